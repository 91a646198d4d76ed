// sort_scan.cu -- device-wide exclusive scan (int64) and stable LSD radix sort of (u64 key, u32 value)
// pairs.  Used once per graph by the Laplacian build (§3.1.1); both are deterministic.
#include "erc_internal.cuh"

namespace erc {

namespace {

constexpr int SCAN_THREADS = 256;
constexpr int SCAN_IPT = 8;
constexpr int SCAN_TILE = SCAN_THREADS * SCAN_IPT;

struct LoadI64 {
  const int64_t* p;
  __device__ int64_t operator()(int64_t i) const { return p[i]; }
};
struct LoadFlag {
  const uint8_t* p;
  __device__ int64_t operator()(int64_t i) const { return (int64_t)p[i]; }
};

// block-wide exclusive scan of one value per thread; returns the exclusive prefix, *block_total
// receives the block's sum
__device__ __forceinline__ int64_t block_exclusive_scan(int64_t v, int64_t* block_total) {
  __shared__ int64_t warp_tot[SCAN_THREADS / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int64_t inc = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int64_t t = __shfl_up_sync(0xffffffffu, inc, o);
    if (lane >= o) inc += t;
  }
  if (lane == 31) warp_tot[warp] = inc;
  __syncthreads();
  if (warp == 0) {
    int64_t t = lane < SCAN_THREADS / 32 ? warp_tot[lane] : 0;
    int64_t ti = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int64_t u = __shfl_up_sync(0xffffffffu, ti, o);
      if (lane >= o) ti += u;
    }
    if (lane < SCAN_THREADS / 32) warp_tot[lane] = ti - t;  // exclusive warp offsets
    if (lane == SCAN_THREADS / 32 - 1) *block_total = ti;
  }
  __syncthreads();
  int64_t r = warp_tot[warp] + inc - v;
  __syncthreads();
  return r;
}

// Single-pass exclusive scan with decoupled look-back (D. Merrill, M. Garland, "Single-pass
// Parallel Prefix Scan with Decoupled Look-back", 2016).  Tiles are claimed in order through an
// atomic ticket, so a tile only waits on tiles that have already started.  Each tile publishes
// its aggregate, then its inclusive prefix, in one 64-bit status word (value << 2 | flag, flag 1
// = aggregate, 2 = inclusive prefix); the tile's first warp walks back over its predecessors,
// 32 at a time, until it meets an inclusive prefix.  Integer sums: the result does not depend on
// the order in which tiles finish.  Inputs are non-negative and their total below 2^62.
// Every poll of a predecessor's status is bounded: after `spin_limit` polls (or once another tile
// has given up) the tile sets the call's abort word and takes the predecessor as an inclusive
// prefix of zero, so its output stays within [0, the true prefix].  A block that starts after the
// abort word is set takes no ticket and does nothing: no tile ever waits on a tile that no block
// has claimed.
constexpr unsigned LOOKBACK_SPINS = 1u << 22;

template <class Load>
__global__ void __launch_bounds__(SCAN_THREADS)
    k_scan_onepass(Load in, int64_t n, unsigned long long* status, unsigned* ticket, int64_t* out,
                   int64_t* total, unsigned* abort, unsigned spin_limit) {
  __shared__ int64_t tile[SCAN_TILE];
  __shared__ unsigned s_tile;
  __shared__ int64_t s_prefix;
  if (threadIdx.x == 0) s_tile = aborted(abort) ? 0xffffffffu : atomicAdd(ticket, 1u);
  __syncthreads();
  if (s_tile == 0xffffffffu) return;
  const int64_t t = s_tile;
  const int64_t base = t * SCAN_TILE;
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    const int j2 = j * SCAN_THREADS + threadIdx.x;
    const int64_t i = base + j2;
    tile[j2] = i < n ? in(i) : 0;
  }
  __syncthreads();
  int64_t v[SCAN_IPT];
  int64_t sum = 0;
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    v[j] = tile[threadIdx.x * SCAN_IPT + j];
    sum += v[j];
  }
  __shared__ int64_t agg;
  const int64_t excl = block_exclusive_scan(sum, &agg);
  volatile unsigned long long* st = status;
  if (threadIdx.x < 32) {  // the first warp publishes and looks back
    const int lane = threadIdx.x;
    if (t == 0) {
      if (lane == 0) {
        st[0] = ((unsigned long long)agg << 2) | 2ull;
        s_prefix = 0;
      }
    } else {
      if (lane == 0) st[t] = ((unsigned long long)agg << 2) | 1ull;
      int64_t prefix = 0;
      int64_t j = t - 1;
      bool done = false;
      while (!done) {
        // lanes read predecessors j, j-1, ..., j-31 (those that exist)
        const int64_t q = j - lane;
        unsigned long long w = 0;
        if (q >= 0) {
          unsigned spins = 0;
          while (((w = st[q]) & 3ull) == 0ull) {
            if (++spins > spin_limit || aborted(abort)) {  // bounded: record it and take zero
              atomicOr(abort, 1u);
              w = 2ull;
              break;
            }
          }
        } else {
          w = 2ull;  // before tile 0: an inclusive prefix of 0
        }
        const unsigned incl = __ballot_sync(0xffffffffu, (w & 3ull) == 2ull);
        const int stop = incl ? __ffs(incl) - 1 : 32;  // nearest inclusive prefix
        int64_t part = lane <= stop ? (int64_t)(w >> 2) : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
        prefix += part;
        done = incl != 0;
        j -= 32;
      }
      if (lane == 0) {
        st[t] = ((unsigned long long)(prefix + agg) << 2) | 2ull;
        s_prefix = prefix;
      }
    }
  }
  __syncthreads();
  int64_t run = excl + s_prefix;
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    tile[threadIdx.x * SCAN_IPT + j] = run;
    run += v[j];
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    const int j2 = j * SCAN_THREADS + threadIdx.x;
    const int64_t i = base + j2;
    if (i < n) out[i] = tile[j2];
  }
  if (total && base + SCAN_TILE >= n && threadIdx.x == 0) *total = s_prefix + agg;
}

inline int64_t scan_blocks(int64_t n) { return (n + SCAN_TILE - 1) / SCAN_TILE; }

// tmp: [status: ntiles u64][ticket]
template <class Load>
erc_status scan_impl(Load in, int64_t n, int64_t* out, int64_t* total, int64_t* tmp,
                     cudaStream_t s, unsigned* abort) {
  if (!abort) return set_error(ERC_ERR_INVALID_ARG, "internal: scan without an abort word");
  if (n <= 0) {
    if (total) ERC_CUDA(cudaMemsetAsync(total, 0, sizeof(int64_t), s));
    return ERC_OK;
  }
  const int64_t nb = scan_blocks(n);
  unsigned long long* status = reinterpret_cast<unsigned long long*>(tmp);
  unsigned* ticket = reinterpret_cast<unsigned*>(status + nb);
  ERC_CUDA(cudaMemsetAsync(status, 0, (size_t)nb * sizeof(unsigned long long) + 8, s));
  k_scan_onepass<<<(unsigned)nb, SCAN_THREADS, 0, s>>>(in, n, status, ticket, out, total, abort,
                                                       wait_limit(LOOKBACK_SPINS));
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  return ERC_OK;
}

// ------------------------------------------------------------------------------------------------
// radix sort: RB-bit digits (8, or 10 while the per-tile count table stays small: 3 passes instead
// of 4 for the 30-bit keys of a 20k-node graph), tiles of 2048 keys; a block's tile is split into
// 8 warp sub-tiles in warp-striped order so that (warp, step, lane) order equals key order, which
// makes the ranks stable.
// ------------------------------------------------------------------------------------------------
constexpr int RS_THREADS = 256;
constexpr int RS_WARPS = RS_THREADS / 32;
constexpr int RS_IPT = 8;
constexpr int RS_TILE = RS_THREADS * RS_IPT;
constexpr int64_t RS_WIDE_MAX_TILES = 4096;  // 10-bit digits up to 8M keys

inline int radix_bits(int64_t n) { return (n + RS_TILE - 1) / RS_TILE <= RS_WIDE_MAX_TILES ? 10 : 8; }

template <int RB>
__global__ void __launch_bounds__(RS_THREADS)
    k_radix_hist(const uint64_t* keys, int64_t n, int shift, int64_t* counts, int64_t nb,
                 const unsigned* abort) {
  constexpr unsigned RADIX = 1u << RB;
  __shared__ unsigned hist[RADIX];
  if (aborted(abort)) return;
  for (unsigned d = threadIdx.x; d < RADIX; d += RS_THREADS) hist[d] = 0;
  __syncthreads();
  const int64_t base = (int64_t)blockIdx.x * RS_TILE;
#pragma unroll
  for (int j = 0; j < RS_IPT; ++j) {
    int64_t i = base + j * RS_THREADS + threadIdx.x;
    if (i < n) atomicAdd(&hist[(unsigned)(keys[i] >> shift) & (RADIX - 1)], 1u);
  }
  __syncthreads();
  for (unsigned d = threadIdx.x; d < RADIX; d += RS_THREADS)
    counts[(int64_t)d * nb + blockIdx.x] = hist[d];
}

template <int RB>
__global__ void __launch_bounds__(RS_THREADS)
    k_radix_scatter(const uint64_t* __restrict__ keys, const uint32_t* __restrict__ vals,
                    uint64_t* __restrict__ keys_out, uint32_t* __restrict__ vals_out, int64_t n,
                    int shift, const int64_t* __restrict__ offsets, int64_t nb,
                    const unsigned* abort) {
  constexpr unsigned RADIX = 1u << RB;
  __shared__ unsigned whist[RS_WARPS][RADIX];
  __shared__ int64_t boff[RADIX];
  if (aborted(abort)) return;  // the offsets of an unfinished scan are not used
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (unsigned d = threadIdx.x; d < RADIX * RS_WARPS; d += RS_THREADS) (&whist[0][0])[d] = 0;
  for (unsigned d = threadIdx.x; d < RADIX; d += RS_THREADS)
    boff[d] = offsets[(int64_t)d * nb + blockIdx.x];
  __syncthreads();
  const int64_t base = (int64_t)blockIdx.x * RS_TILE + (int64_t)warp * 32 * RS_IPT;
  const unsigned lt_mask = (1u << lane) - 1u;
  uint64_t k[RS_IPT];
  uint32_t v[RS_IPT];
  unsigned rank[RS_IPT];
  unsigned dig[RS_IPT];
#pragma unroll
  for (int j = 0; j < RS_IPT; ++j) {
    int64_t i = base + j * 32 + lane;
    bool ok = i < n;
    k[j] = ok ? keys[i] : 0;
    v[j] = ok ? vals[i] : 0;
    unsigned d = ok ? ((unsigned)(k[j] >> shift) & (RADIX - 1)) : RADIX;
    dig[j] = d;
    unsigned peers = __match_any_sync(0xffffffffu, d);
    unsigned before = 0;
    if (ok) before = whist[warp][d];
    __syncwarp();
    if (ok && lane == __ffs(peers) - 1) whist[warp][d] = before + __popc(peers);
    __syncwarp();
    rank[j] = before + __popc(peers & lt_mask);
  }
  __syncthreads();
  // exclusive prefix over warps per digit, plus the block's global offset for the digit
  for (unsigned d = threadIdx.x; d < RADIX; d += RS_THREADS) {
    unsigned run = 0;
    for (int w = 0; w < RS_WARPS; ++w) {
      unsigned t = whist[w][d];
      whist[w][d] = run;
      run += t;
    }
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < RS_IPT; ++j) {
    if (dig[j] < RADIX) {
      int64_t dst = boff[dig[j]] + whist[warp][dig[j]] + rank[j];
      keys_out[dst] = k[j];
      vals_out[dst] = v[j];
    }
  }
}

template <int RB>
erc_status radix_passes(uint64_t* keys, uint32_t* vals, uint64_t* keys_alt, uint32_t* vals_alt,
                        int64_t n, int bits, void* tmp, cudaStream_t s, unsigned* abort) {
  const int64_t nb = (n + RS_TILE - 1) / RS_TILE;
  const size_t cnt = (size_t)nb << RB;
  char* t = static_cast<char*>(tmp);
  int64_t* counts = reinterpret_cast<int64_t*>(t);
  int64_t* offs = reinterpret_cast<int64_t*>(t + ((cnt * sizeof(int64_t) + 255) & ~size_t(255)));
  void* scan_tmp = t + 2 * ((cnt * sizeof(int64_t) + 255) & ~size_t(255));
  uint64_t *ka = keys, *kb = keys_alt;
  uint32_t *va = vals, *vb = vals_alt;
  int passes = 0;
  for (int shift = 0; shift < bits; shift += RB, ++passes) {
    k_radix_hist<RB><<<(unsigned)nb, RS_THREADS, 0, s>>>(ka, n, shift, counts, nb, abort);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    ERC_TRY(exclusive_scan_i64(counts, nullptr, offs, (int64_t)cnt, nullptr, scan_tmp, s, abort));
    k_radix_scatter<RB><<<(unsigned)nb, RS_THREADS, 0, s>>>(ka, va, kb, vb, n, shift, offs, nb,
                                                            abort);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    uint64_t* tk = ka; ka = kb; kb = tk;
    uint32_t* tv = va; va = vb; vb = tv;
  }
  if (passes & 1) {  // the result sits in the alternate buffers: copy it back
    ERC_CUDA(cudaMemcpyAsync(keys, ka, (size_t)n * sizeof(uint64_t), cudaMemcpyDeviceToDevice, s));
    ERC_CUDA(cudaMemcpyAsync(vals, va, (size_t)n * sizeof(uint32_t), cudaMemcpyDeviceToDevice, s));
  }
  return ERC_OK;
}

}  // namespace

size_t scan_temp_bytes(int64_t n) {
  return (size_t)(scan_blocks(n > 0 ? n : 1) + 1) * sizeof(unsigned long long) + 256;
}

erc_status exclusive_scan_i64(const int64_t* in, const uint8_t* flags, int64_t* out, int64_t n,
                              int64_t* total, void* tmp, cudaStream_t s, unsigned* abort) {
  if (in) return scan_impl(LoadI64{in}, n, out, total, static_cast<int64_t*>(tmp), s, abort);
  return scan_impl(LoadFlag{flags}, n, out, total, static_cast<int64_t*>(tmp), s, abort);
}

size_t radix_sort_temp_bytes(int64_t n) {
  const int64_t nb = (n + RS_TILE - 1) / RS_TILE;
  const size_t cnt = (size_t)nb << radix_bits(n);
  return 2 * ((cnt * sizeof(int64_t) + 255) & ~size_t(255)) + scan_temp_bytes((int64_t)cnt);
}

erc_status radix_sort_pairs(uint64_t* keys, uint32_t* vals, uint64_t* keys_alt, uint32_t* vals_alt,
                            int64_t n, int bits, void* tmp, cudaStream_t s, unsigned* abort) {
  if (n <= 1) return ERC_OK;
  if (radix_bits(n) == 10)
    return radix_passes<10>(keys, vals, keys_alt, vals_alt, n, bits, tmp, s, abort);
  return radix_passes<8>(keys, vals, keys_alt, vals_alt, n, bits, tmp, s, abort);
}

}  // namespace erc
