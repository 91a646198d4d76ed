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

template <class Load>
__global__ void __launch_bounds__(SCAN_THREADS) k_scan_reduce(Load in, int64_t n, int64_t* sums) {
  const int64_t base = (int64_t)blockIdx.x * SCAN_TILE;
  int64_t s = 0;
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    int64_t i = base + j * SCAN_THREADS + threadIdx.x;
    if (i < n) s += in(i);
  }
  __shared__ int64_t tot;
  block_exclusive_scan(s, &tot);
  __syncthreads();
  if (threadIdx.x == 0) sums[blockIdx.x] = tot;
}

template <class Load>
__global__ void __launch_bounds__(SCAN_THREADS)
    k_scan_apply(Load in, int64_t n, const int64_t* offsets, int64_t* out, int64_t* total) {
  __shared__ int64_t tile[SCAN_TILE];
  const int64_t base = (int64_t)blockIdx.x * SCAN_TILE;
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    int j2 = j * SCAN_THREADS + threadIdx.x;
    int64_t i = base + j2;
    tile[j2] = i < n ? in(i) : 0;
  }
  __syncthreads();
  int64_t v[SCAN_IPT];
  int64_t s = 0;
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    v[j] = tile[threadIdx.x * SCAN_IPT + j];
    s += v[j];
  }
  __shared__ int64_t tot;
  int64_t run = block_exclusive_scan(s, &tot) + (offsets ? offsets[blockIdx.x] : 0);
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    tile[threadIdx.x * SCAN_IPT + j] = run;
    run += v[j];
  }
  __syncthreads();
#pragma unroll
  for (int j = 0; j < SCAN_IPT; ++j) {
    int j2 = j * SCAN_THREADS + threadIdx.x;
    int64_t i = base + j2;
    if (i < n) out[i] = tile[j2];
  }
  if (total && blockIdx.x == gridDim.x - 1 && threadIdx.x == 0)
    *total = (offsets ? offsets[blockIdx.x] : 0) + tot;
}

inline int64_t scan_blocks(int64_t n) { return (n + SCAN_TILE - 1) / SCAN_TILE; }

template <class Load>
erc_status scan_impl(Load in, int64_t n, int64_t* out, int64_t* total, int64_t* tmp,
                     cudaStream_t s) {
  if (n <= 0) {
    if (total) ERC_CUDA(cudaMemsetAsync(total, 0, sizeof(int64_t), s));
    return ERC_OK;
  }
  int64_t nb = scan_blocks(n);
  if (nb == 1) {
    k_scan_apply<<<1, SCAN_THREADS, 0, s>>>(in, n, (const int64_t*)nullptr, out, total);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    return ERC_OK;
  }
  int64_t* sums = tmp;
  int64_t* rest = tmp + ((nb + 31) & ~int64_t(31));
  k_scan_reduce<<<(unsigned)nb, SCAN_THREADS, 0, s>>>(in, n, sums);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  ERC_TRY(scan_impl(LoadI64{sums}, nb, sums, (int64_t*)nullptr, rest, s));
  k_scan_apply<<<(unsigned)nb, SCAN_THREADS, 0, s>>>(in, n, sums, out, total);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  return ERC_OK;
}

// ------------------------------------------------------------------------------------------------
// radix sort: 8-bit digits, tiles of 2048 keys; a block's tile is split into 8 warp sub-tiles in
// warp-striped order so that (warp, step, lane) order equals key order, which makes the ranks
// stable.
// ------------------------------------------------------------------------------------------------
constexpr int RS_THREADS = 256;
constexpr int RS_WARPS = RS_THREADS / 32;
constexpr int RS_IPT = 8;
constexpr int RS_TILE = RS_THREADS * RS_IPT;
constexpr int RS_RADIX = 256;

__global__ void __launch_bounds__(RS_THREADS)
    k_radix_hist(const uint64_t* keys, int64_t n, int shift, int64_t* counts, int64_t nb) {
  __shared__ unsigned hist[RS_RADIX];
  for (int d = threadIdx.x; d < RS_RADIX; d += RS_THREADS) hist[d] = 0;
  __syncthreads();
  const int64_t base = (int64_t)blockIdx.x * RS_TILE;
#pragma unroll
  for (int j = 0; j < RS_IPT; ++j) {
    int64_t i = base + j * RS_THREADS + threadIdx.x;
    if (i < n) atomicAdd(&hist[(unsigned)(keys[i] >> shift) & 255u], 1u);
  }
  __syncthreads();
  for (int d = threadIdx.x; d < RS_RADIX; d += RS_THREADS)
    counts[(int64_t)d * nb + blockIdx.x] = hist[d];
}

__global__ void __launch_bounds__(RS_THREADS)
    k_radix_scatter(const uint64_t* __restrict__ keys, const uint32_t* __restrict__ vals,
                    uint64_t* __restrict__ keys_out, uint32_t* __restrict__ vals_out, int64_t n,
                    int shift, const int64_t* __restrict__ offsets, int64_t nb) {
  __shared__ unsigned whist[RS_WARPS][RS_RADIX];
  __shared__ int64_t boff[RS_RADIX];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  for (int d = threadIdx.x; d < RS_RADIX * RS_WARPS; d += RS_THREADS) (&whist[0][0])[d] = 0;
  for (int d = threadIdx.x; d < RS_RADIX; d += RS_THREADS)
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
    unsigned d = ok ? ((unsigned)(k[j] >> shift) & 255u) : RS_RADIX;
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
  for (int d = threadIdx.x; d < RS_RADIX; d += RS_THREADS) {
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
    if (dig[j] < RS_RADIX) {
      int64_t dst = boff[dig[j]] + whist[warp][dig[j]] + rank[j];
      keys_out[dst] = k[j];
      vals_out[dst] = v[j];
    }
  }
}

}  // namespace

size_t scan_temp_bytes(int64_t n) {
  size_t total = 0;
  int64_t m = n;
  while (m > SCAN_TILE) {
    int64_t nb = scan_blocks(m);
    total += (size_t)((nb + 31) & ~int64_t(31)) * sizeof(int64_t);
    m = nb;
  }
  return total + 256;
}

erc_status exclusive_scan_i64(const int64_t* in, const uint8_t* flags, int64_t* out, int64_t n,
                              int64_t* total, void* tmp, cudaStream_t s) {
  if (in) return scan_impl(LoadI64{in}, n, out, total, static_cast<int64_t*>(tmp), s);
  return scan_impl(LoadFlag{flags}, n, out, total, static_cast<int64_t*>(tmp), s);
}

size_t radix_sort_temp_bytes(int64_t n) {
  int64_t nb = (n + RS_TILE - 1) / RS_TILE;
  size_t cnt = (size_t)nb * RS_RADIX;
  return 2 * ((cnt * sizeof(int64_t) + 255) & ~size_t(255)) + scan_temp_bytes((int64_t)cnt);
}

erc_status radix_sort_pairs(uint64_t* keys, uint32_t* vals, uint64_t* keys_alt, uint32_t* vals_alt,
                            int64_t n, int bits, void* tmp, cudaStream_t s) {
  if (n <= 1) return ERC_OK;
  int64_t nb = (n + RS_TILE - 1) / RS_TILE;
  size_t cnt = (size_t)nb * RS_RADIX;
  char* t = static_cast<char*>(tmp);
  int64_t* counts = reinterpret_cast<int64_t*>(t);
  int64_t* offs = reinterpret_cast<int64_t*>(t + ((cnt * sizeof(int64_t) + 255) & ~size_t(255)));
  void* scan_tmp = t + 2 * ((cnt * sizeof(int64_t) + 255) & ~size_t(255));
  uint64_t *ka = keys, *kb = keys_alt;
  uint32_t *va = vals, *vb = vals_alt;
  int passes = 0;
  for (int shift = 0; shift < bits; shift += 8, ++passes) {
    k_radix_hist<<<(unsigned)nb, RS_THREADS, 0, s>>>(ka, n, shift, counts, nb);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    ERC_TRY(exclusive_scan_i64(counts, nullptr, offs, (int64_t)cnt, nullptr, scan_tmp, s));
    k_radix_scatter<<<(unsigned)nb, RS_THREADS, 0, s>>>(ka, va, kb, vb, n, shift, offs, nb);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    std::swap(ka, kb);
    std::swap(va, vb);
  }
  if (passes & 1) {
    ERC_CUDA(cudaMemcpyAsync(keys, ka, n * sizeof(uint64_t), cudaMemcpyDeviceToDevice, s));
    ERC_CUDA(cudaMemcpyAsync(vals, va, n * sizeof(uint32_t), cudaMemcpyDeviceToDevice, s));
  }
  return ERC_OK;
}

}  // namespace erc
