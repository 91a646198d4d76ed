// erc_internal.cuh -- shared internals of liberc.so (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <cstddef>
#include <type_traits>
#include <utility>

#include "erc.h"

namespace erc {

// ------------------------------------------------------------------------------------------------
// host-side errors
// ------------------------------------------------------------------------------------------------
erc_status set_error(erc_status code, const char* fmt, ...);
void clear_error();

#define ERC_CUDA(call)                                                                    \
  do {                                                                                    \
    cudaError_t e_ = (call);                                                              \
    if (e_ != cudaSuccess)                                                                \
      return ::erc::set_error(ERC_ERR_CUDA, "%s:%d %s: %s", __FILE__, __LINE__, #call,      \
                              cudaGetErrorString(e_));                                    \
  } while (0)

#define ERC_TRY(expr)                   \
  do {                                  \
    erc_status st_ = (expr);            \
    if (st_ != ERC_OK) return st_;      \
  } while (0)

#define ERC_REQUIRE(cond, ...)                                          \
  do {                                                                  \
    if (!(cond)) return ::erc::set_error(ERC_ERR_INVALID_ARG, __VA_ARGS__); \
  } while (0)

inline cudaStream_t as_stream(erc_stream s) { return reinterpret_cast<cudaStream_t>(s); }

// SM count of the current device (cached per device).
int sm_count();

// Polls a bounded device-side wait makes before it gives up: `dflt` (the wait's own limit) unless
// erc_set_wait_limit() set a process-wide override.  Read when work is enqueued (it is a kernel
// argument, and part of the key of every cached graph that holds such a kernel).
unsigned wait_limit(unsigned dflt);

// process-wide count of kernels this library has launched (graph launches add the kernels they
// contain); launches recorded while a graph is being captured are not counted
void count_launches(long long k);
void set_capturing(bool on);

// A launch sequence replayed as a CUDA graph: `enqueue` is captured once per key (on a private
// stream of the current device) into an executable graph, kept in a small least-recently-used
// cache, and launched on `s`.  The key must hold everything the sequence depends on: pointers,
// sizes, scalars and the device.  Host reads of device results stay outside the sequence.
struct GraphKey {
  static constexpr int WORDS = 32;
  uint64_t w[WORDS] = {};
  int n = 0;
  GraphKey& add(uint64_t v) {
    if (n < WORDS) w[n++] = v;
    return *this;
  }
  GraphKey& add(const void* p) { return add((uint64_t)(uintptr_t)p); }
};
template <class F>
erc_status graph_launch(GraphKey key, F&& enqueue, cudaStream_t s);
erc_status graph_launch_impl(const GraphKey& key, erc_status (*enqueue)(void*, cudaStream_t),
                             void* ctx, cudaStream_t s);
template <class F>
erc_status graph_launch(GraphKey key, F&& enqueue, cudaStream_t s) {
  using Fn = std::remove_reference_t<F>;
  auto thunk = [](void* c, cudaStream_t cs) -> erc_status { return (*static_cast<Fn*>(c))(cs); };
  return graph_launch_impl(key, thunk, const_cast<void*>(static_cast<const void*>(&enqueue)), s);
}

// Internal forms of the entry points for the whole-path driver.
//   build_laplacian_impl: erc_build_laplacian, plus *nonunit (host, may be null) = 1 when some
//     merged weight differs from 1 (always 1 for weighted input), read with m in one round trip.
//   cg_enqueue: erc_batched_cg (erc_batched_pcg with precond) up to the true residual, without
//     reading the status; the status flags accumulate over calls until reset_flags (the
//     multi-kernel solver still polls its own progress).  cg_status reads them once: the status
//     of every batch since the last reset.
erc_status build_laplacian_impl(int32_t n, const int32_t* src, const int32_t* dst, const float* w,
                                int64_t m_in, int32_t dup_policy, int64_t* row_ptr, int32_t* col,
                                float* val, float* deg, int32_t* csr_eid, int32_t* eu, int32_t* ev,
                                float* ew, int64_t* m_out, void* ws, size_t ws_bytes,
                                cudaStream_t s, int* nonunit);
erc_status cg_enqueue(const erc_graph* g, float eps, const float* Y, float* X, int32_t ld,
                      int32_t kc, float tol, int32_t max_iter, int32_t* iters, float* relres,
                      void* ws, size_t ws_bytes, cudaStream_t s, bool reset_flags,
                      cudaEvent_t ev0, cudaEvent_t ev1, int32_t* path, bool precond);
erc_status cg_status(int32_t n, int32_t ld, int32_t columns, int32_t max_iter, void* ws,
                     cudaStream_t s);

// ------------------------------------------------------------------------------------------------
// workspace carving: the same plan runs once to size (base == nullptr) and once to carve
// ------------------------------------------------------------------------------------------------
struct Arena {
  char* base;
  size_t used = 0;
  explicit Arena(void* b) : base(static_cast<char*>(b)) {}
  template <class T>
  T* take(size_t count) {
    used = (used + 255) & ~size_t(255);
    T* p = base ? reinterpret_cast<T*>(base + used) : nullptr;
    used += count * sizeof(T);
    return p;
  }
};

// ------------------------------------------------------------------------------------------------
// double-float ("float2" hi + lo) accumulation: error-free transformations on float32 units.
// GB300 runs float64 at a small fraction of its float32 rate, so long dot products are kept in a
// float pair (about 44 significant bits) and only the final per-column values go to float64.
// ------------------------------------------------------------------------------------------------
__device__ __forceinline__ float2 df_two_sum(float a, float b) {
  float s = __fadd_rn(a, b);
  float bb = __fsub_rn(s, a);
  float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return make_float2(s, e);
}
__device__ __forceinline__ float2 df_norm(float hi, float e) {
  float h = __fadd_rn(hi, e);
  return make_float2(h, __fsub_rn(e, __fsub_rn(h, hi)));
}
__device__ __forceinline__ float2 df_add(float2 a, float2 b) {
  float2 s = df_two_sum(a.x, b.x);
  return df_norm(s.x, __fadd_rn(s.y, __fadd_rn(a.y, b.y)));
}
// acc + a*b with the product kept exact (a*b = p + pe)
__device__ __forceinline__ float2 df_fma(float2 acc, float a, float b) {
  float p = __fmul_rn(a, b);
  float pe = __fmaf_rn(a, b, -p);
  float2 s = df_two_sum(acc.x, p);
  return df_norm(s.x, __fadd_rn(s.y, __fadd_rn(acc.y, pe)));
}
__device__ __forceinline__ double df_value(float2 a) { return (double)a.x + (double)a.y; }
__device__ __forceinline__ float2 df_from_double(double v) {
  const float hi = (float)v;
  return make_float2(hi, (float)(v - (double)hi));
}
// Philox4x32-10 block function (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds of two 32x32->64
// multiplies, with the key bumped by the Weyl constants between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
    k.x += 0x9E3779B9u;
    k.y += 0xBB67AE85u;
  }
  return c;
}

// (a.x + a.y) / (b.x + b.y) rounded to float, without float64 arithmetic: Dekker's pair division
// (T. J. Dekker, "A floating-point technique for extending the available precision", 1971) with
// one correction step.  q0 b.x is subtracted exactly by the fused multiply-add.
__device__ __forceinline__ float df_div(float2 a, float2 b) {
  const float q0 = __fdiv_rn(a.x, b.x);
  const float r = __fadd_rn(__fmaf_rn(-q0, b.x, a.x), a.y);
  return __fadd_rn(q0, __fdiv_rn(__fmaf_rn(-q0, b.y, r), b.x));
}

// ------------------------------------------------------------------------------------------------
// deterministic grid-wide per-column reduction of float2 partials.
// Blocks publish their partial row; the last block of each group of RED_GROUP blocks sums the
// group in block order, and the last group-finisher sums the group rows in group order.  The
// result does not depend on which block arrives when.  Counters must be zero at kernel start; the
// finishers reset them, so consecutive launches on one stream can share the buffers.
// ------------------------------------------------------------------------------------------------
constexpr int RED_GROUP = 32;
constexpr int MAX_GRID = 8192;  // the largest grid any reducing kernel launches

struct ColReduce {
  float2* part1;  // [MAX_GRID][ld]
  float2* part2;  // [MAX_GRID / RED_GROUP][ld]
  unsigned* cnt;  // [MAX_GRID / RED_GROUP + 1]
};

inline void plan_colreduce(Arena& a, ColReduce& cr, int ld) {
  cr.part1 = a.take<float2>((size_t)MAX_GRID * ld);
  cr.part2 = a.take<float2>((size_t)(MAX_GRID / RED_GROUP) * ld);
  cr.cnt = a.take<unsigned>(MAX_GRID / RED_GROUP + 1);
}
inline size_t colreduce_counter_bytes() { return sizeof(unsigned) * (MAX_GRID / RED_GROUP + 1); }

// All threads of every block call this once `bpart` (shared, ld entries) holds the block's
// partial.  Returns true in exactly one block, whose `res` (shared, ld entries) then holds the
// totals.
__device__ __forceinline__ bool grid_colreduce(const ColReduce& cr, const float2* bpart,
                                               float2* res, int ld) {
  __shared__ int s_last;
  const int G = gridDim.x, b = blockIdx.x;
  const int grp = b / RED_GROUP;
  const int ng = (G + RED_GROUP - 1) / RED_GROUP;
  const int gsize = min(RED_GROUP, G - grp * RED_GROUP);
  for (int c = threadIdx.x; c < ld; c += blockDim.x) cr.part1[(size_t)b * ld + c] = bpart[c];
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = (atomicAdd(&cr.cnt[grp], 1u) == (unsigned)(gsize - 1));
  __syncthreads();
  if (!s_last) return false;
  __threadfence();
  for (int c = threadIdx.x; c < ld; c += blockDim.x) {
    float2 acc = make_float2(0.f, 0.f);
    const float2* src = cr.part1 + (size_t)grp * RED_GROUP * ld + c;
    float2 v[RED_GROUP];  // issue every load before the (ordered) additions
#pragma unroll
    for (int k = 0; k < RED_GROUP; ++k)
      v[k] = k < gsize ? __ldcg(src + (size_t)k * ld) : make_float2(0.f, 0.f);
#pragma unroll
    for (int k = 0; k < RED_GROUP; ++k) acc = df_add(acc, v[k]);
    cr.part2[(size_t)grp * ld + c] = acc;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    cr.cnt[grp] = 0;
    s_last = (atomicAdd(&cr.cnt[ng], 1u) == (unsigned)(ng - 1));
  }
  __syncthreads();
  if (!s_last) return false;
  __threadfence();
  for (int c = threadIdx.x; c < ld; c += blockDim.x) {
    float2 acc = make_float2(0.f, 0.f);
    for (int k0 = 0; k0 < ng; k0 += 16) {
      float2 v[16];
#pragma unroll
      for (int k = 0; k < 16; ++k)
        v[k] = k0 + k < ng ? __ldcg(cr.part2 + (size_t)(k0 + k) * ld + c) : make_float2(0.f, 0.f);
#pragma unroll
      for (int k = 0; k < 16; ++k) acc = df_add(acc, v[k]);
    }
    res[c] = acc;
  }
  if (threadIdx.x == 0) cr.cnt[ng] = 0;
  __syncthreads();
  return true;
}

// gpu-scope release/acquire primitives (PTX memory model)
__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* p, unsigned v) {
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v)
               : "memory");
  return old;
}

// Ordered column sums of G rows of partials (part: [G][ld] float pairs, written by other blocks
// of the same launch, read through L2): threads take fixed segments of the rows for a pair of
// columns each, every load of a chunk in flight, then the segments are added in order, so any
// block computes the same totals.  res: ld entries; tmp: shared scratch of 2 * blockDim.x.
__device__ __forceinline__ void colsum_rows(const float2* part, int G, int ld, float2* res,
                                            float2* tmp) {
  const int bd = blockDim.x;
  const int half = ld >> 1;  // column pairs: one float4 of two float-pairs per load
  if (half <= bd) {
    constexpr int CHUNK = 20;
    const int nseg = bd / half;
    const int per = (G + nseg - 1) / nseg;
    const int seg = threadIdx.x / half, cp = threadIdx.x % half;
    if (seg < nseg) {
      const int k0 = seg * per, k1 = min(G, k0 + per);
      float2 a0 = make_float2(0.f, 0.f), a1 = make_float2(0.f, 0.f);
      for (int k = k0; k < k1; k += CHUNK) {
        float4 v[CHUNK];
#pragma unroll
        for (int j = 0; j < CHUNK; ++j)
          v[j] = k + j < k1
                     ? __ldcg(reinterpret_cast<const float4*>(part + (size_t)(k + j) * ld) + cp)
                     : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < CHUNK; ++j) {
          a0 = df_add(a0, make_float2(v[j].x, v[j].y));
          a1 = df_add(a1, make_float2(v[j].z, v[j].w));
        }
      }
      tmp[seg * ld + 2 * cp] = a0;
      tmp[seg * ld + 2 * cp + 1] = a1;
    }
    __syncthreads();
    for (int c = threadIdx.x; c < ld; c += bd) {
      float2 acc = make_float2(0.f, 0.f);
      for (int s = 0; s < nseg; ++s) acc = df_add(acc, tmp[s * ld + c]);
      res[c] = acc;
    }
  } else {
    for (int c = threadIdx.x; c < ld; c += bd) {
      float2 acc = make_float2(0.f, 0.f);
      for (int k = 0; k < G; k += 8) {
        float2 v[8];
#pragma unroll
        for (int j = 0; j < 8; ++j)
          v[j] = k + j < G ? __ldcg(part + (size_t)(k + j) * ld + c) : make_float2(0.f, 0.f);
#pragma unroll
        for (int j = 0; j < 8; ++j) acc = df_add(acc, v[j]);
      }
      res[c] = acc;
    }
  }
  __syncthreads();
}

// colsum_rows for float partials (part: [G][ld] floats, ld a multiple of 4, ld <= 2 blockDim.x):
// four columns per load, float-pair sums in a fixed order; tmp holds 2 * blockDim.x entries.  For partials that are sums of squares, whose
// rounding to float costs at most 2^-24 of the total.
__device__ __forceinline__ void colsum_rows_f(const float* part, int G, int ld, float2* res,
                                              float2* tmp) {
  const int bd = blockDim.x;
  const int quads = ld >> 2;
  constexpr int CHUNK = 20;
  // segments of the rows, as many as the threads and tmp's 2 * blockDim.x entries allow
  const int nseg = max(1, min(quads <= bd ? bd / quads : 1, (2 * bd) / ld));
  const int per = (G + nseg - 1) / nseg;
  for (int t = threadIdx.x; t < nseg * quads; t += bd) {
    const int seg = t / quads, cq = t % quads;
    const int k0 = seg * per, k1 = min(G, k0 + per);
    float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                   make_float2(0.f, 0.f)};
    for (int k = k0; k < k1; k += CHUNK) {
      float4 v[CHUNK];
#pragma unroll
      for (int j = 0; j < CHUNK; ++j)
        v[j] = k + j < k1
                   ? __ldcg(reinterpret_cast<const float4*>(part + (size_t)(k + j) * ld) + cq)
                   : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int j = 0; j < CHUNK; ++j) {
        a[0] = df_add(a[0], make_float2(v[j].x, 0.f));
        a[1] = df_add(a[1], make_float2(v[j].y, 0.f));
        a[2] = df_add(a[2], make_float2(v[j].z, 0.f));
        a[3] = df_add(a[3], make_float2(v[j].w, 0.f));
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) tmp[seg * ld + 4 * cq + i] = a[i];
  }
  __syncthreads();
  for (int c = threadIdx.x; c < ld; c += bd) {
    float2 acc = make_float2(0.f, 0.f);
    for (int s = 0; s < nseg; ++s) acc = df_add(acc, tmp[s * ld + c]);
    res[c] = acc;
  }
  __syncthreads();
}

// ------------------------------------------------------------------------------------------------
// row-block shapes: a row of ld floats is nvec = ld/4 float4s, handled by a group of LPR lanes
// with VPL float4s per lane (LPR * VPL >= nvec).
// ------------------------------------------------------------------------------------------------
template <int V>
using ic = std::integral_constant<int, V>;

template <class F>
inline erc_status dispatch_shape(int nvec, F&& f) {
  if (nvec <= 4) return f(ic<4>{}, ic<1>{});
  if (nvec <= 8) return f(ic<8>{}, ic<1>{});
  if (nvec <= 16) return f(ic<16>{}, ic<1>{});
  if (nvec <= 32) return f(ic<32>{}, ic<1>{});
  if (nvec <= 64) return f(ic<32>{}, ic<2>{});
  if (nvec <= 128) return f(ic<32>{}, ic<4>{});
  if (nvec <= 256) return f(ic<32>{}, ic<8>{});
  return set_error(ERC_ERR_INVALID_ARG, "ld > 1024 is not supported");
}

constexpr int MAX_LD = 1024;

template <int LPR>
__device__ __forceinline__ unsigned group_mask() {
  if constexpr (LPR == 32) {
    return 0xffffffffu;
  } else {
    const unsigned lane = threadIdx.x & 31u;
    return ((1u << LPR) - 1u) << (lane & ~(unsigned)(LPR - 1));
  }
}

// blocks of `kernel` that fit on one SM at `threads` threads (cached per kernel and device)
int resident_per_sm(const void* kernel, int threads, size_t smem = 0);

// a one-wave grid: min(resident blocks on the whole GPU, blocks the work needs), at least 1
inline int one_wave_grid(const void* kernel, int threads, long long work_blocks) {
  long long g = (long long)resident_per_sm(kernel, threads) * sm_count();
  if (work_blocks < g) g = work_blocks;
  if (g > MAX_GRID) g = MAX_GRID;
  return g < 1 ? 1 : (int)g;
}

// grid size for a grid-stride kernel: at most `waves` resident waves of blocks, at least 1
inline int grid_for(long long work_items, int items_per_block, int waves_blocks_per_sm = 8) {
  long long g = (work_items + items_per_block - 1) / items_per_block;
  long long cap = (long long)sm_count() * waves_blocks_per_sm;
  if (g > cap) g = cap;
  if (g > MAX_GRID) g = MAX_GRID;
  if (g < 1) g = 1;
  return (int)g;
}

// A call's abort word (device): a bounded wait that gives up sets it, and every later kernel of
// the same call that would consume the unfinished result returns at once when it is set; the host
// reads it once the call's work has finished and reports ERC_ERR_TIMEOUT.
__device__ __forceinline__ bool aborted(const unsigned* abort) {
  return *reinterpret_cast<const volatile unsigned*>(abort) != 0u;
}

// ------------------------------------------------------------------------------------------------
// internal entry points shared between translation units
// ------------------------------------------------------------------------------------------------
erc_status check_graph(const erc_graph* g);
size_t scan_temp_bytes(int64_t n);
// exclusive scan of int64 `in` (or of the 0/1 flags in `flags` when `in` is null) into `out`;
// `total` (device, may be null) receives the sum.  `abort` (device, required) is the call's abort
// word: the scan does nothing when it is already set, and sets it when a bounded look-back wait
// gives up (the output is then incomplete; every entry stays within [0, the true value]).
erc_status exclusive_scan_i64(const int64_t* in, const uint8_t* flags, int64_t* out, int64_t n,
                              int64_t* total, void* tmp, cudaStream_t s, unsigned* abort);
size_t radix_sort_temp_bytes(int64_t n);
// stable LSD radix sort of (key, value) pairs on the low `bits` key bits; the result is in
// keys/vals (the *_alt buffers are scratch of the same size).  `abort` as for the scan: once it
// is set no further pass runs and the result is undefined.
erc_status radix_sort_pairs(uint64_t* keys, uint32_t* vals, uint64_t* keys_alt, uint32_t* vals_alt,
                            int64_t n, int bits, void* tmp, cudaStream_t s, unsigned* abort);

}  // namespace erc
