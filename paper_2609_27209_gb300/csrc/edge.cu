// edge.cu -- the O(n + m) tail of the path:
//   erc_edge_resistance  R_e += sum_c (X_u,c - X_v,c)^2 over a column batch   (Eq. 6, Algorithm 1)
//   erc_curvature        p_u = 1 - 1/2 sum_v w_uv R_uv, kappa_uv = 2 (p_u + p_v) / R_uv (Eq. 2)
//   erc_sampling_probs   Eq. 7 (with the uniform fallback), Eq. 8, normalisation (§3.2)
#include <cfloat>
#include <mutex>

#include "erc_internal.cuh"

namespace erc {
namespace {

constexpr int T = 256;

__device__ __forceinline__ float4 ld_f4(const float* p) {
  return __ldg(reinterpret_cast<const float4*>(p));
}

// One group of LPR lanes walks a segment of consecutive canonical edges, EB edges at a time with
// every row load of the batch issued before the first use.  Edges are sorted by their smaller
// endpoint, so the X_u loads of a batch mostly hit L1.  The group owns each R_e it touches, so
// the accumulation needs no atomics; per edge the column order and the lane tree are fixed.
template <int LPR, int VPL>
__global__ void __launch_bounds__(T)
    k_edge_resistance(const int32_t* __restrict__ eu, const int32_t* __restrict__ ev, int64_t m,
                      const float* __restrict__ X, int32_t ld, int32_t kc, float* __restrict__ R) {
  constexpr int SEG = 32;
  constexpr int EB = VPL >= 4 ? 1 : 4 / VPL;
  const int gl = threadIdx.x & (LPR - 1);
  const int gpb = T / LPR;
  const int nvec = ld >> 2;
  const unsigned gm = group_mask<LPR>();
  const int64_t nseg = (m + SEG - 1) / SEG;
  for (int64_t sg = (int64_t)blockIdx.x * gpb + threadIdx.x / LPR; sg < nseg;
       sg += (int64_t)gridDim.x * gpb) {
    const int64_t e0 = sg * SEG, e1 = min(m, e0 + SEG);
    for (int64_t eb = e0; eb < e1; eb += EB) {
      float4 xu[EB][VPL], xv[EB][VPL];
      float rold[EB];
#pragma unroll
      for (int k = 0; k < EB; ++k) {
        const bool ok = eb + k < e1;
        const int32_t u = ok ? __ldg(eu + eb + k) : 0, v = ok ? __ldg(ev + eb + k) : 0;
#pragma unroll
        for (int t = 0; t < VPL; ++t) {
          const int q = gl + LPR * t;
          const bool on = ok && q < nvec;
          xu[k][t] = on ? ld_f4(X + (size_t)u * ld + 4 * q) : make_float4(0.f, 0.f, 0.f, 0.f);
          xv[k][t] = on ? ld_f4(X + (size_t)v * ld + 4 * q) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        rold[k] = ok && gl == 0 ? R[eb + k] : 0.f;
      }
#pragma unroll
      for (int k = 0; k < EB; ++k) {
        float s = 0.f;
#pragma unroll
        for (int t = 0; t < VPL; ++t) {
          const int cb = 4 * (gl + LPR * t);
          const float dx = cb + 0 < kc ? xu[k][t].x - xv[k][t].x : 0.f;
          const float dy = cb + 1 < kc ? xu[k][t].y - xv[k][t].y : 0.f;
          const float dz = cb + 2 < kc ? xu[k][t].z - xv[k][t].z : 0.f;
          const float dw = cb + 3 < kc ? xu[k][t].w - xv[k][t].w : 0.f;
          s = fmaf(dx, dx, s);
          s = fmaf(dy, dy, s);
          s = fmaf(dz, dz, s);
          s = fmaf(dw, dw, s);
        }
#pragma unroll
        for (int off = LPR / 2; off > 0; off >>= 1) s += __shfl_xor_sync(gm, s, off, LPR);
        if (gl == 0 && eb + k < e1) R[eb + k] = rold[k] + s;
      }
    }
  }
}


// Row sums of the node kernels: NL lanes per row, each adding its slots in a float pair, then a
// fixed lane tree.  Float pairs keep about 44 bits without float64 arithmetic.
constexpr int NL = 8;

__device__ __forceinline__ float2 group_df_sum(float2 acc, unsigned gm) {
#pragma unroll
  for (int off = NL / 2; off > 0; off >>= 1) {
    float2 o;
    o.x = __shfl_xor_sync(gm, acc.x, off, NL);
    o.y = __shfl_xor_sync(gm, acc.y, off, NL);
    acc = df_add(acc, o);
  }
  return acc;
}

// p_u = 1 - 1/2 sum_{slots j of row u} w_j R[eid_j] (Eq. 2), rounded once to float
inline int node_grid(int32_t n) { return (int)(((int64_t)n + T / NL - 1) / (T / NL)); }

template <bool WEIGHTED>
__global__ void __launch_bounds__(T)
    k_node_curvature(const int64_t* __restrict__ row_ptr, const float* __restrict__ val,
                     const int32_t* __restrict__ eid, const float* __restrict__ R, int32_t n,
                     float* __restrict__ p) {
  const int gl = threadIdx.x & (NL - 1);
  const unsigned gm = group_mask<NL>();
  const int64_t u = (int64_t)blockIdx.x * (T / NL) + threadIdx.x / NL;
  if (u >= n) return;  // whole groups leave together: the grid covers every row once
  float2 acc = make_float2(0.f, 0.f);
  for (int64_t j = row_ptr[u] + gl; j < row_ptr[u + 1]; j += NL) {
    const float r = __ldg(R + __ldg(eid + j));
    acc = WEIGHTED ? df_fma(acc, __ldg(val + j), r) : df_add(acc, make_float2(r, 0.f));
  }
  acc = group_df_sum(acc, gm);
  if (gl == 0) {  // 1 - acc / 2 as a pair, then rounded
    const float2 s = df_two_sum(1.f, -0.5f * acc.x);
    p[u] = __fadd_rn(s.x, __fsub_rn(s.y, 0.5f * acc.y));
  }
}

__global__ void k_edge_curvature(const int32_t* __restrict__ eu, const int32_t* __restrict__ ev,
                                 const float* __restrict__ p, const float* __restrict__ R,
                                 int64_t m, float* __restrict__ kappa) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < m;
       e += (int64_t)gridDim.x * blockDim.x) {
    const float s = p[eu[e]] + p[ev[e]];
    kappa[e] = __fdiv_rn(2.f * s, R[e]);
  }
}

// ---------------------------------------------------------------------------- sampling (§3.2)
struct ProbWork {
  double* qnode;     // [n]
  float* part_min;   // [MAX_GRID]
  float* part_max;   // [MAX_GRID]
  double* part_qn;   // [MAX_GRID]
  double* part_cnt;  // [MAX_GRID]
  double* part_qe;   // [MAX_GRID]
};

void plan_probs(Arena& a, ProbWork& w, int32_t n) {
  w.qnode = a.take<double>(n);
  w.part_min = a.take<float>(MAX_GRID);
  w.part_max = a.take<float>(MAX_GRID);
  w.part_qn = a.take<double>(MAX_GRID);
  w.part_cnt = a.take<double>(MAX_GRID);
  w.part_qe = a.take<double>(MAX_GRID);
}

template <class V, class Op>
__device__ __forceinline__ V block_reduce(V v, Op op, V* sh) {
  sh[threadIdx.x] = v;
  __syncthreads();
  for (int s = blockDim.x / 2; s > 0; s >>= 1) {
    if (threadIdx.x < s) sh[threadIdx.x] = op(sh[threadIdx.x], sh[threadIdx.x + s]);
    __syncthreads();
  }
  V r = sh[0];
  __syncthreads();
  return r;
}

struct MinF {
  __device__ float operator()(float a, float b) const { return fminf(a, b); }
};
struct MaxF {
  __device__ float operator()(float a, float b) const { return fmaxf(a, b); }
};
struct AddD {
  __device__ double operator()(double a, double b) const { return a + b; }
};

__global__ void __launch_bounds__(T)
    k_kappa_minmax(const float* __restrict__ kappa, int64_t m, float* part_min, float* part_max) {
  __shared__ float sh[T];
  float lo = FLT_MAX, hi = -FLT_MAX;
  for (int64_t e = (int64_t)blockIdx.x * T + threadIdx.x; e < m; e += (int64_t)gridDim.x * T) {
    const float k = kappa[e];
    lo = fminf(lo, k);
    hi = fmaxf(hi, k);
  }
  lo = block_reduce(lo, MinF{}, sh);
  hi = block_reduce(hi, MaxF{}, sh);
  if (threadIdx.x == 0) {
    part_min[blockIdx.x] = lo;
    part_max[blockIdx.x] = hi;
  }
}

// Eq. 8: q_e = sqrt(max(-kappa_e + 2 kappa_max, 0)) + 1
__device__ __forceinline__ float edge_weight(float k, float kmax) {
  return sqrtf(fmaxf(-k + 2.f * kmax, 0.f)) + 1.f;
}

// kappa_min and kappa_max from the blocks' partials of k_kappa_minmax, in the same order in every
// block that needs them
__device__ __forceinline__ void kappa_extrema(const float* part_min, const float* part_max,
                                              int nparts, float* sh, float& kmin, float& kmax) {
  float lo = FLT_MAX, hi = -FLT_MAX;
  for (int i = threadIdx.x; i < nparts; i += T) {
    lo = fminf(lo, part_min[i]);
    hi = fmaxf(hi, part_max[i]);
  }
  kmin = block_reduce(lo, MinF{}, sh);
  kmax = block_reduce(hi, MaxF{}, sh);
}

// the Eq. 7 and Eq. 8 weights: blocks [0, gn) take node rows (q_u, per block the sum of q_u and
// the number of non-isolated nodes), blocks [gn, gn + ge) take edges (per block the sum of q_e).
// Node row sums: q_u = sum_{v in N(u)} (kappa_uv - kappa_min) / (kappa_max - kappa_min + eta);
// each difference kappa - kappa_min is exact as a float pair, the row's pair sum is scaled once
// in float64.
__global__ void __launch_bounds__(T)
    k_weights(const int64_t* __restrict__ row_ptr, const int32_t* __restrict__ eid,
              const float* __restrict__ kappa, int32_t n, int64_t m, double eta,
              const float* part_min, const float* part_max, int nmm, int gn,
              double* __restrict__ qnode, double* part_qn, double* part_cnt, double* part_qe) {
  __shared__ float shf[T];
  __shared__ double sh[T];
  float kmin, kmax;
  kappa_extrema(part_min, part_max, nmm, shf, kmin, kmax);
  if ((int)blockIdx.x < gn) {
    const int gl = threadIdx.x & (NL - 1);
    const unsigned gm = group_mask<NL>();
    const double inv = 1.0 / ((double)kmax - (double)kmin + eta);
    double tq = 0.0, tc = 0.0;
    for (int64_t u = (int64_t)blockIdx.x * (T / NL) + threadIdx.x / NL; u < n;
         u += (int64_t)gn * (T / NL)) {  // the same trip count for a group's lanes
      const int64_t j0 = row_ptr[u], j1 = row_ptr[u + 1];
      float2 acc = make_float2(0.f, 0.f);
      for (int64_t j = j0 + gl; j < j1; j += NL)
        acc = df_add(acc, df_two_sum(__ldg(kappa + __ldg(eid + j)), -kmin));
      acc = group_df_sum(acc, gm);
      if (gl == 0) {
        const double q = df_value(acc) * inv;
        qnode[u] = q;
        tq += q;
        tc += j1 > j0 ? 1.0 : 0.0;
      }
    }
    tq = block_reduce(tq, AddD{}, sh);
    tc = block_reduce(tc, AddD{}, sh);
    if (threadIdx.x == 0) {
      part_qn[blockIdx.x] = tq;
      part_cnt[blockIdx.x] = tc;
    }
  } else {
    const int64_t b = (int64_t)blockIdx.x - gn, ge = (int64_t)gridDim.x - gn;
    double acc = 0.0;
    for (int64_t e = b * T + threadIdx.x; e < m; e += ge * T)
      acc += (double)edge_weight(kappa[e], kmax);
    acc = block_reduce(acc, AddD{}, sh);
    if (threadIdx.x == 0) part_qe[b] = acc;
  }
}

// normalisation: every block forms the three totals from all partials itself (same order in
// every block), then scales its share of the node and edge weights
__global__ void k_normalize(const int64_t* __restrict__ row_ptr, const double* __restrict__ qnode,
                            int32_t n, const float* __restrict__ kappa, int64_t m,
                            const float* part_min, const float* part_max, int nmm,
                            const double* part_qn, const double* part_cnt, int gn,
                            const double* part_qe, int ge, float* __restrict__ prob_node,
                            float* __restrict__ prob_edge) {
  __shared__ float shf[T];
  __shared__ double sh[T];
  float kmin, kmax;
  kappa_extrema(part_min, part_max, nmm, shf, kmin, kmax);
  double a = 0.0, b = 0.0, c = 0.0;
  for (int i = threadIdx.x; i < gn; i += T) {
    a += part_qn[i];
    b += part_cnt[i];
  }
  for (int i = threadIdx.x; i < ge; i += T) c += part_qe[i];
  const double tot_n = block_reduce(a, AddD{}, sh);
  const double cnt = block_reduce(b, AddD{}, sh);
  const double tot_e = block_reduce(c, AddD{}, sh);
  const double inv_n = tot_n > 0.0 ? 1.0 / tot_n : 0.0;
  const double uni = cnt > 0.0 ? 1.0 / cnt : 0.0;
  const double inv_e = tot_e > 0.0 ? 1.0 / tot_e : 0.0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n; u += stride) {
    double pr;
    if (tot_n > 0.0)
      pr = qnode[u] * inv_n;
    else  // every Eq. 7 weight vanished: uniform over the nodes with an edge
      pr = row_ptr[u + 1] > row_ptr[u] ? uni : 0.0;
    prob_node[u] = (float)pr;
  }
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < m; e += stride)
    prob_edge[e] = (float)((double)edge_weight(kappa[e], kmax) * inv_e);
}

}  // namespace
}  // namespace erc

using namespace erc;

extern "C" erc_status erc_edge_resistance(const erc_graph* g, const float* X, int32_t ld,
                                          int32_t kc, float* R_acc, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(kc >= 1 && ld >= kc && ld % 4 == 0 && ld <= MAX_LD, "bad kc %d / ld %d", kc, ld);
  ERC_REQUIRE(X && (reinterpret_cast<uintptr_t>(X) & 15) == 0, "X must be 16-byte aligned");
  ERC_REQUIRE(R_acc || g->m == 0, "R_acc is required");
  if (g->m == 0) return ERC_OK;
  cudaStream_t s = as_stream(stream);
  return dispatch_shape(ld / 4, [&](auto lpr, auto vpl) -> erc_status {
    constexpr int LPR = decltype(lpr)::value, VPL = decltype(vpl)::value;
    const int64_t nseg = (g->m + 31) / 32;
    k_edge_resistance<LPR, VPL><<<grid_for(nseg, T / LPR), T, 0, s>>>(g->eu, g->ev, g->m, X, ld,
                                                                       kc, R_acc);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    return ERC_OK;
  });
}

extern "C" erc_status erc_curvature(const erc_graph* g, const float* R, float* p_node,
                                    float* kappa, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(p_node && (kappa || g->m == 0) && (R || g->m == 0), "R, p_node, kappa required");
  cudaStream_t s = as_stream(stream);
  if (g->val)
    k_node_curvature<true><<<node_grid(g->n), T, 0, s>>>(g->row_ptr, g->val, g->csr_eid,
                                                                R, g->n, p_node);
  else
    k_node_curvature<false><<<node_grid(g->n), T, 0, s>>>(g->row_ptr, g->val, g->csr_eid,
                                                                 R, g->n, p_node);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  if (g->m > 0) {
    k_edge_curvature<<<grid_for(g->m, T), T, 0, s>>>(g->eu, g->ev, p_node, R, g->m, kappa);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
  }
  return ERC_OK;
}

extern "C" size_t erc_sampling_probs_workspace_size(int32_t n, int64_t m) {
  (void)m;
  if (n < 1) return 0;
  Arena a(nullptr);
  ProbWork w;
  plan_probs(a, w, n);
  return a.used + 256;
}

extern "C" erc_status erc_sampling_probs(const erc_graph* g, const float* kappa, float eta,
                                         float* prob_node, float* prob_edge, void* ws,
                                         size_t ws_bytes, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(eta > 0.f && isfinite(eta), "eta must be positive");
  ERC_REQUIRE(prob_node && ((kappa && prob_edge) || g->m == 0), "kappa and outputs required");
  if (ws_bytes < erc_sampling_probs_workspace_size(g->n, g->m))
    return set_error(ERC_ERR_CAPACITY, "workspace too small");
  cudaStream_t s = as_stream(stream);
  Arena ar(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  ProbWork w;
  plan_probs(ar, w, g->n);
  if (g->m == 0) {
    ERC_CUDA(cudaMemsetAsync(prob_node, 0, (size_t)g->n * sizeof(float), s));
    return ERC_OK;
  }
  const int ge = grid_for(g->m, T);
  k_kappa_minmax<<<ge, T, 0, s>>>(kappa, g->m, w.part_min, w.part_max);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  const int gn = grid_for(g->n, T / NL);
  const int gq = grid_for(g->m, T);  // edge blocks of the weights kernel (<= MAX_GRID partials)
  k_weights<<<gn + gq, T, 0, s>>>(g->row_ptr, g->csr_eid, kappa, g->n, g->m, (double)eta,
                                  w.part_min, w.part_max, ge, gn, w.qnode, w.part_qn, w.part_cnt,
                                  w.part_qe);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  k_normalize<<<grid_for(g->n > g->m ? g->n : g->m, T), T, 0, s>>>(
      g->row_ptr, w.qnode, g->n, kappa, g->m, w.part_min, w.part_max, ge, w.part_qn,
      w.part_cnt, gn, w.part_qe, gq, prob_node, prob_edge);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  return ERC_OK;
}

// ------------------------------------------------------------------------------------------------
// erc_sampling_probs_noalloc: erc_sampling_probs for callers that cannot allocate device memory.
// Its scratch is this file-scope device array instead of a caller workspace.  The array exists on
// every device that loads the library and stays allocated until the process exits.
// ------------------------------------------------------------------------------------------------
static __device__ __align__(256) unsigned char g_probs_noalloc_scratch[ERC_SAMPLING_PROBS_NOALLOC_SCRATCH_BYTES];

namespace erc {
namespace {
// The identity of the calling thread's current CUDA context (cuCtxGetId, reached through the
// runtime's driver entry points so that the library does not link the driver library): 0 when
// it cannot be read.  Context ids are never reused within a process.
unsigned long long current_context_id() {
  using GetCurrent = int (*)(void**);
  using GetId = int (*)(void*, unsigned long long*);
  static GetCurrent get_current = nullptr;
  static GetId get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 4000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrent>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetId>(f);
    cudaGetLastError();
  });
  void* ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != 0 || !ctx || get_id(ctx, &id) != 0) return 0;
  return id;
}

// The array's device address, looked up with cudaGetSymbolAddress the first time a device is used
// in a context and cached under (device, context id): a device reset destroys the context, the
// module is loaded again in the next one and the array may then sit elsewhere, so a new context
// means a new lookup.  In host code the symbol names a host-side stand-in, never the device
// memory, so kernels only ever receive this looked-up address.
erc_status noalloc_scratch(void** out) {
  static std::mutex mu;
  static void* addr[64] = {};
  static unsigned long long ctx_of[64] = {};
  int dev = 0;
  ERC_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= 64) return set_error(ERC_ERR_CUDA, "device ordinal %d out of range", dev);
  // 0 when no context is current yet (the lookup below makes the primary context current): the
  // next call then looks up once more
  const unsigned long long ctx = current_context_id();
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev] || ctx == 0 || ctx != ctx_of[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_probs_noalloc_scratch);
    if (e != cudaSuccess || !p)
      return set_error(ERC_ERR_CUDA, "cudaGetSymbolAddress(scratch) failed on device %d: %s",
                       dev, cudaGetErrorString(e));
    addr[dev] = p;
    ctx_of[dev] = ctx;
  }
  *out = addr[dev];
  return ERC_OK;
}
}  // namespace
}  // namespace erc

extern "C" erc_status erc_sampling_probs_noalloc(const erc_graph* g, const float* kappa,
                                                 float eta, float* prob_node, float* prob_edge,
                                                 erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  if (g->n > ERC_SAMPLING_PROBS_NOALLOC_MAX_NODES)
    return set_error(ERC_ERR_CAPACITY,
                     "erc_sampling_probs_noalloc handles at most %d nodes (got %d); use "
                     "erc_sampling_probs with a caller workspace",
                     ERC_SAMPLING_PROBS_NOALLOC_MAX_NODES, g->n);
  const size_t need = erc_sampling_probs_workspace_size(g->n, g->m);
  if (need > sizeof(g_probs_noalloc_scratch))
    return set_error(ERC_ERR_CAPACITY, "scratch needs %zu bytes, the static array holds %zu",
                     need, sizeof(g_probs_noalloc_scratch));
  void* scratch = nullptr;
  ERC_TRY(noalloc_scratch(&scratch));
  // every word of the scratch that this call reads is written earlier in the same call, so the
  // previous call's leftovers need no clearing
  return erc_sampling_probs(g, kappa, eta, prob_node, prob_edge, scratch,
                            sizeof(g_probs_noalloc_scratch), stream);
}
