// cg.cu -- column-wise CG on L_eps X = Y (Eq. 5, §3.1.3, Algorithm 1) and the operator
// L_eps P = eps P + (D - A) P it iterates on.
//
// One CG iteration is two kernels over the row-major n x ld block:
//   k_spmm<MODE_STEP>  AP = L_eps P: a group of LPR lanes gathers the neighbour rows of one
//                      light row (float4 along the columns); rows heavier than H are taken by a
//                      whole block, its groups splitting the row and combining in a fixed order.
//                      Per-column p.Ap partials; the last block to finish forms alpha = rr / pAp.
//   k_update_fused     x += alpha p, r -= alpha Ap and r.r; the last block forms beta, counts the
//                      iteration and retires converged columns, then releases a grid barrier;
//                      every block then applies p = r + beta p to its rows.  Launched
//                      cooperatively (all blocks resident), the barrier wait is bounded.
// Reductions are deterministic: fixed groupings and orders, float-pair accumulation.  S
// iterations are captured once into a CUDA graph and relaunched; kernels return at once when no
// column is active, so the host only polls the "any active" flag between graph launches.
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "erc_internal.cuh"

namespace erc {
namespace {

constexpr int T = 256;
constexpr int WARPS = T / 32;
constexpr int SMEM_FLOATS = 8192;  // 32 KB: heavy-row combine buffer, or the reduction buffers
constexpr unsigned SPIN_LIMIT = 1u << 24;
enum { MODE_STEP = 0, MODE_APPLY = 1, MODE_RESID = 2 };

struct HeavyRows {
  uint8_t* flag;    // [n]
  int64_t* pos;     // [n]
  int32_t* list;    // [n] rows with more than H neighbours, ascending
  int64_t* count;   // [1]
  void* scan_tmp;
};

void plan_heavy(Arena& a, HeavyRows& h, int32_t n) {
  h.flag = a.take<uint8_t>(n);
  h.pos = a.take<int64_t>(n);
  h.list = a.take<int32_t>(n);
  h.count = a.take<int64_t>(1);
  h.scan_tmp = a.take<char>(scan_temp_bytes(n));
}

struct CgWork {
  float *R, *P, *AP;
  float *alpha, *beta;
  double *rr, *yy;
  int *active, *conv, *iters;
  int* flags;  // [0] any column active [1] numeric trouble [2] unconverged columns [3] timeout
  unsigned* gen;  // generation counter of the update kernel's grid barrier
  ColReduce cr;
  HeavyRows heavy;
};

void plan_cg(Arena& a, CgWork& w, int32_t n, int32_t ld) {
  const size_t blk = (size_t)n * ld;
  w.R = a.take<float>(blk);
  w.P = a.take<float>(blk);
  w.AP = a.take<float>(blk);
  w.alpha = a.take<float>(ld);
  w.beta = a.take<float>(ld);
  w.rr = a.take<double>(ld);
  w.yy = a.take<double>(ld);
  w.active = a.take<int>(ld);
  w.conv = a.take<int>(ld);
  w.iters = a.take<int>(ld);
  w.flags = a.take<int>(8);
  w.gen = a.take<unsigned>(8);
  plan_colreduce(a, w.cr, ld);
  plan_heavy(a, w.heavy, n);
}

struct SpmmArgs {
  const int64_t* row_ptr;
  const int32_t* col;
  const float* val;
  int32_t n, ld, kc;
  float eps;
  int32_t H;               // rows with more than H neighbours are split over a block
  const int32_t* heavy;    // their ids, ascending
  const int64_t* nheavy;   // their number (device)
  const float* P;  // operand: P (step/apply) or X (residual)
  float* AP;       // output of step/apply
  const float* Y;  // residual mode
  ColReduce cr;
  float* alpha;
  const double* rr;
  int* active;
  int* flags;
  double* pap_out;  // apply mode, may be null
  const double* yy;
  const int* iters;
  const int* conv;
  float* relres_out;
  int32_t* iters_out;
};

__device__ __forceinline__ float4 ld_f4(const float* p) {
  return __ldg(reinterpret_cast<const float4*>(p));
}
__device__ __forceinline__ float4 f4_zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }

// per-warp then per-block combination of per-thread column partials of a row-group kernel with
// NW warps; the cross-warp step runs over chunks of CH columns (scratch holds NW x CH)
template <int LPR, int VPL, int NW, int CH>
__device__ __forceinline__ void block_partials_groups(float2 (&d)[VPL][4], float2* sbuf,
                                                      float2* scratch, int ld) {
#pragma unroll
  for (int off = LPR; off < 32; off <<= 1) {
#pragma unroll
    for (int v = 0; v < VPL; ++v)
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        float2 o;
        o.x = __shfl_xor_sync(0xffffffffu, d[v][t].x, off);
        o.y = __shfl_xor_sync(0xffffffffu, d[v][t].y, off);
        d[v][t] = df_add(d[v][t], o);
      }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int cb = 0; cb < ld; cb += CH) {
    if (lane < LPR) {
#pragma unroll
      for (int v = 0; v < VPL; ++v)
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int c = 4 * (lane + LPR * v) + t;
          if (c >= cb && c < cb + CH && c < ld) scratch[warp * CH + (c - cb)] = d[v][t];
        }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < CH && cb + c < ld; c += blockDim.x) {
      float2 acc = make_float2(0.f, 0.f);
      for (int w = 0; w < NW; ++w) acc = df_add(acc, scratch[w * CH + c]);
      sbuf[cb + c] = acc;
    }
    __syncthreads();
  }
}

// per-warp then per-block combination of per-thread column partials of a row-group kernel
template <int LPR, int VPL>
__device__ __forceinline__ void block_partials_rowgroup(float2 (&d)[VPL][4], float2* sbuf,
                                                        float2* scratch, int ld) {
#pragma unroll
  for (int off = LPR; off < 32; off <<= 1) {
#pragma unroll
    for (int v = 0; v < VPL; ++v)
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        float2 o;
        o.x = __shfl_xor_sync(0xffffffffu, d[v][t].x, off);
        o.y = __shfl_xor_sync(0xffffffffu, d[v][t].y, off);
        d[v][t] = df_add(d[v][t], o);
      }
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int cb = 0; cb < ld; cb += 256) {
    if (lane < LPR) {
#pragma unroll
      for (int v = 0; v < VPL; ++v)
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const int c = 4 * (lane + LPR * v) + t;
          if (c >= cb && c < cb + 256 && c < ld) scratch[warp * 256 + (c - cb)] = d[v][t];
        }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < 256 && cb + c < ld; c += blockDim.x) {
      float2 acc = make_float2(0.f, 0.f);
      for (int w = 0; w < WARPS; ++w) acc = df_add(acc, scratch[w * 256 + c]);
      sbuf[cb + c] = acc;
    }
    __syncthreads();
  }
}

// acc += sum_{j in [j0, j1)} w_j (p_u - p_{col_j}) for this lane's float4 column slots.
// L2ONLY loads p through L2 only: required where p is rewritten within the same launch.
template <int LPR, int VPL, bool WEIGHTED, bool L2ONLY = false>
__device__ __forceinline__ void gather_range(const SpmmArgs& a, int gl, unsigned gm, int nvec,
                                             const float4 (&pu)[VPL], int64_t j0, int64_t j1,
                                             float4 (&acc)[VPL]) {
  constexpr int U = VPL >= 8 ? 1 : 8 / VPL;  // neighbour rows in flight per group
  for (int64_t jb = j0; jb < j1; jb += LPR) {
    const int64_t jj = jb + gl;
    int32_t cidx = 0;
    float wv = 1.f;
    if (jj < j1) {
      cidx = __ldg(a.col + jj);
      if (WEIGHTED) wv = __ldg(a.val + jj);
    }
    const int cnt = (int)min((int64_t)LPR, j1 - jb);
    // batches of U neighbour rows, the last one predicated: every load of a batch is issued
    // before the first FMA, so a row costs ceil(deg / U) dependent trips
    for (int t = 0; t < cnt; t += U) {
      int cj[U];
      float wj[U];
      float4 pv[U][VPL];
#pragma unroll
      for (int k = 0; k < U; ++k) {
        cj[k] = __shfl_sync(gm, cidx, (t + k) & (LPR - 1), LPR);
        wj[k] = WEIGHTED ? __shfl_sync(gm, wv, (t + k) & (LPR - 1), LPR) : 1.f;
        if (t + k >= cnt) wj[k] = 0.f;
      }
#pragma unroll
      for (int k = 0; k < U; ++k)
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          const int q = gl + LPR * v;
          const float* src = a.P + (size_t)cj[k] * a.ld + 4 * q;
          pv[k][v] = (q < nvec && t + k < cnt)
                         ? (L2ONLY ? __ldcg(reinterpret_cast<const float4*>(src)) : ld_f4(src))
                         : pu[v];
        }
#pragma unroll
      for (int k = 0; k < U; ++k)
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          acc[v].x = fmaf(wj[k], pu[v].x - pv[k][v].x, acc[v].x);
          acc[v].y = fmaf(wj[k], pu[v].y - pv[k][v].y, acc[v].y);
          acc[v].z = fmaf(wj[k], pu[v].z - pv[k][v].z, acc[v].z);
          acc[v].w = fmaf(wj[k], pu[v].w - pv[k][v].w, acc[v].w);
        }
    }
  }
}

// L_eps p_u = eps p_u + acc: store it (step/apply) or y_u minus it (residual), and add this
// lane's column contributions to the dot partials (p.Ap, or |y - L x|^2)
template <int LPR, int VPL, int MODE>
__device__ __forceinline__ void finish_row(const SpmmArgs& a, int64_t u, int gl, int nvec,
                                           const float4 (&pu)[VPL], const float4 (&acc)[VPL],
                                           float2 (&dot)[VPL][4]) {
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int q = gl + LPR * v;
    if (q >= nvec) continue;
    float4 o;
    o.x = fmaf(a.eps, pu[v].x, acc[v].x);
    o.y = fmaf(a.eps, pu[v].y, acc[v].y);
    o.z = fmaf(a.eps, pu[v].z, acc[v].z);
    o.w = fmaf(a.eps, pu[v].w, acc[v].w);
    if (MODE == MODE_RESID) {
      const float4 y = ld_f4(a.Y + (size_t)u * a.ld + 4 * q);
      const int cb = 4 * q;
      o.x = cb + 0 < a.kc ? y.x - o.x : 0.f;
      o.y = cb + 1 < a.kc ? y.y - o.y : 0.f;
      o.z = cb + 2 < a.kc ? y.z - o.z : 0.f;
      o.w = cb + 3 < a.kc ? y.w - o.w : 0.f;
      dot[v][0] = df_fma(dot[v][0], o.x, o.x);
      dot[v][1] = df_fma(dot[v][1], o.y, o.y);
      dot[v][2] = df_fma(dot[v][2], o.z, o.z);
      dot[v][3] = df_fma(dot[v][3], o.w, o.w);
    } else {
      reinterpret_cast<float4*>(a.AP + (size_t)u * a.ld)[q] = o;
      dot[v][0] = df_fma(dot[v][0], pu[v].x, o.x);
      dot[v][1] = df_fma(dot[v][1], pu[v].y, o.y);
      dot[v][2] = df_fma(dot[v][2], pu[v].z, o.z);
      dot[v][3] = df_fma(dot[v][3], pu[v].w, o.w);
    }
  }
}

template <int LPR, int VPL>
__device__ __forceinline__ void load_row(const SpmmArgs& a, int64_t u, int gl, int nvec,
                                         float4 (&pu)[VPL], float4 (&acc)[VPL]) {
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int q = gl + LPR * v;
    pu[v] = q < nvec ? ld_f4(a.P + (size_t)u * a.ld + 4 * q) : f4_zero();
    acc[v] = f4_zero();
  }
}

template <int LPR, int VPL, bool WEIGHTED, int MODE>
__global__ void __launch_bounds__(T, VPL <= 2 ? 3 : VPL == 4 ? 2 : 1) k_spmm(SpmmArgs a) {
  if (MODE == MODE_STEP && *(volatile int*)a.flags == 0) return;
  __shared__ __align__(16) float smem[SMEM_FLOATS];
  constexpr int GPB = T / LPR;  // groups per block
  const int gl = threadIdx.x & (LPR - 1);
  const int gi = threadIdx.x / LPR;
  const int nvec = a.ld >> 2;
  const unsigned gm = group_mask<LPR>();
  float2 dot[VPL][4];
#pragma unroll
  for (int v = 0; v < VPL; ++v)
#pragma unroll
    for (int t = 0; t < 4; ++t) dot[v][t] = make_float2(0.f, 0.f);

  // heavy rows: one block per row, its GPB groups take equal slices of the neighbour list and
  // group 0 adds the slices in group order
  const int64_t nheavy = a.nheavy ? *a.nheavy : 0;
  for (int64_t h = blockIdx.x; h < nheavy; h += gridDim.x) {
    const int64_t u = a.heavy[h];
    const int64_t j0 = a.row_ptr[u], j1 = a.row_ptr[u + 1];
    const int64_t per = (j1 - j0 + GPB - 1) / GPB;
    const int64_t s0 = min(j1, j0 + gi * per), s1 = min(j1, s0 + per);
    float4 pu[VPL], acc[VPL];
    load_row<LPR, VPL>(a, u, gl, nvec, pu, acc);
    gather_range<LPR, VPL, WEIGHTED>(a, gl, gm, nvec, pu, s0, s1, acc);
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      if (q < nvec) reinterpret_cast<float4*>(smem + gi * a.ld)[q] = acc[v];
    }
    __syncthreads();
    if (gi == 0) {
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        const int q = gl + LPR * v;
        if (q >= nvec) continue;
        float4 s = f4_zero();
        for (int g = 0; g < GPB; ++g) {
          const float4 c = reinterpret_cast<const float4*>(smem + g * a.ld)[q];
          s.x += c.x;
          s.y += c.y;
          s.z += c.z;
          s.w += c.w;
        }
        acc[v] = s;
      }
      finish_row<LPR, VPL, MODE>(a, u, gl, nvec, pu, acc, dot);
    }
    __syncthreads();
  }

  // light rows: one group per row
  const int64_t ngroups = (int64_t)gridDim.x * GPB;
  for (int64_t u = (int64_t)blockIdx.x * GPB + gi; u < a.n; u += ngroups) {
    const int64_t j0 = a.row_ptr[u], j1 = a.row_ptr[u + 1];
    if (j1 - j0 > a.H) continue;
    float4 pu[VPL], acc[VPL];
    load_row<LPR, VPL>(a, u, gl, nvec, pu, acc);
    gather_range<LPR, VPL, WEIGHTED>(a, gl, gm, nvec, pu, j0, j1, acc);
    finish_row<LPR, VPL, MODE>(a, u, gl, nvec, pu, acc, dot);
  }
  if (MODE == MODE_APPLY && a.pap_out == nullptr) return;

  float2* sbuf = reinterpret_cast<float2*>(smem);
  float2* scratch = reinterpret_cast<float2*>(smem + 2 * MAX_LD);
  __syncthreads();
  block_partials_rowgroup<LPR, VPL>(dot, sbuf, scratch, a.ld);
  if (!grid_colreduce(a.cr, sbuf, sbuf, a.ld)) return;
  for (int c = threadIdx.x; c < a.ld; c += blockDim.x) {
    const double v = df_value(sbuf[c]);
    if (MODE == MODE_STEP) {
      float al = 0.f;
      if (a.active[c]) {
        const double q = a.rr[c] / v;
        if (!(v > 0.0) || !isfinite(q)) {
          a.active[c] = 0;
          atomicOr(&a.flags[1], 1);
        } else {
          al = (float)q;
        }
      }
      a.alpha[c] = al;
    } else if (MODE == MODE_APPLY) {
      if (c < a.kc) a.pap_out[c] = v;
    } else {
      if (c < a.kc) {
        const double y2 = a.yy[c];
        a.relres_out[c] = y2 > 0.0 ? (float)sqrt(v / y2) : 0.f;
        a.iters_out[c] = a.iters[c];
        if (!a.conv[c]) atomicAdd(&a.flags[2], 1);
      }
    }
  }
}

// ---------------------------------------------------------------------------- vector kernels
// Each thread keeps one column quad q (4 columns) and walks the rows, so its partial sums
// belong to fixed columns.  Threads per block = nvec * (256 / nvec).
struct VecArgs {
  int32_t n, ld, kc;
  double tol2;
  int32_t max_iter;
  const float* Y;
  float *X, *R, *P, *AP;
  float *alpha, *beta;
  double *rr, *yy;
  int *active, *conv, *iters, *flags;
  unsigned* gen;
  ColReduce cr;
};

__device__ __forceinline__ void block_partials_quad(const float2 (&d)[4], float2* red,
                                                    float2* sbuf, int ld, int nvec) {
#pragma unroll
  for (int t = 0; t < 4; ++t) red[threadIdx.x * 4 + t] = d[t];
  __syncthreads();
  const int rb = blockDim.x / nvec;
  for (int c = threadIdx.x; c < ld; c += blockDim.x) {
    const int q = c >> 2, t = c & 3;
    float2 acc = make_float2(0.f, 0.f);
    for (int r = 0; r < rb; ++r) acc = df_add(acc, red[(r * nvec + q) * 4 + t]);
    sbuf[c] = acc;
  }
  __syncthreads();
}

__global__ void __launch_bounds__(T) k_cg_init(VecArgs a) {
  __shared__ float2 red[T * 4];
  __shared__ float2 sbuf[MAX_LD];
  const int nvec = a.ld >> 2, rb = blockDim.x / nvec;
  const int q = threadIdx.x % nvec;
  float2 d[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
  const int cb = 4 * q;
  for (int64_t row = (int64_t)blockIdx.x * rb + threadIdx.x / nvec; row < a.n;
       row += (int64_t)gridDim.x * rb) {
    const size_t i = (size_t)row * a.ld + cb;
    float4 y = ld_f4(a.Y + i);
    if (cb + 0 >= a.kc) y.x = 0.f;
    if (cb + 1 >= a.kc) y.y = 0.f;
    if (cb + 2 >= a.kc) y.z = 0.f;
    if (cb + 3 >= a.kc) y.w = 0.f;
    *reinterpret_cast<float4*>(a.R + i) = y;
    *reinterpret_cast<float4*>(a.P + i) = y;
    *reinterpret_cast<float4*>(a.X + i) = f4_zero();
    d[0] = df_fma(d[0], y.x, y.x);
    d[1] = df_fma(d[1], y.y, y.y);
    d[2] = df_fma(d[2], y.z, y.z);
    d[3] = df_fma(d[3], y.w, y.w);
  }
  block_partials_quad(d, red, sbuf, a.ld, nvec);
  if (!grid_colreduce(a.cr, sbuf, sbuf, a.ld)) return;
  int any = 0;
  for (int c = threadIdx.x; c < a.ld; c += blockDim.x) {
    const double v = df_value(sbuf[c]);
    a.yy[c] = v;
    a.rr[c] = v;
    a.iters[c] = 0;
    a.alpha[c] = 0.f;
    a.beta[c] = 0.f;
    int act = 0, cv = 1;
    if (c < a.kc) {
      if (!isfinite(v)) {
        atomicOr(&a.flags[1], 1);
        cv = 0;
      } else if (v > 0.0 && !(v <= a.tol2 * v)) {
        act = 1;
        cv = 0;
      }
    }
    a.active[c] = act;
    a.conv[c] = cv;
    any |= act;
  }
  any = __syncthreads_or(any);
  if (threadIdx.x == 0) a.flags[0] = any;
}

// x += alpha p, r -= alpha Ap, r.r  |grid barrier: beta, convergence|  p = r + beta p
__global__ void __launch_bounds__(T) k_update_fused(VecArgs a) {
  if (*(volatile int*)a.flags == 0) return;
  __shared__ float2 red[T * 4];
  __shared__ float2 sbuf[MAX_LD];
  __shared__ unsigned s_gen;
  if (threadIdx.x == 0) s_gen = ld_acquire(a.gen);
  const int nvec = a.ld >> 2, rb = blockDim.x / nvec;
  const int q = threadIdx.x % nvec;
  const int64_t row0 = (int64_t)blockIdx.x * rb + threadIdx.x / nvec;
  const int64_t rstep = (int64_t)gridDim.x * rb;
  const float4 al = *reinterpret_cast<const float4*>(a.alpha + 4 * q);
  float2 d[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
  if (al.x != 0.f || al.y != 0.f || al.z != 0.f || al.w != 0.f) {
    for (int64_t row = row0; row < a.n; row += rstep) {
      const size_t i = (size_t)row * a.ld + 4 * q;
      float4 x = *reinterpret_cast<const float4*>(a.X + i);
      float4 r = *reinterpret_cast<const float4*>(a.R + i);
      const float4 p = *reinterpret_cast<const float4*>(a.P + i);
      const float4 ap = *reinterpret_cast<const float4*>(a.AP + i);
      x.x = fmaf(al.x, p.x, x.x);
      x.y = fmaf(al.y, p.y, x.y);
      x.z = fmaf(al.z, p.z, x.z);
      x.w = fmaf(al.w, p.w, x.w);
      r.x = fmaf(-al.x, ap.x, r.x);
      r.y = fmaf(-al.y, ap.y, r.y);
      r.z = fmaf(-al.z, ap.z, r.z);
      r.w = fmaf(-al.w, ap.w, r.w);
      *reinterpret_cast<float4*>(a.X + i) = x;
      *reinterpret_cast<float4*>(a.R + i) = r;
      d[0] = df_fma(d[0], r.x, r.x);
      d[1] = df_fma(d[1], r.y, r.y);
      d[2] = df_fma(d[2], r.z, r.z);
      d[3] = df_fma(d[3], r.w, r.w);
    }
  }
  block_partials_quad(d, red, sbuf, a.ld, nvec);
  if (grid_colreduce(a.cr, sbuf, sbuf, a.ld)) {
    int any = 0;
    for (int c = threadIdx.x; c < a.ld; c += blockDim.x) {
      float be = 0.f;
      if (a.active[c]) {
        const double rn = df_value(sbuf[c]);
        const int it = a.iters[c] + 1;
        a.iters[c] = it;
        if (!isfinite(rn)) {
          a.active[c] = 0;
          atomicOr(&a.flags[1], 1);
        } else {
          be = (float)(rn / a.rr[c]);
          a.rr[c] = rn;
          if (rn <= a.tol2 * a.yy[c]) {
            a.conv[c] = 1;
            a.active[c] = 0;
          } else if (it >= a.max_iter) {
            a.active[c] = 0;
          }
        }
      }
      a.beta[c] = be;
      any |= a.active[c];
    }
    any = __syncthreads_or(any);
    if (threadIdx.x == 0) {
      a.flags[0] = any;
      __threadfence();
      red_release_add(a.gen, 1u);  // release the blocks waiting for beta
    }
  } else if (threadIdx.x == 0) {
    unsigned spins = 0;
    while (ld_acquire(a.gen) == s_gen) {
      if (++spins > SPIN_LIMIT) {  // bounded: flag the timeout and fall through
        atomicOr(&a.flags[3], 1);
        break;
      }
      __nanosleep(64);
    }
  }
  __syncthreads();
  const int4 act = __ldcg(reinterpret_cast<const int4*>(a.active + 4 * q));
  if (!(act.x | act.y | act.z | act.w)) return;
  const float4 be = __ldcg(reinterpret_cast<const float4*>(a.beta + 4 * q));
  for (int64_t row = row0; row < a.n; row += rstep) {
    const size_t i = (size_t)row * a.ld + 4 * q;
    const float4 r = *reinterpret_cast<const float4*>(a.R + i);
    float4 p = *reinterpret_cast<const float4*>(a.P + i);
    if (act.x) p.x = fmaf(be.x, p.x, r.x);
    if (act.y) p.y = fmaf(be.y, p.y, r.y);
    if (act.z) p.z = fmaf(be.z, p.z, r.z);
    if (act.w) p.w = fmaf(be.w, p.w, r.w);
    *reinterpret_cast<float4*>(a.P + i) = p;
  }
}

// ---------------------------------------------------------------------------- resident CG
// When r and Ap of every row fit in the SMs' shared memory, one cooperative launch runs the whole
// solve.  Block b owns rows [b rb, b rb + rb): their r and Ap live in its shared memory, x and p
// in global memory (p is gathered by other blocks).  Per iteration:
//   A  Ap = L_eps p for own rows (heavy rows by the whole block), p.Ap   -> reduce, alpha
//   B  x += alpha p, r -= alpha Ap, r.r                                  -> reduce, beta, stop test
//   C  p = r + beta p                                                    -> barrier
// Every reduce and barrier is a bounded wait on one generation counter.  Data written by other
// blocks inside the launch (p, scalars) is read through L2 (ld.global.cg), never through L1.
constexpr int PT = 512;
constexpr int PWARPS = PT / 32;
constexpr int PCH = 64;

struct ResArgs {
  SpmmArgs s;
  VecArgs v;
  int32_t rb;  // rows per block
};

__device__ __forceinline__ float4 ldcg_f4(const float* p) {
  return __ldcg(reinterpret_cast<const float4*>(p));
}

// wait until the generation counter moves past `g` (bounded; sets flags[3] on timeout)
__device__ __forceinline__ void wait_generation(unsigned* gen, unsigned g, int* flags) {
  if (threadIdx.x == 0) {
    unsigned spins = 0;
    while (ld_acquire(gen) == g) {  // one L2 round trip per poll: ~2^22 polls is seconds
      if (++spins > (1u << 22)) {
        atomicOr(&flags[3], 1);
        break;
      }
    }
  }
  __syncthreads();
}

// plain grid barrier on (count, generation); every block calls it the same number of times.
// The __syncthreads before thread 0's acquire-release arrival orders the whole block's writes.
__device__ __forceinline__ void grid_barrier(unsigned* cnt, unsigned* gen, int* flags) {
  __shared__ unsigned s_g;
  __syncthreads();
  if (threadIdx.x == 0) {
    s_g = ld_acquire(gen);
    if (atom_add_acq_rel(cnt, 1u) == gridDim.x - 1) {
      atomicExch(cnt, 0u);
      red_release_add(gen, 1u);
    }
  }
  __syncthreads();
  wait_generation(gen, s_g, flags);
}

template <int LPR, int VPL, bool WEIGHTED>
__global__ void __launch_bounds__(PT, 1) k_cg_resident(ResArgs ra) {
  extern __shared__ __align__(16) float dsm[];
  const SpmmArgs& a = ra.s;
  const VecArgs& va = ra.v;
  constexpr int GPB = PT / LPR;
  const int gl = threadIdx.x & (LPR - 1);
  const int gi = threadIdx.x / LPR;
  const int ld = a.ld, nvec = ld >> 2;
  const unsigned gm = group_mask<LPR>();
  const int64_t r0 = (int64_t)blockIdx.x * ra.rb;
  const int nrows = (int)max((int64_t)0, min((int64_t)a.n, r0 + ra.rb) - r0);
  float* rs = dsm;                                     // [rb][ld]  r of own rows
  float* aps = rs + (size_t)ra.rb * ld;                // [rb][ld]  Ap of own rows
  float* comb = aps + (size_t)ra.rb * ld;              // [GPB][ld] heavy-row slices
  float2* sbuf = reinterpret_cast<float2*>(comb + (size_t)GPB * ld);  // [ld]
  float2* scratch = sbuf + ld;                         // [PWARPS][PCH]
  __shared__ unsigned s_gen;
  __shared__ int64_t s_h0, s_h1;
  unsigned* bar_cnt = va.gen + 1;

  for (int idx = threadIdx.x; idx < nrows * nvec; idx += PT) {
    const int i = idx / nvec, q = idx % nvec;
    reinterpret_cast<float4*>(rs + (size_t)i * ld)[q] = ldcg_f4(va.R + (size_t)(r0 + i) * ld + 4 * q);
  }
  if (threadIdx.x == 0) {  // this block's slice of the ascending heavy-row list
    const int64_t nh = a.nheavy ? *a.nheavy : 0;
    int64_t lo = 0, hi = nh;
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (a.heavy[mid] < r0) lo = mid + 1; else hi = mid;
    }
    s_h0 = lo;
    hi = nh;
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (a.heavy[mid] < r0 + nrows) lo = mid + 1; else hi = mid;
    }
    s_h1 = lo;
  }
  __syncthreads();

  while (true) {
    if (*(volatile int*)&va.flags[0] == 0 || *(volatile int*)&va.flags[3] != 0) break;
    // ---------------- A: Ap = L_eps p on own rows, p.Ap
    float2 dot[VPL][4];
#pragma unroll
    for (int v = 0; v < VPL; ++v)
#pragma unroll
      for (int t = 0; t < 4; ++t) dot[v][t] = make_float2(0.f, 0.f);
    for (int64_t h = s_h0; h < s_h1; ++h) {
      const int64_t u = a.heavy[h];
      const int64_t j0 = a.row_ptr[u], j1 = a.row_ptr[u + 1];
      const int64_t per = (j1 - j0 + GPB - 1) / GPB;
      const int64_t s0 = min(j1, j0 + gi * per), s1 = min(j1, s0 + per);
      float4 pu[VPL], acc[VPL];
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        const int q = gl + LPR * v;
        pu[v] = q < nvec ? ldcg_f4(a.P + (size_t)u * ld + 4 * q) : f4_zero();
        acc[v] = f4_zero();
      }
      gather_range<LPR, VPL, WEIGHTED, true>(a, gl, gm, nvec, pu, s0, s1, acc);
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        const int q = gl + LPR * v;
        if (q < nvec) reinterpret_cast<float4*>(comb + gi * ld)[q] = acc[v];
      }
      __syncthreads();
      if (gi == 0) {
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          const int q = gl + LPR * v;
          if (q >= nvec) continue;
          float4 s = f4_zero();
          for (int g = 0; g < GPB; ++g) {
            const float4 c = reinterpret_cast<const float4*>(comb + g * ld)[q];
            s.x += c.x;
            s.y += c.y;
            s.z += c.z;
            s.w += c.w;
          }
          float4 o;
          o.x = fmaf(a.eps, pu[v].x, s.x);
          o.y = fmaf(a.eps, pu[v].y, s.y);
          o.z = fmaf(a.eps, pu[v].z, s.z);
          o.w = fmaf(a.eps, pu[v].w, s.w);
          reinterpret_cast<float4*>(aps + (size_t)(u - r0) * ld)[q] = o;
          dot[v][0] = df_fma(dot[v][0], pu[v].x, o.x);
          dot[v][1] = df_fma(dot[v][1], pu[v].y, o.y);
          dot[v][2] = df_fma(dot[v][2], pu[v].z, o.z);
          dot[v][3] = df_fma(dot[v][3], pu[v].w, o.w);
        }
      }
      __syncthreads();
    }
    for (int i = gi; i < nrows; i += GPB) {
      const int64_t u = r0 + i;
      const int64_t j0 = a.row_ptr[u], j1 = a.row_ptr[u + 1];
      if (j1 - j0 > a.H) continue;
      float4 pu[VPL], acc[VPL];
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        const int q = gl + LPR * v;
        pu[v] = q < nvec ? ldcg_f4(a.P + (size_t)u * ld + 4 * q) : f4_zero();
        acc[v] = f4_zero();
      }
      gather_range<LPR, VPL, WEIGHTED, true>(a, gl, gm, nvec, pu, j0, j1, acc);
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        const int q = gl + LPR * v;
        if (q >= nvec) continue;
        float4 o;
        o.x = fmaf(a.eps, pu[v].x, acc[v].x);
        o.y = fmaf(a.eps, pu[v].y, acc[v].y);
        o.z = fmaf(a.eps, pu[v].z, acc[v].z);
        o.w = fmaf(a.eps, pu[v].w, acc[v].w);
        reinterpret_cast<float4*>(aps + (size_t)i * ld)[q] = o;
        dot[v][0] = df_fma(dot[v][0], pu[v].x, o.x);
        dot[v][1] = df_fma(dot[v][1], pu[v].y, o.y);
        dot[v][2] = df_fma(dot[v][2], pu[v].z, o.z);
        dot[v][3] = df_fma(dot[v][3], pu[v].w, o.w);
      }
    }
    if (threadIdx.x == 0) s_gen = ld_acquire(va.gen);
    __syncthreads();
    block_partials_groups<LPR, VPL, PWARPS, PCH>(dot, sbuf, scratch, ld);
    if (grid_colreduce_flat(a.cr, sbuf, sbuf, scratch, ld)) {
      for (int c = threadIdx.x; c < ld; c += PT) {
        const double v = df_value(sbuf[c]);
        float al = 0.f;
        if (*(volatile int*)&va.active[c]) {
          const double q = *(volatile double*)&va.rr[c] / v;
          if (!(v > 0.0) || !isfinite(q)) {
            va.active[c] = 0;
            atomicOr(&va.flags[1], 1);
          } else {
            al = (float)q;
          }
        }
        va.alpha[c] = al;
      }
      __syncthreads();
      if (threadIdx.x == 0) red_release_add(va.gen, 1u);  // orders the block's writes above
    } else {
      wait_generation(va.gen, s_gen, va.flags);
    }
    __syncthreads();

    // ---------------- B: x += alpha p, r -= alpha Ap, r.r
    float4 al[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      al[v] = q < nvec ? ldcg_f4(va.alpha + 4 * q) : f4_zero();
    }
#pragma unroll
    for (int v = 0; v < VPL; ++v)
#pragma unroll
      for (int t = 0; t < 4; ++t) dot[v][t] = make_float2(0.f, 0.f);
    for (int i = gi; i < nrows; i += GPB) {
      const size_t ig = (size_t)(r0 + i) * ld;
#pragma unroll
      for (int v = 0; v < VPL; ++v) {
        const int q = gl + LPR * v;
        if (q >= nvec) continue;
        const float4 p = ldcg_f4(a.P + ig + 4 * q);
        float4 x = *reinterpret_cast<const float4*>(va.X + ig + 4 * q);
        float4 r = reinterpret_cast<const float4*>(rs + (size_t)i * ld)[q];
        const float4 ap = reinterpret_cast<const float4*>(aps + (size_t)i * ld)[q];
        x.x = fmaf(al[v].x, p.x, x.x);
        x.y = fmaf(al[v].y, p.y, x.y);
        x.z = fmaf(al[v].z, p.z, x.z);
        x.w = fmaf(al[v].w, p.w, x.w);
        r.x = fmaf(-al[v].x, ap.x, r.x);
        r.y = fmaf(-al[v].y, ap.y, r.y);
        r.z = fmaf(-al[v].z, ap.z, r.z);
        r.w = fmaf(-al[v].w, ap.w, r.w);
        *reinterpret_cast<float4*>(va.X + ig + 4 * q) = x;
        reinterpret_cast<float4*>(rs + (size_t)i * ld)[q] = r;
        dot[v][0] = df_fma(dot[v][0], r.x, r.x);
        dot[v][1] = df_fma(dot[v][1], r.y, r.y);
        dot[v][2] = df_fma(dot[v][2], r.z, r.z);
        dot[v][3] = df_fma(dot[v][3], r.w, r.w);
      }
    }
    if (threadIdx.x == 0) s_gen = ld_acquire(va.gen);
    __syncthreads();
    block_partials_groups<LPR, VPL, PWARPS, PCH>(dot, sbuf, scratch, ld);
    if (grid_colreduce_flat(a.cr, sbuf, sbuf, scratch, ld)) {
      int any = 0;
      for (int c = threadIdx.x; c < ld; c += PT) {
        float be = 0.f;
        int act = *(volatile int*)&va.active[c];
        if (act) {
          const double rn = df_value(sbuf[c]);
          const int it = *(volatile int*)&va.iters[c] + 1;
          va.iters[c] = it;
          if (!isfinite(rn)) {
            act = 0;
            atomicOr(&va.flags[1], 1);
          } else {
            be = (float)(rn / *(volatile double*)&va.rr[c]);
            va.rr[c] = rn;
            if (rn <= va.tol2 * *(volatile double*)&va.yy[c]) {
              va.conv[c] = 1;
              act = 0;
            } else if (it >= va.max_iter) {
              act = 0;
            }
          }
          va.active[c] = act;
        }
        va.beta[c] = be;
        any |= act;
      }
      any = __syncthreads_or(any);
      if (threadIdx.x == 0) {
        va.flags[0] = any;
        red_release_add(va.gen, 1u);  // orders the block's writes above
      }
    } else {
      wait_generation(va.gen, s_gen, va.flags);
    }
    __syncthreads();

    // ---------------- C: p = r + beta p on active columns
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      if (q >= nvec) continue;
      const int4 act = __ldcg(reinterpret_cast<const int4*>(va.active + 4 * q));
      if (!(act.x | act.y | act.z | act.w)) continue;
      const float4 be = ldcg_f4(va.beta + 4 * q);
      for (int i = gi; i < nrows; i += GPB) {
        const size_t ig = (size_t)(r0 + i) * ld + 4 * q;
        const float4 r = reinterpret_cast<const float4*>(rs + (size_t)i * ld)[q];
        float4 p = ldcg_f4(a.P + ig);
        if (act.x) p.x = fmaf(be.x, p.x, r.x);
        if (act.y) p.y = fmaf(be.y, p.y, r.y);
        if (act.z) p.z = fmaf(be.z, p.z, r.z);
        if (act.w) p.w = fmaf(be.w, p.w, r.w);
        *reinterpret_cast<float4*>(const_cast<float*>(a.P) + ig) = p;
      }
    }
    grid_barrier(bar_cnt, va.gen, va.flags);
  }
}

// ---------------------------------------------------------------------------- heavy rows
__global__ void k_mark_heavy(const int64_t* __restrict__ row_ptr, int32_t n, int32_t H,
                             uint8_t* __restrict__ flag) {
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n;
       u += (int64_t)gridDim.x * blockDim.x)
    flag[u] = (row_ptr[u + 1] - row_ptr[u]) > H;
}
__global__ void k_list_heavy(const uint8_t* __restrict__ flag, const int64_t* __restrict__ pos,
                             int32_t n, int32_t* __restrict__ list) {
  for (int64_t u = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; u < n;
       u += (int64_t)gridDim.x * blockDim.x)
    if (flag[u]) list[pos[u]] = (int32_t)u;
}

// ---------------------------------------------------------------------------- launch helpers
inline int vec_threads(int nvec) { return nvec * (T / nvec); }

template <int MODE>
const void* spmm_kernel(int nvec, bool weighted) {
  const void* k = nullptr;
  dispatch_shape(nvec, [&](auto lpr, auto vpl) -> erc_status {
    constexpr int LPR = decltype(lpr)::value, VPL = decltype(vpl)::value;
    k = weighted ? (const void*)k_spmm<LPR, VPL, true, MODE>
                 : (const void*)k_spmm<LPR, VPL, false, MODE>;
    return ERC_OK;
  });
  return k;
}

// grid and heavy threshold of the operator for this graph: one wave of blocks, and rows heavier
// than about twice the mean work of a group are split over a block
void spmm_shape(const erc_graph* g, int ld, int* grid, int32_t* H) {
  const int nvec = ld / 4;
  int lpr = nvec <= 4 ? 4 : nvec <= 8 ? 8 : nvec <= 16 ? 16 : 32;
  const int gpb = T / lpr;
  *grid = one_wave_grid(spmm_kernel<MODE_STEP>(nvec, g->val != nullptr), T,
                        ((long long)g->n + gpb - 1) / gpb);
  const long long groups = (long long)(*grid) * gpb;
  long long h = 2 * g->m / (2 * groups);
  if (h < 32) h = 32;
  if (h > (1 << 20)) h = 1 << 20;
  *H = (int32_t)h;
}

erc_status build_heavy(const erc_graph* g, int32_t H, const HeavyRows& hv, cudaStream_t s) {
  const int grid = grid_for(g->n, 256);
  k_mark_heavy<<<grid, 256, 0, s>>>(g->row_ptr, g->n, H, hv.flag);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  ERC_TRY(exclusive_scan_i64(nullptr, hv.flag, hv.pos, g->n, hv.count, hv.scan_tmp, s));
  k_list_heavy<<<grid, 256, 0, s>>>(hv.flag, hv.pos, g->n, hv.list);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  return ERC_OK;
}

template <int MODE>
erc_status launch_spmm(const SpmmArgs& a, int grid, cudaStream_t s) {
  return dispatch_shape(a.ld / 4, [&](auto lpr, auto vpl) -> erc_status {
    constexpr int LPR = decltype(lpr)::value, VPL = decltype(vpl)::value;
    if (a.val)
      k_spmm<LPR, VPL, true, MODE><<<grid, T, 0, s>>>(a);
    else
      k_spmm<LPR, VPL, false, MODE><<<grid, T, 0, s>>>(a);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    return ERC_OK;
  });
}

int update_grid(int32_t n, int nvec) {
  const int threads = vec_threads(nvec);
  return one_wave_grid((const void*)k_update_fused, threads,
                       ((long long)n + threads / nvec - 1) / (threads / nvec));
}

erc_status launch_update(const VecArgs& va, int grid, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(vec_threads(va.ld / 4));
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // every block resident: the barrier can complete
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  ERC_CUDA(cudaLaunchKernelEx(&cfg, k_update_fused, va));
  count_launches(1);
  return ERC_OK;
}

// ---- resident path selection: the kernel for this shape, its shared memory, and whether it fits
const void* resident_kernel(int nvec, bool weighted) {
  const void* k = nullptr;
  auto pick = [&](auto lpr, auto vpl) {
    constexpr int LPR = decltype(lpr)::value, VPL = decltype(vpl)::value;
    k = weighted ? (const void*)k_cg_resident<LPR, VPL, true>
                 : (const void*)k_cg_resident<LPR, VPL, false>;
  };
  if (nvec <= 4) pick(ic<4>{}, ic<1>{});
  else if (nvec <= 8) pick(ic<8>{}, ic<1>{});
  else if (nvec <= 16) pick(ic<16>{}, ic<1>{});
  else if (nvec <= 32) pick(ic<32>{}, ic<1>{});
  else if (nvec <= 64) pick(ic<32>{}, ic<2>{});
  return k;  // wider rows use the multi-kernel path
}

bool resident_plan(const erc_graph* g, int ld, int32_t* rb, size_t* smem, const void** kern) {
  const char* mode = getenv("ERC_CG_MODE");
  if (mode && strcmp(mode, "graph") == 0) return false;
  const int nvec = ld / 4;
  const void* k = resident_kernel(nvec, g->val != nullptr);
  if (!k) return false;
  const int lpr = nvec <= 4 ? 4 : nvec <= 8 ? 8 : nvec <= 16 ? 16 : 32;
  const int grid = sm_count();
  const int64_t rows = ((int64_t)g->n + grid - 1) / grid;
  const size_t bytes = 4 * (2 * (size_t)rows * ld + (size_t)(PT / lpr) * ld + 2 * (size_t)ld +
                            2 * (size_t)PWARPS * PCH);
  int dev = 0, optin = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
    return false;
  if (bytes > (size_t)optin) return false;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) !=
      cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k, PT, bytes) != cudaSuccess || nb < 1) {
    cudaGetLastError();
    return false;
  }
  *rb = (int32_t)rows;
  *smem = bytes;
  *kern = k;
  return true;
}

erc_status launch_resident(const void* kern, const ResArgs& ra, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(sm_count());
  cfg.blockDim = dim3(PT);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // one block per SM, all resident
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* args[] = {const_cast<ResArgs*>(&ra)};
  ERC_CUDA(cudaLaunchKernelExC(&cfg, kern, args));
  count_launches(1);
  return ERC_OK;
}

erc_status launch_iteration(const SpmmArgs& sa, int sgrid, const VecArgs& va, int ugrid,
                            cudaStream_t s) {
  ERC_TRY(launch_spmm<MODE_STEP>(sa, sgrid, s));
  return launch_update(va, ugrid, s);
}

// ---------------------------------------------------------------------------- graph cache
struct GraphKey {
  const void* ptr[14];
  long long num[10];
  bool operator==(const GraphKey& o) const {
    for (int i = 0; i < 14; ++i)
      if (ptr[i] != o.ptr[i]) return false;
    for (int i = 0; i < 10; ++i)
      if (num[i] != o.num[i]) return false;
    return true;
  }
};
struct GraphEntry {
  GraphKey key;
  cudaGraphExec_t exec = nullptr;
  unsigned long long stamp = 0;
};
constexpr int CACHE = 16;
std::mutex g_mu;
GraphEntry g_cache[CACHE];
unsigned long long g_clock = 0;

cudaStream_t capture_stream() {
  static thread_local cudaStream_t cs[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 0 || dev >= 64) return nullptr;
  if (!cs[dev]) cudaStreamCreateWithFlags(&cs[dev], cudaStreamNonBlocking);
  return cs[dev];
}

erc_status iteration_graph(const SpmmArgs& sa, int sgrid, const VecArgs& va, int ugrid, int S,
                           cudaGraphExec_t* out) {
  int dev = 0;
  ERC_CUDA(cudaGetDevice(&dev));
  GraphKey k{};
  const void* ptrs[14] = {sa.row_ptr, sa.col, sa.val, sa.P, sa.AP, va.X, va.R, va.alpha,
                          va.active, va.flags, sa.cr.part1, va.Y, sa.heavy, va.gen};
  for (int i = 0; i < 14; ++i) k.ptr[i] = ptrs[i];
  int eps_bits = 0;
  long long tol_bits = 0;
  memcpy(&eps_bits, &sa.eps, sizeof eps_bits);
  memcpy(&tol_bits, &va.tol2, sizeof tol_bits);
  long long nums[10] = {sa.n, sa.ld, sa.kc, eps_bits, tol_bits, va.max_iter, S, dev, sgrid,
                        (long long)ugrid << 32 | (unsigned)sa.H};
  for (int i = 0; i < 10; ++i) k.num[i] = nums[i];
  std::lock_guard<std::mutex> lock(g_mu);
  ++g_clock;
  int victim = 0;
  for (int i = 0; i < CACHE; ++i) {
    if (g_cache[i].exec && g_cache[i].key == k) {
      g_cache[i].stamp = g_clock;
      *out = g_cache[i].exec;
      return ERC_OK;
    }
    if (g_cache[i].stamp < g_cache[victim].stamp) victim = i;
  }
  cudaStream_t cs = capture_stream();
  if (!cs) return set_error(ERC_ERR_CUDA, "no capture stream");
  ERC_CUDA(cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal));
  set_capturing(true);
  erc_status st = ERC_OK;
  for (int i = 0; i < S && st == ERC_OK; ++i) st = launch_iteration(sa, sgrid, va, ugrid, cs);
  set_capturing(false);
  cudaGraph_t graph = nullptr;
  cudaError_t ce = cudaStreamEndCapture(cs, &graph);
  if (st != ERC_OK) {
    if (graph) cudaGraphDestroy(graph);
    return st;
  }
  if (ce != cudaSuccess) return set_error(ERC_ERR_CUDA, "graph capture: %s", cudaGetErrorString(ce));
  cudaGraphExec_t exec = nullptr;
  ce = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  if (ce != cudaSuccess)
    return set_error(ERC_ERR_CUDA, "graph instantiate: %s", cudaGetErrorString(ce));
  if (g_cache[victim].exec) cudaGraphExecDestroy(g_cache[victim].exec);
  g_cache[victim].key = k;
  g_cache[victim].exec = exec;
  g_cache[victim].stamp = g_clock;
  *out = exec;
  return ERC_OK;
}

int iterations_per_poll(const erc_graph* g, int ld) {
  const double bytes = (double)(2 * g->m + g->n) * ld * 4.0;  // gathered + streamed per iteration
  if (bytes < 256e6) return 16;
  if (bytes < 2e9) return 4;
  return 2;
}

erc_status check_block(const float* p, const char* name) {
  ERC_REQUIRE(p && (reinterpret_cast<uintptr_t>(p) & 15) == 0, "%s must be 16-byte aligned", name);
  return ERC_OK;
}

}  // namespace
}  // namespace erc

using namespace erc;

extern "C" size_t erc_batched_cg_workspace_size(int32_t n, int32_t ld) {
  if (n < 1 || ld < 4) return 0;
  Arena a(nullptr);
  CgWork w;
  plan_cg(a, w, n, ld);
  return a.used + 256;
}

static erc_status batched_cg_impl(const erc_graph* g, float eps, const float* Y, float* X,
                                  int32_t ld, int32_t kc, float tol, int32_t max_iter,
                                  int32_t* iters, float* relres, void* ws, size_t ws_bytes,
                                  erc_stream stream, float* solve_us, int32_t* path) {
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(kc >= 1 && ld >= kc && ld % 4 == 0 && ld <= MAX_LD, "bad kc %d / ld %d", kc, ld);
  ERC_REQUIRE(eps > 0.f && isfinite(eps), "eps must be positive");
  ERC_REQUIRE(tol >= 0.f && isfinite(tol), "tol must be finite and >= 0");
  ERC_REQUIRE(max_iter >= 1, "max_iter must be >= 1");
  ERC_REQUIRE(iters && relres, "iters and relres are required");
  ERC_TRY(check_block(Y, "Y"));
  ERC_TRY(check_block(X, "X"));
  if (ws_bytes < erc_batched_cg_workspace_size(g->n, ld))
    return set_error(ERC_ERR_CAPACITY, "workspace too small");
  cudaStream_t s = as_stream(stream);
  Arena ar(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  CgWork w;
  plan_cg(ar, w, g->n, ld);
  ERC_CUDA(cudaMemsetAsync(w.cr.cnt, 0, colreduce_counter_bytes(), s));
  ERC_CUDA(cudaMemsetAsync(w.flags, 0, 8 * sizeof(int), s));
  ERC_CUDA(cudaMemsetAsync(w.gen, 0, 8 * sizeof(unsigned), s));

  int sgrid = 1;
  int32_t H = 0;
  spmm_shape(g, ld, &sgrid, &H);
  ERC_TRY(build_heavy(g, H, w.heavy, s));
  const int nvec = ld / 4;
  const int ugrid = update_grid(g->n, nvec);

  VecArgs va{};
  va.n = g->n;
  va.ld = ld;
  va.kc = kc;
  va.tol2 = (double)tol * (double)tol;
  va.max_iter = max_iter;
  va.Y = Y;
  va.X = X;
  va.R = w.R;
  va.P = w.P;
  va.AP = w.AP;
  va.alpha = w.alpha;
  va.beta = w.beta;
  va.rr = w.rr;
  va.yy = w.yy;
  va.active = w.active;
  va.conv = w.conv;
  va.iters = w.iters;
  va.flags = w.flags;
  va.gen = w.gen;
  va.cr = w.cr;

  SpmmArgs sa{};
  sa.row_ptr = g->row_ptr;
  sa.col = g->col;
  sa.val = g->val;
  sa.n = g->n;
  sa.ld = ld;
  sa.kc = kc;
  sa.eps = eps;
  sa.H = H;
  sa.heavy = w.heavy.list;
  sa.nheavy = w.heavy.count;
  sa.P = w.P;
  sa.AP = w.AP;
  sa.Y = Y;
  sa.cr = w.cr;
  sa.alpha = w.alpha;
  sa.rr = w.rr;
  sa.active = w.active;
  sa.flags = w.flags;
  sa.yy = w.yy;
  sa.iters = w.iters;
  sa.conv = w.conv;
  sa.relres_out = relres;
  sa.iters_out = iters;

  k_cg_init<<<grid_for(g->n, vec_threads(nvec) / nvec), vec_threads(nvec), 0, s>>>(va);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());

  int32_t rb = 0;
  size_t smem = 0;
  const void* kres = nullptr;
  const bool resident = resident_plan(g, ld, &rb, &smem, &kres);
  if (path) *path = resident ? 1 : 0;
  cudaEvent_t ev[2] = {nullptr, nullptr};
  if (solve_us) {
    ERC_CUDA(cudaEventCreate(&ev[0]));
    ERC_CUDA(cudaEventCreate(&ev[1]));
    ERC_CUDA(cudaEventRecord(ev[0], s));
  }
  if (resident) {
    // the whole solve in one cooperative launch, no host round trips
    ResArgs ra{sa, va, rb};
    ERC_TRY(launch_resident(kres, ra, smem, s));
  } else {
    const int S = iterations_per_poll(g, ld);
    cudaGraphExec_t exec = nullptr;
    ERC_TRY(iteration_graph(sa, sgrid, va, ugrid, S, &exec));
    int done = 0;
    int h_any = 1;
    while (done < max_iter) {
      ERC_CUDA(cudaGraphLaunch(exec, s));
      count_launches(2LL * S);  // the graph holds S iterations of two kernels
      done += S;
      ERC_CUDA(cudaMemcpyAsync(&h_any, w.flags, sizeof(int), cudaMemcpyDeviceToHost, s));
      ERC_CUDA(cudaStreamSynchronize(s));
      if (!h_any) break;
    }
  }
  if (solve_us) ERC_CUDA(cudaEventRecord(ev[1], s));

  // true residual of the returned iterate, plus the per-column outputs
  SpmmArgs ra = sa;
  ra.P = X;
  ERC_TRY(launch_spmm<MODE_RESID>(ra, sgrid, s));
  int h_flags[4] = {0, 0, 0, 0};
  ERC_CUDA(cudaMemcpyAsync(h_flags, w.flags, 4 * sizeof(int), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaStreamSynchronize(s));
  if (solve_us) {
    float ms = 0.f;
    const cudaError_t e = cudaEventElapsedTime(&ms, ev[0], ev[1]);
    cudaEventDestroy(ev[0]);
    cudaEventDestroy(ev[1]);
    if (e != cudaSuccess) return set_error(ERC_ERR_CUDA, "event timing: %s", cudaGetErrorString(e));
    *solve_us = 1000.f * ms;
  }
  if (h_flags[3]) return set_error(ERC_ERR_TIMEOUT, "update kernel grid barrier timed out");
  if (h_flags[1]) return set_error(ERC_ERR_NUMERIC, "non-finite or non-positive CG scalar");
  if (h_flags[2])
    return set_error(ERC_ERR_NOT_CONVERGED, "%d of %d columns reached max_iter=%d", h_flags[2],
                     kc, max_iter);
  return ERC_OK;
}

extern "C" erc_status erc_batched_cg(const erc_graph* g, float eps, const float* Y, float* X,
                                     int32_t ld, int32_t kc, float tol, int32_t max_iter,
                                     int32_t* iters, float* relres, void* ws, size_t ws_bytes,
                                     erc_stream stream) {
  clear_error();
  return batched_cg_impl(g, eps, Y, X, ld, kc, tol, max_iter, iters, relres, ws, ws_bytes, stream,
                         nullptr, nullptr);
}

extern "C" erc_status erc_batched_cg_timed(const erc_graph* g, float eps, const float* Y,
                                           float* X, int32_t ld, int32_t kc, float tol,
                                           int32_t max_iter, int32_t* iters, float* relres,
                                           void* ws, size_t ws_bytes, float* solve_us,
                                           int32_t* path, erc_stream stream) {
  clear_error();
  ERC_REQUIRE(solve_us && path, "solve_us and path are required");
  return batched_cg_impl(g, eps, Y, X, ld, kc, tol, max_iter, iters, relres, ws, ws_bytes, stream,
                         solve_us, path);
}

extern "C" size_t erc_laplacian_apply_workspace_size(int32_t n, int32_t ld) {
  if (n < 1 || ld < 4) return 0;
  Arena a(nullptr);
  ColReduce cr;
  plan_colreduce(a, cr, ld);
  HeavyRows h;
  plan_heavy(a, h, n);
  return a.used + 256;
}

extern "C" erc_status erc_laplacian_apply(const erc_graph* g, float eps, const float* P,
                                          float* AP, int32_t ld, int32_t kc, double* pAp,
                                          void* ws, size_t ws_bytes, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(kc >= 1 && ld >= kc && ld % 4 == 0 && ld <= MAX_LD, "bad kc %d / ld %d", kc, ld);
  ERC_REQUIRE(eps >= 0.f && isfinite(eps), "eps must be finite and >= 0");
  ERC_TRY(check_block(P, "P"));
  ERC_TRY(check_block(AP, "AP"));
  if (ws_bytes < erc_laplacian_apply_workspace_size(g->n, ld))
    return set_error(ERC_ERR_CAPACITY, "workspace too small");
  cudaStream_t s = as_stream(stream);
  Arena ar(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  SpmmArgs sa{};
  plan_colreduce(ar, sa.cr, ld);
  HeavyRows hv;
  plan_heavy(ar, hv, g->n);
  sa.row_ptr = g->row_ptr;
  sa.col = g->col;
  sa.val = g->val;
  sa.n = g->n;
  sa.ld = ld;
  sa.kc = kc;
  sa.eps = eps;
  sa.P = P;
  sa.AP = AP;
  sa.pap_out = pAp;
  int sgrid = 1;
  spmm_shape(g, ld, &sgrid, &sa.H);
  sa.heavy = hv.list;
  sa.nheavy = hv.count;
  ERC_TRY(build_heavy(g, sa.H, hv, s));
  if (pAp) ERC_CUDA(cudaMemsetAsync(sa.cr.cnt, 0, colreduce_counter_bytes(), s));
  return launch_spmm<MODE_APPLY>(sa, sgrid, s);
}

extern "C" erc_status erc_laplacian_apply_timed(const erc_graph* g, float eps, const float* P,
                                                float* AP, int32_t ld, int32_t kc, double* pAp,
                                                int32_t reps, float* avg_us, void* ws,
                                                size_t ws_bytes, erc_stream stream) {
  clear_error();
  ERC_REQUIRE(reps >= 1 && avg_us, "reps >= 1 and avg_us are required");
  // one untimed call builds the heavy-row list in the workspace and warms the caches
  ERC_TRY(erc_laplacian_apply(g, eps, P, AP, ld, kc, pAp, ws, ws_bytes, stream));
  cudaStream_t s = as_stream(stream);
  Arena ar(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  SpmmArgs sa{};
  plan_colreduce(ar, sa.cr, ld);
  HeavyRows hv;
  plan_heavy(ar, hv, g->n);
  sa.row_ptr = g->row_ptr;
  sa.col = g->col;
  sa.val = g->val;
  sa.n = g->n;
  sa.ld = ld;
  sa.kc = kc;
  sa.eps = eps;
  sa.P = P;
  sa.AP = AP;
  sa.pap_out = pAp;
  int sgrid = 1;
  spmm_shape(g, ld, &sgrid, &sa.H);
  sa.heavy = hv.list;
  sa.nheavy = hv.count;
  cudaEvent_t e0, e1;
  ERC_CUDA(cudaEventCreate(&e0));
  ERC_CUDA(cudaEventCreate(&e1));
  erc_status st = ERC_OK;
  cudaError_t ce = cudaEventRecord(e0, s);
  for (int r = 0; r < reps && st == ERC_OK && ce == cudaSuccess; ++r)
    st = launch_spmm<MODE_APPLY>(sa, sgrid, s);
  if (ce == cudaSuccess) ce = cudaEventRecord(e1, s);
  if (ce == cudaSuccess) ce = cudaEventSynchronize(e1);
  float ms = 0.f;
  if (ce == cudaSuccess) ce = cudaEventElapsedTime(&ms, e0, e1);
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  if (st != ERC_OK) return st;
  if (ce != cudaSuccess) return set_error(ERC_ERR_CUDA, "event timing: %s", cudaGetErrorString(ce));
  *avg_us = 1000.f * ms / (float)reps;
  return ERC_OK;
}
