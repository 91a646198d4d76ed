// cg.cu -- column-wise CG on L_eps X = Y (Eq. 5, §3.1.3, Algorithm 1) and the operator
// L_eps P = eps P + (D - A) P it iterates on.
//
// One CG iteration is two kernels over the row-major n x ld block:
//   k_spmm<MODE_STEP>  AP = L_eps P: a group of LPR lanes gathers the neighbour rows of one
//                      light row (float4 along the columns); rows heavier than H are taken by a
//                      whole block, its groups splitting the row and combining in a fixed order.
//                      Per-column p.Ap partials; the last block to finish forms alpha = rr / pAp.
//   k_update_fused     r -= alpha Ap and r.r; the last block forms beta, counts the iteration
//                      and retires converged columns, then releases a grid barrier; every block
//                      then applies x += alpha p and p = r + beta p to its rows (x's update reads
//                      the p it needs there: 8 vector passes instead of 9).  Launched
//                      cooperatively (all blocks resident), the barrier wait is bounded.
// Reductions are deterministic: fixed groupings and orders, float-pair accumulation.  S
// iterations are captured once into a CUDA graph and relaunched; kernels return at once when no
// column is active, so the host only polls the "any active" flag between graph launches.
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "erc_internal.cuh"
#include "cg_device.cuh"

namespace erc {
namespace {

struct HeavyRows {
  int32_t* list;    // [n] rows with more than H neighbours, ascending
  int64_t* count;   // [1]
  int* bcount;      // [MAX_GRID] heavy rows in each listing block's range of rows
};

void plan_heavy(Arena& a, HeavyRows& h, int32_t n) {
  h.list = a.take<int32_t>(n);
  h.count = a.take<int64_t>(1);
  h.bcount = a.take<int>(MAX_GRID);
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
  // nothing left to do: no active column, or a bounded wait of the solve has given up
  if (MODE == MODE_STEP && (*(volatile int*)a.flags == 0 || *(volatile int*)(a.flags + 3) != 0))
    return;
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
    gather_range<LPR, VPL, WEIGHTED>(a, a.P, gl, gm, 0, nvec, pu, s0, s1, acc);
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
    gather_range<LPR, VPL, WEIGHTED>(a, a.P, gl, gm, 0, nvec, pu, j0, j1, acc);
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

// r = y (columns kc.. zero), x = 0, p = r (with the Jacobi preconditioner, a.deg set: p = z =
// r / (deg + eps)); y.y and r.r (r.z) per column.  With the preconditioner both sums travel in
// one grid reduction of 2 ld columns.
__global__ void __launch_bounds__(T) k_cg_init(VecArgs a) {
  __shared__ float2 red[T * 4];
  __shared__ float2 sbuf[2 * MAX_LD];
  const bool pc = a.deg != nullptr;
  const int nvec = a.ld >> 2, rb = blockDim.x / nvec;
  const int q = threadIdx.x % nvec;
  float2 d[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
  float2 e[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
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
    const float4 p = pc ? f4_scale(y, jacobi_inv(a.deg, row, a.eps)) : y;
    *reinterpret_cast<float4*>(a.R + i) = y;
    *reinterpret_cast<float4*>(a.P + i) = p;
    *reinterpret_cast<float4*>(a.X + i) = f4_zero();
    d[0] = df_fma(d[0], y.x, y.x);
    d[1] = df_fma(d[1], y.y, y.y);
    d[2] = df_fma(d[2], y.z, y.z);
    d[3] = df_fma(d[3], y.w, y.w);
    e[0] = df_fma(e[0], y.x, p.x);
    e[1] = df_fma(e[1], y.y, p.y);
    e[2] = df_fma(e[2], y.z, p.z);
    e[3] = df_fma(e[3], y.w, p.w);
  }
  block_partials_quad(d, red, sbuf, a.ld, nvec);
  if (pc) block_partials_quad(e, red, sbuf + a.ld, a.ld, nvec);
  if (!grid_colreduce(a.cr, sbuf, sbuf, pc ? 2 * a.ld : a.ld)) return;
  int any = 0;
  for (int c = threadIdx.x; c < a.ld; c += blockDim.x) {
    const double v = df_value(sbuf[c]);
    const double rho = pc ? df_value(sbuf[a.ld + c]) : v;
    a.yy[c] = v;
    a.rr[c] = rho;
    a.iters[c] = 0;
    a.alpha[c] = 0.f;
    a.beta[c] = 0.f;
    int act = 0, cv = 1;
    if (c < a.kc) {
      if (!isfinite(v) || !isfinite(rho)) {
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

// r -= alpha Ap, r.r  |grid barrier: beta, convergence|  x += alpha p, p = r + beta p
// The x update uses this iteration's alpha and the p it was formed with, exactly as it would
// before the barrier, so the iterates do not change; it is applied after the barrier because
// that pass reads p anyway (x, p, r read; x, p written: with r, Ap read and r written before
// the barrier, 8 passes over the n x ld block).
// With the Jacobi preconditioner (a.deg set) the first part also sums r.z, z = r / (deg + eps),
// beta is the ratio of successive r.z, and p = z + beta p; the stop test stays on r.r.
constexpr int UPD = 4;  // rows per thread whose loads the vector update keeps in flight

__global__ void __launch_bounds__(T) k_update_fused(VecArgs a) {
  if (*(volatile int*)a.flags == 0 || *(volatile int*)(a.flags + 3) != 0) return;
  __shared__ float2 red[T * 4];
  __shared__ float2 sbuf[2 * MAX_LD];
  const bool pc = a.deg != nullptr;
  __shared__ unsigned s_gen;
  if (threadIdx.x == 0) s_gen = ld_acquire(a.gen);
  const int nvec = a.ld >> 2, rb = blockDim.x / nvec;
  const int q = threadIdx.x % nvec;
  const int64_t row0 = (int64_t)blockIdx.x * rb + threadIdx.x / nvec;
  const int64_t rstep = (int64_t)gridDim.x * rb;
  const float4 al = *reinterpret_cast<const float4*>(a.alpha + 4 * q);
  float2 d[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
  float2 e[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                 make_float2(0.f, 0.f)};
  // UPD rows per thread in flight: every load of a group of rows is issued before the first
  // use, so each thread keeps several rows' loads outstanding (HBM latency otherwise bounds the
  // pass); the rows and the partial sums keep their order
  if (al.x != 0.f || al.y != 0.f || al.z != 0.f || al.w != 0.f) {
    for (int64_t rowb = row0; rowb < a.n; rowb += UPD * rstep) {
      float4 r[UPD], ap[UPD];
#pragma unroll
      for (int k = 0; k < UPD; ++k) {
        const int64_t row = rowb + k * rstep;
        if (row < a.n) {
          const size_t i = (size_t)row * a.ld + 4 * q;
          r[k] = *reinterpret_cast<const float4*>(a.R + i);
          ap[k] = *reinterpret_cast<const float4*>(a.AP + i);
        }
      }
#pragma unroll
      for (int k = 0; k < UPD; ++k) {
        const int64_t row = rowb + k * rstep;
        if (row >= a.n) break;
        float4 rr = r[k];
        rr.x = fmaf(-al.x, ap[k].x, rr.x);
        rr.y = fmaf(-al.y, ap[k].y, rr.y);
        rr.z = fmaf(-al.z, ap[k].z, rr.z);
        rr.w = fmaf(-al.w, ap[k].w, rr.w);
        *reinterpret_cast<float4*>(a.R + (size_t)row * a.ld + 4 * q) = rr;
        d[0] = df_fma(d[0], rr.x, rr.x);
        d[1] = df_fma(d[1], rr.y, rr.y);
        d[2] = df_fma(d[2], rr.z, rr.z);
        d[3] = df_fma(d[3], rr.w, rr.w);
        if (pc) {
          const float4 z = f4_scale(rr, jacobi_inv(a.deg, row, a.eps));
          e[0] = df_fma(e[0], rr.x, z.x);
          e[1] = df_fma(e[1], rr.y, z.y);
          e[2] = df_fma(e[2], rr.z, z.z);
          e[3] = df_fma(e[3], rr.w, z.w);
        }
      }
    }
  }
  block_partials_quad(d, red, sbuf, a.ld, nvec);
  if (pc) block_partials_quad(e, red, sbuf + a.ld, a.ld, nvec);
  if (grid_colreduce(a.cr, sbuf, sbuf, pc ? 2 * a.ld : a.ld)) {
    int any = 0;
    for (int c = threadIdx.x; c < a.ld; c += blockDim.x) {
      float be = 0.f;
      if (a.active[c]) {
        const double rn = df_value(sbuf[c]);
        const double rho = pc ? df_value(sbuf[a.ld + c]) : rn;  // the numerator of beta
        const int it = a.iters[c] + 1;
        a.iters[c] = it;
        if (!isfinite(rn) || !isfinite(rho)) {
          a.active[c] = 0;
          atomicOr(&a.flags[1], 1);
        } else {
          be = (float)(rho / a.rr[c]);
          a.rr[c] = rho;
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
      if (++spins > a.spin_limit) {  // bounded: flag the timeout and fall through
        atomicOr(&a.flags[3], 1);
        break;
      }
      __nanosleep(64);
    }
  }
  __syncthreads();
  // columns with alpha != 0 were active in this iteration: x += alpha p; those still active
  // after it: p = r + beta p (a column that converged now still takes its last x update)
  const int4 act = __ldcg(reinterpret_cast<const int4*>(a.active + 4 * q));
  const float4 be = __ldcg(reinterpret_cast<const float4*>(a.beta + 4 * q));
  const bool any_p = act.x | act.y | act.z | act.w;
  const bool any_x = al.x != 0.f || al.y != 0.f || al.z != 0.f || al.w != 0.f;
  if (!any_x && !any_p) return;
  for (int64_t rowb = row0; rowb < a.n; rowb += UPD * rstep) {
    float4 p[UPD], x[UPD], r[UPD];
#pragma unroll
    for (int k = 0; k < UPD; ++k) {
      const int64_t row = rowb + k * rstep;
      if (row < a.n) {
        const size_t i = (size_t)row * a.ld + 4 * q;
        p[k] = *reinterpret_cast<const float4*>(a.P + i);
        if (any_x) x[k] = *reinterpret_cast<const float4*>(a.X + i);
        if (any_p) r[k] = *reinterpret_cast<const float4*>(a.R + i);
      }
    }
#pragma unroll
    for (int k = 0; k < UPD; ++k) {
      const int64_t row = rowb + k * rstep;
      if (row >= a.n) break;
      const size_t i = (size_t)row * a.ld + 4 * q;
      float4 pp = p[k];
      if (any_x) {
        float4 xx = x[k];
        xx.x = fmaf(al.x, pp.x, xx.x);
        xx.y = fmaf(al.y, pp.y, xx.y);
        xx.z = fmaf(al.z, pp.z, xx.z);
        xx.w = fmaf(al.w, pp.w, xx.w);
        *reinterpret_cast<float4*>(a.X + i) = xx;
      }
      if (!any_p) continue;
      float4 rr = r[k];
      if (pc) rr = f4_scale(rr, jacobi_inv(a.deg, row, a.eps));  // z
      if (act.x) pp.x = fmaf(be.x, pp.x, rr.x);
      if (act.y) pp.y = fmaf(be.y, pp.y, rr.y);
      if (act.z) pp.z = fmaf(be.z, pp.z, rr.z);
      if (act.w) pp.w = fmaf(be.w, pp.w, rr.w);
      *reinterpret_cast<float4*>(a.P + i) = pp;
    }
  }
}


// ---------------------------------------------------------------------------- cluster CG
// The kc columns of Eq. 5 are independent systems, so the solve can also be split by columns:
// a thread-block cluster of CS blocks owns a group of 16 columns for every row and runs the whole
// solve of its group; clusters never wait on one another.  Block k of a cluster owns the rows
// [b_k, b_k+1) (equal shares of the neighbour lists, at most rbmax rows): their r and Ap live in
// its shared memory, x and p in global memory (p is gathered by the cluster's other blocks, from
// L2).  Four lanes take one light row, a float4 of the group's columns each, so a neighbour costs
// one 64-byte line; the next row's bounds and column indices are fetched while the current row's
// neighbours are in flight.  Rows heavier than H are split over the whole block.  Per-column dot
// products are combined in a fixed order: within a block by warp shuffles and shared memory,
// across the cluster by every block reading every block's partial through distributed shared
// memory, so all blocks of a cluster derive the same alpha, beta and stop decisions.
// Per iteration: A (Ap, p.Ap) | B (x, r, r.r) | C (p), each closed by a hardware cluster barrier.
constexpr int CT = 384;
constexpr int CWARPS = CT / 32;
constexpr int CL = 4;            // lanes per row
constexpr int CGR = CT / CL;     // rows in flight per block
constexpr int CW = 4 * CL;       // columns per group
constexpr int CHMAX = 256;       // heavy rows per block
constexpr int CMAXS = 16;        // largest cluster
constexpr int CU = 16;           // neighbour rows per batch
constexpr int CIDX = CU / CL;    // column indices each lane fetches per batch
constexpr int CUNROLL = 4;       // rows per lane in flight in the vector phases

struct ClusterArgs {
  const int64_t* row_ptr;
  const int32_t* col;
  const float* val;
  int32_t n, ld, kc;
  float eps;
  double tol2;
  int32_t max_iter;
  int32_t rbmax;  // rows of r and Ap a block's shared memory holds
  const float* Y;
  float* X;
  float* P;
  double *yy, *rr;
  int *iters, *conv, *flags;
};

__device__ __forceinline__ unsigned cluster_rank() {
  unsigned r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ unsigned cluster_size() {
  unsigned r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ unsigned cluster_index() {
  unsigned r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
// every thread of every block of the cluster; orders shared and global memory at cluster scope
__device__ __forceinline__ void cluster_barrier() {
  asm volatile(
      "barrier.cluster.arrive.release.aligned;\n\t"
      "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// float2 at the same shared-memory offset in block `rank` of this cluster
__device__ __forceinline__ float2 ld_cluster_f2(const float2* local, unsigned rank) {
  const unsigned a = (unsigned)__cvta_generic_to_shared(local);
  unsigned ra;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(a), "r"(rank));
  float2 v;
  asm volatile("ld.shared::cluster.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(ra) : "memory");
  return v;
}

struct ClusterShared {
  float2 red[2][CW];  // this block's partials (two slots: consecutive reductions)
  float2 wsum[CWARPS][CW];
  float2 tot[CW];
  float4 comb[CWARPS][CL];
  double rr[CW], yy[CW];
  float alpha[CW], beta[CW];
  int active[CW], iters[CW], conv[CW];
  int64_t samp[CT];
  int32_t b[CMAXS + 1];
  int32_t heavy[CHMAX];
  int wcnt[CWARPS];
  int nheavy;
};

// d (per-lane partials of its 4 columns) -> cl.tot: block sum in warp/lane order, then the
// cluster's block partials in rank order; every block of the cluster obtains the same totals
__device__ __forceinline__ void cluster_colsum(float2 (&d)[4], ClusterShared& cl, int slot, int S) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = CL; off < 32; off <<= 1)
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      float2 o;
      o.x = __shfl_xor_sync(0xffffffffu, d[t].x, off);
      o.y = __shfl_xor_sync(0xffffffffu, d[t].y, off);
      d[t] = df_add(d[t], o);
    }
  if (lane < CL)
#pragma unroll
    for (int t = 0; t < 4; ++t) cl.wsum[warp][4 * lane + t] = d[t];
  __syncthreads();
  if (threadIdx.x < CW) {
    float2 acc = make_float2(0.f, 0.f);
    for (int w = 0; w < CWARPS; ++w) acc = df_add(acc, cl.wsum[w][threadIdx.x]);
    cl.red[slot][threadIdx.x] = acc;
  }
  cluster_barrier();
  if (threadIdx.x < CW) {
    float2 v[CMAXS];
#pragma unroll
    for (int k = 0; k < CMAXS; ++k)
      v[k] = k < S ? ld_cluster_f2(&cl.red[slot][threadIdx.x], k) : make_float2(0.f, 0.f);
    float2 acc = make_float2(0.f, 0.f);
#pragma unroll
    for (int k = 0; k < CMAXS; ++k)
      if (k < S) acc = df_add(acc, v[k]);
    cl.tot[threadIdx.x] = acc;
  }
  __syncthreads();
}

// column indices (and weights) of neighbours [jb, jb + CU) within [jb, j1): lane gl holds
// entries jb + gl + CL * t
template <bool WEIGHTED>
__device__ __forceinline__ void cluster_fetch_idx(const ClusterArgs& a, int gl, int64_t jb,
                                                  int64_t j1, int (&c)[CIDX], float (&w)[CIDX]) {
#pragma unroll
  for (int t = 0; t < CIDX; ++t) {
    const int64_t j = jb + gl + CL * t;
    c[t] = j < j1 ? __ldg(a.col + j) : 0;
    w[t] = j < j1 ? (WEIGHTED ? __ldg(a.val + j) : 1.f) : 0.f;
  }
}

// acc += sum over the batch [jb, min(jb + CU, j1)) of w_j (p_u - p_{col_j}) for this lane's
// float4.  Slots past j1 load p_u itself, so they add exactly zero.
template <bool WEIGHTED>
__device__ __forceinline__ void cluster_batch(const ClusterArgs& a, bool valid, size_t qoff,
                                              float4 pu, const int (&c)[CIDX],
                                              const float (&w)[CIDX], int64_t jb, int64_t j1,
                                              unsigned gm, float4& acc) {
  float4 v[CU];
#pragma unroll
  for (int k = 0; k < CU; ++k) {
    // entry jb + k sits in lane k % CL, slot k / CL
    const int ck = __shfl_sync(gm, c[k / CL], k % CL, CL);
    v[k] = valid && jb + k < j1
               ? __ldcg(reinterpret_cast<const float4*>(a.P + (size_t)ck * a.ld + qoff))
               : pu;
  }
#pragma unroll
  for (int k = 0; k < CU; ++k) {
    if (WEIGHTED) {
      const float wk = __shfl_sync(gm, w[k / CL], k % CL, CL);
      acc.x = fmaf(wk, pu.x - v[k].x, acc.x);
      acc.y = fmaf(wk, pu.y - v[k].y, acc.y);
      acc.z = fmaf(wk, pu.z - v[k].z, acc.z);
      acc.w = fmaf(wk, pu.w - v[k].w, acc.w);
    } else {
      acc.x += pu.x - v[k].x;
      acc.y += pu.y - v[k].y;
      acc.z += pu.z - v[k].z;
      acc.w += pu.w - v[k].w;
    }
  }
}

__device__ __forceinline__ void dot4(float2 (&d)[4], float4 a, float4 b) {
  d[0] = df_fma(d[0], a.x, b.x);
  d[1] = df_fma(d[1], a.y, b.y);
  d[2] = df_fma(d[2], a.z, b.z);
  d[3] = df_fma(d[3], a.w, b.w);
}
__device__ __forceinline__ float4 fma4(float4 s, float4 a, float4 b) {  // s * a + b
  return make_float4(fmaf(s.x, a.x, b.x), fmaf(s.y, a.y, b.y), fmaf(s.z, a.z, b.z),
                     fmaf(s.w, a.w, b.w));
}
__device__ __forceinline__ float4 eps_fma4(float e, float4 p, float4 acc) {
  return make_float4(fmaf(e, p.x, acc.x), fmaf(e, p.y, acc.y), fmaf(e, p.z, acc.z),
                     fmaf(e, p.w, acc.w));
}

template <bool WEIGHTED>
__global__ void __launch_bounds__(CT, 1) k_cg_cluster(ClusterArgs a) {
  extern __shared__ __align__(16) float4 csm[];
  __shared__ ClusterShared cl;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int gl = tid & (CL - 1), gi = tid / CL;
  const unsigned gm = 0xfu << (lane & ~(CL - 1));
  const int S = (int)cluster_size(), rank = (int)cluster_rank();
  const int q = CL * (int)cluster_index() + gl;  // this lane's float4 slot of the row
  const bool valid = q < (a.ld >> 2);
  const size_t qoff = 4 * (size_t)q;
  const int rbmax = a.rbmax;
  float4* rs = csm;                 // [rbmax][CL] r of own rows
  float4* aps = csm + CL * rbmax;   // [rbmax][CL] Ap of own rows

  // ---- row split: S equal shares of the neighbour lists, each of at most rbmax rows
  const int64_t nnz = a.row_ptr[a.n];
  cl.samp[tid] = a.row_ptr[(int64_t)tid * a.n / (CT - 1)];
  __syncthreads();
  if (tid <= S) {
    const int64_t target = (int64_t)tid * nnz / S;
    int f = 0, fh = CT - 1;  // first sample f with samp[f] >= target (samp[CT - 1] = nnz)
    while (f < fh) {
      const int mid = (f + fh) >> 1;
      if (cl.samp[mid] < target) f = mid + 1; else fh = mid;
    }
    int64_t lo = f > 0 ? (int64_t)(f - 1) * a.n / (CT - 1) : 0;
    int64_t hi = (int64_t)f * a.n / (CT - 1);
    while (lo < hi) {  // first row u with row_ptr[u] >= target
      const int64_t mid = (lo + hi) >> 1;
      if (a.row_ptr[mid] < target) lo = mid + 1; else hi = mid;
    }
    cl.b[tid] = (int32_t)lo;
  }
  __syncthreads();
  if (tid == 0) {
    int32_t b = 0;
    cl.b[0] = 0;
    for (int k = 0; k < S; ++k) {
      const int64_t need = (int64_t)a.n - (int64_t)(S - k - 1) * rbmax;
      int64_t nb = cl.b[k + 1];
      nb = max(nb, max((int64_t)b, need));
      nb = min(nb, (int64_t)b + rbmax);
      b = (int32_t)nb;
      cl.b[k + 1] = b;
    }
    int ok = b == a.n;
    for (int k = 0; k < S; ++k) ok &= cl.b[k + 1] - cl.b[k] <= rbmax;
    cl.nheavy = ok;  // reused below; the host sizes rbmax so that this holds
  }
  __syncthreads();
  if (!cl.nheavy) {  // the same outcome in every block: none reaches a cluster barrier
    if (tid == 0 && rank == 0) atomicOr(&a.flags[1], 1);
    return;
  }
  __syncthreads();
  const int32_t b0 = cl.b[rank];
  const int nr = cl.b[rank + 1] - b0;
  const int64_t* rp = a.row_ptr + b0;
  const int64_t nnz_b = rp[nr] - rp[0];
  const int64_t H = max((int64_t)64, (nnz_b + CHMAX - 1) / CHMAX);  // at most CHMAX heavy rows

  // ---- heavy rows of this block, ascending
  if (tid == 0) cl.nheavy = 0;
  __syncthreads();
  for (int base = 0; base < nr; base += CT) {
    const int i = base + tid;
    const bool hv = i < nr && rp[i + 1] - rp[i] > H;
    const unsigned bal = __ballot_sync(0xffffffffu, hv);
    if (lane == 0) cl.wcnt[warp] = __popc(bal);
    __syncthreads();
    int off = cl.nheavy, tot = 0;
    for (int w = 0; w < CWARPS; ++w) {
      if (w < warp) off += cl.wcnt[w];
      tot += cl.wcnt[w];
    }
    if (hv) cl.heavy[off + __popc(bal & ((1u << lane) - 1u))] = i;
    __syncthreads();
    if (tid == 0) cl.nheavy += tot;
    __syncthreads();
  }
  const int nheavy = cl.nheavy;

  // ---- r = p = y (columns beyond kc zero), x = 0, y.y
  float2 d[4];
#pragma unroll
  for (int t = 0; t < 4; ++t) d[t] = make_float2(0.f, 0.f);
  for (int i = gi; i < nr; i += CGR) {
    const size_t o = (size_t)(b0 + i) * a.ld + qoff;
    float4 y = f4_zero();
    if (valid) {
      y = ld_f4(a.Y + o);
      const int cb = 4 * q;
      if (cb + 0 >= a.kc) y.x = 0.f;
      if (cb + 1 >= a.kc) y.y = 0.f;
      if (cb + 2 >= a.kc) y.z = 0.f;
      if (cb + 3 >= a.kc) y.w = 0.f;
      *reinterpret_cast<float4*>(a.P + o) = y;
      *reinterpret_cast<float4*>(a.X + o) = f4_zero();
    }
    rs[i * CL + gl] = y;
    dot4(d, y, y);
  }
  cluster_colsum(d, cl, 0, S);  // its barrier also publishes p to the cluster
  if (tid < CW) {
    const int c = 4 * CL * (int)cluster_index() + tid;
    const double v = df_value(cl.tot[tid]);
    int act = 0, cv = 1;
    if (c < a.kc) {
      if (!isfinite(v)) {
        if (rank == 0) atomicOr(&a.flags[1], 1);
        cv = 0;
      } else if (v > 0.0 && !(v <= a.tol2 * v)) {
        act = 1;
        cv = 0;
      }
    }
    cl.yy[tid] = v;
    cl.rr[tid] = v;
    cl.iters[tid] = 0;
    cl.active[tid] = act;
    cl.conv[tid] = cv;
  }
  int any = __syncthreads_or(tid < CW && cl.active[tid]);

  int slot = 1;
  while (any) {
    // ---------------- A: Ap = L_eps p on own rows, p.Ap
#pragma unroll
    for (int t = 0; t < 4; ++t) d[t] = make_float2(0.f, 0.f);
    {
      // light rows, software-pipelined: row i's first batch of indices and row i + CGR's bounds
      // are in registers when row i starts; row i + CGR's first indices are fetched with it
      int i = gi;
      int64_t j0 = 0, j1 = 0, nj0 = 0, nj1 = 0;
      if (i < nr) {
        j0 = rp[i];
        j1 = rp[i + 1];
      }
      if (i + CGR < nr) {
        nj0 = rp[i + CGR];
        nj1 = rp[i + CGR + 1];
      }
      bool hv = j1 - j0 > H;
      int c[CIDX], cn[CIDX];
      float w[CIDX], wn[CIDX];
      cluster_fetch_idx<WEIGHTED>(a, gl, j0, hv ? j0 : j1, c, w);
      for (; i < nr; i += CGR) {
        const bool nhv = nj1 - nj0 > H;
        cluster_fetch_idx<WEIGHTED>(a, gl, nj0, nhv ? nj0 : nj1, cn, wn);
        int64_t nnj0 = 0, nnj1 = 0;
        if (i + 2 * CGR < nr) {
          nnj0 = rp[i + 2 * CGR];
          nnj1 = rp[i + 2 * CGR + 1];
        }
        if (!hv) {
          const float4 pu = valid ? __ldcg(reinterpret_cast<const float4*>(
                                        a.P + (size_t)(b0 + i) * a.ld + qoff))
                                  : f4_zero();
          float4 acc = f4_zero();
          cluster_batch<WEIGHTED>(a, valid, qoff, pu, c, w, j0, j1, gm, acc);
          for (int64_t jb = j0 + CU; jb < j1; jb += CU) {  // rows longer than one batch
            cluster_fetch_idx<WEIGHTED>(a, gl, jb, j1, c, w);
            cluster_batch<WEIGHTED>(a, valid, qoff, pu, c, w, jb, j1, gm, acc);
          }
          const float4 o = eps_fma4(a.eps, pu, acc);
          aps[i * CL + gl] = o;
          dot4(d, pu, o);
        }
        j0 = nj0;
        j1 = nj1;
        hv = nhv;
        nj0 = nnj0;
        nj1 = nnj1;
#pragma unroll
        for (int t = 0; t < CIDX; ++t) {
          c[t] = cn[t];
          w[t] = wn[t];
        }
      }
    }
    for (int h = 0; h < nheavy; ++h) {  // the whole block on one row, slices combined in order
      const int i = cl.heavy[h];
      const int64_t j0 = rp[i], j1 = rp[i + 1];
      const int64_t per = (j1 - j0 + CGR - 1) / CGR;
      const int64_t s0 = min(j1, j0 + gi * per), s1 = min(j1, s0 + per);
      const float4 pu = valid ? __ldcg(reinterpret_cast<const float4*>(
                                    a.P + (size_t)(b0 + i) * a.ld + qoff))
                              : f4_zero();
      float4 acc = f4_zero();
      int c[CIDX];
      float w[CIDX];
      for (int64_t jb = s0; jb < s1; jb += CU) {
        cluster_fetch_idx<WEIGHTED>(a, gl, jb, s1, c, w);
        cluster_batch<WEIGHTED>(a, valid, qoff, pu, c, w, jb, s1, gm, acc);
      }
#pragma unroll
      for (int off = CL; off < 32; off <<= 1) {
        acc.x += __shfl_xor_sync(0xffffffffu, acc.x, off);
        acc.y += __shfl_xor_sync(0xffffffffu, acc.y, off);
        acc.z += __shfl_xor_sync(0xffffffffu, acc.z, off);
        acc.w += __shfl_xor_sync(0xffffffffu, acc.w, off);
      }
      if (lane < CL) cl.comb[warp][lane] = acc;
      __syncthreads();
      if (tid < CL) {
        float4 s = f4_zero();
        for (int wp = 0; wp < CWARPS; ++wp) {
          const float4 cv = cl.comb[wp][tid];
          s = make_float4(s.x + cv.x, s.y + cv.y, s.z + cv.z, s.w + cv.w);
        }
        const float4 o = eps_fma4(a.eps, pu, s);
        aps[i * CL + tid] = o;
        dot4(d, pu, o);
      }
      __syncthreads();
    }
    cluster_colsum(d, cl, slot, S);
    slot ^= 1;
    if (tid < CW) {
      float al = 0.f;
      if (cl.active[tid]) {
        const double v = df_value(cl.tot[tid]);
        const double qq = cl.rr[tid] / v;
        if (!(v > 0.0) || !isfinite(qq)) {
          cl.active[tid] = 0;
          if (rank == 0) atomicOr(&a.flags[1], 1);
        } else {
          al = (float)qq;
        }
      }
      cl.alpha[tid] = al;
    }
    __syncthreads();

    // ---------------- B: x += alpha p, r -= alpha Ap, r.r
    {
      const float4 al = make_float4(cl.alpha[4 * gl], cl.alpha[4 * gl + 1], cl.alpha[4 * gl + 2],
                                    cl.alpha[4 * gl + 3]);
      const float4 nal = make_float4(-al.x, -al.y, -al.z, -al.w);
#pragma unroll
      for (int t = 0; t < 4; ++t) d[t] = make_float2(0.f, 0.f);
      if (valid) {
        for (int i0 = gi; i0 < nr; i0 += CUNROLL * CGR) {
          float4 p[CUNROLL], x[CUNROLL];
#pragma unroll
          for (int k = 0; k < CUNROLL; ++k) {
            const int i = i0 + k * CGR;
            if (i < nr) {
              const size_t o = (size_t)(b0 + i) * a.ld + qoff;
              p[k] = __ldcg(reinterpret_cast<const float4*>(a.P + o));
              x[k] = *reinterpret_cast<const float4*>(a.X + o);
            }
          }
#pragma unroll
          for (int k = 0; k < CUNROLL; ++k) {
            const int i = i0 + k * CGR;
            if (i < nr) {
              const size_t o = (size_t)(b0 + i) * a.ld + qoff;
              *reinterpret_cast<float4*>(a.X + o) = fma4(al, p[k], x[k]);
              const float4 r = fma4(nal, aps[i * CL + gl], rs[i * CL + gl]);
              rs[i * CL + gl] = r;
              dot4(d, r, r);
            }
          }
        }
      }
    }
    cluster_colsum(d, cl, slot, S);
    slot ^= 1;
    if (tid < CW) {
      float be = 0.f;
      int act = cl.active[tid];
      if (act) {
        const double rn = df_value(cl.tot[tid]);
        const int it = cl.iters[tid] + 1;
        cl.iters[tid] = it;
        if (!isfinite(rn)) {
          act = 0;
          if (rank == 0) atomicOr(&a.flags[1], 1);
        } else {
          be = (float)(rn / cl.rr[tid]);
          cl.rr[tid] = rn;
          if (rn <= a.tol2 * cl.yy[tid]) {
            cl.conv[tid] = 1;
            act = 0;
          } else if (it >= a.max_iter) {
            act = 0;
          }
        }
        cl.active[tid] = act;
      }
      cl.beta[tid] = be;
    }
    any = __syncthreads_or(tid < CW && cl.active[tid]);
    if (!any) break;

    // ---------------- C: p = r + beta p on active columns
    {
      const int4 act = make_int4(cl.active[4 * gl], cl.active[4 * gl + 1], cl.active[4 * gl + 2],
                                 cl.active[4 * gl + 3]);
      const float4 be = make_float4(cl.beta[4 * gl], cl.beta[4 * gl + 1], cl.beta[4 * gl + 2],
                                    cl.beta[4 * gl + 3]);
      if (valid && (act.x | act.y | act.z | act.w)) {
        for (int i0 = gi; i0 < nr; i0 += CUNROLL * CGR) {
          float4 p[CUNROLL];
#pragma unroll
          for (int k = 0; k < CUNROLL; ++k) {
            const int i = i0 + k * CGR;
            if (i < nr)
              p[k] = __ldcg(reinterpret_cast<const float4*>(a.P + (size_t)(b0 + i) * a.ld + qoff));
          }
#pragma unroll
          for (int k = 0; k < CUNROLL; ++k) {
            const int i = i0 + k * CGR;
            if (i < nr) {
              const float4 r = rs[i * CL + gl];
              if (act.x) p[k].x = fmaf(be.x, p[k].x, r.x);
              if (act.y) p[k].y = fmaf(be.y, p[k].y, r.y);
              if (act.z) p[k].z = fmaf(be.z, p[k].z, r.z);
              if (act.w) p[k].w = fmaf(be.w, p[k].w, r.w);
              *reinterpret_cast<float4*>(a.P + (size_t)(b0 + i) * a.ld + qoff) = p[k];
            }
          }
        }
      }
    }
    cluster_barrier();
  }
  // no block leaves while another may still read its partials
  cluster_barrier();
  const int c = 4 * CL * (int)cluster_index() + tid;
  if (rank == 0 && tid < CW && c < a.ld) {
    a.yy[c] = cl.yy[tid];
    a.rr[c] = cl.rr[tid];
    a.iters[c] = cl.iters[tid];
    a.conv[c] = cl.conv[tid];
  }
}

// ---------------------------------------------------------------------------- heavy rows
// The rows with more than H neighbours, ascending, in two launches and without any wait between
// blocks: block b first counts the heavy rows of its contiguous range [b per, (b + 1) per), then
// writes them, in order, after the counts of the blocks before it.  Integer counts: the list does
// not depend on timing.
constexpr int HLT = 256;

__global__ void __launch_bounds__(HLT) k_count_heavy(const int64_t* __restrict__ row_ptr,
                                                     int32_t n, int32_t H, int64_t per,
                                                     int* __restrict__ bcount) {
  __shared__ int s_cnt;
  if (threadIdx.x == 0) s_cnt = 0;
  __syncthreads();
  const int64_t u0 = (int64_t)blockIdx.x * per, u1 = min((int64_t)n, u0 + per);
  int c = 0;
  for (int64_t u = u0 + threadIdx.x; u < u1; u += HLT) c += (row_ptr[u + 1] - row_ptr[u]) > H;
  if (c) atomicAdd(&s_cnt, c);
  __syncthreads();
  if (threadIdx.x == 0) bcount[blockIdx.x] = s_cnt;
}

__global__ void __launch_bounds__(HLT) k_list_heavy(const int64_t* __restrict__ row_ptr,
                                                    int32_t n, int32_t H, int64_t per,
                                                    const int* __restrict__ bcount,
                                                    int32_t* __restrict__ list,
                                                    int64_t* __restrict__ count) {
  __shared__ unsigned long long s_off;
  __shared__ int s_wcnt[HLT / 32];
  if (threadIdx.x == 0) s_off = 0;
  __syncthreads();
  unsigned long long o = 0;
  for (int b = threadIdx.x; b < (int)blockIdx.x; b += HLT) o += (unsigned)bcount[b];
  if (o) atomicAdd(&s_off, o);
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t u0 = (int64_t)blockIdx.x * per, u1 = min((int64_t)n, u0 + per);
  int64_t off = (int64_t)s_off;
  for (int64_t base = u0; base < u1; base += HLT) {
    const int64_t u = base + threadIdx.x;
    const bool heavy = u < u1 && row_ptr[u + 1] - row_ptr[u] > H;
    const unsigned bal = __ballot_sync(0xffffffffu, heavy);
    if (lane == 0) s_wcnt[warp] = __popc(bal);
    __syncthreads();
    int64_t mine = off, tot = 0;
    for (int w = 0; w < HLT / 32; ++w) {
      if (w < warp) mine += s_wcnt[w];
      tot += s_wcnt[w];
    }
    if (heavy) list[mine + __popc(bal & ((1u << lane) - 1u))] = (int32_t)u;
    off += tot;
    __syncthreads();
  }
  if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) *count = off;
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
  // rows with more neighbours than an eighth of a group's mean share go to whole blocks: on
  // power-law graphs a group that drew a row near the mean share would otherwise hold up its
  // block long after the others finished
  const long long groups = (long long)(*grid) * gpb;
  long long h = 2 * g->m / (8 * groups);
  if (h < 32) h = 32;
  if (h > (1 << 20)) h = 1 << 20;
  *H = (int32_t)h;
}

erc_status build_heavy(const erc_graph* g, int32_t H, const HeavyRows& hv, cudaStream_t s) {
  const int grid = grid_for(g->n, 8 * HLT);  // at most 8 SMs' worth of blocks per SM, <= MAX_GRID
  const int64_t per = ((int64_t)g->n + grid - 1) / grid;
  k_count_heavy<<<grid, HLT, 0, s>>>(g->row_ptr, g->n, H, per, hv.bcount);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  k_list_heavy<<<grid, HLT, 0, s>>>(g->row_ptr, g->n, H, per, hv.bcount, hv.list, hv.count);
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
int resident_lpr(int nvec) { return nvec <= 4 ? 4 : nvec <= 8 ? 8 : nvec <= 16 ? 16 : 32; }

// the resident kernel for this shape (null where the row block is too wide for it); the
// preconditioned instantiations live in their own translation unit
const void* resident_kernel(int nvec, bool weighted, bool ps, bool pc) {
  return pc ? resident_kernel_pc(nvec, weighted, ps) : resident_kernel_for<false>(nvec, weighted, ps);
}

// Raise a kernel's dynamic shared-memory limit to everything the block may use, once per device
// and kernel; each launch then asks for what its plan needs.  Returns the limit (0 on failure).
size_t open_smem(const void* k) {
  static std::mutex mu;
  static const void* done_k[64][32] = {};
  static size_t done_v[64][32] = {};
  int dev = 0, optin = 0;
  cudaFuncAttributes fa;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < 32; ++i)
    if (done_k[dev][i] == k) return done_v[dev][i];
  if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess ||
      cudaFuncGetAttributes(&fa, k) != cudaSuccess || (size_t)optin <= fa.sharedSizeBytes) {
    cudaGetLastError();
    return 0;
  }
  const size_t lim = (size_t)optin - fa.sharedSizeBytes;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)lim) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  for (int i = 0; i < 32; ++i)
    if (!done_k[dev][i]) {
      done_k[dev][i] = k;
      done_v[dev][i] = lim;
      break;
    }
  return lim;
}

// shared memory of the resident kernel: r, Ap (and p with PS) of `rows` rows, the column
// partials, the region shared by the heavy-row slices and the reduction scratch, and the local
// heavy-row list
size_t resident_smem(int64_t rows, int ld, bool ps) {
  const size_t shared = resident_shared_floats_for(PT / resident_lpr(ld / 4), ld);
  return 4 * ((ps ? 3 : 2) * (size_t)rows * ld + 2 * (size_t)ld + shared + (size_t)rows);
}

bool resident_plan(const erc_graph* g, int ld, bool pc, int32_t* rb, size_t* smem,
                   const void** kern) {
  const int nvec = ld / 4;
  const int grid = sm_count();
  const int64_t rows = ((int64_t)g->n + grid - 1) / grid;
  for (int ps = 1; ps >= 0; --ps) {  // p in shared memory when it fits
    const void* k = resident_kernel(nvec, g->val != nullptr, ps, pc);
    if (!k) return false;
    const size_t bytes = resident_smem(rows, ld, ps);
    if (bytes > open_smem(k)) continue;
    int nb = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k, PT, bytes) != cudaSuccess || nb < 1) {
      cudaGetLastError();
      continue;
    }
    *rb = (int32_t)rows;
    *smem = bytes;
    *kern = k;
    return true;
  }
  return false;
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

// ---- cluster path: the largest cluster for which every column group's cluster is resident at
// once, and shared memory for the rows a block may take
struct ClusterPlan {
  const void* k = nullptr;
  int S = 0, groups = 0;
  int32_t rbmax = 0;
  size_t smem = 0;
};

void cluster_config(const ClusterPlan& pl, cudaStream_t s, cudaLaunchConfig_t* cfg,
                    cudaLaunchAttribute* attr) {
  *cfg = cudaLaunchConfig_t{};
  cfg->gridDim = dim3(pl.groups * pl.S);
  cfg->blockDim = dim3(CT);
  cfg->dynamicSmemBytes = pl.smem;
  cfg->stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = pl.S;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg->attrs = attr;
  cfg->numAttrs = 1;
}

bool cluster_plan(const erc_graph* g, int ld, ClusterPlan* pl) {
  const void* k = g->val ? (const void*)k_cg_cluster<true> : (const void*)k_cg_cluster<false>;
  const size_t lim = open_smem(k);
  if (!lim || cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) !=
                  cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  const int64_t row_bytes = 2 * CL * sizeof(float4);  // r and Ap of the group's columns
  const int64_t cap = ((int64_t)lim - 1024) / row_bytes;
  const int groups = (ld / 4 + CL - 1) / CL;
  for (int S = CMAXS; S >= 1; --S) {
    const int64_t even = ((int64_t)g->n + S - 1) / S;
    if (even > cap) break;  // smaller clusters need still more rows per block
    ClusterPlan p;
    p.k = k;
    p.S = S;
    p.groups = groups;
    p.rbmax = (int32_t)std::min(cap, even + even / 8 + 32);  // room to balance neighbour lists
    p.smem = (size_t)p.rbmax * row_bytes;
    cudaLaunchConfig_t cfg;
    cudaLaunchAttribute attr[1];
    cluster_config(p, nullptr, &cfg, attr);
    int nc = 0;
    if (cudaOccupancyMaxActiveClusters(&nc, k, &cfg) != cudaSuccess) {
      cudaGetLastError();
      continue;
    }
    if (nc < groups) continue;  // one wave: every group's cluster at once
    *pl = p;
    return true;
  }
  return false;
}

// Both single-launch plans for a graph shape, computed once per (device, n, ld, weighted,
// preconditioned): the occupancy queries behind them cost more host time than a small solve.
struct SolverPlans {
  bool cluster = false, resident = false;
  ClusterPlan cp;
  int32_t rb = 0;
  size_t smem = 0;
  const void* kres = nullptr;
};

SolverPlans solver_plans(const erc_graph* g, int ld, bool pc) {
  struct Entry {
    int dev = -1;
    int32_t n = 0, ld = 0;
    bool weighted = false, pc = false;
    SolverPlans p;
  };
  static std::mutex mu;
  static Entry cache[16];
  static int next = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  const bool weighted = g->val != nullptr;
  {
    std::lock_guard<std::mutex> lock(mu);
    for (const Entry& e : cache)
      if (e.dev == dev && e.n == g->n && e.ld == ld && e.weighted == weighted && e.pc == pc)
        return e.p;
  }
  SolverPlans p;
  p.cluster = !pc && cluster_plan(g, ld, &p.cp);  // the cluster solver has no preconditioner
  p.resident = resident_plan(g, ld, pc, &p.rb, &p.smem, &p.kres);
  std::lock_guard<std::mutex> lock(mu);
  Entry& e = cache[next];
  next = (next + 1) % 16;
  e.dev = dev;
  e.n = g->n;
  e.ld = ld;
  e.weighted = weighted;
  e.pc = pc;
  e.p = p;
  return p;
}

// Where both single-launch solvers fit, the cheaper per iteration by a model fitted to GB300
// timings: the resident gather costs ~2.4 ns per 128-byte neighbour line per SM plus ~18 us of
// synchronisation and vector work; the cluster gather ~2.6 ns per neighbour per block (one
// request per column group) plus ~10 us.  Small graphs favour the cluster solver.
bool prefer_cluster(const erc_graph* g, int ld, const ClusterPlan& cp) {
  const double nnz = 2.0 * (double)g->m;
  const double lines = std::max(1.0, ld / 32.0);
  const double t_res = 18.0 + nnz * lines * 2.4e-3 / sm_count();
  const double t_cl = 10.0 + nnz / cp.S * 2.6e-3;
  return t_cl < t_res;
}

erc_status launch_cluster(const ClusterPlan& pl, const ClusterArgs& ca, cudaStream_t s) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  cluster_config(pl, s, &cfg, attr);
  void* args[] = {const_cast<ClusterArgs*>(&ca)};
  ERC_CUDA(cudaLaunchKernelExC(&cfg, pl.k, args));
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
  const void* ptr[15];
  long long num[11];
  bool operator==(const GraphKey& o) const {
    for (int i = 0; i < 15; ++i)
      if (ptr[i] != o.ptr[i]) return false;
    for (int i = 0; i < 11; ++i)
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
  const void* ptrs[15] = {sa.row_ptr, sa.col, sa.val, sa.P, sa.AP, va.X, va.R, va.alpha,
                          va.active, va.flags, sa.cr.part1, va.Y, sa.heavy, va.gen, va.deg};
  for (int i = 0; i < 15; ++i) k.ptr[i] = ptrs[i];
  int eps_bits = 0;
  long long tol_bits = 0;
  memcpy(&eps_bits, &sa.eps, sizeof eps_bits);
  memcpy(&tol_bits, &va.tol2, sizeof tol_bits);
  long long nums[11] = {sa.n, sa.ld, sa.kc, eps_bits, tol_bits, va.max_iter, S, dev, sgrid,
                        (long long)ugrid << 32 | (unsigned)sa.H, (long long)va.spin_limit};
  for (int i = 0; i < 11; ++i) k.num[i] = nums[i];
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

erc_status erc::cg_enqueue(const erc_graph* g, float eps, const float* Y, float* X, int32_t ld,
                           int32_t kc, float tol, int32_t max_iter, int32_t* iters, float* relres,
                           void* ws, size_t ws_bytes, cudaStream_t s, bool reset_flags,
                           cudaEvent_t ev0, cudaEvent_t ev1, int32_t* path, bool precond) {
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(!precond || g->deg, "the Jacobi preconditioner needs the degrees (deg)");
  ERC_REQUIRE(kc >= 1 && ld >= kc && ld % 4 == 0 && ld <= MAX_LD, "bad kc %d / ld %d", kc, ld);
  ERC_REQUIRE(eps > 0.f && isfinite(eps), "eps must be positive");
  ERC_REQUIRE(tol >= 0.f && isfinite(tol), "tol must be finite and >= 0");
  ERC_REQUIRE(max_iter >= 1, "max_iter must be >= 1");
  ERC_REQUIRE(iters && relres, "iters and relres are required");
  ERC_TRY(check_block(Y, "Y"));
  ERC_TRY(check_block(X, "X"));
  if (ws_bytes < erc_batched_cg_workspace_size(g->n, ld))
    return set_error(ERC_ERR_CAPACITY, "workspace too small");
  Arena ar(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  CgWork w;
  plan_cg(ar, w, g->n, ld);
  ERC_CUDA(cudaMemsetAsync(w.cr.cnt, 0, colreduce_counter_bytes(), s));
  if (reset_flags) ERC_CUDA(cudaMemsetAsync(w.flags, 0, 8 * sizeof(int), s));
  ERC_CUDA(cudaMemsetAsync(w.gen, 0, 8 * sizeof(unsigned), s));

  int sgrid = 1;
  int32_t H = 0;
  spmm_shape(g, ld, &sgrid, &H);
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
  va.deg = precond ? g->deg : nullptr;
  va.eps = eps;
  va.spin_limit = wait_limit(SPIN_LIMIT);

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

  // path: 2 cluster (column groups), 1 resident (one cooperative launch), 0 multi-kernel graph.
  // ERC_CG_MODE=graph|resident|cluster restricts the choice (testing of every path).
  const char* mode = getenv("ERC_CG_MODE");
  const SolverPlans plans = solver_plans(g, ld, precond);
  const ClusterPlan& cp = plans.cp;
  const int32_t rb = plans.rb;
  const size_t smem = plans.smem;
  const void* kres = plans.kres;
  bool cluster = (!mode || strcmp(mode, "cluster") == 0) && plans.cluster;
  bool resident = (!mode || strcmp(mode, "resident") == 0) && plans.resident;
  if (cluster && resident) {
    if (prefer_cluster(g, ld, cp))
      resident = false;
    else
      cluster = false;
  }
  if (path) *path = cluster ? 2 : resident ? 1 : 0;
  // the resident kernel finds its own heavy rows, initialises its columns and forms the true
  // residual itself; the cluster kernel initialises its own columns
  if (!resident) ERC_TRY(build_heavy(g, H, w.heavy, s));
  if (!cluster && !resident) {
    k_cg_init<<<grid_for(g->n, vec_threads(nvec) / nvec), vec_threads(nvec), 0, s>>>(va);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
  }
  if (ev0) ERC_CUDA(cudaEventRecord(ev0, s));
  if (cluster) {
    ClusterArgs ca{};
    ca.row_ptr = g->row_ptr;
    ca.col = g->col;
    ca.val = g->val;
    ca.n = g->n;
    ca.ld = ld;
    ca.kc = kc;
    ca.eps = eps;
    ca.tol2 = va.tol2;
    ca.max_iter = max_iter;
    ca.rbmax = cp.rbmax;
    ca.Y = Y;
    ca.X = X;
    ca.P = w.P;
    ca.yy = w.yy;
    ca.rr = w.rr;
    ca.iters = w.iters;
    ca.conv = w.conv;
    ca.flags = w.flags;
    ERC_TRY(launch_cluster(cp, ca, s));
  } else if (resident) {
    // the whole solve in one cooperative launch, no host round trips
    ResArgs ra{sa, va, rb};
    ra.v.spin_limit = wait_limit(RES_SPIN_LIMIT);
    ERC_TRY(launch_resident(kres, ra, smem, s));
  } else {
    const int S = iterations_per_poll(g, ld);
    cudaGraphExec_t exec = nullptr;
    ERC_TRY(iteration_graph(sa, sgrid, va, ugrid, S, &exec));
    int done = 0;
    int h_flags[4] = {1, 0, 0, 0};
    while (done < max_iter) {
      ERC_CUDA(cudaGraphLaunch(exec, s));
      count_launches(2LL * S);  // the graph holds S iterations of two kernels
      done += S;
      ERC_CUDA(cudaMemcpyAsync(h_flags, w.flags, 4 * sizeof(int), cudaMemcpyDeviceToHost, s));
      ERC_CUDA(cudaStreamSynchronize(s));
      if (!h_flags[0] || h_flags[3]) break;  // every column stopped, or a wait gave up
    }
  }
  if (ev1) ERC_CUDA(cudaEventRecord(ev1, s));

  // true residual of the returned iterate, plus the per-column outputs
  if (!resident) {
    SpmmArgs ra = sa;
    ra.P = X;
    ERC_TRY(launch_spmm<MODE_RESID>(ra, sgrid, s));
  }
  return ERC_OK;
}

erc_status erc::cg_status(int32_t n, int32_t ld, int32_t columns, int32_t max_iter, void* ws,
                          cudaStream_t s) {
  Arena ar(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  CgWork w;
  plan_cg(ar, w, n, ld);
  int h_flags[4] = {0, 0, 0, 0};
  ERC_CUDA(cudaMemcpyAsync(h_flags, w.flags, 4 * sizeof(int), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaStreamSynchronize(s));
  if (h_flags[3]) return set_error(ERC_ERR_TIMEOUT, "a bounded grid-wide wait timed out");
  if (h_flags[1]) return set_error(ERC_ERR_NUMERIC, "non-finite or non-positive CG scalar");
  if (h_flags[2])
    return set_error(ERC_ERR_NOT_CONVERGED, "%d of %d columns reached max_iter=%d", h_flags[2],
                     columns, max_iter);
  return ERC_OK;
}

static erc_status batched_cg_impl(const erc_graph* g, float eps, const float* Y, float* X,
                                  int32_t ld, int32_t kc, float tol, int32_t max_iter,
                                  int32_t* iters, float* relres, void* ws, size_t ws_bytes,
                                  erc_stream stream, float* solve_us, int32_t* path,
                                  bool precond) {
  cudaStream_t s = as_stream(stream);
  cudaEvent_t ev[2] = {nullptr, nullptr};
  if (solve_us) {
    ERC_CUDA(cudaEventCreate(&ev[0]));
    ERC_CUDA(cudaEventCreate(&ev[1]));
  }
  erc_status st = cg_enqueue(g, eps, Y, X, ld, kc, tol, max_iter, iters, relres, ws, ws_bytes, s,
                             true, ev[0], ev[1], path, precond);
  if (st == ERC_OK) st = cg_status(g->n, ld, kc, max_iter, ws, s);
  if (solve_us) {
    float ms = 0.f;
    const cudaError_t e =
        st == ERC_OK || st == ERC_ERR_NOT_CONVERGED ? cudaEventElapsedTime(&ms, ev[0], ev[1])
                                                    : cudaSuccess;
    cudaEventDestroy(ev[0]);
    cudaEventDestroy(ev[1]);
    if (e != cudaSuccess) return set_error(ERC_ERR_CUDA, "event timing: %s", cudaGetErrorString(e));
    *solve_us = 1000.f * ms;
  }
  return st;
}

extern "C" erc_status erc_batched_cg(const erc_graph* g, float eps, const float* Y, float* X,
                                     int32_t ld, int32_t kc, float tol, int32_t max_iter,
                                     int32_t* iters, float* relres, void* ws, size_t ws_bytes,
                                     erc_stream stream) {
  clear_error();
  return batched_cg_impl(g, eps, Y, X, ld, kc, tol, max_iter, iters, relres, ws, ws_bytes, stream,
                         nullptr, nullptr, false);
}

extern "C" erc_status erc_batched_cg_timed(const erc_graph* g, float eps, const float* Y,
                                           float* X, int32_t ld, int32_t kc, float tol,
                                           int32_t max_iter, int32_t* iters, float* relres,
                                           void* ws, size_t ws_bytes, float* solve_us,
                                           int32_t* path, erc_stream stream) {
  clear_error();
  ERC_REQUIRE(solve_us && path, "solve_us and path are required");
  return batched_cg_impl(g, eps, Y, X, ld, kc, tol, max_iter, iters, relres, ws, ws_bytes, stream,
                         solve_us, path, false);
}

extern "C" erc_status erc_batched_pcg(const erc_graph* g, float eps, const float* Y, float* X,
                                      int32_t ld, int32_t kc, float tol, int32_t max_iter,
                                      int32_t* iters, float* relres, void* ws, size_t ws_bytes,
                                      erc_stream stream) {
  clear_error();
  return batched_cg_impl(g, eps, Y, X, ld, kc, tol, max_iter, iters, relres, ws, ws_bytes, stream,
                         nullptr, nullptr, true);
}

extern "C" erc_status erc_batched_pcg_timed(const erc_graph* g, float eps, const float* Y,
                                            float* X, int32_t ld, int32_t kc, float tol,
                                            int32_t max_iter, int32_t* iters, float* relres,
                                            void* ws, size_t ws_bytes, float* solve_us,
                                            int32_t* path, erc_stream stream) {
  clear_error();
  ERC_REQUIRE(solve_us && path, "solve_us and path are required");
  return batched_cg_impl(g, eps, Y, X, ld, kc, tol, max_iter, iters, relres, ws, ws_bytes, stream,
                         solve_us, path, true);
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
