// cg_device.cuh -- device code shared by the CG translation units: the operator's argument
// block and row gather (L_eps p_u = eps p_u + sum_v w_uv (p_u - p_v), Eq. 5), the per-column
// dot-product combination, and the resident CG kernel (Algorithm 1, §3.1.3), whose plain and
// Jacobi-preconditioned instantiations are compiled in separate units.
#pragma once

#include "erc_internal.cuh"

namespace erc {
namespace {

constexpr int T = 256;
constexpr int WARPS = T / 32;
constexpr int SMEM_FLOATS = 8192;  // 32 KB: heavy-row combine buffer, or the reduction buffers
// default poll limits of the bounded waits: the vector update's grid barrier (which sleeps 64 ns
// between polls) and the resident solver's synchronisations (one L2 round trip per poll); either
// is seconds, far beyond any legitimate wait
constexpr unsigned SPIN_LIMIT = 1u << 24;
constexpr unsigned RES_SPIN_LIMIT = 1u << 22;
enum { MODE_STEP = 0, MODE_APPLY = 1, MODE_RESID = 2 };

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

// acc += sum_{j in [j0, j1)} w_j (p_u - p_{col_j}) for this lane's float4 column slots
// q = qb + gl + LPR v < qend whose bit v of `on` is set (the others keep acc); p is the n x ld
// block src_rows.  L2ONLY loads p through L2 only: required where p is rewritten
// within the same launch.
template <int LPR, int VPL, bool WEIGHTED, bool L2ONLY = false, int UB = 8>
__device__ __forceinline__ void gather_range(const SpmmArgs& a, const float* __restrict__ src_rows,
                                             int gl, unsigned gm, int qb, int qend,
                                             const float4 (&pu)[VPL], int64_t j0, int64_t j1,
                                             float4 (&acc)[VPL], unsigned on = ~0u) {
  constexpr int U = VPL >= UB ? 1 : UB / VPL;  // neighbour rows in flight per group
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
          const int q = qb + gl + LPR * v;
          const float* src = src_rows + (size_t)cj[k] * a.ld + 4 * q;
          pv[k][v] = (q < qend && t + k < cnt && ((on >> v) & 1u))
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

// the vectors and per-column state of one batched solve
struct VecArgs {
  int32_t n, ld, kc;
  double tol2;
  int32_t max_iter;
  const float* Y;
  float *X, *R, *P, *AP;
  float *alpha, *beta;
  double *rr, *yy;  // rr: r.r, or r.z with the Jacobi preconditioner; yy: y.y
  int *active, *conv, *iters, *flags;
  unsigned* gen;
  ColReduce cr;
  // Jacobi preconditioner M = diag(L_eps) = deg + eps (z = r / M): the weighted degrees, or
  // null for plain CG
  const float* deg;
  float eps;
  unsigned spin_limit;  // polls of a bounded wait before it gives up (sets flags[3])
};

// 1 / (deg_u + eps), the inverse diagonal of L_eps at row u
__device__ __forceinline__ float jacobi_inv(const float* deg, int64_t u, float eps) {
  return 1.f / (__ldg(deg + u) + eps);
}

__device__ __forceinline__ float4 f4_scale(float4 v, float s) {
  return make_float4(v.x * s, v.y * s, v.z * s, v.w * s);
}

// ---------------------------------------------------------------------------- resident CG
// When r and Ap of every row fit in the SMs' shared memory, one cooperative launch runs the whole
// solve.  Block b owns rows [b rb, b rb + rb): their r and Ap live in its shared memory, x and p
// in global memory (p is gathered by other blocks); where room is left (PS), the block's own rows
// of p are kept in shared memory too, and global p is only written and gathered.  Per iteration:
//   A  Ap = L_eps p on own rows (heavy rows by the whole block), p.Ap    -> reduce: alpha
//   B  x += alpha p, r -= alpha Ap, r.r                                  -> reduce: beta, stop
//   C  p = r + beta p                                                    -> barrier
// A grid synchronisation is an arrival (a release-add on a counter after the block's partials
// are written) and a bounded wait until all blocks have arrived.  There is no finishing block:
// after a reduction every block sums all blocks' partials itself, in the same fixed order, so
// every block derives the same alpha, beta and stop decisions into its own shared memory.  The
// counter only grows, so the s-th synchronisation waits for s * gridDim arrivals and needs no
// reset.  Data written by other blocks inside the launch (p, the partials) is read through L2
// (ld.global.cg), never through L1.  The vector phases B and C issue the loads of several rows
// before using any of them.
// With the Jacobi preconditioner (PC; an option, not the paper's method) z = r / (deg + eps):
// the start is p = z0, B also sums r.z (alpha and beta then use r.z in place of r.r, the stop
// test keeps r.r), and C forms p = z + beta p.
constexpr int PT = 512;
constexpr int PWARPS = PT / 32;
constexpr int PCH = 64;
constexpr int RMAXLD = 256;  // widest row block the resident kernel takes (64 float4)
constexpr int RU = 2;  // float4 loads per lane in flight in phases B and C
constexpr int RUB = 8;  // neighbour rows in flight per row group in the gathers

struct ResArgs {
  SpmmArgs s;
  VecArgs v;
  int32_t rb;  // rows per block
};

__device__ __forceinline__ float4 ldcg_f4(const float* p) {
  return __ldcg(reinterpret_cast<const float4*>(p));
}

// count this block in at the next synchronisation; the __syncthreads before thread 0's release
// orders the whole block's writes (and its reads of earlier partials) before it
__device__ __forceinline__ void res_arrive(unsigned* arr) {
  __syncthreads();
  if (threadIdx.x == 0) red_release_add(arr, 1u);
}
// bounded wait until `target` arrivals: after `limit` polls it sets flags[3] and returns
__device__ __forceinline__ void res_wait(const unsigned* arr, unsigned target, int* flags,
                                         unsigned limit) {
  if (threadIdx.x == 0) {
    unsigned spins = 0;
    while ((int)(ld_acquire(arr) - target) < 0) {  // one L2 round trip per poll
      if (++spins > limit) {
        atomicOr(&flags[3], 1);
        break;
      }
    }
  }
  __syncthreads();
}

// floats of the region shared by the heavy-row slices [GPB][ld] and the reduction scratch
// [2 * PT float pairs] of the resident kernel
__host__ __device__ constexpr size_t resident_shared_floats_for(int gpb, int ld) {
  return (size_t)gpb * ld > 4 * (size_t)PT ? (size_t)gpb * ld : 4 * (size_t)PT;
}
__device__ __forceinline__ size_t resident_shared_floats(int ld) {
  const int nvec = ld >> 2;
  const int lpr = nvec <= 4 ? 4 : nvec <= 8 ? 8 : nvec <= 16 ? 16 : 32;
  return resident_shared_floats_for(PT / lpr, ld);
}

// o = L_eps s on the block's rows, s = src_rows (n x ld; the block's own rows are read from `own`
// when it is not null): o_u = eps s_u + sum_v w_uv (s_u - s_v).  The block's rows heavier than
// a.H (the ascending local list hv[0..nh)) are split over all its groups and combined in group
// order; the others take one group each.  emit(i, v, s_u, o_u) runs once per row i and valid
// float4 slot v of the lane (for heavy rows in group 0).  Slots whose bit in `on` is clear are
// neither loaded nor gathered (s_u = 0 there).
template <int LPR, int VPL, bool WEIGHTED, class Emit>
__device__ __forceinline__ void block_apply(const SpmmArgs& a, const float* src_rows,
                                            const float* own, int64_t r0, int nrows,
                                            const int* hv, int nh, float* comb, int gl, int gi,
                                            unsigned gm, unsigned on, Emit&& emit) {
  constexpr int GPB = PT / LPR;
  const int ld = a.ld, nvec = ld >> 2;
  auto own_row = [&](int i, int v) -> float4 {
    const int q = gl + LPR * v;
    if (q >= nvec || !((on >> v) & 1u)) return f4_zero();
    return own ? reinterpret_cast<const float4*>(own + (size_t)i * ld)[q]
               : ldcg_f4(src_rows + (size_t)(r0 + i) * ld + 4 * q);
  };
  for (int hh = 0; hh < nh; ++hh) {
    const int i = hv[hh];
    const int64_t u = r0 + i;
    const int64_t j0 = a.row_ptr[u], j1 = a.row_ptr[u + 1];
    const int64_t per = (j1 - j0 + GPB - 1) / GPB;
    const int64_t s0 = min(j1, j0 + gi * per), s1 = min(j1, s0 + per);
    float4 pu[VPL], acc[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      pu[v] = own_row(i, v);
      acc[v] = f4_zero();
    }
    gather_range<LPR, VPL, WEIGHTED, true, RUB>(a, src_rows, gl, gm, 0, nvec, pu, s0, s1, acc, on);
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
        emit(i, v, pu[v], o);
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
      pu[v] = own_row(i, v);
      acc[v] = f4_zero();
    }
    gather_range<LPR, VPL, WEIGHTED, true, RUB>(a, src_rows, gl, gm, 0, nvec, pu, j0, j1, acc, on);
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      if (q >= nvec) continue;
      float4 o;
      o.x = fmaf(a.eps, pu[v].x, acc[v].x);
      o.y = fmaf(a.eps, pu[v].y, acc[v].y);
      o.z = fmaf(a.eps, pu[v].z, acc[v].z);
      o.w = fmaf(a.eps, pu[v].w, acc[v].w);
      emit(i, v, pu[v], o);
    }
  }
}

// the block's part of a grid-wide column sum: publish the block's partials (row blockIdx.x of
// part), count in, wait for every block, then sum all blocks' rows in a fixed order into sbuf
__device__ __forceinline__ void res_reduce(float2* part, int ld, const float2* bpart,
                                           float2* sbuf, float2* scratch, unsigned* arrivals,
                                           unsigned& nsync, int* flags, unsigned limit) {
  for (int c = threadIdx.x; c < ld; c += PT) part[(size_t)blockIdx.x * ld + c] = bpart[c];
  res_arrive(arrivals);
  res_wait(arrivals, ++nsync * gridDim.x, flags, limit);
  colsum_rows(part, gridDim.x, ld, sbuf, scratch);
}

template <int LPR, int VPL, bool WEIGHTED, bool PS, bool PC>
__global__ void __launch_bounds__(PT, 1) k_cg_resident(ResArgs ra) {
  extern __shared__ __align__(16) float dsm[];
  const SpmmArgs& a = ra.s;
  const VecArgs& va = ra.v;
  constexpr int GPB = PT / LPR;
  constexpr int NU = RU > VPL ? RU / VPL : 1;  // rows whose loads are in flight together
  const int gl = threadIdx.x & (LPR - 1);
  const int gi = threadIdx.x / LPR;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int ld = a.ld, nvec = ld >> 2;
  const int G = gridDim.x;
  const unsigned gm = group_mask<LPR>();
  const int64_t r0 = (int64_t)blockIdx.x * ra.rb;
  const int nrows = (int)max((int64_t)0, min((int64_t)a.n, r0 + ra.rb) - r0);
  float* rs = dsm;                                     // [rb][ld]  r of own rows
  float* aps = rs + (size_t)ra.rb * ld;                // [rb][ld]  Ap of own rows
  float* ps = aps + (size_t)ra.rb * ld;                // [rb][ld]  p of own rows (PS only)
  float2* sbuf = reinterpret_cast<float2*>(PS ? ps + (size_t)ra.rb * ld : ps);  // [ld]
  // one region, used as the heavy-row slices [GPB][ld] in the operator and as the reduction
  // scratch [PWARPS][PCH] = 2 * PT float pairs after it; then the local heavy-row list [rb]
  float* comb = reinterpret_cast<float*>(sbuf + ld);
  float2* scratch = sbuf + ld;
  int* hv = reinterpret_cast<int*>(comb + resident_shared_floats(ld));
  // block partials, one region per reduction kind so that no block overwrites partials another
  // block may still be summing: [G][ld] each
  float2* part_pap = a.cr.part1;
  // r.r rounded to float: sums of squares lose at most 2^-24 of their total that way, and every
  // block reads half the bytes
  float* part_rr = reinterpret_cast<float*>(a.cr.part1 + (size_t)G * ld);
  float* part_rz = part_rr + (size_t)G * ld;  // r.z (PC), also a sum of non-negative terms
  float2* part_init = a.cr.part1 + 2 * (size_t)G * ld;
  float2* part_yz = a.cr.part1 + 3 * (size_t)G * ld;  // y.z at the start (PC)
  float2* part_res = a.cr.part1 + 4 * (size_t)G * ld;
  unsigned* arrivals = va.gen;
  // per-column CG state, the same in every block
  __shared__ float2 s_rr[RMAXLD], s_yy[RMAXLD];  // float pairs; s_rr holds r.z with PC
  __shared__ float2 s_rz[PC ? RMAXLD : 1];        // the new r.z of phase B (PC)
  __shared__ __align__(16) float s_alpha[RMAXLD], s_beta[RMAXLD];
  __shared__ __align__(16) int s_active[RMAXLD];
  __shared__ int s_iters[RMAXLD], s_conv[RMAXLD];
  __shared__ int s_nh, s_wcnt[PWARPS];

  // ---- the block's rows heavier than a.H, ascending
  if (threadIdx.x == 0) s_nh = 0;
  __syncthreads();
  for (int base = 0; base < nrows; base += PT) {
    const int i = base + threadIdx.x;
    const bool heavy = i < nrows && a.row_ptr[r0 + i + 1] - a.row_ptr[r0 + i] > a.H;
    const unsigned bal = __ballot_sync(0xffffffffu, heavy);
    if (lane == 0) s_wcnt[warp] = __popc(bal);
    __syncthreads();
    int off = s_nh, tot = 0;
    for (int w = 0; w < PWARPS; ++w) {
      if (w < warp) off += s_wcnt[w];
      tot += s_wcnt[w];
    }
    if (heavy) hv[off + __popc(bal & ((1u << lane) - 1u))] = i;
    __syncthreads();
    if (threadIdx.x == 0) s_nh += tot;
    __syncthreads();
  }
  const int nh = s_nh;

  // ---- r = p = y (columns kc.. zero; with PC p = z = y / (deg + eps)), x = 0; y.y (and y.z)
  // -> the per-column state
  float2 dot[VPL][4];
  float2 dz[PC ? VPL : 1][4];  // r.z partials (PC)
#pragma unroll
  for (int v = 0; v < VPL; ++v)
#pragma unroll
    for (int t = 0; t < 4; ++t) dot[v][t] = make_float2(0.f, 0.f);
#pragma unroll
  for (int v = 0; v < (PC ? VPL : 1); ++v)
#pragma unroll
    for (int t = 0; t < 4; ++t) dz[v][t] = make_float2(0.f, 0.f);
  for (int i = gi; i < nrows; i += GPB) {
    const float di = PC ? jacobi_inv(va.deg, r0 + i, a.eps) : 1.f;
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      if (q >= nvec) continue;
      const size_t o = (size_t)(r0 + i) * ld + 4 * q;
      float4 y = ld_f4(a.Y + o);
      const int cb = 4 * q;
      if (cb + 0 >= a.kc) y.x = 0.f;
      if (cb + 1 >= a.kc) y.y = 0.f;
      if (cb + 2 >= a.kc) y.z = 0.f;
      if (cb + 3 >= a.kc) y.w = 0.f;
      const float4 p0 = PC ? f4_scale(y, di) : y;
      reinterpret_cast<float4*>(rs + (size_t)i * ld)[q] = y;
      if (PS) reinterpret_cast<float4*>(ps + (size_t)i * ld)[q] = p0;
      *reinterpret_cast<float4*>(const_cast<float*>(a.P) + o) = p0;
      *reinterpret_cast<float4*>(va.X + o) = f4_zero();
      dot[v][0] = df_fma(dot[v][0], y.x, y.x);
      dot[v][1] = df_fma(dot[v][1], y.y, y.y);
      dot[v][2] = df_fma(dot[v][2], y.z, y.z);
      dot[v][3] = df_fma(dot[v][3], y.w, y.w);
      if constexpr (PC) {
        dz[v][0] = df_fma(dz[v][0], y.x, p0.x);
        dz[v][1] = df_fma(dz[v][1], y.y, p0.y);
        dz[v][2] = df_fma(dz[v][2], y.z, p0.z);
        dz[v][3] = df_fma(dz[v][3], y.w, p0.w);
      }
    }
  }
  unsigned nsync = 0;
  block_partials_groups<LPR, VPL, PWARPS, PCH>(dot, sbuf, scratch, ld);
  if constexpr (PC) {
    // y.y and y.z of the block published together, one synchronisation (which also publishes
    // p), then both sums: y.z to s_rr, y.y left in sbuf
    for (int c = threadIdx.x; c < ld; c += PT) part_init[(size_t)blockIdx.x * ld + c] = sbuf[c];
    block_partials_groups<LPR, VPL, PWARPS, PCH>(dz, sbuf, scratch, ld);
    for (int c = threadIdx.x; c < ld; c += PT) part_yz[(size_t)blockIdx.x * ld + c] = sbuf[c];
    res_arrive(arrivals);
    res_wait(arrivals, ++nsync * G, va.flags, va.spin_limit);
    colsum_rows(part_yz, G, ld, sbuf, scratch);
    for (int c = threadIdx.x; c < ld; c += PT) s_rr[c] = sbuf[c];
    colsum_rows(part_init, G, ld, sbuf, scratch);
  } else {
    res_reduce(part_init, ld, sbuf, sbuf, scratch, arrivals, nsync, va.flags,
               va.spin_limit);  // also publishes p
  }
  int any = 0;
  for (int c = threadIdx.x; c < ld; c += PT) {
    const float2 v = sbuf[c];
    const double vd = df_value(v);
    int act = 0, cv = 1;
    if (c < a.kc) {
      if (!isfinite(vd) || (PC && !isfinite(s_rr[c].x))) {
        cv = 0;
        if (blockIdx.x == 0) atomicOr(&va.flags[1], 1);
      } else if (vd > 0.0 && !(vd <= va.tol2 * vd)) {
        act = 1;
        cv = 0;
      }
    }
    s_yy[c] = v;
    if (!PC) s_rr[c] = v;
    s_alpha[c] = 0.f;
    s_beta[c] = 0.f;
    s_active[c] = act;
    s_iters[c] = 0;
    s_conv[c] = cv;
    any |= act;
  }
  any = __syncthreads_or(any);

  while (any) {
    if (*(volatile int*)&va.flags[3] != 0) break;
    // ---------------- A: Ap = L_eps p on own rows, p.Ap
    if (nsync > 1) res_wait(arrivals, nsync * G, va.flags, va.spin_limit);  // every p written
    // this lane's float4 slots with an active column: converged columns are neither gathered
    // nor updated (their alpha is 0)
    unsigned on = 0;
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      if (q < nvec) {
        const int4 act = reinterpret_cast<const int4*>(s_active)[q];
        if (act.x | act.y | act.z | act.w) on |= 1u << v;
      }
    }
#pragma unroll
    for (int v = 0; v < VPL; ++v)
#pragma unroll
      for (int t = 0; t < 4; ++t) dot[v][t] = make_float2(0.f, 0.f);
    block_apply<LPR, VPL, WEIGHTED>(
        a, a.P, PS ? ps : nullptr, r0, nrows, hv, nh, comb, gl, gi, gm, on,
        [&](int i, int v, float4 pu, float4 o) {
          reinterpret_cast<float4*>(aps + (size_t)i * ld)[gl + LPR * v] = o;
          dot[v][0] = df_fma(dot[v][0], pu.x, o.x);
          dot[v][1] = df_fma(dot[v][1], pu.y, o.y);
          dot[v][2] = df_fma(dot[v][2], pu.z, o.z);
          dot[v][3] = df_fma(dot[v][3], pu.w, o.w);
        });
    block_partials_groups<LPR, VPL, PWARPS, PCH>(dot, sbuf, scratch, ld);
    res_reduce(part_pap, ld, sbuf, sbuf, scratch, arrivals, nsync, va.flags, va.spin_limit);
    for (int c = threadIdx.x; c < ld; c += PT) {
      const float2 v = sbuf[c];
      float al = 0.f;
      if (s_active[c]) {
        const float q = df_div(s_rr[c], v);
        if (!(v.x > 0.f) || !isfinite(q)) {
          s_active[c] = 0;
          if (blockIdx.x == 0) atomicOr(&va.flags[1], 1);
        } else {
          al = q;
        }
      }
      s_alpha[c] = al;
    }
    __syncthreads();

    // ---------------- B: x += alpha p, r -= alpha Ap, r.r (and r.z)
    float4 al[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      al[v] = q < nvec ? reinterpret_cast<const float4*>(s_alpha)[q] : f4_zero();
      for (int t = 0; t < 4; ++t) dot[v][t] = make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int v = 0; v < (PC ? VPL : 1); ++v)
#pragma unroll
      for (int t = 0; t < 4; ++t) dz[v][t] = make_float2(0.f, 0.f);
    for (int i0 = gi; i0 < nrows; i0 += NU * GPB) {
      float4 p[NU][VPL], x[NU][VPL];
      float di[NU];
#pragma unroll
      for (int k = 0; k < NU; ++k)
        di[k] = PC && i0 + k * GPB < nrows ? jacobi_inv(va.deg, r0 + i0 + k * GPB, a.eps) : 1.f;
#pragma unroll
      for (int k = 0; k < NU; ++k)
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          const int i = i0 + k * GPB, q = gl + LPR * v;
          if (i < nrows && q < nvec && ((on >> v) & 1u)) {
            const size_t o = (size_t)(r0 + i) * ld + 4 * q;
            p[k][v] = PS ? reinterpret_cast<const float4*>(ps + (size_t)i * ld)[q] : ldcg_f4(a.P + o);
            x[k][v] = *reinterpret_cast<const float4*>(va.X + o);
          }
        }
#pragma unroll
      for (int k = 0; k < NU; ++k)
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          const int i = i0 + k * GPB, q = gl + LPR * v;
          if (i >= nrows || q >= nvec || !((on >> v) & 1u)) continue;
          float4 xx = x[k][v], r = reinterpret_cast<const float4*>(rs + (size_t)i * ld)[q];
          const float4 pp = p[k][v], ap = reinterpret_cast<const float4*>(aps + (size_t)i * ld)[q];
          xx.x = fmaf(al[v].x, pp.x, xx.x);
          xx.y = fmaf(al[v].y, pp.y, xx.y);
          xx.z = fmaf(al[v].z, pp.z, xx.z);
          xx.w = fmaf(al[v].w, pp.w, xx.w);
          r.x = fmaf(-al[v].x, ap.x, r.x);
          r.y = fmaf(-al[v].y, ap.y, r.y);
          r.z = fmaf(-al[v].z, ap.z, r.z);
          r.w = fmaf(-al[v].w, ap.w, r.w);
          *reinterpret_cast<float4*>(va.X + (size_t)(r0 + i) * ld + 4 * q) = xx;
          reinterpret_cast<float4*>(rs + (size_t)i * ld)[q] = r;
          dot[v][0] = df_fma(dot[v][0], r.x, r.x);
          dot[v][1] = df_fma(dot[v][1], r.y, r.y);
          dot[v][2] = df_fma(dot[v][2], r.z, r.z);
          dot[v][3] = df_fma(dot[v][3], r.w, r.w);
          if constexpr (PC) {
            const float4 z = f4_scale(r, di[k]);
            dz[v][0] = df_fma(dz[v][0], r.x, z.x);
            dz[v][1] = df_fma(dz[v][1], r.y, z.y);
            dz[v][2] = df_fma(dz[v][2], r.z, z.z);
            dz[v][3] = df_fma(dz[v][3], r.w, z.w);
          }
        }
    }
    block_partials_groups<LPR, VPL, PWARPS, PCH>(dot, sbuf, scratch, ld);
    for (int c = threadIdx.x; c < ld; c += PT)
      part_rr[(size_t)blockIdx.x * ld + c] = __fadd_rn(sbuf[c].x, sbuf[c].y);
    if constexpr (PC) {
      block_partials_groups<LPR, VPL, PWARPS, PCH>(dz, sbuf, scratch, ld);
      for (int c = threadIdx.x; c < ld; c += PT)
        part_rz[(size_t)blockIdx.x * ld + c] = __fadd_rn(sbuf[c].x, sbuf[c].y);
    }
    res_arrive(arrivals);
    res_wait(arrivals, ++nsync * G, va.flags, va.spin_limit);
    if constexpr (PC) {
      colsum_rows_f(part_rz, G, ld, sbuf, scratch);
      for (int c = threadIdx.x; c < ld; c += PT) s_rz[c] = sbuf[c];
    }
    colsum_rows_f(part_rr, G, ld, sbuf, scratch);
    any = 0;
    for (int c = threadIdx.x; c < ld; c += PT) {
      float be = 0.f;
      int act = s_active[c];
      if (act) {
        const float2 rn = sbuf[c];
        const float2 rho = PC ? s_rz[c] : rn;  // the numerator of beta
        const int it = s_iters[c] + 1;
        s_iters[c] = it;
        if (!isfinite(rn.x) || !isfinite(rho.x)) {
          act = 0;
          if (blockIdx.x == 0) atomicOr(&va.flags[1], 1);
        } else {
          be = df_div(rho, s_rr[c]);
          s_rr[c] = rho;
          if (df_value(rn) <= va.tol2 * df_value(s_yy[c])) {
            s_conv[c] = 1;
            act = 0;
          } else if (it >= va.max_iter) {
            act = 0;
          }
        }
        s_active[c] = act;
      }
      s_beta[c] = be;
      any |= act;
    }
    any = __syncthreads_or(any);  // the same in every block
    if (!any) break;

    // ---------------- C: p = r + beta p (PC: p = z + beta p) on active columns
    int4 act[VPL];
    float4 be[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      act[v] = q < nvec ? reinterpret_cast<const int4*>(s_active)[q] : make_int4(0, 0, 0, 0);
      be[v] = q < nvec ? reinterpret_cast<const float4*>(s_beta)[q] : f4_zero();
    }
    for (int i0 = gi; i0 < nrows; i0 += NU * GPB) {
      float4 p[NU][VPL];
      float di[NU];
#pragma unroll
      for (int k = 0; k < NU; ++k)
        di[k] = PC && i0 + k * GPB < nrows ? jacobi_inv(va.deg, r0 + i0 + k * GPB, a.eps) : 1.f;
#pragma unroll
      for (int k = 0; k < NU; ++k)
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          const int i = i0 + k * GPB, q = gl + LPR * v;
          if (i < nrows && (act[v].x | act[v].y | act[v].z | act[v].w))
            p[k][v] = PS ? reinterpret_cast<const float4*>(ps + (size_t)i * ld)[q]
                         : ldcg_f4(a.P + (size_t)(r0 + i) * ld + 4 * q);
        }
#pragma unroll
      for (int k = 0; k < NU; ++k)
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          const int i = i0 + k * GPB, q = gl + LPR * v;
          if (i >= nrows || !(act[v].x | act[v].y | act[v].z | act[v].w)) continue;
          float4 r = reinterpret_cast<const float4*>(rs + (size_t)i * ld)[q];
          if (PC) r = f4_scale(r, di[k]);  // z
          float4 pp = p[k][v];
          if (act[v].x) pp.x = fmaf(be[v].x, pp.x, r.x);
          if (act[v].y) pp.y = fmaf(be[v].y, pp.y, r.y);
          if (act[v].z) pp.z = fmaf(be[v].z, pp.z, r.z);
          if (act[v].w) pp.w = fmaf(be[v].w, pp.w, r.w);
          *reinterpret_cast<float4*>(const_cast<float*>(a.P) + (size_t)(r0 + i) * ld + 4 * q) = pp;
          if (PS) reinterpret_cast<float4*>(ps + (size_t)i * ld)[q] = pp;
        }
    }
    res_arrive(arrivals);
    ++nsync;
  }

  // ---- true residual y - L_eps x of the returned iterate (every block's x is final: the last
  // reduction ordered its writes), relative to ||y||; iterations and the unconverged count
#pragma unroll
  for (int v = 0; v < VPL; ++v)
#pragma unroll
    for (int t = 0; t < 4; ++t) dot[v][t] = make_float2(0.f, 0.f);
  block_apply<LPR, VPL, WEIGHTED>(
      a, va.X, nullptr, r0, nrows, hv, nh, comb, gl, gi, gm, ~0u,
      [&](int i, int v, float4, float4 o) {
        const int q = gl + LPR * v, cb = 4 * q;
        const float4 y = ld_f4(a.Y + (size_t)(r0 + i) * ld + 4 * q);
        const float rx = cb + 0 < a.kc ? y.x - o.x : 0.f;
        const float ry = cb + 1 < a.kc ? y.y - o.y : 0.f;
        const float rz = cb + 2 < a.kc ? y.z - o.z : 0.f;
        const float rw = cb + 3 < a.kc ? y.w - o.w : 0.f;
        dot[v][0] = df_fma(dot[v][0], rx, rx);
        dot[v][1] = df_fma(dot[v][1], ry, ry);
        dot[v][2] = df_fma(dot[v][2], rz, rz);
        dot[v][3] = df_fma(dot[v][3], rw, rw);
      });
  block_partials_groups<LPR, VPL, PWARPS, PCH>(dot, sbuf, scratch, ld);
  res_reduce(part_res, ld, sbuf, sbuf, scratch, arrivals, nsync, va.flags, va.spin_limit);
  if (blockIdx.x == 0)
    for (int c = threadIdx.x; c < a.kc; c += PT) {
      const float q = s_yy[c].x > 0.f ? df_div(sbuf[c], s_yy[c]) : 0.f;
      a.relres_out[c] = sqrtf(fmaxf(q, 0.f));
      a.iters_out[c] = s_iters[c];
      if (!s_conv[c]) atomicAdd(&va.flags[2], 1);
    }
}

// the resident kernel of a row-block shape: nvec float4 per row, weighted or not, p of the own
// rows in shared memory (ps) or not; null for rows wider than 256 floats
template <bool PC>
const void* resident_kernel_for(int nvec, bool weighted, bool ps) {
  const void* k = nullptr;
  auto pick = [&](auto lpr, auto vpl) {
    constexpr int LPR = decltype(lpr)::value, VPL = decltype(vpl)::value;
    if (ps)
      k = weighted ? (const void*)k_cg_resident<LPR, VPL, true, true, PC>
                   : (const void*)k_cg_resident<LPR, VPL, false, true, PC>;
    else
      k = weighted ? (const void*)k_cg_resident<LPR, VPL, true, false, PC>
                   : (const void*)k_cg_resident<LPR, VPL, false, false, PC>;
  };
  if (nvec <= 4) pick(ic<4>{}, ic<1>{});
  else if (nvec <= 8) pick(ic<8>{}, ic<1>{});
  else if (nvec <= 16) pick(ic<16>{}, ic<1>{});
  else if (nvec <= 32) pick(ic<32>{}, ic<1>{});
  else if (nvec <= 64) pick(ic<32>{}, ic<2>{});
  return k;  // wider rows use the multi-kernel path
}

}  // namespace

// the preconditioned (Jacobi) resident kernels, compiled in cg_pcg.cu
const void* resident_kernel_pc(int nvec, bool weighted, bool ps);

}  // namespace erc
