// rhs.cu -- erc_jl_rhs: Y = B^T W^{1/2} Q for a batch of projection columns (§3.1.2), with the
// signs of Q generated in registers by Philox4x32-10 and never stored.
//
// Row u of Y gathers over u's CSR slots: the canonical edge e = (eu, ev) contributes
// sigma * sqrt(w_e) * Q[e, c] with sigma = +1 when u = eu (the smaller id) and -1 otherwise.
// Summing in CSR order makes Y deterministic without atomics.
#include "erc_internal.cuh"

namespace erc {
namespace {

// Row u of Y: the LPR lanes of a group walk u's CSR slots LPR at a time.  Lane l generates the
// Philox blocks of slot jb + l (one per 128-column block its group covers) and the slot's signed
// coefficient; the slots are then applied in CSR order, each lane taking from the generating
// lane, by shuffles, the word that holds its four columns' sign bits.
template <int LPR, int VPL, bool WEIGHTED>
__global__ void __launch_bounds__(256)
    k_jl_rhs(const int64_t* __restrict__ row_ptr, const int32_t* __restrict__ col,
             const float* __restrict__ val, const int32_t* __restrict__ csr_eid, int32_t n,
             uint2 key, float inv_sqrt_k, int32_t c0, int32_t kc, int32_t ld, float* __restrict__ Y) {
  constexpr int NBM = VPL + 1;  // 128-column Philox blocks a group's columns can span
  const int gl = threadIdx.x & (LPR - 1);
  const unsigned gm = group_mask<LPR>();
  const int groups_per_block = blockDim.x / LPR;
  const int64_t ngroups = (int64_t)gridDim.x * groups_per_block;
  const int nvec = ld >> 2;
  const int g0 = c0 >> 7;
  const int nb = ((c0 + 4 * (nvec - 1)) >> 7) - g0 + 1;
  int blk[VPL], wsel[VPL], sh[VPL];
  bool on[VPL];
#pragma unroll
  for (int v = 0; v < VPL; ++v) {
    const int q = gl + LPR * v;
    const int c = c0 + 4 * q;  // c0 % 4 == 0: the four columns share one word
    on[v] = q < nvec && 4 * q < kc;
    blk[v] = (c >> 7) - g0;
    wsel[v] = (c >> 5) & 3;
    sh[v] = c & 31;
  }
  for (int64_t u = (int64_t)blockIdx.x * groups_per_block + threadIdx.x / LPR; u < n;
       u += ngroups) {
    float4 acc[VPL];
#pragma unroll
    for (int v = 0; v < VPL; ++v) acc[v] = make_float4(0.f, 0.f, 0.f, 0.f);
    const int64_t j0 = row_ptr[u], j1 = row_ptr[u + 1];
    for (int64_t jb = j0; jb < j1; jb += LPR) {
      const int64_t j = jb + gl;
      float coef = 0.f;
      uint4 w[NBM];
#pragma unroll
      for (int b = 0; b < NBM; ++b) w[b] = make_uint4(0u, 0u, 0u, 0u);
      if (j < j1) {
        const uint32_t e = (uint32_t)csr_eid[j];
        coef = WEIGHTED ? sqrtf(val[j]) * inv_sqrt_k : inv_sqrt_k;
        if (col[j] < u) coef = -coef;  // u is the larger endpoint: row e of B is e_nb - e_u
#pragma unroll
        for (int b = 0; b < NBM; ++b)
          if (b < nb) w[b] = philox4x32_10(make_uint4((uint32_t)(g0 + b), 0u, e, 0u), key);
      }
      const int cnt = (int)min((int64_t)LPR, j1 - jb);
      for (int k = 0; k < cnt; ++k) {
        const float cf = __shfl_sync(gm, coef, k, LPR);
        uint32_t word[VPL];
#pragma unroll
        for (int v = 0; v < VPL; ++v) word[v] = 0u;
#pragma unroll
        for (int b = 0; b < NBM; ++b) {
          if (b >= nb) break;
          const uint32_t x = __shfl_sync(gm, w[b].x, k, LPR), y = __shfl_sync(gm, w[b].y, k, LPR);
          const uint32_t z = __shfl_sync(gm, w[b].z, k, LPR), t = __shfl_sync(gm, w[b].w, k, LPR);
#pragma unroll
          for (int v = 0; v < VPL; ++v)
            if (blk[v] == b) word[v] = wsel[v] == 0 ? x : wsel[v] == 1 ? y : wsel[v] == 2 ? z : t;
        }
#pragma unroll
        for (int v = 0; v < VPL; ++v) {
          if (!on[v]) continue;
          const uint32_t bits = word[v] >> sh[v];
          acc[v].x += (bits & 1u) ? -cf : cf;
          acc[v].y += (bits & 2u) ? -cf : cf;
          acc[v].z += (bits & 4u) ? -cf : cf;
          acc[v].w += (bits & 8u) ? -cf : cf;
        }
      }
    }
#pragma unroll
    for (int v = 0; v < VPL; ++v) {
      const int q = gl + LPR * v;
      if (q < nvec) {
        float4 o = acc[v];
        const int cb = 4 * q;
        if (cb + 0 >= kc) o.x = 0.f;
        if (cb + 1 >= kc) o.y = 0.f;
        if (cb + 2 >= kc) o.z = 0.f;
        if (cb + 3 >= kc) o.w = 0.f;
        reinterpret_cast<float4*>(Y + (size_t)u * ld)[q] = o;
      }
    }
  }
}

__global__ void k_philox_signs(uint2 key, int64_t e0, int64_t e1, int32_t c0, int32_t c1,
                               uint32_t* __restrict__ out) {
  const int64_t ncol = c1 - c0;
  const int64_t total = (e1 - e0) * ncol;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t e = e0 + t / ncol;
    const int c = c0 + (int)(t % ncol);
    const uint4 w = philox4x32_10(
        make_uint4((uint32_t)(c >> 7), 0u, (uint32_t)(e & 0xffffffff), (uint32_t)(e >> 32)), key);
    const int wi = (c >> 5) & 3;
    const uint32_t word = wi == 0 ? w.x : wi == 1 ? w.y : wi == 2 ? w.z : w.w;
    out[t] = (word >> (c & 31)) & 1u;
  }
}

}  // namespace
}  // namespace erc

using namespace erc;

extern "C" erc_status erc_jl_rhs(const erc_graph* g, uint64_t seed, int32_t K, int32_t c0,
                                 int32_t kc, float* Y, int32_t ld, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(K >= 1 && kc >= 1 && c0 >= 0 && (int64_t)c0 + kc <= K,
              "need 0 <= c0, 1 <= kc, c0 + kc <= K (c0=%d kc=%d K=%d)", c0, kc, K);
  ERC_REQUIRE(c0 % 4 == 0, "c0 must be a multiple of 4 (got %d)", c0);
  ERC_REQUIRE(ld >= kc && ld % 4 == 0 && ld <= MAX_LD, "bad ld %d for kc %d", ld, kc);
  ERC_REQUIRE(Y && (reinterpret_cast<uintptr_t>(Y) & 15) == 0, "Y must be 16-byte aligned");
  ERC_REQUIRE(g->m < (int64_t(1) << 31), "m must be < 2^31");
  cudaStream_t s = as_stream(stream);
  const uint2 key = make_uint2((uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32));
  const float inv_sqrt_k = (float)(1.0 / sqrt((double)K));
  return dispatch_shape(ld / 4, [&](auto lpr, auto vpl) -> erc_status {
    constexpr int LPR = decltype(lpr)::value, VPL = decltype(vpl)::value;
    const int grid = grid_for(g->n, 256 / LPR);
    if (g->val)
      k_jl_rhs<LPR, VPL, true><<<grid, 256, 0, s>>>(g->row_ptr, g->col, g->val, g->csr_eid, g->n,
                                                    key, inv_sqrt_k, c0, kc, ld, Y);
    else
      k_jl_rhs<LPR, VPL, false><<<grid, 256, 0, s>>>(g->row_ptr, g->col, g->val, g->csr_eid, g->n,
                                                     key, inv_sqrt_k, c0, kc, ld, Y);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    return ERC_OK;
  });
}

extern "C" erc_status erc_philox_signs(uint64_t seed, int64_t e0, int64_t e1, int32_t c0,
                                       int32_t c1, uint32_t* out_bits, erc_stream stream) {
  clear_error();
  ERC_REQUIRE(e0 >= 0 && e1 >= e0 && c0 >= 0 && c1 >= c0, "bad ranges");
  ERC_REQUIRE(out_bits || e1 == e0 || c1 == c0, "out_bits is required");
  const int64_t total = (e1 - e0) * (int64_t)(c1 - c0);
  if (total == 0) return ERC_OK;
  const uint2 key = make_uint2((uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32));
  k_philox_signs<<<grid_for(total, 256), 256, 0, as_stream(stream)>>>(key, e0, e1, c0, c1,
                                                                      out_bits);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  return ERC_OK;
}
