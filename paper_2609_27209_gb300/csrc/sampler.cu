// sampler.cu -- curvature-guided subgraph samplers (§3.2, Eq. 7 and Eq. 8: the experiments'
// ERC-LG-sub(node) and ERC-LG-sub(edge), GraphSAINT-style) and GraphSAINT's count normalisation.
//
// A draw is exact integer inverse-CDF sampling: the float32 probabilities become fixed-point
// weights W_i = round(p_i 2^40) (from the float's bits, no float arithmetic), an exclusive scan
// gives E_i = W_0 + .. + W_{i-1} and T, a 64-bit Philox word x gives r = floor(x T / 2^64), and
// the draw is the largest i with E_i <= r (that i has W_i > 0).  Everything is integer, so the
// drawn indices do not depend on summation order.  The drawn nodes (or the drawn edges'
// endpoints) are marked and compacted in id order; the subgraph's edges are the canonical edges
// with both endpoints marked (induced), or the drawn edges themselves, compacted in id order.
#include "erc_internal.cuh"

namespace erc {
namespace {

constexpr int ST = 256;
constexpr uint32_t SAMPLER_TAG = 0x53414D50u;

struct SamplePlan {
  int64_t *W, *E, *draws, *npos, *epos, *totals;  // totals: [0] T [1] nodes [2] edges
  uint8_t *nmark, *emark;
  unsigned* err;  // [0] a probability outside [0, 1]; [1] the abort word of the scans
  void* scan_tmp;
};

void plan_sample(Arena& a, SamplePlan& p, int64_t count, int32_t n, int64_t m, int64_t budget) {
  p.W = a.take<int64_t>(count);
  p.E = a.take<int64_t>(count);
  p.draws = a.take<int64_t>(budget > 0 ? budget : 1);
  p.nmark = a.take<uint8_t>(n);
  p.emark = a.take<uint8_t>(m > 0 ? m : 1);
  p.npos = a.take<int64_t>(n);
  p.epos = a.take<int64_t>(m > 0 ? m : 1);
  p.totals = a.take<int64_t>(4);
  p.err = a.take<unsigned>(4);
  int64_t big = count > n ? count : n;
  if (m > big) big = m;
  p.scan_tmp = a.take<char>(scan_temp_bytes(big));
}

// W_i = round(p_i 2^40) (half up) from the bits of p_i; p_i must lie in [0, 1]
__global__ void k_fixed_weights(const float* __restrict__ prob, int64_t count,
                                int64_t* __restrict__ W, unsigned* __restrict__ err) {
  bool bad = false;
  for (int64_t i = (int64_t)blockIdx.x * ST + threadIdx.x; i < count;
       i += (int64_t)gridDim.x * ST) {
    const float p = prob[i];
    int64_t w = 0;
    if (!(p >= 0.f && p <= 1.f)) {
      bad = true;
    } else if (p > 0.f) {
      const uint32_t bits = __float_as_uint(p);
      const int e = (int)(bits >> 23);
      const uint64_t mant = e ? ((bits & 0x7fffffu) | 0x800000u) : (bits & 0x7fffffu);
      const int shift = (e ? e - 150 : -149) + 40;  // p 2^40 = mant 2^shift
      if (shift >= 0)
        w = (int64_t)(mant << shift);
      else if (shift > -40)
        w = (int64_t)((mant + (1ull << (-shift - 1))) >> (-shift));
    }
    W[i] = w;
  }
  if (__syncthreads_or(bad) && threadIdx.x == 0) atomicOr(err, 1u);
}

// draw k: the largest i with E_i <= floor(x_k T / 2^64)
__global__ void k_draw(const int64_t* __restrict__ E, int64_t count,
                       const int64_t* __restrict__ tot, int64_t budget, uint2 key, int64_t first,
                       uint32_t stream, int64_t* __restrict__ draws) {
  const uint64_t T = (uint64_t)tot[0];
  for (int64_t k = (int64_t)blockIdx.x * ST + threadIdx.x; k < budget;
       k += (int64_t)gridDim.x * ST) {
    const uint64_t d = (uint64_t)(first + k);
    const uint4 w =
        philox4x32_10(make_uint4((uint32_t)d, (uint32_t)(d >> 32), SAMPLER_TAG, stream), key);
    const uint64_t x = ((uint64_t)w.x << 32) | w.y;
    const int64_t r = (int64_t)__umul64hi(x, T);
    int64_t lo = 0, hi = count;  // first index with E > r, minus one
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (E[mid] <= r) lo = mid + 1; else hi = mid;
    }
    draws[k] = lo - 1;
  }
}

__global__ void k_mark_draws(const int64_t* __restrict__ draws, int64_t budget, int edges,
                             const int32_t* __restrict__ eu, const int32_t* __restrict__ ev,
                             uint8_t* __restrict__ nmark, uint8_t* __restrict__ emark) {
  for (int64_t k = (int64_t)blockIdx.x * ST + threadIdx.x; k < budget;
       k += (int64_t)gridDim.x * ST) {
    const int64_t i = draws[k];
    if (edges) {
      emark[i] = 1;
      nmark[eu[i]] = 1;
      nmark[ev[i]] = 1;
    } else {
      nmark[i] = 1;
    }
  }
}

__global__ void k_mark_induced(const int32_t* __restrict__ eu, const int32_t* __restrict__ ev,
                               int64_t m, const uint8_t* __restrict__ nmark,
                               uint8_t* __restrict__ emark) {
  for (int64_t e = (int64_t)blockIdx.x * ST + threadIdx.x; e < m; e += (int64_t)gridDim.x * ST)
    emark[e] = nmark[eu[e]] & nmark[ev[e]];
}

__global__ void k_compact(const uint8_t* __restrict__ mark, const int64_t* __restrict__ pos,
                          int64_t count, int32_t* __restrict__ out) {
  for (int64_t i = (int64_t)blockIdx.x * ST + threadIdx.x; i < count;
       i += (int64_t)gridDim.x * ST)
    if (mark[i]) out[pos[i]] = (int32_t)i;
}

__global__ void k_saint_counts(const int32_t* __restrict__ nodes, int64_t n_s,
                               const int32_t* __restrict__ edges, int64_t m_s,
                               int32_t* __restrict__ node_count, int32_t* __restrict__ edge_count) {
  // ids are distinct within a subgraph, so each counter is touched once per call
  for (int64_t i = (int64_t)blockIdx.x * ST + threadIdx.x; i < n_s + m_s;
       i += (int64_t)gridDim.x * ST) {
    if (i < n_s)
      node_count[nodes[i]] += 1;
    else
      edge_count[edges[i - n_s]] += 1;
  }
}

__global__ void k_saint_norm(const int64_t* __restrict__ row_ptr,
                             const int32_t* __restrict__ csr_eid, int32_t n,
                             const int32_t* __restrict__ node_count,
                             const int32_t* __restrict__ edge_count, int32_t N,
                             float* __restrict__ lam, float* __restrict__ alpha) {
  for (int64_t v = (int64_t)blockIdx.x * ST + threadIdx.x; v < n; v += (int64_t)gridDim.x * ST) {
    const int32_t cv = node_count[v];
    lam[v] = __fdiv_rn((float)cv, (float)N);
    for (int64_t j = row_ptr[v]; j < row_ptr[v + 1]; ++j)
      alpha[j] = cv > 0 ? __fdiv_rn((float)edge_count[csr_eid[j]], (float)cv) : 0.f;
  }
}

}  // namespace
}  // namespace erc

using namespace erc;

extern "C" size_t erc_sample_workspace_size(int32_t n, int64_t m, int64_t budget) {
  if (n < 1 || m < 0 || budget < 0) return 0;
  Arena a(nullptr);
  SamplePlan p;
  plan_sample(a, p, n > m ? n : m, n, m, budget);
  return a.used + 256;
}

extern "C" erc_status erc_sample_subgraph(const erc_graph* g, int32_t kind, const float* prob,
                                          int64_t budget, uint64_t seed, int64_t first_draw,
                                          int32_t induced, int32_t* nodes, int32_t* n_out,
                                          int32_t* edges, int64_t* m_out, void* ws,
                                          size_t ws_bytes, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(kind == ERC_SAMPLE_NODES || kind == ERC_SAMPLE_EDGES, "bad sampler kind %d", kind);
  ERC_REQUIRE(budget >= 0 && first_draw >= 0, "budget and first_draw must be >= 0");
  ERC_REQUIRE(n_out && m_out, "n_out and m_out are required");
  ERC_REQUIRE(g->eu && g->ev, "graph edge list required");
  const bool by_edge = kind == ERC_SAMPLE_EDGES;
  const int64_t count = by_edge ? g->m : g->n;
  ERC_REQUIRE(prob || count == 0, "prob is required");
  ERC_REQUIRE(nodes && (edges || g->m == 0), "nodes and edges are required");
  if (ws_bytes < erc_sample_workspace_size(g->n, g->m, budget))
    return set_error(ERC_ERR_CAPACITY, "workspace too small");
  cudaStream_t s = as_stream(stream);
  Arena ar(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  SamplePlan p;
  plan_sample(ar, p, g->n > g->m ? g->n : g->m, g->n, g->m, budget);
  *n_out = 0;
  *m_out = 0;
  if (count == 0 || budget == 0) return ERC_OK;
  ERC_CUDA(cudaMemsetAsync(p.err, 0, 4 * sizeof(unsigned), s));
  ERC_CUDA(cudaMemsetAsync(p.nmark, 0, (size_t)g->n, s));
  if (g->m > 0) ERC_CUDA(cudaMemsetAsync(p.emark, 0, (size_t)g->m, s));
  k_fixed_weights<<<grid_for(count, ST), ST, 0, s>>>(prob, count, p.W, p.err);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  // the scans' prefixes are only ever below their true values when a bounded wait gives up, so
  // every index derived from them stays in range; the host then reports the timeout
  unsigned* abort = p.err + 1;
  ERC_TRY(exclusive_scan_i64(p.W, nullptr, p.E, count, &p.totals[0], p.scan_tmp, s, abort));
  int64_t T = 0;
  unsigned h_err[2] = {0, 0};
  ERC_CUDA(cudaMemcpyAsync(&T, p.totals, sizeof(int64_t), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaMemcpyAsync(h_err, p.err, 2 * sizeof(unsigned), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaStreamSynchronize(s));
  if (h_err[0]) return set_error(ERC_ERR_INVALID_ARG, "probabilities must lie in [0, 1]");
  if (h_err[1]) return set_error(ERC_ERR_TIMEOUT, "a bounded wait in the sampler's scan ran out");
  if (T == 0) return set_error(ERC_ERR_INVALID_ARG, "every probability rounds to zero");
  const uint2 key = make_uint2((uint32_t)(seed & 0xffffffffu), (uint32_t)(seed >> 32));
  k_draw<<<grid_for(budget, ST), ST, 0, s>>>(p.E, count, p.totals, budget, key, first_draw,
                                             by_edge ? 1u : 0u, p.draws);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  k_mark_draws<<<grid_for(budget, ST), ST, 0, s>>>(p.draws, budget, by_edge, g->eu, g->ev,
                                                   p.nmark, p.emark);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  if ((!by_edge || induced) && g->m > 0) {
    k_mark_induced<<<grid_for(g->m, ST), ST, 0, s>>>(g->eu, g->ev, g->m, p.nmark, p.emark);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
  }
  ERC_TRY(exclusive_scan_i64(nullptr, p.nmark, p.npos, g->n, &p.totals[1], p.scan_tmp, s, abort));
  k_compact<<<grid_for(g->n, ST), ST, 0, s>>>(p.nmark, p.npos, g->n, nodes);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  if (g->m > 0) {
    ERC_TRY(exclusive_scan_i64(nullptr, p.emark, p.epos, g->m, &p.totals[2], p.scan_tmp, s,
                               abort));
    k_compact<<<grid_for(g->m, ST), ST, 0, s>>>(p.emark, p.epos, g->m, edges);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
  }
  int64_t h_tot[3] = {0, 0, 0};
  ERC_CUDA(cudaMemcpyAsync(h_tot, p.totals, 3 * sizeof(int64_t), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaMemcpyAsync(h_err, p.err, 2 * sizeof(unsigned), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaStreamSynchronize(s));
  if (h_err[1]) return set_error(ERC_ERR_TIMEOUT, "a bounded wait in the sampler's scans ran out");
  *n_out = (int32_t)h_tot[1];
  *m_out = g->m > 0 ? h_tot[2] : 0;
  return ERC_OK;
}

extern "C" erc_status erc_saint_counts(const erc_graph* g, const int32_t* nodes, int32_t n_s,
                                       const int32_t* edges, int64_t m_s, int32_t* node_count,
                                       int32_t* edge_count, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(n_s >= 0 && n_s <= g->n && m_s >= 0 && m_s <= g->m, "bad subgraph sizes");
  ERC_REQUIRE((nodes && node_count) || n_s == 0, "nodes and node_count are required");
  ERC_REQUIRE((edges && edge_count) || m_s == 0, "edges and edge_count are required");
  if (n_s + m_s == 0) return ERC_OK;
  k_saint_counts<<<grid_for(n_s + m_s, ST), ST, 0, as_stream(stream)>>>(nodes, n_s, edges, m_s,
                                                                        node_count, edge_count);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  return ERC_OK;
}

extern "C" erc_status erc_saint_norm(const erc_graph* g, const int32_t* node_count,
                                     const int32_t* edge_count, int32_t N, float* lambda,
                                     float* alpha, erc_stream stream) {
  clear_error();
  ERC_TRY(check_graph(g));
  ERC_REQUIRE(N >= 1 && N < (1 << 24), "N must be in [1, 2^24)");
  ERC_REQUIRE(node_count && lambda && (g->m == 0 || (edge_count && alpha && g->csr_eid)),
              "counts and outputs are required");
  k_saint_norm<<<grid_for(g->n, ST), ST, 0, as_stream(stream)>>>(
      g->row_ptr, g->csr_eid, g->n, node_count, edge_count, N, lambda, alpha);
  count_launches(1);
  ERC_CUDA(cudaGetLastError());
  return ERC_OK;
}
