// build.cu -- erc_build_laplacian: the simple undirected graph behind L = D - A = B^T W B (§3.1.1).
//
// Every input edge (u, v), u != v, is emitted as the two directed keys (u<<B | v) and (v<<B | u)
// carrying its input index; a stable LSD radix sort on the low 2B key bits then lays the keys out
// in CSR order with duplicates adjacent and in input order.  A scan over run heads numbers the
// CSR slots, a second scan over the upper-triangle slots (col > row) numbers the canonical edges,
// and the lower slots find their edge id by a binary search in the partner row.
#include "erc_internal.cuh"

namespace erc {
namespace {

constexpr int BT = 256;

struct BuildPlan {
  uint64_t *keys, *keys_alt;
  uint32_t *vals, *vals_alt;
  uint8_t *head, *upper;
  int64_t *slot, *eidx;
  int32_t* row_of;
  float* wmerged;
  int64_t* counters;  // [0] nnz  [1] m
  unsigned* err;      // [0] bit 0: node id out of range, bit 1: bad weight; [1] a merged
                      // weight differs from 1; [2] the abort word (a scan's wait gave up)
  void *sort_tmp, *scan_tmp;
};

void plan_build(Arena& a, BuildPlan& p, int64_t m_in) {
  const int64_t E = 2 * m_in;
  p.keys = a.take<uint64_t>(E);
  p.keys_alt = a.take<uint64_t>(E);
  p.vals = a.take<uint32_t>(E);
  p.vals_alt = a.take<uint32_t>(E);
  p.head = a.take<uint8_t>(E);
  p.upper = a.take<uint8_t>(E);
  p.slot = a.take<int64_t>(E);
  p.eidx = a.take<int64_t>(E);
  p.row_of = a.take<int32_t>(E);
  p.wmerged = a.take<float>(E);
  p.counters = a.take<int64_t>(4);
  p.err = a.take<unsigned>(4);
  p.sort_tmp = a.take<char>(radix_sort_temp_bytes(E));
  p.scan_tmp = a.take<char>(scan_temp_bytes(E));
}

__device__ __forceinline__ int64_t gtid() { return (int64_t)blockIdx.x * blockDim.x + threadIdx.x; }
__device__ __forceinline__ int64_t gstride() { return (int64_t)gridDim.x * blockDim.x; }

__global__ void k_emit(const int32_t* __restrict__ src, const int32_t* __restrict__ dst,
                       const float* __restrict__ w, int64_t m_in, int32_t n, int B, uint64_t sent,
                       uint64_t* __restrict__ keys, uint32_t* __restrict__ vals,
                       unsigned* __restrict__ err) {
  unsigned bad = 0;
  for (int64_t i = gtid(); i < m_in; i += gstride()) {
    int32_t a = src[i], b = dst[i];
    bool range_ok = a >= 0 && a < n && b >= 0 && b < n;
    if (!range_ok) bad |= 1u;
    if (w) {
      float x = w[i];
      if (!(x > 0.f) || !isfinite(x)) bad |= 2u;
    }
    uint64_t k0 = sent, k1 = sent;
    if (range_ok && a != b) {
      k0 = ((uint64_t)a << B) | (uint64_t)b;
      k1 = ((uint64_t)b << B) | (uint64_t)a;
    }
    keys[2 * i] = k0;
    keys[2 * i + 1] = k1;
    vals[2 * i] = (uint32_t)i;
    vals[2 * i + 1] = (uint32_t)i;
  }
  if (bad) atomicOr(err, bad);
}

__global__ void k_heads(const uint64_t* __restrict__ keys, int64_t E, uint64_t sent,
                        uint8_t* __restrict__ head, const unsigned* abort) {
  if (aborted(abort)) return;  // the sort did not finish: nothing after it runs
  for (int64_t i = gtid(); i < E; i += gstride()) {
    uint64_t k = keys[i];
    head[i] = (k != sent) && (i == 0 || keys[i - 1] != k);
  }
}

// nonunit (may be null): set to 1 when some merged weight differs from 1 (unweighted inputs with
// merged duplicates)
__global__ void k_emit_csr(const uint64_t* __restrict__ keys, const uint32_t* __restrict__ vals,
                           const uint8_t* __restrict__ head, const int64_t* __restrict__ slot,
                           const float* __restrict__ w, int64_t E, int B, int dup_first,
                           int32_t* __restrict__ col, float* __restrict__ wmerged,
                           int32_t* __restrict__ row_of, uint8_t* __restrict__ upper,
                           unsigned* __restrict__ nonunit, const unsigned* abort) {
  if (aborted(abort)) return;
  const uint64_t mask = (1ull << B) - 1ull;
  bool other = false;
  for (int64_t i = gtid(); i < E; i += gstride()) {
    if (!head[i]) continue;
    const uint64_t k = keys[i];
    double acc;
    if (dup_first) {
      acc = w ? (double)w[vals[i]] : 1.0;
    } else {
      acc = 0.0;  // float64 sum of the duplicates in input order (the sort is stable)
      for (int64_t j = i; j < E && keys[j] == k; ++j) acc += w ? (double)w[vals[j]] : 1.0;
    }
    const int64_t s = slot[i];
    const int32_t r = (int32_t)(k >> B), c = (int32_t)(k & mask);
    col[s] = c;
    row_of[s] = r;
    wmerged[s] = (float)acc;
    upper[s] = c > r;
    other |= (float)acc != 1.f;
  }
  if (nonunit && __any_sync(0xffffffffu, other) && (threadIdx.x & 31) == 0) atomicOr(nonunit, 1u);
}

__global__ void k_row_ptr(const int32_t* __restrict__ row_of, const int64_t* __restrict__ counters,
                          int32_t n, int64_t* __restrict__ row_ptr, const unsigned* abort) {
  if (aborted(abort)) return;
  const int64_t nnz = counters[0];
  for (int64_t s = gtid(); s < nnz; s += gstride()) {
    int32_t r = row_of[s];
    int32_t prev = s == 0 ? -1 : row_of[s - 1];
    for (int32_t q = prev + 1; q <= r; ++q) row_ptr[q] = s;
    if (s == nnz - 1)
      for (int32_t q = r + 1; q <= n; ++q) row_ptr[q] = nnz;
  }
}

__global__ void k_degree(const int64_t* __restrict__ row_ptr, const float* __restrict__ wmerged,
                         int32_t n, float* __restrict__ deg, float* __restrict__ val,
                         const int64_t* __restrict__ counters, const unsigned* abort) {
  if (aborted(abort)) return;
  for (int64_t r = gtid(); r < n; r += gstride()) {
    double acc = 0.0;  // sequential float64 sum in column order
    for (int64_t j = row_ptr[r]; j < row_ptr[r + 1]; ++j) {
      float x = wmerged[j];
      acc += (double)x;
      if (val) val[j] = x;
    }
    deg[r] = (float)acc;
  }
}

__global__ void k_emit_edges(const uint8_t* __restrict__ upper, const int64_t* __restrict__ eidx,
                             const int32_t* __restrict__ row_of, const int32_t* __restrict__ col,
                             const float* __restrict__ wmerged,
                             const int64_t* __restrict__ counters, int32_t* __restrict__ eu,
                             int32_t* __restrict__ ev, float* __restrict__ ew,
                             int32_t* __restrict__ csr_eid, const unsigned* abort) {
  if (aborted(abort)) return;
  const int64_t nnz = counters[0];
  for (int64_t s = gtid(); s < nnz; s += gstride()) {
    if (!upper[s]) continue;
    const int64_t e = eidx[s];
    eu[e] = row_of[s];
    ev[e] = col[s];
    if (ew) ew[e] = wmerged[s];
    csr_eid[s] = (int32_t)e;
  }
}

__global__ void k_lower_eid(const uint8_t* __restrict__ upper, const int32_t* __restrict__ row_of,
                            const int32_t* __restrict__ col, const int64_t* __restrict__ row_ptr,
                            const int64_t* __restrict__ counters, int32_t* __restrict__ csr_eid,
                            const unsigned* abort) {
  if (aborted(abort)) return;
  const int64_t nnz = counters[0];
  for (int64_t s = gtid(); s < nnz; s += gstride()) {
    if (upper[s]) continue;
    const int32_t r = row_of[s], c = col[s];  // c < r: edge (c, r) sits in row c
    int64_t lo = row_ptr[c], hi = row_ptr[c + 1] - 1;
    while (lo < hi) {
      int64_t mid = (lo + hi) >> 1;
      if (col[mid] < r)
        lo = mid + 1;
      else
        hi = mid;
    }
    csr_eid[s] = (lo < row_ptr[c + 1] && col[lo] == r) ? csr_eid[lo] : -1;
  }
}

inline int bit_length(uint32_t x) { return x ? 32 - __builtin_clz(x) : 0; }

}  // namespace
}  // namespace erc

using namespace erc;

extern "C" size_t erc_build_laplacian_workspace_size(int32_t n, int64_t m_in) {
  (void)n;
  if (m_in < 0) return 0;
  Arena a(nullptr);
  BuildPlan p;
  plan_build(a, p, m_in);
  return a.used + 256;
}

erc_status erc::build_laplacian_impl(int32_t n, const int32_t* src, const int32_t* dst,
                                     const float* w, int64_t m_in, int32_t dup_policy,
                                     int64_t* row_ptr, int32_t* col, float* val, float* deg,
                                     int32_t* csr_eid, int32_t* eu, int32_t* ev, float* ew,
                                     int64_t* m_out, void* ws, size_t ws_bytes, cudaStream_t s,
                                     int* nonunit) {
  ERC_REQUIRE(n >= 1, "n must be >= 1 (got %d)", n);
  ERC_REQUIRE(m_in >= 0 && m_in <= (int64_t(1) << 30), "m_in out of range (%lld)",
              (long long)m_in);
  ERC_REQUIRE(dup_policy == ERC_DUP_SUM || dup_policy == ERC_DUP_FIRST, "bad dup_policy %d",
              dup_policy);
  ERC_REQUIRE(row_ptr && deg && m_out, "row_ptr, deg and m_out are required");
  ERC_REQUIRE(m_in == 0 || (src && dst && col && csr_eid && eu && ev),
              "src, dst, col, csr_eid, eu, ev are required");
  ERC_REQUIRE(!(w && !val && m_in > 0), "val is required for a weighted graph");
  if (ws_bytes < erc_build_laplacian_workspace_size(n, m_in))
    return set_error(ERC_ERR_CAPACITY, "workspace too small: %zu < %zu", ws_bytes,
                     erc_build_laplacian_workspace_size(n, m_in));
  Arena a(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  BuildPlan p;
  plan_build(a, p, m_in);

  // the launch sequence is replayed from a cached CUDA graph: some twenty small kernels whose
  // launch overhead would otherwise exceed their run time
  const int64_t E = 2 * m_in;
  const int B = bit_length((uint32_t)n);  // 2^B > n - 1: every id fits, and the sentinel sorts last
  const uint64_t sent = (2 * B >= 64) ? ~0ull : ((1ull << (2 * B)) - 1ull);
  unsigned* abort = p.err + 2;
  auto enqueue = [&](cudaStream_t cs) -> erc_status {
    ERC_CUDA(cudaMemsetAsync(p.counters, 0, 4 * sizeof(int64_t), cs));
    ERC_CUDA(cudaMemsetAsync(p.err, 0, 4 * sizeof(unsigned), cs));
    ERC_CUDA(cudaMemsetAsync(row_ptr, 0, (size_t)(n + 1) * sizeof(int64_t), cs));
    if (m_in > 0) {
      k_emit<<<grid_for(m_in, BT), BT, 0, cs>>>(src, dst, w, m_in, n, B, sent, p.keys, p.vals,
                                                p.err);
      count_launches(1);
      ERC_CUDA(cudaGetLastError());
      ERC_TRY(radix_sort_pairs(p.keys, p.vals, p.keys_alt, p.vals_alt, E, 2 * B, p.sort_tmp, cs,
                               abort));
      k_heads<<<grid_for(E, BT), BT, 0, cs>>>(p.keys, E, sent, p.head, abort);
      count_launches(1);
      ERC_CUDA(cudaGetLastError());
      ERC_TRY(exclusive_scan_i64(nullptr, p.head, p.slot, E, &p.counters[0], p.scan_tmp, cs,
                                 abort));
      ERC_CUDA(cudaMemsetAsync(p.upper, 0, (size_t)E, cs));  // slots past nnz must not count
      k_emit_csr<<<grid_for(E, BT), BT, 0, cs>>>(p.keys, p.vals, p.head, p.slot, w, E, B,
                                                dup_policy == ERC_DUP_FIRST, col, p.wmerged,
                                                p.row_of, p.upper, w ? nullptr : p.err + 1,
                                                abort);
      count_launches(1);
      ERC_CUDA(cudaGetLastError());
      k_row_ptr<<<grid_for(E, BT), BT, 0, cs>>>(p.row_of, p.counters, n, row_ptr, abort);
      count_launches(1);
      ERC_CUDA(cudaGetLastError());
    }
    k_degree<<<grid_for(n, BT), BT, 0, cs>>>(row_ptr, p.wmerged, n, deg, val, p.counters, abort);
    count_launches(1);
    ERC_CUDA(cudaGetLastError());
    if (m_in > 0) {
      ERC_TRY(exclusive_scan_i64(nullptr, p.upper, p.eidx, E, &p.counters[1], p.scan_tmp, cs,
                                 abort));
      k_emit_edges<<<grid_for(E, BT), BT, 0, cs>>>(p.upper, p.eidx, p.row_of, col, p.wmerged,
                                                  p.counters, eu, ev, ew, csr_eid, abort);
      count_launches(1);
      ERC_CUDA(cudaGetLastError());
      k_lower_eid<<<grid_for(E, BT), BT, 0, cs>>>(p.upper, p.row_of, col, row_ptr, p.counters,
                                                 csr_eid, abort);
      count_launches(1);
      ERC_CUDA(cudaGetLastError());
    }
    return ERC_OK;
  };
  GraphKey key;
  key.add((uint64_t)n).add((uint64_t)m_in).add((uint64_t)dup_policy).add(src).add(dst).add(w);
  key.add(row_ptr).add(col).add(val).add(deg).add(csr_eid).add(eu).add(ev).add(ew).add(a.base);
  key.add((uint64_t)wait_limit(0));
  ERC_TRY(graph_launch(key, enqueue, s));
  int64_t h_counters[2] = {0, 0};
  unsigned h_err[3] = {0, 0, 0};
  ERC_CUDA(cudaMemcpyAsync(h_counters, p.counters, 2 * sizeof(int64_t), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaMemcpyAsync(h_err, p.err, 3 * sizeof(unsigned), cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaStreamSynchronize(s));
  if (h_err[2])
    return set_error(ERC_ERR_TIMEOUT, "a bounded wait in the Laplacian build's scans ran out; "
                                      "the outputs are undefined");
  if (h_err[0] & 1u) return set_error(ERC_ERR_INVALID_ARG, "node id outside [0, %d)", n);
  if (h_err[0] & 2u) return set_error(ERC_ERR_INVALID_ARG, "edge weight not finite and positive");
  if (h_counters[0] != 2 * h_counters[1])
    return set_error(ERC_ERR_CUDA, "internal: nnz %lld != 2 m %lld", (long long)h_counters[0],
                     (long long)h_counters[1]);
  *m_out = h_counters[1];
  if (nonunit) *nonunit = w ? 1 : (int)h_err[1];
  return ERC_OK;
}

extern "C" erc_status erc_build_laplacian(int32_t n, const int32_t* src, const int32_t* dst,
                                          const float* w, int64_t m_in, int32_t dup_policy,
                                          int64_t* row_ptr, int32_t* col, float* val, float* deg,
                                          int32_t* csr_eid, int32_t* eu, int32_t* ev, float* ew,
                                          int64_t* m_out, void* ws, size_t ws_bytes,
                                          erc_stream stream) {
  clear_error();
  return build_laplacian_impl(n, src, dst, w, m_in, dup_policy, row_ptr, col, val, deg, csr_eid,
                              eu, ev, ew, m_out, ws, ws_bytes, as_stream(stream), nullptr);
}

extern "C" erc_status erc_build_laplacian_ex(int32_t n, const int32_t* src, const int32_t* dst,
                                             const float* w, int64_t m_in, int32_t dup_policy,
                                             int64_t* row_ptr, int32_t* col, float* val,
                                             float* deg, int32_t* csr_eid, int32_t* eu,
                                             int32_t* ev, float* ew, int64_t* m_out,
                                             int32_t* unit_weights, void* ws, size_t ws_bytes,
                                             erc_stream stream) {
  clear_error();
  ERC_REQUIRE(unit_weights, "unit_weights is required");
  int nonunit = 1;
  ERC_TRY(build_laplacian_impl(n, src, dst, w, m_in, dup_policy, row_ptr, col, val, deg, csr_eid,
                               eu, ev, ew, m_out, ws, ws_bytes, as_stream(stream), &nonunit));
  *unit_weights = nonunit ? 0 : 1;
  return ERC_OK;
}
