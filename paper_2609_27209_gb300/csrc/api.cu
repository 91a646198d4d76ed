// api.cu -- error reporting, graph checks and the whole-path drivers erc_run / erc_run_host
// (Algorithm 1 followed by §3.2), which stream the K projection columns in batches of kc so the
// n x K embedding is never held.
#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "erc_internal.cuh"

namespace erc {

namespace {
thread_local char g_err[512] = "";
thread_local bool g_capturing = false;
thread_local long long g_captured = 0;  // kernels recorded into the graph being captured
std::atomic<unsigned long long> g_launches{0};
std::atomic<unsigned> g_wait_limit{0};  // 0: every bounded wait keeps its own default
}

unsigned wait_limit(unsigned dflt) {
  const unsigned v = g_wait_limit.load(std::memory_order_relaxed);
  return v ? v : dflt;
}

void count_launches(long long k) {
  if (g_capturing)
    g_captured += k;
  else
    g_launches.fetch_add((unsigned long long)k, std::memory_order_relaxed);
}
void set_capturing(bool on) {
  g_capturing = on;
  if (on) g_captured = 0;
}

// ---- cached launch sequences (see GraphKey)
namespace {
struct CachedGraph {
  GraphKey key;
  cudaGraphExec_t exec = nullptr;
  long long kernels = 0;
  unsigned long long stamp = 0;
};
constexpr int GRAPHS = 32;
std::mutex g_graph_mu;
CachedGraph g_graphs[GRAPHS];
unsigned long long g_graph_clock = 0;

bool same_key(const GraphKey& a, const GraphKey& b) {
  if (a.n != b.n) return false;
  for (int i = 0; i < a.n; ++i)
    if (a.w[i] != b.w[i]) return false;
  return true;
}

cudaStream_t private_stream() {
  static thread_local cudaStream_t cs[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  if (!cs[dev] && cudaStreamCreateWithFlags(&cs[dev], cudaStreamNonBlocking) != cudaSuccess)
    return nullptr;
  return cs[dev];
}
}  // namespace

erc_status graph_launch_impl(const GraphKey& key_in, erc_status (*enqueue)(void*, cudaStream_t),
                             void* ctx, cudaStream_t s) {
  GraphKey key = key_in;
  int dev = 0;
  ERC_CUDA(cudaGetDevice(&dev));
  key.add((uint64_t)dev);
  std::lock_guard<std::mutex> lock(g_graph_mu);
  ++g_graph_clock;
  int victim = 0;
  for (int i = 0; i < GRAPHS; ++i) {
    if (g_graphs[i].exec && same_key(g_graphs[i].key, key)) {
      g_graphs[i].stamp = g_graph_clock;
      ERC_CUDA(cudaGraphLaunch(g_graphs[i].exec, s));
      count_launches(g_graphs[i].kernels);
      return ERC_OK;
    }
    if (g_graphs[i].stamp < g_graphs[victim].stamp) victim = i;
  }
  cudaStream_t cs = private_stream();
  if (!cs) return set_error(ERC_ERR_CUDA, "no capture stream");
  ERC_CUDA(cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal));
  set_capturing(true);
  const erc_status st = enqueue(ctx, cs);
  const long long kernels = g_captured;
  set_capturing(false);
  cudaGraph_t graph = nullptr;
  const cudaError_t ce = cudaStreamEndCapture(cs, &graph);
  if (st != ERC_OK) {
    if (graph) cudaGraphDestroy(graph);
    return st;
  }
  if (ce != cudaSuccess) return set_error(ERC_ERR_CUDA, "graph capture: %s", cudaGetErrorString(ce));
  cudaGraphExec_t exec = nullptr;
  const cudaError_t ie = cudaGraphInstantiate(&exec, graph, 0);
  cudaGraphDestroy(graph);
  if (ie != cudaSuccess)
    return set_error(ERC_ERR_CUDA, "graph instantiate: %s", cudaGetErrorString(ie));
  if (g_graphs[victim].exec) cudaGraphExecDestroy(g_graphs[victim].exec);
  g_graphs[victim].key = key;
  g_graphs[victim].exec = exec;
  g_graphs[victim].kernels = kernels;
  g_graphs[victim].stamp = g_graph_clock;
  ERC_CUDA(cudaGraphLaunch(exec, s));
  count_launches(kernels);
  return ERC_OK;
}

erc_status set_error(erc_status code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof g_err, fmt, ap);
  va_end(ap);
  return code;
}

void clear_error() { g_err[0] = '\0'; }

int sm_count() {
  static int cache[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  if (!cache[dev]) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v < 1)
      v = 148;
    cache[dev] = v;
  }
  return cache[dev];
}

int resident_per_sm(const void* kernel, int threads, size_t smem) {
  struct Entry {
    const void* k;
    int threads, dev, blocks;
    size_t smem;
  };
  static std::mutex mu;
  static Entry cache[256];
  static int used = 0;
  int dev = 0;
  cudaGetDevice(&dev);
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used; ++i)
    if (cache[i].k == kernel && cache[i].threads == threads && cache[i].dev == dev &&
        cache[i].smem == smem)
      return cache[i].blocks;
  int nb = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kernel, threads, smem) != cudaSuccess ||
      nb < 1)
    nb = 1;
  if (used < 256) cache[used++] = Entry{kernel, threads, dev, nb, smem};
  return nb;
}

erc_status check_graph(const erc_graph* g) {
  ERC_REQUIRE(g, "graph is null");
  ERC_REQUIRE(g->n >= 1, "graph has n < 1");
  ERC_REQUIRE(g->m >= 0 && g->m < (int64_t(1) << 31), "graph m out of range");
  ERC_REQUIRE(g->row_ptr, "graph row_ptr is null");
  ERC_REQUIRE(g->m == 0 || (g->col && g->csr_eid && g->eu && g->ev), "graph arrays are null");
  return ERC_OK;
}

namespace {

struct RunPlan {
  int64_t* row_ptr;
  int32_t *col, *csr_eid;
  float *val, *deg, *ew;
  float *Y, *X;
  void* cg_ws;
  size_t cg_bytes;
  void* aux_ws;  // build workspace, later the sampling workspace
  size_t aux_bytes;
};

inline int32_t ld_for(int32_t kc) { return (kc + 3) & ~3; }

void plan_run(Arena& a, RunPlan& p, int32_t n, int64_t m_in, int32_t kc) {
  const int32_t ld = ld_for(kc);
  p.row_ptr = a.take<int64_t>((size_t)n + 1);
  p.col = a.take<int32_t>(2 * m_in);
  p.csr_eid = a.take<int32_t>(2 * m_in);
  p.val = a.take<float>(2 * m_in);
  p.deg = a.take<float>(n);
  p.ew = a.take<float>(m_in);
  p.Y = a.take<float>((size_t)n * ld);
  p.X = a.take<float>((size_t)n * ld);
  p.cg_bytes = erc_batched_cg_workspace_size(n, ld);
  p.cg_ws = a.take<char>(p.cg_bytes);
  const size_t b1 = erc_build_laplacian_workspace_size(n, m_in);
  const size_t b2 = erc_sampling_probs_workspace_size(n, m_in);
  p.aux_bytes = b1 > b2 ? b1 : b2;
  p.aux_ws = a.take<char>(p.aux_bytes);
}

erc_status run_device(const erc_params* prm, int32_t n, const int32_t* src, const int32_t* dst,
                      const float* w, int64_t m_in, int64_t* m_out, int32_t* eu, int32_t* ev,
                      float* R, float* p_node, float* kappa, float* prob_node, float* prob_edge,
                      int32_t* iters, float* relres, const RunPlan& p, cudaStream_t s,
                      bool read_status = true) {
  const int32_t ld = ld_for(prm->kc);
  int64_t m = 0;
  // the build also reports whether an unweighted input kept unit weights (no merged duplicates):
  // then the weight arrays are dropped and the gathers read indices only
  int nonunit = 1;
  ERC_TRY(build_laplacian_impl(n, src, dst, w, m_in, prm->dup_policy, p.row_ptr, p.col, p.val,
                               p.deg, p.csr_eid, eu, ev, p.ew, &m, p.aux_ws, p.aux_bytes, s,
                               &nonunit));
  *m_out = m;
  erc_graph g{n, m, p.row_ptr, p.col, nonunit ? p.val : nullptr, p.deg, p.csr_eid,
              eu, ev, nonunit ? p.ew : nullptr};
  if (m > 0) ERC_CUDA(cudaMemsetAsync(R, 0, (size_t)m * sizeof(float), s));
  // every batch is enqueued without a host round trip (the single-launch solvers need none); the
  // CG status of all batches is read once at the end
  for (int32_t c0 = 0; c0 < prm->K; c0 += prm->kc) {
    const int32_t k = prm->kc < prm->K - c0 ? prm->kc : prm->K - c0;
    ERC_TRY(erc_jl_rhs(&g, prm->seed, prm->K, c0, k, p.Y, ld, reinterpret_cast<erc_stream>(s)));
    ERC_TRY(cg_enqueue(&g, prm->eps, p.Y, p.X, ld, k, prm->tol, prm->max_iter, iters + c0,
                       relres + c0, p.cg_ws, p.cg_bytes, s, c0 == 0, nullptr, nullptr, nullptr,
                       prm->precond == ERC_PRECOND_JACOBI));
    ERC_TRY(erc_edge_resistance(&g, p.X, ld, k, R, reinterpret_cast<erc_stream>(s)));
  }
  ERC_TRY(erc_curvature(&g, R, p_node, kappa, reinterpret_cast<erc_stream>(s)));
  ERC_TRY(erc_sampling_probs(&g, kappa, prm->eta, prob_node, prob_edge, p.aux_ws, p.aux_bytes,
                             reinterpret_cast<erc_stream>(s)));
  return read_status ? cg_status(n, ld, prm->K, prm->max_iter, p.cg_ws, s) : ERC_OK;
}

erc_status check_params(const erc_params* prm, int32_t n, int64_t m_in) {
  ERC_REQUIRE(prm, "params is null");
  ERC_REQUIRE(prm->K >= 1, "K must be >= 1");
  ERC_REQUIRE(prm->kc >= 1 && prm->kc <= MAX_LD, "kc must be in [1, %d]", MAX_LD);
  ERC_REQUIRE(prm->kc % 4 == 0 || prm->kc >= prm->K, "kc must be a multiple of 4 when K > kc");
  ERC_REQUIRE(n >= 1 && m_in >= 0, "bad n / m_in");
  ERC_REQUIRE(prm->precond == ERC_PRECOND_NONE || prm->precond == ERC_PRECOND_JACOBI,
              "precond must be ERC_PRECOND_NONE or ERC_PRECOND_JACOBI");
  return ERC_OK;
}

}  // namespace
}  // namespace erc

using namespace erc;

extern "C" const char* erc_version(void) { return "erc-gb300 0.1 (sm_103a)"; }
extern "C" const char* erc_last_error(void) { return g_err; }
extern "C" uint64_t erc_kernel_launches(void) { return g_launches.load(); }
extern "C" void erc_set_wait_limit(uint32_t polls) {
  g_wait_limit.store(polls, std::memory_order_relaxed);
}

extern "C" size_t erc_run_workspace_size(int32_t n, int64_t m_in, int32_t kc) {
  if (n < 1 || m_in < 0 || kc < 1) return 0;
  Arena a(nullptr);
  RunPlan p;
  plan_run(a, p, n, m_in, kc);
  return a.used + 256;
}

extern "C" erc_status erc_run(const erc_params* prm, int32_t n, const int32_t* src,
                              const int32_t* dst, const float* w, int64_t m_in, int64_t* m_out,
                              int32_t* eu, int32_t* ev, float* R, float* p_node, float* kappa,
                              float* prob_node, float* prob_edge, int32_t* iters, float* relres,
                              void* ws, size_t ws_bytes, erc_stream stream) {
  clear_error();
  ERC_TRY(check_params(prm, n, m_in));
  ERC_REQUIRE(m_out && eu && ev && R && p_node && kappa && prob_node && prob_edge && iters &&
                  relres,
              "output pointers are required");
  if (ws_bytes < erc_run_workspace_size(n, m_in, prm->kc))
    return set_error(ERC_ERR_CAPACITY, "workspace too small");
  Arena a(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  RunPlan p;
  plan_run(a, p, n, m_in, prm->kc);
  return run_device(prm, n, src, dst, w, m_in, m_out, eu, ev, R, p_node, kappa, prob_node,
                    prob_edge, iters, relres, p, as_stream(stream));
}

namespace {
struct HostIo {
  int32_t *src, *dst;
  float* w;
  int32_t *eu, *ev;
  float *R, *p, *kappa, *pn, *pe, *relres;
  int32_t* iters;
};
void plan_host_io(Arena& a, HostIo& h, int32_t n, int64_t m_in, int32_t K) {
  h.src = a.take<int32_t>(m_in);
  h.dst = a.take<int32_t>(m_in);
  h.w = a.take<float>(m_in);
  h.eu = a.take<int32_t>(m_in);
  h.ev = a.take<int32_t>(m_in);
  h.R = a.take<float>(m_in);
  h.kappa = a.take<float>(m_in);
  h.pe = a.take<float>(m_in);
  h.p = a.take<float>(n);
  h.pn = a.take<float>(n);
  h.iters = a.take<int32_t>(K);
  h.relres = a.take<float>(K);
}
}  // namespace

extern "C" size_t erc_run_host_workspace_size(int32_t n, int64_t m_in, int32_t kc, int32_t K) {
  if (n < 1 || m_in < 0 || kc < 1 || K < 1) return 0;
  Arena a(nullptr);
  HostIo h;
  plan_host_io(a, h, n, m_in, K);
  RunPlan p;
  plan_run(a, p, n, m_in, kc);
  return a.used + 256;
}

extern "C" erc_status erc_run_host(const erc_params* prm, int32_t n, const int32_t* src,
                                   const int32_t* dst, const float* w, int64_t m_in,
                                   int64_t* m_out, int32_t* eu, int32_t* ev, float* R,
                                   float* p_node, float* kappa, float* prob_node,
                                   float* prob_edge, int32_t* iters, float* relres, void* ws,
                                   size_t ws_bytes, erc_stream stream) {
  clear_error();
  ERC_TRY(check_params(prm, n, m_in));
  ERC_REQUIRE(m_in == 0 || (src && dst), "src and dst are required");
  ERC_REQUIRE(m_out && eu && ev && R && p_node && kappa && prob_node && prob_edge && iters &&
                  relres,
              "output pointers are required");
  if (ws_bytes < erc_run_host_workspace_size(n, m_in, prm->kc, prm->K))
    return set_error(ERC_ERR_CAPACITY, "workspace too small");
  cudaStream_t s = as_stream(stream);
  Arena a(reinterpret_cast<void*>((reinterpret_cast<uintptr_t>(ws) + 255) & ~uintptr_t(255)));
  HostIo d;
  plan_host_io(a, d, n, m_in, prm->K);
  RunPlan p;
  plan_run(a, p, n, m_in, prm->kc);
  const size_t mi4 = (size_t)m_in * 4;
  if (m_in > 0) {
    ERC_CUDA(cudaMemcpyAsync(d.src, src, mi4, cudaMemcpyHostToDevice, s));
    ERC_CUDA(cudaMemcpyAsync(d.dst, dst, mi4, cudaMemcpyHostToDevice, s));
    if (w) ERC_CUDA(cudaMemcpyAsync(d.w, w, mi4, cudaMemcpyHostToDevice, s));
  }
  // the CG status is read after the output copies are enqueued: its readback is the call's one
  // synchronisation after the build
  ERC_TRY(run_device(prm, n, d.src, d.dst, w ? d.w : nullptr, m_in, m_out, d.eu, d.ev, d.R, d.p,
                     d.kappa, d.pn, d.pe, d.iters, d.relres, p, s, false));
  const size_t m4 = (size_t)(*m_out) * 4, n4 = (size_t)n * 4, k4 = (size_t)prm->K * 4;
  if (m4) {
    ERC_CUDA(cudaMemcpyAsync(eu, d.eu, m4, cudaMemcpyDeviceToHost, s));
    ERC_CUDA(cudaMemcpyAsync(ev, d.ev, m4, cudaMemcpyDeviceToHost, s));
    ERC_CUDA(cudaMemcpyAsync(R, d.R, m4, cudaMemcpyDeviceToHost, s));
    ERC_CUDA(cudaMemcpyAsync(kappa, d.kappa, m4, cudaMemcpyDeviceToHost, s));
    ERC_CUDA(cudaMemcpyAsync(prob_edge, d.pe, m4, cudaMemcpyDeviceToHost, s));
  }
  ERC_CUDA(cudaMemcpyAsync(p_node, d.p, n4, cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaMemcpyAsync(prob_node, d.pn, n4, cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaMemcpyAsync(iters, d.iters, k4, cudaMemcpyDeviceToHost, s));
  ERC_CUDA(cudaMemcpyAsync(relres, d.relres, k4, cudaMemcpyDeviceToHost, s));
  return cg_status(n, ld_for(prm->kc), prm->K, prm->max_iter, p.cg_ws, s);
}
