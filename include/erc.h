/*
 * erc.h -- C ABI of liberc.so: ERC-LG (effective-resistance curvature of every edge of a large graph)
 * on one NVIDIA GB300 GPU (sm_103a).
 *
 * Method: "Scalable Subgraph Sampling via Resistance Curvature" (arxiv 2609.27209), §3.
 *   L = D - A = B^T W B (§3.1.1); Y = B^T W^{1/2} Q with Q_ec uniform on {+-1/sqrt(K)} (§3.1.2);
 *   column-wise CG on L_eps Z = Y, L_eps = L + eps I (Eq. 5, §3.1.3, Algorithm 1);
 *   R_uv = ||Z_u - Z_v||^2 accumulated over column batches (Eq. 6, Algorithm 1);
 *   p_u = 1 - 1/2 sum_v w_uv R_uv, kappa_uv = 2 (p_u + p_v) / R_uv (Eq. 2);
 *   node / edge sampling probabilities (Eq. 7, Eq. 8, §3.2).
 *
 * Conventions for every call
 *   - Returns an erc_status; erc_last_error() gives a message for the last failure on the calling
 *     host thread.
 *   - Array arguments are DEVICE pointers owned by the caller unless marked "host".  The library
 *     never frees or keeps caller memory and performs no device allocation: scratch space comes
 *     from the caller through the matching *_workspace_size() query (16-byte alignment or better;
 *     the library aligns sub-buffers itself).
 *   - Work is ordered on the caller's stream `s` (a cudaStream_t; NULL = legacy default stream)
 *     and is asynchronous, except where a host-visible result is returned (m_out, the CG status):
 *     those calls synchronise `s` before returning.
 *   - Node ids are int32 in [0, n); CSR offsets are int64.  Column blocks (Y, X) are row-major
 *     n x ld float32 with ld >= kc, ld a multiple of 4 and the base 16-byte aligned; only the
 *     first kc columns of a row carry data.
 *   - Precision: float32 storage and arithmetic; dot products and per-column CG scalars are
 *     accumulated in a float32 pair (about 44 significant bits) and finished in float64.
 */
#ifndef ERC_H
#define ERC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef void* erc_stream; /* cudaStream_t */

typedef enum erc_status {
  ERC_OK = 0,
  ERC_ERR_INVALID_ARG = 1,   /* bad size, pointer, alignment, node id or weight */
  ERC_ERR_CUDA = 2,          /* a CUDA runtime call failed (message has the CUDA error) */
  ERC_ERR_CAPACITY = 3,      /* workspace too small, or a size beyond the library's limits */
  ERC_ERR_NOT_CONVERGED = 4, /* some CG column reached max_iter; results are still written */
  ERC_ERR_NUMERIC = 5,       /* a non-finite or non-positive CG scalar was met */
  ERC_ERR_TIMEOUT = 6        /* a bounded device-side wait ran out */
} erc_status;

enum { ERC_DUP_SUM = 0, ERC_DUP_FIRST = 1 };
/* CG preconditioner: none (the paper's plain CG, the default) or Jacobi, M = diag(L_eps) */
enum { ERC_PRECOND_NONE = 0, ERC_PRECOND_JACOBI = 1 };

/* Non-owning view of a graph built by erc_build_laplacian (all pointers device, read-only). */
typedef struct erc_graph {
  int32_t n;              /* nodes */
  int64_t m;              /* undirected edges; the CSR holds 2m slots */
  const int64_t* row_ptr; /* [n+1] CSR offsets of the symmetric adjacency A */
  const int32_t* col;     /* [2m] neighbour ids, strictly ascending within a row */
  const float* val;       /* [2m] edge weights w_uv, or NULL when every weight is 1 */
  const float* deg;       /* [n] weighted degree sum_v w_uv (float64 sum, rounded once) */
  const int32_t* csr_eid; /* [2m] canonical edge id of each CSR slot */
  const int32_t* eu;      /* [m] canonical edges: eu[e] < ev[e], lexicographic order */
  const int32_t* ev;      /* [m] */
  const float* ew;        /* [m] weight of edge e, or NULL when every weight is 1 */
} erc_graph;

/* Parameters of a whole ERC-LG run (Algorithm 1 + §3.2). */
typedef struct erc_params {
  uint64_t seed;      /* Philox key of Q */
  int32_t K;          /* projection dimension (§3.1.2) */
  int32_t kc;         /* columns per streamed batch ("b" in Algorithm 1), 1..1024 */
  float eps;          /* regularisation eps > 0 (Eq. 5) */
  float tol;          /* CG relative residual tolerance tau (Algorithm 1) */
  int32_t max_iter;   /* CG iteration cap per column */
  float eta;          /* eta > 0 of Eq. 7 */
  int32_t dup_policy; /* ERC_DUP_SUM or ERC_DUP_FIRST */
  int32_t precond;    /* ERC_PRECOND_NONE (Algorithm 1's plain CG) or ERC_PRECOND_JACOBI */
} erc_params;

const char* erc_version(void);
const char* erc_last_error(void);
/* Number of CUDA kernels this library has launched in this process so far (a CUDA-graph launch
 * counts the kernels it contains).  For instrumentation only. */
uint64_t erc_kernel_launches(void);

/* erc_set_wait_limit -- failure detection (no counterpart in the paper).  Every device-side wait
 * of the library on work of other thread blocks of the same launch is bounded: the look-back of
 * the single-pass scans (Laplacian build, subgraph sampler), the grid barrier of the CG vector
 * update and the grid synchronisations of the resident CG solver.  A wait that runs out of polls
 * records it in the call's device status and returns; the kernels after it in the same call do
 * no further work on the unfinished result, and the call returns ERC_ERR_TIMEOUT once it reads
 * its status (the outputs are then undefined).  `polls` sets the number of polls every such
 * wait makes before it gives up, for all later calls of the process; 0 (the initial state)
 * restores each wait's default, which is seconds of waiting.  Waits of work already enqueued keep
 * the limit they were enqueued with.  The hardware cluster barriers of the cluster CG solver are
 * not polled and take no limit. */
void erc_set_wait_limit(uint32_t polls);

/* ---------------------------------------------------------------------------------------------
 * erc_build_laplacian -- the simple undirected graph behind L = D - A = B^T W B (§3.1.1).
 *
 * In : n nodes; src, dst [m_in] int32 endpoints (any order/orientation); w [m_in] float32 weights
 *      (> 0, finite) or NULL for unit weights; dup_policy: repeated (u,v) pairs (either
 *      orientation) are merged by summing their weights in float64 in input order and rounding
 *      once (ERC_DUP_SUM) or by keeping the first weight (ERC_DUP_FIRST).  Self-loops are dropped
 *      (they contribute nothing to B^T W B).
 * Out: row_ptr [n+1], col [2 m_in], val [2 m_in] (may be NULL only when w is NULL), deg [n],
 *      csr_eid [2 m_in], eu, ev [m_in], ew [m_in] (may be NULL); capacities in brackets, the first
 *      2m / m entries are written; m_out (host) receives m.  Edge ids e = 0..m-1 number the
 *      canonical pairs (eu < ev) in lexicographic order.  Deterministic (bit-identical reruns).
 * Errors: INVALID_ARG for n < 1, m_in < 0 or > 2^30, an id outside [0, n), a weight <= 0 or
 *      non-finite; CAPACITY if ws_bytes < erc_build_laplacian_workspace_size(n, m_in).
 * Synchronises s.
 * ------------------------------------------------------------------------------------------- */
size_t erc_build_laplacian_workspace_size(int32_t n, int64_t m_in);
erc_status erc_build_laplacian(int32_t n, const int32_t* src, const int32_t* dst, const float* w,
                               int64_t m_in, int32_t dup_policy, int64_t* row_ptr, int32_t* col,
                               float* val, float* deg, int32_t* csr_eid, int32_t* eu, int32_t* ev,
                               float* ew, int64_t* m_out, void* ws, size_t ws_bytes, erc_stream s);
/* erc_build_laplacian_ex -- erc_build_laplacian, plus *unit_weights (host) = 1 when w is NULL and
 * no merged duplicate pair received a weight other than 1, else 0.  When it is 1 every weight of
 * the graph is 1: an erc_graph may then carry val = ew = NULL, and the kernels read neighbour
 * indices only.  The flag comes back with m_out in the same synchronisation. */
erc_status erc_build_laplacian_ex(int32_t n, const int32_t* src, const int32_t* dst,
                                  const float* w, int64_t m_in, int32_t dup_policy,
                                  int64_t* row_ptr, int32_t* col, float* val, float* deg,
                                  int32_t* csr_eid, int32_t* eu, int32_t* ev, float* ew,
                                  int64_t* m_out, int32_t* unit_weights, void* ws,
                                  size_t ws_bytes, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_jl_rhs -- Y[:, 0:kc] = (B^T W^{1/2} Q)[:, c0:c0+kc]  (§3.1.2; Algorithm 1 "form Y").
 *
 * Row e of B is e_u - e_v for the canonical edge (u = eu[e] < v = ev[e]).  Q is never stored: its
 * entry (e, c) is +1/sqrt(K) when a Philox4x32-10 bit is 0 and -1/sqrt(K) when it is 1, the bit
 * being bit (c mod 32) of word ((c div 32) mod 4) of Philox4x32-10 with key (seed lo, seed hi) and
 * counter (c div 128, 0, e lo, e hi).  K is the total projection dimension, so a column's values
 * do not depend on the batch it is produced in.  Requires c0 % 4 == 0, 0 < kc, c0 + kc <= K.
 * Row u is summed in CSR order (deterministic).  Columns kc..ld-1 are set to 0.
 * ------------------------------------------------------------------------------------------- */
erc_status erc_jl_rhs(const erc_graph* g, uint64_t seed, int32_t K, int32_t c0, int32_t kc,
                      float* Y, int32_t ld, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_batched_cg -- solve L_eps X = Y column by column with CG (Eq. 5, §3.1.3, Algorithm 1).
 *
 * Every column c < kc runs Hestenes-Stiefel CG from x = 0 independently of the others and stops
 * once its recursively updated residual satisfies ||r||_2 <= tol ||y||_2, or after max_iter
 * iterations.  L_eps p is applied as eps p_u + sum_v w_uv (p_u - p_v).
 * Out: X [n x ld] (columns kc..ld-1 set to 0); iters [kc] int32 (device) iterations per column;
 *      relres [kc] float (device) true relative residual ||y - L_eps x|| / ||y|| of the returned x.
 * Errors: NOT_CONVERGED if any column stopped at max_iter; NUMERIC if p^T L_eps p <= 0 or a
 *      non-finite scalar appeared (that column is frozen); CAPACITY if ws is too small.
 * Synchronises s (it reads the convergence status).
 * ------------------------------------------------------------------------------------------- */
size_t erc_batched_cg_workspace_size(int32_t n, int32_t ld);
erc_status erc_batched_cg(const erc_graph* g, float eps, const float* Y, float* X, int32_t ld,
                          int32_t kc, float tol, int32_t max_iter, int32_t* iters, float* relres,
                          void* ws, size_t ws_bytes, erc_stream s);

/* erc_batched_cg_timed -- benchmarking helper: erc_batched_cg, plus *solve_us (host) = the time
 * between CUDA events recorded on `s` around the solver kernels (the final residual excluded)
 * and *path (host), the solver that ran:
 *   2  one launch of thread-block clusters, each solving a group of 16 columns over all rows
 *      (graphs whose rows' r and Ap slices fit in the shared memory of a cluster, when a cost
 *      model favours it over 1: small graphs); the launch also initialises r, p and x;
 *   1  one cooperative launch over all rows and columns (r and Ap blocks in the SMs' shared
 *      memory); the launch also initialises r, p and x and forms the true residual;
 *   0  the multi-kernel loop captured in CUDA graphs (larger graphs).
 * The environment variable ERC_CG_MODE=cluster|resident|graph restricts the choice. */
erc_status erc_batched_cg_timed(const erc_graph* g, float eps, const float* Y, float* X,
                                int32_t ld, int32_t kc, float tol, int32_t max_iter,
                                int32_t* iters, float* relres, void* ws, size_t ws_bytes,
                                float* solve_us, int32_t* path, erc_stream s);

/* erc_batched_pcg, erc_batched_pcg_timed -- an optional solver variant, not part of the paper's
 * method: erc_batched_cg with the Jacobi preconditioner M = diag(L_eps) = deg + eps (g->deg
 * required), i.e. preconditioned CG (Y. Saad, "Iterative Methods for Sparse Linear Systems",
 * Algorithm 9.1) with z = r / (deg + eps), p0 = z0, alpha = r.z / p.Ap, beta = r'.z' / r.z.
 * Same arguments, workspace (erc_batched_cg_workspace_size), start (x = 0), stop test (on the
 * unpreconditioned ||r||_2 <= tol ||y||_2), outputs and errors as erc_batched_cg.  It solves
 * the same systems to the same tolerance in fewer iterations where degrees vary widely
 * (power-law graphs).  Paths 1 and 0 only (no cluster solver). */
erc_status erc_batched_pcg(const erc_graph* g, float eps, const float* Y, float* X, int32_t ld,
                           int32_t kc, float tol, int32_t max_iter, int32_t* iters, float* relres,
                           void* ws, size_t ws_bytes, erc_stream s);
erc_status erc_batched_pcg_timed(const erc_graph* g, float eps, const float* Y, float* X,
                                 int32_t ld, int32_t kc, float tol, int32_t max_iter,
                                 int32_t* iters, float* relres, void* ws, size_t ws_bytes,
                                 float* solve_us, int32_t* path, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_edge_resistance -- R_acc[e] += sum_{c < kc} (X[eu[e], c] - X[ev[e], c])^2   (Eq. 6).
 *
 * Called once per column batch on the batch's solution, so R_acc (float32 [m], zeroed by the
 * caller before the first batch) ends as the JL estimate over all K columns without the n x K
 * embedding ever being held (Algorithm 1's streamed accumulation).
 * ------------------------------------------------------------------------------------------- */
erc_status erc_edge_resistance(const erc_graph* g, const float* X, int32_t ld, int32_t kc,
                               float* R_acc, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_curvature -- Eq. 2: p_u = 1 - 1/2 sum_{v in N(u)} w_uv R_uv (float64 row sums),
 *                  kappa_e = 2 (p_u + p_v) / R_e for e = (u, v).
 * In: R [m].  Out: p_node [n], kappa [m].  R_e = 0 gives an IEEE infinity / NaN.
 * ------------------------------------------------------------------------------------------- */
erc_status erc_curvature(const erc_graph* g, const float* R, float* p_node, float* kappa,
                         erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_sampling_probs -- §3.2.
 *   node: q_u = sum_{v in N(u)} (kappa_uv - kappa_min) / (kappa_max - kappa_min + eta)  (Eq. 7);
 *         prob_node = q / sum q, or, when every q_u is 0, uniform over the nodes with an edge.
 *   edge: q_e = sqrt(max(-kappa_e + 2 kappa_max, 0)) + 1 (Eq. 8); prob_edge = q / sum q over the
 *         m canonical edges.
 * Out: prob_node [n], prob_edge [m].  Sums are float64 in a fixed order (deterministic).
 * ------------------------------------------------------------------------------------------- */
size_t erc_sampling_probs_workspace_size(int32_t n, int64_t m);
erc_status erc_sampling_probs(const erc_graph* g, const float* kappa, float eta, float* prob_node,
                              float* prob_edge, void* ws, size_t ws_bytes, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_sampling_probs_noalloc -- erc_sampling_probs with no caller workspace and no allocation.
 *
 * The paper has no counterpart; this is a library convenience.  It serves callers that cannot
 * allocate device memory themselves: plug-ins whose host application owns every device buffer,
 * code that must not call cudaMalloc / cudaFree because those calls can synchronise the whole
 * device, and processes held to a fixed device-memory budget.  Inputs and outputs are as for
 * erc_sampling_probs; the scratch is a file-scope device array of
 * ERC_SAMPLING_PROBS_NOALLOC_SCRATCH_BYTES inside liberc.so, present on every device that loads
 * the library and held until the process exits.  The call allocates nothing.
 * Limits: g->n <= ERC_SAMPLING_PROBS_NOALLOC_MAX_NODES, else ERC_ERR_CAPACITY (nothing is run).
 * The first call on each device looks up the array's device address (cudaGetSymbolAddress) with
 * that device current, and so does the first call after the device's context was destroyed and
 * created again (cudaDeviceReset): make those calls before any stream capture.  All calls share the one
 * array and it keeps the last call's contents (a call never relies on them): calls that may
 * overlap on the GPU -- concurrent streams, or several host threads -- race with each other and
 * must be serialised by the caller.
 * ------------------------------------------------------------------------------------------- */
#define ERC_SAMPLING_PROBS_NOALLOC_MAX_NODES 4000000
#define ERC_SAMPLING_PROBS_NOALLOC_SCRATCH_BYTES (32u << 20)
erc_status erc_sampling_probs_noalloc(const erc_graph* g, const float* kappa, float eta,
                                      float* prob_node, float* prob_edge, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_sample_subgraph -- one curvature-guided subgraph (§3.2: sampling proportional to the node
 * weights of Eq. 7 or the edge weights of Eq. 8; the paper's ERC-LG-sub(node) / (edge) samplers
 * follow GraphSAINT).
 *
 * kind ERC_SAMPLE_NODES: `budget` draws with replacement over the n nodes with probabilities
 *   prob [n] (prob_node of erc_sampling_probs); the subgraph is induced on the distinct drawn
 *   nodes.
 * kind ERC_SAMPLE_EDGES: `budget` draws over the m canonical edges with prob [m] (prob_edge); the
 *   nodes are the drawn edges' endpoints and the edges are the subgraph induced on them
 *   (induced != 0, GraphSAINT) or the distinct drawn edges (induced == 0).
 * A draw is exact: weights W_i = round(prob_i * 2^40) (prob_i must lie in [0, 1]; entries below
 *   2^-41 are never drawn), draw k takes x = (word0 << 32) | word1 of Philox4x32-10 with key
 *   (seed lo, seed hi) and counter (k lo, k hi, 0x53414D50, kind), and picks the smallest i with
 *   W_0 + .. + W_i > floor(x * sum(W) / 2^64).  Draws k = first_draw .. first_draw + budget - 1,
 *   so consecutive calls with advancing first_draw continue one random stream.
 * Out: nodes [capacity n] ascending distinct node ids, *n_out (host); edges [capacity m]
 *   ascending canonical edge ids, *m_out (host).  Deterministic.
 * Errors: INVALID_ARG for a probability outside [0, 1] or all weights rounding to zero;
 *   CAPACITY if ws_bytes < erc_sample_workspace_size(n, m, budget).  Synchronises s.
 * ------------------------------------------------------------------------------------------- */
enum { ERC_SAMPLE_NODES = 0, ERC_SAMPLE_EDGES = 1 };
size_t erc_sample_workspace_size(int32_t n, int64_t m, int64_t budget);
erc_status erc_sample_subgraph(const erc_graph* g, int32_t kind, const float* prob,
                               int64_t budget, uint64_t seed, int64_t first_draw, int32_t induced,
                               int32_t* nodes, int32_t* n_out, int32_t* edges, int64_t* m_out,
                               void* ws, size_t ws_bytes, erc_stream s);

/* erc_saint_counts -- GraphSAINT's pre-sampling counts: node_count[v] += 1 for each of the n_s
 * distinct ids in nodes, edge_count[e] += 1 for each of the m_s distinct ids in edges (device
 * int32 arrays [n] and [m], accumulated over calls; the caller zeroes them first).
 * erc_saint_norm -- from counts over N subgraphs: lambda[v] = node_count[v] / N (loss
 * normalisation, [n]) and, for CSR slot j of row v holding edge e, alpha[j] =
 * edge_count[e] / node_count[v] (aggregator normalisation of the message into v, [2m]; 0 where
 * node_count[v] = 0), each a correctly rounded float32 quotient.  N in [1, 2^24). */
erc_status erc_saint_counts(const erc_graph* g, const int32_t* nodes, int32_t n_s,
                            const int32_t* edges, int64_t m_s, int32_t* node_count,
                            int32_t* edge_count, erc_stream s);
erc_status erc_saint_norm(const erc_graph* g, const int32_t* node_count, const int32_t* edge_count,
                          int32_t N, float* lambda, float* alpha, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_laplacian_apply -- AP = L_eps P for an n x ld block (the CG operator of Eq. 5), and, when
 * pAp is not NULL, pAp[c] = sum_u P[u,c] AP[u,c] as float64 (device [kc]).  Exposed for testing
 * and benchmarking the operator alone.
 * ------------------------------------------------------------------------------------------- */
size_t erc_laplacian_apply_workspace_size(int32_t n, int32_t ld);
erc_status erc_laplacian_apply(const erc_graph* g, float eps, const float* P, float* AP,
                               int32_t ld, int32_t kc, double* pAp, void* ws, size_t ws_bytes,
                               erc_stream s);

/* erc_laplacian_apply_timed -- benchmarking helper: one untimed erc_laplacian_apply, then `reps`
 * back-to-back launches of the operator kernel alone between two CUDA events recorded on `s`;
 * *avg_us (host) receives the mean launch duration in microseconds.  Synchronises s. */
erc_status erc_laplacian_apply_timed(const erc_graph* g, float eps, const float* P, float* AP,
                                     int32_t ld, int32_t kc, double* pAp, int32_t reps,
                                     float* avg_us, void* ws, size_t ws_bytes, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_philox_signs -- the sign bits of Q[e, c] for e in [e0, e1), c in [c0, c1) (see erc_jl_rhs),
 * written to out_bits (device, row-major (e1-e0) x (c1-c0), one uint32 0/1 per entry).
 * ------------------------------------------------------------------------------------------- */
erc_status erc_philox_signs(uint64_t seed, int64_t e0, int64_t e1, int32_t c0, int32_t c1,
                            uint32_t* out_bits, erc_stream s);

/* ---------------------------------------------------------------------------------------------
 * erc_run -- the whole path: erc_build_laplacian, then for c0 = 0, kc, 2kc, ... < K:
 * erc_jl_rhs -> erc_batched_cg -> erc_edge_resistance (Algorithm 1), then erc_curvature and
 * erc_sampling_probs.  Inputs as erc_build_laplacian; outputs (device, capacity m_in for the edge
 * arrays): eu, ev [m], R [m], p_node [n], kappa [m], prob_node [n], prob_edge [m], iters [K],
 * relres [K]; m_out (host).  NOT_CONVERGED is reported after all batches are done.
 * erc_run_host is the same with src, dst, w and every output in HOST memory (pinned memory
 * makes the copies asynchronous); the copies run on s inside the call, and every output is
 * copied back whatever the CG status.
 * ------------------------------------------------------------------------------------------- */
size_t erc_run_workspace_size(int32_t n, int64_t m_in, int32_t kc);
erc_status erc_run(const erc_params* prm, int32_t n, const int32_t* src, const int32_t* dst,
                   const float* w, int64_t m_in, int64_t* m_out, int32_t* eu, int32_t* ev,
                   float* R, float* p_node, float* kappa, float* prob_node, float* prob_edge,
                   int32_t* iters, float* relres, void* ws, size_t ws_bytes, erc_stream s);
size_t erc_run_host_workspace_size(int32_t n, int64_t m_in, int32_t kc, int32_t K);
erc_status erc_run_host(const erc_params* prm, int32_t n, const int32_t* src, const int32_t* dst,
                        const float* w, int64_t m_in, int64_t* m_out, int32_t* eu, int32_t* ev,
                        float* R, float* p_node, float* kappa, float* prob_node,
                        float* prob_edge, int32_t* iters, float* relres, void* ws,
                        size_t ws_bytes, erc_stream s);

#ifdef __cplusplus
}
#endif
#endif /* ERC_H */
