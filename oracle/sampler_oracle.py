"""Oracle of the curvature-guided subgraph samplers (§3.2, Eq. 7 and Eq. 8; the experiments'
ERC-LG-sub(node) and ERC-LG-sub(edge) variants, which follow GraphSAINT's node and edge samplers
with the curvature-based probabilities) and of GraphSAINT's count-based normalisation.

TEST INFRASTRUCTURE ONLY: imported by tests/ (and nothing on the product path).  Plain numpy and
Python integers, written for checking by eye, not for speed.

Readings (the paper names the samplers but not their mechanics):
  * A draw picks index i with probability proportional to the float32 probability p_i, exactly:
    the weights are fixed point, W_i = round(p_i * 2^40) (int64), their inclusive prefix sums
    C_i are exact, and a 64-bit random word x selects r = floor(x * T / 2^64), T = sum W, and
    the smallest i with C_i > r.  Entries with p_i < 2^-41 are never drawn.
  * Draw k of stream s takes its word from Philox4x32-10 (the block function of the oracle's
    sign generator) with key (seed lo, seed hi) and counter (k lo, k hi, 0x53414D50, s): output
    words 0 (high half) and 1 (low half).  Stream 0 is the node sampler, 1 the edge sampler.
  * Node sampler: B draws with replacement over the nodes; the subgraph is induced on the
    distinct drawn nodes (all canonical edges with both endpoints drawn).
  * Edge sampler: B draws over the canonical edges; its nodes are the drawn edges' endpoints and
    its edges are either the subgraph induced on them (GraphSAINT) or the distinct drawn edges
    (the paper's "selected edges and their endpoints").
  * Normalisation over N sampled subgraphs: C_v and C_e count the subgraphs that contain node v
    and edge e; lambda_v = C_v / N (loss normalisation) and, for CSR slot j of row v holding
    edge e, alpha_j = C_e / C_v (aggregator normalisation of the message into v); 0 where
    C_v = 0.
"""
import numpy as np

from .erc_oracle import philox4x32_10

FIX_BITS = 40
SAMPLER_TAG = 0x53414D50
STREAM_NODE = 0
STREAM_EDGE = 1


def integer_weights(prob):
    """Fixed-point weights round(p * 2^40) of float32 probabilities (exact in float64)."""
    p = np.asarray(prob, dtype=np.float32).astype(np.float64)
    return np.floor(p * 2.0 ** FIX_BITS + 0.5).astype(np.int64)


def draw_words(seed, stream, k0, count):
    """The 64-bit words of draws k0 .. k0+count-1 of a stream (Python ints)."""
    k = np.arange(k0, k0 + count, dtype=np.uint64)
    w = philox4x32_10((k & np.uint64(0xFFFFFFFF), k >> np.uint64(32), SAMPLER_TAG, stream),
                      (seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF))
    return [(int(hi) << 32) | int(lo) for hi, lo in zip(w[0], w[1])]


def draw(prob, budget, seed, stream, k0=0):
    """Indices of `budget` draws proportional to `prob` (see the module readings)."""
    W = integer_weights(prob)
    C = np.cumsum(W)  # exact int64 inclusive prefix sums
    T = int(C[-1]) if C.size else 0
    if budget == 0:
        return np.zeros(0, np.int64)
    if T == 0:
        raise ValueError("every weight rounds to zero")
    r = np.array([(x * T) >> 64 for x in draw_words(seed, stream, k0, budget)], dtype=np.int64)
    return np.searchsorted(C, r, side="right").astype(np.int64)


def induced_edges(g, nodes):
    """Ascending ids of the canonical edges with both endpoints in `nodes`."""
    inside = np.zeros(g["n"], dtype=bool)
    inside[np.asarray(nodes, dtype=np.int64)] = True
    return np.flatnonzero(inside[g["eu"]] & inside[g["ev"]]).astype(np.int64)


def sample_nodes(g, prob_node, budget, seed, k0=0):
    """Node sampler: (sorted distinct nodes, ascending induced edge ids)."""
    nodes = np.unique(draw(prob_node, budget, seed, STREAM_NODE, k0))
    return nodes, induced_edges(g, nodes)


def sample_edges(g, prob_edge, budget, seed, k0=0, induced=True):
    """Edge sampler: (sorted distinct endpoints, ascending edge ids)."""
    drawn = np.unique(draw(prob_edge, budget, seed, STREAM_EDGE, k0))
    nodes = np.unique(np.concatenate([g["eu"][drawn], g["ev"][drawn]]).astype(np.int64))
    return nodes, (induced_edges(g, nodes) if induced else drawn)


def saint_counts(g, subgraphs):
    """C_v and C_e over a list of (nodes, edges) subgraphs."""
    cn = np.zeros(g["n"], dtype=np.int64)
    ce = np.zeros(g["m"], dtype=np.int64)
    for nodes, edges in subgraphs:
        cn[np.asarray(nodes, dtype=np.int64)] += 1
        ce[np.asarray(edges, dtype=np.int64)] += 1
    return cn, ce


def saint_norm(g, cn, ce, N):
    """lambda_v = C_v / N and alpha per CSR slot = C_e / C_row (float64; 0 where C_row = 0)."""
    lam = cn.astype(np.float64) / float(N)
    rows = np.repeat(np.arange(g["n"]), np.diff(g["row_ptr"]))
    c_row = cn[rows].astype(np.float64)
    c_e = ce[g["csr_eid"]].astype(np.float64)
    alpha = np.divide(c_e, c_row, out=np.zeros_like(c_e), where=c_row > 0)
    return lam, alpha
