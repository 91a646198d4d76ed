"""Plain fp64 CPU oracle for ERC-LG -- TEST INFRASTRUCTURE ONLY.

This module restates, slowly and in float64, what "Scalable Subgraph Sampling via Resistance
Curvature" (arxiv 2609.27209, §3) computes, so that the CUDA library can be checked against it.
Only the test-suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of ``bench.py`` may import
it; the library itself never does, and this file shares no code with the CUDA path.

Library primitives used as single steps: numpy sorting / reductions and a scipy sparse
matrix product (the products ``A @ P`` and ``B^T @ V``).  Nothing is blocked, fused or reordered
beyond what the paper's steps state.

Steps and where the paper states them
-------------------------------------
* ``build_laplacian``   -- L = D - A = B^T W B on the simple undirected graph (§3.1.1).
* ``philox4x32_10`` / ``jl_sign_bits`` -- the entries of Q, drawn uniformly from {+-1/sqrt(K)}
  (§3.1.2; Algorithm 1 streams them per column batch).  The counter layout is a convention of this
  library, see ``jl_sign_bits``.
* ``jl_rhs``            -- Y = B^T W^{1/2} Q for a column range (§3.1.2, Eq. 4's right-hand side).
* ``laplacian_matvec``  -- L_eps X = L X + eps X (Eq. 5, §3.1.3).
* ``batched_cg``        -- column-wise Hestenes-Stiefel CG on L_eps Z = Y to relative residual
  tolerance tau (§3.1.3; Algorithm 1).
* ``edge_resistance``   -- R_uv = ||Z_u - Z_v||^2 on the original edges, summed over column
  batches (Eq. 6; Algorithm 1's accumulation step).
* ``curvature``         -- node curvature p_u and edge curvature kappa_uv (Eq. 2).
* ``sampling_probs``    -- node weights (Eq. 7, with the uniform fallback), edge weights (Eq. 8),
  each normalised over all nodes / all edges (§3.2).
* ``erc_lg``            -- the whole of Algorithm 1 followed by §3.2.

Readings where the paper is silent (each is a convention shared with the CUDA library):
self-loops are dropped; duplicate edges are merged by summing their weights in float64 in input
order and rounding once to float32 (``dup_policy="first"`` keeps the first weight instead);
edge e of B is oriented from the smaller to the larger node id; edges are numbered in
lexicographic (u, v) order with u < v; the Q scale uses the total K even when columns are streamed
in batches; CG starts from x = 0 and stops a column when its recursive residual satisfies
||r|| <= tau ||y||; the uniform fallback of Eq. 7 applies when the node weights sum to exactly 0.
"""
from __future__ import annotations

import numpy as np
import scipy.sparse as sp

# ------------------------------------------------------------------------------------------------
# §3.1.1  the Laplacian L = D - A = B^T W B of the simple undirected graph
# ------------------------------------------------------------------------------------------------


def build_laplacian(n, src, dst, w=None, dup_policy="sum"):
    """Symmetric CSR of A plus degrees and the canonical edge list (§3.1.1).

    Returns a dict with
      row_ptr int64[n+1], col int32[2m] (ascending within each row), val float32[2m],
      deg float32[n] (= sum of the row's weights, accumulated in float64, rounded once),
      csr_eid int32[2m] (canonical edge id of each CSR slot),
      eu, ev int32[m] with eu < ev in lexicographic order, ew float32[m], and n, m.
    """
    src = np.asarray(src, dtype=np.int64)
    dst = np.asarray(dst, dtype=np.int64)
    m_in = src.size
    if np.any((src < 0) | (src >= n) | (dst < 0) | (dst >= n)):
        raise ValueError("node id out of range")
    w_in = np.ones(m_in, np.float32) if w is None else np.asarray(w, dtype=np.float32)
    if np.any(~np.isfinite(w_in)) or np.any(w_in <= 0):
        raise ValueError("edge weights must be finite and positive")

    keep = src != dst  # a self-loop has an all-zero incidence row: it is not part of B^T W B
    idx = np.nonzero(keep)[0]
    a = np.minimum(src[idx], dst[idx])
    b = np.maximum(src[idx], dst[idx])
    # lexicographic order of (a, b) by one integer key a n + b; stable: equal pairs keep input order
    order = np.argsort(a * n + b, kind="stable")
    a, b, wi = a[order], b[order], w_in[idx][order].astype(np.float64)

    if a.size:
        head = np.ones(a.size, bool)
        head[1:] = (a[1:] != a[:-1]) | (b[1:] != b[:-1])
        starts = np.nonzero(head)[0]
        if dup_policy == "sum":
            merged = np.add.reduceat(wi, starts)   # float64 sum of each run of duplicates
        elif dup_policy == "first":
            merged = wi[starts]
        else:
            raise ValueError(dup_policy)
        eu, ev, ew = a[starts], b[starts], merged.astype(np.float32)
    else:
        eu = ev = np.empty(0, np.int64)
        ew = np.empty(0, np.float32)
    m = eu.size

    # adjacency A: each undirected edge appears in row u and in row v
    rows = np.concatenate([eu, ev])
    cols = np.concatenate([ev, eu])
    eids = np.concatenate([np.arange(m), np.arange(m)])
    o = np.argsort(rows * n + cols)  # (row, col) pairs are distinct: lexicographic order
    rows, cols, eids = rows[o], cols[o], eids[o]
    row_ptr = np.zeros(n + 1, np.int64)
    np.cumsum(np.bincount(rows, minlength=n), out=row_ptr[1:])
    val = ew[eids]
    # deg_u: float64 sum of the row's float32 weights, rounded once to float32.  For weights whose
    # float64 partial sums are exact (every input used here) the value is order-independent.
    deg = np.zeros(n, np.float64)
    nonempty = np.nonzero(np.diff(row_ptr))[0]
    if nonempty.size:
        deg[nonempty] = np.add.reduceat(val.astype(np.float64), row_ptr[nonempty])
    return dict(n=int(n), m=int(m), row_ptr=row_ptr, col=cols.astype(np.int32), val=val,
                deg=deg.astype(np.float32), csr_eid=eids.astype(np.int32),
                eu=eu.astype(np.int32), ev=ev.astype(np.int32), ew=ew)


def adjacency(g):
    """A as a scipy CSR matrix (float64)."""
    return sp.csr_matrix((g["val"].astype(np.float64), g["col"], g["row_ptr"]),
                         shape=(g["n"], g["n"]))


def incidence(g):
    """Oriented incidence B (m x n): row e is e_u - e_v with u = eu[e] < v = ev[e] (§3.1.1)."""
    m, n = g["m"], g["n"]
    rows = np.repeat(np.arange(m), 2)
    cols = np.stack([g["eu"], g["ev"]], axis=1).ravel()
    vals = np.tile([1.0, -1.0], m)
    return sp.csr_matrix((vals, (rows, cols)), shape=(m, n))


# ------------------------------------------------------------------------------------------------
# §3.1.2  Q with entries uniform on {+-1/sqrt(K)}: Philox4x32-10 counter-based generator
# ------------------------------------------------------------------------------------------------
# Philox4x32-10 as published by Salmon, Moraes, Dror and Shaw, "Parallel Random Numbers: As Easy
# as 1, 2, 3" (SC'11): ten rounds of two 32x32->64 multiplies with a Weyl-sequence key schedule.
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
_MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(ctr, key):
    """Philox4x32-10 block function.

    ctr: tuple of four uint32-valued arrays (broadcastable), key: tuple of two uint32 ints.
    Returns the four output words as uint32 arrays.
    """
    c0, c1, c2, c3 = (np.asarray(c, dtype=np.uint64) & _MASK32 for c in ctr)
    k0 = np.uint64(int(key[0]) & 0xFFFFFFFF)
    k1 = np.uint64(int(key[1]) & 0xFFFFFFFF)
    m0, m1 = np.uint64(PHILOX_M0), np.uint64(PHILOX_M1)
    for _ in range(10):
        p0 = m0 * c0           # exact: both factors < 2^32, product < 2^64
        p1 = m1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
        k0 = (k0 + np.uint64(PHILOX_W0)) & _MASK32
        k1 = (k1 + np.uint64(PHILOX_W1)) & _MASK32
    return tuple(x.astype(np.uint32) for x in (c0, c1, c2, c3))


def jl_sign_bits(seed, e, c):
    """Sign bit (0 -> +1, 1 -> -1) of Q[e, c] for broadcastable edge ids e and column ids c.

    Layout convention: one Philox4x32-10 call yields the 128 signs of edge e for the columns
    128*g .. 128*g+127 with key (seed_lo, seed_hi) and counter (g, 0, e_lo, e_hi); column c takes
    bit (c mod 32) of output word ((c div 32) mod 4).
    """
    e = np.asarray(e, dtype=np.int64)
    c = np.asarray(c, dtype=np.int64)
    e, c = np.broadcast_arrays(e, c)
    g = (c >> 7).astype(np.uint64)
    words = philox4x32_10((g, 0, e & 0xFFFFFFFF, e >> 32), (seed & 0xFFFFFFFF, seed >> 32))
    widx = (c >> 5) & 3
    word = np.choose(widx, words)
    return ((word >> (c & 31).astype(np.uint32)) & np.uint32(1)).astype(np.uint8)


def jl_q(seed, K, e, c0, kc):
    """Dense block Q[e, c0:c0+kc] (float64) with entries +-1/sqrt(K) (§3.1.2)."""
    bits = jl_sign_bits(seed, np.asarray(e)[:, None], np.arange(c0, c0 + kc)[None, :])
    return (1.0 - 2.0 * bits.astype(np.float64)) / np.sqrt(K)


def jl_rhs(g, seed, K, c0, kc, edge_block=1 << 16, edge_ids=None):
    """Y = B^T W^{1/2} Q[:, c0:c0+kc]  (n x kc, float64), streamed over blocks of edges (§3.1.2).

    Edge e adds +sqrt(w_e) Q[e, :] to row eu[e] and -sqrt(w_e) Q[e, :] to row ev[e].
    `edge_ids` (optional) gives the id each edge of `g` has in a larger graph, so that rows of a
    subgraph holding every edge of those rows reproduce the larger graph's Y on them.
    """
    n, m = g["n"], g["m"]
    Y = np.zeros((n, kc))
    sw = np.sqrt(g["ew"].astype(np.float64))
    ids = np.arange(m) if edge_ids is None else np.asarray(edge_ids, dtype=np.int64)
    for e0 in range(0, m, edge_block):
        e = np.arange(e0, min(m, e0 + edge_block))
        V = sw[e, None] * jl_q(seed, K, ids[e], c0, kc)
        np.add.at(Y, g["eu"][e], V)
        np.add.at(Y, g["ev"][e], -V)
    return Y


# ------------------------------------------------------------------------------------------------
# §3.1.3  regularised system L_eps Z = Y and its column-wise CG solve
# ------------------------------------------------------------------------------------------------


def laplacian_matvec(g, eps, X, A=None, d=None):
    """L_eps X = (D + eps I) X - A X  (Eq. 5 with L = D - A, D_uu = sum_v A_uv in float64).

    `d` (optional) is the diagonal D + eps I as returned by `regularised_diagonal`, passed by the
    solvers so that it is formed once per solve rather than once per product."""
    A = adjacency(g) if A is None else A
    d = regularised_diagonal(A, eps) if d is None else d
    return d[:, None] * X - A @ X


def regularised_diagonal(A, eps):
    """The diagonal of L_eps = D - A + eps I: the float64 row sums of A plus eps (Eq. 5)."""
    return np.asarray(A.sum(axis=1)).ravel() + eps


def batched_cg(g, eps, Y, tol, max_iter=20000):
    """Column-wise CG (Hestenes-Stiefel) on L_eps X = Y, every column independent (§3.1.3).

    Each column starts at x = 0, r = p = y and stops once ||r|| <= tol ||y|| on the recursively
    updated residual (or after max_iter iterations).  Returns (X, iters, relres) with relres the
    true relative residual ||y - L_eps x|| / ||y|| of the returned X, and `converged`.
    """
    A = adjacency(g)
    d = regularised_diagonal(A, eps)
    Y = np.asarray(Y, dtype=np.float64)
    X = np.zeros_like(Y)
    Rv = Y.copy()
    P = Y.copy()
    rr = np.einsum("ij,ij->j", Rv, Rv)
    yy = rr.copy()
    active = rr > (tol * tol) * yy
    iters = np.zeros(Y.shape[1], np.int64)
    for _ in range(max_iter):
        if not active.any():
            break
        AP = laplacian_matvec(g, eps, P, A, d)
        pAp = np.einsum("ij,ij->j", P, AP)
        alpha = np.where(active, rr / np.where(active, pAp, 1.0), 0.0)
        X += alpha * P
        Rv -= alpha * AP
        rr_new = np.einsum("ij,ij->j", Rv, Rv)
        beta = np.where(active, rr_new / np.where(active, rr, 1.0), 0.0)
        P = np.where(active, Rv + beta * P, P)
        rr = np.where(active, rr_new, rr)
        iters += active
        active = active & (rr > (tol * tol) * yy)
    res = Y - laplacian_matvec(g, eps, X, A, d)
    ny = np.sqrt(yy)
    relres = np.where(ny > 0, np.sqrt(np.einsum("ij,ij->j", res, res)) / np.where(ny > 0, ny, 1),
                      0.0)
    return X, iters, relres, not active.any()


def batched_pcg(g, eps, Y, tol, max_iter=20000):
    """Optional solver variant, not in the paper: column-wise Jacobi-preconditioned CG on
    L_eps X = Y with M = diag(L_eps) = deg + eps (preconditioned CG as in Y. Saad, "Iterative
    Methods for Sparse Linear Systems", Algorithm 9.1).  Same start (x = 0, r = y), same stop test
    on the unpreconditioned recursive residual ||r|| <= tol ||y||, same outputs as batched_cg.
    """
    A = adjacency(g)
    d = regularised_diagonal(A, eps)  # the diagonal of L_eps, float64
    Y = np.asarray(Y, dtype=np.float64)
    X = np.zeros_like(Y)
    Rv = Y.copy()
    Z = Rv / d[:, None]
    P = Z.copy()
    rz = np.einsum("ij,ij->j", Rv, Z)
    yy = np.einsum("ij,ij->j", Y, Y)
    active = yy > (tol * tol) * yy
    iters = np.zeros(Y.shape[1], np.int64)
    for _ in range(max_iter):
        if not active.any():
            break
        AP = laplacian_matvec(g, eps, P, A, d)
        pAp = np.einsum("ij,ij->j", P, AP)
        alpha = np.where(active, rz / np.where(active, pAp, 1.0), 0.0)
        X += alpha * P
        Rv -= alpha * AP
        rr = np.einsum("ij,ij->j", Rv, Rv)
        Z = Rv / d[:, None]
        rz_new = np.einsum("ij,ij->j", Rv, Z)
        beta = np.where(active, rz_new / np.where(active, rz, 1.0), 0.0)
        P = np.where(active, Z + beta * P, P)
        rz = np.where(active, rz_new, rz)
        iters += active
        active = active & (rr > (tol * tol) * yy)
    res = Y - laplacian_matvec(g, eps, X, A, d)
    ny = np.sqrt(yy)
    relres = np.where(ny > 0, np.sqrt(np.einsum("ij,ij->j", res, res)) / np.where(ny > 0, ny, 1),
                      0.0)
    return X, iters, relres, not active.any()


# ------------------------------------------------------------------------------------------------
# Eq. 6, Eq. 2: resistances on the original edges, then curvature
# ------------------------------------------------------------------------------------------------


def edge_resistance(g, X):
    """sum over the columns of X of (X[u, c] - X[v, c])^2 for every edge (u, v) (Eq. 6)."""
    D = X[g["eu"]] - X[g["ev"]]
    return np.einsum("ij,ij->i", D, D)


def curvature(g, R):
    """p_u = 1 - 1/2 sum_{v in N(u)} w_uv R_uv,  kappa_uv = 2 (p_u + p_v) / R_uv  (Eq. 2)."""
    R = np.asarray(R, dtype=np.float64)
    wR = g["ew"].astype(np.float64) * R
    s = np.bincount(g["eu"], weights=wR, minlength=g["n"]) + \
        np.bincount(g["ev"], weights=wR, minlength=g["n"])
    p = 1.0 - 0.5 * s
    with np.errstate(divide="ignore", invalid="ignore"):
        kappa = 2.0 * (p[g["eu"]] + p[g["ev"]]) / R
    return p, kappa


# ------------------------------------------------------------------------------------------------
# §3.2: curvature-guided sampling probabilities (Eq. 7, Eq. 8, normalisation)
# ------------------------------------------------------------------------------------------------


def sampling_probs(g, kappa, eta=1e-8):
    """Node probabilities from Eq. 7 and edge probabilities from Eq. 8, each normalised (§3.2).

    q_u = sum_{v in N(u)} (kappa_uv - kappa_min) / (kappa_max - kappa_min + eta); when every q_u is
    zero the node distribution is uniform over the nodes with at least one edge.
    q_uv = sqrt(max(-kappa_uv + 2 kappa_max, 0)) + 1.
    """
    kappa = np.asarray(kappa, dtype=np.float64)
    n, m = g["n"], g["m"]
    if m == 0:
        return np.zeros(n), np.zeros(0)
    kmin, kmax = kappa.min(), kappa.max()
    score = (kappa - kmin) / (kmax - kmin + eta)
    q_node = np.bincount(g["eu"], weights=score, minlength=n) + \
        np.bincount(g["ev"], weights=score, minlength=n)
    tot = q_node.sum()
    if tot == 0.0:
        nonisolated = np.diff(g["row_ptr"]) > 0
        prob_node = nonisolated / nonisolated.sum()
    else:
        prob_node = q_node / tot
    q_edge = np.sqrt(np.maximum(-kappa + 2.0 * kmax, 0.0)) + 1.0
    return prob_node, q_edge / q_edge.sum()


# ------------------------------------------------------------------------------------------------
# Algorithm 1 + §3.2
# ------------------------------------------------------------------------------------------------


def erc_lg(n, src, dst, w, K, kc, eps, tol, seed, max_iter=20000, eta=1e-8, dup_policy="sum",
           columns=None, precond=None):
    """Algorithm 1 on one device: stream the K columns in batches of kc, accumulate R, then Eq. 2
    and §3.2.  `columns` = (c0, c1) restricts the run to that column range (R then holds only
    those columns' contributions).  precond="jacobi" solves with batched_pcg instead of the
    paper's CG."""
    g = build_laplacian(n, src, dst, w, dup_policy)
    c_lo, c_hi = (0, K) if columns is None else columns
    R = np.zeros(g["m"])
    iters = []
    relres = []
    converged = True
    for c0 in range(c_lo, c_hi, kc):
        k = min(kc, c_hi - c0)
        Y = jl_rhs(g, seed, K, c0, k)
        solve = batched_pcg if precond == "jacobi" else batched_cg
        X, it, rr, ok = solve(g, eps, Y, tol, max_iter)
        R += edge_resistance(g, X)
        iters.append(it)
        relres.append(rr)
        converged &= ok
    p, kappa = curvature(g, R)
    prob_node, prob_edge = sampling_probs(g, kappa, eta)
    return dict(graph=g, R=R, p=p, kappa=kappa, prob_node=prob_node, prob_edge=prob_edge,
                iters=np.concatenate(iters) if iters else np.zeros(0, np.int64),
                relres=np.concatenate(relres) if relres else np.zeros(0),
                converged=converged)
