"""Pins for the oracle's right-hand sides, operator and CG (§3.1.2-§3.1.3, Eq. 4-5).

* Y = B^T W^{1/2} Q is compared with the dense incidence product, checked to lie in range(L)
  (1^T Y = 0 on every connected component) and checked statistically against E[Y Y^T] = L.
* L_eps X is compared with the dense (B^T W B + eps I) X.
* CG is compared with a direct dense solve (the paper's ERC-JL) and its true residual with tau,
  and its iterates (and those of the optional Jacobi PCG) step by step with scipy's cg.
"""
import numpy as np
import pytest
import scipy.sparse as sp
import scipy.sparse.csgraph as csg
import scipy.sparse.linalg as sla

from oracle import dense as D
from oracle import erc_oracle as O
from paper_2609_27209_gb300 import synth


def _graph(seed=0, n=60, extra=150):
    n, src, dst, w = synth.random_connected(n, extra, seed)
    return O.build_laplacian(n, src, dst, w)


def test_rhs_equals_dense_incidence_product():
    g = _graph(1)
    K, c0, kc = 300, 40, 200
    Y = O.jl_rhs(g, 99, K, c0, kc, edge_block=37)
    B = D.dense_incidence(g["n"], g["eu"], g["ev"])
    Q = O.jl_q(99, K, np.arange(g["m"]), c0, kc)
    ref = B.T @ (np.sqrt(g["ew"].astype(np.float64))[:, None] * Q)
    np.testing.assert_allclose(Y, ref, rtol=0, atol=1e-13)


def test_rhs_lies_in_range_of_laplacian_per_component():
    n, src, dst, w = synth.random_multigraph(80, 70, 5, self_loops=True)
    g = O.build_laplacian(n, src, dst, w)
    ncomp, lab = csg.connected_components(O.adjacency(g), directed=False)
    assert ncomp > 1
    Y = O.jl_rhs(g, 3, 64, 0, 64)
    for c in range(ncomp):
        np.testing.assert_allclose(Y[lab == c].sum(axis=0), 0.0, atol=1e-12)


def test_rhs_second_moment_is_laplacian():
    g = _graph(2, n=12, extra=20)
    K = 16384
    Y = O.jl_rhs(g, 11, K, 0, K)
    L = D.dense_laplacian(g["n"], g["eu"], g["ev"], g["ew"])
    M = Y @ Y.T
    d = np.diag(L)
    bound = 6.0 * np.sqrt(2.0 * np.outer(d, d) / K)
    assert np.all(np.abs(M - L) <= bound + 1e-12)


def test_matvec_equals_dense_regularized_laplacian():
    g = _graph(3)
    rng = np.random.default_rng(0)
    X = rng.standard_normal((g["n"], 7))
    L = D.dense_laplacian(g["n"], g["eu"], g["ev"], g["ew"])
    np.testing.assert_allclose(O.laplacian_matvec(g, 1e-3, X),
                               (L + 1e-3 * np.eye(g["n"])) @ X, rtol=0, atol=1e-11)


@pytest.mark.parametrize("eps", [1e-3, 1e-1])
def test_cg_matches_direct_solve(eps):
    g = _graph(4, n=150, extra=300)
    Y = O.jl_rhs(g, 5, 32, 0, 32)
    X, iters, relres, ok = O.batched_cg(g, eps, Y, 1e-11)
    assert ok
    Z = D.jl_dense_solve(D.dense_laplacian(g["n"], g["eu"], g["ev"], g["ew"]), eps, Y)
    np.testing.assert_allclose(X, Z, rtol=0, atol=1e-7 * np.abs(Z).max())
    assert np.all(relres <= 1e-11 * 1.01)
    assert np.all(iters > 0) and np.all(iters <= 3 * g["n"])


def test_cg_zero_column_and_max_iter():
    g = _graph(5)
    Y = O.jl_rhs(g, 6, 8, 0, 8)
    Y[:, 3] = 0.0
    X, iters, relres, ok = O.batched_cg(g, 1e-3, Y, 1e-8)
    assert ok and iters[3] == 0 and np.all(X[:, 3] == 0) and relres[3] == 0
    X, iters, relres, ok = O.batched_cg(g, 1e-3, Y, 1e-8, max_iter=2)
    assert not ok and np.all(iters[np.arange(8) != 3] == 2)


def test_cg_stops_columns_independently():
    """Each column's iterate equals a single-column solve of that column alone."""
    g = _graph(6, n=100, extra=200)
    Y = O.jl_rhs(g, 8, 16, 0, 16)
    Y[:, 0] *= 1e-3  # differently scaled columns still stop on their own relative residual
    X, iters, _, _ = O.batched_cg(g, 1e-3, Y, 1e-6)
    for c in [0, 5, 15]:
        x1, it1, _, _ = O.batched_cg(g, 1e-3, Y[:, c:c + 1], 1e-6)
        assert it1[0] == iters[c]
        np.testing.assert_allclose(X[:, c], x1[:, 0], rtol=1e-12, atol=1e-15)


def test_rhs_rows_of_a_subgraph_with_global_edge_ids():
    """Rows whose every edge is in a subgraph get the full graph's Y when edges keep their ids."""
    n, src, dst, w = synth.random_connected(300, 1200, seed=12)
    g = O.build_laplacian(n, src, dst, w)
    Y = O.jl_rhs(g, 7, 96, 32, 40)
    S = np.array([0, 5, 17, 123, 299])
    keep = np.isin(src, S) | np.isin(dst, S)
    sub = O.build_laplacian(n, src[keep], dst[keep], w[keep])
    keys = g["eu"].astype(np.int64) * n + g["ev"]
    ids = np.searchsorted(keys, sub["eu"].astype(np.int64) * n + sub["ev"])
    Ys = O.jl_rhs(sub, 7, 96, 32, 40, edge_ids=ids)
    np.testing.assert_allclose(Ys[S], Y[S], rtol=0, atol=1e-14)


# ---- the optional Jacobi-preconditioned variant (not in the paper)

@pytest.mark.parametrize("eps", [1e-3, 1e-1])
def test_pcg_matches_direct_solve(eps):
    g = _graph(4, n=150, extra=300)
    Y = O.jl_rhs(g, 5, 32, 0, 32)
    X, iters, relres, ok = O.batched_pcg(g, eps, Y, 1e-11)
    assert ok
    Z = D.jl_dense_solve(D.dense_laplacian(g["n"], g["eu"], g["ev"], g["ew"]), eps, Y)
    np.testing.assert_allclose(X, Z, rtol=0, atol=1e-7 * np.abs(Z).max())
    assert np.all(relres <= 1e-11 * 1.01)


@pytest.mark.parametrize("graph", ["cycle", "complete"])
def test_pcg_equals_cg_on_regular_graphs(graph):
    """Every degree equal: M = cI, and preconditioned CG takes exactly CG's steps."""
    n, src, dst, w = synth.cycle(200) if graph == "cycle" else synth.complete(40)
    g = O.build_laplacian(n, src, dst, w)
    Y = O.jl_rhs(g, 3, 16, 0, 16)
    Xc, ic, _, _ = O.batched_cg(g, 1e-3, Y, 1e-9)
    Xp, ip, _, _ = O.batched_pcg(g, 1e-3, Y, 1e-9)
    np.testing.assert_array_equal(ip, ic)
    np.testing.assert_allclose(Xp, Xc, rtol=1e-9, atol=1e-12 * np.abs(Xc).max())


def test_pcg_needs_fewer_iterations_with_hubs():
    """A 3,000-node Chung-Lu graph (degree exponent 2.2): degrees spread over orders of magnitude,
    which Jacobi scaling removes (measured: 88 CG against 23 preconditioned iterations)."""
    n, src, dst, w = synth.chung_lu(3000, 2.2, 20000, "unit", 7)
    g = O.build_laplacian(n, src, dst, w)
    Y = O.jl_rhs(g, 4, 8, 0, 8)
    _, ic, _, okc = O.batched_cg(g, 1e-3, Y, 1e-6)
    _, ip, rp, okp = O.batched_pcg(g, 1e-3, Y, 1e-6)
    assert okc and okp and np.all(rp <= 1.01e-6)
    assert ip.max() * 2 <= ic.max(), (ip.max(), ic.max())


@pytest.mark.parametrize("precond", [None, "jacobi"])
def test_iterates_match_scipy_cg(precond):
    """After k iterations from x = 0 the oracle's CG (and Jacobi PCG) iterate equals that of
    scipy.sparse.linalg.cg on the same L_eps and right-hand side (with the preconditioner
    M^-1 = diag(1 / (deg + eps)) for PCG), on a power-law graph whose diagonal varies widely: the
    alpha, beta and direction updates are pinned step by step, not only at convergence."""
    n, src, dst, w = synth.chung_lu(400, 2.2, 2000, "unit", 3)
    g = O.build_laplacian(n, src, dst, w)
    A = O.adjacency(g)
    eps = 1e-3
    d = np.asarray(A.sum(axis=1)).ravel() + eps
    L = sp.diags(d) - A
    M = sla.LinearOperator((n, n), matvec=lambda v: v / d) if precond else None
    Y = O.jl_rhs(g, 5, 4, 0, 4)
    solve = O.batched_pcg if precond else O.batched_cg
    for k in (1, 2, 5, 20):
        X, iters, _, _ = solve(g, eps, Y, 1e-30, max_iter=k)
        assert np.all(iters == k)
        for c in range(Y.shape[1]):
            ref, _ = sla.cg(L, Y[:, c], x0=np.zeros(n), rtol=1e-30, atol=0.0, maxiter=k, M=M)
            assert np.linalg.norm(X[:, c] - ref) <= 1e-11 * np.linalg.norm(ref), (k, c)
