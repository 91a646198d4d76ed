"""Pins for resistances and curvature (Eq. 1, Eq. 2, Eq. 6) against closed forms and theorems.

Exact resistances (pseudoinverse, Eq. 1): Foster's theorem sum_e w_e R_e = n - #components, tree
edges R = 1/w, the cycle R = (n-1)/(n w), the complete graph R = 2/n, parallel edges merged into one
conductance.  Curvature (Eq. 2) on exact resistances: cycle p = 1/n, kappa = 4/(n-1); K_n p = 1/n,
kappa = 2; trees p_u = 1 - d_u/2, kappa_uv = w_uv (4 - d_u - d_v); sum_u p_u = 1 when connected.
The JL estimate (Eq. 6) is checked against its exact mean and variance over Q.
"""
import numpy as np
import pytest
import scipy.sparse.csgraph as csg

from oracle import dense as D
from oracle import erc_oracle as O
from paper_2609_27209_gb300 import synth


def _exact(n, src, dst, w=None):
    g = O.build_laplacian(n, src, dst, w)
    L = D.dense_laplacian(n, g["eu"], g["ev"], g["ew"])
    return g, L, D.exact_resistance(L, g["eu"], g["ev"])


def test_foster_connected():
    g, L, R = _exact(*synth.random_connected(120, 400, seed=1))
    assert abs(np.dot(g["ew"].astype(np.float64), R) - (g["n"] - 1)) < 1e-9


def test_foster_disconnected():
    n, src, dst, w = synth.random_multigraph(60, 50, 2)
    g, L, R = _exact(n, src, dst, w)
    ncomp = csg.connected_components(O.adjacency(g), directed=False)[0]
    assert abs(np.dot(g["ew"].astype(np.float64), R) - (n - ncomp)) < 1e-9


def test_tree_resistance_is_inverse_weight():
    g, L, R = _exact(*synth.random_tree(50, seed=3))
    np.testing.assert_allclose(R, 1.0 / g["ew"].astype(np.float64), rtol=1e-10)


@pytest.mark.parametrize("n", [3, 7, 40])
def test_cycle_resistance(n):
    g, L, R = _exact(*synth.cycle(n, weight=2.5))
    np.testing.assert_allclose(R, (n - 1) / (n * 2.5), rtol=1e-10)


def test_complete_graph_resistance():
    g, L, R = _exact(*synth.complete(9))
    np.testing.assert_allclose(R, 2.0 / 9, rtol=1e-10)


def test_parallel_edges_merge_into_one_conductance():
    g, L, R = _exact(2, np.array([0, 1, 0]), np.array([1, 0, 1]),
                     np.array([1.5, 0.25, 2.0], np.float32))
    assert g["m"] == 1
    np.testing.assert_allclose(R, 1.0 / 3.75, rtol=1e-12)


def test_regularized_resistance_tends_to_exact():
    g, L, R = _exact(*synth.random_connected(80, 200, seed=4))
    prev = np.inf
    for eps in [1e-2, 1e-4, 1e-6]:
        Rr = D.regularized_resistance(L, eps, g["eu"], g["ev"])
        assert np.all(Rr <= R + 1e-12)
        err = np.max(np.abs(Rr - R))
        assert err < prev
        prev = err
    assert prev < 1e-5


# ---------------------------------------------------------------- curvature (Eq. 2) closed forms


@pytest.mark.parametrize("n", [5, 12])
def test_cycle_curvature(n):
    g, L, R = _exact(*synth.cycle(n))
    p, kappa = O.curvature(g, R)
    np.testing.assert_allclose(p, 1.0 / n, rtol=1e-9)
    np.testing.assert_allclose(kappa, 4.0 / (n - 1), rtol=1e-9)


def test_complete_graph_curvature():
    g, L, R = _exact(*synth.complete(8))
    p, kappa = O.curvature(g, R)
    np.testing.assert_allclose(p, 1.0 / 8, rtol=1e-9)
    np.testing.assert_allclose(kappa, 2.0, rtol=1e-9)


def test_tree_curvature_closed_form():
    g, L, R = _exact(*synth.random_tree(40, seed=5))
    p, kappa = O.curvature(g, R)
    d = np.diff(g["row_ptr"]).astype(np.float64)
    np.testing.assert_allclose(p, 1.0 - d / 2.0, atol=1e-9)
    w = g["ew"].astype(np.float64)
    np.testing.assert_allclose(kappa, w * (4.0 - d[g["eu"]] - d[g["ev"]]), atol=1e-8)


def test_node_curvature_sums_to_one():
    g, L, R = _exact(*synth.random_connected(90, 300, seed=6))
    p, _ = O.curvature(g, R)
    assert abs(p.sum() - 1.0) < 1e-9


# ---------------------------------------------------------------- JL estimate (Eq. 6)


def _jl(g, L, eps, K, seed):
    Y = O.jl_rhs(g, seed, K, 0, K)
    return O.edge_resistance(g, D.jl_dense_solve(L, eps, Y))


def test_jl_estimate_mean_and_variance():
    """R_hat has mean b^T L_eps^-1 L L_eps^-1 b and the exact JL variance; both <= R."""
    g, L, R = _exact(*synth.random_connected(40, 90, seed=7))
    eps, K = 1e-3, 64
    mean = D.jl_expected_resistance(L, eps, g["eu"], g["ev"])
    std = D.jl_resistance_std(L, eps, g["eu"], g["ev"], g["ew"], K)
    assert np.all(mean <= R + 1e-12)
    assert np.all(std <= np.sqrt(2.0 / K) * mean + 1e-12)
    z = []
    for seed in range(40):
        z.append((_jl(g, L, eps, K, seed) - mean) / std)
    z = np.array(z)
    assert abs(z.mean()) < 0.1
    assert 0.7 < z.var() < 1.3


def test_jl_estimate_converges_with_k():
    g, L, R = _exact(*synth.random_connected(30, 60, seed=8))
    err = [np.mean(np.abs(_jl(g, L, 1e-6, K, 3) - R) / R) for K in (64, 1024, 16384)]
    assert err[0] > err[1] > err[2]
    assert err[2] < 0.03


def test_foster_in_expectation_for_jl():
    g, L, R = _exact(*synth.random_connected(200, 800, seed=9))
    eps, K = 1e-3, 256
    lam = np.linalg.eigvalsh(L)
    expect = np.sum(lam ** 2 / (lam + eps) ** 2)
    tot = np.dot(g["ew"].astype(np.float64), _jl(g, L, eps, K, 1))
    assert abs(tot - expect) < 6 * np.sqrt(2.0 / (K * (g["n"] - 1))) * (g["n"] - 1)
    # each non-null mode loses 1 - lam^2/(lam+eps)^2 <= 2 eps / lam of its unit contribution
    nz = lam[1:]
    assert 0 <= (g["n"] - 1) - expect <= np.sum(2 * eps / nz)
