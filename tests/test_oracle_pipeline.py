"""The whole oracle pipeline (Algorithm 1 + §3.2) on the 2,000-node ring-with-chords workload.

Pinned against the dense definitions: ERC-LG with CG agrees with the direct-solve ERC-JL on the same
projection (Table 3 reports the two as nearly identical), the estimate is unbiased for its exact
JL mean, Foster's theorem holds in expectation, and streaming columns in batches changes nothing.
"""
import numpy as np
import pytest

from oracle import dense as D
from oracle import erc_oracle as O
from paper_2609_27209_gb300 import synth


@pytest.fixture(scope="module")
def c1():
    wl = synth.WORKLOADS["ring_chords_n2000"]
    n, src, dst, w = synth.make_graph(wl.name)
    out = O.erc_lg(n, src, dst, w, wl.K[0], wl.kc, wl.eps, wl.tol, synth.JL_SEED)
    g = out["graph"]
    L = D.dense_laplacian(n, g["eu"], g["ev"], g["ew"])
    return wl, (n, src, dst, w), out, L


def test_workload_shape(c1):
    wl, (n, src, dst, w), out, L = c1
    g = out["graph"]
    assert n == 2000 and g["m"] == 10000 and w is None
    assert out["converged"] and np.all(out["relres"] <= 1.5 * wl.tol)


def test_cg_agrees_with_direct_solve(c1):
    wl, _, out, L = c1
    g = out["graph"]
    Y = O.jl_rhs(g, synth.JL_SEED, wl.K[0], 0, wl.K[0])
    R_jl = O.edge_resistance(g, D.jl_dense_solve(L, wl.eps, Y))
    rel = np.abs(out["R"] - R_jl) / R_jl
    assert np.median(rel) < 1e-6 and rel.max() < 1e-4


def test_unbiased_for_exact_jl_mean_and_foster(c1):
    wl, _, out, L = c1
    g = out["graph"]
    mean = D.jl_expected_resistance(L, wl.eps, g["eu"], g["ev"])
    rel = out["R"] / mean - 1
    K = wl.K[0]
    assert abs(rel.mean()) < 6 * np.sqrt(2.0 / K) / np.sqrt(50)   # edges are weakly dependent
    assert np.std(rel) < 1.2 * np.sqrt(2.0 / K)
    n = g["n"]
    tot = np.dot(g["ew"].astype(np.float64), out["R"])
    assert abs(tot - (n - 1)) < 6 * np.sqrt(2.0 / (K * (n - 1))) * (n - 1)
    assert abs(out["p"].sum() - 1) < 6 * np.sqrt(2.0 / (K * (n - 1))) * (n - 1)


def test_column_batches_sum_to_the_whole(c1):
    wl, (n, src, dst, w), out, L = c1
    a = O.erc_lg(n, src, dst, w, 64, 16, wl.eps, wl.tol, synth.JL_SEED, columns=(0, 32))
    b = O.erc_lg(n, src, dst, w, 64, 32, wl.eps, wl.tol, synth.JL_SEED, columns=(32, 64))
    np.testing.assert_allclose(a["R"] + b["R"], out["R"], rtol=1e-9)
