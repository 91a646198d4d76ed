"""GPU parity of each C-ABI call against the CPU oracle on the same seeded inputs.

Integer work (CSR build, Philox signs) must match bit for bit; float32 work is held to bounds
derived from the arithmetic (relative float32 rounding times the magnitude of the summed terms).
"""
import numpy as np
import pytest
import torch

from oracle import erc_oracle as O
from paper_2609_27209_gb300 import erc, synth

from ._gpu import assert_graph_equal, build_both, dev, host, to_dev

pytestmark = pytest.mark.gpu
U32 = 2.0 ** -24


# ------------------------------------------------------------------ erc_build_laplacian (§3.1.1)
@pytest.mark.parametrize("seed", range(4))
@pytest.mark.parametrize("policy", [0, 1])
@pytest.mark.parametrize("weighted", [True, False])
def test_build_multigraph_bit_exact(seed, policy, weighted):
    n, src, dst, w = synth.random_multigraph(97, 3000, seed, weighted=weighted)
    g, ref = build_both(n, src, dst, w, policy)
    assert_graph_equal(g, ref)


@pytest.mark.parametrize("policy", [0, 1])
def test_build_reports_unit_weights(policy):
    """erc_build_laplacian_ex's unit-weight flag: 1 exactly when no weights were given and every
    merged weight is 1 (duplicates summed under ERC_DUP_SUM give 2; ERC_DUP_FIRST keeps 1)."""
    n, src, dst, _ = synth.random_connected(300, 900, seed=5)
    g = erc.erc_build_laplacian(n, to_dev(src), to_dev(dst), None, policy)
    assert g.unit_weights and bool((g.ew == 1).all())
    g = erc.erc_build_laplacian(n, to_dev(src), to_dev(dst),
                                to_dev(np.ones(src.size, np.float32)), policy)
    assert not g.unit_weights  # weights were given: the graph keeps its weight arrays
    dup_src, dup_dst = np.concatenate([src, dst[:5]]), np.concatenate([dst, src[:5]])
    g = erc.erc_build_laplacian(n, to_dev(dup_src), to_dev(dup_dst), None, policy)
    assert g.unit_weights == (policy == 1)
    assert bool((g.ew == 1).all()) == (policy == 1)


@pytest.mark.parametrize("name", ["ring_chords_n2000", "sbm_n20000"])
def test_build_workload_bit_exact(name):
    g, ref = build_both(*synth.make_graph(name))
    assert_graph_equal(g, ref)


def test_build_edge_cases():
    # only self-loops, isolated nodes, n = 1, empty edge list
    for n, src, dst in [(5, [1, 3], [1, 3]), (1, [0], [0]), (7, [], []), (9, [8, 0, 8], [0, 8, 0])]:
        s = np.array(src, np.int32)
        d = np.array(dst, np.int32)
        g, ref = build_both(n, s, d)
        assert_graph_equal(g, ref)
    # ids up to n - 1 with n a power of two and n one below it (key-width boundaries)
    for n in [1024, 1023, 1025]:
        s = np.array([0, n - 1, n - 2, 5], np.int32)
        d = np.array([n - 1, 0, n - 1, n - 1], np.int32)
        g, ref = build_both(n, s, d, np.array([1, 2, 3, 4], np.float32))
        assert_graph_equal(g, ref)


def test_build_rejects_bad_input():
    src = to_dev(np.array([0, 5], np.int32))
    dst = to_dev(np.array([1, 1], np.int32))
    with pytest.raises(erc.ErcError) as e:
        erc.erc_build_laplacian(5, src, dst)
    assert e.value.status == erc.ERC_ERR_INVALID_ARG
    src = to_dev(np.array([0, 2], np.int32))
    for bad in [0.0, -1.0, np.nan, np.inf]:
        with pytest.raises(erc.ErcError):
            erc.erc_build_laplacian(5, src, dst, to_dev(np.array([1.0, bad], np.float32)))


def test_build_is_deterministic():
    n, src, dst, w = synth.make_graph("sbm_n20000")
    a = erc.erc_build_laplacian(n, to_dev(src), to_dev(dst), to_dev(w))
    b = erc.erc_build_laplacian(n, to_dev(src), to_dev(dst), to_dev(w))
    for k in ["row_ptr", "col", "val", "deg", "csr_eid", "eu", "ev", "ew"]:
        assert torch.equal(getattr(a, k), getattr(b, k)), k


# ------------------------------------------------------------------ Philox signs and Y (§3.1.2)
@pytest.mark.parametrize("seed", [0xE2C1, 0xFFFFFFFF00000001])
def test_philox_signs_bit_exact(seed):
    for e0, e1, c0, c1 in [(0, 300, 0, 300), (70000, 70100, 100, 600), ((1 << 31) + 5, (1 << 31) + 40, 1000, 1030)]:
        got = host(erc.erc_philox_signs(seed, e0, e1, c0, c1))
        ref = O.jl_sign_bits(seed, np.arange(e0, e1)[:, None], np.arange(c0, c1)[None, :])
        np.testing.assert_array_equal(got, ref)


def _rhs_bound(ref, K):
    """|sum of float32 terms| error bound per row: a few ulps of the sum of |terms|."""
    rp = ref["row_ptr"]
    sw = np.sqrt(ref["val"].astype(np.float64)) / np.sqrt(K)
    rows = np.repeat(np.arange(ref["n"]), np.diff(rp))
    mag = np.bincount(rows, weights=sw, minlength=ref["n"])
    deg = np.diff(rp)
    return (4 + deg) * U32 * mag


@pytest.mark.parametrize("name,K,c0,kc", [("ring_chords_n2000", 64, 0, 64),
                                          ("sbm_n20000", 128, 0, 128),
                                          ("sbm_n20000", 1024, 256, 200),
                                          ("ring_chords_n2000", 300, 4, 33)])
def test_jl_rhs(name, K, c0, kc):
    n, src, dst, w = synth.make_graph(name)
    g, ref = build_both(n, src, dst, w)
    Y = host(erc.erc_jl_rhs(g, synth.JL_SEED, K, c0, kc))
    Yr = O.jl_rhs(ref, synth.JL_SEED, K, c0, kc)
    assert np.all(Y[:, kc:] == 0)
    bound = _rhs_bound(ref, K)[:, None]
    assert np.all(np.abs(Y[:, :kc] - Yr) <= bound + 1e-30)


# ------------------------------------------------------------------ L_eps P (Eq. 5)
def _matvec_bound(ref, eps, P):
    """float32 error bound of eps p_u + sum_v w (p_u - p_v), elementwise."""
    A = O.adjacency(ref)
    absP = np.abs(P.astype(np.float64))
    deg = np.asarray(A.sum(axis=1)).ravel()
    mag = eps * absP + deg[:, None] * absP + A @ absP
    d = np.diff(ref["row_ptr"])[:, None]
    return (4 + 2 * d) * U32 * mag


@pytest.mark.parametrize("kc", [3, 4, 16, 32, 64, 100, 128, 256, 512, 1024])
def test_laplacian_apply(kc):
    n, src, dst, w = synth.random_connected(1500, 6000, seed=kc, weighted=kc % 2 == 0)
    g, ref = build_both(n, src, dst, w)
    ld = erc.padded_ld(kc)
    P = synth.random_block(n, kc, ld, seed=kc + 1)
    eps = 1e-3
    AP, pap = erc.erc_laplacian_apply(g, eps, to_dev(P), kc, want_pap=True)
    AP = host(AP)
    APr = O.laplacian_matvec(ref, eps, P[:, :kc].astype(np.float64))
    assert np.all(np.abs(AP[:, :kc] - APr) <= _matvec_bound(ref, eps, P[:, :kc]))
    pr = np.einsum("ij,ij->j", P[:, :kc].astype(np.float64), APr)
    np.testing.assert_allclose(host(pap), pr, rtol=2e-6)


def test_laplacian_apply_hub_rows():
    """A star with a 20k-neighbour hub plus a path: long and short rows in one launch."""
    n = 20001
    src = np.concatenate([np.zeros(n - 1, np.int32), np.arange(1, n - 1, dtype=np.int32)])
    dst = np.concatenate([np.arange(1, n, dtype=np.int32), np.arange(2, n, dtype=np.int32)])
    g, ref = build_both(n, src, dst)
    for kc in [8, 128]:
        P = synth.random_block(n, kc, kc, seed=3)
        AP, _ = erc.erc_laplacian_apply(g, 1e-3, to_dev(P), kc)
        APr = O.laplacian_matvec(ref, 1e-3, P.astype(np.float64))
        assert np.all(np.abs(host(AP) - APr) <= _matvec_bound(ref, 1e-3, P))


# ------------------------------------------------------------------ R accumulation (Eq. 6)
@pytest.mark.parametrize("kc", [5, 32, 128, 256])
def test_edge_resistance_accumulates(kc):
    n, src, dst, w = synth.random_connected(3000, 9000, seed=7)
    g, ref = build_both(n, src, dst, w)
    ld = erc.padded_ld(kc)
    X1 = synth.random_block(n, kc, ld, seed=1)
    X2 = synth.random_block(n, kc, ld, seed=2)
    R0 = synth.random_positive(g.m, seed=3)
    R = to_dev(R0.copy())
    erc.erc_edge_resistance(g, to_dev(X1), kc, R)
    erc.erc_edge_resistance(g, to_dev(X2), kc, R)
    Rr = R0.astype(np.float64) + O.edge_resistance(ref, X1[:, :kc].astype(np.float64)) + \
        O.edge_resistance(ref, X2[:, :kc].astype(np.float64))
    np.testing.assert_allclose(host(R), Rr, rtol=(kc + 8) * U32)


# ------------------------------------------------------------------ curvature (Eq. 2)
@pytest.mark.parametrize("weighted", [True, False])
def test_curvature(weighted):
    n, src, dst, w = synth.random_connected(5000, 30000, seed=8, weighted=weighted)
    g, ref = build_both(n, src, dst, w)
    R = synth.random_positive(g.m, seed=9, lo=0.02, hi=1.0)
    p, kappa = erc.erc_curvature(g, to_dev(R))
    pr, kr = O.curvature(ref, R.astype(np.float64))
    half_sum = 1.0 - pr  # = 1/2 sum w R >= 0
    assert np.all(np.abs(host(p) - pr) <= 4 * U32 * (np.abs(pr) + half_sum + 1))
    # kappa = 2 (p_u + p_v) / R from float32 p: error from the rounding of p and of the division
    pe = 4 * U32 * (np.abs(pr) + half_sum + 1)
    kb = 2 * (pe[ref["eu"]] + pe[ref["ev"]]) / R + 4 * U32 * np.abs(kr)
    assert np.all(np.abs(host(kappa) - kr) <= kb)


# ------------------------------------------------------------------ sampling (§3.2)
def test_sampling_probs_random_kappa():
    n, src, dst, w = synth.random_connected(4000, 20000, seed=10)
    g, ref = build_both(n, src, dst, w)
    kappa = synth.random_normal(g.m, seed=11, scale=3.0)
    pn, pe = erc.erc_sampling_probs(g, to_dev(kappa), 1e-8)
    pnr, per = O.sampling_probs(ref, kappa.astype(np.float64), 1e-8)
    np.testing.assert_allclose(host(pn), pnr, rtol=1e-6, atol=1e-12)
    np.testing.assert_allclose(host(pe), per, rtol=1e-6)


def test_sampling_probs_golden_trees():
    import json
    import math
    import os
    cases = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                        "sampling_trees.json")))["cases"]
    ev = lambda xs: np.array([eval(x, {"sqrt": math.sqrt}) for x in xs])  # noqa: E731
    for c in cases:
        e = np.array(c["edges"], np.int32)
        g, ref = build_both(c["n"], e[:, 0], e[:, 1])
        kappa = ev(c["kappa"]).astype(np.float32)
        pn, pe = erc.erc_sampling_probs(g, to_dev(kappa), 1e-8)
        np.testing.assert_allclose(host(pn), ev(c["prob_node"]), rtol=1e-6, atol=1e-9)
        np.testing.assert_allclose(host(pe), ev(c["prob_edge"]), rtol=1e-6)


def test_sampling_probs_uniform_fallback_with_isolated_nodes():
    n = 12
    src = np.arange(8, dtype=np.int32)
    dst = ((np.arange(8) + 1) % 8).astype(np.int32)  # an 8-cycle, nodes 8..11 isolated
    g, ref = build_both(n, src, dst)
    kappa = np.full(g.m, 0.5, np.float32)
    pn, pe = erc.erc_sampling_probs(g, to_dev(kappa), 1e-8)
    np.testing.assert_allclose(host(pn), [1 / 8] * 8 + [0] * 4, rtol=1e-7)
    np.testing.assert_allclose(host(pe), 1 / 8, rtol=1e-7)
