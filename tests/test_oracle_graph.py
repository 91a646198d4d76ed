"""Pins for the oracle's Laplacian construction (§3.1.1: L = D - A = B^T W B).

Checked against a brute-force dictionary build of the simple graph, against the dense incidence
definition B^T W B, and against invariants (symmetry, sorted rows, L 1 = 0, sum deg = 2 sum w).
"""
import math

import numpy as np
import pytest

from oracle import dense as D
from oracle import erc_oracle as O
from paper_2609_27209_gb300 import synth


def brute_force(n, src, dst, w, policy):
    merged = {}
    for i, (a, b) in enumerate(zip(src.tolist(), dst.tolist())):
        if a == b:
            continue
        key = (min(a, b), max(a, b))
        merged.setdefault(key, []).append(1.0 if w is None else float(w[i]))
    edges = sorted(merged)
    weight = {}
    for k in edges:
        ws = merged[k]
        weight[k] = np.float32(math.fsum(ws) if policy == "sum" else ws[0])
    nbrs = [[] for _ in range(n)]
    for e, (a, b) in enumerate(edges):
        nbrs[a].append((b, e))
        nbrs[b].append((a, e))
    row_ptr = [0]
    col, val, eid = [], [], []
    deg = []
    for u in range(n):
        lst = sorted(nbrs[u])
        for v, e in lst:
            col.append(v)
            eid.append(e)
            val.append(weight[edges[e]])
        row_ptr.append(len(col))
        deg.append(np.float32(math.fsum(float(weight[edges[e]]) for _, e in lst)))
    return dict(row_ptr=np.array(row_ptr), col=np.array(col), val=np.array(val, np.float32),
                csr_eid=np.array(eid), deg=np.array(deg, np.float32),
                eu=np.array([a for a, _ in edges]), ev=np.array([b for _, b in edges]),
                ew=np.array([weight[k] for k in edges], np.float32), m=len(edges))


@pytest.mark.parametrize("seed", range(6))
@pytest.mark.parametrize("policy", ["sum", "first"])
@pytest.mark.parametrize("weighted", [True, False])
def test_csr_matches_brute_force(seed, policy, weighted):
    n, src, dst, w = synth.random_multigraph(23, 90, seed, weighted=weighted)
    g = O.build_laplacian(n, src, dst, w, policy)
    ref = brute_force(n, src, dst, w, policy)
    assert g["m"] == ref["m"]
    for k in ["row_ptr", "col", "csr_eid", "eu", "ev"]:
        np.testing.assert_array_equal(g[k], ref[k], err_msg=k)
    for k in ["val", "deg", "ew"]:
        np.testing.assert_array_equal(g[k], ref[k], err_msg=k)


def test_dense_laplacian_equals_degree_minus_adjacency():
    n, src, dst, w = synth.random_connected(40, 120, seed=3)
    g = O.build_laplacian(n, src, dst, w)
    L_inc = D.dense_laplacian(n, g["eu"], g["ev"], g["ew"])           # B^T W B
    A = O.adjacency(g).toarray()
    L_csr = np.diag(A.sum(axis=1)) - A  # D - A
    np.testing.assert_allclose(L_inc, L_csr, rtol=0, atol=1e-12)
    # the float32 degree output is that diagonal rounded once
    np.testing.assert_array_equal(g["deg"], np.diag(L_inc).astype(np.float32))
    np.testing.assert_allclose(L_inc @ np.ones(n), 0, atol=1e-12)


def test_csr_invariants_on_sbm():
    n, src, dst, w = synth.make_graph("sbm_n20000")
    g = O.build_laplacian(n, src, dst, w)
    A = O.adjacency(g)
    assert (A - A.T).nnz == 0
    rp, col = g["row_ptr"], g["col"]
    same_row = np.repeat(np.arange(n), np.diff(rp))
    assert np.all(np.diff(col.astype(np.int64))[np.diff(same_row) == 0] > 0)  # strictly sorted
    e = g["csr_eid"]
    lo = np.minimum(same_row, col)
    hi = np.maximum(same_row, col)
    np.testing.assert_array_equal(lo, g["eu"][e])
    np.testing.assert_array_equal(hi, g["ev"][e])
    assert np.all(g["eu"] < g["ev"])
    assert np.all(np.diff(g["eu"].astype(np.int64) * n + g["ev"]) > 0)
    np.testing.assert_allclose(g["deg"].astype(np.float64).sum(),
                               2 * g["ew"].astype(np.float64).sum(), rtol=1e-6)


@pytest.mark.parametrize("name", ["sbm_n20000"])
def test_degree_sum_is_exact_for_workload_weights(name):
    """deg is a float64 sum; for these weight ranges it is exact, hence order-independent."""
    n, src, dst, w = synth.make_graph(name)
    g = O.build_laplacian(n, src, dst, w)
    rp, val = g["row_ptr"], g["val"]
    rng = np.random.default_rng(0)
    rows = np.concatenate([rng.integers(0, n, 300), [int(np.argmax(np.diff(rp)))]])
    for u in rows:
        exact = math.fsum(val[rp[u]:rp[u + 1]].astype(np.float64).tolist())
        seq = 0.0
        for x in val[rp[u]:rp[u + 1]].astype(np.float64)[::-1]:
            seq += x
        assert seq == exact
        assert g["deg"][u] == np.float32(exact)


def test_uniform_weight_range_degree_exact():
    rng = np.random.default_rng(1)
    x = rng.uniform(0.5, 2.0, 20000).astype(np.float32).astype(np.float64)
    s = 0.0
    for v in x:
        s += v
    assert s == math.fsum(x.tolist())


def test_invalid_inputs_rejected():
    with pytest.raises(ValueError):
        O.build_laplacian(3, np.array([0, 3]), np.array([1, 1]))
    with pytest.raises(ValueError):
        O.build_laplacian(3, np.array([0]), np.array([1]), np.array([0.0], np.float32))
    with pytest.raises(ValueError):
        O.build_laplacian(3, np.array([0]), np.array([1]), np.array([np.nan], np.float32))


def test_self_loops_only_and_isolated_nodes():
    g = O.build_laplacian(4, np.array([1, 2]), np.array([1, 2]))
    assert g["m"] == 0
    np.testing.assert_array_equal(g["row_ptr"], np.zeros(5))
    g = O.build_laplacian(5, np.array([0, 4]), np.array([4, 0]))
    assert g["m"] == 1 and g["ew"][0] == 2.0  # duplicate (reversed) merged by summing
    np.testing.assert_array_equal(g["deg"], [2, 0, 0, 0, 2])
