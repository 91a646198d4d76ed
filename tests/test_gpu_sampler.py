"""GPU parity of the curvature-guided subgraph samplers and GraphSAINT normalisation (§3.2).

Draws, node sets, edge sets and counts are integer results: bit-exact against the oracle.  The
normalisation coefficients are correctly rounded float32 quotients of integers: within one ulp
of the oracle's float64 quotients.
"""
import numpy as np
import pytest
import torch

from oracle import sampler_oracle as S
from paper_2609_27209_gb300 import erc, synth

from ._gpu import build_both, dev, host, to_dev

pytestmark = pytest.mark.gpu


def _probs(count, seed, zeros=0.2):
    rng = np.random.default_rng(seed)
    q = rng.random(count) ** 3
    q[rng.random(count) < zeros] = 0.0
    return (q / q.sum()).astype(np.float32)


@pytest.fixture(scope="module")
def graph():
    n, src, dst, w = synth.random_connected(700, 2800, seed=21, weighted=True)
    return build_both(n, src, dst, w)


@pytest.mark.parametrize("budget,seed,first", [(1, 3, 0), (64, 4, 0), (600, 5, 1000),
                                               (5000, 6, (1 << 33) + 7)])
def test_node_sampler_matches_oracle(graph, budget, seed, first):
    g, ref = graph
    p = _probs(g.n, seed)
    nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, to_dev(p), budget, seed, first)
    rn, re_ = S.sample_nodes(ref, p, budget, seed, first)
    np.testing.assert_array_equal(host(nodes), rn)
    np.testing.assert_array_equal(host(edges), re_)


@pytest.mark.parametrize("induced", [True, False])
@pytest.mark.parametrize("budget,seed", [(1, 7), (200, 8), (3000, 9)])
def test_edge_sampler_matches_oracle(graph, budget, seed, induced):
    g, ref = graph
    p = _probs(g.m, seed)
    nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_EDGES, to_dev(p), budget, seed,
                                           induced=induced)
    rn, re_ = S.sample_edges(ref, p, budget, seed, induced=induced)
    np.testing.assert_array_equal(host(nodes), rn)
    np.testing.assert_array_equal(host(edges), re_)


def test_stream_continues_across_calls(graph):
    g, _ = graph
    p = to_dev(_probs(g.n, 10))
    a, _ = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, p, 400, 11, 0)
    b1, _ = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, p, 150, 11, 0)
    b2, _ = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, p, 250, 11, 150)
    np.testing.assert_array_equal(host(a), np.union1d(host(b1), host(b2)))


def test_saint_counts_and_norm_match_oracle(graph):
    g, ref = graph
    p = _probs(g.n, 12, zeros=0.0)
    N = 25
    cn = torch.zeros(g.n, dtype=torch.int32, device=dev())
    ce = torch.zeros(g.m, dtype=torch.int32, device=dev())
    subs = []
    for t in range(N):
        nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, to_dev(p), 150, 13,
                                               150 * t)
        erc.erc_saint_counts(g, nodes, edges, cn, ce)
        subs.append(S.sample_nodes(ref, p, 150, 13, 150 * t))
    rcn, rce = S.saint_counts(ref, subs)
    np.testing.assert_array_equal(host(cn), rcn)
    np.testing.assert_array_equal(host(ce), rce)
    lam, alpha = erc.erc_saint_norm(g, cn, ce, N)
    rlam, ralpha = S.saint_norm(ref, rcn, rce, N)
    ulp = 2.0 ** -23
    assert np.all(np.abs(host(lam) - rlam) <= ulp * rlam)
    assert np.all(np.abs(host(alpha) - ralpha) <= ulp * ralpha)
    assert np.any(host(alpha) > 0) and np.any(host(alpha) < 1)


def test_sampler_edge_cases(graph):
    g, ref = graph
    p = np.zeros(g.n, np.float32)
    p[123] = 1.0
    nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, to_dev(p), 50, 1)
    np.testing.assert_array_equal(host(nodes), [123])
    assert edges.numel() == 0
    nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, to_dev(p), 0, 1)
    assert nodes.numel() == 0 and edges.numel() == 0
    for bad in [np.full(g.n, 0.0, np.float32), np.full(g.n, 2.0, np.float32)]:
        with pytest.raises(erc.ErcError) as e:
            erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, to_dev(bad), 10, 1)
        assert e.value.status == erc.ERC_ERR_INVALID_ARG
    q = _probs(g.n, 2)
    q[5] = np.nan
    with pytest.raises(erc.ErcError):
        erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, to_dev(q), 10, 1)


def test_sampler_on_pipeline_probabilities_full_size():
    """The 169k-node workload: probabilities from the whole path, one node and one edge
    subgraph, against the oracle fed the same float32 probabilities."""
    name = "chung_lu_n169343_g2.5"
    wl = synth.WORKLOADS[name]
    n, src, dst, w = synth.make_graph(name)
    prm = erc.Params(K=32, kc=32, eps=wl.eps, tol=wl.tol, seed=synth.JL_SEED)
    out = erc.erc_run(n, to_dev(src), to_dev(dst), None if w is None else to_dev(w), prm)
    g, ref = build_both(n, src, dst, w)
    pn, pe = host(out["prob_node"]), host(out["prob_edge"])
    nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, out["prob_node"], 8000, 77)
    rn, re_ = S.sample_nodes(ref, pn, 8000, 77)
    np.testing.assert_array_equal(host(nodes), rn)
    np.testing.assert_array_equal(host(edges), re_)
    nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_EDGES, out["prob_edge"], 8000, 78)
    rn, re_ = S.sample_edges(ref, pe, 8000, 78)
    np.testing.assert_array_equal(host(nodes), rn)
    np.testing.assert_array_equal(host(edges), re_)
