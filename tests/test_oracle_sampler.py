"""Pins for the sampler oracle (§3.2 samplers, GraphSAINT normalisation).

Each check is against something the sampler's definition implies rather than against the oracle's
own formula: leading bits of the random word for dyadic probabilities, empirical frequencies,
inclusion probabilities 1 - (1 - p)^B, set-based induced subgraphs, and hand-derived
normalisation coefficients.
"""
import numpy as np

from oracle import erc_oracle as O
from oracle import sampler_oracle as S
from paper_2609_27209_gb300 import synth


def _graph(seed=0, n=60, extra=150):
    n, src, dst, w = synth.random_connected(n, extra, seed)
    return O.build_laplacian(n, src, dst, w)


def test_dyadic_probabilities_follow_the_leading_bits():
    # p = (1/4, 3/4): T = 2^40 and r = x >> 24, so index 0 exactly when x < 2^62
    p = np.array([0.25, 0.75], np.float32)
    idx = S.draw(p, 4000, seed=17, stream=0)
    words = S.draw_words(17, 0, 0, 4000)
    np.testing.assert_array_equal(idx, [0 if x < (1 << 62) else 1 for x in words])
    # p = (1/2, 0, 1/2): the middle entry is never drawn, the top bit decides the rest
    p = np.array([0.5, 0.0, 0.5], np.float32)
    idx = S.draw(p, 4000, seed=5, stream=1)
    words = S.draw_words(5, 1, 0, 4000)
    np.testing.assert_array_equal(idx, [0 if x < (1 << 63) else 2 for x in words])


def test_single_support_and_zero_weights():
    p = np.zeros(9, np.float32)
    p[6] = 1.0
    assert np.all(S.draw(p, 500, seed=1, stream=0) == 6)
    p = np.array([0.0, 0.3, 0.0, 0.7, 0.0], np.float32)
    idx = S.draw(p, 5000, seed=2, stream=0)
    assert set(np.unique(idx)) <= {1, 3}


def test_frequencies_match_probabilities():
    rng = np.random.default_rng(3)
    q = rng.random(8) ** 2
    p = (q / q.sum()).astype(np.float32)
    B = 100_000
    cnt = np.bincount(S.draw(p, B, seed=99, stream=0), minlength=8)
    pe = p.astype(np.float64)
    assert np.all(np.abs(cnt - B * pe) <= 5 * np.sqrt(B * pe * (1 - pe)) + 1), (cnt, B * pe)


def test_words_are_uniform_and_offset_consistent():
    w = S.draw_words(123, 0, 0, 50_000)
    u = np.array(w, dtype=np.float64) / 2.0 ** 64
    assert abs(u.mean() - 0.5) < 5 * np.sqrt(1 / 12 / u.size)
    assert S.draw_words(123, 0, 7, 20) == w[7:27]
    assert S.draw_words(123, 1, 0, 20) != w[:20]  # the two streams differ
    assert len(set(w)) == len(w)


def test_induced_edges_against_sets():
    g = _graph(4)
    rng = np.random.default_rng(4)
    nodes = np.unique(rng.integers(0, g["n"], 25))
    ns = set(nodes.tolist())
    ref = [e for e in range(g["m"]) if g["eu"][e] in ns and g["ev"][e] in ns]
    np.testing.assert_array_equal(S.induced_edges(g, nodes), ref)
    np.testing.assert_array_equal(S.induced_edges(g, np.arange(g["n"])), np.arange(g["m"]))
    assert S.induced_edges(g, [3]).size == 0
    e = 11
    np.testing.assert_array_equal(S.induced_edges(g, [g["eu"][e], g["ev"][e]]), [e])


def test_node_sampler_inclusion_probability():
    g = _graph(5, n=12, extra=20)
    rng = np.random.default_rng(5)
    q = rng.random(g["n"]) + 0.2
    p = (q / q.sum()).astype(np.float32)
    B, trials = 6, 4000
    hits = np.zeros(g["n"])
    for t in range(trials):
        nodes, _ = S.sample_nodes(g, p, B, seed=1000 + t)
        hits[nodes] += 1
    incl = 1 - (1 - p.astype(np.float64)) ** B
    assert np.all(np.abs(hits / trials - incl) <= 5 * np.sqrt(incl * (1 - incl) / trials))


def test_edge_sampler_structure():
    g = _graph(6)
    rng = np.random.default_rng(6)
    q = rng.random(g["m"])
    p = (q / q.sum()).astype(np.float32)
    nodes, drawn = S.sample_edges(g, p, 40, seed=8, induced=False)
    ends = set(g["eu"][drawn].tolist()) | set(g["ev"][drawn].tolist())
    assert set(nodes.tolist()) == ends
    nodes2, ind = S.sample_edges(g, p, 40, seed=8, induced=True)
    np.testing.assert_array_equal(nodes, nodes2)
    assert set(drawn.tolist()) <= set(ind.tolist())
    assert np.all(np.diff(ind) > 0)


def test_saint_norm_full_graph_and_path():
    g = _graph(7)
    full = (np.arange(g["n"]), np.arange(g["m"]))
    cn, ce = S.saint_counts(g, [full] * 5)
    lam, alpha = S.saint_norm(g, cn, ce, 5)
    assert np.all(lam == 1.0) and np.all(alpha == 1.0)
    # path 0-1-2: subgraphs {0,1}+(0,1) and {1,2}+(1,2) -> C = (1, 2, 1), C_e = (1, 1)
    p = O.build_laplacian(3, np.array([0, 1]), np.array([1, 2]))
    cn, ce = S.saint_counts(p, [([0, 1], [0]), ([1, 2], [1])])
    lam, alpha = S.saint_norm(p, cn, ce, 2)
    np.testing.assert_array_equal(lam, [0.5, 1.0, 0.5])
    # CSR slots: row 0 -> 1 (edge 0); row 1 -> 0 (edge 0), 2 (edge 1); row 2 -> 1 (edge 1)
    np.testing.assert_array_equal(alpha, [1.0, 0.5, 0.5, 1.0])
