"""Pins for the sampling probabilities (§3.2: Eq. 7, Eq. 8, normalisation, uniform fallback).

Hand-derived tree cases live in ``tests/golden/sampling_trees.json``; each one also re-derives its
kappa from exact resistances through Eq. 2 to check the tree closed form it relies on.
"""
import json
import math
import os

import numpy as np
import pytest

from oracle import dense as D
from oracle import erc_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "sampling_trees.json")
CASES = json.load(open(GOLDEN))["cases"]


def _ev(exprs):
    return np.array([eval(x, {"sqrt": math.sqrt}) for x in exprs], dtype=np.float64)


@pytest.mark.parametrize("case", CASES, ids=[c["name"] for c in CASES])
def test_golden_tree_probabilities(case):
    e = np.array(case["edges"], dtype=np.int32)
    g = O.build_laplacian(case["n"], e[:, 0], e[:, 1])
    np.testing.assert_array_equal(np.diff(g["row_ptr"]), case["degrees"])
    kappa = _ev(case["kappa"])
    # the tree closed form used by the fixture agrees with Eq. 2 on exact resistances
    L = D.dense_laplacian(g["n"], g["eu"], g["ev"], g["ew"])
    _, kappa_exact = O.curvature(g, D.exact_resistance(L, g["eu"], g["ev"]))
    np.testing.assert_allclose(kappa_exact, kappa, atol=1e-9)
    pn, pe = O.sampling_probs(g, kappa, eta=1e-8)
    np.testing.assert_allclose(pn, _ev(case["prob_node"]), rtol=1e-7, atol=1e-9)
    np.testing.assert_allclose(pe, _ev(case["prob_edge"]), rtol=1e-12)
    assert abs(pn.sum() - 1) < 1e-12 and abs(pe.sum() - 1) < 1e-12


def test_probabilities_are_normalised_on_random_input():
    rng = np.random.default_rng(0)
    n = 300
    src = rng.integers(0, n, 2000)
    dst = rng.integers(0, n, 2000)
    g = O.build_laplacian(n, src, dst)
    kappa = rng.normal(0, 2, g["m"])
    pn, pe = O.sampling_probs(g, kappa, eta=1e-8)
    assert abs(pn.sum() - 1) < 1e-12 and abs(pe.sum() - 1) < 1e-12
    assert np.all(pn >= 0) and np.all(pe > 0)
    # Eq. 8 favours low curvature: edge probability is non-increasing in kappa
    o = np.argsort(kappa)
    assert np.all(np.diff(pe[o]) <= 1e-15)
