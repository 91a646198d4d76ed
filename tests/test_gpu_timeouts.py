"""Failure detection: every bounded device-side wait reports ERC_ERR_TIMEOUT when it runs out.

erc_set_wait_limit(1) makes every wait of the library give up after one poll: the look-back of
the single-pass scans (Laplacian build, subgraph sampler), the grid barrier of the multi-kernel
CG update and the grid synchronisations of the resident CG solver.  With other blocks still
working, such a wait runs out at once, the call's kernels stop consuming the unfinished result,
and the call returns ERC_ERR_TIMEOUT.  Nothing faults or hangs: a call either completes with
exact results (every wait it made happened to be satisfied already) or reports the timeout, and
over a few calls on inputs of thousands of blocks the timeout path is taken.  With the default
limits restored the same calls succeed again on the same context.
"""
import os

import numpy as np
import pytest
import torch

from paper_2609_27209_gb300 import erc, synth

from ._gpu import assert_graph_equal, build_both, host, to_dev

pytestmark = pytest.mark.gpu
TRIES = 3


@pytest.fixture(autouse=True)
def default_limits_after():
    yield
    erc.erc_set_wait_limit(0)
    os.environ.pop("ERC_CG_MODE", None)


def _status(fn):
    try:
        fn()
        return erc.ERC_OK
    except erc.ErcError as e:
        return e.status


def test_build_scan_timeout_is_reported():
    n, src, dst, w = synth.random_connected(400_000, 1_600_000, seed=41, weighted=True)
    src_d, dst_d, w_d = to_dev(src), to_dev(dst), to_dev(w)
    ref_g, ref = build_both(n, src, dst, w)
    erc.erc_set_wait_limit(1)
    seen = []
    for _ in range(TRIES):
        st = _status(lambda: erc.erc_build_laplacian(n, src_d, dst_d, w_d))
        assert st in (erc.ERC_OK, erc.ERC_ERR_TIMEOUT), st
        if st == erc.ERC_ERR_TIMEOUT:
            assert b"bounded wait" in erc.lib().erc_last_error()
        seen.append(st)
    assert erc.ERC_ERR_TIMEOUT in seen, seen
    erc.erc_set_wait_limit(0)
    assert_graph_equal(erc.erc_build_laplacian(n, src_d, dst_d, w_d), ref)


def test_sampler_scan_timeout_is_reported():
    n, src, dst, w = synth.random_connected(2_000_000, 4_000_000, seed=43)
    g = erc.erc_build_laplacian(n, to_dev(src), to_dev(dst))
    prob = torch.full((n,), 1.0 / n, dtype=torch.float32, device="cuda:0")
    ref_nodes, ref_edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, prob, 50_000, 9)
    erc.erc_set_wait_limit(1)
    seen = []
    for _ in range(TRIES):
        out = {}

        def call():
            out["r"] = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, prob, 50_000, 9)

        st = _status(call)
        assert st in (erc.ERC_OK, erc.ERC_ERR_TIMEOUT), st
        if st == erc.ERC_OK:  # a call that completed is exact
            assert torch.equal(out["r"][0], ref_nodes) and torch.equal(out["r"][1], ref_edges)
        seen.append(st)
    assert erc.ERC_ERR_TIMEOUT in seen, seen
    erc.erc_set_wait_limit(0)
    nodes, edges = erc.erc_sample_subgraph(g, erc.ERC_SAMPLE_NODES, prob, 50_000, 9)
    assert torch.equal(nodes, ref_nodes) and torch.equal(edges, ref_edges)


@pytest.mark.parametrize("mode", ["resident", "graph"])
def test_cg_wait_timeout_is_reported(mode):
    """resident: the single-launch solver's grid synchronisations; graph: the grid barrier of the
    multi-kernel path's fused vector update."""
    n, src, dst, w = synth.make_graph("sbm_n20000")
    g = erc.erc_build_laplacian(n, to_dev(src), to_dev(dst), to_dev(w))
    kc = 128
    Y = erc.erc_jl_rhs(g, synth.JL_SEED, kc, 0, kc)
    os.environ["ERC_CG_MODE"] = mode
    _, _, _, _, _, path = erc.erc_batched_cg_timed(g, 1e-3, Y, kc, 1e-6)
    assert path == (1 if mode == "resident" else 0)
    X0, it0, _, st0 = erc.erc_batched_cg(g, 1e-3, Y, kc, 1e-6)
    assert st0 == erc.ERC_OK
    erc.erc_set_wait_limit(1)
    seen = []
    for _ in range(TRIES):
        out = {}

        def call():
            out["r"] = erc.erc_batched_cg(g, 1e-3, Y, kc, 1e-6)

        st = _status(call)
        assert st in (erc.ERC_OK, erc.ERC_ERR_TIMEOUT), st
        if st == erc.ERC_OK:
            assert torch.equal(out["r"][0], X0)
        else:
            assert b"timed out" in erc.lib().erc_last_error()
        seen.append(st)
    assert erc.ERC_ERR_TIMEOUT in seen, seen
    erc.erc_set_wait_limit(0)
    X1, it1, _, st1 = erc.erc_batched_cg(g, 1e-3, Y, kc, 1e-6)
    assert st1 == erc.ERC_OK
    assert torch.equal(X1, X0) and torch.equal(it1, it0)


def test_wait_limit_is_exported_and_resets():
    erc.erc_set_wait_limit(5)
    erc.erc_set_wait_limit(0)
    n, src, dst, w = synth.random_connected(1000, 4000, seed=2)
    g, ref = build_both(n, src, dst, w)
    assert_graph_equal(g, ref)
    assert np.all(host(g.deg) == ref["deg"])
