"""The library's multi-rank path on one GPU: paper_2609_27209_gb300.dist.run_sharded, which is
what bench.py runs under torchrun (Algorithm 1: each rank solves its own block of projection
columns, the per-rank edge accumulators r^(g) are summed, R = sum_g r^(g), then Eq. 2 and §3.2).

Ranks 0 and 1 of a world of 2 run one after the other on the same device; the all-reduce is a
host-side stand-in.  A first pass records each rank's accumulator; a second pass hands every rank
the sum, as a sum all-reduce would, so that curvature and probabilities come from the combined R.
The summed R, and kappa and the probabilities of both ranks, must match the float64 oracle run on
all 2K columns of the same projection (spec tolerances).
"""
import numpy as np
import pytest
import torch

from oracle import erc_oracle as O
from paper_2609_27209_gb300 import dist as edist
from paper_2609_27209_gb300 import erc, synth

from ._gpu import host, to_dev

pytestmark = pytest.mark.gpu


def test_run_sharded_ranks_in_turn_match_the_oracle():
    n, src, dst, w = synth.random_connected(3000, 12000, seed=61, weighted=True)
    src_d, dst_d, w_d = to_dev(src), to_dev(dst), to_dev(w)
    world, K, kc, eps, tol = 2, 32, 16, 1e-3, 1e-6
    prm = erc.Params(K=K, kc=kc, eps=eps, tol=tol, seed=synth.JL_SEED)

    partial = {}

    def keep(rank):
        def allreduce(t):
            partial[rank] = t.clone()
            return t
        return allreduce

    for rank in range(world):
        out = edist.run_sharded(n, src_d, dst_d, w_d, prm, world, rank, keep(rank))
        assert out["status"] == erc.ERC_OK
    total = partial[0] + partial[1]

    outs = []
    for rank in range(world):
        def allreduce(t, rank=rank):
            assert torch.equal(t, partial[rank])  # the rank's accumulator is deterministic
            t.copy_(total)
            return t
        outs.append(edist.run_sharded(n, src_d, dst_d, w_d, prm, world, rank, allreduce))

    ref = O.erc_lg(n, src, dst, w, K * world, kc, eps, tol, synth.JL_SEED)
    assert ref["converged"]
    R = host(outs[0]["R"]).astype(np.float64)
    rel = np.abs(R - ref["R"]) / ref["R"]
    assert rel.max() <= 1e-3 and np.median(rel) <= 1e-5, (rel.max(), np.median(rel))
    # each rank's own block is a different part of the projection: neither alone is R
    for rank in range(world):
        assert not np.allclose(host(partial[rank]), ref["R"], rtol=1e-2)
    kap = host(outs[0]["kappa"]).astype(np.float64)
    assert np.max(np.abs(kap - ref["kappa"])) <= 1e-3 * np.max(np.abs(ref["kappa"]))
    np.testing.assert_allclose(host(outs[0]["prob_node"]), ref["prob_node"], rtol=2e-3,
                               atol=1e-9)
    np.testing.assert_allclose(host(outs[0]["prob_edge"]), ref["prob_edge"], rtol=2e-3)
    for key in ("R", "p", "kappa", "prob_node", "prob_edge"):  # every rank holds the same result
        assert torch.equal(outs[0][key], outs[1][key]), key


def test_shards_cover_the_projection_in_order():
    """Rank g's batches are exactly the columns [g K, (g + 1) K) of the K * world projection, so
    the sum of the two ranks' accumulators equals one rank running every column."""
    n, src, dst, w = synth.random_connected(800, 3000, seed=62)
    src_d, dst_d = to_dev(src), to_dev(dst)
    prm1 = erc.Params(K=16, kc=8, eps=1e-3, tol=1e-7, seed=synth.JL_SEED)
    prm2 = erc.Params(K=32, kc=8, eps=1e-3, tol=1e-7, seed=synth.JL_SEED)
    parts = [edist.run_sharded(n, src_d, dst_d, None, prm1, 2, r, lambda t: t)["R"]
             for r in range(2)]
    whole = edist.run_sharded(n, src_d, dst_d, None, prm2, 1, 0, lambda t: t)["R"]
    torch.testing.assert_close(parts[0] + parts[1], whole, rtol=1e-6, atol=0)
