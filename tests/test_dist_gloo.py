"""Multi-rank column partition of Algorithm 1, on CPU with world-size-2 gloo ranks.

Each rank takes its own block of projection columns and the per-rank edge accumulators are summed
with one all-reduce; the result must equal a single rank running every column.  The per-rank
column work here is the CPU oracle (there is no GPU in these tests); the partition and the
aggregation are the library's own (paper_2609_27209_gb300.dist).
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2609_27209_gb300 import dist as edist

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, K, kc, out_path):
    import sys

    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from oracle import erc_oracle as O
        from paper_2609_27209_gb300 import synth

        n, src, dst, w = synth.random_connected(300, 900, seed=3)
        g = O.build_laplacian(n, src, dst, w)

        def shard_fn(c0, k, K_total):
            Y = O.jl_rhs(g, synth.JL_SEED, K_total, c0, k)
            X, _, _, _ = O.batched_cg(g, 1e-3, Y, 1e-10)
            return torch.from_numpy(O.edge_resistance(g, X))

        def allreduce(t):
            dist.all_reduce(t, op=dist.ReduceOp.SUM)
            return t

        R = edist.sharded_resistance(shard_fn, K, kc, world, rank, allreduce)
        np.save(f"{out_path}.{rank}.npy", R.numpy())
    finally:
        dist.destroy_process_group()


def test_shard_columns_cover_the_projection_once():
    for world in (1, 2, 3, 8):
        cols = []
        for rank in range(world):
            b, e, K_total = edist.shard_columns(16, world, rank)
            assert K_total == 16 * world
            for c0, k in edist.batches(b, e, 5):
                cols.extend(range(c0, c0 + k))
        assert cols == list(range(16 * world))
    with pytest.raises(ValueError):
        edist.shard_columns(16, 2, 2)


def test_two_gloo_ranks_sum_to_the_single_rank_result(tmp_path):
    from oracle import erc_oracle as O
    from paper_2609_27209_gb300 import synth

    K, kc, world = 16, 8, 2
    out = str(tmp_path / "R")
    mp.spawn(_worker, args=(world, _free_port(), K, kc, out), nprocs=world, join=True)
    R0 = np.load(out + ".0.npy")
    R1 = np.load(out + ".1.npy")
    np.testing.assert_array_equal(R0, R1)  # every rank holds the same aggregated result
    n, src, dst, w = synth.random_connected(300, 900, seed=3)
    ref = O.erc_lg(n, src, dst, w, K * world, kc, 1e-3, 1e-10, synth.JL_SEED)
    np.testing.assert_allclose(R0, ref["R"], rtol=1e-9)
