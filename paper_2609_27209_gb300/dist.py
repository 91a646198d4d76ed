"""Column-sharded ERC-LG across ranks (Algorithm 1's multi-GPU partition of the K projection columns).

Each rank owns a contiguous block of projection columns, runs the streamed batches of its block
on its own device through the C ABI, and the per-rank edge accumulators r^(g) are summed with one
all-reduce -- the only exchange in Algorithm 1 -- before curvature (Eq. 2) and the sampling
probabilities (§3.2) are formed (replicated on every rank).

Weak scaling: every rank owns `K` columns of a projection of total dimension K * world, so the
per-rank work is fixed as ranks are added.  With world = 1 this is exactly ``erc.erc_run``.
"""
from __future__ import annotations


def shard_columns(K_per_rank, world, rank):
    """(c_begin, c_end, K_total) of this rank's projection columns."""
    if world < 1 or not 0 <= rank < world or K_per_rank < 1:
        raise ValueError("bad shard request")
    return rank * K_per_rank, (rank + 1) * K_per_rank, K_per_rank * world


def batches(c_begin, c_end, kc):
    """The streamed column batches [c0, c0 + k) of one rank's block (Algorithm 1's inner loop)."""
    return [(c0, min(kc, c_end - c0)) for c0 in range(c_begin, c_end, kc)]


def sharded_resistance(shard_fn, K_per_rank, kc, world, rank, allreduce_sum):
    """Sum over ranks of each rank's batch contributions to R.

    shard_fn(c0, k, K_total) -> the R contribution of columns [c0, c0 + k) (a tensor or array);
    allreduce_sum(x) -> the elementwise sum of x over all ranks.
    """
    c_begin, c_end, K_total = shard_columns(K_per_rank, world, rank)
    R = None
    for c0, k in batches(c_begin, c_end, kc):
        part = shard_fn(c0, k, K_total)
        R = part if R is None else R + part
    return allreduce_sum(R)


def run_sharded(n, src, dst, w, params, world, rank, allreduce_sum):
    """The whole path on this rank's device, with the column block of `rank` out of `world`."""
    import torch

    from . import erc

    g = erc.erc_build_laplacian(n, src, dst, w, params.dup_policy)
    R = torch.zeros(max(g.m, 1), dtype=torch.float32, device=src.device)[:g.m]
    ld = erc.padded_ld(params.kc)
    ws = erc._workspace(erc.lib().erc_batched_cg_workspace_size(n, ld), src.device)
    Y = torch.empty(n, ld, dtype=torch.float32, device=src.device)
    X = torch.empty_like(Y)
    status = erc.ERC_OK

    solve = erc.erc_batched_pcg if params.precond == erc.ERC_PRECOND_JACOBI else erc.erc_batched_cg

    def shard_fn(c0, k, K_total):
        nonlocal status
        erc.erc_jl_rhs(g, params.seed, K_total, c0, k, ld=ld, out=Y)
        _, _, _, st = solve(g, params.eps, Y, k, params.tol, params.max_iter, X=X, ws=ws)
        status = max(status, st)
        erc.erc_edge_resistance(g, X, k, R)
        return R

    # shard_fn accumulates in place, so each batch returns the running sum: keep the last one
    c_begin, c_end, K_total = shard_columns(params.K, world, rank)
    for c0, k in batches(c_begin, c_end, params.kc):
        shard_fn(c0, k, K_total)
    R = allreduce_sum(R)
    p, kappa = erc.erc_curvature(g, R)
    pn, pe = erc.erc_sampling_probs(g, kappa, params.eta)
    return dict(m=g.m, eu=g.eu, ev=g.ev, R=R, p=p, kappa=kappa, prob_node=pn, prob_edge=pe,
                status=status)
