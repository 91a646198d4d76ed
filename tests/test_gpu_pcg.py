"""GPU parity of the optional Jacobi-preconditioned solve (M = diag(L_eps) = deg + eps; not the
paper's solver) with the oracle's batched_pcg, on both solver paths that carry it (resident
cooperative, multi-kernel graph), and through erc_run with params.precond.

Same bars as the plain CG: R_hat per edge max relative error 1e-3 and median 1e-5 against the fp64
oracle on the same right-hand sides; iteration counts within 10 % + 2 of the oracle's.
"""
import numpy as np
import pytest
import torch

from oracle import erc_oracle as O
from paper_2609_27209_gb300 import erc, synth

from ._gpu import build_both, dev, host, to_dev

pytestmark = pytest.mark.gpu
PATHS = {"graph": 0, "resident": 1}


def _R(g, X, kc):
    R = torch.zeros(g.m, device=dev())
    erc.erc_edge_resistance(g, X, kc, R)
    return host(R)


def _check_R(R, Rr, max_rel=1e-3, med_rel=1e-5):
    rel = np.abs(R.astype(np.float64) - Rr) / Rr
    assert rel.max() <= max_rel and np.median(rel) <= med_rel, (rel.max(), np.median(rel))


@pytest.mark.parametrize("mode", list(PATHS))
@pytest.mark.parametrize("kc,weighted,heavy", [(16, True, False), (128, False, False),
                                               (64, True, True), (12, True, False)])
def test_pcg_paths_match_oracle(monkeypatch, mode, kc, weighted, heavy):
    monkeypatch.setenv("ERC_CG_MODE", mode)
    n, src, dst, w = synth.random_connected(4000, 16000, seed=kc + 1, weighted=weighted)
    if heavy:  # a hub joined to 3000 nodes: block-split rows and a wide spread of degrees
        src = np.concatenate([src, np.zeros(3000, np.int32)])
        dst = np.concatenate([dst, np.arange(1, 3001, dtype=np.int32)])
        if w is not None:
            w = np.concatenate([w, np.full(3000, 0.75, np.float32)])
    g, ref = build_both(n, src, dst, w)
    Y = erc.erc_jl_rhs(g, 9, 256, 0, kc)
    X, iters, relres, st, _, path = erc.erc_batched_pcg_timed(g, 1e-3, Y, kc, 1e-6)
    assert st == erc.ERC_OK and path == PATHS[mode]
    Xr, itr, _, ok = O.batched_pcg(ref, 1e-3, O.jl_rhs(ref, 9, 256, 0, kc), 1e-6)
    assert ok
    _check_R(_R(g, X, kc), O.edge_resistance(ref, Xr))
    assert np.all(np.abs(host(iters) - itr) <= 0.1 * itr + 2), (host(iters), itr)
    assert np.all(host(relres) <= (4e-6 if heavy else 2e-6))
    assert torch.all(X[:, kc:] == 0)


@pytest.mark.parametrize("mode", list(PATHS))
def test_pcg_cuts_iterations_on_a_power_law_graph(monkeypatch, mode):
    """On a Chung-Lu graph (exponent 2.2) the preconditioned solve reaches the same tolerance in
    far fewer iterations than plain CG, and both give the same resistances."""
    monkeypatch.setenv("ERC_CG_MODE", mode)
    n, src, dst, w = synth.chung_lu(3000, 2.2, 20000, "unit", 7)
    g, ref = build_both(n, src, dst, w)
    kc = 32
    Y = erc.erc_jl_rhs(g, 3, 32, 0, kc)
    Xc, itc, _, stc, _, pc_ = erc.erc_batched_cg_timed(g, 1e-3, Y, kc, 1e-6)
    Xp, itp, rrp, stp, _, pp = erc.erc_batched_pcg_timed(g, 1e-3, Y, kc, 1e-6)
    assert stc == erc.ERC_OK and stp == erc.ERC_OK and pp == PATHS[mode]
    assert host(itp).max() * 2 <= host(itc).min(), (host(itp), host(itc))
    Rc, Rp = _R(g, Xc, kc), _R(g, Xp, kc)
    np.testing.assert_allclose(Rp, Rc, rtol=1e-3)
    cols = np.arange(0, kc, 4)
    _, itr, _, _ = O.batched_pcg(ref, 1e-3, O.jl_rhs(ref, 3, 32, 0, kc)[:, cols], 1e-6)
    assert np.all(np.abs(host(itp)[cols] - itr) <= 0.1 * itr + 2)


def test_pcg_in_cluster_mode_takes_the_multi_kernel_path(monkeypatch):
    """The cluster solver has no preconditioner: restricted to it, the preconditioned solve runs
    on the multi-kernel path."""
    monkeypatch.setenv("ERC_CG_MODE", "cluster")
    n, src, dst, w = synth.random_connected(1500, 6000, seed=3, weighted=True)
    g, ref = build_both(n, src, dst, w)
    Y = erc.erc_jl_rhs(g, 9, 16, 0, 16)
    X, _, _, st, _, path = erc.erc_batched_pcg_timed(g, 1e-3, Y, 16, 1e-6)
    assert st == erc.ERC_OK and path == 0
    Xr, _, _, _ = O.batched_pcg(ref, 1e-3, O.jl_rhs(ref, 9, 16, 0, 16), 1e-6)
    _check_R(_R(g, X, 16), O.edge_resistance(ref, Xr))


def test_pcg_resident_without_p_in_shared_memory(monkeypatch):
    """12,000 nodes x 256 columns: the resident kernel keeps p in global memory only."""
    monkeypatch.setenv("ERC_CG_MODE", "resident")
    n, src, dst, w = synth.random_connected(12000, 36000, seed=31, weighted=True)
    g, ref = build_both(n, src, dst, w)
    kc = 256
    Y = erc.erc_jl_rhs(g, 9, 256, 0, kc)
    X, iters, relres, st, _, path = erc.erc_batched_pcg_timed(g, 1e-3, Y, kc, 1e-6)
    assert st == erc.ERC_OK and path == 1
    cols = np.arange(0, kc, 16)
    Xr, itr, _, _ = O.batched_pcg(ref, 1e-3, O.jl_rhs(ref, 9, 256, 0, kc)[:, cols], 1e-6)
    Xs = X[:, torch.as_tensor(cols, device=dev())].contiguous()
    _check_R(_R(g, Xs, len(cols)), O.edge_resistance(ref, Xr))
    assert np.all(np.abs(host(iters)[cols] - itr) <= 0.1 * itr + 2)
    assert np.all(host(relres) <= 2e-6)


@pytest.mark.parametrize("mode", list(PATHS))
def test_pcg_not_converged_and_zero_columns(monkeypatch, mode):
    monkeypatch.setenv("ERC_CG_MODE", mode)
    n, src, dst, w = synth.random_connected(1000, 3000, seed=5)
    g, _ = build_both(n, src, dst, w)
    Y = erc.erc_jl_rhs(g, 5, 16, 0, 16)
    Y[:, 3] = 0
    X, iters, _, st, _, path = erc.erc_batched_pcg_timed(g, 1e-3, Y, 16, 1e-6, max_iter=2)
    assert st == erc.ERC_ERR_NOT_CONVERGED and path == PATHS[mode]
    it = host(iters)
    assert it[3] == 0 and np.all(np.delete(it, 3) == 2)
    X, iters, relres, st, _, _ = erc.erc_batched_pcg_timed(g, 1e-3, Y, 16, 1e-6)
    assert st == erc.ERC_OK and host(iters)[3] == 0 and float(host(relres)[3]) == 0.0
    assert torch.all(X[:, 3] == 0)
    X, iters, relres, st, _, _ = erc.erc_batched_pcg_timed(g, 1e-3, torch.zeros_like(Y), 16, 1e-6)
    assert st == erc.ERC_OK and torch.all(iters == 0) and torch.all(relres == 0)
    assert torch.all(X == 0)


def test_run_with_jacobi_matches_oracle():
    """The whole path with params.precond = Jacobi against the oracle's erc_lg(precond="jacobi"),
    on the 2000-node ring-with-chords workload."""
    name = "ring_chords_n2000"
    wl = synth.WORKLOADS[name]
    n, src, dst, w = synth.make_graph(name)
    K = wl.K[0]
    prm = erc.Params(K=K, kc=wl.kc, eps=wl.eps, tol=wl.tol, seed=synth.JL_SEED,
                     precond=erc.ERC_PRECOND_JACOBI)
    out = erc.erc_run(n, to_dev(src), to_dev(dst), to_dev(w), prm)
    assert out["status"] == erc.ERC_OK
    ref = O.erc_lg(n, src, dst, w, K, wl.kc, wl.eps, wl.tol, synth.JL_SEED, precond="jacobi")
    _check_R(host(out["R"]), ref["R"])
    k, kr = host(out["kappa"]).astype(np.float64), ref["kappa"]
    assert np.abs(k - kr).max() <= 1e-3 * np.abs(kr).max()
    assert np.all(np.abs(host(out["iters"]) - ref["iters"]) <= 0.1 * ref["iters"] + 2)
    bad = erc.Params(K=K, kc=wl.kc, eps=wl.eps, tol=wl.tol, precond=7)
    with pytest.raises(erc.ErcError) as e:
        erc.erc_run(n, to_dev(src), to_dev(dst), to_dev(w), bad)
    assert e.value.status == erc.ERC_ERR_INVALID_ARG
