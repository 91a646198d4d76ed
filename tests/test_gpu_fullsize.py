"""Full-size checks on the three large workloads, in the launch shapes bench.py times.

Every workload runs at its largest projection dimension K in batches of its kc columns, as
bench.py does: 169k nodes at K = 256 in one batch, 233k nodes at K = 128 in batches of 32, 2.45M
nodes at K = 1024 in batches of 128 (plus the smaller K = 64 and 256 of that workload's sweep).

Against the float64 oracle (one spawned process per column, tests/_oracle_pool.py):
  * the first batch [0, kc) is solved on the GPU exactly as inside erc_run; on 8-16 columns spread
    over it the per-edge resistances (Eq. 6 summed over those columns) must match the oracle's to
    a relative error of 1e-3 (max) and 1e-5 (median), and the iteration counts must agree;
  * the CSR rows of sampled nodes and the canonical edge list are bit-exact, Philox signs of
    sampled edges bit-exact, rows of Y within float32 rounding (first and last batch).
At any size, on the whole K-column run:
  * the true residual of the returned solution, curvature consistent with the resistances (Eq. 2),
    probabilities that sum to 1;
  * Foster's theorem in expectation: sum_e w_e R_e equals K times the oracle's mean per-column
    Foster sum within six standard deviations of the JL estimate (each column's sum has standard
    deviation at most sqrt(2 (n - 1)) / K), and never exceeds n - 1 beyond that.
"""
import numpy as np
import pytest
import torch

from oracle import erc_oracle as O
from paper_2609_27209_gb300 import erc, synth

from ._gpu import host, to_dev
from ._oracle_pool import oracle_columns

pytestmark = pytest.mark.gpu
LARGE = ["chung_lu_n169343_g2.5", "chung_lu_n232965_g2.1", "chung_lu_n2449029_g2.3"]
U32 = 2.0 ** -24
ORACLE_COLUMNS = {"chung_lu_n169343_g2.5": 16, "chung_lu_n232965_g2.1": 8,
                  "chung_lu_n2449029_g2.3": 8}


def bench_shape(wl, K=None):
    """(K, kc) of bench.py's run of workload wl: its largest K, batches of its kc columns."""
    K = max(wl.K) if K is None else K
    return K, min(wl.kc, K)


@pytest.fixture(scope="module", params=LARGE)
def big(request):
    name = request.param
    wl = synth.WORKLOADS[name]
    n, src, dst, w = synth.make_graph(name)
    K, kc = bench_shape(wl)
    prm = erc.Params(K=K, kc=kc, eps=wl.eps, tol=wl.tol, seed=synth.JL_SEED)
    src_d, dst_d, w_d = to_dev(src), to_dev(dst), to_dev(w)
    out = erc.erc_run(n, src_d, dst_d, w_d, prm)
    g = erc.erc_build_laplacian(n, src_d, dst_d, w_d)
    torch.cuda.synchronize()
    keys = np.sort(np.minimum(src, dst).astype(np.int64) * n + np.maximum(src, dst))
    keys = keys[np.concatenate([[True], keys[1:] != keys[:-1]])]  # distinct pairs, ascending
    rng = np.random.default_rng(7)
    rp = host(g.row_ptr)
    deg = np.diff(rp)
    S = np.unique(np.concatenate([rng.integers(0, n, 300), [0, n - 1, int(np.argmax(deg))]]))
    yield dict(name=name, wl=wl, n=n, src=src, dst=dst, w=w, src_d=src_d, dst_d=dst_d, w_d=w_d,
               prm=prm, out=out, g=g, keys=keys, rp=rp, S=S)
    del out, g
    torch.cuda.empty_cache()


@pytest.fixture(scope="module")
def chunk(big):
    """The first batch [0, kc) solved on the GPU as erc_run solves it."""
    g, prm = big["g"], big["prm"]
    Y = erc.erc_jl_rhs(g, prm.seed, prm.K, 0, prm.kc)
    X, iters, relres, st = erc.erc_batched_cg(g, prm.eps, Y, prm.kc, prm.tol)
    yield dict(Y=Y, X=X, iters=host(iters), relres=host(relres), status=st)
    del Y, X
    torch.cuda.empty_cache()


@pytest.fixture(scope="module")
def ora(big):
    """The oracle on columns spread over the first batch of the same projection."""
    prm = big["prm"]
    cols = np.unique(np.linspace(0, prm.kc - 1, ORACLE_COLUMNS[big["name"]]).round().astype(int))
    ref = O.build_laplacian(big["n"], big["src"], big["dst"], big["w"])
    res = oracle_columns(ref, prm.seed, prm.K, cols, prm.eps, prm.tol)
    res["cols"] = cols
    res["graph"] = ref
    return res


def test_canonical_edges_and_sampled_rows_bit_exact(big):
    n, g, keys, rp, S = big["n"], big["g"], big["keys"], big["rp"], big["S"]
    assert g.m == keys.size
    eu, ev = host(g.eu).astype(np.int64), host(g.ev).astype(np.int64)
    np.testing.assert_array_equal(eu * n + ev, keys)  # every unique pair, u < v, lexicographic
    if big["w"] is not None:  # the generators emit no duplicates: ew is the input weight
        ikeys = np.minimum(big["src"], big["dst"]).astype(np.int64) * n + np.maximum(big["src"], big["dst"])
        order = np.argsort(ikeys)
        np.testing.assert_array_equal(host(g.ew), big["w"][order])
    src, dst, w = big["src"], big["dst"], big["w"]
    keep = np.isin(src, S) | np.isin(dst, S)
    sub = O.build_laplacian(n, src[keep], dst[keep], None if w is None else w[keep])
    col = host(g.col)
    val = host(g.val)
    eid = host(g.csr_eid)
    gdeg = host(g.deg)
    srp = sub["row_ptr"]
    for u in S:
        a, b = rp[u], rp[u + 1]
        sa, sb = srp[u], srp[u + 1]
        np.testing.assert_array_equal(col[a:b], sub["col"][sa:sb])
        np.testing.assert_array_equal(val[a:b], sub["val"][sa:sb])
        assert gdeg[u] == sub["deg"][u]
        lo = np.minimum(u, col[a:b]).astype(np.int64)
        hi = np.maximum(u, col[a:b]).astype(np.int64)
        np.testing.assert_array_equal(eid[a:b], np.searchsorted(keys, lo * n + hi))


def test_signs_and_rhs_rows(big):
    n, g, keys, S, prm = big["n"], big["g"], big["keys"], big["S"], big["prm"]
    m, K, kc = g.m, prm.K, prm.kc
    for e0, e1 in [(0, 512), (m - 512, m)]:
        got = host(erc.erc_philox_signs(prm.seed, e0, e1, 0, K))
        np.testing.assert_array_equal(got, O.jl_sign_bits(prm.seed, np.arange(e0, e1)[:, None],
                                                          np.arange(K)[None, :]))
    src, dst, w = big["src"], big["dst"], big["w"]
    keep = np.isin(src, S) | np.isin(dst, S)
    sub = O.build_laplacian(n, src[keep], dst[keep], None if w is None else w[keep])
    ids = np.searchsorted(keys, sub["eu"].astype(np.int64) * n + sub["ev"])
    srp = sub["row_ptr"]
    for c0 in sorted({0, K - kc}):  # the first and the last streamed batch
        Y = host(erc.erc_jl_rhs(g, prm.seed, K, c0, kc))
        Yr = O.jl_rhs(sub, prm.seed, K, c0, kc, edge_ids=ids)
        for u in S:
            sw = np.sqrt(sub["val"][srp[u]:srp[u + 1]].astype(np.float64)) / np.sqrt(K)
            bound = (4 + srp[u + 1] - srp[u]) * U32 * sw.sum()
            assert np.all(np.abs(Y[u, :kc] - Yr[u]) <= bound + 1e-30), (c0, u)


def test_first_batch_matches_oracle(big, chunk, ora):
    """The bench's first batch, solved in the bench's launch shape, against the float64 oracle on
    the same columns: per-edge R over those columns and the iteration counts."""
    g, prm = big["g"], big["prm"]
    assert chunk["status"] == erc.ERC_OK
    assert ora["converged"]
    cols = ora["cols"]
    XS = chunk["X"][:, torch.as_tensor(cols, device=chunk["X"].device)].contiguous()
    ldS = erc.padded_ld(len(cols))
    if ldS != len(cols):
        XS = torch.nn.functional.pad(XS, (0, ldS - len(cols))).contiguous()
    Rg = torch.zeros(g.m, device="cuda:0")
    erc.erc_edge_resistance(g, XS, len(cols), Rg)
    Rr = ora["R"]
    rel = np.abs(host(Rg).astype(np.float64) - Rr) / Rr
    print(f"\n{big['name']}: batch [0, {prm.kc}), oracle columns {cols.tolist()}: R max rel "
          f"{rel.max():.2e}, median {np.median(rel):.2e}; iterations GPU "
          f"{chunk['iters'][cols].tolist()} oracle {ora['iters'].tolist()}")
    assert rel.max() <= 1e-3 and np.median(rel) <= 1e-5, (rel.max(), np.median(rel))
    itg = chunk["iters"][cols]
    assert np.all(np.abs(itg - ora["iters"]) <= 0.1 * ora["iters"] + 3)


def _foster_bounds(n, K, n_cols):
    """Six standard deviations of (sum_e w_e R_e over K columns) - K * (mean per-column Foster
    sum over n_cols other columns): one column's sum is s^T M s / K with s a sign vector and
    ||M||_F^2 <= n - 1, so its variance is at most 2 (n - 1) / K^2."""
    return 6.0 * (np.sqrt(2.0 * (n - 1) / K) + np.sqrt(2.0 * (n - 1) / n_cols))


def _check_run(name, n, g, prm, out, ora):
    assert out["status"] == erc.ERC_OK, out["status"]
    assert float(out["relres"].max()) <= 2 * prm.tol
    R = host(out["R"]).astype(np.float64)
    assert np.all(np.isfinite(R)) and np.all(R > 0)
    ew = host(g.ew).astype(np.float64) if not g.unit_weights else np.ones(g.m)
    eu, ev = host(out["eu"]), host(out["ev"])
    # Eq. 2 consistency on the full outputs (float64 recomputation from the returned R)
    half = 0.5 * (np.bincount(eu, weights=ew * R, minlength=n) +
                  np.bincount(ev, weights=ew * R, minlength=n))
    p = host(out["p"]).astype(np.float64)
    assert np.all(np.abs(p - (1.0 - half)) <= 8 * U32 * (1.0 + half))
    kappa = host(out["kappa"]).astype(np.float64)
    kref = 2.0 * (p[eu] + p[ev]) / R
    assert np.all(np.abs(kappa - kref) <=
                  4 * U32 * (np.abs(kref) + 2 * (np.abs(p[eu]) + np.abs(p[ev])) / R))
    assert abs(out["prob_node"].double().sum().item() - 1) < 1e-5
    assert abs(out["prob_edge"].double().sum().item() - 1) < 1e-5
    # Foster in expectation: the oracle's columns of the K_o-column projection estimate
    # E[sum_e w_e R_e] = n - 1 - (regularisation deficit), independently of K
    tot = float(np.dot(ew, R))
    K_o = ora["K"]
    mu = K_o * float(ora["foster"].mean())
    bound = _foster_bounds(n, prm.K, len(ora["foster"]))
    print(f"\n{name} K={prm.K}: sum w R = {tot:.1f}, oracle estimate {mu:.1f} "
          f"(n - 1 = {n - 1}, deficit {n - 1 - mu:.1f}), bound {bound:.1f}")
    assert abs(tot - mu) <= bound
    assert tot <= (n - 1) + 6.0 * np.sqrt(2.0 * (n - 1) / prm.K)


def test_solution_residual_and_curvature_properties(big, chunk, ora):
    """The whole run at the largest K, and the workload's smaller projections of its K sweep
    (the 2.45M-node graph: K = 64 in one batch, K = 256 in two batches of 128), each with the
    sampling epilogue."""
    n, g, prm, out = big["n"], big["g"], big["prm"], big["out"]
    # independent check of one batch: ||y - L_eps x|| / ||y|| through the operator kernel
    Y, X = chunk["Y"], chunk["X"]
    AX, _ = erc.erc_laplacian_apply(g, prm.eps, X, prm.kc)
    res = (Y - AX).double().norm(dim=0) / Y.double().norm(dim=0)
    assert float(res[:prm.kc].max()) <= 2 * prm.tol, float(res.max())
    del AX
    ora["K"] = prm.K  # the oracle's columns belong to the largest projection
    _check_run(big["name"], n, g, prm, out, ora)
    wl = big["wl"]
    for Ks in sorted(set(wl.K) - {prm.K}):
        K, kc = bench_shape(wl, Ks)
        p2 = erc.Params(K=K, kc=kc, eps=wl.eps, tol=wl.tol, seed=synth.JL_SEED)
        out2 = erc.erc_run(n, big["src_d"], big["dst_d"], big["w_d"], p2)
        _check_run(big["name"], n, g, p2, out2, ora)
        del out2


def test_jacobi_pcg_full_size(big, chunk):
    """The optional Jacobi-preconditioned solve of the first batch in the configuration bench.py
    times: its true residual meets tau, it needs far fewer iterations than plain CG on these
    power-law graphs, and its resistances equal plain CG's; on the 169k-node graph a column
    subset also matches the oracle's preconditioned solve."""
    n, g, prm = big["n"], big["g"], big["prm"]
    Y, Xc, itc = chunk["Y"], chunk["X"], chunk["iters"]
    Xp, itp, rrp, stp = erc.erc_batched_pcg(g, prm.eps, Y, prm.kc, prm.tol)
    assert stp == erc.ERC_OK
    AX, _ = erc.erc_laplacian_apply(g, prm.eps, Xp, prm.kc)
    res = (Y - AX).double().norm(dim=0) / Y.double().norm(dim=0)
    assert float(res[:prm.kc].max()) <= 2 * prm.tol, float(res.max())
    del AX
    assert 2 * int(itp.max()) <= int(itc.min()), (int(itp.max()), int(itc.min()))
    Rc = torch.zeros(g.m, device="cuda:0")
    Rp = torch.zeros(g.m, device="cuda:0")
    erc.erc_edge_resistance(g, Xc, prm.kc, Rc)
    erc.erc_edge_resistance(g, Xp, prm.kc, Rp)
    # both solves stop at ||r|| <= tau ||y||: their resistances differ by O(tau) (the bars of
    # the oracle parity tests, 1e-3 max and 1e-5 median at tau = 1e-6, scaled with tau)
    rel = (Rp.double() - Rc.double()).abs() / Rc.double()
    print(f"\n{big['name']}: PCG {int(itp.max())} vs CG {int(itc.max())} iterations; "
          f"R max rel {float(rel.max()):.2e}, median {float(rel.median()):.2e}")
    assert float(rel.max()) <= 1e3 * prm.tol and float(rel.median()) <= 10 * prm.tol
    del Xp, Rc, Rp, rel
    if big["name"] == "chung_lu_n169343_g2.5":
        ref = O.build_laplacian(n, big["src"], big["dst"], big["w"])
        cols = np.arange(8)
        r = oracle_columns(ref, prm.seed, prm.K, cols, prm.eps, prm.tol, precond=True)
        Xs, its, _, st = erc.erc_batched_pcg(g, prm.eps, Y[:, :8].contiguous(), 8, prm.tol)
        assert st == erc.ERC_OK and r["converged"]
        Rg = torch.zeros(g.m, device="cuda:0")
        erc.erc_edge_resistance(g, Xs, 8, Rg)
        rel = np.abs(host(Rg).astype(np.float64) - r["R"]) / r["R"]
        assert rel.max() <= 1e-3 and np.median(rel) <= 1e-5, (rel.max(), np.median(rel))
        assert np.all(np.abs(host(its) - r["iters"]) <= 0.1 * r["iters"] + 3)
