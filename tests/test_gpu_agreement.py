"""Curvature agreement study in the style of the paper's SBM accuracy table (§4): ERC-REG (the
regularised resistance, dense), ERC-JL (the dense solve of the same projected systems) and the
GPU's ERC-LG (CG, Algorithm 1) against exact resistance curvature from the pseudoinverse (Eq. 1,
Eq. 2), on a 1,000-node graph drawn like the 20k-node SBM workload, at K = 1024, 2048 and 4096.

Reported per method and K: mean absolute curvature error, Spearman rank correlation and the
fraction of edges whose curvature sign agrees with the exact one.  Checked: ERC-LG reproduces
ERC-JL's errors (CG to tau on the same Y), the JL error falls like 1/sqrt(K), and rank and sign
agreement grow with K.  The paper's own numbers are for an SBM of unstated size and are not
expected to match.
"""
import numpy as np
import pytest
from scipy.stats import spearmanr

from oracle import dense as D
from oracle import erc_oracle as O
from paper_2609_27209_gb300 import erc, synth

from ._gpu import host, to_dev

pytestmark = pytest.mark.gpu
EPS, TOL = 1e-3, 1e-6


def _metrics(k, k_exact):
    return (float(np.mean(np.abs(k - k_exact))), float(spearmanr(k, k_exact).statistic),
            float(np.mean(np.sign(k) == np.sign(k_exact))))


def test_curvature_agreement_with_exact_erc():
    n, src, dst, w = synth.sbm(1000, 10, 8.0, 0.5, 0.5, seed=2)
    g = O.build_laplacian(n, src, dst, w)
    L = D.dense_laplacian(n, g["eu"], g["ev"], g["ew"])
    _, k_exact = O.curvature(g, D.exact_resistance(L, g["eu"], g["ev"]))
    _, k_reg = O.curvature(g, D.regularized_resistance(L, EPS, g["eu"], g["ev"]))
    rows = [("ERC-REG", "-", *_metrics(k_reg, k_exact))]
    table = {}
    for K in (1024, 2048, 4096):
        X = D.jl_dense_solve(L, EPS, O.jl_rhs(g, synth.JL_SEED, K, 0, K))
        _, k_jl = O.curvature(g, O.edge_resistance(g, X))
        prm = erc.Params(K=K, kc=128, eps=EPS, tol=TOL, seed=synth.JL_SEED)
        out = erc.erc_run(n, to_dev(src), to_dev(dst), to_dev(w), prm)
        assert out["status"] == erc.ERC_OK
        k_lg = host(out["kappa"]).astype(np.float64)
        table[K] = (_metrics(k_jl, k_exact), _metrics(k_lg, k_exact))
        rows.append(("ERC-JL", K, *table[K][0]))
        rows.append(("ERC-LG", K, *table[K][1]))
    print(f"\nn={n} m={g['m']} eps={EPS} tau={TOL}")
    print(f"{'method':8s} {'K':>5s} {'MAE':>9s} {'Spearman':>9s} {'sign':>7s}")
    for name, K, mae, rho, sign in rows:
        print(f"{name:8s} {K!s:>5s} {mae:9.5f} {rho:9.4f} {sign:7.4f}")

    assert rows[0][2] < 0.1 * table[4096][0][0]  # the regularisation error is negligible
    for K in table:
        (mae_jl, rho_jl, s_jl), (mae_lg, rho_lg, s_lg) = table[K]
        assert abs(mae_lg - mae_jl) <= 0.02 * mae_jl, (K, mae_lg, mae_jl)
        assert abs(rho_lg - rho_jl) <= 0.01 and abs(s_lg - s_jl) <= 0.01
    maes = [table[K][1][0] for K in (1024, 2048, 4096)]
    assert maes[0] > maes[1] > maes[2]
    assert 1.5 <= maes[0] / maes[2] <= 2.8, maes  # 1/sqrt(K): a factor 2 over K x 4
    rhos = [table[K][1][1] for K in (1024, 2048, 4096)]
    signs = [table[K][1][2] for K in (1024, 2048, 4096)]
    assert rhos[0] < rhos[1] < rhos[2] and signs[0] <= signs[2]
