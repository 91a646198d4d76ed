"""The spawned per-column oracle runner used by the full-size GPU tests gives exactly what the
oracle computes when it solves the same columns in one process (Eq. 4-6 column by column)."""
import numpy as np

from oracle import erc_oracle as O
from paper_2609_27209_gb300 import synth

from ._oracle_pool import oracle_columns


def test_pool_equals_direct_oracle_solve():
    n, src, dst, w = synth.random_connected(500, 2000, seed=17, weighted=True)
    g = O.build_laplacian(n, src, dst, w)
    K, eps, tol = 64, 1e-3, 1e-8
    cols = [0, 9, 31, 63]
    res = oracle_columns(g, synth.JL_SEED, K, cols, eps, tol, procs=2)
    R = np.zeros(g["m"])
    for i, c in enumerate(cols):
        X, it, rr, ok = O.batched_cg(g, eps, O.jl_rhs(g, synth.JL_SEED, K, c, 1), tol)
        Rc = O.edge_resistance(g, X)
        R += Rc
        assert ok and res["iters"][i] == it[0]
        assert res["relres"][i] == rr[0]
        assert res["foster"][i] == np.dot(g["ew"].astype(np.float64), Rc)
    assert res["converged"]
    np.testing.assert_allclose(res["R"], R, rtol=1e-13)
    # columns solved in one batch give the same per-column results (the systems are independent)
    Xb, itb, _, _ = O.batched_cg(g, eps, np.concatenate(
        [O.jl_rhs(g, synth.JL_SEED, K, c, 1) for c in cols], axis=1), tol)
    np.testing.assert_array_equal(itb, res["iters"])
    np.testing.assert_allclose(O.edge_resistance(g, Xb), R, rtol=1e-10)
