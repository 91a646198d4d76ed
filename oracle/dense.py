"""Dense fp64 helpers for small graphs -- TEST INFRASTRUCTURE ONLY (n up to a few thousand).

Only the test-suite and the benchmark's CPU-baseline leg use this module; the CUDA library never
does.  Each function is the plain matrix definition the paper gives:

* ``dense_laplacian``        -- L = B^T W B (§3.1.1) from the oriented incidence matrix.
* ``exact_resistance``       -- R_uv = b_uv^T L^+ b_uv with the Moore-Penrose pseudoinverse (Eq. 1).
* ``regularized_resistance`` -- b_uv^T (L + eps I)^{-1} b_uv, the diagonal-perturbation scheme the
  paper calls ERC-REG (§3.1.3, Table 3).
* ``jl_dense_solve``         -- Z_eps = (L + eps I)^{-1} Y by a direct solve: the paper's ERC-JL
  comparison (JL projection without CG, Table 3).
* ``jl_expected_resistance`` -- the exact mean over Q of the JL estimate with exact solves,
  E[R_uv] = b^T L_eps^{-1} L L_eps^{-1} b, since E[Q Q^T] = I for entries +-1/sqrt(K).
"""
from __future__ import annotations

import numpy as np


def dense_incidence(n, eu, ev):
    """B in R^{m x n}: row e is e_u - e_v (§3.1.1)."""
    m = len(eu)
    B = np.zeros((m, n))
    B[np.arange(m), eu] = 1.0
    B[np.arange(m), ev] = -1.0
    return B


def dense_laplacian(n, eu, ev, ew):
    """L = B^T W B (§3.1.1)."""
    B = dense_incidence(n, eu, ev)
    return B.T @ (np.asarray(ew, np.float64)[:, None] * B)


def _pairs(n, eu, ev):
    B = dense_incidence(n, eu, ev)
    return B


def exact_resistance(L, eu, ev):
    """R_e = b_e^T L^+ b_e (Eq. 1)."""
    Lp = np.linalg.pinv(L, hermitian=True)
    B = _pairs(L.shape[0], eu, ev)
    return np.einsum("ij,jk,ik->i", B, Lp, B)


def regularized_resistance(L, eps, eu, ev):
    """b_e^T (L + eps I)^{-1} b_e: ERC-REG's diagonal perturbation (§3.1.3)."""
    n = L.shape[0]
    Li = np.linalg.inv(L + eps * np.eye(n))
    B = _pairs(n, eu, ev)
    return np.einsum("ij,jk,ik->i", B, Li, B)


def jl_dense_solve(L, eps, Y):
    """Z_eps = (L + eps I)^{-1} Y by a direct solve (ERC-JL in Table 3)."""
    return np.linalg.solve(L + eps * np.eye(L.shape[0]), Y)


def jl_expected_resistance(L, eps, eu, ev):
    """E_Q[ ||b_e^T L_eps^{-1} B^T W^{1/2} Q||^2 ] = b_e^T L_eps^{-1} L L_eps^{-1} b_e."""
    n = L.shape[0]
    Li = np.linalg.inv(L + eps * np.eye(n))
    M = Li @ L @ Li
    B = _pairs(n, eu, ev)
    return np.einsum("ij,jk,ik->i", B, M, B)


def jl_resistance_std(L, eps, eu, ev, ew, K):
    """Exact standard deviation of the JL estimate of each edge with exact solves.

    With a_e = W^{1/2} B L_eps^{-1} b_e and i.i.d. +-1/sqrt(K) entries,
    Var = (2/K) (||a_e||_2^4 - ||a_e||_4^4).
    """
    n = L.shape[0]
    Li = np.linalg.inv(L + eps * np.eye(n))
    B = dense_incidence(n, eu, ev)
    A = (np.sqrt(np.asarray(ew, np.float64))[:, None] * B) @ Li @ B.T  # column e is a_e
    s2 = np.sum(A * A, axis=0)
    s4 = np.sum(A ** 4, axis=0)
    return np.sqrt(2.0 / K * (s2 * s2 - s4))
