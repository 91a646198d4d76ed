"""Pins for the oracle's projection signs (§3.1.2: Q entries uniform on {+-1/sqrt(K)}).

The Philox4x32-10 block function is checked against an independent implementation: cuRAND's host
(CPU-side) Philox4_32_10 generator, run as a library.  With the default ordering that generator
emits output block b from counter (b >> 16, 0, b & 0xffff, 0) under key (seed_lo, seed_hi), which
covers counter words 0 and 2 -- the words that carry the column group and the edge id here.
Statistical checks pin what the method needs from Q: balanced, uncorrelated signs.
"""
import ctypes
import ctypes.util
import os

import numpy as np
import pytest

from oracle import erc_oracle as O


def _curand():
    for cand in [os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "lib64",
                              "libcurand.so"), ctypes.util.find_library("curand")]:
        if cand:
            try:
                return ctypes.CDLL(cand)
            except OSError:
                pass
    return None


@pytest.mark.parametrize("seed", [0xE2C1, 0x0123456789ABCDEF, 0xFFFFFFFF00000001])
def test_philox_matches_curand_host_generator(seed):
    lib = _curand()
    if lib is None:
        pytest.skip("libcurand not available")
    gen = ctypes.c_void_p()
    CURAND_RNG_PSEUDO_PHILOX4_32_10 = 161
    if lib.curandCreateGeneratorHost(ctypes.byref(gen), CURAND_RNG_PSEUDO_PHILOX4_32_10) != 0:
        pytest.skip("cuRAND host generator unavailable")
    try:
        assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        nblk = 3 << 16  # counter word 0 takes the values 0, 1, 2
        out = np.zeros(4 * nblk, np.uint32)
        assert lib.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p),
                                  ctypes.c_size_t(out.size)) == 0
    finally:
        lib.curandDestroyGenerator(gen)
    b = np.arange(nblk, dtype=np.int64)
    words = O.philox4x32_10((b >> 16, 0, b & 0xFFFF, 0), (seed & 0xFFFFFFFF, seed >> 32))
    np.testing.assert_array_equal(np.stack(words, axis=1).ravel(), out)


def test_sign_balance_and_independence():
    seed, K = 0xE2C1, 256
    e = np.arange(20000)
    bits = O.jl_sign_bits(seed, e[:, None], np.arange(K)[None, :]).astype(np.float64)
    s = 1.0 - 2.0 * bits
    N = s.size
    assert abs(s.mean()) < 5.0 / np.sqrt(N)
    # every column balanced
    assert np.max(np.abs(s.mean(axis=0))) < 5.0 / np.sqrt(e.size) * 1.3
    # Q^T Q close to I: off-diagonals of (1/m) S^T S are ~ N(0, 1/m)
    C = s.T @ s / e.size
    off = C[~np.eye(K, dtype=bool)]
    assert np.max(np.abs(off)) < 6.0 / np.sqrt(e.size)
    np.testing.assert_allclose(np.diag(C), 1.0)
    # consecutive edges uncorrelated too
    assert abs(np.mean(s[1:] * s[:-1])) < 5.0 / np.sqrt(N)


def test_q_scale_uses_total_dimension():
    q = O.jl_q(7, 1024, np.arange(5), 128, 16)
    np.testing.assert_allclose(np.abs(q), 1.0 / 32.0)
    # a column's value does not depend on the batch it is produced in
    a = O.jl_q(7, 1024, np.arange(50), 100, 60)
    b = O.jl_q(7, 1024, np.arange(50), 130, 30)
    np.testing.assert_array_equal(a[:, 30:], b)
