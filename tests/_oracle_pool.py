"""Oracle CG on chosen projection columns of a large graph, one spawned process per column.

Test infrastructure.  The K systems of Eq. 4 / Eq. 5 are independent, so the float64 oracle
(`oracle.erc_oracle`) can solve any subset of columns, each on its own; on the multi-million-edge
workloads one column takes minutes in numpy/scipy, so the columns run in parallel processes.  The
pool is started with the "spawn" method (a process forked after CUDA has been initialised would
hang) and its workers import numpy, scipy and the oracle only.  The oracle graph travels through
.npy files; each worker adds its column's squared edge differences (Eq. 6) into one shared float64
accumulator under a lock and returns its iteration count, true residual and Foster sum
sum_e w_e (x_u - x_v)^2.
"""
from __future__ import annotations

import multiprocessing as mp
import os
import tempfile
from multiprocessing import shared_memory

import numpy as np

_KEYS = ("row_ptr", "col", "val", "deg", "csr_eid", "eu", "ev", "ew")
_lock = None


def _init(lock):
    global _lock
    _lock = lock
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[k] = "1"


def _load_graph(d):
    g = {k: np.load(os.path.join(d, k + ".npy"), mmap_mode="r") for k in _KEYS}
    n, m = np.load(os.path.join(d, "nm.npy"))
    g["n"], g["m"] = int(n), int(m)
    return g


def _solve_column(task):
    d, seed, K, c, eps, tol, shm_name, precond = task
    from oracle import erc_oracle as O

    g = _load_graph(d)
    Y = O.jl_rhs(g, seed, K, c, 1)
    solve = O.batched_pcg if precond else O.batched_cg
    X, it, relres, ok = solve(g, eps, Y, tol)
    R = O.edge_resistance(g, X)
    foster = float(np.dot(np.asarray(g["ew"], dtype=np.float64), R))
    shm = shared_memory.SharedMemory(name=shm_name)
    acc = None
    try:
        acc = np.ndarray((g["m"],), dtype=np.float64, buffer=shm.buf)
        with _lock:
            acc += R
    finally:
        acc = None  # the view must go before the mapping is closed
        shm.close()
    return c, int(it[0]), float(relres[0]), bool(ok), foster


def oracle_columns(g, seed, K, cols, eps, tol, procs=None, precond=False):
    """Solve the oracle's columns `cols` of the K-column projection on graph `g` (an
    `oracle.erc_oracle.build_laplacian` dict).  Returns a dict with R (float64 [m], the sum over
    `cols` of Eq. 6's squared differences), iters, relres, foster (per column, in `cols` order)
    and converged."""
    cols = [int(c) for c in cols]
    procs = max(1, min(len(cols), procs or os.cpu_count() or 1))
    m = int(g["m"])
    with tempfile.TemporaryDirectory() as d:
        for k in _KEYS:
            np.save(os.path.join(d, k + ".npy"), np.ascontiguousarray(g[k]))
        np.save(os.path.join(d, "nm.npy"), np.array([g["n"], m], dtype=np.int64))
        shm = shared_memory.SharedMemory(create=True, size=max(8, 8 * m))
        acc = None
        try:
            acc = np.ndarray((m,), dtype=np.float64, buffer=shm.buf)
            acc[:] = 0.0
            ctx = mp.get_context("spawn")
            lock = ctx.Lock()
            tasks = [(d, seed, K, c, eps, tol, shm.name, precond) for c in cols]
            with ctx.Pool(procs, initializer=_init, initargs=(lock,)) as pool:
                res = pool.map(_solve_column, tasks, chunksize=1)
            R = acc.copy()
        finally:
            acc = None  # the view must go before the mapping is closed
            shm.close()
            shm.unlink()
    by_col = {r[0]: r for r in res}
    return dict(R=R,
                iters=np.array([by_col[c][1] for c in cols]),
                relres=np.array([by_col[c][2] for c in cols]),
                converged=all(by_col[c][3] for c in cols),
                foster=np.array([by_col[c][4] for c in cols]))
