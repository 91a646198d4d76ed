#!/usr/bin/env python
"""ERC-LG curvature throughput on GB300.

One step = the whole path on one synthetic graph with its inputs resident in HBM: Laplacian build,
then for every batch of projection columns the Philox right-hand sides, the column-wise CG solve
and the edge-resistance accumulation, then curvature (Eq. 2) and the sampling probabilities
(Eq. 7-8).  The metric is curvature edges per second (m / step time).  The default workload is the
largest: the 2.45M-node, 64.3M-edge power-law graph at K = 1024 in batches of 128 columns (its
smaller K = 64 and 256 are reported under "k_sweep").  The JSON line also carries the end-to-end
number through the host-memory C-ABI call, the roofline of the dominant kernel, the CPU oracle as
a reported baseline, clocks and the kernel-launch count.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config NAME]
Under torchrun (N > 1) every rank owns K projection columns of a K*N projection (weak scaling)
and the per-rank edge accumulators are summed with one all-reduce (Algorithm 1).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time
import warnings

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ERC-LG curvature edges/s end-to-end; CG SpMM HBM GB/s vs GB300 peak"
DEFAULT_CONFIG = "chung_lu_n2449029_g2.3"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default=DEFAULT_CONFIG)
    ap.add_argument("--K", type=int, default=None,
                    help="projection dimension (per rank; default: the workload's largest)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-sweep", action="store_true",
                    help="skip the workload's other projection dimensions")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--spmm-reps", type=int, default=50)
    ap.add_argument("--precond", choices=["none", "jacobi"], default="none",
                    help="CG preconditioner of the whole step (the paper's method: none)")
    return ap.parse_args()


# ------------------------------------------------------------------------------------ helpers
class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) >= 9:
                rows.append(f)
        os.unlink(self.path)
        if not rows:
            return None

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d.get("hbm_gbs"), "measured"
    return 6800.0, "fallback"


def spmm_traffic(workload):
    """DRAM bytes per launch of the operator kernel from a committed ncu summary, if current."""
    return _traffic("spmm", workload)


# CG vector update per iteration: read x, r, p, Ap and write x, r, p (7 passes of 4 bytes)
UPDATE_BYTES_PER_ELEM = 28


def _traffic(kernel, workload, field="dram_bytes_per_launch"):
    """A per-launch ncu counter of `kernel` on `workload` from profiles/traffic.json, or None
    when it was not captured or was captured on other solver sources."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p))
    e = d.get(kernel, {}).get(workload)
    if not e or e.get("solver_src_sha1") != solver_src_sha1():
        return None
    return e.get(field)


def solver_src_sha1():
    """sha1 of the solver's sources (cg.cu, then cg_device.cuh): ncu counters taken on other
    sources do not describe the kernels that run."""
    h = hashlib.sha1()
    for f in ("cg.cu", "cg_device.cuh"):
        h.update(open(os.path.join(ROOT, "paper_2609_27209_gb300", "csrc", f), "rb").read())
    return h.hexdigest()


def spmm_algorithmic_bytes(n, m, kc, weighted):
    """Bytes the operator must move once: CSR (col, weights, row_ptr) + read P + write AP."""
    return 4 * 2 * m + (4 * 2 * m if weighted else 0) + 8 * (n + 1) + 2 * 4 * n * kc


def solve_algorithmic_bytes(n, m, kc, weighted, column_iters, resident):
    """Bytes a single-launch CG solve must move: the CSR once per iteration while any column is
    active; per column and iteration it runs, its column of P once, of Ap once and the update's
    7 vector passes (a stopped column is neither gathered nor updated); the launch's own
    initialisation (read Y; write P, X); and, in the resident kernel, the true residual (one
    operator pass and Y read)."""
    T = max(column_iters) if len(column_iters) else 0
    csr = spmm_algorithmic_bytes(n, m, kc, weighted) - 2 * 4 * n * kc
    algo = T * csr + sum(column_iters) * (8 + UPDATE_BYTES_PER_ELEM) * n + 12 * n * kc
    if resident:
        algo += spmm_algorithmic_bytes(n, m, kc, weighted) + 4 * n * kc
    return algo


# ------------------------------------------------------------------------------------ oracle leg
# The float64 oracle (oracle/erc_oracle.py, as it stands) timed on the host cores on a bounded
# sample of the workload.  A run costs build + K x (one column's right-hand side, CG solve and
# edge distances: the K systems are independent and cost alike) + the curvature/probability tail.
# Up to CAPPED_EDGES edges the sample solves whole columns; beyond that one column's solve takes
# minutes, so the sample runs CAP_ITERS CG iterations of one column and scales them to the
# column's iteration count.
CAPPED_EDGES = 10_000_000
CAP_ITERS = 20
REF_CAP_ITERS = 10  # CG iterations per step of the reference arm on such graphs


def _oracle_solver(precond):
    from oracle import erc_oracle as O
    return O.batched_pcg if precond == "jacobi" else O.batched_cg


class OracleRun:
    """The oracle's graph of one workload, with the seconds its build took."""

    def __init__(self, name, precond="none", graph=None):
        from oracle import erc_oracle as O
        from paper_2609_27209_gb300 import synth

        self.name, self.precond = name, precond
        self.wl = synth.WORKLOADS[name]
        self.seed = synth.JL_SEED
        n, src, dst, w = synth.make_graph(name) if graph is None else graph
        t0 = time.perf_counter()
        self.g = O.build_laplacian(n, src, dst, w)
        self.t_build = time.perf_counter() - t0
        self.n, self.m = n, self.g["m"]
        self.capped = self.m > CAPPED_EDGES

    def columns(self, K, c0, cols, max_iter=20000):
        """(t_rhs, t_cg, t_edge, iterations, R) of columns [c0, c0 + cols) of the K projection."""
        from oracle import erc_oracle as O

        t0 = time.perf_counter()
        Y = O.jl_rhs(self.g, self.seed, K, c0, cols)
        t1 = time.perf_counter()
        X, it, _, _ = _oracle_solver(self.precond)(self.g, self.wl.eps, Y, self.wl.tol, max_iter)
        t2 = time.perf_counter()
        R = O.edge_resistance(self.g, X)
        t3 = time.perf_counter()
        return t1 - t0, t2 - t1, t3 - t2, it, R

    def tail(self, R):
        from oracle import erc_oracle as O

        t0 = time.perf_counter()
        _, kappa = O.curvature(self.g, R)
        O.sampling_probs(self.g, kappa)
        return time.perf_counter() - t0

    def column_iterations(self, K):
        """CG iterations of column 0 solved to the tolerance (the capped samples' scale)."""
        return int(self.columns(K, 0, 1)[3][0])

    def cg_only(self, Y, max_iter):
        """(seconds, iterations) of the CG solve of the columns Y, capped at max_iter."""
        t0 = time.perf_counter()
        _, it, _, _ = _oracle_solver(self.precond)(self.g, self.wl.eps, Y, self.wl.tol, max_iter)
        return time.perf_counter() - t0, int(it.max())


def oracle_sample(run, K, cols):
    """Whole columns: the full graph with `cols` of the K columns, the column work scaled to K.
    Returns (edges/s, seconds sampled, description, estimated seconds of the whole run)."""
    t0 = time.perf_counter()
    tr, tc, te, _, R = run.columns(K, 0, cols)
    t_tail = run.tail(R * (K / cols))
    est = run.t_build + (tr + tc + te) * (K / cols) + t_tail
    desc = (f"full graph (n={run.n}, m={run.m}), {cols} of {K} projection columns solved to the "
            f"tolerance; build ({run.t_build:.1f} s) and curvature/probability tail timed once, "
            f"the column work scaled by {K}/{cols}")
    return run.m / est, time.perf_counter() - t0 + run.t_build, desc, est


def oracle_sample_capped(run, K, T, t_tail=None, cap=CAP_ITERS):
    """One column with its CG capped at `cap` iterations, scaled to T iterations per column and to
    K columns.  Returns (edges/s, seconds sampled, description, estimated seconds)."""
    t0 = time.perf_counter()
    tr, tc, te, it, R = run.columns(K, 0, 1, max_iter=cap)
    done = max(1, int(it[0]))
    if t_tail is None:
        t_tail = run.tail(R * K)
    est = run.t_build + K * (tr + tc * (T / done) + te) + t_tail
    desc = (f"full graph (n={run.n}, m={run.m}); build ({run.t_build:.1f} s) and "
            f"curvature/probability tail ({t_tail:.1f} s) timed once; one column's right-hand "
            f"side, {done} CG iterations and edge distances timed, the iterations scaled to "
            f"{T:.1f} per column and the column to {K} columns")
    return run.m / est, time.perf_counter() - t0, desc, est


def cpu_cores_used():
    return 1  # numpy elementwise and scipy sparse products run single-threaded here


_THREAD_VARS = ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")


def _oracle_warm(_):
    import numpy  # noqa: F401
    import scipy.sparse  # noqa: F401

    from oracle import erc_oracle  # noqa: F401
    time.sleep(0.05)  # long enough that every worker of the pool takes a warm-up task
    return os.getpid()


def _oracle_columns(task):
    """One worker's share of the oracle's column-proportional work (RHS, CG, distances)."""
    name, K, c0, kc, g, precond = task
    from oracle import erc_oracle as O
    from paper_2609_27209_gb300 import synth
    wl = synth.WORKLOADS[name]
    X, _, _, _ = _oracle_solver(precond)(g, wl.eps, O.jl_rhs(g, synth.JL_SEED, K, c0, kc),
                                         wl.tol)
    return O.edge_resistance(g, X)


def oracle_sample_all_cores(run, K, cols, procs):
    """The same sample as oracle_sample with the `cols` columns split over `procs` processes
    (spawn context, one BLAS thread each, warmed up before timing); the build and the
    curvature/probability tail are not parallel and are counted once on one core."""
    import multiprocessing as mp

    from oracle import erc_oracle as O
    saved = {k: os.environ.get(k) for k in _THREAD_VARS}
    for k in _THREAD_VARS:
        os.environ[k] = "1"
    try:
        with mp.get_context("spawn").Pool(procs) as pool:
            pool.map(_oracle_warm, range(4 * procs), chunksize=1)
            bounds = [(cols * i // procs, cols * (i + 1) // procs) for i in range(procs)]
            tasks = [(run.name, K, a, b - a, run.g, run.precond) for a, b in bounds if b > a]
            t0 = time.perf_counter()
            parts = pool.map(_oracle_columns, tasks, chunksize=1)
            t_cols = time.perf_counter() - t0
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    R = sum(parts)
    t0 = time.perf_counter()
    _, kappa = O.curvature(run.g, R * (K / cols))
    O.sampling_probs(run.g, kappa)
    t_tail = time.perf_counter() - t0
    est = run.t_build + t_cols * (K / cols) + t_tail
    desc = (f"full graph (n={run.n}, m={run.m}), {cols} of {K} projection columns split over "
            f"{len(tasks)} processes; build and curvature/probability tail on one core, the "
            f"column work scaled by {K}/{cols}")
    return run.m / est, desc


# ------------------------------------------------------------------------------------ main legs
def workload_K(args, wl):
    """The projection dimension of the run: --K, else the workload's largest."""
    return args.K or max(wl.K)


def run_reference(args, world, rank):
    """The float64 oracle on the host cores as the reference arm: every step is a bounded sample
    of the workload (see the oracle leg); rank 0 alone runs it."""
    from paper_2609_27209_gb300 import synth

    wl = synth.WORKLOADS[args.config]
    K = workload_K(args, wl)
    if rank != 0:
        return
    run = OracleRun(args.config, args.precond)
    if run.capped:
        # once: one full oracle solve of column 0 (its right-hand side, iteration count and edge
        # distances) and the tail; every step then times REF_CAP_ITERS CG iterations of that
        # column and scales them to its iteration count
        from oracle import erc_oracle as O

        t_rhs, _, t_edge, it0, R = run.columns(K, 0, 1)
        T = int(it0[0])
        t_tail = run.tail(R * K)
        Y = O.jl_rhs(run.g, run.seed, K, 0, 1)

        def sample():
            t_cg, done = run.cg_only(Y, REF_CAP_ITERS)
            est = run.t_build + K * (t_rhs + t_cg * (T / max(1, done)) + t_edge) + t_tail
            desc = (f"full graph (n={run.n}, m={run.m}); build ({run.t_build:.1f} s), one "
                    f"column's right-hand side ({t_rhs:.1f} s) and edge distances "
                    f"({t_edge:.1f} s) from a full oracle solve of column 0 ({T} iterations), "
                    f"and the curvature/probability tail ({t_tail:.1f} s) timed once; each "
                    f"step times {done} CG iterations of that column, scaled to {T} per column "
                    f"and to {K} columns")
            return run.m / est, t_cg, desc, est
    else:
        cols = min(K, max(4, K // 8))

        def sample():
            return oracle_sample(run, K, cols)
    for _ in range(args.warmup):
        sample()
    vals, ests = [], []
    desc = ""
    for _ in range(args.steps):
        v, _, desc, est = sample()
        vals.append(v)
        ests.append(est)
    value = len(vals) / sum(1.0 / v for v in vals)  # harmonic mean = m / mean time
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "edges/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * statistics.mean(ests), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.config, "K": K, "kc": min(wl.kc, K), "eps": wl.eps,
                       "tol": wl.tol, "precond": args.precond},
            "cpu_baseline": {"value": value, "unit": "edges/s", "cores": cpu_cores_used(),
                             "kind": "oracle", "sample": desc},
            "e2e": {"value": value, "unit": "edges/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def _timed_steps(step, n_steps, flush, stream):
    """CUDA-event time (ms) of each of n_steps calls of step(), L2 flushed before each."""
    import torch

    times = []
    res = None
    for _ in range(n_steps):
        flush.fill_(1)  # evict L2 between timed steps (outside the timed interval)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        res = step()
        b.record(stream)
        b.synchronize()
        times.append(a.elapsed_time(b))
    return times, res


def run_ours(args, world, rank, local_rank):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2609_27209_gb300 import dist as edist
    from paper_2609_27209_gb300 import erc, synth

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    wl = synth.WORKLOADS[args.config]
    K = workload_K(args, wl)
    kc = min(wl.kc, K)
    graph = synth.make_graph(args.config)
    n, src, dst, w = graph
    m_in = src.size
    precond = erc.ERC_PRECOND_JACOBI if args.precond == "jacobi" else erc.ERC_PRECOND_NONE
    prm = erc.Params(K=K, kc=kc, eps=wl.eps, tol=wl.tol, seed=synth.JL_SEED, precond=precond)
    src_d = torch.from_numpy(src).to(dev)
    dst_d = torch.from_numpy(dst).to(dev)
    w_d = None if w is None else torch.from_numpy(w).to(dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # > 129 MB of L2
    stream = torch.cuda.current_stream()

    mem = None
    if world == 1:
        ws = erc.erc_run_workspace(n, m_in, prm, dev)
        out = erc._run_outputs(n, m_in, K, dev)
        # the library allocates nothing: a step's device memory is its workspace, outputs, inputs
        nbytes = lambda t: t.numel() * t.element_size()
        mem = {"workspace": nbytes(ws),
               "outputs": sum(nbytes(t) for t in out.values() if torch.is_tensor(t)),
               "inputs": nbytes(src_d) + nbytes(dst_d) + (0 if w_d is None else nbytes(w_d))}
        mem["total"] = sum(mem.values())

        def step():
            return erc.erc_run(n, src_d, dst_d, w_d, prm, ws=ws, out=out)
    else:
        def allreduce(t):
            dist.all_reduce(t, op=dist.ReduceOp.SUM)
            return t

        def step():
            return edist.run_sharded(n, src_d, dst_d, w_d, prm, world, rank, allreduce)

    res = None
    for _ in range(args.warmup):
        res = step()
    torch.cuda.synchronize()
    m = int(res["m"])
    sampler = ClockSampler(local_rank)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    launches0 = erc.erc_kernel_launches()
    sampler.start()
    times, res = _timed_steps(step, args.steps, flush, stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    launches = erc.erc_kernel_launches() - launches0
    if world > 1:
        dist.barrier()
    ms = statistics.mean(times)
    t = torch.tensor([ms], dtype=torch.float64, device=dev)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    ms_max = float(t.item())
    value = world * m / (ms_max / 1000.0)
    iters = res.get("iters")
    it = iters.float() if iters is not None else None
    slow = ms_max > 2000.0  # steps of seconds: fewer repetitions of the extra measurements
    if world == 1:
        del ws, out

    # ---- end to end through the host-memory C-ABI call (copies inside the timed region)
    e2e = None
    if not args.no_e2e and world == 1:
        src_h = torch.from_numpy(src).pin_memory()
        dst_h = torch.from_numpy(dst).pin_memory()
        w_h = None if w is None else torch.from_numpy(w).pin_memory()
        hws = erc.erc_run_host_workspace(n, m_in, prm, dev)
        hout = erc._run_outputs(n, m_in, K, None, pin=True)
        for _ in range(1 if slow else 2):
            erc.erc_run_host(n, src_h, dst_h, w_h, prm, ws=hws, out=hout)
        et = []
        for _ in range(3 if slow else max(3, args.steps // 2)):
            flush.fill_(1)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            erc.erc_run_host(n, src_h, dst_h, w_h, prm, ws=hws, out=hout)
            torch.cuda.synchronize()
            et.append(time.perf_counter() - t0)
        h2d = m_in * 4 * (2 if w is None else 3)
        d2h = 5 * 4 * m + 2 * 4 * n + 2 * 4 * K
        e2e = {"value": m / statistics.mean(et), "unit": "edges/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": 1000 * statistics.mean(et),
               "repetitions": len(et)}
        del hws, hout

    # ---- the workload's other projection dimensions (its K sweep), the same path and batches
    sweep = None
    if world == 1 and not args.no_sweep and len(wl.K) > 1:
        sweep = []
        for Ks in wl.K:
            if Ks == K:
                continue
            p2 = erc.Params(K=Ks, kc=min(wl.kc, Ks), eps=wl.eps, tol=wl.tol, seed=synth.JL_SEED,
                            precond=precond)
            ws2 = erc.erc_run_workspace(n, m_in, p2, dev)
            out2 = erc._run_outputs(n, m_in, Ks, dev)
            st2 = lambda: erc.erc_run(n, src_d, dst_d, w_d, p2, ws=ws2, out=out2)
            st2()
            t2, r2 = _timed_steps(st2, 3, flush, stream)
            sweep.append({"K": Ks, "kc": p2.kc, "ms_per_step": statistics.mean(t2),
                          "value": m / (statistics.mean(t2) / 1000.0), "status": r2["status"],
                          "cg_iters_mean": float(r2["iters"].float().mean())})
            del ws2, out2
        torch.cuda.empty_cache()

    # ---- roofline of the dominant kernel.  On graphs whose r and Ap blocks fit in shared memory
    # the whole CG solve is one launch (k_cg_cluster over column groups, else k_cg_resident),
    # timed by CUDA events the library records around it on its stream; its bytes stay in L2.
    # Otherwise the operator k_spmm dominates (HBM: P exceeds L2) and is timed alone, back to back
    # as inside the CG loop.  The operator alone is always reported under "spmm".
    roof = spmm = cusparse = samp = cpu_all = variants = None
    if rank == 0:
        g = erc.erc_build_laplacian(n, src_d, dst_d, w_d)
        P = erc.erc_jl_rhs(g, synth.JL_SEED, K, 0, kc)
        weighted = not g.unit_weights
        peak, src_kind = measured_peaks()
        op_bytes = spmm_algorithmic_bytes(n, g.m, kc, weighted)
        erc.erc_laplacian_apply_timed(g, prm.eps, P, kc, reps=5)
        t_spmm = erc.erc_laplacian_apply_timed(g, prm.eps, P, kc, reps=args.spmm_reps) * 1e-6
        traffic = spmm_traffic(args.config)
        spmm = {"kernel": "k_spmm (L_eps P + p.Ap)", "launch_us": t_spmm * 1e6,
                "algorithmic_bytes": op_bytes, "achieved": op_bytes / t_spmm / 1e9,
                "frac": op_bytes / t_spmm / 1e9 / peak, "traffic": traffic,
                "gathered_row_bytes": 4 * 2 * g.m * kc}
        if traffic:
            spmm["dram_achieved"] = traffic / t_spmm / 1e9
            spmm["dram_frac"] = spmm["dram_achieved"] / peak
        # library comparison point (run only): cuSPARSE SpMM of the adjacency, A P, through
        # torch's CSR x dense product, timed with events on the current stream
        vals = g.val if not g.unit_weights else torch.ones(2 * g.m, device=dev)
        with warnings.catch_warnings():  # torch flags its sparse CSR support as beta
            warnings.simplefilter("ignore", UserWarning)
            A = torch.sparse_csr_tensor(g.row_ptr, g.col.long(), vals, size=(n, n))
        for _ in range(3):
            A @ P
        reps = 10 if slow else args.spmm_reps
        ca, cb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ca.record()
        for _ in range(reps):
            A @ P
        cb.record()
        cb.synchronize()
        t_cs = ca.elapsed_time(cb) / 1e3 / reps
        cusparse = {"kernel": "cuSPARSE SpMM A P (torch sparse CSR @ dense), run only",
                    "launch_us": t_cs * 1e6, "achieved": op_bytes / t_cs / 1e9,
                    "frac": op_bytes / t_cs / 1e9 / peak}
        del A, vals
        # the curvature-guided subgraph samplers on this run's probabilities (§3.2), one call
        # each (node budget n/10, edge budget m/10); each call synchronises to return its sizes
        if res.get("prob_node") is not None and res.get("prob_edge") is not None:
            samp = {"node_budget": max(1, n // 10), "edge_budget": max(1, g.m // 10)}
            runs = [(erc.ERC_SAMPLE_NODES, "node", res["prob_node"], samp["node_budget"]),
                    (erc.ERC_SAMPLE_EDGES, "edge", res["prob_edge"], samp["edge_budget"])]
            for kind, key, prob, b in runs:
                sws = erc._workspace(erc.lib().erc_sample_workspace_size(n, g.m, b), dev)
                erc.erc_sample_subgraph(g, kind, prob, b, 1, ws=sws)
                torch.cuda.synchronize()
                t0 = time.perf_counter()
                for r in range(5):
                    nodes_s, edges_s = erc.erc_sample_subgraph(g, kind, prob, b, 1, b * r, ws=sws)
                torch.cuda.synchronize()
                samp[key + "_subgraph_us"] = (time.perf_counter() - t0) / 5 * 1e6
                samp[key + "_subgraph_size"] = [int(nodes_s.numel()), int(edges_s.numel())]
                del sws
        erc.erc_batched_cg_timed(g, prm.eps, P, kc, prm.tol)  # warm
        _, it_cg, _, _, solve_us, path = erc.erc_batched_cg_timed(g, prm.eps, P, kc, prm.tol)
        # the optional Jacobi-preconditioned solve of the same batch (not the paper's solver)
        erc.erc_batched_pcg_timed(g, prm.eps, P, kc, prm.tol)
        _, it_pc, _, _, pcg_us, pcg_path = erc.erc_batched_pcg_timed(g, prm.eps, P, kc, prm.tol)
        variants = {"batch_columns": kc,
                    "cg": {"path": path, "solve_us": solve_us,
                           "iters_max": int(it_cg.max().item()),
                           "iters_mean": float(it_cg.float().mean().item())},
                    "jacobi_pcg": {"path": pcg_path, "solve_us": pcg_us,
                                   "iters_max": int(it_pc.max().item()),
                                   "iters_mean": float(it_pc.float().mean().item())}}
        pc = args.precond == "jacobi"  # the roofline follows the solver the step runs
        if pc:
            it_cg, solve_us, path = it_pc, pcg_us, pcg_path
        if path in (1, 2):
            # bytes the solve must move: the CSR once per iteration while any column is active,
            # per column and iteration it runs P once, Ap once and the update's 7 vector passes
            # (a converged column is neither gathered nor updated), plus the launch's own
            # initialisation (read Y; write P, X) and, in the resident kernel, the true residual
            its = it_cg.double()
            T = int(its.max().item())
            algo = solve_algorithmic_bytes(n, g.m, kc, weighted, [int(x) for x in it_cg.tolist()],
                                           path == 1)
            ach = algo / (solve_us * 1e-6) / 1e9
            kname = "k_cg_cluster" if path == 2 else "k_cg_resident"
            roof = {"bound": "l2", "achieved": ach, "peak": peak, "unit": "GB/s",
                    "frac": ach / peak,
                    "traffic": None if pc else _traffic(kname[2:], args.config),
                    "kernel": f"{kname}{' (Jacobi)' if pc else ''} (one launch = whole CG solve "
                              "of a batch; its working set stays in L2, so frac is an effective "
                              "rate against the HBM peak)",
                    "iterations": T, "column_iterations": float(its.sum().item()),
                    "algorithmic_bytes": algo, "launch_us": solve_us, "peak_source": src_kind}
            l2 = None if pc else _traffic(kname[2:], args.config, "l2_bytes_per_launch")
            if l2:  # what the solve moved through L2, by ncu's lts__t_bytes.sum
                roof["l2_traffic"] = l2
                roof["l2_achieved"] = l2 / (solve_us * 1e-6) / 1e9
        else:
            roof = {"bound": "hbm", "achieved": spmm["achieved"], "peak": peak, "unit": "GB/s",
                    "frac": spmm["frac"], "traffic": spmm["traffic"], "kernel": spmm["kernel"],
                    "algorithmic_bytes": op_bytes, "launch_us": t_spmm * 1e6,
                    "peak_source": src_kind, "gathered_row_bytes": spmm["gathered_row_bytes"]}
            if traffic:
                roof["dram_achieved"] = spmm["dram_achieved"]
                roof["dram_frac"] = spmm["dram_frac"]
        del g, P

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        run = OracleRun(args.config, args.precond, graph=graph)
        if run.capped:
            T_gpu = float(it.mean())  # the solver's iterations per column on this workload
            v, secs, desc, _ = oracle_sample_capped(run, K, T_gpu)
            desc += " (the iteration count is the GPU solve's mean)"
        else:
            # size the sample to roughly 15 s of CPU work from a 4-column probe
            _, _, _, est4 = oracle_sample(run, K, min(K, 4))
            per_col = (est4 - run.t_build) / K
            cols = int(min(K, max(4, (15.0 / max(per_col, 1e-9)) // 4 * 4)))
            v, secs, desc, _ = oracle_sample(run, K, cols)
            procs = max(1, min(os.cpu_count() or 1, cols))
            va, desc_all = oracle_sample_all_cores(run, K, cols, procs)
            cpu_all = {"value": va, "unit": "edges/s", "cores": procs, "kind": "oracle",
                       "sample": desc_all}
        cpu = {"value": v, "unit": "edges/s", "cores": cpu_cores_used(), "kind": "oracle",
               "sample": desc, "seconds": secs}
        del run

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "edges/s", "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_max,
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "f32", "data": "synthetic",
                "config": {"workload": args.config, "n": n, "m": m, "K": K, "kc": kc,
                           "eps": wl.eps, "tol": wl.tol, "precond": args.precond,
                           "l2": "flushed (256 MiB write) before every timed step",
                           "parallelism": f"projection columns over {world} rank(s)"},
                "roofline": roof, "spmm": spmm, "cusparse_spmm": cusparse, "sampler": samp,
                "solver_variants": variants, "k_sweep": sweep, "cpu_baseline": cpu,
                "cpu_baseline_all_cores": cpu_all,
                "e2e": e2e, "gpu_launches": launches, "device_memory_bytes": mem,
                "clocks": clocks,
                "cg_iters": None if it is None else {"mean": float(it.mean()),
                                                     "max": float(it.max())}}
        print(json.dumps(line), flush=True)


def main():
    args = parse()
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, world, rank)
        return
    if world > 1:
        import torch
        import torch.distributed as dist

        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    try:
        run_ours(args, world, rank, local_rank)
    finally:
        if world > 1:
            import torch.distributed as dist

            dist.destroy_process_group()


if __name__ == "__main__":
    main()
