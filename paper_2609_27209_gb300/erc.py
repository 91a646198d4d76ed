"""Python binding of liberc.so (the C ABI in include/erc.h): argument marshalling only.

Every function here has the name of the C entry point it calls and does nothing but allocate
torch tensors for outputs / workspace, pass raw device pointers and the current CUDA stream, and
turn error codes into exceptions.  All arithmetic runs in the library's CUDA kernels; there is no
CPU path, and loading fails loudly when the library has not been built.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liberc.so")

ERC_OK = 0
ERC_ERR_INVALID_ARG = 1
ERC_ERR_CUDA = 2
ERC_ERR_CAPACITY = 3
ERC_ERR_NOT_CONVERGED = 4
ERC_ERR_NUMERIC = 5
ERC_ERR_TIMEOUT = 6
ERC_DUP_SUM = 0
ERC_DUP_FIRST = 1
ERC_PRECOND_NONE = 0
ERC_PRECOND_JACOBI = 1

_c_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_u64 = ctypes.c_uint64
_f32 = ctypes.c_float
_sz = ctypes.c_size_t


class ErcError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"erc status {status}: {message}")
        self.status = status


class ErcGraphC(ctypes.Structure):
    _fields_ = [("n", _i32), ("m", _i64), ("row_ptr", _c_p), ("col", _c_p), ("val", _c_p),
                ("deg", _c_p), ("csr_eid", _c_p), ("eu", _c_p), ("ev", _c_p), ("ew", _c_p)]


class ErcParamsC(ctypes.Structure):
    _fields_ = [("seed", _u64), ("K", _i32), ("kc", _i32), ("eps", _f32), ("tol", _f32),
                ("max_iter", _i32), ("eta", _f32), ("dup_policy", _i32), ("precond", _i32)]


_SIGS = {
    "erc_version": (ctypes.c_char_p, []),
    "erc_last_error": (ctypes.c_char_p, []),
    "erc_kernel_launches": (ctypes.c_uint64, []),
    "erc_set_wait_limit": (None, [ctypes.c_uint32]),
    "erc_build_laplacian_workspace_size": (_sz, [_i32, _i64]),
    "erc_build_laplacian": (_i32, [_i32, _c_p, _c_p, _c_p, _i64, _i32, _c_p, _c_p, _c_p, _c_p,
                                   _c_p, _c_p, _c_p, _c_p, ctypes.POINTER(_i64), _c_p, _sz, _c_p]),
    "erc_build_laplacian_ex": (_i32, [_i32, _c_p, _c_p, _c_p, _i64, _i32, _c_p, _c_p, _c_p, _c_p,
                                      _c_p, _c_p, _c_p, _c_p, ctypes.POINTER(_i64),
                                      ctypes.POINTER(_i32), _c_p, _sz, _c_p]),
    "erc_jl_rhs": (_i32, [ctypes.POINTER(ErcGraphC), _u64, _i32, _i32, _i32, _c_p, _i32, _c_p]),
    "erc_batched_cg_workspace_size": (_sz, [_i32, _i32]),
    "erc_batched_cg": (_i32, [ctypes.POINTER(ErcGraphC), _f32, _c_p, _c_p, _i32, _i32, _f32,
                              _i32, _c_p, _c_p, _c_p, _sz, _c_p]),
    "erc_batched_cg_timed": (_i32, [ctypes.POINTER(ErcGraphC), _f32, _c_p, _c_p, _i32, _i32,
                                    _f32, _i32, _c_p, _c_p, _c_p, _sz, ctypes.POINTER(_f32),
                                    ctypes.POINTER(_i32), _c_p]),
    "erc_batched_pcg": (_i32, [ctypes.POINTER(ErcGraphC), _f32, _c_p, _c_p, _i32, _i32, _f32,
                               _i32, _c_p, _c_p, _c_p, _sz, _c_p]),
    "erc_batched_pcg_timed": (_i32, [ctypes.POINTER(ErcGraphC), _f32, _c_p, _c_p, _i32, _i32,
                                     _f32, _i32, _c_p, _c_p, _c_p, _sz, ctypes.POINTER(_f32),
                                     ctypes.POINTER(_i32), _c_p]),
    "erc_edge_resistance": (_i32, [ctypes.POINTER(ErcGraphC), _c_p, _i32, _i32, _c_p, _c_p]),
    "erc_curvature": (_i32, [ctypes.POINTER(ErcGraphC), _c_p, _c_p, _c_p, _c_p]),
    "erc_sampling_probs_workspace_size": (_sz, [_i32, _i64]),
    "erc_sampling_probs": (_i32, [ctypes.POINTER(ErcGraphC), _c_p, _f32, _c_p, _c_p, _c_p, _sz,
                                  _c_p]),
    "erc_sampling_probs_noalloc": (_i32, [ctypes.POINTER(ErcGraphC), _c_p, _f32, _c_p, _c_p,
                                          _c_p]),
    "erc_sample_workspace_size": (_sz, [_i32, _i64, _i64]),
    "erc_sample_subgraph": (_i32, [ctypes.POINTER(ErcGraphC), _i32, _c_p, _i64, _u64, _i64, _i32,
                                   _c_p, ctypes.POINTER(_i32), _c_p, ctypes.POINTER(_i64), _c_p,
                                   _sz, _c_p]),
    "erc_saint_counts": (_i32, [ctypes.POINTER(ErcGraphC), _c_p, _i32, _c_p, _i64, _c_p, _c_p,
                                _c_p]),
    "erc_saint_norm": (_i32, [ctypes.POINTER(ErcGraphC), _c_p, _c_p, _i32, _c_p, _c_p, _c_p]),
    "erc_laplacian_apply_workspace_size": (_sz, [_i32, _i32]),
    "erc_laplacian_apply": (_i32, [ctypes.POINTER(ErcGraphC), _f32, _c_p, _c_p, _i32, _i32, _c_p,
                                   _c_p, _sz, _c_p]),
    "erc_laplacian_apply_timed": (_i32, [ctypes.POINTER(ErcGraphC), _f32, _c_p, _c_p, _i32,
                                         _i32, _c_p, _i32, ctypes.POINTER(_f32), _c_p, _sz,
                                         _c_p]),
    "erc_philox_signs": (_i32, [_u64, _i64, _i64, _i32, _i32, _c_p, _c_p]),
    "erc_run_workspace_size": (_sz, [_i32, _i64, _i32]),
    "erc_run": (_i32, [ctypes.POINTER(ErcParamsC), _i32, _c_p, _c_p, _c_p, _i64,
                       ctypes.POINTER(_i64), _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                       _c_p, _sz, _c_p]),
    "erc_run_host_workspace_size": (_sz, [_i32, _i64, _i32, _i32]),
    "erc_run_host": (_i32, [ctypes.POINTER(ErcParamsC), _i32, _c_p, _c_p, _c_p, _i64,
                            ctypes.POINTER(_i64), _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p, _c_p,
                            _c_p, _c_p, _sz, _c_p]),
}

_lib = None


def lib():
    """The loaded liberc.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build(); "
                               "there is no CPU fallback")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def exported_symbols():
    return list(_SIGS)


def _check(status, allow=()):
    if status != ERC_OK and status not in allow:
        raise ErcError(status, lib().erc_last_error().decode(errors="replace"))
    return status


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _workspace(nbytes, device):
    return torch.empty(max(int(nbytes), 1), dtype=torch.uint8, device=device)


def erc_version():
    return lib().erc_version().decode()


def erc_kernel_launches():
    return int(lib().erc_kernel_launches())


def erc_set_wait_limit(polls):
    """Polls every bounded device-side wait makes before giving up (0 restores the defaults)."""
    lib().erc_set_wait_limit(int(polls))


@dataclass
class Graph:
    """Tensors of a graph built by erc_build_laplacian plus the matching C struct."""

    n: int
    m: int
    row_ptr: torch.Tensor
    col: torch.Tensor
    val: torch.Tensor
    deg: torch.Tensor
    csr_eid: torch.Tensor
    eu: torch.Tensor
    ev: torch.Tensor
    ew: torch.Tensor
    unit_weights: bool

    def c(self):
        g = ErcGraphC()
        g.n, g.m = self.n, self.m
        g.row_ptr, g.col, g.deg, g.csr_eid = (_ptr(self.row_ptr), _ptr(self.col), _ptr(self.deg),
                                              _ptr(self.csr_eid))
        g.val = None if self.unit_weights else _ptr(self.val)
        g.ew = None if self.unit_weights else _ptr(self.ew)
        g.eu, g.ev = _ptr(self.eu), _ptr(self.ev)
        return g


def erc_build_laplacian(n, src, dst, w=None, dup_policy=ERC_DUP_SUM):
    """Device int32 src/dst (and float32 w or None) -> Graph (see include/erc.h)."""
    dev = src.device
    m_in = src.numel()
    cap2, cap1 = max(2 * m_in, 1), max(m_in, 1)
    row_ptr = torch.empty(n + 1, dtype=torch.int64, device=dev)
    col = torch.empty(cap2, dtype=torch.int32, device=dev)
    val = torch.empty(cap2, dtype=torch.float32, device=dev)
    deg = torch.empty(n, dtype=torch.float32, device=dev)
    csr_eid = torch.empty(cap2, dtype=torch.int32, device=dev)
    eu = torch.empty(cap1, dtype=torch.int32, device=dev)
    ev = torch.empty(cap1, dtype=torch.int32, device=dev)
    ew = torch.empty(cap1, dtype=torch.float32, device=dev)
    ws = _workspace(lib().erc_build_laplacian_workspace_size(n, m_in), dev)
    m = _i64(0)
    unit = _i32(0)
    _check(lib().erc_build_laplacian_ex(n, _ptr(src), _ptr(dst), _ptr(w), m_in, dup_policy,
                                        _ptr(row_ptr), _ptr(col), _ptr(val), _ptr(deg),
                                        _ptr(csr_eid), _ptr(eu), _ptr(ev), _ptr(ew),
                                        ctypes.byref(m), ctypes.byref(unit), _ptr(ws), ws.numel(),
                                        _stream()))
    m = m.value
    return Graph(n, m, row_ptr, col[:2 * m], val[:2 * m], deg, csr_eid[:2 * m], eu[:m], ev[:m],
                 ew[:m], bool(unit.value))


def padded_ld(kc):
    return (kc + 3) // 4 * 4


def erc_jl_rhs(g, seed, K, c0, kc, ld=None, out=None):
    ld = padded_ld(kc) if ld is None else ld
    Y = torch.empty(g.n, ld, dtype=torch.float32, device=g.row_ptr.device) if out is None else out
    gc = g.c()
    _check(lib().erc_jl_rhs(ctypes.byref(gc), seed, K, c0, kc, _ptr(Y), ld, _stream()))
    return Y


def _solve(fn, g, eps, Y, kc, tol, max_iter, X, ws, timed):
    n, ld = Y.shape
    dev = Y.device
    X = torch.empty_like(Y) if X is None else X
    iters = torch.empty(kc, dtype=torch.int32, device=dev)
    relres = torch.empty(kc, dtype=torch.float32, device=dev)
    if ws is None:
        ws = _workspace(lib().erc_batched_cg_workspace_size(n, ld), dev)
    gc = g.c()
    args = [ctypes.byref(gc), eps, _ptr(Y), _ptr(X), ld, kc, tol, max_iter, _ptr(iters),
            _ptr(relres), _ptr(ws), ws.numel()]
    if not timed:
        st = _check(getattr(lib(), fn)(*args, _stream()), allow=(ERC_ERR_NOT_CONVERGED,))
        return X, iters, relres, st
    us = _f32(0)
    path = _i32(0)
    st = _check(getattr(lib(), fn)(*args, ctypes.byref(us), ctypes.byref(path), _stream()),
                allow=(ERC_ERR_NOT_CONVERGED,))
    return X, iters, relres, st, float(us.value), int(path.value)


def erc_batched_cg(g, eps, Y, kc, tol, max_iter=20000, X=None, ws=None):
    """Returns (X, iters, relres, status); status is ERC_OK or ERC_ERR_NOT_CONVERGED."""
    return _solve("erc_batched_cg", g, eps, Y, kc, tol, max_iter, X, ws, False)


def erc_batched_cg_timed(g, eps, Y, kc, tol, max_iter=20000, X=None, ws=None):
    """erc_batched_cg plus (solve microseconds, path): 2 = cluster column-group solver, 1 = resident
    cooperative solver, 0 = multi-kernel graph loop."""
    return _solve("erc_batched_cg_timed", g, eps, Y, kc, tol, max_iter, X, ws, True)


def erc_batched_pcg(g, eps, Y, kc, tol, max_iter=20000, X=None, ws=None):
    """Jacobi-preconditioned variant of erc_batched_cg (an option, not the paper's solver)."""
    return _solve("erc_batched_pcg", g, eps, Y, kc, tol, max_iter, X, ws, False)


def erc_batched_pcg_timed(g, eps, Y, kc, tol, max_iter=20000, X=None, ws=None):
    """erc_batched_pcg plus (solve microseconds, path: 1 resident, 0 multi-kernel)."""
    return _solve("erc_batched_pcg_timed", g, eps, Y, kc, tol, max_iter, X, ws, True)


def erc_edge_resistance(g, X, kc, R_acc):
    gc = g.c()
    _check(lib().erc_edge_resistance(ctypes.byref(gc), _ptr(X), X.shape[1], kc, _ptr(R_acc),
                                     _stream()))
    return R_acc


def erc_curvature(g, R):
    dev = R.device
    p = torch.empty(g.n, dtype=torch.float32, device=dev)
    kappa = torch.empty(max(g.m, 1), dtype=torch.float32, device=dev)[:g.m]
    gc = g.c()
    _check(lib().erc_curvature(ctypes.byref(gc), _ptr(R), _ptr(p), _ptr(kappa), _stream()))
    return p, kappa


def erc_sampling_probs(g, kappa, eta=1e-8):
    dev = kappa.device
    pn = torch.empty(g.n, dtype=torch.float32, device=dev)
    pe = torch.empty(max(g.m, 1), dtype=torch.float32, device=dev)[:g.m]
    ws = _workspace(lib().erc_sampling_probs_workspace_size(g.n, g.m), dev)
    gc = g.c()
    _check(lib().erc_sampling_probs(ctypes.byref(gc), _ptr(kappa), eta, _ptr(pn), _ptr(pe),
                                    _ptr(ws), ws.numel(), _stream()))
    return pn, pe


ERC_SAMPLE_NODES, ERC_SAMPLE_EDGES = 0, 1


def erc_sample_subgraph(g, kind, prob, budget, seed, first_draw=0, induced=True, ws=None):
    """One curvature-guided subgraph (see include/erc.h): (nodes int32, edges int32) on device."""
    dev = g.row_ptr.device
    nodes = torch.empty(max(g.n, 1), dtype=torch.int32, device=dev)
    edges = torch.empty(max(g.m, 1), dtype=torch.int32, device=dev)
    if ws is None:
        ws = _workspace(lib().erc_sample_workspace_size(g.n, g.m, budget), dev)
    n_s, m_s = _i32(0), _i64(0)
    gc = g.c()
    _check(lib().erc_sample_subgraph(ctypes.byref(gc), kind, _ptr(prob), budget, seed, first_draw,
                                     int(bool(induced)), _ptr(nodes), ctypes.byref(n_s),
                                     _ptr(edges), ctypes.byref(m_s), _ptr(ws), ws.numel(),
                                     _stream()))
    return nodes[:n_s.value], edges[:m_s.value]


def erc_saint_counts(g, nodes, edges, node_count, edge_count):
    gc = g.c()
    _check(lib().erc_saint_counts(ctypes.byref(gc), _ptr(nodes), nodes.numel(), _ptr(edges),
                                  edges.numel(), _ptr(node_count), _ptr(edge_count), _stream()))


def erc_saint_norm(g, node_count, edge_count, N):
    dev = g.row_ptr.device
    lam = torch.empty(g.n, dtype=torch.float32, device=dev)
    alpha = torch.empty(max(2 * g.m, 1), dtype=torch.float32, device=dev)[:2 * g.m]
    gc = g.c()
    _check(lib().erc_saint_norm(ctypes.byref(gc), _ptr(node_count), _ptr(edge_count), N,
                                _ptr(lam), _ptr(alpha), _stream()))
    return lam, alpha


def erc_sampling_probs_noalloc(g, kappa, eta=1e-8, out=None):
    """erc_sampling_probs without a workspace: the library's static device scratch is used.

    For callers that cannot allocate device memory; pass preallocated `out` = (prob_node,
    prob_edge) to keep the call itself free of allocations on the Python side too.
    """
    dev = kappa.device
    if out is None:
        out = (torch.empty(g.n, dtype=torch.float32, device=dev),
               torch.empty(max(g.m, 1), dtype=torch.float32, device=dev)[:g.m])
    pn, pe = out
    gc = g.c()
    _check(lib().erc_sampling_probs_noalloc(ctypes.byref(gc), _ptr(kappa), eta, _ptr(pn),
                                            _ptr(pe), _stream()))
    return pn, pe


def erc_laplacian_apply(g, eps, P, kc, want_pap=False):
    n, ld = P.shape
    AP = torch.empty_like(P)
    pap = torch.empty(kc, dtype=torch.float64, device=P.device) if want_pap else None
    ws = _workspace(lib().erc_laplacian_apply_workspace_size(n, ld), P.device)
    gc = g.c()
    _check(lib().erc_laplacian_apply(ctypes.byref(gc), eps, _ptr(P), _ptr(AP), ld, kc, _ptr(pap),
                                     _ptr(ws), ws.numel(), _stream()))
    return AP, pap


def erc_laplacian_apply_timed(g, eps, P, kc, reps=50):
    """Mean duration (microseconds) of the operator kernel over `reps` back-to-back launches."""
    n, ld = P.shape
    AP = torch.empty_like(P)
    pap = torch.empty(kc, dtype=torch.float64, device=P.device)
    ws = _workspace(lib().erc_laplacian_apply_workspace_size(n, ld), P.device)
    us = _f32(0)
    gc = g.c()
    _check(lib().erc_laplacian_apply_timed(ctypes.byref(gc), eps, _ptr(P), _ptr(AP), ld, kc,
                                           _ptr(pap), reps, ctypes.byref(us), _ptr(ws),
                                           ws.numel(), _stream()))
    return float(us.value)


def erc_philox_signs(seed, e0, e1, c0, c1, device="cuda"):
    out = torch.empty(max((e1 - e0) * (c1 - c0), 1), dtype=torch.int32, device=device)
    _check(lib().erc_philox_signs(seed, e0, e1, c0, c1, _ptr(out), _stream()))
    return out[:(e1 - e0) * (c1 - c0)].view(e1 - e0, c1 - c0)


@dataclass
class Params:
    K: int
    kc: int
    eps: float = 1e-3
    tol: float = 1e-6
    seed: int = 0xE2C1
    max_iter: int = 20000
    eta: float = 1e-8
    dup_policy: int = ERC_DUP_SUM
    precond: int = ERC_PRECOND_NONE

    def c(self):
        p = ErcParamsC()
        p.seed, p.K, p.kc, p.eps, p.tol = self.seed, self.K, self.kc, self.eps, self.tol
        p.max_iter, p.eta, p.dup_policy = self.max_iter, self.eta, self.dup_policy
        p.precond = self.precond
        return p


def _run_outputs(n, m_in, K, device, pin=False):
    kw = dict(device=device) if not pin else dict(pin_memory=True)
    c1 = max(m_in, 1)
    return dict(eu=torch.empty(c1, dtype=torch.int32, **kw),
                ev=torch.empty(c1, dtype=torch.int32, **kw),
                R=torch.empty(c1, dtype=torch.float32, **kw),
                p=torch.empty(n, dtype=torch.float32, **kw),
                kappa=torch.empty(c1, dtype=torch.float32, **kw),
                prob_node=torch.empty(n, dtype=torch.float32, **kw),
                prob_edge=torch.empty(c1, dtype=torch.float32, **kw),
                iters=torch.empty(K, dtype=torch.int32, **kw),
                relres=torch.empty(K, dtype=torch.float32, **kw))


def _trim(out, m):
    for k in ("eu", "ev", "R", "kappa", "prob_edge"):
        out[k] = out[k][:m]
    out["m"] = m
    return out


def erc_run_workspace(n, m_in, params, device="cuda"):
    return _workspace(lib().erc_run_workspace_size(n, m_in, params.kc), device)


def erc_run(n, src, dst, w, params, ws=None, out=None):
    """The whole path on device-resident inputs; returns a dict of device tensors + status."""
    dev = src.device
    m_in = src.numel()
    if ws is None:
        ws = erc_run_workspace(n, m_in, params, dev)
    o = _run_outputs(n, m_in, params.K, dev) if out is None else out
    m = _i64(0)
    pc = params.c()
    st = _check(lib().erc_run(ctypes.byref(pc), n, _ptr(src), _ptr(dst), _ptr(w), m_in,
                              ctypes.byref(m), _ptr(o["eu"]), _ptr(o["ev"]), _ptr(o["R"]),
                              _ptr(o["p"]), _ptr(o["kappa"]), _ptr(o["prob_node"]),
                              _ptr(o["prob_edge"]), _ptr(o["iters"]), _ptr(o["relres"]),
                              _ptr(ws), ws.numel(), _stream()), allow=(ERC_ERR_NOT_CONVERGED,))
    res = _trim(dict(o), m.value)
    res["status"] = st
    return res


def erc_run_host_workspace(n, m_in, params, device="cuda"):
    return _workspace(lib().erc_run_host_workspace_size(n, m_in, params.kc, params.K), device)


def erc_run_host(n, src, dst, w, params, ws=None, out=None):
    """The whole path from host (ideally pinned) inputs to host outputs, copies included."""
    m_in = src.numel()
    if ws is None:
        ws = erc_run_host_workspace(n, m_in, params)
    o = _run_outputs(n, m_in, params.K, None, pin=True) if out is None else out
    m = _i64(0)
    pc = params.c()
    st = _check(lib().erc_run_host(ctypes.byref(pc), n, _ptr(src), _ptr(dst), _ptr(w), m_in,
                                   ctypes.byref(m), _ptr(o["eu"]), _ptr(o["ev"]), _ptr(o["R"]),
                                   _ptr(o["p"]), _ptr(o["kappa"]), _ptr(o["prob_node"]),
                                   _ptr(o["prob_edge"]), _ptr(o["iters"]), _ptr(o["relres"]),
                                   _ptr(ws), ws.numel(), _stream()),
                allow=(ERC_ERR_NOT_CONVERGED,))
    res = _trim(dict(o), m.value)
    res["status"] = st
    return res
