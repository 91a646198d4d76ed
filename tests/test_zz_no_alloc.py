"""erc_sampling_probs_noalloc: the workspace-free variant for callers that cannot allocate.

Some callers cannot allocate device memory (plug-ins whose host owns every device buffer, code
that must not let cudaMalloc / cudaFree synchronise the device, fixed memory budgets).  This entry
point takes its scratch from a static device array inside the library instead of a caller
workspace.  Its results must match erc_sampling_probs on the same inputs, on consecutive calls
that reuse the shared array.  This file is named to be collected last.
"""
import numpy as np
import pytest
import torch

from paper_2609_27209_gb300 import erc, synth

pytestmark = pytest.mark.gpu


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).to("cuda:0")


def test_noalloc_matches_workspace_variant_on_consecutive_calls():
    n, src, dst, w = synth.random_connected(6000, 30000, seed=21, weighted=True)
    g = erc.erc_build_laplacian(n, _dev(src), _dev(dst), _dev(w))
    for call, seed in enumerate([31, 32]):
        kappa = _dev(synth.random_normal(g.m, seed=seed, scale=2.0 + call))
        ref_n, ref_e = erc.erc_sampling_probs(g, kappa, 1e-8)
        pn, pe = erc.erc_sampling_probs_noalloc(g, kappa, 1e-8)
        torch.cuda.synchronize()
        np.testing.assert_allclose(pn.cpu().numpy(), ref_n.cpu().numpy(), rtol=1e-6, atol=1e-12)
        np.testing.assert_allclose(pe.cpu().numpy(), ref_e.cpu().numpy(), rtol=1e-6)


def test_noalloc_uniform_fallback_after_a_regular_call():
    # an 8-cycle plus 4 isolated nodes with equal curvature: the node weights of Eq. 7 vanish
    n = 12
    src = np.arange(8, dtype=np.int32)
    dst = ((np.arange(8) + 1) % 8).astype(np.int32)
    g = erc.erc_build_laplacian(n, _dev(src), _dev(dst))
    kappa = _dev(np.full(g.m, 0.5, np.float32))
    pn, pe = erc.erc_sampling_probs_noalloc(g, kappa, 1e-8)
    np.testing.assert_allclose(pn.cpu().numpy(), [1 / 8] * 8 + [0] * 4, rtol=1e-7)
    np.testing.assert_allclose(pe.cpu().numpy(), 1 / 8, rtol=1e-7)


def test_noalloc_rejects_graphs_beyond_its_limit():
    n, src, dst, w = synth.random_connected(100, 300, seed=5)
    g = erc.erc_build_laplacian(n, _dev(src), _dev(dst))
    import ctypes

    # the size check runs on the host before anything touches the device
    big = erc.ErcGraphC.from_buffer_copy(g.c())
    big.n = 4000001  # one node past ERC_SAMPLING_PROBS_NOALLOC_MAX_NODES
    kappa = _dev(np.zeros(g.m, np.float32))
    out = torch.empty(g.m, dtype=torch.float32, device="cuda:0")
    st = erc.lib().erc_sampling_probs_noalloc(ctypes.byref(big), erc._ptr(kappa), 1e-8,
                                              erc._ptr(out), erc._ptr(out), erc._stream())
    assert st == erc.ERC_ERR_CAPACITY
    assert b"at most 4000000 nodes" in erc.lib().erc_last_error()


def test_noalloc_call_allocates_no_device_memory():
    """With its outputs preallocated, a warmed-up call leaves the device's free memory and the
    torch allocator's reservation unchanged: the scratch is the library's static array."""
    n, src, dst, w = synth.random_connected(50_000, 200_000, seed=23, weighted=True)
    g = erc.erc_build_laplacian(n, _dev(src), _dev(dst), _dev(w))
    kappa = _dev(synth.random_normal(g.m, seed=33, scale=1.5))
    out = (torch.empty(g.n, dtype=torch.float32, device="cuda:0"),
           torch.empty(g.m, dtype=torch.float32, device="cuda:0"))
    erc.erc_sampling_probs_noalloc(g, kappa, 1e-8, out=out)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    reserved0 = torch.cuda.memory_reserved()
    for _ in range(3):
        erc.erc_sampling_probs_noalloc(g, kappa, 1e-8, out=out)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert torch.cuda.memory_reserved() == reserved0
    ref_n, ref_e = erc.erc_sampling_probs(g, kappa, 1e-8)
    np.testing.assert_allclose(out[0].cpu().numpy(), ref_n.cpu().numpy(), rtol=1e-6, atol=1e-12)
    np.testing.assert_allclose(out[1].cpu().numpy(), ref_e.cpu().numpy(), rtol=1e-6)
