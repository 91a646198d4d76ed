"""Helpers shared by the GPU parity tests (inputs come from synth, references from oracle)."""
import numpy as np
import torch

from oracle import erc_oracle as O
from paper_2609_27209_gb300 import erc


def dev():
    return torch.device("cuda:0")


def to_dev(a):
    return None if a is None else torch.from_numpy(np.ascontiguousarray(a)).to(dev())


def host(t):
    return t.detach().cpu().numpy()


def build_both(n, src, dst, w=None, policy=0):
    """(GPU graph, oracle graph) of the same edge list."""
    g = erc.erc_build_laplacian(n, to_dev(src), to_dev(dst), to_dev(w), policy)
    ref = O.build_laplacian(n, src, dst, w, "sum" if policy == 0 else "first")
    return g, ref


def assert_graph_equal(g, ref):
    assert g.m == ref["m"]
    np.testing.assert_array_equal(host(g.row_ptr), ref["row_ptr"])
    np.testing.assert_array_equal(host(g.col), ref["col"])
    np.testing.assert_array_equal(host(g.csr_eid), ref["csr_eid"])
    np.testing.assert_array_equal(host(g.eu), ref["eu"])
    np.testing.assert_array_equal(host(g.ev), ref["ev"])
    np.testing.assert_array_equal(host(g.val), ref["val"])
    np.testing.assert_array_equal(host(g.ew), ref["ew"])
    np.testing.assert_array_equal(host(g.deg), ref["deg"])
