"""The C ABI library builds for sm_103a, loads, and exports every entry point include/erc.h declares.

No compute call is made here, so these tests run without a GPU.
"""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "erc.h")


def declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(erc_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def libpath():
    import __graft_entry__

    __graft_entry__.build()
    from paper_2609_27209_gb300 import erc

    return erc.LIB_PATH


def test_header_declares_the_path_calls():
    names = declared()
    for must in ["erc_build_laplacian", "erc_jl_rhs", "erc_batched_cg", "erc_edge_resistance",
                 "erc_curvature", "erc_sampling_probs", "erc_run", "erc_run_host"]:
        assert must in names


def test_library_exports_every_declared_symbol(libpath):
    lib = ctypes.CDLL(libpath)
    for name in declared():
        assert hasattr(lib, name), name
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True)
    if out.returncode == 0:
        exported = set(re.findall(r"\s(erc_[a-z0-9_]+)$", out.stdout, flags=re.M))
        assert set(declared()) <= exported


def test_binding_covers_every_declared_symbol(libpath):
    from paper_2609_27209_gb300 import erc

    assert set(erc.exported_symbols()) == set(declared())
    assert "sm_103a" in erc.erc_version()


def test_library_is_built_for_sm_103a(libpath):
    from paper_2609_27209_gb300 import build

    assert build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
    assert os.path.getmtime(libpath) >= max(
        os.path.getmtime(os.path.join(build.CSRC, f)) for f in os.listdir(build.CSRC))


def test_struct_layouts_match_the_header(tmp_path):
    """sizeof and every field offset of erc_graph and erc_params, as a C compiler lays them out
    from include/erc.h, equal the binding's ctypes structures."""
    from paper_2609_27209_gb300 import erc

    structs = {"erc_graph": erc.ErcGraphC, "erc_params": erc.ErcParamsC}
    lines = ['#include <stddef.h>', '#include <stdio.h>', '#include "erc.h"', "int main(void) {"]
    for cname, cls in structs.items():
        lines.append(f'  printf("{cname} size %zu\\n", sizeof({cname}));')
        for field, _ in cls._fields_:
            lines.append(f'  printf("{cname} {field} %zu\\n", offsetof({cname}, {field}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    cc = subprocess.run(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o",
                         str(exe)], capture_output=True, text=True)
    if cc.returncode != 0 and "cuda_runtime" in cc.stderr:
        pytest.skip("the header needs the CUDA include path")
    assert cc.returncode == 0, cc.stderr
    got = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    seen = 0
    for line in got:
        if not line:
            continue
        cname, field, value = line.split()
        cls = structs[cname]
        expect = ctypes.sizeof(cls) if field == "size" else getattr(cls, field).offset
        assert int(value) == expect, (cname, field, value, expect)
        seen += 1
    assert seen == sum(len(c._fields_) + 1 for c in structs.values())


def test_binding_fails_loudly_without_library(monkeypatch):
    from paper_2609_27209_gb300 import erc

    monkeypatch.setattr(erc, "_lib", None)
    monkeypatch.setattr(erc, "LIB_PATH", os.path.join(ROOT, "does-not-exist.so"))
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        erc.lib()


def test_workspace_queries_need_no_gpu(libpath):
    from paper_2609_27209_gb300 import erc

    L = erc.lib()
    assert L.erc_build_laplacian_workspace_size(100, 1000) > 0
    assert L.erc_batched_cg_workspace_size(100, 64) > 100 * 64 * 4 * 3
    assert L.erc_run_workspace_size(100, 1000, 64) > L.erc_batched_cg_workspace_size(100, 64)
