"""The C-ABI library builds for sm_103a, loads without a GPU, and exports
every entry point include/csrtrain.h declares (no compute calls here)."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def libpath():
    from paper_1905_07931_gb300 import build
    return build.build()


def _declared():
    with open(os.path.join(ROOT, "include", "csrtrain.h")) as f:
        src = f.read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?(?:int|int64_t|char\s*\*|const char\s*\*)\s*\*?\s*(\w+)\s*\(", src, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_paper_calls():
    names = _declared()
    for n in ["csr_from_dense", "spmm_fwd", "spmm_bwd_t", "weight_grad_dense", "weight_grad_sddmm",
              "prox_update_compact", "debias_update", "csr_transpose"]:
        assert n in names


def test_library_exports_every_declared_symbol(libpath):
    lib = ctypes.CDLL(libpath)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_covers_the_header(libpath):
    from paper_1905_07931_gb300 import csrtrain
    assert sorted(csrtrain.exported_symbols()) == _declared()


def test_host_only_calls_work_without_gpu(libpath):
    from paper_1905_07931_gb300 import csrtrain
    L = csrtrain.lib()
    n = ctypes.c_size_t(0)
    assert L.csrt_workspace_bytes(4096, 9216, 256, ctypes.byref(n)) == 0
    assert n.value >= 256
    assert L.csrt_workspace_bytes(-1, 3, 3, ctypes.byref(n)) == csrtrain.CSRT_ERR_ARG
    assert b"negative" in L.csrt_last_error()
