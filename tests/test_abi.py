"""The C-ABI library builds for sm_103a, loads without a GPU and exports every symbol
include/dcleap.h declares; the product path is independent of the oracle."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(dcl_[a-z0-9_]+)\s*\(", src))
    return names


@pytest.fixture(scope="module")
def built():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_20467_gb300 as pkg
    return pkg


def test_library_exports_every_declared_symbol(built):
    handle = ctypes.CDLL(built.LIB_PATH)
    declared = _declared()
    assert len(declared) >= 15
    for name in sorted(declared):
        assert hasattr(handle, name), f"{name} declared in include/ but not exported"
    # the binding wraps exactly the declared calls, under the same names
    assert set(built.SIGNATURES) == declared


def test_create_without_gpu_reports_error(built):
    """With no GPU the ABI returns a status (never aborts) and records a message."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    L = built.lib()
    out = ctypes.c_void_p()
    st = L.dcl_create(None, 1, 1, None, None, ctypes.byref(out))
    assert st != built.DCL_OK and out.value is None
    assert len(L.dcl_last_error(None)) > 0


def test_null_context_is_rejected(built):
    L = built.lib()
    assert L.dcl_step(None, None) == built.DCL_ERR_INVALID_ARG
    assert L.dcl_generate(None, 1, None, None) == built.DCL_ERR_INVALID_ARG
    L.dcl_destroy(None)


def test_product_path_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2607_20467_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                src = open(os.path.join(dirpath, fn)).read()
                assert not re.search(r"^\s*(from|import)\s+oracle\b", src, re.M), fn
                assert "oracle/" not in src, fn


def test_missing_library_fails_loudly(built, monkeypatch, tmp_path):
    """With libdcleap.so absent the binding raises instead of falling back to anything."""
    pkg = built
    monkeypatch.setattr(pkg, "LIB_PATH", str(tmp_path / "libdcleap.so"))
    monkeypatch.setattr(pkg, "_lib", None)
    with pytest.raises(ImportError, match="no CPU fallback"):
        pkg.lib()
    with pytest.raises(ImportError):
        pkg.Context(None, 1, 1)
