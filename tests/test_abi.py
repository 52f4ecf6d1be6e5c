"""The C-ABI library loads (without a GPU) and exports every function the
headers in include/ declare.  No compute call is made here."""
import ctypes
import os
import re

import pytest

from paper_2403_00835_gb300 import cllm

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"^\s*(?:const\s+)?\w+\s*\**\s*(cllm_\w+)\s*\(", src, flags=re.M))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    return cllm.load()


def test_headers_declare_the_boundary():
    names = declared_functions()
    for required in ("cllm_create", "cllm_prefill", "cllm_jacobi_step", "cllm_jacobi_decode",
                     "cllm_ar_decode", "cllm_destroy", "cllm_status_string"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing
    assert set(cllm.EXPORTS) <= set(declared_functions())


def test_status_strings(lib):
    for code, name in cllm.STATUS.items():
        s = lib.cllm_status_string(code).decode()
        assert s and s != "unknown status", name
    assert lib.cllm_status_string(12345).decode() == "unknown status"


def test_create_rejects_null_arguments(lib):
    h = ctypes.c_void_p()
    assert lib.cllm_create(None, None, None, ctypes.byref(h)) == -1  # CLLM_EINVAL, no CUDA call
    lib.cllm_destroy(None)  # no-op


def test_library_is_in_tree():
    assert cllm.library_path().startswith(os.path.join(ROOT, "paper_2403_00835_gb300"))


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """No CPU fallback: without the built library the binding raises."""
    monkeypatch.setattr(cllm, "_lib", None)
    monkeypatch.setattr(cllm._build, "LIB", str(tmp_path / "absent" / "libcllm.so"))
    with pytest.raises(RuntimeError, match="not built"):
        cllm.load(build_if_missing=False)


def test_engine_rejects_host_weights():
    """The engine takes device weights only (PyTorch supplies memory, never compute)."""
    torch = pytest.importorskip("torch")
    from paper_2403_00835_gb300 import synthetic as syn
    w = syn.make_weights(syn.TINY, seed=0, device="cpu")
    with pytest.raises(ValueError, match="CUDA"):
        cllm.Engine(syn.TINY, w, max_batch=1, max_seq=64, max_block=8)
