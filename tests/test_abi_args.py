"""Argument checks of the C ABI that run before any CUDA call (CPU, no GPU):
bad shapes are CLLM_EINVAL, shapes this build does not handle are
CLLM_EUNSUPPORTED, and every call on a null context is CLLM_EINVAL.  Only
invalid inputs are passed: a valid one would go on to touch the device."""
import ctypes

import pytest

from paper_2403_00835_gb300 import cllm

EINVAL, EUNSUPPORTED = -1, -8


@pytest.fixture(scope="module")
def lib():
    return cllm.load()


def _arch(**kw):
    a = dict(n_layers=2, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64, ffn=688, vocab=2048,
             rms_eps=1e-6, rope_theta=1e4, dtype=cllm.CLLM_BF16, max_batch=2, max_seq=128,
             max_block=16)
    a.update(kw)
    return cllm.Arch(*[a[f] for f, _ in cllm.Arch._fields_])


def _weights(null=None):
    arr = (ctypes.c_void_p * 2)(0x1000, 0x2000)  # never dereferenced: the checks fail first
    pp = ctypes.cast(arr, ctypes.POINTER(ctypes.c_void_p))
    w = cllm.Weights(0x1000, 0x2000, 0x3000, *([pp] * 9))
    if null is not None:
        setattr(w, null, None)
    return w, arr


def _create(lib, arch, w):
    h = ctypes.c_void_p()
    rc = lib.cllm_create(ctypes.byref(arch), ctypes.byref(w), None, ctypes.byref(h))
    assert not h.value
    return rc


@pytest.mark.parametrize("field,value", [
    ("n_layers", 0), ("d_model", 64), ("n_heads", 0), ("n_kv_heads", 0), ("vocab", 1),
    ("ffn", 4), ("max_batch", 0), ("max_batch", 129), ("max_seq", 1), ("max_block", 0),
    ("rms_eps", float("nan")), ("rms_eps", -1.0), ("rope_theta", 0.0), ("dtype", 7)])
def test_create_rejects_bad_shapes(lib, field, value):
    w, _keep = _weights()
    assert _create(lib, _arch(**{field: value}), w) == EINVAL


@pytest.mark.parametrize("kw", [
    dict(head_dim=96, n_heads=4, n_kv_heads=4, d_model=384),  # head dim other than 64 / 128
    dict(d_model=320),                                         # not a multiple of 128
    dict(n_heads=6, n_kv_heads=4, d_model=384),                # heads not a multiple of kv heads
    dict(ffn=690),                                             # ffn not a multiple of 8
])
def test_create_reports_unsupported_shapes(lib, kw):
    w, _keep = _weights()
    assert _create(lib, _arch(**kw), w) == EUNSUPPORTED


@pytest.mark.parametrize("name", [f for f, _ in cllm.Weights._fields_])
def test_create_rejects_missing_weights(lib, name):
    w, _keep = _weights(null=name)
    assert _create(lib, _arch(), w) == EINVAL


def test_calls_on_a_null_context(lib):
    i32 = ctypes.c_int32
    toks = (i32 * 4)(1, 2, 3, 4)
    lens = (i32 * 1)(4)
    out = (i32 * 16)()
    acc = (i32 * 1)()
    assert lib.cllm_prefill(None, 1, toks, lens, out) == EINVAL
    assert lib.cllm_jacobi_step(None, toks, 4, out, acc, None, None) == EINVAL
    assert lib.cllm_jacobi_decode(None, 1, toks, lens, 4, 8, None, out, acc) == EINVAL
    assert lib.cllm_ar_decode(None, 1, toks, lens, 8, -1, out) == EINVAL
    assert lib.cllm_decode_begin(None, 4, 8, None) == EINVAL
    assert lib.cllm_decode_run(None, 1, None, None) == EINVAL
    assert lib.cllm_decode_read(None, out, acc) == EINVAL
    assert lib.cllm_decode_read_trajectory(None, out) == EINVAL
    assert lib.cllm_committed_lengths(None, out) == EINVAL
    assert lib.cllm_set_profiling(None, 1) == EINVAL
