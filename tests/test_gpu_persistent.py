"""The persistent per-iteration kernel (one launch per Jacobi iteration, grid
barriers between phases) against the one-kernel-per-phase path: same work
split, reductions and epilogues, so predictions, gaps, accepted counts,
committed lengths and decoded tokens must be bit-identical."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2403_00835_gb300 import synthetic as syn
from tests.parity_util import engine_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny_bf16():
    cfg = syn.TINY_BF16
    w = syn.make_weights(cfg, seed=0, device="cuda")
    eng = engine_for(cfg, w, max_batch=4, max_seq=160, max_block=16)
    yield cfg, eng
    eng.close()


def _steps(eng, prompts, guesses_list, persistent):
    eng.set_persistent(persistent)
    eng.prefill(prompts)
    outs = []
    for g in guesses_list:
        r = eng.jacobi_step(g, want_gap=True)
        outs.append((r["next"].copy(), r["accepted"].copy(), r["gap"].copy()))
    return outs, eng.committed_lengths().copy()


@pytest.mark.parametrize("n", [1, 8, 16])
def test_persistent_steps_bit_identical(tiny_bf16, n):
    cfg, eng = tiny_bf16
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=1)
    gl = [syn.make_guesses(cfg.vocab, 3, n, seed=s) for s in (2, 3, 4)]
    eng.set_persistent(True)
    eng.prefill(prompts)
    assert eng.uses_persistent(n)
    a, la = _steps(eng, prompts, gl, True)
    b, lb = _steps(eng, prompts, gl, False)
    for (n1, a1, g1), (n2, a2, g2) in zip(a, b):
        np.testing.assert_array_equal(n1, n2)
        np.testing.assert_array_equal(a1, a2)
        np.testing.assert_array_equal(g1, g2)
    np.testing.assert_array_equal(la, lb)
    eng.set_persistent(True)


@pytest.mark.parametrize("n", [8, 16])
def test_persistent_logits_bit_identical(tiny_bf16, n):
    """A step asked for its logits runs the persistent kernel (the one the
    decode loop runs) and stores them from its LM-head phase; they equal the
    per-GEMM path's logits bit for bit."""
    cfg, eng = tiny_bf16
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=1)
    g = syn.make_guesses(cfg.vocab, 3, n, seed=2)
    out = []
    for persistent in (True, False):
        eng.set_persistent(persistent)
        eng.prefill(prompts)
        assert eng.uses_persistent(n) == persistent
        out.append(eng.jacobi_step(g, want_gap=True, want_logits=True))
    eng.set_persistent(True)
    a, b = out
    assert np.isfinite(a["logits"]).all()
    np.testing.assert_array_equal(a["logits"], b["logits"])
    np.testing.assert_array_equal(a["next"], b["next"])
    np.testing.assert_array_equal(a["gap"], b["gap"])
    np.testing.assert_array_equal(a["accepted"], b["accepted"])


def test_persistent_decode_bit_identical(tiny_bf16):
    cfg, eng = tiny_bf16
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45, 8], seed=5)
    eng.set_persistent(True)
    pa, ia = eng.jacobi_decode(prompts, 8, 64, seed=3)
    eng.set_persistent(False)
    pb, ib = eng.jacobi_decode(prompts, 8, 64, seed=3)
    eng.set_persistent(True)
    np.testing.assert_array_equal(pa, pb)
    np.testing.assert_array_equal(ia, ib)
    ar = eng.ar_decode(prompts, 64)
    np.testing.assert_array_equal(pa, ar)


def test_persistent_7b_decode_bit_identical():
    cfg = syn.LLAMA7B
    w = syn.make_weights(cfg, seed=0, device="cuda")
    eng = engine_for(cfg, w, max_batch=2, max_seq=128 + 64 + 64, max_block=64)
    prompts = syn.make_prompts(cfg.vocab, [128, 100], seed=1)
    try:
        for n in (16, 64):
            eng.set_persistent(True)
            eng.prefill(prompts)
            assert eng.uses_persistent(n)
            pa, ia = eng.jacobi_decode(prompts, n, 48, seed=2)
            eng.set_persistent(False)
            pb, ib = eng.jacobi_decode(prompts, n, 48, seed=2)
            np.testing.assert_array_equal(pa, pb)
            np.testing.assert_array_equal(ia, ib)
    finally:
        eng.close()


@pytest.mark.parametrize("n", [1, 16])
def test_persistent_dataflow_flags_bit_identical(tiny_bf16, n):
    """Attention and the O projection opened by completion flags (the
    default) or by grid barriers compute the same logits bit for bit."""
    cfg, eng = tiny_bf16
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=11)
    g = syn.make_guesses(cfg.vocab, 3, n, seed=12)
    out = []
    try:
        for flags in (True, False):
            eng.set_dataflow(flags)
            eng.prefill(prompts)
            assert eng.uses_persistent(n)
            out.append(eng.jacobi_step(g, want_gap=True, want_logits=True))
    finally:
        eng.set_dataflow(True)
    a, b = out
    np.testing.assert_array_equal(a["logits"], b["logits"])
    np.testing.assert_array_equal(a["next"], b["next"])
    np.testing.assert_array_equal(a["accepted"], b["accepted"])
