"""Parity above 128 block rows (B * n > 128), where a step runs the per-GEMM
kernels with a 256-wide token tile (129..256 rows) or several token tiles
(more than 256 rows) instead of the persistent kernel.

Tiny bf16 decoder: ragged batches of 9 and 18 sequences at n = 16 (144 and
288 rows) against the oracle, step by step and as a free-running decode.
Coder-style 7B shape: the benchmark's batched configuration (8 sequences,
n = 32, 256 rows) with its ragged prompt lengths; the oracle checks a sample
of the batch (the shortest sequence) row by row at full size, and every
sequence of a short-prompt batch."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from tests.parity_util import FLAG_GAP, engine_for, first_flag, logits_ok, oracle_for

pytestmark = pytest.mark.gpu

MAX_SEQ = 192


@pytest.fixture(scope="module")
def tiny():
    cfg = syn.TINY_BF16
    w_cpu = syn.make_weights(cfg, seed=0, device="cpu")
    w_gpu = syn.weights_to(w_cpu, "cuda")
    eng = engine_for(cfg, w_gpu, max_batch=18, max_seq=MAX_SEQ, max_block=16)
    yield cfg, eng, oracle_for(cfg, w_cpu)
    eng.close()


def _check_step(cfg, om, prompts, guesses, r, n, dtype):
    """Oracle step of every sequence vs the GPU's step outputs."""
    flagged = 0
    worst_all = 0.0
    for b, p in enumerate(prompts):
        s = om.session(len(p) + n + 1)
        head, _, _ = orc.prefill(s, p)
        st = orc.jacobi_step(s, [head] + list(guesses[b][1:]), len(p), keep_logits=True)
        ok, worst = logits_ok(r["logits"][b], st.logits, dtype)
        assert ok, f"b={b}: logits err/bound {worst:.3f}"
        worst_all = max(worst_all, worst)
        for k in range(n):
            if st.gap[k] < FLAG_GAP:
                flagged += 1
            else:
                assert r["next"][b][k] == st.pred[k], (b, k)
        if all(g >= FLAG_GAP for g in st.gap[: st.accepted]):
            assert r["accepted"][b] == st.accepted, b
        s.close()
    return worst_all, flagged


@pytest.mark.parametrize("B", [9, 18])
def test_tiny_wide_step(tiny, B):
    cfg, eng, om = tiny
    n = 16
    lens = syn.ragged_lens(B, 5, 60, seed=3)
    prompts = syn.make_prompts(cfg.vocab, lens, seed=1)
    guesses = syn.make_guesses(cfg.vocab, B, n, seed=2)
    eng.prefill(prompts)
    assert not eng.uses_persistent(n)
    r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
    worst, flagged = _check_step(cfg, om, prompts, guesses, r, n, "bf16")
    print(f"B={B} ({B * n} rows): worst logit err/bound {worst:.3f}, flagged {flagged}/{B * n}")


def test_tiny_wide_decode_matches_oracle_ar(tiny):
    cfg, eng, om = tiny
    B, n, max_new = 18, 16, 48
    lens = syn.ragged_lens(B, 5, 60, seed=4)
    prompts = syn.make_prompts(cfg.vocab, lens, seed=5)
    out, iters = eng.jacobi_decode(prompts, n, max_new, seed=2)
    for b, p in enumerate(prompts):
        ar = orc.ar_decode(om, p, max_new)
        k = first_flag(ar.min_gap)
        assert out[b][:k].tolist() == ar.tokens[:k], b
        assert 1 <= iters[b] <= max_new
    # the fixed point is the greedy AR output (Sec. 3.1), bit for bit on the GPU
    np.testing.assert_array_equal(out, eng.ar_decode(prompts, max_new))


@pytest.fixture(scope="module")
def coder():
    cfg = syn.CODER7B
    w_gpu = syn.make_weights(cfg, seed=0, device="cuda")
    w_cpu = syn.weights_to(w_gpu, "cpu")
    yield cfg, w_gpu, oracle_for(cfg, w_cpu)


def test_coder7b_b8_n32_benchmark_batch_sampled(coder):
    """The benchmark's batch (8 ragged prompts of 256..1024 tokens, n = 32):
    the GPU steps all 8 sequences in one 256-row forward; the oracle checks
    the shortest sequence's 32 rows (logits, predictions, accepted count)."""
    cfg, w_gpu, om = coder
    B, n = 8, 32
    lens = syn.ragged_lens(B, 256, 1024, seed=1)
    prompts = syn.make_prompts(cfg.vocab, lens, seed=1)
    guesses = syn.make_guesses(cfg.vocab, B, n, seed=2)
    eng = engine_for(cfg, w_gpu, max_batch=B, max_seq=max(lens) + n + 16, max_block=n)
    try:
        eng.prefill(prompts)
        assert not eng.uses_persistent(n)
        r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
    finally:
        eng.close()
    b = int(np.argmin(lens))
    sub = {k: (v[b:b + 1] if v is not None else None) for k, v in r.items()}
    worst, flagged = _check_step(cfg, om, [prompts[b]], guesses[b:b + 1], sub, n, "bf16")
    print(f"sequence {b} (len {lens[b]}) of {lens}: worst logit err/bound {worst:.3f}, "
          f"flagged {flagged}/{n}")


def test_coder7b_b8_n32_short_prompts_every_sequence(coder):
    """Same 256-row forward with short ragged prompts, so that the oracle can
    check every sequence of the batch."""
    cfg, w_gpu, om = coder
    B, n = 8, 32
    lens = syn.ragged_lens(B, 8, 48, seed=6)
    prompts = syn.make_prompts(cfg.vocab, lens, seed=7)
    guesses = syn.make_guesses(cfg.vocab, B, n, seed=8)
    eng = engine_for(cfg, w_gpu, max_batch=B, max_seq=max(lens) + n + 16, max_block=n)
    try:
        eng.prefill(prompts)
        r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
    finally:
        eng.close()
    worst, flagged = _check_step(cfg, om, prompts, guesses, r, n, "bf16")
    print(f"lens {lens}: worst logit err/bound {worst:.3f}, flagged {flagged}/{B * n}")
