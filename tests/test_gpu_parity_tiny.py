"""Parity of the CUDA path (through the C ABI) with the oracle on the tiny
decoder (2 layers, d 256, 4 x 64 heads, SwiGLU 688, vocab 2048): in fp32 (the
SIMT kernels) and in bf16 (the tcgen05 GEMMs and tensor-core attention, with
ragged 688-wide tiles).  Same seeded weights, prompts and guesses on both
sides."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from tests.parity_util import FLAG_GAP, engine_for, first_flag, logits_ok, oracle_for

pytestmark = pytest.mark.gpu

MAX_SEQ = 160


@pytest.fixture(scope="module", params=["f32", "bf16"])
def pair(request):
    cfg = syn.TINY if request.param == "f32" else syn.TINY_BF16
    w_cpu = syn.make_weights(cfg, seed=0, device="cpu")
    w_gpu = syn.weights_to(w_cpu, "cuda")
    eng = engine_for(cfg, w_gpu, max_batch=4, max_seq=MAX_SEQ, max_block=16)
    yield cfg, eng, oracle_for(cfg, w_cpu)
    eng.close()


def test_prefill_head(pair):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=1)
    heads = eng.prefill(prompts)
    for b, p in enumerate(prompts):
        tok, gap, _ = orc.prefill(om.session(MAX_SEQ), p)
        if gap >= FLAG_GAP:
            assert heads[b] == tok


@pytest.mark.parametrize("n", [1, 8, 16])
def test_step_logits_tokens_accepted(pair, n):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=1)
    guesses = syn.make_guesses(cfg.vocab, len(prompts), n, seed=2)
    eng.prefill(prompts)
    r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
    flagged = 0
    for b, p in enumerate(prompts):
        s = om.session(MAX_SEQ)
        head, _, _ = orc.prefill(s, p)
        blk = [head] + guesses[b][1:]
        st = orc.jacobi_step(s, blk, len(p), keep_logits=True)
        ok, worst = logits_ok(r["logits"][b], st.logits, cfg.dtype)
        assert ok, f"b={b} logits err/bound={worst:.3g}"
        for k in range(n):
            if st.gap[k] < FLAG_GAP:
                flagged += 1
            else:
                assert r["next"][b][k] == st.pred[k], (b, k)
        rows_ok = all(g >= FLAG_GAP for g in st.gap[: st.accepted])
        if rows_ok:
            assert r["accepted"][b] == st.accepted
        np.testing.assert_allclose(r["gap"][b], st.gap, atol=1e-2 if cfg.dtype == "bf16" else 1e-4)
    print(f"flagged rows: {flagged}/{n * len(prompts)}")


def test_step_commits_and_continues(pair):
    """Two consecutive steps: the second one runs on the KV committed by the first."""
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 20], seed=3)
    n = 8
    eng.prefill(prompts)
    g1 = syn.make_guesses(cfg.vocab, 2, n, seed=4)
    g2 = syn.make_guesses(cfg.vocab, 2, n, seed=5)
    r1 = eng.jacobi_step(g1)
    r2 = eng.jacobi_step(g2, want_logits=True)
    for b, p in enumerate(prompts):
        s = om.session(MAX_SEQ)
        head, _, _ = orc.prefill(s, p)
        st1 = orc.jacobi_step(s, [head] + g1[b][1:], len(p))
        if min(st1.gap) < FLAG_GAP:
            continue  # trajectories may legitimately differ after a near-tie
        assert r1["accepted"][b] == st1.accepted
        L = len(p) + st1.accepted
        st2 = orc.jacobi_step(s, [st1.pred[st1.accepted - 1]] + g2[b][1:], L, keep_logits=True)
        ok, worst = logits_ok(r2["logits"][b], st2.logits, cfg.dtype)
        assert ok, worst
    assert list(eng.committed_lengths()) == [len(p) + a for p, a in
                                             zip(prompts, (r1["accepted"] + r2["accepted"]).tolist())]


@pytest.mark.parametrize("n,seed", [(8, 2), (4, 7)])
def test_decode_matches_oracle(pair, n, seed):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=1)
    max_new = 64
    out, iters = eng.jacobi_decode(prompts, n, max_new, seed=seed)
    thr = 1e-4 if cfg.dtype == "f32" else FLAG_GAP
    for b, p in enumerate(prompts):
        ar = orc.ar_decode(om, p, max_new)
        k = first_flag(ar.min_gap, thr)
        assert out[b][:k].tolist() == ar.tokens[:k], f"b={b} first flag {k}"
        jr = orc.jacobi_decode(om, p, n, max_new, seed=seed, b=b)
        if min(jr.min_gap_all) >= thr and k == max_new:
            assert iters[b] == jr.iterations
            assert out[b].tolist() == jr.tokens


def test_ar_decode_matches_oracle(pair):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 9], seed=6)
    out = eng.ar_decode(prompts, 40)
    thr = 1e-4 if cfg.dtype == "f32" else FLAG_GAP
    for b, p in enumerate(prompts):
        ar = orc.ar_decode(om, p, 40)
        k = first_flag(ar.min_gap, thr)
        assert out[b][:k].tolist() == ar.tokens[:k]


def test_gpu_jacobi_equals_gpu_ar(pair):
    """The fixed point is the greedy AR output (Sec. 3.1) on the GPU itself,
    bit for bit: every kernel's result for a row is independent of n."""
    cfg, eng, _ = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=8)
    ar = eng.ar_decode(prompts, 48)
    for n in (4, 16):
        jac, _ = eng.jacobi_decode(prompts, n, 48, seed=3)
        np.testing.assert_array_equal(jac, ar)


def test_guess_from_prompt_and_eos(pair):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32], seed=1)
    ar = orc.ar_decode(om, prompts[0], 30)
    thr = 1e-4 if cfg.dtype == "f32" else FLAG_GAP
    k = first_flag(ar.min_gap, thr)
    out, _ = eng.jacobi_decode(prompts, 8, 30, seed=4, guess_init=1)
    assert out[0][:k].tolist() == ar.tokens[:k]
    if k >= 12:
        eos = ar.tokens[10]
        stop = ar.tokens.index(eos)
        out, _ = eng.jacobi_decode(prompts, 8, 30, seed=4, eos_id=eos)
        assert out[0][: stop + 1].tolist() == ar.tokens[: stop + 1]
        assert (out[0][stop + 1:] == -1).all()


def test_errors_are_reported(pair):
    from paper_2403_00835_gb300.cllm import CllmError
    cfg, eng, _ = pair
    with pytest.raises(CllmError) as e:
        eng.prefill([[cfg.vocab]])  # token outside the vocabulary
    assert e.value.status == -1
    with pytest.raises(CllmError) as e:
        eng.jacobi_decode([[1] * 100], 16, 60)  # 100 + 60 + 16 > max_seq
    assert e.value.status == -4
    eng.prefill([[1, 2, 3]])
    with pytest.raises(CllmError) as e:
        eng.jacobi_step([[0] * 17])  # n > max_block
    assert e.value.status == -1


@pytest.mark.parametrize("n", [32, 48, 64])
def test_wide_block_step(n):
    """Blocks of 2-4 query tiles per sequence: the tensor-core attention runs a
    group of tiles against each staged key chunk; logits and tokens against the
    oracle, batch 2 with ragged prompts."""
    cfg = syn.TINY_BF16
    w_cpu = syn.make_weights(cfg, seed=0, device="cpu")
    eng = engine_for(cfg, syn.weights_to(w_cpu, "cuda"), max_batch=2, max_seq=256, max_block=64)
    om = oracle_for(cfg, w_cpu)
    try:
        prompts = syn.make_prompts(cfg.vocab, [150, 37], seed=11)
        guesses = syn.make_guesses(cfg.vocab, len(prompts), n, seed=12)
        eng.prefill(prompts)
        r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
        for b, p in enumerate(prompts):
            s = om.session(256)
            head, _, _ = orc.prefill(s, p)
            st = orc.jacobi_step(s, [head] + guesses[b][1:], len(p), keep_logits=True)
            ok, worst = logits_ok(r["logits"][b], st.logits, cfg.dtype)
            assert ok, f"b={b} logits err/bound={worst:.3g}"
            for k in range(n):
                if st.gap[k] >= FLAG_GAP:
                    assert r["next"][b][k] == st.pred[k], (b, k)
    finally:
        eng.close()
