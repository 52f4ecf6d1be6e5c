"""Edge cases of the CUDA path against the fp64 oracle and against the CUDA
path's own greedy decode:

  * context lengths at and around the attention's key-chunk (128) and range
    (512 keys) boundaries, up to a 4096-token prefix, in ragged batches;
  * the accept rule (Alg. 3's i*) with planted correct prefixes of every
    length, several lengths in one batch;
  * the argmax with planted exact ties (duplicated LM-head rows): the lowest
    vocabulary index wins and the reported top-1/top-2 gap is exactly 0;
  * EOS in a ragged batch (one sequence stops while the others run on);
  * max_new truncation of the last block;
  * resume: prefill(prompt + committed tokens) and continuing gives the
    uninterrupted decode's remaining tokens (greedy decoding is deterministic;
    the fixed point of every Jacobi block is the greedy continuation, Sec. 3.1).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from paper_2403_00835_gb300.cllm import CLLM_BLOCK_REFILL, CLLM_BLOCK_SHRINK
from tests.parity_util import FLAG_GAP, engine_for, logits_ok, oracle_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tiny_bf16():
    cfg = syn.TINY_BF16
    w_cpu = syn.make_weights(cfg, seed=0, device="cpu")
    return cfg, w_cpu, syn.weights_to(w_cpu, "cuda")


@pytest.mark.parametrize("lens", [[1, 127, 128, 129], [255, 256, 257, 511], [512, 513, 1023, 4096]])
def test_context_lengths(tiny_bf16, lens):
    """One Jacobi step (n = 16) over prefixes that end just before, at and
    just after the key-chunk and range boundaries; logits and tokens against
    the oracle."""
    cfg, w_cpu, w_gpu = tiny_bf16
    n = 16
    max_seq = max(lens) + n + 16
    eng = engine_for(cfg, w_gpu, max_batch=len(lens), max_seq=max_seq, max_block=n)
    om = oracle_for(cfg, w_cpu)
    try:
        prompts = syn.make_prompts(cfg.vocab, lens, seed=21)
        guesses = syn.make_guesses(cfg.vocab, len(lens), n, seed=22)
        heads = eng.prefill(prompts)
        r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
        for b, p in enumerate(prompts):
            s = om.session(len(p) + n + 1)
            ohead, ogap, _ = orc.prefill(s, p)
            if ogap >= FLAG_GAP:
                assert heads[b] == ohead, f"L={len(p)}: prefill head"
            st = orc.jacobi_step(s, [ohead] + guesses[b][1:], len(p), keep_logits=True)
            s.close()
            ok, worst = logits_ok(r["logits"][b], st.logits, cfg.dtype)
            assert ok, f"L={len(p)}: logits err/bound {worst:.3g}"
            for k in range(n):
                if st.gap[k] >= FLAG_GAP:
                    assert r["next"][b][k] == st.pred[k], (len(p), k)
    finally:
        eng.close()


def test_empty_prompt_is_rejected(tiny_bf16):
    from paper_2403_00835_gb300.cllm import CllmError
    cfg, _, w_gpu = tiny_bf16
    eng = engine_for(cfg, w_gpu, max_batch=2, max_seq=64, max_block=8)
    try:
        with pytest.raises(CllmError) as e:
            eng.prefill([[1, 2, 3], []])
        assert e.value.status == -1
    finally:
        eng.close()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_planted_prefixes(dtype):
    """A block whose first m + 1 tokens are the greedy continuation (the head
    and m correct guesses) followed by wrong guesses commits exactly m + 1
    tokens (Alg. 3: i* is the first position whose guess differs from the
    prediction), and its first m + 1 predictions are the next greedy tokens.
    The greedy continuation is the CUDA path's own AR decode, so the check is
    exact; the oracle's step agrees wherever it has no near-tie."""
    cfg = syn.TINY if dtype == "f32" else syn.TINY_BF16
    w_cpu = syn.make_weights(cfg, seed=0, device="cpu")
    n = 16
    ms = [0, 1, 5, 14, 15]
    eng = engine_for(cfg, syn.weights_to(w_cpu, "cuda"), max_batch=len(ms), max_seq=128, max_block=n)
    om = oracle_for(cfg, w_cpu)
    try:
        prompts = syn.make_prompts(cfg.vocab, [40, 23, 57, 31, 18], seed=31)
        ar = eng.ar_decode(prompts, n + 1)          # y_0 .. y_n of every sequence
        noise = syn.make_guesses(cfg.vocab, len(ms), n, seed=32)
        guesses = []
        for b, m in enumerate(ms):
            g = ar[b][: m + 1].tolist()
            for k in range(m + 1, n):
                t = noise[b][k]
                g.append(t if t != ar[b][k] else (t + 1) % cfg.vocab)
            guesses.append(g)
        eng.prefill(prompts)
        r = eng.jacobi_step(guesses, want_gap=True)
        for b, m in enumerate(ms):
            assert r["accepted"][b] == m + 1, (b, m)
            assert r["next"][b][: m + 1].tolist() == ar[b][1: m + 2].tolist(), (b, m)
            s = om.session(len(prompts[b]) + n + 1)
            orc.prefill(s, prompts[b])
            st = orc.jacobi_step(s, guesses[b], len(prompts[b]))
            s.close()
            thr = 1e-4 if dtype == "f32" else FLAG_GAP
            if min(st.gap[: m + 1]) >= thr:
                assert st.accepted == m + 1, (b, m)
        assert (eng.committed_lengths() == np.array([len(p) + m + 1 for p, m in zip(prompts, ms)])).all()
    finally:
        eng.close()


def test_argmax_planted_ties():
    """LM-head rows duplicated in pairs (row 2i + 1 = row 2i): every logit ties
    exactly with its partner, so the argmax must return the even index (the
    lowest index among equal maxima) and the top-1/top-2 gap must be 0.  The
    winning pair is compared with the oracle where the oracle's best and
    second-best pair are at least 0.05 apart."""
    cfg = syn.TINY_BF16
    w_cpu = syn.make_weights(cfg, seed=5, device="cpu")
    lm = w_cpu["lm_head"]
    lm[1::2] = lm[0::2]
    n = 16
    eng = engine_for(cfg, syn.weights_to(w_cpu, "cuda"), max_batch=2, max_seq=128, max_block=n)
    om = oracle_for(cfg, w_cpu)
    try:
        prompts = syn.make_prompts(cfg.vocab, [33, 60], seed=41)
        guesses = syn.make_guesses(cfg.vocab, 2, n, seed=42)
        heads = eng.prefill(prompts)
        assert (heads % 2 == 0).all()
        r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
        assert (r["next"] % 2 == 0).all(), r["next"]
        assert (r["gap"] == 0.0).all()
        compared = 0
        for b, p in enumerate(prompts):
            s = om.session(len(p) + n + 1)
            orc.prefill(s, p)
            st = orc.jacobi_step(s, [int(heads[b])] + guesses[b][1:], len(p), keep_logits=True)
            s.close()
            for k in range(n):
                pairs = np.asarray(st.logits[k], dtype=np.float64)[0::2]
                top = np.sort(pairs)[-2:]
                assert st.pred[k] % 2 == 0 and st.gap[k] == 0.0
                if top[1] - top[0] >= FLAG_GAP:
                    compared += 1
                    assert r["next"][b][k] == st.pred[k], (b, k)
        assert compared > 0
    finally:
        eng.close()


def test_eos_in_ragged_batch(tiny_bf16):
    """A sequence that emits EOS stops (its later slots stay -1, its iteration
    count stops growing) while the other sequences of the batch run on to
    max_new; every sequence's tokens are the greedy ones up to its stop."""
    cfg, _, w_gpu = tiny_bf16
    eng = engine_for(cfg, w_gpu, max_batch=3, max_seq=160, max_block=16)
    try:
        prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=51)
        max_new = 40
        ar = eng.ar_decode(prompts, max_new)
        # an EOS token that sequence 0 emits early and sequence 2 never emits
        eos = None
        for t in ar[0][3:12]:
            if int(t) not in ar[2].tolist():
                eos = int(t)
                break
        if eos is None:
            pytest.skip("no token of sequence 0 is absent from sequence 2")
        stops = []
        for b in range(3):
            row = ar[b].tolist()
            stops.append(row.index(eos) if eos in row else max_new)
        ar_eos = eng.ar_decode(prompts, max_new, eos_id=eos)
        for n in (4, 16):
            for mode in (CLLM_BLOCK_REFILL, CLLM_BLOCK_SHRINK):
                out, its = eng.jacobi_decode(prompts, n, max_new, seed=7, eos_id=eos, block_mode=mode)
                np.testing.assert_array_equal(out, ar_eos)
                for b in range(3):
                    k = stops[b]
                    assert out[b][: min(k + 1, max_new)].tolist() == ar[b][: min(k + 1, max_new)].tolist()
                    assert (out[b][k + 1:] == -1).all()
                assert stops[2] == max_new and (out[2] >= 0).all()
                assert its[0] <= its[2]
    finally:
        eng.close()


@pytest.mark.parametrize("max_new", [1, 7, 13, 16, 17])
def test_max_new_truncation(tiny_bf16, max_new):
    """The last block is cut at max_new: exactly max_new tokens, the greedy
    ones, and the committed lengths grow by max_new."""
    cfg, _, w_gpu = tiny_bf16
    eng = engine_for(cfg, w_gpu, max_batch=2, max_seq=128, max_block=8)
    try:
        prompts = syn.make_prompts(cfg.vocab, [21, 34], seed=61)
        ar = eng.ar_decode(prompts, 24)
        out, its = eng.jacobi_decode(prompts, 8, max_new, seed=2)
        assert out.shape == (2, max_new)
        np.testing.assert_array_equal(out, ar[:, :max_new])
        assert (its >= 1).all() and (its <= max_new).all()
        assert eng.committed_lengths().tolist() == [len(p) + max_new for p in prompts]
    finally:
        eng.close()


@pytest.mark.parametrize("m", [7, 16])
def test_resume_equals_uninterrupted(tiny_bf16, m):
    """Checkpoint/resume: the state of a decode is its prompt plus committed
    tokens.  Prefilling that and decoding the rest gives the uninterrupted
    decode's remaining tokens, for AR and for Jacobi decoding (refill and
    shrink).  (The resumed Jacobi decode draws its guesses from a restarted
    iteration counter, so its iteration counts may differ; its tokens may not.)"""
    cfg, _, w_gpu = tiny_bf16
    eng = engine_for(cfg, w_gpu, max_batch=3, max_seq=192, max_block=16)
    try:
        prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=71)
        total = 40
        full = eng.ar_decode(prompts, total)
        resumed_prompts = [p + full[b][:m].tolist() for b, p in enumerate(prompts)]
        rest = eng.ar_decode(resumed_prompts, total - m)
        np.testing.assert_array_equal(rest, full[:, m:])
        for mode in (CLLM_BLOCK_REFILL, CLLM_BLOCK_SHRINK):
            jac, _ = eng.jacobi_decode(prompts, 8, total, seed=3, block_mode=mode)
            np.testing.assert_array_equal(jac, full)
            jrest, _ = eng.jacobi_decode(resumed_prompts, 8, total - m, seed=3, block_mode=mode)
            np.testing.assert_array_equal(jrest, full[:, m:])
    finally:
        eng.close()
