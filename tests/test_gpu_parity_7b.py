"""Parity at full model size: the LLaMA-2-7B shape in bf16 with random-init
weights, in the launch configuration the benchmark times (batch 1, 128-token
prompt, n = 16), and the wide-block configuration (512-token prompt, n = 64).
The oracle computes the same forward in fp64 on the host cores (tens of
seconds per configuration)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from tests.parity_util import FLAG_GAP, engine_for, first_flag, logits_ok, oracle_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def llama():
    cfg = syn.LLAMA7B
    w_gpu = syn.make_weights(cfg, seed=0, device="cuda")
    w_cpu = syn.weights_to(w_gpu, "cpu")
    eng = engine_for(cfg, w_gpu, max_batch=1, max_seq=512 + 64 + 64, max_block=64)
    yield cfg, eng, oracle_for(cfg, w_cpu)
    eng.close()


def _step_parity(cfg, eng, om, plen, n):
    prompt = syn.make_prompts(cfg.vocab, [plen], seed=1)[0]
    guess = syn.make_guesses(cfg.vocab, 1, n, seed=2)
    head = eng.prefill([prompt])[0]
    r = eng.jacobi_step(guess, want_gap=True, want_logits=True)
    s = om.session(plen + n + 1)
    ohead, ogap, _ = orc.prefill(s, prompt)
    if ogap >= FLAG_GAP:
        assert head == ohead
    st = orc.jacobi_step(s, [ohead] + guess[0][1:], plen, keep_logits=True)
    ok, worst = logits_ok(r["logits"][0], st.logits, "bf16")
    assert ok, f"logits max err / (2e-2 std) = {worst:.3f}"
    flagged = [k for k in range(n) if st.gap[k] < FLAG_GAP]
    for k in range(n):
        if k not in flagged:
            assert r["next"][0][k] == st.pred[k], k
    if all(g >= FLAG_GAP for g in st.gap[: st.accepted]):
        assert r["accepted"][0] == st.accepted
    print(f"n={n}: worst logit err/bound {worst:.3f}, flagged {len(flagged)}/{n}")
    return s, st


def test_7b_step_n16_prompt128(llama):
    cfg, eng, om = llama
    _step_parity(cfg, eng, om, 128, 16)


def test_7b_step_n64_prompt512(llama):
    cfg, eng, om = llama
    _step_parity(cfg, eng, om, 512, 64)


def test_7b_decode_prefix_matches_oracle_ar(llama):
    cfg, eng, om = llama
    prompt = syn.make_prompts(cfg.vocab, [128], seed=1)[0]
    out, _ = eng.jacobi_decode([prompt], 16, 24, seed=2)
    ar = orc.ar_decode(om, prompt, 24)
    k = first_flag(ar.min_gap)
    assert out[0][:k].tolist() == ar.tokens[:k]
    print(f"first flagged position {k} of 24")


def test_7b_gpu_jacobi_equals_gpu_ar(llama):
    """Sec. 3.1's fixed point = greedy AR, on the GPU at full size: the n = 16
    Jacobi decode and the n = 1 decode produce the same 256 tokens."""
    cfg, eng, _ = llama
    prompt = syn.make_prompts(cfg.vocab, [128], seed=1)[0]
    ar = eng.ar_decode([prompt], 256)
    jac, iters = eng.jacobi_decode([prompt], 16, 256, seed=2)
    np.testing.assert_array_equal(jac, ar)
    assert 1 <= iters[0] <= 256
