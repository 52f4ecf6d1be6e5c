"""Parity on the coder-style 7B shape (vocab 32256, RoPE theta 1e5) with a
ragged batch: two sequences of different prompt lengths in one Jacobi step of
n = 32 (the batched, ragged-commit configuration), against the fp64 oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from tests.parity_util import FLAG_GAP, engine_for, logits_ok, oracle_for

pytestmark = pytest.mark.gpu


def test_coder7b_ragged_batch_step():
    cfg = syn.CODER7B
    w_gpu = syn.make_weights(cfg, seed=0, device="cuda")
    w_cpu = syn.weights_to(w_gpu, "cpu")
    n = 32
    lens = [256, 289]
    eng = engine_for(cfg, w_gpu, max_batch=2, max_seq=max(lens) + n + 16, max_block=n)
    try:
        om = oracle_for(cfg, w_cpu)
        prompts = syn.make_prompts(cfg.vocab, lens, seed=1)
        guesses = syn.make_guesses(cfg.vocab, 2, n, seed=2)
        heads = eng.prefill(prompts)
        r = eng.jacobi_step(guesses, want_gap=True, want_logits=True)
        for b, p in enumerate(prompts):
            s = om.session(len(p) + n + 1)
            ohead, ogap, _ = orc.prefill(s, p)
            if ogap >= FLAG_GAP:
                assert heads[b] == ohead
            st = orc.jacobi_step(s, [ohead] + guesses[b][1:], len(p), keep_logits=True)
            ok, worst = logits_ok(r["logits"][b], st.logits, "bf16")
            assert ok, f"b={b}: logits max err / (2e-2 std) = {worst:.3f}"
            flagged = [k for k in range(n) if st.gap[k] < FLAG_GAP]
            for k in range(n):
                if k not in flagged:
                    assert r["next"][b][k] == st.pred[k], (b, k)
            if all(g >= FLAG_GAP for g in st.gap[: st.accepted]):
                assert r["accepted"][b] == st.accepted
            print(f"b={b} len={len(p)}: worst logit err/bound {worst:.3f}, flagged {len(flagged)}/{n}")
    finally:
        eng.close()
