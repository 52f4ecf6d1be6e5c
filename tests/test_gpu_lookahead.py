"""The lookahead combination (Sec. 3.3) on the CUDA path: the refill block with
an n-gram pool kept on the device (each iteration's predictions give n-grams;
the next block takes the pooled continuation of its head).  Compared with the
oracle's decode of the same seeded weights, prompts and guesses -- tokens,
iteration counts and the recorded blocks -- and with the GPU's greedy AR
decode, which the pool cannot change (a token is committed only when the step
verifies it)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from paper_2403_00835_gb300.cllm import CLLM_BLOCK_LOOKAHEAD, CLLM_BLOCK_REFILL, CllmError
from tests.parity_util import FLAG_GAP, engine_for, first_flag, oracle_for

pytestmark = pytest.mark.gpu

MAX_SEQ = 192


@pytest.fixture(scope="module", params=["f32", "bf16"])
def pair(request):
    cfg = syn.TINY if request.param == "f32" else syn.TINY_BF16
    w_cpu = syn.make_weights(cfg, seed=0, device="cpu")
    w_gpu = syn.weights_to(w_cpu, "cuda")
    eng = engine_for(cfg, w_gpu, max_batch=4, max_seq=MAX_SEQ, max_block=16)
    yield cfg, eng, oracle_for(cfg, w_cpu)
    eng.close()


@pytest.mark.parametrize("n,ngram", [(4, 2), (8, 3), (8, 5), (16, 4)])
def test_lookahead_decode_and_trajectory_match_oracle(pair, n, ngram):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=1)
    max_new = 48
    out, iters, traj = eng.jacobi_decode(prompts, n, max_new, seed=3, block_mode=CLLM_BLOCK_LOOKAHEAD,
                                         ngram=ngram, record_cap=max_new + 1)
    thr = 1e-4 if cfg.dtype == "f32" else FLAG_GAP
    compared = 0
    for b, p in enumerate(prompts):
        ar = orc.ar_decode(om, p, max_new)
        k = first_flag(ar.min_gap, thr)
        assert out[b][:k].tolist() == ar.tokens[:k], f"b={b} first flag {k}"
        jr = orc.jacobi_decode(om, p, n, max_new, seed=3, b=b, mode="lookahead", ngram=ngram, record=True)
        if min(jr.min_gap_all) >= thr and k == max_new:
            compared += 1
            assert iters[b] == jr.iterations
            assert out[b].tolist() == jr.tokens
            np.testing.assert_array_equal(traj[: jr.iterations, b, :].astype(np.int64),
                                          np.array(jr.trajectory, dtype=np.int64))
            assert (traj[jr.iterations:, b, :] == -1).all()
    print(f"sequences compared iteration by iteration: {compared}/{len(prompts)}")
    if cfg.dtype == "f32":
        assert compared >= 1  # (sequences with a near-tie anywhere in a block are skipped)


def test_lookahead_equals_gpu_ar_and_saves_iterations(pair):
    """The decode is the GPU's greedy AR output; on these random-init models,
    whose greedy continuations repeat, the pool also cuts iterations."""
    cfg, eng, _ = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=8)
    ar = eng.ar_decode(prompts, 64)
    base, it_base = eng.jacobi_decode(prompts, 8, 64, seed=3, block_mode=CLLM_BLOCK_REFILL)
    la, it_la = eng.jacobi_decode(prompts, 8, 64, seed=3, block_mode=CLLM_BLOCK_LOOKAHEAD, ngram=4)
    np.testing.assert_array_equal(base, ar)
    np.testing.assert_array_equal(la, ar)
    print("iterations refill", it_base.tolist(), "lookahead", it_la.tolist())
    assert it_la.sum() <= it_base.sum()


def test_lookahead_rejects_bad_ngram(pair):
    cfg, eng, _ = pair
    prompts = syn.make_prompts(cfg.vocab, [16], seed=9)
    for bad in (0, 1, 17):
        with pytest.raises(CllmError):
            eng.jacobi_decode(prompts, 4, 8, seed=1, block_mode=CLLM_BLOCK_LOOKAHEAD, ngram=bad)


def test_lookahead_7b_persistent_equals_ar():
    """The 7B shape at n = 16 runs the persistent kernel, whose accept phase
    keeps the pool: the decode equals the greedy AR decode."""
    cfg = syn.LLAMA7B
    w = syn.make_weights(cfg, seed=0, device="cuda")
    eng = engine_for(cfg, w, max_batch=2, max_seq=128 + 64 + 32, max_block=16)
    prompts = syn.make_prompts(cfg.vocab, [128, 100], seed=1)
    try:
        eng.prefill(prompts)
        assert eng.uses_persistent(16)
        la, its = eng.jacobi_decode(prompts, 16, 48, seed=2, block_mode=CLLM_BLOCK_LOOKAHEAD, ngram=4)
        ar = eng.ar_decode(prompts, 48)
        np.testing.assert_array_equal(la, ar)
        print("7B lookahead iterations", its.tolist())
    finally:
        eng.close()
