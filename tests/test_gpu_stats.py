"""The acceptance statistics the accept step keeps on the device (Sec. 3.3,
Table 3): the histogram of fast-forwarded (accepted) tokens per iteration and
the stationary tokens per n-token window, read back with one call
(cllm_decode_read_stats), against the host-side profiler
(trajectory.analyse) run on the oracle's own recorded Jacobi trajectories --
and on the GPU's recorded trajectory, which must give the same numbers.

Prompts of 4 tokens with guesses drawn from the prompt (Alg. 3's "random
tokens from x") make the random-weight decoder accept several tokens per
iteration and hold stationary tokens now and then, so the counters are not
trivially one and zero."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from paper_2403_00835_gb300 import trajectory as tj
from paper_2403_00835_gb300.cllm import (CLLM_BLOCK_REFILL, CLLM_BLOCK_SHRINK, CLLM_GUESS_FROM_PROMPT,
                                         CllmError)
from tests.parity_util import engine_for, oracle_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pair():
    cfg = syn.TINY
    w_cpu = syn.make_weights(cfg, seed=0, device="cpu")
    w_gpu = syn.weights_to(w_cpu, "cuda")
    eng = engine_for(cfg, w_gpu, max_batch=4, max_seq=160, max_block=16)
    yield cfg, eng, oracle_for(cfg, w_cpu)
    eng.close()


def _expected(stats: tj.TrajectoryStats, n):
    acc = np.bincount(np.asarray(stats.accepted, dtype=np.int64), minlength=n + 1)
    win = np.bincount(np.asarray(stats.window_stationary, dtype=np.int64), minlength=n + 1)
    return acc, win


def _check(dev, stats, n):
    acc, win = _expected(stats, n)
    np.testing.assert_array_equal(dev["acc_hist"], acc)
    np.testing.assert_array_equal(dev["win_hist"], win)
    assert dev["iterations"] == len(stats.accepted)
    assert dev["accepted"] == sum(stats.accepted)
    assert dev["windows"] == len(stats.window_stationary)
    assert dev["stationary"] == sum(stats.window_stationary)


@pytest.mark.parametrize("mode", ["shrink", "refill"])
@pytest.mark.parametrize("n", [8, 16])
def test_device_counters_match_oracle_trajectories(pair, mode, n):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [4, 4, 4, 4], seed=1)
    max_new = 64
    bm = CLLM_BLOCK_SHRINK if mode == "shrink" else CLLM_BLOCK_REFILL
    out, iters, traj = eng.jacobi_decode(prompts, n, max_new, seed=2, block_mode=bm,
                                         guess_init=CLLM_GUESS_FROM_PROMPT,
                                         record_cap=max_new + 1, stats=True)
    dev = eng.decode_read_stats()
    # the GPU's own trajectory through the host profiler: the same counts
    _check(dev, tj.analyse_batch(traj, out, iters, n), n)
    # the oracle's decode of the same prompts and guesses, recorded and profiled
    ref = tj.TrajectoryStats()
    for b, p in enumerate(prompts):
        jr = orc.jacobi_decode(om, p, n, max_new, seed=2, b=b, mode=mode, guess_init="prompt",
                               record=True)
        assert out[b].tolist() == jr.tokens and iters[b] == jr.iterations, b
        blocks = np.array([list(x) + [-1] * (n - len(x)) for x in jr.trajectory])
        s = tj.analyse(blocks, jr.tokens, jr.iterations, n)
        ref.accepted += s.accepted
        ref.window_stationary += s.window_stationary
    _check(dev, ref, n)
    assert dev["accepted"] == len(prompts) * max_new
    print(f"{mode} n={n}: accepted histogram {dev['acc_hist'][1:].tolist()}, "
          f"windows {dev['windows']}, stationary {dev['stationary']}")
    if mode == "shrink" and n == 8:
        assert dev["acc_hist"][2:].sum() > 0 and dev["stationary"] > 0


def test_counters_reset_per_decode_and_need_opt_in(pair):
    cfg, eng, _ = pair
    prompts = syn.make_prompts(cfg.vocab, [4, 4], seed=3)
    eng.jacobi_decode(prompts, 8, 32, seed=2, guess_init=CLLM_GUESS_FROM_PROMPT, stats=True)
    first = eng.decode_read_stats()
    eng.jacobi_decode(prompts, 8, 32, seed=2, guess_init=CLLM_GUESS_FROM_PROMPT, stats=True)
    second = eng.decode_read_stats()
    for k in ("iterations", "accepted", "windows", "stationary"):
        assert first[k] == second[k], k
    np.testing.assert_array_equal(first["acc_hist"], second["acc_hist"])
    eng.jacobi_decode(prompts, 8, 32, seed=2)
    with pytest.raises(CllmError):
        eng.decode_read_stats()
