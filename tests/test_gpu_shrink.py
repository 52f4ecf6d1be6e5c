"""Alg. 3's two block policies on the CUDA path, with the trajectory capture:
the shrinking window (the block narrows by the accepted tokens until it is
fixed, then a fresh n-wide block) and the fixed-width refill, each compared
with the oracle's decode of the same seeded weights, prompts and guesses --
tokens, iteration counts and the recorded blocks y^(0), y^(1), ... (Sec. 3.1)."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn
from paper_2403_00835_gb300.cllm import CLLM_BLOCK_REFILL, CLLM_BLOCK_SHRINK, CllmError
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


def _padded(blocks, n):
    return np.array([list(b) + [-1] * (n - len(b)) for b in blocks], dtype=np.int64)


@pytest.mark.parametrize("mode", ["shrink", "refill"])
@pytest.mark.parametrize("n", [4, 8, 16])
def test_decode_and_trajectory_match_oracle(pair, mode, n):
    cfg, eng, om = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=1)
    max_new = 48
    bm = CLLM_BLOCK_SHRINK if mode == "shrink" else CLLM_BLOCK_REFILL
    out, iters, traj = eng.jacobi_decode(prompts, n, max_new, seed=3, block_mode=bm,
                                         record_cap=max_new + 1)
    thr = 1e-4 if cfg.dtype == "f32" else FLAG_GAP
    compared = 0
    for b, p in enumerate(prompts):
        ar = orc.ar_decode(om, p, max_new)
        k = first_flag(ar.min_gap, thr)
        # the fixed point is the greedy output whatever the policy (Sec. 3.1)
        assert out[b][:k].tolist() == ar.tokens[:k], f"b={b} first flag {k}"
        jr = orc.jacobi_decode(om, p, n, max_new, seed=3, b=b, mode=mode, record=True)
        if min(jr.min_gap_all) >= thr and k == max_new:
            compared += 1
            assert iters[b] == jr.iterations
            assert out[b].tolist() == jr.tokens
            got = traj[: jr.iterations, b, :].astype(np.int64)
            np.testing.assert_array_equal(got, _padded(jr.trajectory, n))
            assert (traj[jr.iterations:, b, :] == -1).all()
    print(f"sequences compared iteration by iteration: {compared}/{len(prompts)}")


def test_shrink_window_widths(pair):
    """In shrink mode every recorded block is a suffix-shrunk window: its width
    is n after a fully fixed window and (previous width - accepted) otherwise."""
    cfg, eng, _ = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17], seed=4)
    n, max_new = 8, 40
    out, iters, traj = eng.jacobi_decode(prompts, n, max_new, seed=5, block_mode=CLLM_BLOCK_SHRINK,
                                         record_cap=max_new + 1)
    for b in range(len(prompts)):
        widths = [(traj[it, b] >= 0).sum() for it in range(iters[b])]
        assert widths[0] == n
        for it in range(1, iters[b]):
            w_prev, w = widths[it - 1], widths[it]
            assert 1 <= w <= n
            assert w == n or w < w_prev


def test_shrink_equals_gpu_ar(pair):
    cfg, eng, _ = pair
    prompts = syn.make_prompts(cfg.vocab, [32, 17, 45], seed=8)
    ar = eng.ar_decode(prompts, 40)
    for n in (4, 16):
        jac, _ = eng.jacobi_decode(prompts, n, 40, seed=3, block_mode=CLLM_BLOCK_SHRINK)
        np.testing.assert_array_equal(jac, ar)


def test_trajectory_needs_recording(pair):
    cfg, eng, _ = pair
    prompts = syn.make_prompts(cfg.vocab, [16], seed=9)
    eng.jacobi_decode(prompts, 4, 8, seed=1)
    with pytest.raises(CllmError):
        traj = np.zeros((4, 1, 4), dtype=np.int32)
        from paper_2403_00835_gb300.cllm import _check, _ip
        _check(eng._lib.cllm_decode_read_trajectory(eng._h, _ip(traj)), "trajectory")
