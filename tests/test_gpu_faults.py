"""Failure paths of the CUDA path, made on purpose without faulting the GPU:

  * bounded on-device waits: a host-armed hook makes one grid barrier of the
    persistent kernel wait for an arrival that never comes; every CTA's wait
    runs out after the wait budget, the kernel unwinds (copies and
    tensor-core work in flight are waited for, tensor memory is freed), the
    call returns CLLM_ETIMEOUT, and the context decodes correctly afterwards;
  * allocation failure: a countdown makes the k-th device or pinned
    allocation fail; the call returns CLLM_ENOMEM, releases what it had taken
    and leaves the process able to create and run a context.
"""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2403_00835_gb300 import synthetic as syn
from paper_2403_00835_gb300.cllm import CllmError, load
from tests.parity_util import engine_for

pytestmark = pytest.mark.gpu

CLLM_ENOMEM = -2
CLLM_ETIMEOUT = -5


def _hooks():
    lib = load()
    lib.cllm_test_hold_barrier.argtypes = [ctypes.c_void_p, ctypes.c_int]
    lib.cllm_test_hold_barrier.restype = ctypes.c_int
    lib.cllm_test_fail_alloc.argtypes = [ctypes.c_int]
    lib.cllm_test_fail_alloc.restype = None
    return lib


@pytest.fixture(scope="module")
def tiny():
    cfg = syn.TINY_BF16
    w = syn.weights_to(syn.make_weights(cfg, seed=0, device="cpu"), "cuda")
    return cfg, w


def test_hold_barrier_times_out_and_context_survives(tiny):
    cfg, w = tiny
    lib = _hooks()
    n = 16
    eng = engine_for(cfg, w, max_batch=2, max_seq=128, max_block=n)
    try:
        prompts = syn.make_prompts(cfg.vocab, [29, 40], seed=81)
        guesses = syn.make_guesses(cfg.vocab, 2, n, seed=82)
        eng.prefill(prompts)
        assert eng.uses_persistent(n)
        ref = eng.jacobi_step(guesses)
        n_phases = 1 + 5 * cfg.n_layers + 2  # embed, 5 per layer, LM head, accept
        # first GEMM, a later attention phase, the commit
        for phase in (1, 7, n_phases - 1):
            eng.prefill(prompts)
            assert lib.cllm_test_hold_barrier(eng._h, phase) == 0
            with pytest.raises(CllmError) as e:
                eng.jacobi_step(guesses)
            assert e.value.status == CLLM_ETIMEOUT, phase
            # the commit did not run: the committed lengths are the prompts'
            assert eng.committed_lengths().tolist() == [len(p) for p in prompts]
            assert lib.cllm_test_hold_barrier(eng._h, -1) == 0
            r = eng.jacobi_step(guesses)
            np.testing.assert_array_equal(r["next"], ref["next"])
            np.testing.assert_array_equal(r["accepted"], ref["accepted"])
        # a held decode iteration ends the decode with the same status
        ar = eng.ar_decode(prompts, 24)
        assert lib.cllm_test_hold_barrier(eng._h, 3) == 0
        with pytest.raises(CllmError) as e:
            eng.jacobi_decode(prompts, n, 24, seed=1)
        assert e.value.status == CLLM_ETIMEOUT
        assert lib.cllm_test_hold_barrier(eng._h, -1) == 0
        out, _ = eng.jacobi_decode(prompts, n, 24, seed=1)
        np.testing.assert_array_equal(out, ar)
    finally:
        lib.cllm_test_hold_barrier(eng._h, -1)
        eng.close()


def test_hold_barrier_rejects_bad_phase(tiny):
    cfg, w = tiny
    lib = _hooks()
    eng = engine_for(cfg, w, max_batch=1, max_seq=64, max_block=8)
    try:
        assert lib.cllm_test_hold_barrier(eng._h, 0) == -1
        assert lib.cllm_test_hold_barrier(eng._h, -2) == -1
        assert lib.cllm_test_hold_barrier(None, 1) == -1
    finally:
        eng.close()


def _free_bytes():
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def test_allocation_failure_injection(tiny):
    cfg, w = tiny
    lib = _hooks()
    prompts = syn.make_prompts(cfg.vocab, [19, 33], seed=91)
    guesses = syn.make_guesses(cfg.vocab, 2, 8, seed=92)
    # a clean context first: reference results and a warmed-up device
    eng = engine_for(cfg, w, max_batch=2, max_seq=96, max_block=8)
    eng.prefill(prompts)
    ref = eng.jacobi_step(guesses)
    ref_dec = eng.jacobi_decode(prompts, 8, 20, seed=2, record_cap=21)
    eng.close()
    free0 = _free_bytes()
    try:
        # every allocation of cllm_create in turn
        k = 0
        while True:
            lib.cllm_test_fail_alloc(k)
            try:
                eng = engine_for(cfg, w, max_batch=2, max_seq=96, max_block=8)
            except CllmError as e:
                assert e.status == CLLM_ENOMEM, k
                assert abs(_free_bytes() - free0) <= 8 << 20, k
                k += 1
                assert k < 500
                continue
            break
        lib.cllm_test_fail_alloc(-1)
        assert k >= 10  # the context's buffers were each made to fail once
        try:
            eng.prefill(prompts)
            # the step's first launch captures a graph and allocates its tables
            lib.cllm_test_fail_alloc(0)
            with pytest.raises(CllmError) as e:
                eng.jacobi_step(guesses)
            assert e.value.status == CLLM_ENOMEM
            lib.cllm_test_fail_alloc(-1)
            r = eng.jacobi_step(guesses)
            np.testing.assert_array_equal(r["next"], ref["next"])
            np.testing.assert_array_equal(r["accepted"], ref["accepted"])
            # a trajectory recording allocates its buffer at decode start
            lib.cllm_test_fail_alloc(0)
            with pytest.raises(CllmError) as e:
                eng.jacobi_decode(prompts, 8, 20, seed=2, record_cap=21)
            assert e.value.status == CLLM_ENOMEM
            lib.cllm_test_fail_alloc(-1)
            dec = eng.jacobi_decode(prompts, 8, 20, seed=2, record_cap=21)
            for a, b in zip(dec, ref_dec):
                np.testing.assert_array_equal(a, b)
        finally:
            eng.close()
        assert abs(_free_bytes() - free0) <= 8 << 20
    finally:
        lib.cllm_test_fail_alloc(-1)
