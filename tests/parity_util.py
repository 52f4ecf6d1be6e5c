"""Shared helpers of the GPU parity tests: build the CUDA engine and the oracle
from the same seeded weights, and the comparison rules.

Comparison rules (stated once here, used by every parity test):
  * logits: per row, max |gpu - oracle| <= 2e-2 * std_vocab(oracle row) in bf16,
    <= 1e-4 absolute in fp32;
  * tokens and accepted counts: bit-exact, except at rows whose oracle top-1 /
    top-2 gap is below 0.05 ("flagged"); flagged rows are counted, not compared;
  * free-running decodes are compared token by token up to the first flagged
    position of the oracle's trajectory.
"""
import numpy as np

from oracle import oracle as orc
from paper_2403_00835_gb300 import synthetic as syn

FLAG_GAP = 0.05
LOGIT_TOL_BF16 = 2e-2
LOGIT_TOL_F32 = 1e-4


def oracle_for(cfg, weights_cpu):
    wd = orc.ORC_F32 if cfg.dtype == "f32" else orc.ORC_BF16
    return orc.OracleModel(orc.OracleArch(**syn.oracle_arch_kwargs(cfg)), weights_cpu, wd)


def engine_for(cfg, weights_gpu, max_batch, max_seq, max_block):
    from paper_2403_00835_gb300.cllm import Engine
    return Engine(cfg, weights_gpu, max_batch=max_batch, max_seq=max_seq, max_block=max_block)


def logits_ok(gpu, ref, dtype):
    """Returns (ok, worst ratio err/bound) per the logit rule."""
    gpu = np.asarray(gpu, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    err = np.abs(gpu - ref).max(axis=-1)
    if dtype == "bf16":
        bound = LOGIT_TOL_BF16 * ref.std(axis=-1)
    else:
        bound = np.full(err.shape, LOGIT_TOL_F32)
    ratio = err / bound
    return bool((ratio <= 1.0).all()), float(ratio.max())


def first_flag(gaps, thr=FLAG_GAP):
    for i, g in enumerate(gaps):
        if g < thr:
            return i
    return len(gaps)
