"""The bf16 weight-streaming GEMM (tcgen05 + TMA, split-K with fixed-order
reduction) in isolation, through the test hook of include/cllm_testing.h:
Y[t][m] = sum_k W[m][k] X[t][k] against an fp64 matmul of the same bf16
values, over ragged M/K/T tiles, split and whole-tile work partitions; and a
token's column must be bit-identical whatever the number of tokens in the
launch (the property that makes a Jacobi step and an AR step agree)."""
import ctypes

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2403_00835_gb300 import cllm

pytestmark = pytest.mark.gpu


def _lib():
    lib = cllm.load()
    lib.cllm_test_gemm_bf16.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_int] * 4
    lib.cllm_test_gemm_bf16.restype = ctypes.c_int
    return lib


def split_hilo(x):
    """fp32 activations -> stacked bf16 planes [2][rows][K]: hi = bf16(x), lo = bf16(x - hi)."""
    hi = x.bfloat16()
    lo = (x - hi.float()).bfloat16()
    return torch.stack([hi, lo]).contiguous()


def run_gemm(W, X2, T):
    M, K = W.shape
    Y = torch.zeros(T, M, device="cuda", dtype=torch.float32)
    rc = _lib().cllm_test_gemm_bf16(W.data_ptr(), X2.data_ptr(), Y.data_ptr(), M, K, T, X2.shape[1])
    assert rc == 0, cllm.STATUS.get(rc, rc)
    return Y


def x_rows(T):
    return max((T + 15) // 16 * 16, 256 if T > 256 else 0)


@pytest.mark.parametrize("M,K,T", [
    (128, 64, 1), (128, 64, 16), (768, 256, 8), (256, 688, 17), (512, 256, 100),
    (256, 512, 256), (384, 256, 300), (4096, 4096, 16), (4096, 11008, 64), (12288, 4096, 32),
    (256, 4096, 520)])
def test_gemm_matches_fp64(M, K, T):
    g = torch.Generator(device="cuda").manual_seed(M * 7 + K * 3 + T)
    W = (torch.randn(M, K, device="cuda", generator=g) * 0.02).bfloat16()
    X2 = split_hilo(torch.randn(x_rows(T), K, device="cuda", generator=g))
    Y = run_gemm(W, X2, T).cpu().double().numpy()
    Wd = W.cpu().double().numpy()
    Xd = (X2[0, :T].double() + X2[1, :T].double()).cpu().numpy()
    ref = Xd @ Wd.T
    bound = 1e-5 * (np.abs(Xd) @ np.abs(Wd).T) + 1e-7
    assert (np.abs(Y - ref) <= bound).all(), float((np.abs(Y - ref) / bound).max())


@pytest.mark.parametrize("M,K", [(4096, 4096), (768, 688)])
def test_gemm_column_independent_of_token_count(M, K):
    g = torch.Generator(device="cuda").manual_seed(5)
    W = (torch.randn(M, K, device="cuda", generator=g) * 0.02).bfloat16()
    X2 = split_hilo(torch.randn(256, K, device="cuda", generator=g))
    ys = {T: run_gemm(W, X2, T) for T in (1, 16, 48, 64, 256)}
    for T in (16, 48, 64, 256):
        assert torch.equal(ys[T][:1], ys[1])
    assert torch.equal(ys[64][:48], ys[48])
    assert torch.equal(ys[256][:64], ys[64])
