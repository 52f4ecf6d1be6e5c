"""The allocation-free GEMM entry point, cllm_gemm_bf16_noalloc.

It exists for callers that cannot call cudaMalloc (a caching allocator owns
the device memory, or the path cannot take cudaMalloc's implicit
synchronisation); all of its scratch lives in one static device array.  Its
output must match the allocating entry point cllm_test_gemm_bf16 (same kernel,
same work split) within the GEMM tests' tolerance, on two calls in a row, so
that a second call sees the array exactly as the first call left it."""
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


def _inputs(M, K, T, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    W = (torch.randn(M, K, device="cuda", generator=g) * 0.02).bfloat16()
    rows = max((T + 15) // 16 * 16, 256 if T > 256 else 0)
    x = torch.randn(rows, K, device="cuda", generator=g)
    hi = x.bfloat16()
    X2 = torch.stack([hi, (x - hi.float()).bfloat16()]).contiguous()
    return W, X2, rows


@pytest.mark.parametrize("M,K,T", [(4096, 4096, 16), (768, 688, 17)])
def test_noalloc_matches_allocating_gemm_twice(M, K, T):
    """Y is accumulated into: both entry points start from the same nonzero Y0
    and must give Y0 + W.X.  The second call must not change the device's
    free memory or the caching allocator's reservation."""
    lib = _lib()
    stream = torch.cuda.current_stream()
    for call in range(2):
        W, X2, rows = _inputs(M, K, T, seed=100 * call + M + K + T)
        g = torch.Generator(device="cuda").manual_seed(7 + call)
        Y0 = torch.randn(T, M, device="cuda", generator=g)
        ref = Y0.clone()
        assert lib.cllm_test_gemm_bf16(W.data_ptr(), X2.data_ptr(), ref.data_ptr(), M, K, T, rows) == 0
        out = Y0.clone()
        torch.cuda.synchronize()
        free0, reserved0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_reserved()
        rc = lib.cllm_gemm_bf16_noalloc(W.data_ptr(), X2.data_ptr(), out.data_ptr(), M, K, T, rows,
                                        ctypes.c_void_p(stream.cuda_stream))
        assert rc == 0, cllm.STATUS.get(rc, rc)
        torch.cuda.synchronize()
        if call == 1:  # the first call may load the library's device code
            assert torch.cuda.mem_get_info()[0] == free0
            assert torch.cuda.memory_reserved() == reserved0
        Wd = W.cpu().double().numpy()
        Xd = (X2[0, :T].double() + X2[1, :T].double()).cpu().numpy()
        exact = Y0.cpu().double().numpy() + Xd @ Wd.T
        bound = 1e-5 * (np.abs(Xd) @ np.abs(Wd).T + np.abs(Y0.cpu().double().numpy())) + 1e-7
        diff = np.abs(out.cpu().double().numpy() - ref.cpu().double().numpy())
        assert (diff <= bound).all(), float((diff / bound).max())
        assert (np.abs(out.cpu().double().numpy() - exact) <= 4e-3 * np.abs(exact).max()).all()


def test_noalloc_rejects_sizes_beyond_its_scratch():
    lib = _lib()
    M, K, T = 16384, 4096, 256  # the epilogue side outputs alone exceed the 8 MiB array
    W = torch.zeros(M, K, device="cuda", dtype=torch.bfloat16)
    X2 = torch.zeros(2, T, K, device="cuda", dtype=torch.bfloat16)
    out = torch.zeros(T, M, device="cuda", dtype=torch.float32)
    rc = lib.cllm_gemm_bf16_noalloc(W.data_ptr(), X2.data_ptr(), out.data_ptr(), M, K, T, T,
                                    ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == -4  # CLLM_ECAPACITY, before any launch


def test_noalloc_refuses_stream_capture():
    """The call synchronises its stream, so it cannot be captured: on a
    capturing stream it returns CLLM_EUNSUPPORTED and queues nothing."""
    lib = _lib()
    W, X2, rows = _inputs(256, 256, 16, seed=3)
    Y = torch.zeros(16, 256, device="cuda")
    side = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.stream(side):
        graph.capture_begin()
        try:
            rc = lib.cllm_gemm_bf16_noalloc(W.data_ptr(), X2.data_ptr(), Y.data_ptr(), 256, 256, 16, rows,
                                            ctypes.c_void_p(side.cuda_stream))
            Y.add_(1.0)  # the capture stays valid after the refusal
        finally:
            graph.capture_end()
    assert cllm.STATUS.get(rc) == "CLLM_EUNSUPPORTED", rc
    graph.replay()
    torch.cuda.synchronize()
    assert float(Y.max()) == 1.0 and float(Y.min()) == 1.0
