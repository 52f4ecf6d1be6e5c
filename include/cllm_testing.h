/*
 * cllm_testing.h -- test hooks of the cllm library (not part of the decoding
 * API).  They run one kernel of the block forward in isolation so that a
 * parity failure can be attributed to it.
 */
#ifndef CLLM_TESTING_H
#define CLLM_TESTING_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/*
 * The bf16 weight-streaming GEMM of the block forward (tcgen05/TMA kernel with
 * its work split and fixed-order split-K reduction) with the residual
 * epilogue:  Y[t][m] += sum_k W[m][k] * (Xhi[t][k] + Xlo[t][k])  for t < T, m < M.
 * W: device bf16 [M][K]; X: device bf16 [2][x_rows][K], the hi plane then the
 * lo plane of the activations (the engine carries every GEMM input as
 * hi = bf16(v), lo = bf16(v - hi)), x_rows >= T rounded up to 16 (and >= 256
 * when T > 256); Y: device fp32 [T][M], accumulated into.
 * Constraints: M a multiple of 128, K a multiple of 8, 1 <= T.  Allocates and
 * frees its own scratch; synchronises the device.  Returns a CLLM_* status.
 * Cited operation: the projections of the block forward, one pass over all
 * n block rows (Eq. 3: one forward pass computes every row).
 */
int cllm_test_gemm_bf16(const void *W, const void *X, float *Y, int M, int K, int T, int x_rows);

#ifdef __cplusplus
}
#endif

#endif /* CLLM_TESTING_H */
