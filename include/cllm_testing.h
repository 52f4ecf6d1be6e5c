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

/*
 * Timing of the same kernel in a chain: `iters` launches captured in one CUDA
 * graph, launch i reading weights W + (i % n_w) * w_stride_bytes (distinct
 * matrices keep the chain from being served by L2), all accumulating into Y.
 * pdl: launch with programmatic dependent launch; l2_ahead: weight tiles per
 * CTA prefetched into L2 before waiting on the previous launch (the engine
 * uses 16).  T <= 256.  The graph runs once to warm up, then once timed with
 * CUDA events; *us_per_launch = elapsed / iters.  Returns a CLLM_* status.
 */
int cllm_test_gemm_bf16_timed(const void *W, long long w_stride_bytes, int n_w, const void *X,
                              float *Y, int M, int K, int T, int x_rows, int iters, int pdl,
                              int l2_ahead, float *us_per_launch);

/*
 * Raw phase timestamps (globaltimer ns) of the last profiled iteration of the
 * persistent kernel (cllm_set_profiling(ctx, 1)): out[0..P] CTA 0's phase
 * starts and end; then, per phase p, out[P+1+p] first and out[2P+1+p] last
 * start over the CTAs, out[3P+1+p] first and out[4P+1+p] last arrival at the
 * grid barrier.  names[p] = phase class.  Returns the number of values (5P+1),
 * 0 if nothing was profiled.
 */
int cllm_test_phase_stamps(cllm_ctx *ctx, unsigned long long *out, int cap, const char **names,
                           int names_cap);

/* Per-CTA timestamps of the last profiled persistent iteration (global
 * timer, ns): out[(k * P + p) * G + cta] for k = 0..12 -- 0 phase start
 * (barrier seen), 1 MMA issuer done with the phase (GEMM phases), 2 arrival
 * at the grid barrier, 3-5 the epilogue's last segment (accumulator ready,
 * after the split-K ticket, done), 6 producer enters the phase, 8 producer
 * done, 7 the split-K owner's partials summed (its last segment), 10/11
 * first/last stage arrival at the MMA, 12 largest gap between arrivals (ns);
 * slot 9 is unused (0).  Then 256 * G traced arrivals
 * (see cllm_test_set_trace_phase).  G = SM count.  Returns the number of
 * values, (13 * P + 256) * G. */
int cllm_test_cta_stamps(cllm_ctx *ctx, unsigned long long *out, long long cap);

/* Profiling: trace every MMA stage arrival (global timer, ns) of phase
 * `phase` of the persistent kernel, up to 256 per CTA; they follow the
 * per-CTA stamps in cllm_test_cta_stamps' output ([cta][256], 0 = unused).
 * -1 turns tracing off.  Drops the captured graphs.  EINVAL on a null ctx. */
int cllm_test_set_trace_phase(cllm_ctx *ctx, int phase);

/*
 * Failure injection for the bounded on-device waits.  From the next captured
 * iteration on, the grid barrier of the persistent kernel before phase
 * `phase` (1 <= phase < the iteration's phase count; phase 0 has no barrier)
 * waits for one arrival more than the grid makes.  Every CTA's wait there
 * runs out after the kernel's wait budget (2 s), the CTA waits for its own
 * copies and tensor-core operations in flight, frees its tensor memory and
 * returns, and the call that ran the iteration returns CLLM_ETIMEOUT.  No
 * phase from `phase` on runs, so the commit of the iteration does not happen
 * and the context stays usable.  -1 disarms.  Drops the captured graphs.
 * Only iterations that run the persistent kernel (cllm_uses_persistent) are
 * affected.  EINVAL on a null ctx, phase 0 or phase < -1.
 */
int cllm_test_hold_barrier(cllm_ctx *ctx, int phase);

/*
 * Allocation-failure injection: the k-th device (or pinned host) allocation
 * the library makes from now on (k = 0: the next one) fails as if memory
 * were exhausted; the call that made it returns CLLM_ENOMEM after releasing
 * what it had allocated.  One-shot; k < 0 disarms.  Process-wide.
 */
void cllm_test_fail_alloc(int k);

/*
 * Host-only (no CUDA call): the work split of one weight-GEMM launch of
 * `mtiles` 128-row weight tiles over K (inner dimension) for T token columns
 * on `sms` SMs, as the library plans it.  out[8] = {mtiles, ntiles (token
 * tiles), kchunks (64-column chunks of K), cpc (chunks per CTA), bn (token
 * columns of a tile), bn_max (kernel variant), maxc (most CTAs sharing one
 * tile), grid (CTAs)}.  T <= 256: one token tile and the (tile, chunk) space
 * cut into equal contiguous ranges that depend on the weight shape and the SM
 * count only; T > 256: whole 128 x 256 tiles per CTA.  EINVAL on a null out
 * or a non-positive argument.
 */
int cllm_test_plan_gemm(int mtiles, int K, int T, int sms, int *out);

#ifdef __cplusplus
}
#endif

#endif /* CLLM_TESTING_H */
