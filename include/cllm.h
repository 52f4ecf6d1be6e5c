/*
 * cllm.h -- C ABI of a single-GPU (sm_103a) Jacobi-decoding engine for
 * LLaMA-style decoders, the computation that Consistency LLMs (CLLMs,
 * arXiv 2403.00835) accelerate.
 *
 * Problem statement (Sec. 3.1).  Given a prompt x, greedy AR decoding produces
 * y_i = argmax_y p(y | y_<i, x) one token per forward pass (Eq. 1).  Jacobi
 * decoding instead iterates an n-token guess y^(j): one causal forward pass
 * over [x ; y^(j)] yields y^(j+1)_i = argmax p(. | y^(j)_<i, x) for all n
 * positions at once (Eq. 3).  With a KV cache (Sec. 3.1 "Jacobi Decoding with
 * KV Cache", App. C Alg. 3) the keys/values of the prefix are kept, every
 * iteration fixes the longest correct prefix of the block (at least one token),
 * commits its K/V, and the fixed point reached this way is the greedy AR output.
 *
 * Conventions for every call:
 *   - Return value: CLLM_OK (0) or a negative CLLM_E* code.  No exception or
 *     abort crosses the ABI.  On error the outputs are left untouched.
 *   - Token arrays passed to these calls are HOST memory owned by the caller,
 *     int32, row-major.  Weights are DEVICE memory owned by the caller.
 *   - A context is bound to one CUDA stream and one device and is not
 *     thread-safe; calls on one context must not overlap.
 *   - Every call on a context synchronises its stream before returning
 *     (unless stated otherwise), so host outputs are valid on return.
 */
#ifndef CLLM_H
#define CLLM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---------------------------------------------------------- */
#define CLLM_OK 0
#define CLLM_EINVAL -1      /* bad argument, shape or pointer                       */
#define CLLM_ENOMEM -2      /* device or host allocation failed                     */
#define CLLM_ECUDA -3       /* a CUDA runtime/driver call failed                    */
#define CLLM_ECAPACITY -4   /* committed length + block would exceed max_seq        */
#define CLLM_ETIMEOUT -5    /* a bounded on-device wait ran out (kernel returned)  */
#define CLLM_EDEVICE -6     /* a device-side check failed (bounds, token id, ...)   */
#define CLLM_ESTATE -7      /* call out of order (e.g. a step before prefill)       */
#define CLLM_EUNSUPPORTED -8 /* shape or device this build does not handle          */

/* ---- element types ----------------------------------------------------------- */
#define CLLM_F32 0   /* fp32 weights and activations (parity configurations)         */
#define CLLM_BF16 1  /* bf16 weights; every GEMM input carried as two bf16 planes     */
                     /* (hi + lo), fp32 accumulation and residual stream; Q, K, V and */
                     /* the attention probabilities in fp16 with fp32 accumulation    */

/* ---- decode options ---------------------------------------------------------- */
#define CLLM_GUESS_UNIFORM 0      /* initial/refill guesses uniform over the vocab   */
#define CLLM_GUESS_FROM_PROMPT 1  /* guesses drawn from the prompt's tokens (Alg. 3) */
#define CLLM_BLOCK_REFILL 0       /* block stays n wide: fresh guesses after commits */
#define CLLM_BLOCK_SHRINK 1       /* Alg. 3: the window narrows by the accepted tokens
                                     until it is fixed, then a fresh n-wide block */
#define CLLM_BLOCK_LOOKAHEAD 2    /* refill, with an n-gram pool (Sec. 3.3's combination
                                     with lookahead decoding): each iteration's
                                     predictions P give n-grams (key P[k], value
                                     P[k+1..k+ngram-1]); the next block takes the
                                     pooled continuation of its head in slots
                                     1..ngram-1 (from earlier iterations' n-grams),
                                     and the step verifies it */

/*
 * Model shape and capacity.  The decoder is the pre-norm LLaMA layer:
 * RMSNorm -> Q/K/V projections -> rotate-half RoPE -> causal softmax attention
 * -> output projection + residual -> RMSNorm -> SwiGLU MLP + residual, then a
 * final RMSNorm and an untied LM head (no biases, unscaled embedding).
 * Constraints of this build: head_dim in {64, 128}; n_heads*head_dim,
 * n_kv_heads*head_dim and d_model multiples of 128; n_heads a multiple of
 * n_kv_heads; ffn and d_model multiples of 8.
 */
typedef struct {
  int n_layers, d_model, n_heads, n_kv_heads, head_dim, ffn, vocab;
  float rms_eps, rope_theta;
  int dtype;     /* CLLM_F32 | CLLM_BF16: element type of weights and activations */
  int max_batch; /* sequences decoded together                                   */
  int max_seq;   /* KV-cache positions per sequence (prompt + new tokens + n)     */
  int max_block; /* largest block width n                                        */
} cllm_arch;

/*
 * Borrowed DEVICE pointers to the weights, element type = arch.dtype, every
 * matrix [out_features][in_features] row-major, 16-byte aligned, and alive for
 * the lifetime of the context.  The per-layer members are HOST arrays of
 * n_layers device pointers (copied at cllm_create).
 *   tok_emb [vocab][d]   final_norm [d]   lm_head [vocab][d]
 *   attn_norm[l] [d]     wq[l] [n_heads*hd][d]   wk[l], wv[l] [n_kv_heads*hd][d]
 *   wo[l] [d][n_heads*hd]   mlp_norm[l] [d]   w_gate[l], w_up[l] [ffn][d]
 *   w_down[l] [d][ffn]
 */
typedef struct {
  const void *tok_emb, *final_norm, *lm_head;
  const void *const *attn_norm, *const *wq, *const *wk, *const *wv, *const *wo,
      *const *mlp_norm, *const *w_gate, *const *w_up, *const *w_down;
} cllm_weights;

typedef struct {
  uint64_t seed;   /* key of the counter-based guess generator                    */
  int eos_id;      /* -1: off.  Else a sequence stops after committing this token   */
  int guess_init;  /* CLLM_GUESS_UNIFORM | CLLM_GUESS_FROM_PROMPT                  */
  int block_mode;  /* CLLM_BLOCK_REFILL | CLLM_BLOCK_SHRINK | CLLM_BLOCK_LOOKAHEAD  */
  int record_cap;  /* > 0: record the first record_cap blocks of every sequence
                      (the Jacobi trajectory), read with cllm_decode_read_trajectory */
  int stats;       /* 1: keep the acceptance statistics on the device, read with
                      cllm_decode_read_stats; 0: off                           */
  int ngram;       /* CLLM_BLOCK_LOOKAHEAD: n-gram size, 2..16 (the pool keeps
                      ngram - 1 tokens per key token, one pool per sequence,
                      batch * vocab * (ngram - 1) ints of device memory); other
                      modes: ignored                                             */
} cllm_decode_opts;

/* Acceptance statistics of a decode (Sec. 3.3, Table 3), summed over the
 * batch.  See cllm_decode_read_stats. */
typedef struct {
  int64_t iterations; /* sequence-iterations run                                  */
  int64_t accepted;   /* tokens they committed (fast-forwarded, head included)     */
  int64_t windows;    /* n-token windows opened                                   */
  int64_t stationary; /* stationary tokens inside those windows                   */
} cllm_accept_stats;

typedef struct cllm_ctx cllm_ctx;

/*
 * Create a context: validates the shape, builds the TMA descriptors of the
 * weights, and allocates (owns) the KV cache K,V[layer][b][kv_head][pos][hd]
 * (fp32 for CLLM_F32, fp16 for CLLM_BF16),
 * the activation scratch and the device status word.  cuda_stream is a
 * cudaStream_t (NULL = a stream the context creates and owns).  The current
 * device at the call is the context's device.
 * Errors: EINVAL (shape/pointers/alignment), EUNSUPPORTED (not an sm_103
 * device, or a shape outside the constraints above), ENOMEM, ECUDA.
 */
int cllm_create(const cllm_arch *arch, const cllm_weights *w, void *cuda_stream,
                cllm_ctx **out);

/* Release everything the context owns (not the weights).  NULL is a no-op. */
void cllm_destroy(cllm_ctx *ctx);

/*
 * Prefill (Alg. 3, first line of the loop's set-up: y_0, K <- LLM(x)).
 * tokens: the B prompts concatenated, sum(lens) entries; lens[b] >= 1.
 * Runs the causal forward over every prompt, fills the KV cache at positions
 * 0..lens[b]-1 of sequence b, sets its committed length to lens[b] and its
 * head to y_1 = argmax p(. | x_b) (Eq. 3 first row), returned in head_out[B]
 * (may be NULL).  Resets any decode in progress.
 * Errors: EINVAL (B outside [1, max_batch], a length < 1, a token outside the
 * vocab), ECAPACITY (lens[b] > max_seq), ECUDA, EDEVICE, ETIMEOUT.
 */
int cllm_prefill(cllm_ctx *ctx, int B, const int32_t *tokens, const int32_t *lens,
                 int32_t *head_out);

/*
 * One Jacobi iteration with KV cache (Eq. 3 + Alg. 3) on the B sequences of
 * the last prefill.  guess[B][n]: the block y^(j); guess[b][0] is replaced by
 * the context's head of sequence b (the token already known to be correct).
 * One forward pass over the block rows at positions L_b .. L_b+n-1 writes their
 * K/V into the cache and computes, for every row k, P[b][k] = argmax of its
 * logits (lowest id on ties) and gap[b][k] = top1 - top2 logit.
 * The accepted count is a_b = 1 + #{leading k >= 1 : block[k] == P[k-1]}
 * (1 <= a_b <= n); the tokens block[0..a_b-1] are committed (their K/V stay,
 * L_b += a_b) and the new head is P[b][a_b-1].
 * Outputs (host): next_out[B][n] = P (y^(j+1) shifted: P[k] predicts block
 * position k+1), accepted_out[B] = a_b; gap_out[B][n] or NULL; logits_out
 * [B][n][vocab] fp32 or NULL (debug: logits are otherwise never stored).
 * The step runs the kernel(s) the decode loop runs for this shape (the
 * persistent per-iteration kernel where cllm_uses_persistent(ctx, n) holds);
 * with logits_out that kernel's LM-head phase also stores the logits.
 * Errors: EINVAL (n outside [1, max_block], token outside the vocab),
 * ESTATE (no prefill), ECAPACITY (L_b + n > max_seq), ECUDA, EDEVICE, ETIMEOUT.
 */
int cllm_jacobi_step(cllm_ctx *ctx, const int32_t *guess, int n, int32_t *next_out,
                     int32_t *accepted_out, float *gap_out, float *logits_out);

/*
 * Jacobi decoding with KV cache of B prompts, max_new tokens each: prefill,
 * then iterations of the step above on a fixed-width block (refill policy:
 * after committing a tokens the block is P[a-1..n-1] followed by a-1 fresh
 * guesses), run entirely on the device as one CUDA graph per iteration with a
 * single 8-byte device->host read per iteration.  A sequence stops after
 * max_new committed tokens (the last commit is truncated) or after committing
 * eos_id.  Guess for (sequence b, iteration j, slot s): the
 * ((b<<40 | j<<16 | s) + 1)-th output of splitmix64 seeded with opts->seed,
 * top 32 bits r mapped to (r*vocab)>>32 (or to prompt_b[(r*len_b)>>32]).
 * tokens_out[B][max_new] (entries past a sequence's end are -1);
 * iters_out[B] = iterations in which the sequence committed tokens (may be NULL).
 * opts may be NULL (seed 0, eos off, uniform guesses).
 * Errors: as cllm_prefill and cllm_jacobi_step, plus ECAPACITY if
 * lens[b] + max_new + n > max_seq.
 */
int cllm_jacobi_decode(cllm_ctx *ctx, int B, const int32_t *tokens, const int32_t *lens,
                       int n, int max_new, const cllm_decode_opts *opts,
                       int32_t *tokens_out, int32_t *iters_out);

/*
 * Greedy AR decoding (Eq. 1) through the same kernels: the Jacobi decode with
 * n = 1 (every iteration commits exactly the head).  tokens_out[B][max_new].
 */
int cllm_ar_decode(cllm_ctx *ctx, int B, const int32_t *tokens, const int32_t *lens,
                   int max_new, int eos_id, int32_t *tokens_out);

/* Static description of a status code. */
const char *cllm_status_string(int status);

/* The last CUDA call that made a call of this thread return CLLM_ECUDA
 * ("<where>: <cudaError name>"), or "none". */
const char *cllm_last_cuda_error(void);

/* ---- device-resident decode loop ---------------------------------------------
 * The three calls cllm_jacobi_decode is made of, for callers that time or
 * drive the loop themselves (inputs and state stay in device memory).
 */

/* Start a decode of the sequences of the last prefill: block width n,
 * max_new tokens each.  Device-only work (resets the per-sequence state to the
 * prefill, draws the first guesses); does not synchronise. */
int cllm_decode_begin(cllm_ctx *ctx, int n, int max_new, const cllm_decode_opts *opts);

/* Run up to max_iters iterations (graph replays).  After each iteration the
 * host reads one 8-byte status {active sequences, committed tokens}; it stops
 * early when no sequence is active.  iters_run and committed (tokens committed
 * by these iterations, summed over sequences) may be NULL. */
int cllm_decode_run(cllm_ctx *ctx, int max_iters, int *iters_run, int64_t *committed);

/* Copy out the decode's tokens [B][max_new] (-1 past the end) and the
 * per-sequence iteration counts [B] (either may be NULL). */
int cllm_decode_read(cllm_ctx *ctx, int32_t *tokens_out, int32_t *iters_out);

/* Copy out the recorded trajectory (Sec. 3.1: the sequence of blocks
 * y^(0), y^(1), ... of Jacobi decoding; Alg. 3 with the decode's block
 * policy): blocks_out[it][b][k] for it < record_cap of cllm_decode_begin's
 * options, k < n; slots beyond a shrunken window and iterations a sequence
 * did not run are -1.  Host buffer of record_cap*B*n ints, owned by the
 * caller.  ESTATE when the decode did not record. */
int cllm_decode_read_trajectory(cllm_ctx *ctx, int32_t *blocks_out);

/*
 * Acceptance statistics of the decode in progress (or just finished), kept
 * on the device by the accept step when cllm_decode_begin's opts->stats = 1
 * (Sec. 3.3 and Table 3 define both quantities in words):
 *  - fast-forwarded count of an iteration: its accepted count a (the head
 *    included, as Table 3 counts it).  acc_hist[a] (host, [n+1] or NULL) =
 *    sequence-iterations that accepted a tokens; out->iterations and
 *    out->accepted are its count and weighted sum.
 *  - stationary tokens: a position is stationary when, before it is
 *    committed, it already holds its final token while an earlier slot of the
 *    block is wrong, and keeps it in every later block until it is committed.
 *    A window is the run of positions covered by the first block that starts
 *    at or after the previous window's end (under CLLM_BLOCK_SHRINK exactly
 *    one n-token window of Alg. 3); stationary tokens count toward the window
 *    that holds them.  win_hist[s] (host, [n+1] or NULL) = windows with s
 *    stationary tokens, windows still open included; out->windows and
 *    out->stationary are the totals.
 * Synchronises the context's stream.  ESTATE without a decode begun with
 * stats = 1; EINVAL on a null ctx or out.
 */
int cllm_decode_read_stats(cllm_ctx *ctx, cllm_accept_stats *out, int64_t *acc_hist,
                           int64_t *win_hist);

/* ---- options --------------------------------------------------------------------
 * CLLM_OPT_PERSISTENT (default 1): run each decode/step iteration of the bf16
 * engine as ONE persistent kernel (one CTA per SM; phases embed, per layer
 * QKV / attention / O / gate-up / down, LM head, accept, separated by grid
 * barriers) when B*n <= 128 and head_dim is 64 or 128; 0 = one kernel per
 * phase.  Both paths compute bit-identical results.  Takes effect for graphs
 * captured after the call.  Returns CLLM_OK or EINVAL (unknown option).
 */
#define CLLM_OPT_PERSISTENT 1
/* CLLM_OPT_PARK_SLOTS (default 0 = all): in the persistent kernel, the weight
 * pairs (32 KB each) a CTA may hold in tensor memory ahead of its MMAs.  The
 * weight stream runs ahead of the grid barriers into these slots, so HBM keeps
 * streaming while a phase drains; 1..64 limits it (values above the kernel's
 * slot count mean all).  Results do not depend on it.  Takes effect for
 * graphs captured after the call. */
#define CLLM_OPT_PARK_SLOTS 3
/* CLLM_OPT_L2_PAIRS (default 0): in the persistent kernel, while a CTA's weight
 * ring and tensor-memory slots are full, its producer prefetches the current
 * phase's next this-many weight pairs (32 KB each) into L2.  0..64.  Results
 * do not depend on it.  Takes effect for graphs captured after the call. */
#define CLLM_OPT_L2_PAIRS 2
/* CLLM_OPT_DATAFLOW (default 1): in the persistent kernel, attention and the
 * O projection start on per-tile completion flags instead of grid barriers:
 * an attention item waits for its head's Q, K and V tiles of the QKV GEMM, a
 * pair of O-projection K chunks for its heads' attention outputs.  0 = grid
 * barriers before both.  Results do not depend on it.  Takes effect for
 * graphs captured after the call. */
#define CLLM_OPT_DATAFLOW 4
int cllm_set_option(cllm_ctx *ctx, int option, int value);

/* 1 if an iteration of width n on the current batch runs as the persistent
 * kernel, 0 if as one kernel per phase, or a negative status. */
int cllm_uses_persistent(cllm_ctx *ctx, int n);

/* ---- introspection ----------------------------------------------------------- */

/* Per-launch device time of each kernel class in the last profiled iteration
 * (cllm_set_profiling(ctx, 1) captures CUDA events around every kernel of the
 * iteration graph).  names/ms: up to cap entries; returns the entry count.
 * Kernel classes: "embed", "gemm_qkv", "attention", "attn_combine", "gemm_o",
 * "gemm_gateup", "gemm_down", "gemm_lmhead", "accept"; for the persistent
 * kernel: "step_persistent" (the kernel) and "phase:<class>" (per-phase time
 * from in-kernel timestamps of CTA 0). */
int cllm_set_profiling(cllm_ctx *ctx, int on);
int cllm_profile_read(cllm_ctx *ctx, const char **names, float *ms_total, int *launches,
                      int cap);

/* Number of kernel launches of one decode iteration at block width n for the
 * current batch (what one graph replay launches). */
int cllm_kernels_per_iteration(cllm_ctx *ctx, int n);

/* Committed length L_b of each sequence (host array [B]). */
int cllm_committed_lengths(cllm_ctx *ctx, int32_t *lens_out);

/* ---- allocation-free GEMM -----------------------------------------------------
 * The paper has no counterpart of this call; it serves callers that cannot
 * call cudaMalloc -- code under a caching allocator that has reserved the
 * device's memory, or a latency-critical path that cannot take the implicit
 * device synchronisation of cudaMalloc/cudaFree.
 * Computes, with the library's bf16 weight-streaming GEMM kernel,
 *   Y[t][m] += sum_k W[m][k] * (Xhi[t][k] + Xlo[t][k])   for t < T, m < M.
 * W: device bf16 [M][K]; X: device bf16 [2][x_rows][K] (hi plane, then lo
 * plane), x_rows >= T rounded up to 16 (and >= 256 when T > 256); Y: device
 * fp32 [T][M], accumulated into.  M a multiple of 128, K a multiple of 8.
 * cuda_stream: the cudaStream_t to run on (NULL = the legacy default stream);
 * the call synchronises it before returning, so it can never be captured into
 * a CUDA graph: on a stream that is capturing it returns CLLM_EUNSUPPORTED
 * before any work is queued.
 * No memory is allocated: all scratch (split-K partial tiles, arrival tickets,
 * the device error word, epilogue side outputs) lives in one static device
 * array of 8 MiB that each device loading the library holds until exit.  Sizes
 * whose scratch would exceed it return CLLM_ECAPACITY before any launch.  Each
 * call looks up the array's device address in the current device's current
 * context (a host-side lookup), so a reset device or a second context on the
 * same device gets its own copy.  Every call reuses the same array (tickets
 * and the error word are cleared at the start of each call; the rest keeps
 * the previous call's contents and is overwritten before it is read), so calls
 * that overlap on the GPU -- from several threads or streams -- race and must
 * not be issued.
 * Returns CLLM_OK, EINVAL, ECAPACITY, EUNSUPPORTED, ECUDA, EDEVICE or ETIMEOUT.
 */
int cllm_gemm_bf16_noalloc(const void *W, const void *X, float *Y, int M, int K, int T,
                           int x_rows, void *cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* CLLM_H */
