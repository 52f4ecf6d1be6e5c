// Internal declarations shared by the kernels and the host engine.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace cllm {

// Device error bits (the device status word); never __trap()/assert.
enum : int {
  DERR_TOKEN = 1,     // a token id outside [0, vocab)
  DERR_CAPACITY = 2,  // a position at or past max_seq
  DERR_TIMEOUT = 4,   // a bounded wait ran out
  DERR_SHAPE = 8,     // an internal shape check failed
};

constexpr int kAttnChunk = 128;  // keys per attention chunk, anchored at absolute positions
// Tensor-core attention: a work item covers a range of kAttnRange consecutive
// chunks (anchored the same way, so a row's split does not depend on the
// block size); partials are per range.
constexpr int kAttnRange = 4;
constexpr int kQTile = 16;       // query rows per attention tile
constexpr int kBK = 64;          // K elements per pipeline stage (128 B of bf16)
constexpr int kBM = 128;         // weight rows per tile (MMA M)
constexpr int kEpiCols = 16;     // columns per epilogue chunk
// Weight tiles per CTA prefetched into L2 ahead of the shared-memory ring by
// the per-GEMM kernels.  Measured on chains of GEMM launches: it adds traffic
// without shortening the chain, so it is off.
constexpr int kL2AheadDefault = 0;

enum EpiKind : int { EPI_QKV = 0, EPI_GATEUP = 1, EPI_RESID = 2, EPI_ARGMAX = 3 };

// Per-launch epilogue arguments (passed by value; one struct for all kinds).
struct EpiArgs {
  int T;      // valid token rows of this launch
  int ldt;    // row stride (tokens) of the per-token partial arrays (ssq, argmax)
  // RMSNorm scale of the GEMM input: rs[t] = 1/sqrt(sum_i ssq_in[i*ldt+t] / d + eps)
  const float* ssq_in;
  int ssq_tiles;
  float inv_d, eps;
  // QKV: rotate-half RoPE, Q out, K/V into the cache at (bidx[t], pos[t])
  void* q_out;
  void* k_cache;  // this layer's [B][Hkv][max_seq][hd]
  void* v_cache;
  int dq, dkv, hd, n_kv_heads, max_seq;
  const int* pos;
  const int* bidx;
  const float2* rope;  // [max_seq][hd/2] (cos, sin)
  // GATEUP: h[t][f] = silu(gate) * up
  void* h_out;
  int F;
  size_t plane_h;  // element offset of h's lo plane (bf16 engine)
  // RESID: x += D; xg = x * gnext; ssq_out per 128-row tile
  float* x;
  void* xg;
  const void* gnext;
  float* ssq_out;
  int d;
  size_t plane_x;  // element offset of xg's lo plane (bf16 engine)
  // ARGMAX: per-tile (max, argmax, second max); last unit reduces to pred/gap
  float* am_part;  // [mtiles][ldt][3]
  int* am_ticket;
  int am_units;
  int am_mtiles;
  int* pred;
  float* gap;
  float* logits;  // optional debug [T][V]
  int V;
  int* err;
  // persistent kernel: completion flag of each finished output tile (QKV:
  // released after the tile's Q/K/V stores; null: none)
  unsigned* tile_done;
  // optional timing of the epilogue's last segment (persistent kernel
  // profiling): dbg[k * dbg_stride + cta], k = 0 accumulator ready, 1 after
  // the arrival ticket, 2 epilogue done, 4 split-K partials summed (owner)
  unsigned long long* dbg;
  long long dbg_stride;
};

// Work decomposition of one weight-streaming GEMM launch.
//   D[m][t] = sum_k W[m][k] X[t][k]  (m: weight rows, t: tokens)
// The chunk space (unit, k-chunk) is split into contiguous ranges of `cpc`
// chunks, one per CTA; a unit is one 128-row tile x one N-tile of tokens.
struct GemmArgs {
  int M, K, T;
  int mtiles, ntiles, kchunks, cpc, bn, maxc;
  int rows_q, rows_qk;  // QKV: first rows of the K and V sections (weight-map select)
  int lo_rows;          // row offset of the activations' lo plane in the B map
  int l2_ahead;         // weight tiles per CTA prefetched into L2 before the PDL wait
  int pre_stages;       // weight tiles issued before the phase's dependency is met (<= ring)
  float* partial;       // [units*maxc][bn][128] split-K partial tiles
  int* tickets;         // [units] arrival counters (self-resetting)
  // SIMT (fp32) path only
  const void* A0;
  const void* A1;
  const void* A2;
  const void* X;
  int ldx;
  int* err;
};

struct AttnArgs {
  const void* q;        // [T][n_heads*hd]
  const void* k_cache;  // this layer's [B][Hkv][max_seq][hd]
  const void* v_cache;
  const int* seq_start;  // [B] position of the sequence's first row
  const int* seq_row0;   // [B] index of the sequence's first row
  const int* seq_nrows;  // [B]
  const int2* qtiles;    // (b, first row within sequence) per 16-row query tile
  int n_qtiles;
  int H, Hkv, hd, max_seq, nch_max;
  float scale_log2;   // log2(e) / sqrt(hd)
  float* part_o;      // [row][H][nch_max][hd], unnormalised
  float2* part_ml;    // [row][H][nch_max]: (running max in log2 units, sum)
  const int* pos;     // [T]
  void* out;          // [T][H*hd] (+ lo plane in the bf16 engine)
  size_t plane_out;
  int T;
  int* err;
};

struct EmbedArgs {
  const void* emb;    // [V][d]
  const void* gain;   // first layer's attention-norm gain [d]
  int V, d, T, ldt;
  // step mode (block != nullptr): row t = b*n + k, token block[b][k], position L[b] + k
  const int* block;
  const int* L;
  int n, B, max_seq;
  // prefill mode: per-row token / position / sequence given
  const int* tok_in;
  const int* pos_in;
  const int* bidx_in;
  // outputs
  float* x;
  void* xg;
  size_t plane;  // element offset of xg's lo plane (bf16 engine)
  float* ssq;  // [d/128][ldt]
  int* pos;
  int* bidx;
  int* seq_start;
  int* seq_row0;
  int* seq_nrows;
  int* err;
};

struct AcceptArgs {
  int B, n, V;
  int decode;  // 1: decode loop (commit to out, done flags, refill); 0: single step
  int max_new, eos;
  unsigned long long seed;
  int guess_mode;
  const int* pred;  // [B*n]
  int* block;       // [B][n]
  int* L;
  int* head;
  int* committed;
  int* iters;
  int* done;
  int* out;  // [B][max_new]
  int* accepted;
  const int* prompts;  // [B][max_seq]
  const int* plen;
  int prompt_ld;
  int* status;  // [0] active sequences, [1] tokens committed by this iteration
  // block policy (Alg. 3): 0 refill (always n wide), 1 shrink (the window
  // narrows by the accepted count until it is fixed, then a fresh n-wide block)
  int shrink;
  int* width;  // [B] current block width (shrink)
  // lookahead policy (refill with an n-gram pool; null: off): pool[b][tok]
  // holds the pool_w tokens that followed tok in the latest n-gram of
  // sequence b's predictions, pool[b][tok][0] = -1 when there is none
  int* pool;
  int pool_w;
  // optional trajectory: traj[it][b][k] = the block of sequence b at its
  // iteration it (slot k < width, -1 beyond), for it < traj_cap
  int* traj;
  int traj_cap;
  // acceptance statistics of a decode (Sec. 3.3, Table 3), kept on the device
  // (null: off).  acc_hist[a]: sequence-iterations that accepted a tokens;
  // win_hist[s]: closed n-token windows with s stationary tokens; totals[0]
  // windows opened, totals[1] stationary tokens inside windows.  Per sequence
  // b and window slot q = position mod n: st_pos/st_val the position and value
  // the slot last held, st_cand whether, since that value arrived, an earlier
  // slot of the block was wrong; win_end/win_cnt the open window's end and its
  // stationary count.  Positions count committed tokens from the decode start.
  unsigned long long* acc_hist;  // [n + 1]
  unsigned long long* win_hist;  // [n + 1]
  unsigned long long* totals;    // [2]
  int* st_pos;                   // [B][n]
  int* st_val;                   // [B][n]
  int* st_cand;                  // [B][n]
  int* win_end;                  // [B]
  int* win_cnt;                  // [B]
};

// ---- persistent per-iteration kernel (persistent.cu) ---------------------------------

enum PhaseKind : int { PH_EMBED = 0, PH_GEMM = 1, PH_ATTN = 2, PH_ACCEPT = 3 };

// One phase of an iteration.  GEMM phases name their tensor maps by index
// into the map table; attention phases carry their layer's K/V cache.
struct PhaseDesc {
  int kind, epi;
  int map_a0, map_a1, map_a2, map_b;
  GemmArgs g;
  EpiArgs e;
  const void* k_cache;
  const void* v_cache;
  int kv_row0;  // attention: the layer's first row in the K/V cache tensor maps
  // Dependencies narrower than the grid barrier (no_barrier = 1: the phase
  // does not wait for it).  Attention: the item of head h waits until the
  // QKV tile flags qkv_done[] of h's Q, K and V tiles reach flag_target (the
  // QKV GEMM's column tiles), and adds 1 to head_done[h] for every query tile
  // whose output it completes.  O projection: a pair of K chunks waits for
  // its heads' head_done[] to reach flag_target (the query tiles) and for
  // this CTA's attention phase to end.
  int no_barrier;
  const unsigned* qkv_done;
  unsigned* head_done;
  int flag_target;
};

struct StepArgs {
  const PhaseDesc* phases;
  int n_phases;
  unsigned* bar;            // grid barrier counter, zero at launch
  EmbedArgs embed;
  AttnArgs attn;            // K/V cache set per phase
  int* attn_tickets;        // [qtiles][heads], self-resetting
  AcceptArgs accept;
  unsigned long long* stamps;  // optional: phase start times (CTA 0)
  // optional: [kCtaStampSlots][phase][cta] -- epilogue group start, MMA done,
  // arrival, 3 epilogue stamps, producer start, (unused), producer done,
  // (unused), first and last stage arrival at the MMA, largest gap between
  // arrivals (ns); then kTraceCap stage arrivals per CTA of phase trace_phase
  unsigned long long* cta_stamps;
  int trace_phase;  // -1: none
  // test hook: the grid barrier before this phase waits for one arrival more
  // than the grid makes, so its bounded waits run out (-1: none)
  int hold_phase;
  // attention tile loads: indices of the K-cache, V-cache and Q tensor maps
  int map_attn_k, map_attn_v, map_attn_q;
  // tensor-memory park slots the weight stream may fill ahead of the MMAs
  // (0: all the kernel has)
  int park_limit;
  // weight pairs of the current phase prefetched into L2 while the weight
  // ring is full (0: none)
  int l2_ahead;
  int* err;
};

constexpr int kCtaStampSlots = 13;
constexpr int kTraceCap = 256;
constexpr int kMaxQTilesStep = 256;  // query tiles of one iteration (persistent kernel)

// Tensor maps travel by value in the kernel's parameter space (TMA reads
// descriptors there as it does for per-GEMM kernels): 7 per layer + the LM
// head + 4 activation maps + the attention's K, V and Q maps, at most 32
// layers (29.7 KB of the 32 KB limit).
constexpr int kMaxStepMaps = 7 * 32 + 8;
struct StepParams {
  StepArgs a;
  CUtensorMap maps[kMaxStepMaps];
};
static_assert(sizeof(StepParams) <= 32764, "kernel parameter space");

// Launch of the persistent kernel (bn_max 16/32/64/128, head_dim 64/128).
cudaError_t launch_step_persistent(const StepParams& p, int bn_max, int hd, int grid,
                                   cudaStream_t s, bool cooperative);
cudaError_t step_persistent_set_attributes();
size_t step_persistent_smem_bytes(int bn_max, int hd);

// ---- launchers (kernels.cu) --------------------------------------------------------
struct GemmMaps {
  CUtensorMap a0, a1, a2, b;
};

// Tensor maps of the attention tiles: the K and V caches of all layers as rows
// of hd values (128-row boxes) and Q (16-row boxes), 64-column halves with the
// 128-byte swizzle.
struct AttnMaps {
  CUtensorMap k, v, q;
};

inline int ceil_div(int a, int b) { return (a + b - 1) / b; }
inline int round_up(int a, int b) { return ceil_div(a, b) * b; }

// Work split of one GEMM launch (api.cu).
struct Part {
  int mtiles, ntiles, kchunks, cpc, bn, bn_max, maxc, grid;
};
Part plan_gemm(int mtiles, int K, int T, int sms);
// bf16 [outer][inner] tensor map: 64-column x box_outer-row tiles, 128-byte swizzle.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint32_t box_outer);

cudaError_t launch_embed(const EmbedArgs& a, int act_bf16, cudaStream_t s, bool pdl);
cudaError_t launch_gemm_tc(int kind, int bn_max, const GemmMaps& maps, const GemmArgs& g,
                           const EpiArgs& e, int grid, cudaStream_t s, bool pdl);
cudaError_t launch_gemm_simt(int kind, const GemmArgs& g, const EpiArgs& e, cudaStream_t s,
                             bool pdl);
cudaError_t launch_attention(const AttnArgs& a, int act_bf16, int grid, cudaStream_t s, bool pdl);
// bf16 engine with tensor maps: Q, K and V tiles by TMA (kv_row0: the layer's
// first cache row in the maps)
cudaError_t launch_attention_tma(const AttnArgs& a, const AttnMaps& m, int kv_row0, int grid,
                                 cudaStream_t s, bool pdl);
cudaError_t launch_attn_combine(const AttnArgs& a, int act_bf16, cudaStream_t s, bool pdl);
cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t s, bool pdl);
cudaError_t launch_decode_init(const AcceptArgs& a, cudaStream_t s);
cudaError_t launch_set_head(int* block, const int* head, int B, int n, int V, int* err,
                            cudaStream_t s);
cudaError_t launch_gather_rows(const void* xg_src, const float* ssq_src, void* xg_dst,
                               float* ssq_dst, const int* rows, int B, int d, int ldt_src,
                               int ldt_dst, size_t plane_src, size_t plane_dst, int act_bf16,
                               cudaStream_t s);
int gemm_tc_stages(int bn_max);
size_t gemm_tc_smem_bytes(int bn_max);
cudaError_t gemm_tc_set_attributes();
cudaError_t attention_set_attributes();
size_t attention_smem_bytes(int act_bf16, int hd);

}  // namespace cllm
