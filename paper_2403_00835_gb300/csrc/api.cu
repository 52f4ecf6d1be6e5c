// Host engine behind include/cllm.h: context, device buffers, TMA
// descriptors, GEMM work partitioning, and the recorder that issues one block
// forward (embed -> layers -> LM head -> accept) eagerly, into a CUDA graph,
// or into a profiled graph with timing events between kernels.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <map>
#include <memory>
#include <new>
#include <string>
#include <tuple>
#include <vector>

#include "../../include/cllm.h"
#include "internal.cuh"

using namespace cllm;


namespace cllm {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// bf16 row-major [outer][inner] matrix, tiles of box_outer rows x 64 columns,
// 128-byte swizzle (the layout the tcgen05 descriptors expect).
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint32_t box_outer) {
  EncodeTiledFn enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), box_outer};
  cuuint32_t estr[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Split of one GEMM launch over the SMs.  T <= 256: one N-tile holding every
// token and the (tile, k-chunk) space cut into equal contiguous ranges; the
// cut depends on the weight shape and the SM count only.  T > 256: whole
// 128 x 256 tiles per CTA, no split.  Chunks per tile and per CTA are even,
// so that every range and every tile starts on a pair of chunks: the
// persistent kernel moves weights in pairs (32 KB per pipeline stage), in the
// same order as the per-chunk kernels, which keeps the two paths bit-identical.
// (A K that is not a multiple of 128 gets one chunk past its end, which TMA
// fills with zeros.)
Part plan_gemm(int mtiles, int K, int T, int sms) {
  Part p{};
  p.mtiles = mtiles;
  p.kchunks = round_up(ceil_div(K, kBK), 2);
  if (T <= 256) {
    p.ntiles = 1;
    p.bn = round_up(std::max(T, 1), 16);
    p.bn_max = p.bn <= 32 ? 32 : (p.bn <= 64 ? 64 : (p.bn <= 128 ? 128 : 256));
    const int C = mtiles * p.kchunks;
    p.cpc = round_up(ceil_div(C, sms), 2);
    p.grid = ceil_div(C, p.cpc);
    p.maxc = 1;
    for (int u = 0; u < mtiles; ++u) {
      const int first = (u * p.kchunks) / p.cpc, last = ((u + 1) * p.kchunks - 1) / p.cpc;
      p.maxc = std::max(p.maxc, last - first + 1);
    }
  } else {
    p.bn = p.bn_max = 256;
    p.ntiles = ceil_div(T, 256);
    const int units = mtiles * p.ntiles;
    const int upc = ceil_div(units, sms);
    p.cpc = upc * p.kchunks;
    p.grid = ceil_div(units, upc);
    p.maxc = 1;
  }
  return p;
}

}  // namespace cllm

namespace {

struct LayerW {
  const void *attn_norm, *wq, *wk, *wv, *wo, *mlp_norm, *w_gate, *w_up, *w_down;
  CUtensorMap mq, mk, mv, mo, mgate, mup, mdown;
};

enum Mode { MODE_PREFILL = 0, MODE_STEP = 1, MODE_DECODE = 2 };


}  // namespace

struct cllm_ctx {
  cllm_arch arch{};
  int dev = 0, sms = 0;
  cudaStream_t stream = nullptr;
  bool own_stream = false;
  bool bf16 = true;
  size_t esz = 2;
  int d = 0, H = 0, Hkv = 0, hd = 0, dq = 0, dkv = 0, F = 0, V = 0, NL = 0;
  int Tcap = 0, prefill_cap = 0, nch_max = 0, max_qtiles = 0;
  int planes = 1;  // GEMM activation planes: 2 (bf16 hi + lo) in the bf16 engine
  // weights
  const void *tok_emb = nullptr, *final_norm = nullptr, *lm_head = nullptr;
  CUtensorMap mlm{};
  std::vector<LayerW> layers;
  // activations and scratch
  float* x = nullptr;
  void* xg = nullptr;
  float* ssq = nullptr;
  void* q = nullptr;
  void* attn = nullptr;
  void* h = nullptr;
  void* xg_last = nullptr;
  float* ssq_last = nullptr;
  int* last_rows = nullptr;
  void* kc = nullptr;
  void* vc = nullptr;
  size_t layer_kv_elems = 0;
  float2* rope = nullptr;
  float* part_o = nullptr;
  float2* part_ml = nullptr;
  float* gemm_part = nullptr;
  size_t gemm_part_elems = 0;
  int* tickets = nullptr;
  int max_mtiles = 0;
  float* am_part = nullptr;
  int* am_ticket = nullptr;
  int* pred = nullptr;
  float* gap = nullptr;
  float* logits_dbg = nullptr;
  int *tok_in = nullptr, *pos_in = nullptr, *bidx_in = nullptr, *pos = nullptr, *bidx = nullptr;
  int *seq_start = nullptr, *seq_row0 = nullptr, *seq_nrows = nullptr;
  int2* qtiles_prefill = nullptr;
  // sequence state
  int *Ld = nullptr, *head = nullptr, *head0 = nullptr, *block = nullptr, *committed = nullptr,
      *iters = nullptr, *done = nullptr, *out = nullptr, *accepted = nullptr, *prompts = nullptr,
      *plen = nullptr, *status = nullptr, *err = nullptr, *width = nullptr;
  size_t out_cap = 0;
  // acceptance statistics (cllm_decode_opts.stats): histograms [max_block+1],
  // totals [2], per-sequence slot state [max_batch][max_block], windows [max_batch]
  unsigned long long *acc_hist = nullptr, *win_hist = nullptr, *st_totals = nullptr;
  int *st_pos = nullptr, *st_val = nullptr, *st_cand = nullptr, *win_end = nullptr,
      *win_cnt = nullptr;
  int* traj = nullptr;  // recorded trajectory [traj_cap][B][n]
  size_t traj_alloc = 0;
  int* pool = nullptr;  // lookahead policy's n-gram pools [B][V][ngram - 1]
  size_t pool_alloc = 0;
  AttnMaps attn_maps{};     // bf16 engine: tensor maps of the attention tiles
  bool attn_maps_ok = false;
  int traj_cap = 0;
  int* status_host = nullptr;  // pinned: slots of 4 ints {active, committed, device error, -}
  cudaEvent_t iter_ev[2] = {nullptr, nullptr};
  // host state
  int B = 0;
  std::vector<int> lens, Lh;
  bool prefilled = false;
  bool dec_active = false;
  int dec_n = 0, dec_max_new = 0;
  cllm_decode_opts dec_opts{};
  std::vector<void*> allocs;
  struct GraphEntry {
    cudaGraphExec_t exec = nullptr;
    int2* qtiles = nullptr;
    int launches = 0;
    bool persistent = false;
    int n_phases = 0;
    std::vector<int> phase_kind;       // PhaseKind / EPI_* per phase (profiling)
    std::vector<std::string> phase_names;
    std::vector<void*> bufs;           // device tables owned by the graph
    unsigned long long* stamps = nullptr;
    unsigned long long* cta_stamps = nullptr;
    size_t bar_bytes = 64;             // grid-barrier counter and completion flags
  };
  bool persistent = true;  // one persistent kernel per iteration where supported
  int park_slots = 0;  // persistent kernel: tensor-memory park slots in use (0: all)
  int l2_pairs = 0;    // persistent kernel: weight pairs prefetched into L2 when the ring is full
  bool dataflow = true;  // persistent kernel: attention and O open on completion flags
  std::vector<unsigned long long> last_stamps;  // last profiled persistent iteration
  std::vector<std::string> last_phase_names;
  std::vector<unsigned long long> last_cta_stamps;
  int trace_phase = -1;  // profiling: phase whose MMA stage arrivals are traced
  int hold_phase = -1;   // test hook: grid barrier that cannot open (bounded-wait path)
  bool step_logits = false;  // the step graph being built stores the LM head's logits
  std::map<std::tuple<int, int, int, int, int, unsigned long long, int, int, int, int>, GraphEntry>
      graphs;
  // profiling
  bool profiling = false;
  std::vector<cudaEvent_t> prof_events;
  std::vector<std::string> prof_names;
  std::map<std::string, std::pair<double, int>> prof_acc;
  // recorder state
  std::vector<const char*>* rec_names = nullptr;
  int rec_count = 0;
};

namespace {

thread_local char g_last_cuda_error[160] = "none";

// Record a failed CUDA call (name and where) and return CLLM_ECUDA.
int cuda_fail(cudaError_t e, const char* where) {
  snprintf(g_last_cuda_error, sizeof g_last_cuda_error, "%s: %s", where, cudaGetErrorName(e));
  return CLLM_ECUDA;
}

// Test hook (cllm_test_fail_alloc): the device or pinned allocation that
// brings the countdown from 0 to -1 fails as if the memory were exhausted.
std::atomic<int> g_alloc_countdown{-1};

bool alloc_injected_failure() {
  int v = g_alloc_countdown.load();
  while (v >= 0 && !g_alloc_countdown.compare_exchange_weak(v, v - 1)) {
  }
  return v == 0;
}

cudaError_t lib_malloc(void** p, size_t bytes) {
  if (alloc_injected_failure()) return cudaErrorMemoryAllocation;
  return cudaMalloc(p, bytes);
}

template <typename T>
bool dev_alloc(cllm_ctx* c, T** p, size_t bytes) {
  void* v = nullptr;
  if (bytes == 0) bytes = 16;
  if (lib_malloc(&v, bytes) != cudaSuccess) return false;
  if (cudaMemset(v, 0, bytes) != cudaSuccess) return false;
  c->allocs.push_back(v);
  *p = static_cast<T*>(v);
  return true;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// after each kernel in the recorder: count, and in profiled capture, time
cudaError_t after_launch(cllm_ctx* c, cudaStream_t s, const char* name, cudaError_t e) {
  if (e != cudaSuccess) return e;
  c->rec_count++;
  if (c->rec_names) {
    c->rec_names->push_back(name);
    const size_t i = c->rec_names->size();
    if (i < c->prof_events.size())
      return cudaEventRecordWithFlags(c->prof_events[i], s, cudaEventRecordExternal);
  }
  return cudaSuccess;
}

EpiArgs base_epi(cllm_ctx* c, int T) {
  EpiArgs e{};
  e.T = T;
  e.ldt = c->Tcap;
  e.inv_d = 1.f / static_cast<float>(c->d);
  e.eps = c->arch.rms_eps;
  e.ssq_tiles = c->d / kBM;
  e.dq = c->dq;
  e.dkv = c->dkv;
  e.hd = c->hd;
  e.n_kv_heads = c->Hkv;
  e.max_seq = c->arch.max_seq;
  e.pos = c->pos;
  e.bidx = c->bidx;
  e.rope = c->rope;
  e.F = c->F;
  e.d = c->d;
  e.V = c->V;
  e.err = c->err;
  e.plane_x = c->planes == 2 ? static_cast<size_t>(c->Tcap) * c->d : 0;
  e.plane_h = c->planes == 2 ? static_cast<size_t>(c->Tcap) * c->F : 0;
  return e;
}

// Work split and epilogue bookkeeping of one bf16 GEMM of T tokens.
GemmArgs tc_gemm_args(cllm_ctx* c, int mtiles, int M, int K, int T, EpiArgs& e, Part* part) {
  GemmArgs g{};
  g.M = M;
  g.K = K;
  g.T = T;
  g.rows_q = c->dq;
  g.rows_qk = c->dq + c->dkv;
  g.err = c->err;
  g.tickets = c->tickets;
  g.partial = c->gemm_part;
  g.lo_rows = c->Tcap;
  g.l2_ahead = kL2AheadDefault;
  g.pre_stages = 1 << 20;
  const Part p = plan_gemm(mtiles, K, T, c->sms);
  g.mtiles = p.mtiles;
  g.ntiles = p.ntiles;
  g.kchunks = p.kchunks;
  g.cpc = p.cpc;
  g.bn = p.bn;
  g.maxc = p.maxc;
  e.am_units = mtiles * p.ntiles;
  e.am_mtiles = mtiles;
  if (part) *part = p;
  return g;
}

// One GEMM launch: D[m][t] = W[m] . X[t] with epilogue `kind`.
cudaError_t gemm(cllm_ctx* c, cudaStream_t s, bool pdl, int kind, int mtiles, int M, int K, int T,
                 const void* X, const void* A0, const void* A1, const void* A2,
                 const CUtensorMap* m0, const CUtensorMap* m1, const CUtensorMap* m2,
                 const EpiArgs& e, const char* name) {
  GemmArgs g{};
  g.M = M;
  g.K = K;
  g.T = T;
  g.rows_q = c->dq;
  g.rows_qk = c->dq + c->dkv;
  g.err = c->err;
  g.tickets = c->tickets;
  g.partial = c->gemm_part;
  g.lo_rows = c->Tcap;
  g.l2_ahead = kL2AheadDefault;
  g.pre_stages = 1 << 20;
  cudaError_t err;
  if (!c->bf16) {
    g.mtiles = mtiles;
    g.ntiles = ceil_div(T, kEpiCols);
    g.A0 = A0;
    g.A1 = A1;
    g.A2 = A2;
    g.X = X;
    g.ldx = K;
    EpiArgs ee = e;
    ee.am_units = mtiles * g.ntiles;
    ee.am_mtiles = mtiles;
    err = launch_gemm_simt(kind, g, ee, s, pdl);
  } else {
    EpiArgs ee = e;
    Part p;
    g = tc_gemm_args(c, mtiles, M, K, T, ee, &p);
    if (static_cast<size_t>(mtiles) * p.maxc * p.bn * kBM > c->gemm_part_elems && p.ntiles == 1)
      return cudaErrorInvalidValue;
    GemmMaps maps{};
    maps.a0 = *m0;
    maps.a1 = m1 ? *m1 : *m0;
    maps.a2 = m2 ? *m2 : *m0;
    if (!make_map(&maps.b, X, static_cast<uint64_t>(K), static_cast<uint64_t>(2 * c->Tcap),
                  static_cast<uint32_t>(p.bn)))
      return cudaErrorInvalidValue;
    err = launch_gemm_tc(kind, p.bn_max, maps, g, ee, p.grid, s, pdl);
  }
  return after_launch(c, s, name, err);
}

struct FwdSpec {
  int mode;  // MODE_*
  int T;     // block rows (step) or prefill rows
  int B, n;  // step/decode shape
  int n_qtiles;
  const int2* qtiles;
  int attn_grid;
  int n_last;  // prefill: rows whose logits are needed (gathered)
  bool want_logits;
  AcceptArgs acc;  // step/decode
};

EmbedArgs make_embed_args(cllm_ctx* c, const FwdSpec& f) {
  const int T = f.T;
  EmbedArgs ea{};
  ea.emb = c->tok_emb;
  ea.gain = c->layers[0].attn_norm;
  ea.V = c->V;
  ea.d = c->d;
  ea.T = T;
  ea.ldt = c->Tcap;
  ea.max_seq = c->arch.max_seq;
  if (f.mode == MODE_PREFILL) {
    ea.tok_in = c->tok_in;
    ea.pos_in = c->pos_in;
    ea.bidx_in = c->bidx_in;
  } else {
    ea.block = c->block;
    ea.L = c->Ld;
    ea.n = f.n;
    ea.B = f.B;
  }
  ea.x = c->x;
  ea.xg = c->xg;
  ea.plane = c->planes == 2 ? static_cast<size_t>(c->Tcap) * c->d : 0;
  ea.ssq = c->ssq;
  ea.pos = c->pos;
  ea.bidx = c->bidx;
  ea.seq_start = c->seq_start;
  ea.seq_row0 = c->seq_row0;
  ea.seq_nrows = c->seq_nrows;
  ea.err = c->err;
  return ea;
}

AttnArgs make_attn_args(cllm_ctx* c, const FwdSpec& f) {
  const int T = f.T;
  AttnArgs aa{};
  aa.q = c->q;
  aa.seq_start = c->seq_start;
  aa.seq_row0 = c->seq_row0;
  aa.seq_nrows = c->seq_nrows;
  aa.qtiles = f.qtiles;
  aa.n_qtiles = f.n_qtiles;
  aa.H = c->H;
  aa.Hkv = c->Hkv;
  aa.hd = c->hd;
  aa.max_seq = c->arch.max_seq;
  aa.nch_max = c->nch_max;
  aa.scale_log2 = 1.4426950408889634f / std::sqrt(static_cast<float>(c->hd));
  aa.part_o = c->part_o;
  aa.part_ml = c->part_ml;
  aa.pos = c->pos;
  aa.out = c->attn;
  aa.plane_out = c->planes == 2 ? static_cast<size_t>(c->Tcap) * c->dq : 0;
  aa.T = T;
  aa.err = c->err;
  return aa;
}

// Issue one forward (+ accept) on stream s.
cudaError_t record_forward(cllm_ctx* c, cudaStream_t s, const FwdSpec& f, bool pdl) {
  cudaError_t err;
  const int T = f.T;
  const int ab = c->bf16 ? 1 : 0;
  const EmbedArgs ea = make_embed_args(c, f);
  if ((err = after_launch(c, s, "embed", launch_embed(ea, ab, s, pdl))) != cudaSuccess) return err;
  AttnArgs aa = make_attn_args(c, f);

  for (int l = 0; l < c->NL; ++l) {
    const LayerW& L = c->layers[l];
    const size_t kvoff = static_cast<size_t>(l) * c->layer_kv_elems * c->esz;
    void* kl = static_cast<char*>(c->kc) + kvoff;
    void* vl = static_cast<char*>(c->vc) + kvoff;
    // (a2) RMSNorm scale + QKV + RoPE + K/V into the cache
    EpiArgs e = base_epi(c, T);
    e.ssq_in = c->ssq;
    e.q_out = c->q;
    e.k_cache = kl;
    e.v_cache = vl;
    const int Mqkv = c->dq + 2 * c->dkv;
    if ((err = gemm(c, s, pdl, EPI_QKV, Mqkv / kBM, Mqkv, c->d, T, c->xg, L.wq, L.wk, L.wv, &L.mq,
                    &L.mk, &L.mv, e, "gemm_qkv")) != cudaSuccess)
      return err;
    // (a3) block attention, split over position-anchored key chunks
    aa.k_cache = kl;
    aa.v_cache = vl;
    {
      const int kv_row0 = static_cast<int>(static_cast<size_t>(l) * c->layer_kv_elems / c->hd);
      const cudaError_t la = c->attn_maps_ok
                                 ? launch_attention_tma(aa, c->attn_maps, kv_row0, f.attn_grid, s, pdl)
                                 : launch_attention(aa, ab, f.attn_grid, s, pdl);
      if ((err = after_launch(c, s, "attention", la)) != cudaSuccess) return err;
    }
    if ((err = after_launch(c, s, "attn_combine", launch_attn_combine(aa, ab, s, pdl))) !=
        cudaSuccess)
      return err;
    // (a4) O-proj + residual; leaves the MLP norm's input and statistics
    e = base_epi(c, T);
    e.x = c->x;
    e.xg = c->xg;
    e.gnext = L.mlp_norm;
    e.ssq_out = c->ssq;
    if ((err = gemm(c, s, pdl, EPI_RESID, c->d / kBM, c->d, c->dq, T, c->attn, L.wo, nullptr,
                    nullptr, &L.mo, nullptr, nullptr, e, "gemm_o")) != cudaSuccess)
      return err;
    // (a5) RMSNorm scale + gate/up + SwiGLU
    e = base_epi(c, T);
    e.ssq_in = c->ssq;
    e.h_out = c->h;
    if ((err = gemm(c, s, pdl, EPI_GATEUP, ceil_div(c->F, 64), c->F, c->d, T, c->xg, L.w_gate,
                    L.w_up, nullptr, &L.mgate, &L.mup, nullptr, e, "gemm_gateup")) != cudaSuccess)
      return err;
    // (a6) down + residual; leaves the next norm's input and statistics
    e = base_epi(c, T);
    e.x = c->x;
    e.xg = c->xg;
    e.gnext = (l + 1 < c->NL) ? c->layers[l + 1].attn_norm : c->final_norm;
    e.ssq_out = c->ssq;
    if ((err = gemm(c, s, pdl, EPI_RESID, c->d / kBM, c->d, c->F, T, c->h, L.w_down, nullptr,
                    nullptr, &L.mdown, nullptr, nullptr, e, "gemm_down")) != cudaSuccess)
      return err;
  }
  // (a7) final norm scale + LM head + argmax / top-2 gap
  EpiArgs e = base_epi(c, T);
  e.am_part = c->am_part;
  e.am_ticket = c->am_ticket;
  e.pred = c->pred;
  e.gap = c->gap;
  e.logits = f.want_logits ? c->logits_dbg : nullptr;
  const int mt_v = ceil_div(c->V, kBM);
  if (f.mode == MODE_PREFILL) {
    if ((err = after_launch(c, s, "gather",
                            launch_gather_rows(c->xg, c->ssq, c->xg_last, c->ssq_last, c->last_rows,
                                               f.n_last, c->d, c->Tcap, c->Tcap,
                                               static_cast<size_t>(c->Tcap) * c->d * (c->planes - 1),
                                               static_cast<size_t>(c->Tcap) * c->d * (c->planes - 1),
                                               ab, s))) !=
        cudaSuccess)
      return err;
    e.T = f.n_last;
    e.ssq_in = c->ssq_last;
    if ((err = gemm(c, s, false, EPI_ARGMAX, mt_v, c->V, c->d, f.n_last, c->xg_last, c->lm_head,
                    nullptr, nullptr, &c->mlm, nullptr, nullptr, e, "gemm_lmhead")) != cudaSuccess)
      return err;
    return cudaSuccess;
  }
  e.ssq_in = c->ssq;
  if ((err = gemm(c, s, pdl, EPI_ARGMAX, mt_v, c->V, c->d, T, c->xg, c->lm_head, nullptr, nullptr,
                  &c->mlm, nullptr, nullptr, e, "gemm_lmhead")) != cudaSuccess)
    return err;
  // (a8) accept / commit / refill
  return after_launch(c, s, "accept", launch_accept(f.acc, s, pdl));
}

AcceptArgs make_accept(cllm_ctx* c, int B, int n, bool decode) {
  AcceptArgs a{};
  a.B = B;
  a.n = n;
  a.V = c->V;
  a.decode = decode ? 1 : 0;
  a.max_new = c->dec_max_new;
  a.eos = c->dec_opts.eos_id;
  a.seed = c->dec_opts.seed;
  a.guess_mode = c->dec_opts.guess_init;
  a.pred = c->pred;
  a.block = c->block;
  a.L = c->Ld;
  a.head = c->head;
  a.committed = c->committed;
  a.iters = c->iters;
  a.done = c->done;
  a.out = c->out;
  a.accepted = c->accepted;
  a.prompts = c->prompts;
  a.plen = c->plen;
  a.prompt_ld = c->arch.max_seq;
  a.status = c->status;
  a.shrink = (decode && c->dec_opts.block_mode == CLLM_BLOCK_SHRINK) ? 1 : 0;
  a.width = c->width;
  if (decode && c->dec_opts.block_mode == CLLM_BLOCK_LOOKAHEAD) {
    a.pool = c->pool;
    a.pool_w = c->dec_opts.ngram - 1;
  }
  a.traj = (decode && c->traj_cap > 0) ? c->traj : nullptr;
  a.traj_cap = decode ? c->traj_cap : 0;
  if (decode && c->dec_opts.stats) {
    a.acc_hist = c->acc_hist;
    a.win_hist = c->win_hist;
    a.totals = c->st_totals;
    a.st_pos = c->st_pos;
    a.st_val = c->st_val;
    a.st_cand = c->st_cand;
    a.win_end = c->win_end;
    a.win_cnt = c->win_cnt;
  }
  return a;
}

// Read the device status (active, committed, error) after a synchronisation.
int check_device_error(cllm_ctx* c) {
  int e = 0;
  cudaError_t ce = cudaMemcpyAsync(&c->status_host[2], c->err, sizeof(int), cudaMemcpyDeviceToHost,
                                   c->stream);
  if (ce != cudaSuccess) return cuda_fail(ce, "status copy");
  ce = cudaStreamSynchronize(c->stream);
  if (ce != cudaSuccess) return cuda_fail(ce, "stream sync");
  e = c->status_host[2];
  if (e == 0) return CLLM_OK;
  cudaMemsetAsync(c->err, 0, sizeof(int), c->stream);
  cudaStreamSynchronize(c->stream);
  if (e & DERR_TIMEOUT) return CLLM_ETIMEOUT;
  if (e & DERR_CAPACITY) return CLLM_ECAPACITY;
  return CLLM_EDEVICE;
}

std::vector<int2> step_qtiles(int B, int n) {
  std::vector<int2> v;
  for (int b = 0; b < B; ++b)
    for (int r0 = 0; r0 < n; r0 += kQTile) v.push_back(make_int2(b, r0));
  return v;
}

int attn_grid_for(cllm_ctx* c, int n_qtiles) {
  const long items = static_cast<long>(n_qtiles) * c->H * c->nch_max;
  return static_cast<int>(std::max(1L, std::min(items, 2L * c->sms)));
}


// Tables of the persistent per-iteration kernel for B sequences x n rows:
// tensor maps [7 per layer: q k v o gate up down][LM head][xg, attn, h] and
// the phases [embed][per layer: QKV, attention, O, gate/up, down][LM head][accept].
int build_persistent(cllm_ctx* c, int mode, int B, int n, const int2* qtiles, int n_qtiles,
                     cllm_ctx::GraphEntry& ge, StepParams& prm, int& bn_max) {
  StepArgs& sa = prm.a;
  const int T = B * n;
  const int NL = c->NL;
  const int mapB = 7 * NL + 1;
  std::vector<CUtensorMap> maps(7 * NL + 7);
  for (int l = 0; l < NL; ++l) {
    const LayerW& L = c->layers[l];
    maps[7 * l + 0] = L.mq;
    maps[7 * l + 1] = L.mk;
    maps[7 * l + 2] = L.mv;
    maps[7 * l + 3] = L.mo;
    maps[7 * l + 4] = L.mgate;
    maps[7 * l + 5] = L.mup;
    maps[7 * l + 6] = L.mdown;
  }
  maps[7 * NL] = c->mlm;
  const uint32_t bn = static_cast<uint32_t>(round_up(T, 16));
  const uint64_t rows = 2 * static_cast<uint64_t>(c->Tcap);
  if (!make_map(&maps[mapB], c->xg, c->d, rows, bn) ||
      !make_map(&maps[mapB + 1], c->attn, c->dq, rows, bn) ||
      !make_map(&maps[mapB + 2], c->h, c->F, rows, bn))
    return CLLM_EINVAL;
  // attention tiles: K/V caches of all layers as rows of hd values, Q rows
  const int mapA = 7 * NL + 4;
  const uint64_t kv_rows = static_cast<uint64_t>(NL) * c->layer_kv_elems / c->hd;
  if (!make_map(&maps[mapA], c->kc, c->hd, kv_rows, kAttnChunk) ||
      !make_map(&maps[mapA + 1], c->vc, c->hd, kv_rows, kAttnChunk) ||
      !make_map(&maps[mapA + 2], c->q, c->dq, static_cast<uint64_t>(c->Tcap), kQTile))
    return CLLM_EINVAL;

  FwdSpec f{};
  f.mode = mode;
  f.T = T;
  f.B = B;
  f.n = n;
  f.qtiles = qtiles;
  f.n_qtiles = n_qtiles;
  // grid-barrier counter (16 words) then, per layer, the QKV tile flags and
  // the per-head attention counts; zeroed with the counter every launch
  const int Mqkv = c->dq + 2 * c->dkv;
  const int n_flags_layer = Mqkv / kBM + c->H;
  const size_t bar_bytes = 64 + sizeof(unsigned) * static_cast<size_t>(NL) * n_flags_layer;
  void* bar_d = nullptr;
  if (lib_malloc(&bar_d, bar_bytes) != cudaSuccess) return CLLM_ENOMEM;
  ge.bufs.push_back(bar_d);
  if (cudaMemset(bar_d, 0, bar_bytes) != cudaSuccess) return CLLM_ECUDA;
  ge.bar_bytes = bar_bytes;
  unsigned* flags = static_cast<unsigned*>(bar_d) + 16;
  std::vector<PhaseDesc> ph;
  auto gemm_phase = [&](int epi, int m0, int m1, int m2, int mb, int mtiles, int M, int K,
                        EpiArgs e) {
    PhaseDesc d{};
    d.kind = PH_GEMM;
    d.epi = epi;
    d.map_a0 = m0;
    d.map_a1 = m1;
    d.map_a2 = m2;
    d.map_b = mb;
    Part p;
    d.g = tc_gemm_args(c, mtiles, M, K, T, e, &p);
    d.e = e;
    // the persistent kernel also has a 16-column variant (4 KB activation tiles)
    bn_max = p.bn <= 16 ? 16 : p.bn_max;
    ph.push_back(d);
  };
  {
    PhaseDesc d{};
    d.kind = PH_EMBED;
    ph.push_back(d);
  }
  for (int l = 0; l < NL; ++l) {
    const LayerW& L = c->layers[l];
    const size_t kvoff = static_cast<size_t>(l) * c->layer_kv_elems * c->esz;
    void* kl = static_cast<char*>(c->kc) + kvoff;
    void* vl = static_cast<char*>(c->vc) + kvoff;
    EpiArgs e = base_epi(c, T);
    e.ssq_in = c->ssq;
    e.q_out = c->q;
    e.k_cache = kl;
    e.v_cache = vl;
    unsigned* qkv_done = flags + static_cast<size_t>(l) * n_flags_layer;
    unsigned* head_done = qkv_done + Mqkv / kBM;
    if (c->dataflow) e.tile_done = qkv_done;
    gemm_phase(EPI_QKV, 7 * l, 7 * l + 1, 7 * l + 2, mapB, Mqkv / kBM, Mqkv, c->d, e);
    const int qkv_ntiles = ph.back().g.ntiles;
    PhaseDesc at{};
    at.kind = PH_ATTN;
    at.k_cache = kl;
    at.v_cache = vl;
    at.kv_row0 = static_cast<int>(static_cast<size_t>(l) * c->layer_kv_elems / c->hd);
    if (c->dataflow) {
      at.no_barrier = 1;
      at.qkv_done = qkv_done;
      at.head_done = head_done;
      at.flag_target = qkv_ntiles;
    }
    ph.push_back(at);
    e = base_epi(c, T);
    e.x = c->x;
    e.xg = c->xg;
    e.gnext = L.mlp_norm;
    e.ssq_out = c->ssq;
    gemm_phase(EPI_RESID, 7 * l + 3, 7 * l + 3, 7 * l + 3, mapB + 1, c->d / kBM, c->d, c->dq, e);
    if (c->dataflow) {
      ph.back().no_barrier = 1;
      ph.back().head_done = head_done;
      ph.back().flag_target = n_qtiles;
    }
    e = base_epi(c, T);
    e.ssq_in = c->ssq;
    e.h_out = c->h;
    gemm_phase(EPI_GATEUP, 7 * l + 4, 7 * l + 5, 7 * l + 4, mapB, ceil_div(c->F, 64), c->F, c->d, e);
    e = base_epi(c, T);
    e.x = c->x;
    e.xg = c->xg;
    e.gnext = (l + 1 < NL) ? c->layers[l + 1].attn_norm : c->final_norm;
    e.ssq_out = c->ssq;
    gemm_phase(EPI_RESID, 7 * l + 6, 7 * l + 6, 7 * l + 6, mapB + 2, c->d / kBM, c->d, c->F, e);
  }
  {
    EpiArgs e = base_epi(c, T);
    e.am_part = c->am_part;
    e.am_ticket = c->am_ticket;
    e.pred = c->pred;
    e.gap = c->gap;
    // single steps asked for the logits (debug/parity) store them from the
    // same kernel that the decode loop runs
    e.logits = (mode == MODE_STEP && c->step_logits) ? c->logits_dbg : nullptr;
    e.ssq_in = c->ssq;
    gemm_phase(EPI_ARGMAX, 7 * NL, 7 * NL, 7 * NL, mapB, ceil_div(c->V, kBM), c->V, c->d, e);
    PhaseDesc d{};
    d.kind = PH_ACCEPT;
    ph.push_back(d);
  }
  ge.phase_kind.clear();
  ge.phase_names.clear();
  int resid_seen = 0;
  for (const PhaseDesc& d : ph) {
    ge.phase_kind.push_back(d.kind == PH_GEMM ? 10 + d.epi : d.kind);
    const char* nm = "accept";
    if (d.kind == PH_EMBED) nm = "embed";
    else if (d.kind == PH_ATTN) nm = "attention";
    else if (d.kind == PH_GEMM && d.epi == EPI_QKV) nm = "gemm_qkv";
    else if (d.kind == PH_GEMM && d.epi == EPI_GATEUP) nm = "gemm_gateup";
    else if (d.kind == PH_GEMM && d.epi == EPI_ARGMAX) nm = "gemm_lmhead";
    else if (d.kind == PH_GEMM && d.epi == EPI_RESID) nm = (resid_seen++ % 2 == 0) ? "gemm_o" : "gemm_down";
    ge.phase_names.push_back(nm);
  }
  // device copies
  auto upload = [&](const void* src, size_t bytes) -> void* {
    void* p = nullptr;
    if (lib_malloc(&p, bytes) != cudaSuccess) return nullptr;
    ge.bufs.push_back(p);
    if (src && cudaMemcpy(p, src, bytes, cudaMemcpyHostToDevice) != cudaSuccess) return nullptr;
    if (!src && cudaMemset(p, 0, bytes) != cudaSuccess) return nullptr;
    return p;
  };
  if (maps.size() > static_cast<size_t>(kMaxStepMaps)) return CLLM_EUNSUPPORTED;
  for (size_t i = 0; i < maps.size(); ++i) prm.maps[i] = maps[i];
  void* ph_d = upload(ph.data(), ph.size() * sizeof(PhaseDesc));
  void* tk_d = upload(nullptr, static_cast<size_t>(n_qtiles) * c->H * sizeof(int) + 16);
  void* st_d = upload(nullptr, (5 * ph.size() + 1) * sizeof(unsigned long long));
  void* cst_d = upload(nullptr, (kCtaStampSlots * ph.size() + kTraceCap) * c->sms *
                                    sizeof(unsigned long long));
  if (!ph_d || !tk_d || !st_d || !cst_d) return CLLM_ENOMEM;
  ge.cta_stamps = static_cast<unsigned long long*>(cst_d);
  if (c->profiling) {
    // epilogue stamps k = 3..5 of the per-CTA stamp array
    const long long PG = static_cast<long long>(ph.size()) * c->sms;
    for (size_t p = 0; p < ph.size(); ++p)
      if (ph[p].kind == PH_GEMM) {
        ph[p].e.dbg = ge.cta_stamps + 3 * PG + static_cast<long long>(p) * c->sms;
        ph[p].e.dbg_stride = PG;
      }
    if (cudaMemcpy(ph_d, ph.data(), ph.size() * sizeof(PhaseDesc), cudaMemcpyHostToDevice) !=
        cudaSuccess)
      return CLLM_ECUDA;
  }
  ge.n_phases = static_cast<int>(ph.size());
  ge.stamps = static_cast<unsigned long long*>(st_d);
  sa = StepArgs{};
  sa.phases = static_cast<const PhaseDesc*>(ph_d);
  sa.n_phases = ge.n_phases;
  sa.bar = static_cast<unsigned*>(bar_d);
  sa.embed = make_embed_args(c, f);
  sa.attn = make_attn_args(c, f);
  sa.attn_tickets = static_cast<int*>(tk_d);
  sa.accept = make_accept(c, B, n, mode == MODE_DECODE);
  sa.stamps = c->profiling ? ge.stamps : nullptr;
  sa.cta_stamps = c->profiling ? ge.cta_stamps : nullptr;
  sa.trace_phase = c->trace_phase;
  sa.hold_phase = c->hold_phase;
  sa.map_attn_k = mapA;
  sa.map_attn_v = mapA + 1;
  sa.map_attn_q = mapA + 2;
  sa.park_limit = c->park_slots;
  sa.l2_ahead = c->l2_pairs;
  sa.err = c->err;
  return CLLM_OK;
}

bool persistent_ok(cllm_ctx* c, int B, int n) {
  // (the attention's K/V tensor maps address cache rows with 32-bit coordinates)
  return c->bf16 && c->persistent && B * n <= 128 && 7 * c->NL + 7 <= kMaxStepMaps &&
         static_cast<uint64_t>(c->NL) * c->layer_kv_elems / c->hd + kAttnChunk < (1ull << 31) &&
         B * ceil_div(n, kQTile) <= kMaxQTilesStep && (c->hd == 64 || c->hd == 128);
}

// Get (capturing on first use) the graph of one decode/step iteration.
int get_graph(cllm_ctx* c, int mode, int n, cllm_ctx::GraphEntry** out) {
  const int B = c->B;
  auto key = std::make_tuple(mode, B, n, mode == MODE_DECODE ? c->dec_max_new : 0,
                             mode == MODE_DECODE ? c->dec_opts.eos_id : 0,
                             mode == MODE_DECODE ? static_cast<unsigned long long>(c->dec_opts.seed) : 0ull,
                             mode == MODE_DECODE ? (c->dec_opts.guess_init | (c->dec_opts.block_mode << 2) |
                                                    (c->traj_cap << 4))
                                                 : 0,
                             (c->profiling ? 1 : 0) | (mode == MODE_STEP && c->step_logits ? 2 : 0) |
                                 (mode == MODE_DECODE && c->dec_opts.stats ? 4 : 0) |
                                 (mode == MODE_DECODE ? (c->dec_opts.ngram << 3) : 0),
                             c->persistent ? 1 : 0,
                             (c->park_slots * 4096 + c->l2_pairs) * 2 + (c->dataflow ? 1 : 0));
  auto it = c->graphs.find(key);
  if (it != c->graphs.end()) {
    *out = &it->second;
    return CLLM_OK;
  }
  cllm_ctx::GraphEntry ge;
  std::vector<int2> qt = step_qtiles(B, n);
  if (lib_malloc(reinterpret_cast<void**>(&ge.qtiles), qt.size() * sizeof(int2)) != cudaSuccess)
    return CLLM_ENOMEM;
  if (cudaMemcpy(ge.qtiles, qt.data(), qt.size() * sizeof(int2), cudaMemcpyHostToDevice) !=
      cudaSuccess) {
    cudaFree(ge.qtiles);
    return CLLM_ECUDA;
  }
  if (persistent_ok(c, B, n)) {
    std::unique_ptr<StepParams> prm(new (std::nothrow) StepParams());
    if (!prm) return CLLM_ENOMEM;
    StepArgs& sa = prm->a;
    int bn_max = 32;
    int rc = build_persistent(c, mode, B, n, ge.qtiles, static_cast<int>(qt.size()), ge, *prm, bn_max);
    if (rc != CLLM_OK) {
      cudaFree(ge.qtiles);
      for (void* p : ge.bufs) cudaFree(p);
      return rc;
    }
    ge.persistent = true;
    const bool prof = c->profiling;
    if (prof) {
      while (c->prof_events.size() < 2) {
        cudaEvent_t ev;
        if (cudaEventCreate(&ev) != cudaSuccess) return CLLM_ECUDA;
        c->prof_events.push_back(ev);
      }
    }
    cudaGraph_t g = nullptr;
    cudaError_t e = cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal);
    if (e != cudaSuccess) return cuda_fail(e, "begin capture (persistent)");
    e = cudaMemsetAsync(sa.bar, 0, ge.bar_bytes, c->stream);
    if (e == cudaSuccess && prof) {
      // first-of slots start at all-ones (atomicMin), last-of slots at zero
      const size_t P = ge.n_phases;
      e = cudaMemsetAsync(ge.stamps + P + 1, 0xff, 2 * P * 8, c->stream);
      if (e == cudaSuccess) e = cudaMemsetAsync(ge.stamps + P + 1 + P, 0, P * 8, c->stream);
      if (e == cudaSuccess) e = cudaMemsetAsync(ge.stamps + P + 1 + 2 * P, 0xff, P * 8, c->stream);
      if (e == cudaSuccess) e = cudaMemsetAsync(ge.stamps + P + 1 + 3 * P, 0, P * 8, c->stream);
    }
    if (e == cudaSuccess && prof)
      e = cudaEventRecordWithFlags(c->prof_events[0], c->stream, cudaEventRecordExternal);
    if (e == cudaSuccess) {
      e = launch_step_persistent(*prm, bn_max, c->hd, c->sms, c->stream, false);
    }
    const cudaError_t first = e;
    if (e == cudaSuccess && prof)
      e = cudaEventRecordWithFlags(c->prof_events[1], c->stream, cudaEventRecordExternal);
    cudaError_t e2 = cudaStreamEndCapture(c->stream, &g);
    if (e != cudaSuccess || e2 != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      cudaFree(ge.qtiles);
      for (void* p : ge.bufs) cudaFree(p);
      return first != cudaSuccess ? cuda_fail(first, "capture of the persistent iteration")
                                  : cuda_fail(e2, "end capture (persistent)");
    }
    ge.launches = 1;
    {  // mark the kernel node cooperative where the driver supports it
      size_t nn = 0;
      if (cudaGraphGetNodes(g, nullptr, &nn) == cudaSuccess && nn > 0) {
        std::vector<cudaGraphNode_t> nodes(nn);
        if (cudaGraphGetNodes(g, nodes.data(), &nn) == cudaSuccess) {
          for (auto nd : nodes) {
            cudaGraphNodeType ty;
            if (cudaGraphNodeGetType(nd, &ty) == cudaSuccess && ty == cudaGraphNodeTypeKernel) {
              cudaLaunchAttributeValue v{};
              v.cooperative = 1;
              if (cudaGraphKernelNodeSetAttribute(nd, cudaLaunchAttributeCooperative, &v) !=
                  cudaSuccess)
                cudaGetLastError();
            }
          }
        }
      }
    }
    e = cudaGraphInstantiate(&ge.exec, g, 0);
    if (e != cudaSuccess) {
      // without the cooperative attribute (co-residency by construction)
      cudaGetLastError();
      size_t nn = 0;
      std::vector<cudaGraphNode_t> nodes;
      if (cudaGraphGetNodes(g, nullptr, &nn) == cudaSuccess) {
        nodes.resize(nn);
        cudaGraphGetNodes(g, nodes.data(), &nn);
        for (auto nd : nodes) {
          cudaGraphNodeType ty;
          if (cudaGraphNodeGetType(nd, &ty) == cudaSuccess && ty == cudaGraphNodeTypeKernel) {
            cudaLaunchAttributeValue v{};
            v.cooperative = 0;
            cudaGraphKernelNodeSetAttribute(nd, cudaLaunchAttributeCooperative, &v);
          }
        }
      }
      e = cudaGraphInstantiate(&ge.exec, g, 0);
    }
    cudaGraphDestroy(g);
    if (e != cudaSuccess) {
      cudaFree(ge.qtiles);
      for (void* p : ge.bufs) cudaFree(p);
      return cuda_fail(e, "instantiate (persistent)");
    }
    auto res = c->graphs.emplace(key, ge);
    *out = &res.first->second;
    return CLLM_OK;
  }
  FwdSpec f{};
  f.mode = mode;
  f.T = B * n;
  f.B = B;
  f.n = n;
  f.qtiles = ge.qtiles;
  f.n_qtiles = static_cast<int>(qt.size());
  f.attn_grid = attn_grid_for(c, f.n_qtiles);
  f.acc = make_accept(c, B, n, mode == MODE_DECODE);
  cudaGraph_t g = nullptr;
  std::vector<const char*> names;
  const bool prof = c->profiling;
  if (prof) {
    // events: [0] before the first kernel, [i] after kernel i
    const size_t need = 4 + static_cast<size_t>(c->NL) * 6 + 8;
    while (c->prof_events.size() < need) {
      cudaEvent_t ev;
      if (cudaEventCreate(&ev) != cudaSuccess) return CLLM_ECUDA;
      c->prof_events.push_back(ev);
    }
    c->rec_names = &names;
  }
  if (cudaStreamBeginCapture(c->stream, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    c->rec_names = nullptr;
    cudaFree(ge.qtiles);
    return CLLM_ECUDA;
  }
  c->rec_count = 0;
  cudaError_t e = cudaSuccess;
  if (prof) e = cudaEventRecordWithFlags(c->prof_events[0], c->stream, cudaEventRecordExternal);
  if (e == cudaSuccess) e = record_forward(c, c->stream, f, !prof);
  cudaError_t e2 = cudaStreamEndCapture(c->stream, &g);
  c->rec_names = nullptr;
  if (e != cudaSuccess || e2 != cudaSuccess) {
    if (g) cudaGraphDestroy(g);
    cudaFree(ge.qtiles);
    return CLLM_ECUDA;
  }
  ge.launches = c->rec_count;
  e = cudaGraphInstantiate(&ge.exec, g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) {
    cudaFree(ge.qtiles);
    return CLLM_ECUDA;
  }
  if (prof) c->prof_names.assign(names.begin(), names.end());
  auto res = c->graphs.emplace(key, ge);
  *out = &res.first->second;
  return CLLM_OK;
}

void accumulate_profile(cllm_ctx* c, const cllm_ctx::GraphEntry* ge) {
  if (ge && ge->persistent) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, c->prof_events[0], c->prof_events[1]) == cudaSuccess) {
      auto& a = c->prof_acc["step_persistent"];
      a.first += ms;
      a.second += 1;
    }
    std::vector<unsigned long long> st(5 * ge->n_phases + 1);
    if (cudaMemcpy(st.data(), ge->stamps, st.size() * 8, cudaMemcpyDeviceToHost) != cudaSuccess)
      return;
    c->last_stamps = st;
    c->last_phase_names = ge->phase_names;
    c->last_cta_stamps.resize((kCtaStampSlots * static_cast<size_t>(ge->n_phases) + kTraceCap) *
                              c->sms);
    cudaMemcpy(c->last_cta_stamps.data(), ge->cta_stamps, c->last_cta_stamps.size() * 8,
               cudaMemcpyDeviceToHost);
    // phase p runs from CTA 0 seeing its dependency met to the next phase's
    for (int p = 0; p < ge->n_phases; ++p) {
      if (st[p + 1] < st[p] || st[p] == 0) continue;
      auto& a = c->prof_acc["phase:" + ge->phase_names[p]];
      a.first += (st[p + 1] - st[p]) * 1e-6;
      a.second += 1;
    }
    return;
  }
  for (size_t i = 0; i < c->prof_names.size() && i + 1 < c->prof_events.size(); ++i) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, c->prof_events[i], c->prof_events[i + 1]) == cudaSuccess) {
      auto& a = c->prof_acc[c->prof_names[i]];
      a.first += ms;
      a.second += 1;
    }
  }
}

int read_status(cllm_ctx* c, int slot) {
  const int e = c->status_host[4 * slot + 2];
  if (e == 0) return CLLM_OK;
  cudaMemsetAsync(c->err, 0, sizeof(int), c->stream);
  cudaStreamSynchronize(c->stream);
  if (e & DERR_TIMEOUT) return CLLM_ETIMEOUT;
  if (e & DERR_CAPACITY) return CLLM_ECAPACITY;
  return CLLM_EDEVICE;
}

}  // namespace

// =====================================================================================
// C ABI
// =====================================================================================

extern "C" const char* cllm_last_cuda_error(void) { return g_last_cuda_error; }

extern "C" const char* cllm_status_string(int s) {
  switch (s) {
    case CLLM_OK: return "ok";
    case CLLM_EINVAL: return "invalid argument";
    case CLLM_ENOMEM: return "out of memory";
    case CLLM_ECUDA: return "CUDA error";
    case CLLM_ECAPACITY: return "KV-cache capacity exceeded";
    case CLLM_ETIMEOUT: return "bounded device wait timed out";
    case CLLM_EDEVICE: return "device-side check failed";
    case CLLM_ESTATE: return "call out of order";
    case CLLM_EUNSUPPORTED: return "unsupported shape or device";
    default: return "unknown status";
  }
}

extern "C" void cllm_destroy(cllm_ctx* c) {
  if (!c) return;
  cudaSetDevice(c->dev);
  if (c->stream) cudaStreamSynchronize(c->stream);
  for (auto& kv : c->graphs) {
    if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
    if (kv.second.qtiles) cudaFree(kv.second.qtiles);
    for (void* p : kv.second.bufs) cudaFree(p);
  }
  for (auto ev : c->prof_events) cudaEventDestroy(ev);
  for (void* p : c->allocs) cudaFree(p);
  if (c->status_host) cudaFreeHost(c->status_host);
  for (auto ev : c->iter_ev)
    if (ev) cudaEventDestroy(ev);
  if (c->own_stream && c->stream) cudaStreamDestroy(c->stream);
  delete c;
}

extern "C" int cllm_create(const cllm_arch* arch, const cllm_weights* w, void* cuda_stream,
                           cllm_ctx** out) {
  if (!arch || !w || !out) return CLLM_EINVAL;
  *out = nullptr;
  const cllm_arch& a = *arch;
  if (a.n_layers < 1 || a.d_model < 128 || a.n_heads < 1 || a.n_kv_heads < 1 || a.vocab < 2 ||
      a.ffn < 8 || a.max_batch < 1 || a.max_batch > 128 || a.max_seq < 2 || a.max_block < 1 ||
      !(a.rms_eps >= 0.f) || !(a.rope_theta > 0.f) || (a.dtype != CLLM_F32 && a.dtype != CLLM_BF16))
    return CLLM_EINVAL;
  if ((a.head_dim != 64 && a.head_dim != 128) || a.d_model % 128 ||
      (a.n_heads * a.head_dim) % 128 || (a.n_kv_heads * a.head_dim) % 128 ||
      a.n_heads % a.n_kv_heads || a.ffn % 8)
    return CLLM_EUNSUPPORTED;
  if (!w->tok_emb || !w->final_norm || !w->lm_head || !w->attn_norm || !w->wq || !w->wk || !w->wv ||
      !w->wo || !w->mlp_norm || !w->w_gate || !w->w_up || !w->w_down)
    return CLLM_EINVAL;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return CLLM_ECUDA;
  cudaDeviceProp prop;
  if (cudaGetDeviceProperties(&prop, dev) != cudaSuccess) return CLLM_ECUDA;
  if (prop.major != 10 || prop.minor != 3) return CLLM_EUNSUPPORTED;

  cllm_ctx* c = new (std::nothrow) cllm_ctx();
  if (!c) return CLLM_ENOMEM;
  c->arch = a;
  c->dev = dev;
  c->sms = prop.multiProcessorCount;
  c->bf16 = a.dtype == CLLM_BF16;
  c->esz = c->bf16 ? 2 : 4;
  c->planes = c->bf16 ? 2 : 1;
  c->d = a.d_model;
  c->H = a.n_heads;
  c->Hkv = a.n_kv_heads;
  c->hd = a.head_dim;
  c->dq = a.n_heads * a.head_dim;
  c->dkv = a.n_kv_heads * a.head_dim;
  c->F = a.ffn;
  c->V = a.vocab;
  c->NL = a.n_layers;
  c->tok_emb = w->tok_emb;
  c->final_norm = w->final_norm;
  c->lm_head = w->lm_head;
  c->layers.resize(a.n_layers);
  std::vector<const void*> all = {w->tok_emb, w->final_norm, w->lm_head};
  for (int l = 0; l < a.n_layers; ++l) {
    LayerW& L = c->layers[l];
    L.attn_norm = w->attn_norm[l];
    L.wq = w->wq[l];
    L.wk = w->wk[l];
    L.wv = w->wv[l];
    L.wo = w->wo[l];
    L.mlp_norm = w->mlp_norm[l];
    L.w_gate = w->w_gate[l];
    L.w_up = w->w_up[l];
    L.w_down = w->w_down[l];
    for (const void* p : {L.attn_norm, L.wq, L.wk, L.wv, L.wo, L.mlp_norm, L.w_gate, L.w_up, L.w_down})
      all.push_back(p);
  }
  for (const void* p : all)
    if (!p || !aligned16(p)) {
      delete c;
      return CLLM_EINVAL;
    }

  if (cuda_stream) {
    c->stream = static_cast<cudaStream_t>(cuda_stream);
  } else {
    if (cudaStreamCreateWithFlags(&c->stream, cudaStreamNonBlocking) != cudaSuccess) {
      delete c;
      return CLLM_ECUDA;
    }
    c->own_stream = true;
  }

  int rc = CLLM_OK;
  do {
    if (c->bf16) {
      if (!get_encode()) {
        rc = CLLM_ECUDA;
        break;
      }
      bool ok = make_map(&c->mlm, c->lm_head, c->d, c->V, kBM);
      for (int l = 0; l < a.n_layers && ok; ++l) {
        LayerW& L = c->layers[l];
        ok = make_map(&L.mq, L.wq, c->d, c->dq, kBM) && make_map(&L.mk, L.wk, c->d, c->dkv, kBM) &&
             make_map(&L.mv, L.wv, c->d, c->dkv, kBM) && make_map(&L.mo, L.wo, c->dq, c->d, kBM) &&
             make_map(&L.mgate, L.w_gate, c->d, c->F, 64) && make_map(&L.mup, L.w_up, c->d, c->F, 64) &&
             make_map(&L.mdown, L.w_down, c->F, c->d, kBM);
      }
      if (!ok) {
        rc = CLLM_EINVAL;
        break;
      }
      if (gemm_tc_set_attributes() != cudaSuccess || attention_set_attributes() != cudaSuccess ||
          step_persistent_set_attributes() != cudaSuccess) {
        rc = CLLM_ECUDA;
        break;
      }
    }
    // capacities
    const int step_rows = a.max_batch * a.max_block;
    c->prefill_cap = std::min(2048, round_up(std::max(a.max_batch * a.max_seq, 16), 16));
    c->Tcap = round_up(std::max(step_rows, c->prefill_cap), 16);
    c->nch_max = ceil_div(a.max_seq, kAttnChunk);
    c->max_qtiles = c->Tcap / kQTile + a.max_batch;
    const size_t T = c->Tcap;
    const size_t es = c->esz;
    const size_t P = c->planes;
    const int dmax = std::max(c->dq, std::max(c->d, c->F));
    (void)dmax;
    bool ok = dev_alloc(c, &c->x, T * c->d * 4) && dev_alloc(c, &c->xg, P * T * c->d * es) &&
              dev_alloc(c, &c->ssq, (c->d / kBM) * T * 4) && dev_alloc(c, &c->q, T * c->dq * es) &&
              dev_alloc(c, &c->attn, P * T * c->dq * es) && dev_alloc(c, &c->h, P * T * c->F * es) &&
              dev_alloc(c, &c->xg_last, P * T * c->d * es) &&
              dev_alloc(c, &c->ssq_last, (c->d / kBM) * T * 4) &&
              dev_alloc(c, &c->last_rows, a.max_batch * 4);
    if (!ok) {
      rc = CLLM_ENOMEM;
      break;
    }
    c->layer_kv_elems = static_cast<size_t>(a.max_batch) * c->Hkv * a.max_seq * c->hd;
    ok = dev_alloc(c, &c->kc, c->layer_kv_elems * a.n_layers * es) &&
         dev_alloc(c, &c->vc, c->layer_kv_elems * a.n_layers * es);
    if (!ok) {
      rc = CLLM_ENOMEM;
      break;
    }
    // tensor maps of the per-GEMM attention's TMA tiles (the cache rows of
    // all layers must be addressable with 32-bit coordinates)
    if (c->bf16 && (c->hd == 64 || c->hd == 128)) {
      const uint64_t kv_rows = static_cast<uint64_t>(a.n_layers) * c->layer_kv_elems / c->hd;
      c->attn_maps_ok = kv_rows + kAttnChunk < (1ull << 31) &&
                        make_map(&c->attn_maps.k, c->kc, c->hd, kv_rows, kAttnChunk) &&
                        make_map(&c->attn_maps.v, c->vc, c->hd, kv_rows, kAttnChunk) &&
                        make_map(&c->attn_maps.q, c->q, c->dq, static_cast<uint64_t>(c->Tcap), kQTile);
    }
    // RoPE table (cos, sin) of pos * theta^(-2i/hd), evaluated in double
    {
      const int half = c->hd / 2;
      std::vector<float2> tab(static_cast<size_t>(a.max_seq) * half);
      for (int p = 0; p < a.max_seq; ++p)
        for (int i = 0; i < half; ++i) {
          const double ang =
              static_cast<double>(p) * std::pow(static_cast<double>(a.rope_theta), -2.0 * i / c->hd);
          tab[static_cast<size_t>(p) * half + i] =
              make_float2(static_cast<float>(std::cos(ang)), static_cast<float>(std::sin(ang)));
        }
      if (!dev_alloc(c, &c->rope, tab.size() * sizeof(float2)) ||
          cudaMemcpy(c->rope, tab.data(), tab.size() * sizeof(float2), cudaMemcpyHostToDevice) !=
              cudaSuccess) {
        rc = CLLM_ENOMEM;
        break;
      }
    }
    // attention partials: rows x heads x chunks
    const size_t prow = T * c->H * c->nch_max;
    ok = dev_alloc(c, &c->part_o, prow * c->hd * 4) && dev_alloc(c, &c->part_ml, prow * 8);
    // GEMM split-K partials (T <= 256 launches)
    const int mt_list[5] = {(c->dq + 2 * c->dkv) / kBM, c->d / kBM, ceil_div(c->F, 64), c->d / kBM,
                            ceil_div(c->V, kBM)};
    const int k_list[5] = {c->d, c->dq, c->d, c->F, c->d};
    const int bn_split = std::min(256, round_up(std::max(step_rows, c->prefill_cap), 16));
    size_t need = 0;
    c->max_mtiles = 0;
    for (int i = 0; i < 5; ++i) {
      const Part p = plan_gemm(mt_list[i], k_list[i], std::min(256, bn_split), c->sms);
      need = std::max(need, static_cast<size_t>(mt_list[i]) * p.maxc * p.bn * kBM);
      c->max_mtiles = std::max(c->max_mtiles, mt_list[i]);
    }
    c->gemm_part_elems = need;
    ok = ok && dev_alloc(c, &c->gemm_part, need * 4) && dev_alloc(c, &c->tickets, c->max_mtiles * 4) &&
         dev_alloc(c, &c->am_part, static_cast<size_t>(ceil_div(c->V, kBM)) * T * 12) &&
         dev_alloc(c, &c->am_ticket, 16) && dev_alloc(c, &c->pred, T * 4) &&
         dev_alloc(c, &c->gap, T * 4);
    ok = ok && dev_alloc(c, &c->tok_in, T * 4) && dev_alloc(c, &c->pos_in, T * 4) &&
         dev_alloc(c, &c->bidx_in, T * 4) && dev_alloc(c, &c->pos, T * 4) &&
         dev_alloc(c, &c->bidx, T * 4) && dev_alloc(c, &c->seq_start, a.max_batch * 4) &&
         dev_alloc(c, &c->seq_row0, a.max_batch * 4) && dev_alloc(c, &c->seq_nrows, a.max_batch * 4) &&
         dev_alloc(c, &c->qtiles_prefill, c->max_qtiles * sizeof(int2));
    const size_t Bm = a.max_batch;
    ok = ok && dev_alloc(c, &c->Ld, Bm * 4) && dev_alloc(c, &c->head, Bm * 4) &&
         dev_alloc(c, &c->head0, Bm * 4) && dev_alloc(c, &c->block, Bm * a.max_block * 4) &&
         dev_alloc(c, &c->committed, Bm * 4) && dev_alloc(c, &c->iters, Bm * 4) &&
         dev_alloc(c, &c->done, Bm * 4) && dev_alloc(c, &c->accepted, Bm * 4) &&
         dev_alloc(c, &c->width, Bm * 4) &&
         dev_alloc(c, &c->acc_hist, (a.max_block + 1) * 8) &&
         dev_alloc(c, &c->win_hist, (a.max_block + 1) * 8) && dev_alloc(c, &c->st_totals, 16) &&
         dev_alloc(c, &c->st_pos, Bm * a.max_block * 4) &&
         dev_alloc(c, &c->st_val, Bm * a.max_block * 4) &&
         dev_alloc(c, &c->st_cand, Bm * a.max_block * 4) && dev_alloc(c, &c->win_end, Bm * 4) &&
         dev_alloc(c, &c->win_cnt, Bm * 4) &&
         dev_alloc(c, &c->prompts, Bm * a.max_seq * 4) && dev_alloc(c, &c->plen, Bm * 4) &&
         dev_alloc(c, &c->status, 16) && dev_alloc(c, &c->err, 16);
    if (!ok) {
      rc = CLLM_ENOMEM;
      break;
    }
    if (alloc_injected_failure() || cudaMallocHost(&c->status_host, 32) != cudaSuccess) {
      rc = CLLM_ENOMEM;
      break;
    }
    std::memset(c->status_host, 0, 32);
    if (cudaEventCreateWithFlags(&c->iter_ev[0], cudaEventDisableTiming) != cudaSuccess ||
        cudaEventCreateWithFlags(&c->iter_ev[1], cudaEventDisableTiming) != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    if (cudaDeviceSynchronize() != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
  } while (0);
  if (rc != CLLM_OK) {
    cllm_destroy(c);
    return rc;
  }
  *out = c;
  return CLLM_OK;
}

extern "C" int cllm_prefill(cllm_ctx* c, int B, const int32_t* tokens, const int32_t* lens,
                            int32_t* head_out) {
  if (!c || !tokens || !lens) return CLLM_EINVAL;
  if (B < 1 || B > c->arch.max_batch) return CLLM_EINVAL;
  long total = 0;
  for (int b = 0; b < B; ++b) {
    if (lens[b] < 1) return CLLM_EINVAL;
    if (lens[b] > c->arch.max_seq) return CLLM_ECAPACITY;
    total += lens[b];
  }
  for (long i = 0; i < total; ++i)
    if (tokens[i] < 0 || tokens[i] >= c->V) return CLLM_EINVAL;
  cudaSetDevice(c->dev);
  c->prefilled = false;
  c->dec_active = false;
  c->B = B;
  c->lens.assign(lens, lens + B);
  // prompts (guesses drawn from the prompt) and lengths
  std::vector<int> pbuf(static_cast<size_t>(B) * c->arch.max_seq, 0);
  std::vector<long> off(B + 1, 0);
  for (int b = 0; b < B; ++b) {
    off[b + 1] = off[b] + lens[b];
    std::memcpy(&pbuf[static_cast<size_t>(b) * c->arch.max_seq], tokens + off[b], lens[b] * 4);
  }
  if (cudaMemcpyAsync(c->prompts, pbuf.data(), pbuf.size() * 4, cudaMemcpyHostToDevice, c->stream) !=
          cudaSuccess ||
      cudaMemcpyAsync(c->plen, lens, B * 4, cudaMemcpyHostToDevice, c->stream) != cudaSuccess)
    return CLLM_ECUDA;

  std::vector<int> heads(B, 0);
  // rounds of at most prefill_cap rows; a prompt may span several rounds
  std::vector<int> done_rows(B, 0);
  int cur = 0;
  while (cur < B) {
    std::vector<int> tok, pos, bidx, start(B, 0), row0(B, 0), nrows(B, 0), lastb;
    std::vector<int2> qt;
    std::vector<int> last_rows;
    int used = 0;
    for (int b = cur; b < B && used < c->prefill_cap; ++b) {
      const int remain = lens[b] - done_rows[b];
      const int take = std::min(remain, c->prefill_cap - used);
      if (take <= 0) continue;
      start[b] = done_rows[b];
      row0[b] = used;
      nrows[b] = take;
      for (int i = 0; i < take; ++i) {
        tok.push_back(tokens[off[b] + done_rows[b] + i]);
        pos.push_back(done_rows[b] + i);
        bidx.push_back(b);
      }
      for (int r0 = 0; r0 < take; r0 += kQTile) qt.push_back(make_int2(b, r0));
      done_rows[b] += take;
      used += take;
      if (done_rows[b] == lens[b]) {
        last_rows.push_back(used - 1);
        lastb.push_back(b);
      }
    }
    const int T = used;
    if (cudaMemcpyAsync(c->tok_in, tok.data(), T * 4, cudaMemcpyHostToDevice, c->stream) ||
        cudaMemcpyAsync(c->pos_in, pos.data(), T * 4, cudaMemcpyHostToDevice, c->stream) ||
        cudaMemcpyAsync(c->bidx_in, bidx.data(), T * 4, cudaMemcpyHostToDevice, c->stream) ||
        cudaMemcpyAsync(c->seq_start, start.data(), B * 4, cudaMemcpyHostToDevice, c->stream) ||
        cudaMemcpyAsync(c->seq_row0, row0.data(), B * 4, cudaMemcpyHostToDevice, c->stream) ||
        cudaMemcpyAsync(c->seq_nrows, nrows.data(), B * 4, cudaMemcpyHostToDevice, c->stream) ||
        cudaMemcpyAsync(c->qtiles_prefill, qt.data(), qt.size() * sizeof(int2),
                        cudaMemcpyHostToDevice, c->stream))
      return CLLM_ECUDA;
    if (!last_rows.empty() &&
        cudaMemcpyAsync(c->last_rows, last_rows.data(), last_rows.size() * 4,
                        cudaMemcpyHostToDevice, c->stream))
      return CLLM_ECUDA;
    FwdSpec f{};
    f.mode = MODE_PREFILL;
    f.T = T;
    f.B = B;
    f.qtiles = c->qtiles_prefill;
    f.n_qtiles = static_cast<int>(qt.size());
    long items = 0;
    for (auto& q : qt) {
      const int nr = std::min(kQTile, nrows[q.x] - q.y);
      items += static_cast<long>(c->H) * ((start[q.x] + q.y + nr - 1) / kAttnChunk + 1);
    }
    f.attn_grid = static_cast<int>(std::max(1L, std::min(items, 4L * c->sms)));
    f.n_last = static_cast<int>(last_rows.size());
    if (f.n_last == 0) {
      // no prompt ends in this round: skip the LM head by running the layers
      // only (the LM head call is harmless with zero rows, so run it on row 0)
      f.n_last = 1;
      int zero = 0;
      if (cudaMemcpyAsync(c->last_rows, &zero, 4, cudaMemcpyHostToDevice, c->stream))
        return CLLM_ECUDA;
    }
    c->rec_names = nullptr;
    if (record_forward(c, c->stream, f, false) != cudaSuccess) return CLLM_ECUDA;
    std::vector<int> pr(f.n_last);
    if (cudaMemcpyAsync(pr.data(), c->pred, f.n_last * 4, cudaMemcpyDeviceToHost, c->stream))
      return CLLM_ECUDA;
    int rc = check_device_error(c);  // synchronises
    if (rc != CLLM_OK) return rc;
    for (size_t i = 0; i < lastb.size(); ++i) heads[lastb[i]] = pr[i];
    while (cur < B && done_rows[cur] == lens[cur]) ++cur;
  }
  if (cudaMemcpyAsync(c->head0, heads.data(), B * 4, cudaMemcpyHostToDevice, c->stream) ||
      cudaMemcpyAsync(c->head, heads.data(), B * 4, cudaMemcpyHostToDevice, c->stream) ||
      cudaMemcpyAsync(c->Ld, lens, B * 4, cudaMemcpyHostToDevice, c->stream))
    return CLLM_ECUDA;
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return CLLM_ECUDA;
  c->Lh.assign(lens, lens + B);
  c->prefilled = true;
  if (head_out) std::memcpy(head_out, heads.data(), B * 4);
  return CLLM_OK;
}

extern "C" int cllm_jacobi_step(cllm_ctx* c, const int32_t* guess, int n, int32_t* next_out,
                                int32_t* accepted_out, float* gap_out, float* logits_out) {
  if (!c || !guess || !next_out || !accepted_out) return CLLM_EINVAL;
  if (!c->prefilled) return CLLM_ESTATE;
  if (n < 1 || n > c->arch.max_block) return CLLM_EINVAL;
  const int B = c->B;
  for (long i = 0; i < static_cast<long>(B) * n; ++i)
    if (guess[i] < 0 || guess[i] >= c->V) return CLLM_EINVAL;
  for (int b = 0; b < B; ++b)
    if (c->Lh[b] + n > c->arch.max_seq) return CLLM_ECAPACITY;
  cudaSetDevice(c->dev);
  c->dec_active = false;
  if (logits_out && !c->logits_dbg) {
    if (!dev_alloc(c, &c->logits_dbg, static_cast<size_t>(c->Tcap) * c->V * 4)) return CLLM_ENOMEM;
  }
  if (cudaMemcpyAsync(c->block, guess, static_cast<size_t>(B) * n * 4, cudaMemcpyHostToDevice,
                      c->stream) != cudaSuccess)
    return CLLM_ECUDA;
  if (launch_set_head(c->block, c->head, B, n, c->V, c->err, c->stream) != cudaSuccess)
    return CLLM_ECUDA;
  if (logits_out && !persistent_ok(c, B, n)) {
    std::vector<int2> qt = step_qtiles(B, n);
    if (cudaMemcpyAsync(c->qtiles_prefill, qt.data(), qt.size() * sizeof(int2),
                        cudaMemcpyHostToDevice, c->stream) != cudaSuccess)
      return CLLM_ECUDA;
    FwdSpec f{};
    f.mode = MODE_STEP;
    f.T = B * n;
    f.B = B;
    f.n = n;
    f.qtiles = c->qtiles_prefill;
    f.n_qtiles = static_cast<int>(qt.size());
    f.attn_grid = attn_grid_for(c, f.n_qtiles);
    f.want_logits = true;
    f.acc = make_accept(c, B, n, false);
    if (record_forward(c, c->stream, f, false) != cudaSuccess) return CLLM_ECUDA;
  } else {
    // the persistent kernel of the decode loop; with logits_out its LM-head
    // phase also stores the logits
    cllm_ctx::GraphEntry* ge = nullptr;
    const bool prof = c->profiling;
    c->profiling = false;
    c->step_logits = logits_out != nullptr;
    int rc = get_graph(c, MODE_STEP, n, &ge);
    c->profiling = prof;
    c->step_logits = false;
    if (rc != CLLM_OK) return rc;
    cudaError_t e = cudaGraphLaunch(ge->exec, c->stream);
    if (e != cudaSuccess) return cuda_fail(e, "graph launch (step)");
  }
  std::vector<int> acc(B);
  if (cudaMemcpyAsync(next_out, c->pred, static_cast<size_t>(B) * n * 4, cudaMemcpyDeviceToHost,
                      c->stream) ||
      cudaMemcpyAsync(acc.data(), c->accepted, B * 4, cudaMemcpyDeviceToHost, c->stream))
    return CLLM_ECUDA;
  if (gap_out && cudaMemcpyAsync(gap_out, c->gap, static_cast<size_t>(B) * n * 4,
                                 cudaMemcpyDeviceToHost, c->stream))
    return CLLM_ECUDA;
  if (logits_out && cudaMemcpyAsync(logits_out, c->logits_dbg, static_cast<size_t>(B) * n * c->V * 4,
                                    cudaMemcpyDeviceToHost, c->stream))
    return CLLM_ECUDA;
  int rc = check_device_error(c);
  if (rc != CLLM_OK) return rc;
  for (int b = 0; b < B; ++b) {
    accepted_out[b] = acc[b];
    c->Lh[b] += acc[b];
  }
  return CLLM_OK;
}

extern "C" int cllm_decode_begin(cllm_ctx* c, int n, int max_new, const cllm_decode_opts* opts) {
  if (!c) return CLLM_EINVAL;
  if (!c->prefilled) return CLLM_ESTATE;
  if (n < 1 || n > c->arch.max_block || max_new < 1 || max_new >= (1 << 24)) return CLLM_EINVAL;
  cllm_decode_opts o{};
  o.seed = 0;
  o.eos_id = -1;
  o.guess_init = CLLM_GUESS_UNIFORM;
  o.block_mode = CLLM_BLOCK_REFILL;
  if (opts) o = *opts;
  if (o.guess_init != CLLM_GUESS_UNIFORM && o.guess_init != CLLM_GUESS_FROM_PROMPT) return CLLM_EINVAL;
  if (o.block_mode != CLLM_BLOCK_REFILL && o.block_mode != CLLM_BLOCK_SHRINK &&
      o.block_mode != CLLM_BLOCK_LOOKAHEAD)
    return CLLM_EINVAL;
  if (o.block_mode == CLLM_BLOCK_LOOKAHEAD && (o.ngram < 2 || o.ngram > 16)) return CLLM_EINVAL;
  if (o.block_mode != CLLM_BLOCK_LOOKAHEAD) o.ngram = 0;
  if (o.record_cap < 0 || o.record_cap > (1 << 20)) return CLLM_EINVAL;
  if (o.stats != 0 && o.stats != 1) return CLLM_EINVAL;
  if (o.eos_id >= c->V) return CLLM_EINVAL;
  for (int b = 0; b < c->B; ++b)
    if (static_cast<long>(c->lens[b]) + max_new + n > c->arch.max_seq) return CLLM_ECAPACITY;
  cudaSetDevice(c->dev);
  const size_t need = static_cast<size_t>(c->B) * max_new;
  const size_t traj_need = static_cast<size_t>(o.record_cap) * c->B * n;
  bool stale = false;
  if (traj_need > c->traj_alloc) {
    int* p = nullptr;
    if (!dev_alloc(c, &p, traj_need * 4)) return CLLM_ENOMEM;
    c->traj = p;
    c->traj_alloc = traj_need;
    stale = true;
  }
  if (need > c->out_cap) {
    int* p = nullptr;
    if (!dev_alloc(c, &p, need * 4)) return CLLM_ENOMEM;
    c->out = p;
    c->out_cap = need;
    stale = true;
  }
  const size_t pool_need = o.ngram > 0 ? static_cast<size_t>(c->B) * c->V * (o.ngram - 1) : 0;
  if (pool_need > c->pool_alloc) {
    int* p = nullptr;
    if (!dev_alloc(c, &p, pool_need * 4)) return CLLM_ENOMEM;
    c->pool = p;
    c->pool_alloc = pool_need;
    stale = true;
  }
  if (stale) {
    // graphs captured against the old output buffer are stale
    for (auto& kv : c->graphs) {
      if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
      if (kv.second.qtiles) cudaFree(kv.second.qtiles);
      for (void* p : kv.second.bufs) cudaFree(p);
    }
    c->graphs.clear();
  }
  c->dec_n = n;
  c->dec_max_new = max_new;
  c->dec_opts = o;
  c->traj_cap = o.record_cap;
  if (traj_need > 0 && cudaMemsetAsync(c->traj, 0xff, traj_need * 4, c->stream) != cudaSuccess)
    return CLLM_ECUDA;
  // an empty pool: every entry -1
  if (pool_need > 0 && cudaMemsetAsync(c->pool, 0xff, pool_need * 4, c->stream) != cudaSuccess)
    return CLLM_ECUDA;
  if (cudaMemcpyAsync(c->head, c->head0, c->B * 4, cudaMemcpyDeviceToDevice, c->stream) !=
      cudaSuccess)
    return CLLM_ECUDA;
  AcceptArgs a = make_accept(c, c->B, n, true);
  if (launch_decode_init(a, c->stream) != cudaSuccess) return CLLM_ECUDA;
  c->dec_active = true;
  c->Lh = c->lens;
  return CLLM_OK;
}

extern "C" int cllm_decode_run(cllm_ctx* c, int max_iters, int* iters_run, int64_t* committed) {
  if (!c || max_iters < 0) return CLLM_EINVAL;
  if (!c->dec_active) return CLLM_ESTATE;
  cudaSetDevice(c->dev);
  cllm_ctx::GraphEntry* ge = nullptr;
  int rc = get_graph(c, MODE_DECODE, c->dec_n, &ge);
  if (rc != CLLM_OK) return rc;
  // Iteration j+1 is queued before iteration j's 12-byte status is read, so
  // the device never waits for the host; once no sequence is active the
  // queued iteration commits nothing.  (Profiling reads per-iteration timing
  // and runs one iteration at a time.)
  auto issue = [&](int j) -> cudaError_t {
    const int slot = j & 1;
    cudaError_t e = cudaGraphLaunch(ge->exec, c->stream);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(&c->status_host[4 * slot], c->status, 2 * sizeof(int),
                          cudaMemcpyDeviceToHost, c->stream);
    if (e == cudaSuccess)
      e = cudaMemcpyAsync(&c->status_host[4 * slot + 2], c->err, sizeof(int),
                          cudaMemcpyDeviceToHost, c->stream);
    if (e == cudaSuccess) e = cudaEventRecord(c->iter_ev[slot], c->stream);
    return e;
  };
  const bool pipelined = !c->profiling;
  int it = 0;
  int64_t com = 0;
  int queued = 0;  // iterations issued
  cudaError_t e = cudaSuccess;
  if (max_iters > 0) {
    e = issue(0);
    if (e != cudaSuccess) return cuda_fail(e, "graph launch");
    queued = 1;
  }
  while (it < max_iters) {
    if (pipelined && queued < max_iters && queued == it + 1) {
      e = issue(queued);
      if (e != cudaSuccess) return cuda_fail(e, "graph launch");
      ++queued;
    }
    e = cudaEventSynchronize(c->iter_ev[it & 1]);
    if (e != cudaSuccess) return cuda_fail(e, "iteration sync");
    if (c->profiling) accumulate_profile(c, ge);
    const int slot = it & 1;
    ++it;
    rc = read_status(c, slot);
    if (rc != CLLM_OK) {
      cudaStreamSynchronize(c->stream);
      return rc;
    }
    com += c->status_host[4 * slot + 1];
    if (c->status_host[4 * slot] == 0) break;
    if (!pipelined && it < max_iters) {
      e = issue(it);
      if (e != cudaSuccess) return cuda_fail(e, "graph launch");
      ++queued;
    }
  }
  // a queued iteration past the end committed nothing; let it finish
  e = cudaStreamSynchronize(c->stream);
  if (e != cudaSuccess) return cuda_fail(e, "stream sync");
  if (iters_run) *iters_run = it;
  if (committed) *committed = com;
  return CLLM_OK;
}

extern "C" int cllm_decode_read(cllm_ctx* c, int32_t* tokens_out, int32_t* iters_out) {
  if (!c) return CLLM_EINVAL;
  if (!c->dec_active) return CLLM_ESTATE;
  cudaSetDevice(c->dev);
  if (tokens_out && cudaMemcpyAsync(tokens_out, c->out, static_cast<size_t>(c->B) * c->dec_max_new * 4,
                                    cudaMemcpyDeviceToHost, c->stream))
    return CLLM_ECUDA;
  if (iters_out &&
      cudaMemcpyAsync(iters_out, c->iters, c->B * 4, cudaMemcpyDeviceToHost, c->stream))
    return CLLM_ECUDA;
  return check_device_error(c);
}

extern "C" int cllm_decode_read_trajectory(cllm_ctx* c, int32_t* blocks_out) {
  if (!c || !blocks_out) return CLLM_EINVAL;
  if (!c->dec_active || c->traj_cap <= 0) return CLLM_ESTATE;
  cudaSetDevice(c->dev);
  const size_t bytes = static_cast<size_t>(c->traj_cap) * c->B * c->dec_n * 4;
  if (cudaMemcpyAsync(blocks_out, c->traj, bytes, cudaMemcpyDeviceToHost, c->stream) != cudaSuccess)
    return cuda_fail(cudaGetLastError(), "trajectory copy");
  return check_device_error(c);
}

extern "C" int cllm_decode_read_stats(cllm_ctx* c, cllm_accept_stats* out, int64_t* acc_hist,
                                     int64_t* win_hist) {
  if (!c || !out) return CLLM_EINVAL;
  if (!c->dec_active || !c->dec_opts.stats) return CLLM_ESTATE;
  cudaSetDevice(c->dev);
  const int n = c->dec_n, B = c->B;
  std::vector<unsigned long long> ah(n + 1), wh(n + 1), tot(2);
  std::vector<int> wend(B), wcnt(B);
  if (cudaMemcpyAsync(ah.data(), c->acc_hist, (n + 1) * 8, cudaMemcpyDeviceToHost, c->stream) ||
      cudaMemcpyAsync(wh.data(), c->win_hist, (n + 1) * 8, cudaMemcpyDeviceToHost, c->stream) ||
      cudaMemcpyAsync(tot.data(), c->st_totals, 16, cudaMemcpyDeviceToHost, c->stream) ||
      cudaMemcpyAsync(wend.data(), c->win_end, B * 4, cudaMemcpyDeviceToHost, c->stream) ||
      cudaMemcpyAsync(wcnt.data(), c->win_cnt, B * 4, cudaMemcpyDeviceToHost, c->stream))
    return cuda_fail(cudaGetLastError(), "statistics copy");
  const int rc = check_device_error(c);  // synchronises
  if (rc != CLLM_OK) return rc;
  // windows still open count with their stationary tokens so far
  for (int b = 0; b < B; ++b)
    if (wend[b] > 0) wh[std::min(wcnt[b], n)] += 1;
  cllm_accept_stats st{};
  for (int a = 0; a <= n; ++a) {
    st.iterations += static_cast<int64_t>(ah[a]);
    st.accepted += static_cast<int64_t>(ah[a]) * a;
  }
  st.windows = static_cast<int64_t>(tot[0]);
  st.stationary = static_cast<int64_t>(tot[1]);
  *out = st;
  for (int a = 0; a <= n; ++a) {
    if (acc_hist) acc_hist[a] = static_cast<int64_t>(ah[a]);
    if (win_hist) win_hist[a] = static_cast<int64_t>(wh[a]);
  }
  return CLLM_OK;
}

extern "C" int cllm_jacobi_decode(cllm_ctx* c, int B, const int32_t* tokens, const int32_t* lens,
                                  int n, int max_new, const cllm_decode_opts* opts,
                                  int32_t* tokens_out, int32_t* iters_out) {
  if (!c || !tokens || !lens || !tokens_out) return CLLM_EINVAL;
  if (n < 1 || n > c->arch.max_block || max_new < 1) return CLLM_EINVAL;
  if (B < 1 || B > c->arch.max_batch) return CLLM_EINVAL;
  for (int b = 0; b < B; ++b)
    if (lens[b] >= 1 && static_cast<long>(lens[b]) + max_new + n > c->arch.max_seq)
      return CLLM_ECAPACITY;
  int rc = cllm_prefill(c, B, tokens, lens, nullptr);
  if (rc != CLLM_OK) return rc;
  rc = cllm_decode_begin(c, n, max_new, opts);
  if (rc != CLLM_OK) return rc;
  // every iteration commits >= 1 token per active sequence
  rc = cllm_decode_run(c, max_new + 1, nullptr, nullptr);
  if (rc != CLLM_OK) return rc;
  return cllm_decode_read(c, tokens_out, iters_out);
}

extern "C" int cllm_ar_decode(cllm_ctx* c, int B, const int32_t* tokens, const int32_t* lens,
                              int max_new, int eos_id, int32_t* tokens_out) {
  cllm_decode_opts o{};
  o.seed = 0;
  o.eos_id = eos_id;
  o.guess_init = CLLM_GUESS_UNIFORM;
  o.block_mode = CLLM_BLOCK_REFILL;
  return cllm_jacobi_decode(c, B, tokens, lens, 1, max_new, &o, tokens_out, nullptr);
}

extern "C" int cllm_set_option(cllm_ctx* c, int option, int value) {
  if (!c) return CLLM_EINVAL;
  if (option == CLLM_OPT_PERSISTENT) {
    c->persistent = value != 0;
    return CLLM_OK;
  }
  if (option == CLLM_OPT_L2_PAIRS) {
    if (value < 0 || value > 64) return CLLM_EINVAL;
    c->l2_pairs = value;
    return CLLM_OK;
  }
  if (option == CLLM_OPT_PARK_SLOTS) {
    if (value < -1 || value > 64) return CLLM_EINVAL;
    c->park_slots = value;
    return CLLM_OK;
  }
  if (option == CLLM_OPT_DATAFLOW) {
    c->dataflow = value != 0;
    return CLLM_OK;
  }
  return CLLM_EINVAL;
}

extern "C" int cllm_uses_persistent(cllm_ctx* c, int n) {
  if (!c || !c->prefilled) return CLLM_EINVAL;
  return persistent_ok(c, c->B, n) ? 1 : 0;
}

extern "C" int cllm_set_profiling(cllm_ctx* c, int on) {
  if (!c) return CLLM_EINVAL;
  c->profiling = on != 0;
  c->prof_acc.clear();
  return CLLM_OK;
}

extern "C" int cllm_profile_read(cllm_ctx* c, const char** names, float* ms_total, int* launches,
                                 int cap) {
  if (!c) return CLLM_EINVAL;
  static thread_local std::vector<std::string> keep;
  keep.clear();
  int i = 0;
  for (auto& kv : c->prof_acc) {
    if (i < cap) {
      keep.push_back(kv.first);
      if (ms_total) ms_total[i] = static_cast<float>(kv.second.first);
      if (launches) launches[i] = kv.second.second;
    }
    ++i;
  }
  if (names)
    for (int j = 0; j < static_cast<int>(keep.size()); ++j) names[j] = keep[j].c_str();
  return i;
}

extern "C" int cllm_kernels_per_iteration(cllm_ctx* c, int n) {
  if (!c || !c->prefilled || n < 1 || n > c->arch.max_block) return CLLM_EINVAL;
  cllm_ctx::GraphEntry* ge = nullptr;
  const bool prof = c->profiling;
  c->profiling = false;
  int rc = get_graph(c, MODE_STEP, n, &ge);
  c->profiling = prof;
  if (rc != CLLM_OK) return rc;
  return ge->launches;
}

extern "C" int cllm_committed_lengths(cllm_ctx* c, int32_t* lens_out) {
  if (!c || !lens_out) return CLLM_EINVAL;
  if (!c->prefilled) return CLLM_ESTATE;
  cudaSetDevice(c->dev);
  if (cudaMemcpyAsync(lens_out, c->Ld, c->B * 4, cudaMemcpyDeviceToHost, c->stream) != cudaSuccess)
    return CLLM_ECUDA;
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return CLLM_ECUDA;
  return CLLM_OK;
}

// ---- test hook (include/cllm_testing.h) -------------------------------------------

#include "../../include/cllm_testing.h"

extern "C" int cllm_test_gemm_bf16(const void* W, const void* X, float* Y, int M, int K, int T,
                                   int x_rows) {
  if (!W || !X || !Y || M < 128 || M % 128 || K < 8 || K % 8 || T < 1) return CLLM_EINVAL;
  if (x_rows < round_up(T, 16) || (T > 256 && x_rows < 256)) return CLLM_EINVAL;
  if (!aligned16(W) || !aligned16(X) || !aligned16(Y)) return CLLM_EINVAL;
  int dev = 0;
  cudaDeviceProp prop;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&prop, dev) != cudaSuccess)
    return CLLM_ECUDA;
  if (prop.major != 10 || prop.minor != 3) return CLLM_EUNSUPPORTED;
  if (!get_encode() || gemm_tc_set_attributes() != cudaSuccess) return CLLM_ECUDA;
  const int mtiles = M / kBM;
  const Part p = plan_gemm(mtiles, K, T, prop.multiProcessorCount);
  const int ldt = round_up(T, 16);
  GemmMaps maps{};
  if (!make_map(&maps.a0, W, K, M, kBM) || !make_map(&maps.b, X, K, 2 * x_rows, p.bn))
    return CLLM_EINVAL;
  maps.a1 = maps.a2 = maps.a0;
  std::vector<void*> tmp;
  auto alloc = [&](size_t bytes) -> void* {
    void* v = nullptr;
    if (cudaMalloc(&v, bytes) != cudaSuccess || cudaMemset(v, 0, bytes) != cudaSuccess) return nullptr;
    tmp.push_back(v);
    return v;
  };
  int rc = CLLM_OK;
  do {
    float* part = static_cast<float*>(alloc(static_cast<size_t>(mtiles) * p.maxc * p.bn * kBM * 4));
    int* tickets = static_cast<int*>(alloc(mtiles * 4));
    int* err = static_cast<int*>(alloc(16));
    float* ssq = static_cast<float*>(alloc(static_cast<size_t>(mtiles) * ldt * 4));
    void* xg = alloc(static_cast<size_t>(T) * M * 2 * 2);
    __nv_bfloat16* ones = static_cast<__nv_bfloat16*>(alloc(static_cast<size_t>(M) * 2));
    if (!part || !tickets || !err || !ssq || !xg || !ones) {
      rc = CLLM_ENOMEM;
      break;
    }
    std::vector<__nv_bfloat16> h1(M, __float2bfloat16(1.f));
    if (cudaMemcpy(ones, h1.data(), M * 2, cudaMemcpyHostToDevice) != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    GemmArgs g{};
    g.M = M;
    g.K = K;
    g.T = T;
    g.mtiles = p.mtiles;
    g.ntiles = p.ntiles;
    g.kchunks = p.kchunks;
    g.cpc = p.cpc;
    g.bn = p.bn;
    g.maxc = p.maxc;
    g.rows_q = M;
    g.rows_qk = M;
    g.lo_rows = x_rows;
    g.l2_ahead = kL2AheadDefault;
    g.pre_stages = 1 << 20;
    g.partial = part;
    g.tickets = tickets;
    g.err = err;
    EpiArgs e{};
    e.T = T;
    e.ldt = ldt;
    e.x = Y;
    e.xg = xg;
    e.gnext = ones;
    e.plane_x = static_cast<size_t>(T) * M;
    e.ssq_out = ssq;
    e.d = M;
    e.err = err;
    if (launch_gemm_tc(EPI_RESID, p.bn_max, maps, g, e, p.grid, 0, false) != cudaSuccess ||
        cudaDeviceSynchronize() != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    int herr = 0;
    if (cudaMemcpy(&herr, err, 4, cudaMemcpyDeviceToHost) != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    if (herr) rc = (herr & DERR_TIMEOUT) ? CLLM_ETIMEOUT : CLLM_EDEVICE;
  } while (0);
  for (void* v : tmp) cudaFree(v);
  return rc;
}

extern "C" int cllm_test_gemm_bf16_timed(const void* W, long long w_stride_bytes, int n_w,
                                         const void* X, float* Y, int M, int K, int T, int x_rows,
                                         int iters, int pdl, int l2_ahead, float* us_per_launch) {
  if (!W || !X || !Y || !us_per_launch || M < 128 || M % 128 || K < 8 || K % 8 || T < 1 ||
      T > 256 || iters < 1 || n_w < 1 || l2_ahead < 0)
    return CLLM_EINVAL;
  if (x_rows < round_up(T, 16)) return CLLM_EINVAL;
  int dev = 0;
  cudaDeviceProp prop;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&prop, dev) != cudaSuccess)
    return CLLM_ECUDA;
  if (prop.major != 10 || prop.minor != 3) return CLLM_EUNSUPPORTED;
  if (!get_encode() || gemm_tc_set_attributes() != cudaSuccess) return CLLM_ECUDA;
  const int mtiles = M / kBM;
  const Part p = plan_gemm(mtiles, K, T, prop.multiProcessorCount);
  const int ldt = round_up(T, 16);
  std::vector<GemmMaps> maps(n_w);
  for (int i = 0; i < n_w; ++i) {
    const char* wi = static_cast<const char*>(W) + static_cast<long long>(i) * w_stride_bytes;
    if (!make_map(&maps[i].a0, wi, K, M, kBM) || !make_map(&maps[i].b, X, K, 2 * x_rows, p.bn))
      return CLLM_EINVAL;
    maps[i].a1 = maps[i].a2 = maps[i].a0;
  }
  std::vector<void*> tmp;
  auto alloc = [&](size_t bytes) -> void* {
    void* v = nullptr;
    if (cudaMalloc(&v, bytes) != cudaSuccess || cudaMemset(v, 0, bytes) != cudaSuccess) return nullptr;
    tmp.push_back(v);
    return v;
  };
  int rc = CLLM_OK;
  cudaStream_t s = nullptr;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  do {
    float* part = static_cast<float*>(alloc(static_cast<size_t>(mtiles) * p.maxc * p.bn * kBM * 4));
    int* tickets = static_cast<int*>(alloc(mtiles * 4));
    int* err = static_cast<int*>(alloc(16));
    float* ssq = static_cast<float*>(alloc(static_cast<size_t>(mtiles) * ldt * 4));
    void* xg = alloc(static_cast<size_t>(T) * M * 2 * 2);
    void* ones = alloc(static_cast<size_t>(M) * 2);
    if (!part || !tickets || !err || !ssq || !xg || !ones) {
      rc = CLLM_ENOMEM;
      break;
    }
    if (cudaStreamCreateWithFlags(&s, cudaStreamNonBlocking) != cudaSuccess ||
        cudaEventCreate(&e0) != cudaSuccess || cudaEventCreate(&e1) != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    GemmArgs g{};
    g.M = M;
    g.K = K;
    g.T = T;
    g.mtiles = p.mtiles;
    g.ntiles = p.ntiles;
    g.kchunks = p.kchunks;
    g.cpc = p.cpc;
    g.bn = p.bn;
    g.maxc = p.maxc;
    g.rows_q = M;
    g.rows_qk = M;
    g.lo_rows = x_rows;
    g.l2_ahead = l2_ahead;
    g.pre_stages = 1 << 20;
    g.partial = part;
    g.tickets = tickets;
    g.err = err;
    EpiArgs e{};
    e.T = T;
    e.ldt = ldt;
    e.x = Y;
    e.xg = xg;
    e.gnext = ones;
    e.plane_x = static_cast<size_t>(T) * M;
    e.ssq_out = ssq;
    e.d = M;
    e.err = err;
    if (cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    cudaError_t le = cudaSuccess;
    for (int i = 0; i < iters && le == cudaSuccess; ++i)
      le = launch_gemm_tc(EPI_RESID, p.bn_max, maps[i % n_w], g, e, p.grid, s, pdl != 0);
    cudaError_t ce = cudaStreamEndCapture(s, &graph);
    if (le != cudaSuccess || ce != cudaSuccess ||
        cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    if (cudaGraphLaunch(exec, s) != cudaSuccess || cudaEventRecord(e0, s) != cudaSuccess ||
        cudaGraphLaunch(exec, s) != cudaSuccess || cudaEventRecord(e1, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess) {
      rc = CLLM_ECUDA;
      break;
    }
    float ms = 0.f;
    cudaEventElapsedTime(&ms, e0, e1);
    *us_per_launch = ms * 1000.f / iters;
    int herr = 0;
    cudaMemcpy(&herr, err, 4, cudaMemcpyDeviceToHost);
    if (herr) rc = (herr & DERR_TIMEOUT) ? CLLM_ETIMEOUT : CLLM_EDEVICE;
  } while (0);
  if (exec) cudaGraphExecDestroy(exec);
  if (graph) cudaGraphDestroy(graph);
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  if (s) cudaStreamDestroy(s);
  for (void* v : tmp) cudaFree(v);
  return rc;
}

extern "C" int cllm_test_phase_stamps(cllm_ctx* c, unsigned long long* out, int cap,
                                      const char** names, int names_cap) {
  if (!c) return CLLM_EINVAL;
  const int n = static_cast<int>(c->last_stamps.size());
  for (int i = 0; i < n && i < cap; ++i) out[i] = c->last_stamps[i];
  for (int i = 0; i < static_cast<int>(c->last_phase_names.size()) && i < names_cap; ++i)
    names[i] = c->last_phase_names[i].c_str();
  return n;
}

namespace {
int drop_graphs(cllm_ctx* c) {
  cudaSetDevice(c->dev);
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return cuda_fail(cudaGetLastError(), "sync");
  for (auto& kv : c->graphs) {
    if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
    if (kv.second.qtiles) cudaFree(kv.second.qtiles);
    for (void* p : kv.second.bufs) cudaFree(p);
  }
  c->graphs.clear();
  return CLLM_OK;
}
}  // namespace

extern "C" int cllm_test_set_trace_phase(cllm_ctx* c, int phase) {
  if (!c) return CLLM_EINVAL;
  c->trace_phase = phase;
  return drop_graphs(c);
}

extern "C" int cllm_test_hold_barrier(cllm_ctx* c, int phase) {
  if (!c || phase == 0 || phase < -1) return CLLM_EINVAL;
  c->hold_phase = phase;
  return drop_graphs(c);
}

extern "C" void cllm_test_fail_alloc(int k) { g_alloc_countdown.store(k < 0 ? -1 : k); }

extern "C" int cllm_test_plan_gemm(int mtiles, int K, int T, int sms, int* out) {
  if (!out || mtiles < 1 || K < 1 || T < 1 || sms < 1) return CLLM_EINVAL;
  const Part p = plan_gemm(mtiles, K, T, sms);
  const int v[8] = {p.mtiles, p.ntiles, p.kchunks, p.cpc, p.bn, p.bn_max, p.maxc, p.grid};
  for (int i = 0; i < 8; ++i) out[i] = v[i];
  return CLLM_OK;
}

extern "C" int cllm_test_cta_stamps(cllm_ctx* c, unsigned long long* out, long long cap) {
  if (!c) return CLLM_EINVAL;
  const long long n = static_cast<long long>(c->last_cta_stamps.size());
  for (long long i = 0; i < n && i < cap; ++i) out[i] = c->last_cta_stamps[i];
  return static_cast<int>(n);
}
