// Persistent per-iteration kernel: one Jacobi iteration (embed, every decoder
// layer's QKV GEMM / attention / O GEMM / gate-up GEMM / down GEMM, the LM
// head and the accept step) as one launch of one CTA per SM.
//
// Phases run in order from a table in global memory.  Phase p may start only
// when every CTA has finished phases 0..p-1: a grid barrier on a monotonic
// counter (each CTA's epilogue warps add 1 after each phase; waits are
// bounded and poll `counter >= p * gridDim`).  Weight tiles do not depend on
// any phase, so their producer never waits for a barrier: it streams the
// CTA's weight tiles of every GEMM phase back to back, and the MMA thread
// parks each landed tile in tensor memory (tcgen05.cp), which frees its
// shared-memory stage for the next load.  While a phase drains (split-K
// reductions, epilogues, attention, the barrier) HBM keeps streaming the next
// phase's weights into the park slots.  Activation tiles are loaded by a
// second producer after each phase's barrier.  Work split, reductions and
// epilogues are those of the per-GEMM kernels (gemm_roles.cuh), and the MMAs
// multiply the same operands in the same order, so the results are
// bit-identical to that path.
#include "attn_item.cuh"
#include "gemm_roles.cuh"
#include "step_items.cuh"

namespace cllm {

namespace {

struct EpiGroupSync {
  __device__ void operator()() const { named_bar_sync(1, 128); }
};

__host__ __device__ constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

constexpr int kPersistThreads = 224;  // producer A, MMA, 4 epilogue warps, producer B
constexpr int kTmemCols = 512;
// The kernel moves weights in pairs of 64-column chunks (the work split puts
// every range and tile on a pair boundary): one 32 KB weight stage, one
// activation stage, one barrier wait and one commit per pair.  A tcgen05.mma
// of M = 128, K = 16 occupies the tensor pipe about as long whatever its N
// (measured: ~62 ns, the same for N = 32 and 64), so four MMAs per 16 KB of
// weights give the MMA thread ~66 GB/s per SM against a ~45 GB/s share of
// HBM; per-chunk barrier waits and commits (~40-60 ns each) would eat most of
// that margin, per-pair ones half of it.
constexpr int kPairChunks = 2;
constexpr int kPairK = kPairChunks * kBK;          // 128 K columns per stage
constexpr int kParkCols = kPairK / 2;              // one parked pair: 128 x 128 bf16 = 64 columns

// Pipeline shape of the persistent kernel for up to BNMAX token columns.
//   Weight pairs (A, 32 KB) stream through a ring of SA shared-memory stages.
//   While the MMA thread cannot proceed (its next activation tile waits for a
//   grid barrier, or its accumulator is still being drained), it moves landed
//   weight pairs into NPARK tensor-memory slots (tcgen05.cp) and frees their
//   stages, so the weight stream runs on across phase boundaries; the MMAs of
//   parked pairs read A from tensor memory, the others from shared memory.
//   Weight tiles do not depend on any phase, so their producer never waits
//   for a barrier; it keeps at most kMaxWeightPairs pairs in flight.
//   Activation pairs (B: hi and lo planes of two chunks, BNMAX x 64 each)
//   go through their own ring of SB stages, issued after the phase's grid
//   barrier.  The activation ring is idle during attention phases and during
//   a phase's last split-K reduction, so it shares its shared memory with the
//   attention tile and the reduction's staging blocks.  Accumulators: NACC of
//   ACC_COLS columns at the start of tensor memory, the park slots after them.
// Shared memory: [A ring][activation ring | attention tile | split-K staging]
// [EpiSmem][attention metadata][barriers].
template <int BNMAX, int HD>
struct PersistCfg {
  static constexpr size_t ATTN_BYTES = align_up(sizeof(AttnTileSmemTma<HD>), 1024);
  static constexpr int A_BYTES = kBM * kPairK * 2;          // 32 KB: two 16 KB chunk tiles
  static constexpr int A_CHUNK = kBM * kBK * 2;
  static constexpr int B_REGION = 2 * BNMAX * kBK * 2;       // one chunk: hi rows, then lo rows
  static constexpr int B_BYTES = kPairChunks * B_REGION;
  static constexpr int SB_FIT = static_cast<int>(ATTN_BYTES / B_BYTES);
  static constexpr int SB = SB_FIT > 8 ? 8 : (SB_FIT < 2 ? 2 : SB_FIT);
  static constexpr size_t SHARED_MIN = align_up(
      ATTN_BYTES > static_cast<size_t>(SB) * B_BYTES ? ATTN_BYTES : static_cast<size_t>(SB) * B_BYTES,
      1024);
  static constexpr size_t SHARED_B =
      SHARED_MIN > 4 * kRedSlotBytes ? SHARED_MIN : align_up(4 * kRedSlotBytes, 1024);
  static constexpr int RED_FIT = static_cast<int>(SHARED_B / kRedSlotBytes);
  static constexpr int RED_SLOTS = RED_FIT > 8 ? 8 : RED_FIT;
  static constexpr size_t EPI_AREA = align_up(sizeof(EpiSmem), 16);
  // the attention work-item prefix and the iteration's metadata: computed at
  // the first attention phase, kept for every layer
  static constexpr size_t PRE_BYTES = align_up(4 * (kMaxQTilesStep + 1), 16);
  static constexpr size_t META_BYTES = PRE_BYTES + align_up(sizeof(AttnMetaSmem), 16);

  static constexpr bool STACKED = true;  // lo rows follow the bn hi rows: one MMA, N = 2 bn
  static constexpr int ACC_COLS = 2 * BNMAX;
  static constexpr int NACC = BNMAX <= 64 ? 2 : 1;
  static constexpr int BN = BNMAX;
  static constexpr int PARK_COL0 = NACC * ACC_COLS;
  static constexpr int NPARK = (kTmemCols - PARK_COL0) / kParkCols;
  static constexpr size_t BAR_FIXED = 8 * (static_cast<size_t>(2 * SB + NPARK + 2 * NACC + 2)) + 16;
  static constexpr size_t BUDGET = 227 * 1024 - 256;  // minus the kernel's static shared memory
  static constexpr size_t FIXED0 = 1024 + SHARED_B + EPI_AREA + META_BYTES + BAR_FIXED + 64;
  static constexpr int FIT = static_cast<int>((BUDGET - FIXED0 - 16 * 6) / (A_BYTES + 16));
  static constexpr int SA = FIT > 6 ? 6 : FIT;
  static constexpr size_t BAR_BYTES = BAR_FIXED + 16 * static_cast<size_t>(SA);
  static constexpr size_t SMEM = 1024 + static_cast<size_t>(SA) * A_BYTES + SHARED_B + EPI_AREA +
                                 META_BYTES + BAR_BYTES + 64;
  static_assert(SA >= 2, "weight ring too small");
  static_assert(NPARK >= 2, "too few tensor-memory park slots");
  static_assert(RED_SLOTS >= 4, "split-K staging");
  static_assert(SMEM <= BUDGET, "shared memory over budget");
};

struct PkPipe {
  uint8_t* sA;  // SA x A_BYTES, 1024-aligned
  uint8_t* sB;  // SB x B_BYTES, 1024-aligned (shared with the attention tile)
  uint64_t* afull;
  uint64_t* aempty;
  uint64_t* bfull;
  uint64_t* bempty;
  uint64_t* pempty;  // [NPARK]: the MMAs reading a park slot are done
  uint64_t* tfull;   // [NACC]
  uint64_t* tempty;  // [NACC]
  uint64_t* drain;
  uint64_t* attn_free;  // one phase per attention phase: its shared memory is free again
  volatile int* abort;
  uint32_t tmem;
  int park_limit;  // park slots in use (0: none)
};

template <class PC>
__device__ PkPipe pk_pipe_init(uint8_t* ring, uint8_t* bars) {
  PkPipe P;
  P.sA = ring;
  P.sB = ring + PC::SA * PC::A_BYTES;
  uint64_t* b = reinterpret_cast<uint64_t*>(bars);
  P.afull = b;
  P.aempty = P.afull + PC::SA;
  P.bfull = P.aempty + PC::SA;
  P.bempty = P.bfull + PC::SB;
  P.pempty = P.bempty + PC::SB;
  P.tfull = P.pempty + PC::NPARK;
  P.tempty = P.tfull + PC::NACC;
  P.drain = P.tempty + PC::NACC;
  P.attn_free = P.drain + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(P.attn_free + 1);
  P.abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int i = 0; i < PC::SA; ++i) {
      mbar_init(&P.afull[i], 1);
      mbar_init(&P.aempty[i], 1);
    }
    for (int i = 0; i < PC::SB; ++i) {
      mbar_init(&P.bfull[i], 1);
      mbar_init(&P.bempty[i], 1);
    }
    for (int i = 0; i < PC::NPARK; ++i) mbar_init(&P.pempty[i], 1);
    for (int i = 0; i < PC::NACC; ++i) {
      mbar_init(&P.tfull[i], 1);
      mbar_init(&P.tempty[i], 4);
    }
    mbar_init(P.drain, 1);
    mbar_init(P.attn_free, 1);
    *P.abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  P.tmem = *tmem_slot;
  return P;
}

// The epilogue's view of the pipeline (accumulator handshake and staging).
__device__ __forceinline__ TcPipe pk_epi_pipe(const PkPipe& K, float* red, int red_slots) {
  TcPipe P{};
  P.tfull = K.tfull;
  P.tempty = K.tempty;
  P.abort = K.abort;
  P.tmem = K.tmem;
  P.red = red;
  P.red_slots = red_slots;
  return P;
}

// ---- producer A: weight pairs, every GEMM phase back to back -------------------------

// Weight pairs in flight per SM.  Four outstanding 16 KB tiles per SM already
// stream HBM at its copy bandwidth; TMA serves an SM's requests in order, so
// every further outstanding weight load delays the (latency-critical)
// activation loads behind it: measured 0.23 us for a 4 KB load on an idle SM,
// 0.26 us behind 4 outstanding weight tiles, 0.53 us behind 8, 1.2 us behind 12.
constexpr int kMaxWeightPairs = 2;

template <int KIND, class PC>
__device__ __forceinline__ void pk_load_a_chunk(uint8_t* dst, uint64_t* bar, const GemmArgs& g,
                                                const CUtensorMap* mA0, const CUtensorMap* mA1,
                                                const CUtensorMap* mA2, int c, uint64_t pol) {
  const int u = c / g.kchunks, k = c - u * g.kchunks;
  const int mt = u / g.ntiles;
  if (KIND == EPI_GATEUP) {
    tma_load_2d(dst, mA0, bar, k * kBK, mt * 64, pol);
    tma_load_2d(dst + PC::A_CHUNK / 2, mA1, bar, k * kBK, mt * 64, pol);
  } else if (KIND == EPI_QKV) {
    const int row = mt * kBM;
    if (row < g.rows_q)
      tma_load_2d(dst, mA0, bar, k * kBK, row, pol);
    else if (row < g.rows_qk)
      tma_load_2d(dst, mA1, bar, k * kBK, row - g.rows_q, pol);
    else
      tma_load_2d(dst, mA2, bar, k * kBK, row - g.rows_qk, pol);
  } else {
    tma_load_2d(dst, mA0, bar, k * kBK, mt * kBM, pol);
  }
}

template <int KIND>
__device__ __forceinline__ void pk_prefetch_chunk(const GemmArgs& g, const CUtensorMap* mA0,
                                                  const CUtensorMap* mA1, const CUtensorMap* mA2,
                                                  int c) {
  const int u = c / g.kchunks, k = c - u * g.kchunks;
  const int mt = u / g.ntiles;
  if (KIND == EPI_GATEUP) {
    tma_prefetch_l2_2d(mA0, k * kBK, mt * 64);
    tma_prefetch_l2_2d(mA1, k * kBK, mt * 64);
  } else if (KIND == EPI_QKV) {
    const int row = mt * kBM;
    if (row < g.rows_q)
      tma_prefetch_l2_2d(mA0, k * kBK, row);
    else if (row < g.rows_qk)
      tma_prefetch_l2_2d(mA1, k * kBK, row - g.rows_q);
    else
      tma_prefetch_l2_2d(mA2, k * kBK, row - g.rows_qk);
  } else {
    tma_prefetch_l2_2d(mA0, k * kBK, mt * kBM);
  }
}

template <int KIND, class PC>
__device__ bool pk_produce_a(const PkPipe& P, int& ia, const GemmArgs& g, const CUtensorMap* mA0,
                             const CUtensorMap* mA1, const CUtensorMap* mA2, int c0, int c1,
                             int l2_ahead) {
  constexpr int S = PC::SA;
  const uint64_t pol_w = l2_policy_evict_first();
  int pf = c0;  // next chunk of this phase to prefetch into L2
  for (int c = c0; c < c1; c += kPairChunks, ++ia) {
    const int st = ia % S;
    if (l2_ahead > 0 && !mbar_test_wait(&P.aempty[st], ((ia / S) & 1) ^ 1)) {
      // the ring is full (shared and tensor memory hold every tile they
      // can): fetch the phase's next tiles into L2 meanwhile
      if (pf < c + kPairChunks) pf = c + kPairChunks;
      for (; pf < c1 && pf < c + kPairChunks * (1 + l2_ahead); ++pf)
        pk_prefetch_chunk<KIND>(g, mA0, mA1, mA2, pf);
    }
    if (!mbar_wait(&P.aempty[st], ((ia / S) & 1) ^ 1, P.abort)) return false;
    if (S > kMaxWeightPairs && ia >= kMaxWeightPairs) {  // at most kMaxWeightPairs in flight
      const int o = ia - kMaxWeightPairs;  // (its stage is not reused before this pair)
      if (!mbar_wait(&P.afull[o % S], (o / S) & 1, P.abort)) return false;
    }
    mbar_arrive_expect_tx(&P.afull[st], PC::A_BYTES);
    uint8_t* dst = P.sA + st * PC::A_BYTES;
    pk_load_a_chunk<KIND, PC>(dst, &P.afull[st], g, mA0, mA1, mA2, c, pol_w);
    pk_load_a_chunk<KIND, PC>(dst + PC::A_CHUNK, &P.afull[st], g, mA0, mA1, mA2, c + 1, pol_w);
  }
  return true;
}

__device__ __forceinline__ unsigned ld_relaxed_gpu(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Smallest of the flags f[i0..i1], up to 8 loads in flight at a time.
__device__ inline unsigned flags_min(const unsigned* f, int i0, int i1) {
  unsigned mn = ~0u;
  for (int b = i0; b <= i1; b += 8) {
    unsigned v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) v[j] = (b + j <= i1) ? ld_relaxed_gpu(f + b + j) : ~0u;
#pragma unroll
    for (int j = 0; j < 8; ++j) mn = min(mn, v[j]);
  }
  return mn;
}

// Bounded wait until the flags in `idx` (cnt of them, or the range
// idx[0]..idx[1] when range) reach target; then an acquire fence, and the
// TMA reads that follow are ordered after the generic stores the flags
// publish.  Sets *abort when the wait runs out.
__device__ inline bool wait_flags(const unsigned* f, const int* idx, int cnt, bool range,
                                  unsigned target, volatile int* abort) {
  auto low = [&]() -> unsigned {
    if (range) return flags_min(f, idx[0], idx[1]);
    unsigned v[3];
#pragma unroll
    for (int j = 0; j < 3; ++j) v[j] = j < cnt ? ld_relaxed_gpu(f + idx[j]) : ~0u;
    return min(v[0], min(v[1], v[2]));
  };
  if (low() < target) {
    const uint64_t t0 = globaltimer_ns();
    while (low() < target) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        *abort = 1;
        return false;
      }
      __nanosleep(32);
    }
  }
  asm volatile("fence.acq_rel.gpu;" ::: "memory");
  asm volatile("fence.proxy.async.global;" ::: "memory");
  return true;
}

// ---- producer B: activation pairs, after the phase's grid barrier --------------------

// gate != nullptr (O projection after attention): instead of the grid barrier,
// the CTA waits for the heads its K chunks cover (columns 64k.. of head
// 64k/hd) to reach target completions, once its own attention phase has
// released the shared memory (attn_free, phase attn_phase).
template <class PC>
__device__ bool pk_produce_b(const PkPipe& P, int& ib, const GemmArgs& g, const CUtensorMap* mB,
                             int c0, int c1, const GridDep& dep, const unsigned* gate,
                             unsigned target, int hd, int nheads, int attn_phase) {
  constexpr int S = PC::SB;
  if (c0 >= c1) return true;
  if (gate == nullptr) {
    if (!dep.wait(P.abort)) return false;
    dep.after();
  } else {
    if (!mbar_wait(P.attn_free, attn_phase & 1, P.abort)) return false;
    const int u0 = c0 / g.kchunks, u1 = (c1 - 1) / g.kchunks;
    int hr[2] = {0, nheads - 1};
    if (u0 == u1) {  // (K is padded to whole pairs: clamp to the last head)
      hr[0] = min(((c0 - u0 * g.kchunks) * kBK) / hd, nheads - 1);
      hr[1] = min(((c1 - u1 * g.kchunks) * kBK - 1) / hd, nheads - 1);
    }
    if (!wait_flags(gate, hr, 2, true, target, P.abort)) return false;
  }
  const uint64_t pol_x = l2_policy_evict_last();
  const uint32_t b_bytes = 2u * static_cast<uint32_t>(g.bn) * kBK * 2;
  const bool tile_mode = g.ntiles > 1;
  for (int c = c0; c < c1; c += kPairChunks, ++ib) {
    const int st = ib % S;
    if (!mbar_wait(&P.bempty[st], ((ib / S) & 1) ^ 1, P.abort)) return false;
    mbar_arrive_expect_tx(&P.bfull[st], kPairChunks * b_bytes);
    for (int h = 0; h < kPairChunks; ++h) {
      const int cc = c + h;
      const int u = cc / g.kchunks, k = cc - u * g.kchunks;
      const int nt = u % g.ntiles;
      const int row0 = tile_mode ? nt * PC::BN : 0;
      uint8_t* dst = P.sB + st * PC::B_BYTES + h * PC::B_REGION;
      tma_load_2d(dst, mB, &P.bfull[st], k * kBK, row0, pol_x);
      tma_load_2d(dst + g.bn * kBK * 2, mB, &P.bfull[st], k * kBK, g.lo_rows + row0, pol_x);
    }
  }
  return true;
}

// Before exit: every issued load of a ring has landed (bounded).
__device__ __forceinline__ void pk_ring_drain(uint64_t* full, int stages, int issued) {
  for (int i = max(0, issued - stages); i < issued; ++i)
    mbar_wait(&full[i % stages], (i / stages) & 1, nullptr);
}

// ---- MMA issuer ----------------------------------------------------------------------

// State of the weight stream at the MMA thread, in pairs: pairs [im, ia)
// have their weights parked in tensor memory (park ring entries [pm, pa),
// entry j in slot j % NPARK); pairs from ia on are read from their
// shared-memory stage.
struct PkMmaState {
  int ia, im, pa, pm, total;
};

// Park landed weight pairs, oldest first, into free park slots (non-blocking).
// Only called while the MMAs cannot proceed (a grid barrier or a busy
// accumulator): a copy costs tensor-pipe time comparable to an MMA, which is
// free while the pipe idles.
template <class PC>
__device__ __forceinline__ void pk_park(const PkPipe& P, PkMmaState& q) {
  if (q.ia < q.im) q.ia = q.im;
  while (q.ia < q.total && q.pa - q.pm < P.park_limit) {
    const int st = q.ia % PC::SA, sl = q.pa % PC::NPARK;
    if (!mbar_test_wait(&P.pempty[sl], ((q.pa / PC::NPARK) & 1) ^ 1)) return;
    if (!mbar_test_wait(&P.afull[st], (q.ia / PC::SA) & 1)) return;
    tc_fence_after();
    const uint32_t a_addr = smem_u32(P.sA + st * PC::A_BYTES);
    const uint32_t t = P.tmem + static_cast<uint32_t>(PC::PARK_COL0 + sl * kParkCols);
#pragma unroll
    for (int kk = 0; kk < kPairK / 16; ++kk)
      tc_cp_128x256b(t + kk * 8,
                     sdesc_kmajor_sw128(a_addr + (kk >> 2) * PC::A_CHUNK + (kk & 3) * 32));
    tc_commit(&P.aempty[st]);  // the stage is free once the copies are done
    ++q.ia;
    ++q.pa;
  }
}

// Spin (bounded) until ready(); with may_park, park weight pairs meanwhile.
template <class PC, class F>
__device__ bool pk_wait(const PkPipe& P, PkMmaState& q, bool may_park, F ready) {
  if (ready()) return true;
  const uint64_t t0 = globaltimer_ns();
  uint32_t it = 0;
  for (;;) {
    if (may_park) pk_park<PC>(P, q);
    if (ready()) return true;
    if ((++it & 63u) == 0) {
      if (*P.abort) return false;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        *P.abort = 1;
        return false;
      }
    }
  }
}

// MMAs of one GEMM phase, a pair of chunks at a time.  Pair im reads its
// activations from B stage im % SB and its weights from its park slot (if it
// was parked) or from A stage im % SA.
template <class PC>
__device__ bool pk_mma(const PkPipe& P, PkMmaState& q, int& acc, uint32_t& accph,
                       const GemmArgs& g, int c0, int c1, unsigned long long* prof,
                       long long prof_stride, unsigned long long* trace) {
  unsigned long long t_first = 0, t_last = 0, gap = 0;
  int ntrace = 0;
  const uint32_t idesc = idesc_bf16_f32(kBM, 2 * g.bn);
  const bool can_park = P.park_limit > 0;
  int c = c0;
  bool first = true;
  Segment sg;
  while (next_segment(c, c1, g.kchunks, sg)) {
    const int a_now = acc;
    const uint32_t ph_now = accph;
    if (!pk_wait<PC>(P, q, can_park, [&] { return mbar_test_wait(&P.tempty[a_now], ph_now ^ 1); }))
      return false;
    tc_fence_after();
    const uint32_t dt = P.tmem + static_cast<uint32_t>(acc * PC::ACC_COLS);
    for (int k = sg.k0; k < sg.k1; k += kPairChunks) {
      const int im = q.im;
      const int sb = im % PC::SB, sa = im % PC::SA;
      // the phase's first activation pair waits for the grid barrier: park
      // the weight stream meanwhile
      if (!pk_wait<PC>(P, q, can_park && first, [&] {
            return (q.ia > im || mbar_test_wait(&P.afull[sa], (im / PC::SA) & 1)) &&
                   mbar_test_wait(&P.bfull[sb], (im / PC::SB) & 1);
          }))
        return false;
      first = false;
      tc_fence_after();
      if (prof != nullptr) {
        const unsigned long long now = globaltimer_ns();
        if (trace != nullptr && ntrace < kTraceCap) trace[ntrace++] = now;
        if (t_first == 0) t_first = now;
        else if (now - t_last > gap) gap = now - t_last;
        t_last = now;
      }
      const uint32_t b_addr = smem_u32(P.sB + sb * PC::B_BYTES);
      const uint32_t accum0 = k > sg.k0 ? 1u : 0u;
      if (q.ia > im) {  // parked
        const int sl = q.pm % PC::NPARK;
        const uint32_t a_t = P.tmem + static_cast<uint32_t>(PC::PARK_COL0 + sl * kParkCols);
#pragma unroll
        for (int kk = 0; kk < kPairK / 16; ++kk)
          tc_mma_f16_ts(dt, a_t + kk * 8,
                        sdesc_kmajor_sw128(b_addr + (kk >> 2) * PC::B_REGION + (kk & 3) * 32), idesc,
                        (accum0 || kk > 0) ? 1u : 0u);
        tc_commit(&P.pempty[sl]);
        ++q.pm;
      } else {
        const uint32_t a_addr = smem_u32(P.sA + sa * PC::A_BYTES);
#pragma unroll
        for (int kk = 0; kk < kPairK / 16; ++kk)
          tc_mma_f16(dt, sdesc_kmajor_sw128(a_addr + (kk >> 2) * PC::A_CHUNK + (kk & 3) * 32),
                     sdesc_kmajor_sw128(b_addr + (kk >> 2) * PC::B_REGION + (kk & 3) * 32), idesc,
                     (accum0 || kk > 0) ? 1u : 0u);
        tc_commit(&P.aempty[sa]);
      }
      tc_commit(&P.bempty[sb]);
      ++q.im;
    }
    tc_commit(&P.tfull[acc]);
    if (++acc == PC::NACC) {
      acc = 0;
      accph ^= 1;
    }
  }
  if (prof != nullptr) {
    prof[0] = t_first;
    prof[prof_stride] = t_last;
    prof[2 * prof_stride] = gap;
  }
  return true;
}

// The phase's arguments are copied into registers first: read through a
// reference into the phase table, every asm statement with a memory clobber
// (TMA issue, mbarrier operations) would force them to be reloaded.
template <class PC>
__device__ bool produce_a_phase(const PkPipe& P, int& ia, const PhaseDesc& ph,
                                const CUtensorMap* maps, int cta, int l2_ahead) {
  const GemmArgs g = ph.g;
  const CUtensorMap* m0 = maps + ph.map_a0;
  const CUtensorMap* m1 = maps + ph.map_a1;
  const CUtensorMap* m2 = maps + ph.map_a2;
  int c0, c1;
  cta_range(g, cta, c0, c1);
  switch (ph.epi) {
    case EPI_QKV: return pk_produce_a<EPI_QKV, PC>(P, ia, g, m0, m1, m2, c0, c1, l2_ahead);
    case EPI_GATEUP: return pk_produce_a<EPI_GATEUP, PC>(P, ia, g, m0, m1, m2, c0, c1, l2_ahead);
    default: return pk_produce_a<EPI_RESID, PC>(P, ia, g, m0, m1, m2, c0, c1, l2_ahead);
  }
}

template <class PC>
__device__ bool epilogue_phase(const TcPipe& P, int& acc, uint32_t& accph, const PhaseDesc& ph,
                               int cta, EpiSmem& es) {
  const GemmArgs g = ph.g;
  const EpiArgs e = ph.e;
  const int epi = ph.epi;
  int c0, c1;
  cta_range(g, cta, c0, c1);
  switch (epi) {
    case EPI_QKV: return tc_epilogue<EPI_QKV, PC>(P, acc, accph, g, e, c0, c1, cta, es);
    case EPI_GATEUP: return tc_epilogue<EPI_GATEUP, PC>(P, acc, accph, g, e, c0, c1, cta, es);
    case EPI_RESID: return tc_epilogue<EPI_RESID, PC>(P, acc, accph, g, e, c0, c1, cta, es);
    default: return tc_epilogue<EPI_ARGMAX, PC>(P, acc, accph, g, e, c0, c1, cta, es);
  }
}

// Arrivals the grid barrier must count before phase p starts: every CTA
// arrives once after each earlier phase.  (The hold hook asks for one more.)
__device__ __forceinline__ unsigned barrier_target(const StepArgs& A, int p, int G) {
  return static_cast<unsigned>(p) * static_cast<unsigned>(G) + (p == A.hold_phase ? 1u : 0u);
}

}  // namespace

template <int BNMAX, int HD>
__global__ void __launch_bounds__(kPersistThreads, 1)
    step_persistent_kernel(const __grid_constant__ StepParams PRM) {
  const StepArgs& A = PRM.a;
  using PC = PersistCfg<BNMAX, HD>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ float s_red[4];
  __shared__ int s_act[4], s_com[4];
  __shared__ int s_flag;
  uint8_t* base =
      reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* shb = base + static_cast<size_t>(PC::SA) * PC::A_BYTES;  // 1024-aligned
  AttnTileSmemTma<HD>& at = *reinterpret_cast<AttnTileSmemTma<HD>*>(shb);
  uint8_t* epi = shb + PC::SHARED_B;
  EpiSmem& es = *reinterpret_cast<EpiSmem*>(epi);
  int* pre = reinterpret_cast<int*>(epi + PC::EPI_AREA);
  AttnMetaSmem& meta = *reinterpret_cast<AttnMetaSmem*>(epi + PC::EPI_AREA + PC::PRE_BYTES);
  uint8_t* bars = epi + PC::EPI_AREA + PC::META_BYTES;
  PkPipe K = pk_pipe_init<PC>(base, bars);
  // park_limit < 0: no parking; 0: every slot; else that many
  K.park_limit =
      A.park_limit < 0 ? 0 : (A.park_limit > 0 && A.park_limit < PC::NPARK ? A.park_limit : PC::NPARK);
  const TcPipe P = pk_epi_pipe(K, reinterpret_cast<float*>(shb), PC::RED_SLOTS);
  const int G = gridDim.x, cta = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer: weight tiles ----------------
      int ia = 0;
      const size_t PG = static_cast<size_t>(A.n_phases) * G;
      for (int p = 0; p < A.n_phases; ++p) {
        const PhaseDesc& ph = A.phases[p];
        if (ph.kind != PH_GEMM) continue;
        unsigned long long* cs =
            A.cta_stamps != nullptr ? A.cta_stamps + static_cast<size_t>(p) * G + cta : nullptr;
        if (cs != nullptr) cs[6 * PG] = globaltimer_ns();
        const bool ok = produce_a_phase<PC>(K, ia, ph, PRM.maps, cta, A.l2_ahead);
        if (cs != nullptr) cs[8 * PG] = globaltimer_ns();
        if (!ok) break;
      }
      pk_ring_drain(K.afull, PC::SA, ia);
    }
  } else if (warp == 6) {
    if (lane == 0) {
      // ---------------- TMA producer: activation tiles ----------------
      int ib = 0, attn_phases = 0;
      for (int p = 0; p < A.n_phases; ++p) {
        const PhaseDesc& ph = A.phases[p];
        if (ph.kind == PH_ATTN) ++attn_phases;
        if (ph.kind != PH_GEMM) continue;
        const GemmArgs g = ph.g;
        int c0, c1;
        cta_range(g, cta, c0, c1);
        const GridDep dep{A.bar, barrier_target(A, p, G)};
        const unsigned* gate = ph.no_barrier ? ph.head_done : nullptr;
        const unsigned target = static_cast<unsigned>(ph.flag_target) + (p == A.hold_phase ? 1u : 0u);
        if (!pk_produce_b<PC>(K, ib, g, PRM.maps + ph.map_b, c0, c1, dep, gate, target, A.attn.hd,
                              A.attn.H, attn_phases - 1))
          break;
      }
      pk_ring_drain(K.bfull, PC::SB, ib);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int total = 0;  // weight tiles of this CTA over the whole iteration
      for (int p = 0; p < A.n_phases; ++p) {
        const PhaseDesc& ph = A.phases[p];
        if (ph.kind != PH_GEMM) continue;
        int c0, c1;
        cta_range(ph.g, cta, c0, c1);
        total += max(0, c1 - c0) / kPairChunks;
      }
      PkMmaState q{0, 0, 0, 0, total};
      int acc = 0;
      uint32_t accph = 0;
      const long long PG = static_cast<long long>(A.n_phases) * G;
      for (int p = 0; p < A.n_phases; ++p) {
        const PhaseDesc& ph = A.phases[p];
        if (ph.kind != PH_GEMM) continue;
        unsigned long long* prof = nullptr;
        unsigned long long* trace = nullptr;
        if (A.cta_stamps != nullptr) {
          prof = A.cta_stamps + 10 * PG + static_cast<long long>(p) * G + cta;
          if (p == A.trace_phase)
            trace = A.cta_stamps + kCtaStampSlots * PG + static_cast<long long>(cta) * kTraceCap;
        }
        const GemmArgs g = ph.g;
        int c0, c1;
        cta_range(g, cta, c0, c1);
        if (!pk_mma<PC>(K, q, acc, accph, g, c0, c1, prof, PG, trace)) break;
        if (A.cta_stamps != nullptr)
          A.cta_stamps[(static_cast<size_t>(A.n_phases) + p) * G + cta] = globaltimer_ns();
      }
      // before exit: every issued copy and MMA has completed (bounded)
      tc_commit(K.drain);
      mbar_wait(K.drain, 0, nullptr);
    }
  } else {
    // ---------------- epilogue / attention / embed / accept (128 threads) ----------------
    const int r = (warp & 3) * 32 + lane;
    const EpiGroupSync sync;
    int acc = 0;
    uint32_t accph = 0;
    int attn_total = -1;  // attention work items of this iteration (prefix in smem)
    for (int p = 0; p < A.n_phases; ++p) {
      const PhaseDesc& ph = A.phases[p];
      const int kind = ph.kind;
      if (kind == PH_ACCEPT && cta != 0) break;
      if (p > 0 && !ph.no_barrier) {
        const GridDep dep{A.bar, barrier_target(A, p, G)};
        if (r == 0) s_flag = dep.wait(P.abort) ? 1 : 0;
        sync();
        const bool ok = s_flag != 0;
        sync();
        if (!ok) break;
      }
      if (A.stamps != nullptr && r == 0) {
        // [0, P]: CTA 0's phase starts; then per phase: first/last start and
        // first/last arrival over the CTAs
        const unsigned long long now = globaltimer_ns();
        if (cta == 0) A.stamps[p] = now;
        if (A.cta_stamps != nullptr) A.cta_stamps[static_cast<size_t>(p) * G + cta] = now;
        unsigned long long* st = A.stamps + (A.n_phases + 1);
        atomicMin(&st[p], now);
        atomicMax(&st[A.n_phases + p], now);
      }
      bool ok = true;
      if (kind == PH_EMBED) {
        const int ngrp = A.embed.d / 128;
        const int units = A.embed.T * ngrp;
        for (int u = cta; u < units; u += G)
          embed_unit<__nv_bfloat16>(A.embed, u / ngrp, u % ngrp, r, s_red, sync);
      } else if (kind == PH_GEMM) {
        ok = epilogue_phase<PC>(P, acc, accph, ph, cta, es);
      } else if (kind == PH_ATTN) {
        AttnArgs a = A.attn;
        a.k_cache = ph.k_cache;
        a.v_cache = ph.v_cache;
        const SmemMeta md{meta};
        if (attn_total < 0) {  // the first attention phase of the launch
          attn_meta_load(a, meta, r, A.accept.B);
          sync();
          attn_total = attn_item_prefix(a, pre, r, sync, md);
        }
        const int total = attn_total;
        const AttnTma tma{PRM.maps + A.map_attn_k, PRM.maps + A.map_attn_v, PRM.maps + A.map_attn_q,
                          ph.kv_row0};
        // an item's head's output is complete once per query tile: publish it
        // (read next through TMA by the O projection)
        auto publish_head = [&](int hh) {
          asm volatile("fence.proxy.async.global;" ::: "memory");
          sync();
          if (r == 0)
            asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ph.head_done + hh) : "memory");
        };
        for (int item = cta; item < total; item += G) {
          if (ph.qkv_done != nullptr) {
            // wait for this item's head's Q, K and V tiles instead of the grid barrier
            const int qi0 = attn_find_qtile(pre, a.n_qtiles, item);
            const int hh = (item - pre[qi0]) % a.H;
            const int kvh = hh / (a.H / a.Hkv);
            const int dq = a.H * HD, dkv = a.Hkv * HD;
            const int tq = (hh * HD) / kBM, tk = (dq + kvh * HD) / kBM, tv = (dq + dkv + kvh * HD) / kBM;
            if (r == 0) {
              const unsigned tgt = static_cast<unsigned>(ph.flag_target) + (p == A.hold_phase ? 1u : 0u);
              const int tiles[3] = {tq, tk, tv};
              s_flag = wait_flags(ph.qkv_done, tiles, 3, false, tgt, P.abort) ? 1 : 0;
            }
            sync();
            const bool ready = s_flag != 0;
            sync();
            if (!ready) {
              ok = false;
              break;
            }
            asm volatile("fence.proxy.async.global;" ::: "memory");  // the item's TMA reads
          }
          int qi, h;
          if (attn_mma_item<HD>(a, item, pre, at, r, sync, qi, h, md, true, &tma)) {
            if (ph.head_done != nullptr) publish_head(h);
            continue;  // output written
          }
          // the last range of (tile, head) to finish merges the tile's ranges
          sync();
          if (r == 0) {
            const int old = ticket_add(&A.attn_tickets[qi * a.H + h], 1);
            s_flag = (old == attn_tile_ranges(a, md, qi) - 1) ? 1 : 0;
          }
          sync();
          const bool last = s_flag != 0;
          sync();
          if (last) {
            attn_combine_tile<__nv_bfloat16, HD>(a, qi, h, r, md);
            if (r == 0) A.attn_tickets[qi * a.H + h] = 0;
            if (ph.head_done != nullptr) publish_head(h);
          }
        }
      } else {  // PH_ACCEPT (CTA 0)
        accept_body(A.accept, r, s_act, s_com, sync);
      }
      if (!ok) break;
      if (p + 1 < A.n_phases) {
        // this CTA's global writes of phase p are read next by other CTAs,
        // some through TMA (async proxy); thread 0's release after the
        // barrier covers every thread's writes
        asm volatile("fence.proxy.async.global;" ::: "memory");
        // and this phase's generic shared-memory accesses (split-K staging,
        // attention tile) precede the next phase's TMA writes to that area
        fence_proxy_async_smem();
        sync();
        if (r == 0) {
          if (A.stamps != nullptr) {
            const unsigned long long now = globaltimer_ns();
            unsigned long long* st = A.stamps + (A.n_phases + 1);
            atomicMin(&st[2 * A.n_phases + p], now);
            atomicMax(&st[3 * A.n_phases + p], now);
            if (A.cta_stamps != nullptr)
              A.cta_stamps[(2 * static_cast<size_t>(A.n_phases) + p) * G + cta] = now;
          }
          asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(A.bar) : "memory");
          // the attention tile's shared memory is the activation ring again
          if (kind == PH_ATTN) mbar_arrive(K.attn_free);
        }
      }
    }
    if (A.stamps != nullptr && cta == 0 && r == 0) A.stamps[A.n_phases] = globaltimer_ns();
  }
  // release tensor memory once every role has finished and drained
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(K.tmem, kTmemCols);
  }
  if (threadIdx.x == 0 && *K.abort) atomicOr(A.err, DERR_TIMEOUT);
}

// ---- launch ----------------------------------------------------------------------------

size_t step_persistent_smem_bytes(int bn_max, int hd) {
  if (hd == 64) {
    switch (bn_max) {
      case 16: return PersistCfg<16, 64>::SMEM;
      case 32: return PersistCfg<32, 64>::SMEM;
      case 64: return PersistCfg<64, 64>::SMEM;
      default: return PersistCfg<128, 64>::SMEM;
    }
  }
  switch (bn_max) {
    case 16: return PersistCfg<16, 128>::SMEM;
    case 32: return PersistCfg<32, 128>::SMEM;
    case 64: return PersistCfg<64, 128>::SMEM;
    default: return PersistCfg<128, 128>::SMEM;
  }
}

template <int BN, int HD>
static cudaError_t set_one() {
  cudaError_t e = cudaFuncSetAttribute(step_persistent_kernel<BN, HD>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(PersistCfg<BN, HD>::SMEM));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(step_persistent_kernel<BN, HD>,
                              cudaFuncAttributePreferredSharedMemoryCarveout,
                              static_cast<int>(cudaSharedmemCarveoutMaxShared));
}

cudaError_t step_persistent_set_attributes() {
  cudaError_t e;
  if ((e = set_one<16, 64>()) != cudaSuccess) return e;
  if ((e = set_one<32, 64>()) != cudaSuccess) return e;
  if ((e = set_one<64, 64>()) != cudaSuccess) return e;
  if ((e = set_one<128, 64>()) != cudaSuccess) return e;
  if ((e = set_one<16, 128>()) != cudaSuccess) return e;
  if ((e = set_one<32, 128>()) != cudaSuccess) return e;
  if ((e = set_one<64, 128>()) != cudaSuccess) return e;
  return set_one<128, 128>();
}

// Grid = SM count and one CTA per SM (shared memory): every CTA is resident on
// an otherwise idle device.  Inside a CUDA graph the cooperative attribute is
// set on the captured node (stream capture of a cooperative launch is not
// supported); the grid-barrier waits are bounded either way.
template <int BN, int HD>
static cudaError_t launch_one(const StepParams& a, int grid, cudaStream_t s, bool cooperative) {
  cudaLaunchConfig_t cfg = cudaLaunchConfig_t{};
  cudaLaunchAttribute attr[1];
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kPersistThreads);
  cfg.dynamicSmemBytes = PersistCfg<BN, HD>::SMEM;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = cooperative ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, step_persistent_kernel<BN, HD>, a);
}

cudaError_t launch_step_persistent(const StepParams& a, int bn_max, int hd, int grid,
                                   cudaStream_t s, bool cooperative) {
  if (hd == 64) {
    switch (bn_max) {
      case 16: return launch_one<16, 64>(a, grid, s, cooperative);
      case 32: return launch_one<32, 64>(a, grid, s, cooperative);
      case 64: return launch_one<64, 64>(a, grid, s, cooperative);
      case 128: return launch_one<128, 64>(a, grid, s, cooperative);
      default: return cudaErrorInvalidValue;
    }
  }
  if (hd == 128) {
    switch (bn_max) {
      case 16: return launch_one<16, 128>(a, grid, s, cooperative);
      case 32: return launch_one<32, 128>(a, grid, s, cooperative);
      case 64: return launch_one<64, 128>(a, grid, s, cooperative);
      case 128: return launch_one<128, 128>(a, grid, s, cooperative);
      default: return cudaErrorInvalidValue;
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace cllm
