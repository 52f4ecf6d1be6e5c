// The three warp roles of the weight-streaming GEMM, as device functions that
// carry their pipeline state across calls.  A standalone GEMM kernel runs one
// phase; the persistent per-iteration kernel runs many phases back to back on
// the same shared-memory ring and TMEM accumulators.
//
//   producer (one thread): TMA of weight tiles (A, evict-first) and the
//     activation tile's hi/lo planes (B, evict-last) into the stage ring.
//     Weight tiles do not depend on earlier work, so they are issued before
//     the phase's dependency (previous kernel / grid barrier) is satisfied;
//     activation tiles only after.
//   MMA issuer (one thread): tcgen05.mma M=128 into a TMEM accumulator pair.
//   epilogue (warps 2..5, 128 threads): tcgen05.ld, split-K partials with a
//     last-arriver fixed-order reduction, fused epilogue (epilogue.cuh).
#pragma once
#include "epilogue.cuh"

namespace cllm {

// Stage = one 128 x 64 weight tile + the hi and lo planes of a BNMAX x 64
// activation tile.
template <int BNMAX, int STAGES_>
struct TcCfg {
  static constexpr int STAGES = STAGES_;
  static constexpr int A_BYTES = kBM * kBK * 2;
  static constexpr int B_HALF = BNMAX * kBK * 2;
  static constexpr int B_BYTES = 2 * B_HALF;
  // The hi and lo products land in separate accumulator columns and are summed
  // in the epilogue, for every BNMAX, so a token's result is the same
  // whatever the launch's token count.  BNMAX <= 128: the lo rows follow the
  // bn hi rows in shared memory and one MMA with N = 2*bn covers both (lo at
  // column bn + t); BNMAX = 256: two MMAs, lo into columns 256 + t.
  static constexpr bool STACKED = BNMAX <= 128;
  static constexpr int ACC_COLS = 2 * BNMAX;
  static constexpr int NACC = ACC_COLS <= 256 ? 2 : 1;  // accumulators in TMEM (512 columns)
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int TMEM_COLS = NACC * ACC_COLS;  // 128, 256, 512 or 512
  static constexpr int BN = BNMAX;
};

struct TcPipe {
  uint8_t* sA;  // STAGES x A_BYTES, 1024-aligned
  uint8_t* sB;  // STAGES x B_BYTES
  uint64_t* full;
  uint64_t* empty;
  uint64_t* tfull;   // [2]
  uint64_t* tempty;  // [2]
  uint64_t* drain;
  volatile int* abort;
  uint32_t tmem;
  // staging of split-K partials for the last arriver's reduction: red_slots
  // blocks of kEpiCols x kBM floats (set by the kernel after tc_pipe_init)
  float* red;
  int red_slots;
  int* jflag;  // two epilogue groups, shared memory: [0] the split-K wait's result, [1] the accumulator wait's
};

constexpr size_t kRedSlotBytes = sizeof(float) * kEpiCols * kBM;

// Shared-memory bytes of the barrier block that follows the ring.
__host__ __device__ constexpr size_t tc_bar_bytes(int stages) { return 8 * (2 * stages + 5) + 16; }

// Carve the pipeline from shared memory and initialise it (all threads call).
// `bars` must be 8-byte aligned and hold tc_bar_bytes(STAGES) bytes.
// NG: epilogue groups of 4 warps (each warp releases the accumulator).
template <class Cfg, int NG = 1>
__device__ TcPipe tc_pipe_init(uint8_t* ring, uint8_t* bars) {
  constexpr int S = Cfg::STAGES;
  TcPipe P;
  P.sA = ring;
  P.sB = ring + S * Cfg::A_BYTES;
  uint64_t* b = reinterpret_cast<uint64_t*>(bars);
  P.full = b;
  P.empty = b + S;
  P.tfull = b + 2 * S;
  P.tempty = P.tfull + 2;
  P.drain = P.tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(P.drain + 1);
  P.abort = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&P.full[i], 1);
      mbar_init(&P.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&P.tfull[i], 1);
      mbar_init(&P.tempty[i], 4 * NG);
    }
    mbar_init(P.drain, 1);
    *P.abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  P.tmem = *tmem_slot;
  return P;
}

// Release TMEM (all threads call; every role has finished and drained).
template <class Cfg>
__device__ void tc_pipe_release(const TcPipe& P) {
  tc_fence_before();
  __syncthreads();
  if ((threadIdx.x >> 5) == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(P.tmem, Cfg::TMEM_COLS);
  }
}

// ---- dependency policies --------------------------------------------------------

// Standalone kernels: the previous kernel in the stream (programmatic
// dependent launch); not pollable.
struct PdlDep {
  static constexpr bool kPollable = false;
  __device__ bool ready() const { return false; }
  __device__ bool wait(volatile int*) const {
    pdl_wait();
    return true;
  }
  __device__ void after() const {}
};

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Persistent kernel: grid barrier counter >= target (every CTA finished the
// phases this one depends on).  Waits are bounded.
struct GridDep {
  static constexpr bool kPollable = true;
  const unsigned* counter;
  unsigned target;
  __device__ bool ready() const { return ld_acquire_gpu(counter) >= target; }
  __device__ bool wait(volatile int* abort) const {
    if (ready()) return true;
    const uint64_t t0 = globaltimer_ns();
    while (!ready()) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > kWaitBudgetNs) {
        *abort = 1;
        return false;
      }
      __nanosleep(32);
    }
    return true;
  }
  // global data written by other CTAs' generic stores is read next by TMA
  __device__ void after() const { asm volatile("fence.proxy.async.global;" ::: "memory"); }
};

// ---- work decomposition -----------------------------------------------------------

struct Segment {
  int unit, k0, k1;
};

// Iterate the (unit, k-range) segments of the chunk range [c, c1).
__device__ __forceinline__ bool next_segment(int& c, int c1, int kchunks, Segment& sg) {
  if (c >= c1) return false;
  sg.unit = c / kchunks;
  sg.k0 = c - sg.unit * kchunks;
  const int end = min(c1, (sg.unit + 1) * kchunks);
  sg.k1 = end - sg.unit * kchunks;
  c = end;
  return true;
}

// Chunk range of CTA `cta` in a launch's work split.
__device__ __forceinline__ void cta_range(const GemmArgs& g, int cta, int& c0, int& c1) {
  const int total = g.mtiles * g.ntiles * g.kchunks;
  c0 = min(total, cta * g.cpc);
  c1 = min(total, c0 + g.cpc);
}

// ---- producer -------------------------------------------------------------------------

// Issue this CTA's chunks [c0, c1) of one GEMM phase.  `idx` counts chunks
// issued so far (ring position).  Returns false if a bounded wait gave up.
template <int KIND, class Cfg, class Dep>
__device__ bool tc_produce(const TcPipe& P, int& idx, int& issued_b, const GemmArgs& g,
                           const CUtensorMap* mA0, const CUtensorMap* mA1, const CUtensorMap* mA2,
                           const CUtensorMap* mB, int c0, int c1, const Dep& dep) {
  constexpr int S = Cfg::STAGES;
  const int n = c1 - c0;
  if (n <= 0) {
    if (!Dep::kPollable) dep.wait(P.abort);
    return true;
  }
  const uint64_t pol_w = l2_policy_evict_first();
  const uint64_t pol_x = l2_policy_evict_last();
  const bool tile_mode = g.ntiles > 1;
  const uint32_t b_bytes = 2u * static_cast<uint32_t>(g.bn) * kBK * 2;
  auto load_a = [&](int j, int st) {
    const int c = c0 + j;
    const int u = c / g.kchunks, k = c - u * g.kchunks;
    const int mt = u / g.ntiles;
    uint8_t* dst = P.sA + st * Cfg::A_BYTES;
    if (KIND == EPI_GATEUP) {
      tma_load_2d(dst, mA0, &P.full[st], k * kBK, mt * 64, pol_w);
      tma_load_2d(dst + Cfg::A_BYTES / 2, mA1, &P.full[st], k * kBK, mt * 64, pol_w);
    } else if (KIND == EPI_QKV) {
      const int row = mt * kBM;
      if (row < g.rows_q)
        tma_load_2d(dst, mA0, &P.full[st], k * kBK, row, pol_w);
      else if (row < g.rows_qk)
        tma_load_2d(dst, mA1, &P.full[st], k * kBK, row - g.rows_q, pol_w);
      else
        tma_load_2d(dst, mA2, &P.full[st], k * kBK, row - g.rows_qk, pol_w);
    } else {
      tma_load_2d(dst, mA0, &P.full[st], k * kBK, mt * kBM, pol_w);
    }
  };
  auto load_b = [&](int j, int st) {
    const int c = c0 + j;
    const int u = c / g.kchunks, k = c - u * g.kchunks;
    const int nt = u % g.ntiles;
    const int row0 = tile_mode ? nt * Cfg::BN : 0;
    uint8_t* dst = P.sB + st * Cfg::B_BYTES;
    tma_load_2d(dst, mB, &P.full[st], k * kBK, row0, pol_x);
    tma_load_2d(dst + (Cfg::STACKED ? g.bn * kBK * 2 : Cfg::B_HALF), mB, &P.full[st], k * kBK,
                g.lo_rows + row0, pol_x);
  };
  auto prefetch_l2 = [&](int j) {
    const int c = c0 + j;
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
  };
  // Weight tiles into free stages while the dependency is not satisfied; once
  // the ring is full, the next l2_ahead tiles into L2 (once), so that HBM
  // keeps streaming while the previous phase drains.
  int j = 0;
  bool open = Dep::kPollable ? dep.ready() : false;
  bool prefetched = false;
  uint64_t t0 = 0;
  while (j < n && !open) {
    const int gi = idx + j, st = gi % S;
    if (j < g.pre_stages && mbar_try_wait(&P.empty[st], ((gi / S) & 1) ^ 1)) {
      mbar_arrive_expect_tx(&P.full[st], Cfg::A_BYTES + b_bytes);
      load_a(j, st);
      ++j;
      if (Dep::kPollable) open = dep.ready();
      continue;
    }
    if (!Dep::kPollable) break;
    if (!prefetched) {
      for (int jj = j; jj < min(n, j + g.l2_ahead); ++jj) prefetch_l2(jj);
      prefetched = true;
    }
    open = dep.ready();
    if (open) break;
    if (*P.abort) break;  // gave up: dep.wait below returns false at once
    if (t0 == 0) {
      t0 = globaltimer_ns();
    } else if (globaltimer_ns() - t0 > kWaitBudgetNs) {
      *P.abort = 1;
      break;
    }
    __nanosleep(32);
  }
  const bool dep_ok = open || dep.wait(P.abort);
  if (dep_ok) dep.after();
  // Activation tiles of the stages issued so far.  (On a failed wait they are
  // still issued -- in-bounds reads of stale data -- so that every stage this
  // thread started completes and can be drained before the CTA exits.)
  for (int jj = 0; jj < j; ++jj) load_b(jj, (idx + jj) % S);
  issued_b = idx + j;
  if (!dep_ok) {
    idx += j;
    return false;
  }
  for (; j < n; ++j) {
    const int gi = idx + j, st = gi % S;
    if (!mbar_wait(&P.empty[st], ((gi / S) & 1) ^ 1, P.abort)) {
      idx += j;
      return false;
    }
    mbar_arrive_expect_tx(&P.full[st], Cfg::A_BYTES + b_bytes);
    load_a(j, st);
    load_b(j, st);
    issued_b = gi + 1;
  }
  idx += n;
  return true;
}

// Before exit: every fully issued stage has landed (bounded).
template <class Cfg>
__device__ void tc_produce_drain(const TcPipe& P, int issued) {
  constexpr int S = Cfg::STAGES;
  for (int i = max(0, issued - S); i < issued; ++i) mbar_wait(&P.full[i % S], (i / S) & 1, nullptr);
}

// ---- MMA issuer ------------------------------------------------------------------------

template <class Cfg>
__device__ bool tc_mma(const TcPipe& P, int& idx, int& acc, uint32_t& accph, const GemmArgs& g,
                       int c0, int c1, unsigned long long* prof = nullptr, long long prof_stride = 0,
                       unsigned long long* trace = nullptr) {
  constexpr int S = Cfg::STAGES;
  // optional profile: first and last stage arrival, largest gap between
  // arrivals, and (trace) every arrival
  unsigned long long t_first = 0, t_last = 0, gap = 0;
  int ntrace = 0;
  const uint32_t idesc = idesc_bf16_f32(kBM, Cfg::STACKED ? 2 * g.bn : g.bn);
  int c = c0;
  Segment sg;
  while (next_segment(c, c1, g.kchunks, sg)) {
    if (!mbar_wait(&P.tempty[acc], accph ^ 1, P.abort)) return false;
    tc_fence_after();
    const uint32_t dt = P.tmem + static_cast<uint32_t>(acc * Cfg::ACC_COLS);
    for (int k = sg.k0; k < sg.k1; ++k, ++idx) {
      const int st = idx % S;
      if (!mbar_wait(&P.full[st], (idx / S) & 1, P.abort)) return false;
      tc_fence_after();
      if (prof != nullptr) {
        const unsigned long long now = globaltimer_ns();
        if (trace != nullptr && ntrace < kTraceCap) trace[ntrace++] = now;
        if (t_first == 0) t_first = now;
        else if (now - t_last > gap) gap = now - t_last;
        t_last = now;
      }
      const uint32_t a_addr = smem_u32(P.sA + st * Cfg::A_BYTES);
      const uint32_t b_addr = smem_u32(P.sB + st * Cfg::B_BYTES);
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk) {
        const uint64_t ad = sdesc_kmajor_sw128(a_addr + kk * 32);
        tc_mma_f16(dt, ad, sdesc_kmajor_sw128(b_addr + kk * 32), idesc,
                   (k > sg.k0 || kk > 0) ? 1u : 0u);
        if (!Cfg::STACKED)
          tc_mma_f16(dt + Cfg::BN, ad, sdesc_kmajor_sw128(b_addr + Cfg::B_HALF + kk * 32), idesc,
                     (k > sg.k0 || kk > 0) ? 1u : 0u);
      }
      tc_commit(&P.empty[st]);
    }
    tc_commit(&P.tfull[acc]);
    if (++acc == Cfg::NACC) {
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

// Before exit: every issued MMA has completed (bounded).
__device__ __forceinline__ void tc_mma_drain(const TcPipe& P) {
  tc_commit(P.drain);
  mbar_wait(P.drain, 0, nullptr);
}

// ---- epilogue (128 threads; r = TMEM lane = weight row of the tile) -------------------

__device__ __forceinline__ void red_release_gpu(int* p, int v) {
  asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Bounded wait until *p >= target (acquire).  On timeout sets *abort.
__device__ inline bool count_wait(const int* p, int target, volatile int* abort) {
  const uint64_t t0 = globaltimer_ns();
  while (static_cast<int>(ld_acquire_gpu(reinterpret_cast<const unsigned*>(p))) < target) {
    if (*abort) return false;
    if (globaltimer_ns() - t0 > kWaitBudgetNs) {
      *abort = 1;
      return false;
    }
    __nanosleep(32);
  }
  return true;
}


// hi + lo accumulator columns of 16 token columns (chunk ch) of this thread's row
template <class Cfg>
__device__ __forceinline__ void tmem_ld_sum_cfg(uint32_t taddr, int ch, int bn, float (&v)[kEpiCols]) {
  tmem_ld16(taddr + ch * kEpiCols, v);
  float vlo[kEpiCols];
  tmem_ld16(taddr + (Cfg::STACKED ? bn : Cfg::BN) + ch * kEpiCols, vlo);
#pragma unroll
  for (int j = 0; j < kEpiCols; ++j) v[j] += vlo[j];
}

// Persistent kernel: publish a finished output tile (its stores are read next
// by other CTAs, some through TMA) on its completion flag.
__device__ __forceinline__ void epi_publish(const EpiArgs& e, int mt, int r) {
  if (e.tile_done == nullptr) return;
  asm volatile("fence.proxy.async.global;" ::: "memory");
  epi_sync();
  if (r == 0) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(e.tile_done + mt) : "memory");
}

// NG = 2 (per-GEMM kernel, 256 token columns): two groups of 4 epilogue warps
// (warps 2-5 and 6-9, each with its own named barrier, EpiSmem and staging
// slots) take alternate 16-column chunks of each unit; a barrier over both
// groups orders their stores before the split-K release, the ticket reset
// and the argmax reduction.  Per column the arithmetic is unchanged.
template <int KIND, class Cfg, int NG = 1>
__device__ bool tc_epilogue(const TcPipe& P, int& acc, uint32_t& accph, const GemmArgs& g,
                            const EpiArgs& e, int c0, int c1, int cta, EpiSmem& es) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = warp & 3;
  const int r = grp * 32 + lane;
  const int gi = NG > 1 ? (warp >= 6 ? 1 : 0) : 0;  // this thread's group
  auto joint = [&]() {
    if constexpr (NG > 1) named_bar_sync(3, 128 * NG);
    else epi_sync();
  };
  const bool tile_mode = g.ntiles > 1;
  if (c0 < c1) epi_prepare<KIND>(e, r, es);
  int c = c0;
  Segment sg;
  while (next_segment(c, c1, g.kchunks, sg)) {
    const int u = sg.unit;
    const int mt = u / g.ntiles, nt = u - mt * g.ntiles;
    EpiPre pre;
    epi_prefetch<KIND, __nv_bfloat16>(e, mt, (tile_mode ? nt * Cfg::BN : 0) + gi * kEpiCols, r, es, pre);
    bool seg_ok;
    if constexpr (NG > 1) {
      // one wait for both groups: a group that returned alone would leave the
      // other at the joint barrier, which has no time limit
      if (gi == 0 && r == 0) P.jflag[1] = mbar_wait(&P.tfull[acc], accph, P.abort) ? 1 : 0;
      joint();
      seg_ok = P.jflag[1] != 0;
      joint();  // read by all before the next unit's wait writes it again
    } else {
      if (r == 0) es.ok = mbar_wait(&P.tfull[acc], accph, P.abort) ? 1 : 0;
      epi_sync();
      seg_ok = es.ok != 0;
      epi_sync();
    }
    if (!seg_ok) return false;
    const bool dbg = e.dbg != nullptr && r == 0 && c >= c1;  // last segment
    if (dbg) e.dbg[cta] = globaltimer_ns();
    tc_fence_after();
    const int first = (u * g.kchunks) / g.cpc;
    const int last = ((u + 1) * g.kchunks - 1) / g.cpc;
    const int nc = last - first + 1;
    const int slot = cta - first;
    const int tbase = tile_mode ? nt * Cfg::BN : 0;
    const int ncols = min(g.bn, e.T - tbase);
    const int nchunk = (ncols + kEpiCols - 1) / kEpiCols;
    const uint32_t taddr = P.tmem + (static_cast<uint32_t>(grp * 32) << 16) +
                           static_cast<uint32_t>(acc * Cfg::ACC_COLS);
    float* mypart = g.partial + (static_cast<size_t>(u) * g.maxc + slot) * g.bn * kBM;
    // Split-K: the unit's contributors are CTAs first..last (slots 0..nc-1).
    // Slot 0 -- for which this unit is the last segment of its range, so it
    // finishes with the phase -- owns the reduction: the others store their
    // partial sums and release a count; the owner waits for nc - 1, then adds
    // the partials to its own accumulator in slot order.
    const bool owner = nc > 1 && slot == 0;
    if (!owner) {
      for (int ch = gi; ch < nchunk; ch += NG) {
        float v[kEpiCols];
        tmem_ld_sum_cfg<Cfg>(taddr, ch, g.bn, v);
        if (nc == 1) {
          epi_apply<KIND, __nv_bfloat16>(e, mt, tbase + ch * kEpiCols, v, r, es, &pre);
        } else {
#pragma unroll
          for (int j = 0; j < kEpiCols; ++j) mypart[(ch * kEpiCols + j) * kBM + r] = v[j];
        }
      }
      if (nc == 1) epi_publish(e, mt, r);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&P.tempty[acc]);
      if (nc > 1) {
        joint();  // every thread's partial stores precede the release
        if (gi == 0 && r == 0) red_release_gpu(&g.tickets[u], 1);
        if (dbg) e.dbg[e.dbg_stride + cta] = globaltimer_ns();
      } else if (KIND == EPI_ARGMAX) {
        if constexpr (NG > 1) joint();  // both groups' partial maxima are written
        if (gi == 0) epi_argmax_finish(e, r, es);
      }
    } else {
      bool got;
      if constexpr (NG > 1) {
        // one wait for both groups, so that they agree on its outcome
        if (gi == 0 && r == 0) *P.jflag = count_wait(&g.tickets[u], nc - 1, P.abort) ? 1 : 0;
        joint();
        got = *P.jflag != 0;
      } else {
        if (r == 0) es.ok = count_wait(&g.tickets[u], nc - 1, P.abort) ? 1 : 0;
        epi_sync();
        got = es.ok != 0;
        epi_sync();
      }
      if (!got) {
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&P.tempty[acc]);
        return false;
      }
      if (dbg) e.dbg[e.dbg_stride + cta] = globaltimer_ns();
      for (int ch = gi; ch < nchunk; ch += NG) {
        float v[kEpiCols];
        tmem_ld_sum_cfg<Cfg>(taddr, ch, g.bn, v);
        // slots 1..nc-1: a group of up to red_slots partial blocks
        // (kEpiCols x kBM contiguous floats each) is copied to shared memory
        // by all 128 threads at once (cp.async at L2, no registers held),
        // then each thread adds its row
        for (int s0 = 1; s0 < nc; s0 += P.red_slots) {
          const int ns = min(P.red_slots, nc - s0);
          for (int q = 0; q < ns; ++q) {
            const float* src = g.partial + (static_cast<size_t>(u) * g.maxc + s0 + q) * g.bn * kBM +
                               static_cast<size_t>(ch) * kEpiCols * kBM;
            float* dst = P.red + q * (kEpiCols * kBM);
#pragma unroll
            for (int i = 0; i < kEpiCols * kBM / (4 * 128); ++i)
              cp_async16(dst + 4 * (i * 128 + r), src + 4 * (i * 128 + r));
          }
          cp_async_commit();
          // the chunk's own epilogue inputs travel in the same round trip
          if (ch > gi && s0 == 1)
            epi_prefetch<KIND, __nv_bfloat16>(e, mt, tbase + ch * kEpiCols, r, es, pre);
          cp_async_wait_all();
          epi_sync();
          for (int q = 0; q < ns; ++q) {
            const float* blk = P.red + q * (kEpiCols * kBM);
#pragma unroll
            for (int j = 0; j < kEpiCols; ++j) v[j] += blk[j * kBM + r];
          }
          epi_sync();
        }
        if (dbg && ch == 0) e.dbg[4 * e.dbg_stride + cta] = globaltimer_ns();
        epi_apply<KIND, __nv_bfloat16>(e, mt, tbase + ch * kEpiCols, v, r, es, &pre);
      }
      // (the count is reset before the tile is published: a later phase that
      // the flag opens may count on the same ticket)
      if constexpr (NG > 1) joint();  // both groups are past the wait and done
      if (gi == 0 && r == 0) g.tickets[u] = 0;
      epi_publish(e, mt, r);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&P.tempty[acc]);
      if (KIND == EPI_ARGMAX && gi == 0) epi_argmax_finish(e, r, es);
    }
    if (dbg) e.dbg[2 * e.dbg_stride + cta] = globaltimer_ns();
    if (++acc == Cfg::NACC) {
      acc = 0;
      accph ^= 1;
    }
  }
  return true;
}

}  // namespace cllm
