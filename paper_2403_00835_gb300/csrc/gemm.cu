// Weight-streaming GEMMs of the block forward, with fused epilogues.
//
//   D[m][t] = sum_k W[m][k] * X[t][k]      (W: [M][K] weights, X: [T][K] activations)
//
// At the small token counts of a Jacobi step (T = batch * n <= 256) every
// weight byte is used T times, so the GEMMs are bound by streaming W from
// HBM.  The bf16 kernel is "swap-AB": the weight tile is the MMA's A operand
// (M = 128 rows), the tokens are its N (16..256 columns), and the fp32
// accumulator lives in tensor memory (TMEM).  A producer warp streams W and X
// tiles with TMA into a ring of shared-memory stages, one thread issues
// tcgen05.mma, and four epilogue warps read TMEM.  The grid is one CTA per SM;
// the (tile, k-chunk) space is cut into equal contiguous ranges, so a tile
// whose K range is split over several CTAs is finished by the last one to
// arrive (atomic ticket, no waiting), which sums the partial tiles in a fixed
// order.  The partition depends only on the weight shape and SM count, never
// on T, so a token's result does not depend on how many rows share the launch.
//
// Fused epilogues (each reads the RMSNorm statistics its producer left):
//   EPI_QKV    : x rms-scale, rotate-half RoPE, Q -> scratch, K/V -> cache
//   EPI_GATEUP : x rms-scale, silu(gate) * up -> h
//   EPI_RESID  : residual add into the fp32 stream, next norm's input and
//                per-tile sum of squares
//   EPI_ARGMAX : x rms-scale, per-tile (max, argmax, 2nd max) of the logits;
//                the last tile to finish reduces them to argmax and top-2 gap
#include <float.h>
#include <limits.h>

#include "act.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace cllm {

// ---------------------------------------------------------------------------------
// Epilogues.  128 threads; thread r owns weight row r of the tile and 16
// consecutive token columns t0..t0+15.  Named barrier 1 syncs the 128 threads.
// ---------------------------------------------------------------------------------

struct EpiSmem {
  float x[kEpiCols][kBM + 1];
  float rs[kEpiCols];
  float red[4][kEpiCols];
  float am[4][kEpiCols][3];
  int flag;
  int ok;
};

__device__ __forceinline__ void epi_sync() { named_bar_sync(1, 128); }

__device__ __forceinline__ void epi_norm_scale(const EpiArgs& e, int t0, int r, EpiSmem& s) {
  if (r < kEpiCols) {
    const int t = t0 + r;
    float rs = 0.f;
    if (t < e.T) {
      float acc = 0.f;
      for (int i = 0; i < e.ssq_tiles; ++i) acc += e.ssq_in[static_cast<size_t>(i) * e.ldt + t];
      rs = rsqrtf(acc * e.inv_d + e.eps);
    }
    s.rs[r] = rs;
  }
  epi_sync();
}

// (max, argmax with lowest index on ties, second max) merge
__device__ __forceinline__ void am_merge(float& v1, int& i1, float& v2, float w1, int j1, float w2) {
  const bool other_hi = (w1 > v1) || (w1 == v1 && j1 < i1);
  if (other_hi) {
    v2 = fmaxf(w2, v1);
    v1 = w1;
    i1 = j1;
  } else {
    v2 = fmaxf(v2, w1);
  }
}

template <int KIND, typename Act>
__device__ void epi_apply(const EpiArgs& e, int mt, int t0, float (&v)[kEpiCols], int r,
                          EpiSmem& s) {
  const int lane = r & 31, grp = r >> 5;
  if (KIND == EPI_QKV) {
    epi_norm_scale(e, t0, r, s);
    const int m = mt * kBM + r;
    const int sec = (m < e.dq) ? 0 : (m < e.dq + e.dkv ? 1 : 2);  // uniform over the tile
    const int ms = m - (sec == 0 ? 0 : (sec == 1 ? e.dq : e.dq + e.dkv));
    const int head = ms / e.hd, i = ms - head * e.hd, half = e.hd >> 1;
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) v[j] *= s.rs[j];
    if (sec < 2) {
#pragma unroll
      for (int j = 0; j < kEpiCols; ++j) s.x[j][r] = v[j];
      epi_sync();
      const int rp = (i < half) ? r + half : r - half;
      const int fi = (i < half) ? i : i - half;
#pragma unroll
      for (int j = 0; j < kEpiCols; ++j) {
        const int t = t0 + j;
        if (t < e.T) {
          const int p = min(e.pos[t], e.max_seq - 1);
          const float2 cs = e.rope[static_cast<size_t>(p) * half + fi];
          const float pv = s.x[j][rp];
          v[j] = (i < half) ? (v[j] * cs.x - pv * cs.y) : (v[j] * cs.x + pv * cs.y);
        }
      }
      epi_sync();
    }
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      const int t = t0 + j;
      if (t >= e.T) continue;
      using AT = typename AttnType<Act>::T;
      if (sec == 0) {
        st_act(reinterpret_cast<AT*>(e.q_out), static_cast<size_t>(t) * e.dq + m, v[j]);
      } else {
        const int p = e.pos[t], b = e.bidx[t];
        if (p < 0 || p >= e.max_seq) {
          atomicOr(e.err, DERR_CAPACITY);
          continue;
        }
        const size_t off =
            ((static_cast<size_t>(b) * e.n_kv_heads + head) * e.max_seq + p) * e.hd + i;
        st_act(reinterpret_cast<AT*>(sec == 1 ? e.k_cache : e.v_cache), off, v[j]);
      }
    }
  } else if (KIND == EPI_GATEUP) {
    epi_norm_scale(e, t0, r, s);
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      v[j] *= s.rs[j];
      s.x[j][r] = v[j];
    }
    epi_sync();
    if (r < 64) {
      const int f = mt * 64 + r;
      if (f < e.F) {
#pragma unroll
        for (int j = 0; j < kEpiCols; ++j) {
          const int t = t0 + j;
          if (t < e.T) {
            const float gt = v[j], up = s.x[j][r + 64];
            st_gin(reinterpret_cast<Act*>(e.h_out), static_cast<size_t>(t) * e.F + f, e.plane_h,
                   gt / (1.f + expf(-gt)) * up);
          }
        }
      }
    }
    epi_sync();
  } else if (KIND == EPI_RESID) {
    const int m = mt * kBM + r;
    const float gn = ld_act(reinterpret_cast<const Act*>(e.gnext), m);
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      const int t = t0 + j;
      float sq = 0.f;
      if (t < e.T) {
        const size_t o = static_cast<size_t>(t) * e.d + m;
        const float xi = e.x[o] + v[j];
        e.x[o] = xi;
        st_gin(reinterpret_cast<Act*>(e.xg), o, e.plane_x, xi * gn);
        sq = xi * xi;
      }
      sq = warp_sum(sq);
      if (lane == 0) s.red[grp][j] = sq;
    }
    epi_sync();
    if (r < kEpiCols) {
      const int t = t0 + r;
      if (t < e.T)
        e.ssq_out[static_cast<size_t>(mt) * e.ldt + t] =
            ((s.red[0][r] + s.red[1][r]) + s.red[2][r]) + s.red[3][r];
    }
    epi_sync();
  } else {  // EPI_ARGMAX
    epi_norm_scale(e, t0, r, s);
    const int m = mt * kBM + r;
    const bool vrow = m < e.V;
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      const int t = t0 + j;
      const float lg = v[j] * s.rs[j];
      if (e.logits != nullptr && t < e.T && vrow) e.logits[static_cast<size_t>(t) * e.V + m] = lg;
      float v1 = vrow ? lg : -INFINITY, v2 = -INFINITY;
      int i1 = m;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float w1 = __shfl_xor_sync(0xffffffffu, v1, o);
        const int j1 = __shfl_xor_sync(0xffffffffu, i1, o);
        const float w2 = __shfl_xor_sync(0xffffffffu, v2, o);
        am_merge(v1, i1, v2, w1, j1, w2);
      }
      if (lane == 0) {
        s.am[grp][j][0] = v1;
        s.am[grp][j][1] = __int_as_float(i1);
        s.am[grp][j][2] = v2;
      }
    }
    epi_sync();
    if (r < kEpiCols) {
      const int t = t0 + r;
      if (t < e.T) {
        float v1 = s.am[0][r][0], v2 = s.am[0][r][2];
        int i1 = __float_as_int(s.am[0][r][1]);
        for (int gq = 1; gq < 4; ++gq)
          am_merge(v1, i1, v2, s.am[gq][r][0], __float_as_int(s.am[gq][r][1]), s.am[gq][r][2]);
        float* dst = e.am_part + (static_cast<size_t>(mt) * e.ldt + t) * 3;
        dst[0] = v1;
        dst[1] = __int_as_float(i1);
        dst[2] = v2;
      }
    }
    epi_sync();
  }
}

// After a unit's argmax partials are written: the last unit of the launch to
// finish reduces all tiles to pred[t] (argmax, lowest index on ties) and
// gap[t] = top1 - top2.  The merge is exact, so the order does not matter.
__device__ void epi_argmax_finish(const EpiArgs& e, int r, EpiSmem& s) {
  __threadfence();
  epi_sync();
  if (r == 0) {
    const int old = atomicAdd(e.am_ticket, 1);
    s.flag = (old == e.am_units - 1);
  }
  epi_sync();
  const bool last = s.flag;
  epi_sync();
  if (!last) return;
  __threadfence();
  for (int tb = 0; tb < e.T; tb += 16) {
    const int t = tb + (r >> 3), part = r & 7;
    float v1 = -INFINITY, v2 = -INFINITY;
    int i1 = INT_MAX;
    if (t < e.T) {
      for (int mt = part; mt < e.am_mtiles; mt += 8) {
        const float* p = e.am_part + (static_cast<size_t>(mt) * e.ldt + t) * 3;
        am_merge(v1, i1, v2, __ldcg(p), __float_as_int(__ldcg(p + 1)), __ldcg(p + 2));
      }
    }
#pragma unroll
    for (int o = 1; o < 8; o <<= 1) {
      const float w1 = __shfl_xor_sync(0xffffffffu, v1, o);
      const int j1 = __shfl_xor_sync(0xffffffffu, i1, o);
      const float w2 = __shfl_xor_sync(0xffffffffu, v2, o);
      am_merge(v1, i1, v2, w1, j1, w2);
    }
    if (part == 0 && t < e.T) {
      e.pred[t] = i1;
      e.gap[t] = v1 - v2;
    }
  }
  if (r == 0) *e.am_ticket = 0;
}

// ---------------------------------------------------------------------------------
// tcgen05 kernel (bf16)
// ---------------------------------------------------------------------------------

// Stage = one 128 x 64 weight tile + the hi and lo planes of a BNMAX x 64
// activation tile.  One CTA per SM with as many stages as fit: the weight
// stream is latency-bound by the bytes in flight per SM (~45 GB/s per SM at
// ~1.8 us loaded DRAM latency needs > 80 KB in flight).
template <int BNMAX>
struct TcCfg {
  static constexpr int STAGES = BNMAX <= 32 ? 8 : (BNMAX <= 64 ? 6 : (BNMAX <= 128 ? 4 : 2));
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
  static constexpr size_t BAR_BYTES = 8 * (2 * STAGES + 5) + 16;
  static constexpr size_t SMEM =
      1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + sizeof(EpiSmem) + 16 + BAR_BYTES;
};

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

template <int KIND, int BNMAX>
__global__ void __launch_bounds__(192, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mA1,
                   const __grid_constant__ CUtensorMap mA2, const __grid_constant__ CUtensorMap mB,
                   const GemmArgs g, const EpiArgs e) {
  using Cfg = TcCfg<BNMAX>;
  constexpr int S = Cfg::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base =
      reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = base;
  uint8_t* sB = base + S * Cfg::A_BYTES;
  EpiSmem& es = *reinterpret_cast<EpiSmem*>(base + S * Cfg::STAGE_BYTES);
  uint64_t* bars = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(&es + 1) + 15) & ~uintptr_t(15));
  uint64_t* full = bars;
  uint64_t* empty = bars + S;
  uint64_t* tfull = bars + 2 * S;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull[i], 1);
      mbar_init(&tempty[i], 4);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mA0);
    tma_prefetch_desc(&mA1);
    tma_prefetch_desc(&mA2);
    tma_prefetch_desc(&mB);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, Cfg::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // Every CTA of this grid is resident (one per SM): let the next kernel in
  // the stream start its independent prologue (weight prefetch) now.
  pdl_launch_dependents();

  const int total = g.mtiles * g.ntiles * g.kchunks;
  const int c0 = blockIdx.x * g.cpc;
  const int c1 = min(total, c0 + g.cpc);
  const bool tile_mode = g.ntiles > 1;
  const uint32_t b_bytes = 2u * static_cast<uint32_t>(g.bn) * kBK * 2;

  if (warp == 0) {
    if (lane == 0 && c0 < c1) {
      // ---------------- TMA producer ----------------
      const uint64_t pol_w = l2_policy_evict_first();
      const uint64_t pol_x = l2_policy_evict_last();
      const int nchunks = c1 - c0;
      auto unit_of = [&](int c) { return c / g.kchunks; };
      auto load_a = [&](int idx) {
        const int c = c0 + idx;
        const int u = unit_of(c), k = c - u * g.kchunks;
        const int mt = u / g.ntiles;
        const int st = idx % S;
        uint8_t* dst = sA + st * Cfg::A_BYTES;
        if (KIND == EPI_GATEUP) {
          tma_load_2d(dst, &mA0, &full[st], k * kBK, mt * 64, pol_w);
          tma_load_2d(dst + Cfg::A_BYTES / 2, &mA1, &full[st], k * kBK, mt * 64, pol_w);
        } else if (KIND == EPI_QKV) {
          const int row = mt * kBM;
          if (row < g.rows_q)
            tma_load_2d(dst, &mA0, &full[st], k * kBK, row, pol_w);
          else if (row < g.rows_qk)
            tma_load_2d(dst, &mA1, &full[st], k * kBK, row - g.rows_q, pol_w);
          else
            tma_load_2d(dst, &mA2, &full[st], k * kBK, row - g.rows_qk, pol_w);
        } else {
          tma_load_2d(dst, &mA0, &full[st], k * kBK, mt * kBM, pol_w);
        }
      };
      auto load_b = [&](int idx) {
        const int c = c0 + idx;
        const int u = unit_of(c), k = c - u * g.kchunks;
        const int nt = u % g.ntiles;
        const int st = idx % S;
        const int row0 = tile_mode ? nt * BNMAX : 0;
        uint8_t* dst = sB + st * Cfg::B_BYTES;
        tma_load_2d(dst, &mB, &full[st], k * kBK, row0, pol_x);
        tma_load_2d(dst + (Cfg::STACKED ? g.bn * kBK * 2 : Cfg::B_HALF), &mB, &full[st], k * kBK,
                    g.lo_rows + row0, pol_x);
      };
      // Weights do not depend on earlier kernels: start streaming them before
      // waiting for the previous kernel (programmatic dependent launch) --
      // the first S tiles into shared memory, the next g.l2_ahead into L2.
      const int pre = min(S, nchunks);
      for (int idx = 0; idx < pre; ++idx) {
        mbar_arrive_expect_tx(&full[idx], Cfg::A_BYTES + b_bytes);
        load_a(idx);
      }
      for (int idx = pre; idx < min(nchunks, pre + g.l2_ahead); ++idx) {
        const int c = c0 + idx;
        const int u = unit_of(c), k = c - u * g.kchunks;
        const int mt = u / g.ntiles;
        if (KIND == EPI_GATEUP) {
          tma_prefetch_l2_2d(&mA0, k * kBK, mt * 64);
          tma_prefetch_l2_2d(&mA1, k * kBK, mt * 64);
        } else if (KIND == EPI_QKV) {
          const int row = mt * kBM;
          if (row < g.rows_q)
            tma_prefetch_l2_2d(&mA0, k * kBK, row);
          else if (row < g.rows_qk)
            tma_prefetch_l2_2d(&mA1, k * kBK, row - g.rows_q);
          else
            tma_prefetch_l2_2d(&mA2, k * kBK, row - g.rows_qk);
        } else {
          tma_prefetch_l2_2d(&mA0, k * kBK, mt * kBM);
        }
      }
      pdl_wait();
      for (int idx = 0; idx < pre; ++idx) load_b(idx);
      int issued = pre;
      for (int idx = pre; idx < nchunks; ++idx) {
        const int st = idx % S;
        const uint32_t ph = ((idx / S) & 1) ^ 1;
        if (!mbar_wait(&empty[st], ph, abort_flag)) break;
        mbar_arrive_expect_tx(&full[st], Cfg::A_BYTES + b_bytes);
        load_a(idx);
        load_b(idx);
        issued = idx + 1;
      }
      // Drain: every issued copy has landed before the CTA may exit.
      for (int idx = max(0, issued - S); idx < issued; ++idx) {
        const int st = idx % S;
        mbar_wait(&full[st], (idx / S) & 1, nullptr);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && c0 < c1) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = idesc_bf16_f32(kBM, Cfg::STACKED ? 2 * g.bn : g.bn);
      int c = c0, idx = 0, acc = 0;
      uint32_t accph = 0;
      Segment sg;
      bool ok = true;
      while (ok && next_segment(c, c1, g.kchunks, sg)) {
        if (!mbar_wait(&tempty[acc], accph ^ 1, abort_flag)) break;
        tc_fence_after();
        const uint32_t dt = tmem + static_cast<uint32_t>(acc * Cfg::ACC_COLS);
        for (int k = sg.k0; k < sg.k1; ++k, ++idx) {
          const int st = idx % S;
          if (!mbar_wait(&full[st], (idx / S) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a_addr = smem_u32(sA + st * Cfg::A_BYTES);
          const uint32_t b_addr = smem_u32(sB + st * Cfg::B_BYTES);
#pragma unroll
          for (int kk = 0; kk < kBK / 16; ++kk) {
            const uint64_t ad = sdesc_kmajor_sw128(a_addr + kk * 32);
            tc_mma_f16(dt, ad, sdesc_kmajor_sw128(b_addr + kk * 32), idesc,
                       (k > sg.k0 || kk > 0) ? 1u : 0u);
            if (!Cfg::STACKED)
              tc_mma_f16(dt + BNMAX, ad, sdesc_kmajor_sw128(b_addr + Cfg::B_HALF + kk * 32), idesc,
                         (k > sg.k0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(&empty[st]);
        }
        if (!ok) break;
        tc_commit(&tfull[acc]);
        if (++acc == Cfg::NACC) {
          acc = 0;
          accph ^= 1;
        }
      }
      // Every issued MMA has completed before TMEM is released.
      tc_commit(drain);
      mbar_wait(drain, 0, nullptr);
    }
  } else {
    // ---------------- epilogue (warps 2..5) ----------------
    pdl_wait();
    const int grp = warp & 3;
    const int r = grp * 32 + lane;
    int c = c0, acc = 0;
    uint32_t accph = 0;
    Segment sg;
    while (next_segment(c, c1, g.kchunks, sg)) {
      const int u = sg.unit;
      const int mt = u / g.ntiles, nt = u - mt * g.ntiles;
      if (r == 0) es.ok = mbar_wait(&tfull[acc], accph, abort_flag) ? 1 : 0;
      epi_sync();
      const bool seg_ok = es.ok != 0;
      epi_sync();
      if (!seg_ok) break;
      tc_fence_after();
      const int first = (u * g.kchunks) / g.cpc;
      const int last = ((u + 1) * g.kchunks - 1) / g.cpc;
      const int nc = last - first + 1;
      const int slot = blockIdx.x - first;
      const int tbase = tile_mode ? nt * BNMAX : 0;
      const int ncols = min(g.bn, e.T - tbase);
      const int nchunk = (ncols + kEpiCols - 1) / kEpiCols;
      const uint32_t taddr =
          tmem + (static_cast<uint32_t>(grp * 32) << 16) + static_cast<uint32_t>(acc * Cfg::ACC_COLS);
      float* mypart = g.partial + (static_cast<size_t>(u) * g.maxc + slot) * g.bn * kBM;
      for (int ch = 0; ch < nchunk; ++ch) {
        float v[kEpiCols];
        tmem_ld16(taddr + ch * kEpiCols, v);
        {
          float vlo[kEpiCols];
          tmem_ld16(taddr + (Cfg::STACKED ? g.bn : BNMAX) + ch * kEpiCols, vlo);
#pragma unroll
          for (int j = 0; j < kEpiCols; ++j) v[j] += vlo[j];
        }
        if (nc == 1) {
          epi_apply<KIND, __nv_bfloat16>(e, mt, tbase + ch * kEpiCols, v, r, es);
        } else {
#pragma unroll
          for (int j = 0; j < kEpiCols; ++j) mypart[(ch * kEpiCols + j) * kBM + r] = v[j];
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      if (nc > 1) {
        __threadfence();
        epi_sync();
        if (r == 0) {
          const int old = atomicAdd(&g.tickets[u], 1);
          es.flag = (old == nc - 1);
        }
        epi_sync();
        const bool last_arrival = es.flag;
        epi_sync();
        if (last_arrival) {
          __threadfence();
          for (int ch = 0; ch < nchunk; ++ch) {
            float v[kEpiCols];
#pragma unroll
            for (int j = 0; j < kEpiCols; ++j) v[j] = 0.f;
            for (int s = 0; s < nc; ++s) {
              const float* p = g.partial + (static_cast<size_t>(u) * g.maxc + s) * g.bn * kBM;
#pragma unroll
              for (int j = 0; j < kEpiCols; ++j) v[j] += __ldcg(p + (ch * kEpiCols + j) * kBM + r);
            }
            epi_apply<KIND, __nv_bfloat16>(e, mt, tbase + ch * kEpiCols, v, r, es);
          }
          if (r == 0) g.tickets[u] = 0;
          if (KIND == EPI_ARGMAX) epi_argmax_finish(e, r, es);
        }
      } else if (KIND == EPI_ARGMAX) {
        epi_argmax_finish(e, r, es);
      }
      if (++acc == Cfg::NACC) {
        acc = 0;
        accph ^= 1;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::TMEM_COLS);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(g.err, DERR_TIMEOUT);
}

// ---------------------------------------------------------------------------------
// SIMT kernel (fp32 weights and activations; the fp32 parity configuration)
// One CTA computes a 128-row x 16-token tile over the full K, then runs the
// same epilogue.
// ---------------------------------------------------------------------------------

template <int KIND>
__global__ void __launch_bounds__(128) gemm_simt_kernel(const GemmArgs g, const EpiArgs e) {
  __shared__ float xs[kEpiCols][kBK + 1];
  __shared__ EpiSmem es;
  pdl_launch_dependents();
  pdl_wait();
  const int mt = blockIdx.x, nt = blockIdx.y, r = threadIdx.x;
  const int t0 = nt * kEpiCols;
  const float* W;
  int row;
  bool vrow;
  if (KIND == EPI_GATEUP) {
    W = static_cast<const float*>(r < 64 ? g.A0 : g.A1);
    row = mt * 64 + (r & 63);
    vrow = row < g.M;
  } else if (KIND == EPI_QKV) {
    const int m = mt * kBM + r;
    if (m < g.rows_q) {
      W = static_cast<const float*>(g.A0);
      row = m;
    } else if (m < g.rows_qk) {
      W = static_cast<const float*>(g.A1);
      row = m - g.rows_q;
    } else {
      W = static_cast<const float*>(g.A2);
      row = m - g.rows_qk;
    }
    vrow = m < g.M;
  } else {
    W = static_cast<const float*>(g.A0);
    row = mt * kBM + r;
    vrow = row < g.M;
  }
  const float* X = static_cast<const float*>(g.X);
  float acc[kEpiCols];
#pragma unroll
  for (int j = 0; j < kEpiCols; ++j) acc[j] = 0.f;
  for (int k0 = 0; k0 < g.K; k0 += kBK) {
    for (int i = r; i < kEpiCols * kBK; i += 128) {
      const int j = i / kBK, kk = i - j * kBK;
      const int t = t0 + j, k = k0 + kk;
      xs[j][kk] = (t < g.T && k < g.K) ? X[static_cast<size_t>(t) * g.ldx + k] : 0.f;
    }
    __syncthreads();
    if (vrow) {
      const int kend = min(kBK, g.K - k0);
      const float* wr = W + static_cast<size_t>(row) * g.K + k0;
      for (int kk = 0; kk < kend; ++kk) {
        const float w = wr[kk];
#pragma unroll
        for (int j = 0; j < kEpiCols; ++j) acc[j] = fmaf(w, xs[j][kk], acc[j]);
      }
    }
    __syncthreads();
  }
  epi_apply<KIND, float>(e, mt, t0, acc, r, es);
  if (KIND == EPI_ARGMAX) epi_argmax_finish(e, r, es);
}

// ---------------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------------

int gemm_tc_stages(int bn_max) {
  switch (bn_max) {
    case 32: return TcCfg<32>::STAGES;
    case 64: return TcCfg<64>::STAGES;
    case 128: return TcCfg<128>::STAGES;
    default: return TcCfg<256>::STAGES;
  }
}

size_t gemm_tc_smem_bytes(int bn_max) {
  switch (bn_max) {
    case 32: return TcCfg<32>::SMEM;
    case 64: return TcCfg<64>::SMEM;
    case 128: return TcCfg<128>::SMEM;
    default: return TcCfg<256>::SMEM;
  }
}

template <int KIND, int BN>
static cudaError_t set_attr_one() {
  cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<KIND, BN>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(TcCfg<BN>::SMEM));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(gemm_tc_kernel<KIND, BN>,
                              cudaFuncAttributePreferredSharedMemoryCarveout,
                              static_cast<int>(cudaSharedmemCarveoutMaxShared));
}

template <int KIND>
static cudaError_t set_attr_kind() {
  cudaError_t err;
  if ((err = set_attr_one<KIND, 32>()) != cudaSuccess) return err;
  if ((err = set_attr_one<KIND, 64>()) != cudaSuccess) return err;
  if ((err = set_attr_one<KIND, 128>()) != cudaSuccess) return err;
  return set_attr_one<KIND, 256>();
}

cudaError_t gemm_tc_set_attributes() {
  cudaError_t err;
  if ((err = set_attr_kind<EPI_QKV>()) != cudaSuccess) return err;
  if ((err = set_attr_kind<EPI_GATEUP>()) != cudaSuccess) return err;
  if ((err = set_attr_kind<EPI_RESID>()) != cudaSuccess) return err;
  return set_attr_kind<EPI_ARGMAX>();
}

static void fill_launch(cudaLaunchConfig_t& cfg, cudaLaunchAttribute* attr, dim3 grid, dim3 block,
                        size_t smem, cudaStream_t s, bool pdl) {
  cfg = cudaLaunchConfig_t{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
}

template <int KIND, int BN>
static cudaError_t launch_tc_one(const GemmMaps& m, const GemmArgs& g, const EpiArgs& e, int grid,
                                 cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  fill_launch(cfg, attr, dim3(grid), dim3(192), TcCfg<BN>::SMEM, s, pdl);
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<KIND, BN>, m.a0, m.a1, m.a2, m.b, g, e);
}

template <int KIND>
static cudaError_t launch_tc_kind(int bn_max, const GemmMaps& m, const GemmArgs& g,
                                  const EpiArgs& e, int grid, cudaStream_t s, bool pdl) {
  switch (bn_max) {
    case 32: return launch_tc_one<KIND, 32>(m, g, e, grid, s, pdl);
    case 64: return launch_tc_one<KIND, 64>(m, g, e, grid, s, pdl);
    case 128: return launch_tc_one<KIND, 128>(m, g, e, grid, s, pdl);
    case 256: return launch_tc_one<KIND, 256>(m, g, e, grid, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_gemm_tc(int kind, int bn_max, const GemmMaps& maps, const GemmArgs& g,
                           const EpiArgs& e, int grid, cudaStream_t s, bool pdl) {
  switch (kind) {
    case EPI_QKV: return launch_tc_kind<EPI_QKV>(bn_max, maps, g, e, grid, s, pdl);
    case EPI_GATEUP: return launch_tc_kind<EPI_GATEUP>(bn_max, maps, g, e, grid, s, pdl);
    case EPI_RESID: return launch_tc_kind<EPI_RESID>(bn_max, maps, g, e, grid, s, pdl);
    case EPI_ARGMAX: return launch_tc_kind<EPI_ARGMAX>(bn_max, maps, g, e, grid, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

template <int KIND>
static cudaError_t launch_simt_one(const GemmArgs& g, const EpiArgs& e, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  fill_launch(cfg, attr, dim3(g.mtiles, g.ntiles), dim3(128), 0, s, pdl);
  return cudaLaunchKernelEx(&cfg, gemm_simt_kernel<KIND>, g, e);
}

cudaError_t launch_gemm_simt(int kind, const GemmArgs& g, const EpiArgs& e, cudaStream_t s,
                             bool pdl) {
  switch (kind) {
    case EPI_QKV: return launch_simt_one<EPI_QKV>(g, e, s, pdl);
    case EPI_GATEUP: return launch_simt_one<EPI_GATEUP>(g, e, s, pdl);
    case EPI_RESID: return launch_simt_one<EPI_RESID>(g, e, s, pdl);
    case EPI_ARGMAX: return launch_simt_one<EPI_ARGMAX>(g, e, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace cllm
