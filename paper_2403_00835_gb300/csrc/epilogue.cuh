// Fused epilogues of the weight-streaming GEMMs (shared by the per-GEMM kernels
// and the persistent per-iteration kernel).
//   EPI_QKV    : x rms-scale, rotate-half RoPE, Q -> scratch, K/V -> cache
//   EPI_GATEUP : x rms-scale, silu(gate) * up -> h
//   EPI_RESID  : residual add into the fp32 stream, next norm's input and
//                per-tile sum of squares
//   EPI_ARGMAX : x rms-scale, per-tile (max, argmax, 2nd max) of the logits;
//                the last tile to finish reduces them to argmax and top-2 gap
#pragma once
#include <type_traits>
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

// Columns whose per-token epilogue inputs (RMSNorm scale, position, sequence)
// are prepared once per launch / phase (launches with more tokens prepare them
// per 16-column chunk).
constexpr int kEpiPrepMax = 256;

struct EpiSmem {
  float x[kEpiCols][kBM + 1];
  float rs[kEpiCols];
  float red[4][kEpiCols];
  float am[4][kEpiCols][3];
  int flag;
  int ok;
  int prepared;  // rs_all / pos_all / bidx_all hold this launch's columns
  float rs_all[kEpiPrepMax];
  int pos_all[kEpiPrepMax];
  int bidx_all[kEpiPrepMax];
};

// Barrier of the thread's group of 4 epilogue warps: named barrier 1; in a
// translation unit that defines CLLM_EPI_GROUPS (kernels with a second group
// in warps 6-9), named barrier 2 for that group.
#ifdef CLLM_EPI_GROUPS
__device__ __forceinline__ void epi_sync() { named_bar_sync((threadIdx.x >> 5) >= 6 ? 2 : 1, 128); }
#else
__device__ __forceinline__ void epi_sync() { named_bar_sync(1, 128); }
#endif

// rs[t] = 1 / sqrt(sum of the per-tile sums of squares / d + eps) for the 16
// columns t0..t0+15: 8 threads per column each sum the tiles i = part (mod 8)
// in order, then a fixed shuffle tree adds the 8 parts (every load of the
// column is in flight at once; the order does not depend on the launch).
// Sum of column t's per-tile squares by the 8 threads part = 0..7 (tiles
// part, part + 8, ... in order) followed by a fixed shuffle tree.
__device__ __forceinline__ float epi_ssq_column(const EpiArgs& e, int t, int part, bool valid) {
  float acc = 0.f;
  if (valid) {
    float v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const int i = part + 8 * u;
      v[u] = i < e.ssq_tiles ? __ldcg(e.ssq_in + static_cast<size_t>(i) * e.ldt + t) : 0.f;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) acc += v[u];
    for (int i = part + 64; i < e.ssq_tiles; i += 8) acc += __ldcg(e.ssq_in + static_cast<size_t>(i) * e.ldt + t);
  }
  acc += __shfl_xor_sync(0xffffffffu, acc, 1);
  acc += __shfl_xor_sync(0xffffffffu, acc, 2);
  acc += __shfl_xor_sync(0xffffffffu, acc, 4);
  return acc;
}

// Once per launch / phase, before the first accumulator is ready: the RMSNorm
// scale (kinds that need it), position and sequence index of every column.
template <int KIND>
__device__ void epi_prepare(const EpiArgs& e, int r, EpiSmem& s) {
  s.prepared = 0;
  if (e.T > kEpiPrepMax) {
    epi_sync();
    return;
  }
  if (KIND != EPI_RESID) {
    const int col = r >> 3, part = r & 7;
    for (int t0 = 0; t0 < e.T; t0 += kEpiCols) {
      const int t = t0 + col;
      const float acc = epi_ssq_column(e, t, part, t < e.T);
      if (part == 0 && t < e.T) s.rs_all[t] = rsqrtf(acc * e.inv_d + e.eps);
    }
  }
  if (KIND == EPI_QKV) {
    for (int t = r; t < e.T; t += 128) {
      s.pos_all[t] = e.pos[t];
      s.bidx_all[t] = e.bidx[t];
    }
  }
  if (r == 0) s.prepared = 1;
  epi_sync();
}

__device__ __forceinline__ void epi_norm_scale(const EpiArgs& e, int t0, int r, EpiSmem& s) {
  if (s.prepared) {
    if (r < kEpiCols) s.rs[r] = (t0 + r < e.T) ? s.rs_all[t0 + r] : 0.f;
    epi_sync();
    return;
  }
  const int col = r >> 3, part = r & 7;
  const int t = t0 + col;
  const float acc = epi_ssq_column(e, t, part, t < e.T);
  if (part == 0) s.rs[col] = (t < e.T) ? rsqrtf(acc * e.inv_d + e.eps) : 0.f;
  epi_sync();
}

// Arrival ticket of the last-arriver pattern: one thread, after a barrier of
// the 128 epilogue threads; release of the CTA's prior writes (cumulative
// over the barrier) and acquire of the earlier arrivals' writes.
__device__ __forceinline__ int ticket_add(int* p, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// Column sums of a warp: every lane holds one value per column (16 columns);
// the result for column c = lane >> 1 ends in lanes 2c and 2c + 1.  Halving
// exchanges (16 shuffles in 5 independent rounds) instead of 16 separate
// 5-shuffle trees; the association order is fixed.
__device__ __forceinline__ float warp_colsum16(const float (&v)[kEpiCols], int lane) {
  static_assert(kEpiCols == 16, "16 columns");
  float a[8], b[4], c[2];
  const bool h16 = lane & 16, h8 = lane & 8, h4 = lane & 4, h2 = lane & 2;
#pragma unroll
  for (int i = 0; i < 8; ++i)
    a[i] = (h16 ? v[i + 8] : v[i]) + __shfl_xor_sync(0xffffffffu, h16 ? v[i] : v[i + 8], 16);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    b[i] = (h8 ? a[i + 4] : a[i]) + __shfl_xor_sync(0xffffffffu, h8 ? a[i] : a[i + 4], 8);
#pragma unroll
  for (int i = 0; i < 2; ++i)
    c[i] = (h4 ? b[i + 2] : b[i]) + __shfl_xor_sync(0xffffffffu, h4 ? b[i] : b[i + 2], 4);
  float d = (h2 ? c[1] : c[0]) + __shfl_xor_sync(0xffffffffu, h2 ? c[0] : c[1], 2);
  return d + __shfl_xor_sync(0xffffffffu, d, 1);
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

// Epilogue inputs that do not depend on the accumulator, loaded before the
// accumulator / split-K ticket is waited for, so their latency overlaps it:
// RESID -- the residual stream values and the next norm's gain; QKV -- the
// RoPE (cos, sin) of each column.  Valid for the 16 columns from t0.
struct EpiPre {
  float a[kEpiCols];
  float b[kEpiCols];
  float g;
  int ok;
  int t0;
};

template <int KIND, typename Act>
__device__ __forceinline__ void epi_prefetch(const EpiArgs& e, int mt, int t0, int r,
                                             const EpiSmem& s, EpiPre& p) {
  p.ok = 0;
  p.t0 = t0;
  if (KIND == EPI_RESID) {
    const int m = mt * kBM + r;
    p.g = ld_act(reinterpret_cast<const Act*>(e.gnext), m);
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      const int t = t0 + j;
      p.a[j] = (t < e.T) ? __ldcg(e.x + static_cast<size_t>(t) * e.d + m) : 0.f;
    }
    p.ok = 1;
  } else if (KIND == EPI_QKV) {
    if (!s.prepared) return;
    const int m = mt * kBM + r;
    const int sec = (m < e.dq) ? 0 : (m < e.dq + e.dkv ? 1 : 2);
    if (sec == 2) return;
    const int ms = m - (sec == 0 ? 0 : e.dq);
    const int i = ms % e.hd, half = e.hd >> 1;
    const int fi = (i < half) ? i : i - half;
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      const int t = t0 + j;
      float2 cs = make_float2(1.f, 0.f);
      if (t < e.T) {
        const int pp = min(s.pos_all[t], e.max_seq - 1);
        cs = e.rope[static_cast<size_t>(pp) * half + fi];
      }
      p.a[j] = cs.x;
      p.b[j] = cs.y;
    }
    p.ok = 1;
  }
}

template <int KIND, typename Act>
__device__ void epi_apply(const EpiArgs& e, int mt, int t0, float (&v)[kEpiCols], int r,
                          EpiSmem& s, const EpiPre* pre = nullptr) {
  const bool use_pre = pre != nullptr && pre->ok && pre->t0 == t0;
  const int lane = r & 31, grp = r >> 5;
  // Every 16-column chunk but a ragged last one is full: its loops run
  // without per-column guards (the epilogue warps run one per scheduler, so
  // each branch and dependent step is exposed latency).
  const bool full = t0 + kEpiCols <= e.T;
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
      // rotate-half RoPE: v' = v cos + sgn * partner sin, sgn = -1 in the
      // first half of the head
      const bool lowhalf = i < half;
      const int rp = lowhalf ? r + half : r - half;
      const int fi = lowhalf ? i : i - half;
      float cs_c[kEpiCols], cs_s[kEpiCols], pv[kEpiCols];
#pragma unroll
      for (int j = 0; j < kEpiCols; ++j) {
        const int t = min(t0 + j, e.T - 1);
        if (use_pre) {
          cs_c[j] = pre->a[j];
          cs_s[j] = pre->b[j];
        } else {
          const int p = min(s.prepared ? s.pos_all[t] : e.pos[t], e.max_seq - 1);
          const float2 cs = e.rope[static_cast<size_t>(p) * half + fi];
          cs_c[j] = cs.x;
          cs_s[j] = cs.y;
        }
        pv[j] = s.x[j][rp];
      }
#pragma unroll
      for (int j = 0; j < kEpiCols; ++j) {
        const float ps = pv[j] * cs_s[j];
        v[j] = lowhalf ? (v[j] * cs_c[j] - ps) : (v[j] * cs_c[j] + ps);
      }
      epi_sync();
    }
    using AT = typename AttnType<Act>::T;
    if (sec == 0) {
      AT* q = reinterpret_cast<AT*>(e.q_out) + static_cast<size_t>(t0) * e.dq + m;
#pragma unroll
      for (int j = 0; j < kEpiCols; ++j)
        if (full || t0 + j < e.T) st_act(q, static_cast<size_t>(j) * e.dq, v[j]);
    } else {
      // every column's cache row first: a load may not move above an
      // earlier store, so reading them between the stores would serialise
      AT* cache = reinterpret_cast<AT*>(sec == 1 ? e.k_cache : e.v_cache) +
                  static_cast<size_t>(head) * e.max_seq * e.hd + i;
      const size_t bstride = static_cast<size_t>(e.n_kv_heads) * e.max_seq * e.hd;
      int pj[kEpiCols], bj[kEpiCols];
#pragma unroll
      for (int j = 0; j < kEpiCols; ++j) {
        const int t = min(t0 + j, e.T - 1);
        pj[j] = s.prepared ? s.pos_all[t] : e.pos[t];
        bj[j] = s.prepared ? s.bidx_all[t] : e.bidx[t];
      }
      bool bad = false;
#pragma unroll
      for (int j = 0; j < kEpiCols; ++j) {
        const bool live = full || t0 + j < e.T;
        const bool inside = static_cast<unsigned>(pj[j]) < static_cast<unsigned>(e.max_seq);
        if (live && inside)
          st_act(cache, static_cast<size_t>(bj[j]) * bstride + static_cast<size_t>(pj[j]) * e.hd,
                 v[j]);
        bad |= live && !inside;
      }
      if (bad) atomicOr(e.err, DERR_CAPACITY);
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
        float h[kEpiCols];  // SwiGLU of every column first, then the stores
#pragma unroll
        for (int j = 0; j < kEpiCols; ++j) {
          const float gt = v[j], up = s.x[j][r + 64];
          if constexpr (std::is_same<Act, float>::value)
            h[j] = gt / (1.f + expf(-gt)) * up;
          else  // bf16 engine: the fast intrinsics' error is far below the lo plane's
            h[j] = __fdividef(gt, 1.f + __expf(-gt)) * up;
        }
        Act* hp = reinterpret_cast<Act*>(e.h_out) + static_cast<size_t>(t0) * e.F + f;
#pragma unroll
        for (int j = 0; j < kEpiCols; ++j)
          if (full || t0 + j < e.T) st_gin(hp, static_cast<size_t>(j) * e.F, e.plane_h, h[j]);
      }
    }
    epi_sync();
  } else if (KIND == EPI_RESID) {
    const int m = mt * kBM + r;
    const float gn = use_pre ? pre->g : ld_act(reinterpret_cast<const Act*>(e.gnext), m);
    float* xp = e.x + static_cast<size_t>(t0) * e.d + m;
    Act* gp = reinterpret_cast<Act*>(e.xg) + static_cast<size_t>(t0) * e.d + m;
    float xi[kEpiCols], sq[kEpiCols];
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      const bool live = full || t0 + j < e.T;
      // L2 read: other CTAs rewrite the residual stream in earlier phases
      // of the persistent kernel, and L1 is not coherent across SMs
      const float x0 = use_pre ? pre->a[j] : (live ? __ldcg(xp + static_cast<size_t>(j) * e.d) : 0.f);
      xi[j] = x0 + v[j];
      sq[j] = live ? xi[j] * xi[j] : 0.f;
    }
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      if (full || t0 + j < e.T) {
        const size_t o = static_cast<size_t>(j) * e.d;
        xp[o] = xi[j];
        st_gin(gp, o, e.plane_x, xi[j] * gn);
      }
    }
    const float col = warp_colsum16(sq, lane);
    if ((lane & 1) == 0) s.red[grp][lane >> 1] = col;
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
    // per column (max, argmax, second max) over the warp's 32 rows, by the
    // same halving exchanges as warp_colsum16 (the merge is exact, so the
    // order does not matter); column c ends in lanes 2c, 2c + 1
    float c1[kEpiCols], c2[kEpiCols];
    int ci[kEpiCols];
#pragma unroll
    for (int j = 0; j < kEpiCols; ++j) {
      const int t = t0 + j;
      const float lg = v[j] * s.rs[j];
      if (e.logits != nullptr && t < e.T && vrow) e.logits[static_cast<size_t>(t) * e.V + m] = lg;
      c1[j] = vrow ? lg : -INFINITY;
      c2[j] = -INFINITY;
      ci[j] = m;
    }
#pragma unroll
    for (int o = 16, half = 8; o >= 2; o >>= 1, half >>= 1) {
      const bool hi = lane & o;
#pragma unroll
      for (int i = 0; i < half; ++i) {
        // keep column i (low lanes) or i + half (high lanes), merge the
        // partner's copy of it (selects between statically indexed values)
        const float w1 = __shfl_xor_sync(0xffffffffu, hi ? c1[i] : c1[i + half], o);
        const int wj = __shfl_xor_sync(0xffffffffu, hi ? ci[i] : ci[i + half], o);
        const float w2 = __shfl_xor_sync(0xffffffffu, hi ? c2[i] : c2[i + half], o);
        float a1 = hi ? c1[i + half] : c1[i], a2 = hi ? c2[i + half] : c2[i];
        int ai = hi ? ci[i + half] : ci[i];
        am_merge(a1, ai, a2, w1, wj, w2);
        c1[i] = a1;
        ci[i] = ai;
        c2[i] = a2;
      }
    }
    {
      float a1 = c1[0], a2 = c2[0];
      int ai = ci[0];
      am_merge(a1, ai, a2, __shfl_xor_sync(0xffffffffu, c1[0], 1),
               __shfl_xor_sync(0xffffffffu, ci[0], 1), __shfl_xor_sync(0xffffffffu, c2[0], 1));
      if ((lane & 1) == 0) {
        s.am[grp][lane >> 1][0] = a1;
        s.am[grp][lane >> 1][1] = __int_as_float(ai);
        s.am[grp][lane >> 1][2] = a2;
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
__device__ inline void epi_argmax_finish(const EpiArgs& e, int r, EpiSmem& s) {
  epi_sync();
  if (r == 0) {
    const int old = ticket_add(e.am_ticket, 1);
    s.flag = (old == e.am_units - 1);
  }
  epi_sync();
  const bool last = s.flag;
  epi_sync();
  if (!last) return;
  for (int tb = 0; tb < e.T; tb += 16) {
    const int t = tb + (r >> 3), part = r & 7;
    float v1 = -INFINITY, v2 = -INFINITY;
    int i1 = INT_MAX;
    if (t < e.T) {
      // every tile of a 256-tile vocabulary in one round trip (32 loads of
      // each kind in flight per thread)
      for (int mt0 = part; mt0 < e.am_mtiles; mt0 += 256) {
        float w1[32], w2[32];
        int j1[32];
#pragma unroll
        for (int u = 0; u < 32; ++u) {
          const int mt = mt0 + 8 * u;
          if (mt < e.am_mtiles) {
            const float* p = e.am_part + (static_cast<size_t>(mt) * e.ldt + t) * 3;
            w1[u] = __ldcg(p);
            j1[u] = __float_as_int(__ldcg(p + 1));
            w2[u] = __ldcg(p + 2);
          } else {
            w1[u] = -INFINITY;
            j1[u] = INT_MAX;
            w2[u] = -INFINITY;
          }
        }
#pragma unroll
        for (int u = 0; u < 32; ++u) am_merge(v1, i1, v2, w1[u], j1[u], w2[u]);
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

}  // namespace cllm
