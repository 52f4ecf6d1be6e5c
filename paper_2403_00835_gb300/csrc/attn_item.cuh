// One work item of the block attention (16-row query tile x head x 128-key
// chunk) on tensor cores, and the merge of a query tile's chunk partials.
// Shared by the attention kernel (a CTA of 128 threads) and the persistent
// per-iteration kernel (its four epilogue warps); `sync` is the barrier of
// those 128 threads and `tid` their index 0..127.
#pragma once
#include "act.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace cllm {

template <int HD>
struct AttnTileSmem {
  __half q[kQTile][HD + 8];
  __half k[kAttnChunk][HD + 8];  // reused as float co[4][kQTile][HD + 8] for the warp merge
  __half v[kAttnChunk][HD + 8];
  float m[4][kQTile];
  float l[4][kQTile];
};

// The same tile filled by TMA tensor-map loads (persistent kernel): Q, K and V
// as 64-column halves of [rows][128 B] with the 128-byte swizzle (16-byte
// chunk c of row r stored at chunk c ^ (r mod 8)), which keeps ldmatrix free
// of bank conflicts without padding; one TMA operation moves a whole
// 128-row half.  After the key loop K and V hold the warps' merge area.
template <int HD>
struct AttnTileSmemTma {
  alignas(1024) uint8_t q[kQTile * HD * 2];
  alignas(1024) uint8_t k[kAttnChunk * HD * 2];
  alignas(1024) uint8_t v[kAttnChunk * HD * 2];
  float m[4][kQTile];
  float l[4][kQTile];
  uint64_t bar[2];  // completion of the K (with Q) and V loads; fresh per work item
};

// Tensor maps of the TMA tile loads: the K and V caches of all layers as
// [layer][b][kv_head][pos] rows of hd fp16 values (boxes of 128 rows x 64
// columns), Q as [row][n_heads*hd] (boxes of 16 rows x 64 columns); kv_row0 =
// the first row of this layer.
struct AttnTma {
  const CUtensorMap* k;
  const CUtensorMap* v;
  const CUtensorMap* q;
  int kv_row0;
};

template <class T>
struct IsTmaTile {
  static constexpr bool value = false;
};
template <int HD>
struct IsTmaTile<AttnTileSmemTma<HD>> {
  static constexpr bool value = true;
};

// Byte address of 16-byte chunk `chunk` of row `row` in a swizzled tile of
// `rows` rows per 64-column half.
__device__ __forceinline__ uint32_t sw128_addr(uint32_t base, int rows, int row, int chunk) {
  return base + static_cast<uint32_t>((chunk >> 3) * rows * 128 + row * 128 +
                                      (((chunk & 7) ^ (row & 7)) << 4));
}

// Where the iteration's query-tile and sequence metadata are read from: the
// kernel arguments (global memory), or a shared-memory copy made once per
// phase (AttnMetaSmem) so that work items do not chain dependent loads.
struct GlobalMeta {
  const AttnArgs& a;
  __device__ int2 qtile(int q) const { return a.qtiles[q]; }
  __device__ int start(int b) const { return a.seq_start[b]; }
  __device__ int row0(int b) const { return a.seq_row0[b]; }
  __device__ int nrows(int b) const { return a.seq_nrows[b]; }
};

constexpr int kMetaMaxBatch = 128;

struct AttnMetaSmem {
  int2 qt[kMaxQTilesStep];
  int start[kMetaMaxBatch];
  int row0[kMetaMaxBatch];
  int nrows[kMetaMaxBatch];
};

struct SmemMeta {
  const AttnMetaSmem& m;
  __device__ int2 qtile(int q) const { return m.qt[q]; }
  __device__ int start(int b) const { return m.start[b]; }
  __device__ int row0(int b) const { return m.row0[b]; }
  __device__ int nrows(int b) const { return m.nrows[b]; }
};

// Copy the metadata of `a` into shared memory (128 threads, one round trip).
__device__ __forceinline__ void attn_meta_load(const AttnArgs& a, AttnMetaSmem& m, int tid, int B) {
  for (int q = tid; q < a.n_qtiles; q += 128) m.qt[q] = a.qtiles[q];
  for (int b = tid; b < B; b += 128) {
    m.start[b] = __ldcg(a.seq_start + b);
    m.row0[b] = __ldcg(a.seq_row0 + b);
    m.nrows[b] = __ldcg(a.seq_nrows + b);
  }
}

// Number of key chunks the query tile qi reaches (its last row's position).
template <class Meta>
__device__ __forceinline__ int attn_tile_chunks(const AttnArgs& a, const Meta& md, int qi) {
  const int2 qt = md.qtile(qi);
  const int nr = min(kQTile, md.nrows(qt.x) - qt.y);
  if (nr <= 0) return 0;
  const int pos_last = md.start(qt.x) + qt.y + nr - 1;
  return min(pos_last / kAttnChunk + 1, a.nch_max);
}
__device__ __forceinline__ int attn_tile_chunks(const AttnArgs& a, int qi) {
  return attn_tile_chunks(a, GlobalMeta{a}, qi);
}

// Prefix sum of work items over query tiles into pre[0..n_qtiles];
// items(q) = H * ceil(chunks(q) / range), range = chunks per item (1 for the
// per-chunk fp32 path).  Warp 0 of the group scans; returns the total.
template <class Sync, class Meta = GlobalMeta>
__device__ int attn_item_prefix(const AttnArgs& a, int* pre, int tid, Sync sync, const Meta& md,
                                int range = kAttnRange) {
  if (tid < 32) {
    int carry = 0;
    for (int base = 0; base < a.n_qtiles; base += 32) {
      const int q = base + tid;
      const int cnt = q < a.n_qtiles ? a.H * ((attn_tile_chunks(a, md, q) + range - 1) / range) : 0;
      int incl = cnt;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (tid >= o) incl += y;
      }
      if (q < a.n_qtiles) pre[q] = carry + incl - cnt;
      carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (tid == 0) pre[a.n_qtiles] = carry;
  }
  sync();
  return pre[a.n_qtiles];
}
template <class Sync>
__device__ int attn_item_prefix(const AttnArgs& a, int* pre, int tid, Sync sync,
                                int range = kAttnRange) {
  return attn_item_prefix(a, pre, tid, sync, GlobalMeta{a}, range);
}

__device__ __forceinline__ int attn_find_qtile(const int* pre, int n, int item) {
  int lo = 0, hi = n - 1;  // largest q with pre[q] <= item
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (pre[mid] <= item) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// Rows of query tile qi and their number of chunk ranges (the last row's).
template <class Meta>
__device__ __forceinline__ int attn_tile_ranges(const AttnArgs& a, const Meta& md, int qi) {
  return (attn_tile_chunks(a, md, qi) + kAttnRange - 1) / kAttnRange;
}

// Work item `item`: one (query tile, head, range of kAttnRange key chunks).
// The 4 warps split each 128-key chunk (32 keys each) and keep an online
// softmax over the range's chunks; K of the next chunk is loaded while the
// current chunk's P.V runs, V while the next Q.K runs.  Then the warps' (m, l,
// O) are merged.  A tile with a single range writes its attention output
// (O / l, the GEMM input planes) directly and returns true when direct_ok;
// otherwise the range's partial (O, m, l) goes to slot `range` of the
// partials (merged by the combine, which gives the same bits for one range).
// Returns the tile index and head in qi_out, h_out.
template <int HD, class Sync, class Meta = GlobalMeta, class Tile = AttnTileSmem<HD>>
__device__ bool attn_mma_item(const AttnArgs& a, int item, const int* pre, Tile& sm, int tid,
                              Sync sync, int& qi_out, int& h_out, const Meta& md,
                              bool direct_ok = true, const AttnTma* tma = nullptr) {
  constexpr bool kTma = IsTmaTile<Tile>::value;
  // merge area: rows padded by 8 floats, so that the 8 row groups of a warp's
  // accumulator fragment fall in distinct banks
  constexpr int CLD = HD + 8;
  static_assert(sizeof(float) * 4 * kQTile * CLD <= (kTma ? 2 : 1) * sizeof(sm.k),
                "merge area must fit in the K (and V) tile");
  const int warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, cq = lane & 3;
  const int group = a.H / a.Hkv;
  const int ldq = a.H * HD;
  const __half* Q = static_cast<const __half*>(a.q);
  const __half* KC = static_cast<const __half*>(a.k_cache);
  const __half* VC = static_cast<const __half*>(a.v_cache);
  float (*co)[kQTile][CLD] = reinterpret_cast<float (*)[kQTile][CLD]>(&sm.k[0]);
  const int qi = attn_find_qtile(pre, a.n_qtiles, item);
  const int local = item - pre[qi];
  const int rg = local / a.H, h = local - rg * a.H;
  const int nrange = attn_tile_ranges(a, md, qi);
  const int2 qt = md.qtile(qi);
  const int b = qt.x, r0 = qt.y;
  const int nr = min(kQTile, md.nrows(b) - r0);
  const int start = md.start(b);
  const int row_g0 = md.row0(b) + r0;
  const int pos0 = start + r0;  // position of tile row 0
  const int c0 = rg * kAttnRange;
  const int c1 = min(c0 + kAttnRange, attn_tile_chunks(a, md, qi));
  const int kend = min(pos0 + nr, a.max_seq);  // keys of the tile: [0, kend)
  if (pos0 + nr > a.max_seq && tid == 0) atomicOr(a.err, DERR_CAPACITY);
  const int kvh = h / group;
  const size_t kvbase = ((static_cast<size_t>(b) * a.Hkv + kvh) * a.max_seq) * HD;
  constexpr int CPR = HD * 2 / 16;  // 16-byte pieces per row
  constexpr int NHALF = HD / 64;     // 64-column halves of a row (TMA boxes per tile)
  uint64_t* barK = nullptr;
  uint64_t* barV = nullptr;
  uint32_t phK = 0, phV = 0;
  int kvrow = 0;

  // cp.async path: per-thread 16-byte copies, zero rows past the tile's keys
  auto load_kv = [&](auto* dstm, const __half* src, int c) {
    const int kb = c * kAttnChunk;
    for (int i = tid; i < kAttnChunk * CPR; i += 128) {
      const int rr = i / CPR, pc = i - rr * CPR;
      void* dst = &dstm[rr][pc * 8];
      if (kb + rr < kend)
        cp_async16(dst, src + kvbase + static_cast<size_t>(kb + rr) * HD + pc * 8);
      else
        *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
  };
  // TMA path: one thread posts the byte count and issues a box per 64-column
  // half.  Rows past the tile's keys hold other positions' (finite) cache
  // values or the map's zero fill: their scores are masked to -inf, so their
  // probabilities are exactly 0.
  auto tma_kv = [&](uint8_t* dst, const CUtensorMap* map, int c, uint64_t* bar, bool with_q) {
    if (tid == 0) {
      mbar_arrive_expect_tx(bar, (with_q ? NHALF * kQTile * 128 : 0) + NHALF * kAttnChunk * 128);
      if (with_q)
        for (int hh = 0; hh < NHALF; ++hh)
          tma_load_2d_nohint(sm.q + hh * kQTile * 128, tma->q, bar, h * HD + hh * 64, row_g0);
      for (int hh = 0; hh < NHALF; ++hh)
        tma_load_2d_nohint(dst + hh * kAttnChunk * 128, map, bar, hh * 64,
                           kvrow + c * kAttnChunk);
    }
  };
  auto wait_buf = [&](uint64_t* bar, uint32_t& ph) {
    if (!mbar_wait(bar, ph & 1u, nullptr) && tid == 0) atomicOr(a.err, DERR_TIMEOUT);
    ++ph;
  };

  if constexpr (kTma) {
    barK = &sm.bar[0];
    barV = &sm.bar[1];
    kvrow = tma->kv_row0 + (b * a.Hkv + kvh) * a.max_seq;
    // fresh barrier phases per work item; every earlier generic write to this
    // shared memory (merge area, GEMM epilogue) ordered before the TMA writes
    fence_proxy_async_smem();
    if (tid == 0) {
      mbar_init(barK, 1);
      mbar_init(barV, 1);
      fence_mbar_init();
    }
    sync();
    // ---- Q (16 rows) with the first chunk's K on barK; its V on barV ----
    tma_kv(sm.k, tma->k, c0, barK, true);
    tma_kv(sm.v, tma->v, c0, barV, false);
  } else {
    // ---- Q (16 rows) and the first chunk's K: group 1; its V: group 2 ----
    for (int i = tid; i < kQTile * CPR; i += 128) {
      const int rr = i / CPR, pc = i - rr * CPR;
      void* dst = &sm.q[rr][pc * 8];
      if (rr < nr)
        cp_async16(dst, Q + static_cast<size_t>(row_g0 + rr) * ldq + h * HD + pc * 8);
      else
        *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
    load_kv(sm.k, KC, c0);
    cp_async_commit();
    load_kv(sm.v, VC, c0);
    cp_async_commit();
  }
  (void)phK;
  (void)phV;

  const int wk0 = warp * 32;  // first key of this warp within a chunk
  const int posA = pos0 + g, posB = pos0 + g + 8;
  const bool rowA = g < nr, rowB = g + 8 < nr;
  float o[HD / 8][4];
#pragma unroll
  for (int dn = 0; dn < HD / 8; ++dn) o[dn][0] = o[dn][1] = o[dn][2] = o[dn][3] = 0.f;
  float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
  for (int c = c0; c < c1; ++c) {
    const int kb = c * kAttnChunk;
    if constexpr (kTma) {
      wait_buf(barK, phK);  // (Q and) this chunk's K: TMA writes, seen by every waiter
    } else {
      cp_async_wait_but1();  // Q and this chunk's K
      sync();
    }
    float sc[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j) sc[j][0] = sc[j][1] = sc[j][2] = sc[j][3] = 0.f;
    const bool live = kb + wk0 < kend;
    if (live) {
#pragma unroll
      for (int ks = 0; ks < HD / 16; ks += 2) {
        uint32_t qa0[4], qa1[4];
        if constexpr (kTma) {
          const uint32_t qb = smem_u32(sm.q);
          ldmatrix_x4_a(qa0, sw128_addr(qb, kQTile, lane & 15, ks * 2 + (lane >> 4)));
          ldmatrix_x4_a(qa1, sw128_addr(qb, kQTile, lane & 15, (ks + 1) * 2 + (lane >> 4)));
        } else {
          ldmatrix_x4(qa0, &sm.q[lane & 15][ks * 16 + (lane >> 4) * 8]);
          ldmatrix_x4(qa1, &sm.q[lane & 15][(ks + 1) * 16 + (lane >> 4) * 8]);
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          uint32_t kb4[4];
          const int mi = lane >> 3;
          if constexpr (kTma)
            ldmatrix_x4_a(kb4, sw128_addr(smem_u32(sm.k), kAttnChunk, wk0 + 8 * j + (lane & 7),
                                          (ks + (mi >> 1)) * 2 + (mi & 1)));
          else
            ldmatrix_x4(kb4, &sm.k[wk0 + 8 * j + (lane & 7)][(ks + (mi >> 1)) * 16 + (mi & 1) * 8]);
          mma_f16_16816(sc[j], qa0, kb4[0], kb4[1]);
          mma_f16_16816(sc[j], qa1, kb4[2], kb4[3]);
        }
      }
    }
    sync();  // every warp is done with K
    if constexpr (kTma) {
      if (c + 1 < c1) tma_kv(sm.k, tma->k, c + 1, barK, false);
    } else {
      if (c + 1 < c1) load_kv(sm.k, KC, c + 1);
      cp_async_commit();  // (possibly empty) group: the next chunk's K
    }
    if (live) {
      // mask + scale (log2 domain), online softmax over the range's chunks
      float nA = mA, nB = mB;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = kb + wk0 + 8 * j + 2 * cq + (e & 1);
          const bool top = e < 2;
          const bool valid = key < kend && (top ? (rowA && key <= posA) : (rowB && key <= posB));
          sc[j][e] = valid ? sc[j][e] * a.scale_log2 : -INFINITY;
        }
        nA = fmaxf(nA, fmaxf(sc[j][0], sc[j][1]));
        nB = fmaxf(nB, fmaxf(sc[j][2], sc[j][3]));
      }
      nA = fmaxf(nA, __shfl_xor_sync(0xffffffffu, nA, 1));
      nA = fmaxf(nA, __shfl_xor_sync(0xffffffffu, nA, 2));
      nB = fmaxf(nB, __shfl_xor_sync(0xffffffffu, nB, 1));
      nB = fmaxf(nB, __shfl_xor_sync(0xffffffffu, nB, 2));
      const float uA = (nA == -INFINITY) ? 0.f : nA;
      const float uB = (nB == -INFINITY) ? 0.f : nB;
      const float fA = exp2f(mA - uA), fB = exp2f(mB - uB);  // rescale of the running sums
      mA = nA;
      mB = nB;
      float sA = 0.f, sB = 0.f;
      uint32_t pa[2][4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float p0 = exp2f(sc[j][0] - uA), p1 = exp2f(sc[j][1] - uA);
        const float p2 = exp2f(sc[j][2] - uB), p3 = exp2f(sc[j][3] - uB);
        sA += p0 + p1;
        sB += p2 + p3;
        pa[j >> 1][(j & 1) * 2 + 0] = pack_f16x2(p0, p1);
        pa[j >> 1][(j & 1) * 2 + 1] = pack_f16x2(p2, p3);
      }
      sA += __shfl_xor_sync(0xffffffffu, sA, 1);
      sA += __shfl_xor_sync(0xffffffffu, sA, 2);
      sB += __shfl_xor_sync(0xffffffffu, sB, 1);
      sB += __shfl_xor_sync(0xffffffffu, sB, 2);
      lA = lA * fA + sA;
      lB = lB * fB + sB;
#pragma unroll
      for (int dn = 0; dn < HD / 8; ++dn) {
        o[dn][0] *= fA;
        o[dn][1] *= fA;
        o[dn][2] *= fB;
        o[dn][3] *= fB;
      }
      if constexpr (kTma) {
        wait_buf(barV, phV);  // this chunk's V (the next K may be in flight)
      } else {
        cp_async_wait_but1();  // this chunk's V (the next K may be in flight)
        sync();
      }
      // O += P V: A fragments of P for keys 16kk..16kk+15 are the S
      // accumulators of n-tiles 2kk, 2kk+1 (a0: row g keys 2c.., a1: row g+8,
      // a2/a3: +8 keys).
#pragma unroll
      for (int kk = 0; kk < 2; ++kk) {
        const uint32_t af[4] = {pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3]};
#pragma unroll
        for (int dn = 0; dn < HD / 8; dn += 2) {
          uint32_t vb[4];
          const int mi = lane >> 3;
          if constexpr (kTma)
            ldmatrix_x4_trans_a(vb, sw128_addr(smem_u32(sm.v), kAttnChunk,
                                               wk0 + 16 * kk + (mi & 1) * 8 + (lane & 7), dn + (mi >> 1)));
          else
            ldmatrix_x4_trans(vb, &sm.v[wk0 + 16 * kk + (mi & 1) * 8 + (lane & 7)][(dn + (mi >> 1)) * 8]);
          mma_f16_16816(o[dn], af, vb[0], vb[1]);
          mma_f16_16816(o[dn + 1], af, vb[2], vb[3]);
        }
      }
    } else {
      if constexpr (kTma) {
        wait_buf(barV, phV);
      } else {
        cp_async_wait_but1();
        sync();
      }
    }
    sync();  // every warp is done with V
    if constexpr (kTma) {
      if (c + 1 < c1) tma_kv(sm.v, tma->v, c + 1, barV, false);
    } else {
      if (c + 1 < c1) load_kv(sm.v, VC, c + 1);
      cp_async_commit();  // (possibly empty) group: the next chunk's V
    }
  }
  if constexpr (!kTma) cp_async_wait_all();
  sync();
#pragma unroll
  for (int dn = 0; dn < HD / 8; ++dn) {
    const int d0 = dn * 8 + 2 * cq;
    *reinterpret_cast<float2*>(&co[warp][g][d0]) = make_float2(o[dn][0], o[dn][1]);
    *reinterpret_cast<float2*>(&co[warp][g + 8][d0]) = make_float2(o[dn][2], o[dn][3]);
  }
  if (cq == 0) {
    sm.m[warp][g] = mA;
    sm.m[warp][g + 8] = mB;
    sm.l[warp][g] = lA;
    sm.l[warp][g + 8] = lB;
  }
  sync();
  const bool single = direct_ok && nrange == 1;
  {
    // thread -> (row, 4 consecutive dims): a row's HD floats are written by
    // HD/4 consecutive threads as float4 (coalesced)
    constexpr int TPR = HD / 4;     // threads per row
    constexpr int RPP = 128 / TPR;  // rows per pass
    constexpr int NP = kQTile / RPP;  // passes
    const int d = (tid % TPR) * 4;
    // all passes' shared-memory reads and arithmetic first, then the global
    // stores: a store may not be reordered above a later pass's loads, so
    // interleaving them would serialise the passes
    float4 ov[NP];
    float lsum[NP], Mrow[NP];
#pragma unroll
    for (int k = 0; k < NP; ++k) {
      const int row = tid / TPR + k * RPP;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < 4; ++w) M = fmaxf(M, sm.m[w][row]);
      ov[k] = make_float4(0.f, 0.f, 0.f, 0.f);
      float l = 0.f;
      if (row < nr && M != -INFINITY) {
        float f[4];
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          f[w] = exp2f(sm.m[w][row] - M);
          l += f[w] * sm.l[w][row];
        }
        const float4 w0 = *reinterpret_cast<const float4*>(&co[0][row][d]);
        const float4 w1 = *reinterpret_cast<const float4*>(&co[1][row][d]);
        const float4 w2 = *reinterpret_cast<const float4*>(&co[2][row][d]);
        const float4 w3 = *reinterpret_cast<const float4*>(&co[3][row][d]);
        ov[k] = make_float4(((f[0] * w0.x + f[1] * w1.x) + f[2] * w2.x) + f[3] * w3.x,
                            ((f[0] * w0.y + f[1] * w1.y) + f[2] * w2.y) + f[3] * w3.y,
                            ((f[0] * w0.z + f[1] * w1.z) + f[2] * w2.z) + f[3] * w3.z,
                            ((f[0] * w0.w + f[1] * w1.w) + f[2] * w2.w) + f[3] * w3.w);
      }
      lsum[k] = l;
      Mrow[k] = M;
    }
#pragma unroll
    for (int k = 0; k < NP; ++k) {
      const int row = tid / TPR + k * RPP;
      if (row < nr) {
        if (single) {
          // the tile's only range: the attention output itself
          const float l = lsum[k];
          st_gin4(static_cast<__nv_bfloat16*>(a.out),
                  static_cast<size_t>(row_g0 + row) * a.H * HD + h * HD + d, a.plane_out,
                  make_float4(ov[k].x / l, ov[k].y / l, ov[k].z / l, ov[k].w / l));
        } else {
          const size_t pidx = (static_cast<size_t>(row_g0 + row) * a.H + h) * a.nch_max + rg;
          *reinterpret_cast<float4*>(a.part_o + pidx * HD + d) = ov[k];
          if (d == 0) a.part_ml[pidx] = make_float2(Mrow[k], lsum[k]);
        }
      }
    }
  }
  sync();
  if constexpr (kTma) {
    if (tid == 0) {  // every load of the item has been waited for
      mbar_inval(barK);
      mbar_inval(barV);
    }
  }
  qi_out = qi;
  h_out = h;
  return single;
}
template <int HD, class Sync>
__device__ bool attn_mma_item(const AttnArgs& a, int item, const int* pre, AttnTileSmem<HD>& sm,
                              int tid, Sync sync, int& qi_out, int& h_out, bool direct_ok) {
  return attn_mma_item<HD>(a, item, pre, sm, tid, sync, qi_out, h_out, GlobalMeta{a}, direct_ok);
}

// Merge of the range partials 0..ceil((pos/128 + 1) / kAttnRange) - 1 of every
// row of query tile qi for head h, in range order; out = O / l, written as the
// GEMM input planes.
// Per output element: l = sum_c f_c l_c and acc = sum_c f_c O_c with
// f_c = 2^(m_c - M), both accumulated with fmaf in chunk order (the attention
// combine kernel computes the same sums).  Thread -> (row, 4 consecutive
// dims), HD/4 consecutive threads per row, so loads and stores are coalesced
// vectors; the rows of all passes and the partials of 2 chunks are loaded
// together, so a tile of up to 256 keys costs one round trip.
template <typename Act, int HD, class Meta>
__device__ void attn_combine_tile(const AttnArgs& a, int qi, int h, int tid, const Meta& md) {
  const int2 qt = md.qtile(qi);
  const int b = qt.x, r0 = qt.y;
  const int nr = min(kQTile, md.nrows(b) - r0);
  constexpr int TPR = HD / 4;        // threads per row
  constexpr int RPP = 128 / TPR;     // rows per pass
  constexpr int NP = kQTile / RPP;   // passes
  constexpr int CG = 2;              // chunks per load group
  const int d = (tid % TPR) * 4;
  int nch[NP];
  size_t base[NP];
  float2 ml[NP][CG];
  float4 ov[NP][CG];
  auto load_group = [&](int c0) {
#pragma unroll
    for (int ps = 0; ps < NP; ++ps)
#pragma unroll
      for (int q = 0; q < CG; ++q)
        if (c0 + q < nch[ps]) {
          ml[ps][q] = __ldcg(&a.part_ml[base[ps] + c0 + q]);
          ov[ps][q] = __ldcg(reinterpret_cast<const float4*>(a.part_o + (base[ps] + c0 + q) * HD + d));
        }
  };
  int nch_max = 0;
#pragma unroll
  for (int ps = 0; ps < NP; ++ps) {
    const int row = ps * RPP + tid / TPR;
    const int t = md.row0(b) + r0 + row;
    const int pos = md.start(b) + r0 + row;  // the row's position (pos[t])
    nch[ps] = row < nr ? (min(pos / kAttnChunk + 1, a.nch_max) + kAttnRange - 1) / kAttnRange : 0;
    base[ps] = (static_cast<size_t>(t) * a.H + h) * a.nch_max;
    nch_max = max(nch_max, nch[ps]);
  }
  load_group(0);
  float M[NP];
#pragma unroll
  for (int ps = 0; ps < NP; ++ps) {
    M[ps] = -INFINITY;
#pragma unroll
    for (int q = 0; q < CG; ++q)
      if (q < nch[ps]) M[ps] = fmaxf(M[ps], ml[ps][q].x);
    for (int c = CG; c < nch[ps]; ++c) M[ps] = fmaxf(M[ps], __ldcg(&a.part_ml[base[ps] + c].x));
  }
  float4 acc[NP];
  float l[NP];
#pragma unroll
  for (int ps = 0; ps < NP; ++ps) {
    acc[ps] = make_float4(0.f, 0.f, 0.f, 0.f);
    l[ps] = 0.f;
  }
  for (int c0 = 0; c0 < nch_max; c0 += CG) {
    if (c0 > 0) load_group(c0);
#pragma unroll
    for (int ps = 0; ps < NP; ++ps)
#pragma unroll
      for (int q = 0; q < CG; ++q)
        if (c0 + q < nch[ps]) {
          const float f = exp2f(ml[ps][q].x - M[ps]);
          l[ps] = fmaf(f, ml[ps][q].y, l[ps]);
          acc[ps].x = fmaf(f, ov[ps][q].x, acc[ps].x);
          acc[ps].y = fmaf(f, ov[ps][q].y, acc[ps].y);
          acc[ps].z = fmaf(f, ov[ps][q].z, acc[ps].z);
          acc[ps].w = fmaf(f, ov[ps][q].w, acc[ps].w);
        }
  }
#pragma unroll
  for (int ps = 0; ps < NP; ++ps) {
    const int row = ps * RPP + tid / TPR;
    if (row >= nr) continue;
    const int t = md.row0(b) + r0 + row;
    const float L = l[ps];
    st_gin4(static_cast<Act*>(a.out), static_cast<size_t>(t) * a.H * HD + h * HD + d, a.plane_out,
            make_float4(acc[ps].x / L, acc[ps].y / L, acc[ps].z / L, acc[ps].w / L));
  }
}

}  // namespace cllm
