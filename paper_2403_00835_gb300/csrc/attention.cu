// Block attention of a Jacobi step: the n rows of each sequence's block attend
// to the cached prefix and, causally, to the block rows up to their own
// (Eq. 3's causal mask: row k of the block, at position L_b + k, sees keys at
// positions 0..L_b+k).  The block's own K/V were already written into the
// cache by the QKV epilogue, so every key comes from the cache.
//
// Split-KV: work items are (16-row query tile, head, key chunk of 128
// positions anchored at absolute position 0).  Each item writes an
// unnormalised partial (O, running max m, sum l); the combine kernel merges a
// row's chunks 0..pos/128 in chunk order.  A row's result therefore depends
// only on its own position, query and keys, not on how many rows share the
// step, so a Jacobi step and an AR step produce the same bits for a token.
//
// bf16 engine (Q, K, V and P held in fp16): each of 4 warps takes 32 keys of
// the chunk for the tile's 16 rows; S = Q K^T and O = P V run on mma.sync
// m16n8k16 f16 x f16 -> fp32 with
// ldmatrix loads from padded shared memory; the softmax is computed on the
// accumulator fragments with quad shuffles; the 4 warps' partials are merged
// in warp order.  fp32: a SIMT kernel with a per-row online softmax.
#include <float.h>

#include "act.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace cllm {

constexpr int kMaxQTilesSmem = 2048;

// Prefix sum of work items over query tiles, in shared memory.
// items(q) = H * (number of chunks the tile's last row reaches).
__device__ int attn_item_prefix(const AttnArgs& a, int* pre) {
  const int tid = threadIdx.x;
  if (tid < 32) {
    int carry = 0;
    for (int base = 0; base < a.n_qtiles; base += 32) {
      const int q = base + tid;
      int cnt = 0;
      if (q < a.n_qtiles) {
        const int2 qt = a.qtiles[q];
        const int nr = min(kQTile, a.seq_nrows[qt.x] - qt.y);
        if (nr > 0) {
          const int pos_last = a.seq_start[qt.x] + qt.y + nr - 1;
          cnt = a.H * min(pos_last / kAttnChunk + 1, a.nch_max);
        }
      }
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
  __syncthreads();
  return pre[a.n_qtiles];
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

template <int HD>
struct AttnSmemF16 {
  __half q[kQTile][HD + 8];
  __half k[kAttnChunk][HD + 8];  // reused as float co[4][kQTile][HD] for the warp merge
  __half v[kAttnChunk][HD + 8];
  float m[4][kQTile];
  float l[4][kQTile];
  int pre[kMaxQTilesSmem + 1];
};

template <int HD>
__global__ void __launch_bounds__(128) attn_chunk_mma_kernel(const AttnArgs a) {
  static_assert(sizeof(float) * 4 * kQTile * HD <= sizeof(__half) * kAttnChunk * (HD + 8),
                "merge area must fit in the K tile");
  extern __shared__ __align__(16) uint8_t smem_raw[];
  AttnSmemF16<HD>& sm = *reinterpret_cast<AttnSmemF16<HD>*>(smem_raw);
  pdl_launch_dependents();
  pdl_wait();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, cq = lane & 3;
  const int total = attn_item_prefix(a, sm.pre);
  const int group = a.H / a.Hkv;
  const int ldq = a.H * HD;
  const __half* Q = static_cast<const __half*>(a.q);
  const __half* KC = static_cast<const __half*>(a.k_cache);
  const __half* VC = static_cast<const __half*>(a.v_cache);
  float (*co)[kQTile][HD] = reinterpret_cast<float (*)[kQTile][HD]>(&sm.k[0][0]);

  for (int item = blockIdx.x; item < total; item += gridDim.x) {
    const int qi = attn_find_qtile(sm.pre, a.n_qtiles, item);
    const int local = item - sm.pre[qi];
    const int c = local / a.H, h = local - c * a.H;
    const int2 qt = a.qtiles[qi];
    const int b = qt.x, r0 = qt.y;
    const int nr = min(kQTile, a.seq_nrows[b] - r0);
    const int start = a.seq_start[b];
    const int row_g0 = a.seq_row0[b] + r0;
    const int pos0 = start + r0;  // position of tile row 0
    const int kb = c * kAttnChunk;
    int ke = min(kb + kAttnChunk, pos0 + nr);
    if (ke > a.max_seq) {
      if (tid == 0) atomicOr(a.err, DERR_CAPACITY);
      ke = a.max_seq;
    }
    const int kvh = h / group;
    const size_t kvbase = ((static_cast<size_t>(b) * a.Hkv + kvh) * a.max_seq) * HD;

    // ---- stage Q (16 rows), K and V (chunk rows) into shared memory ----
    constexpr int CPR = HD * 2 / 16;  // 16-byte pieces per row
    for (int i = tid; i < kQTile * CPR; i += 128) {
      const int rr = i / CPR, pc = i - rr * CPR;
      void* dst = &sm.q[rr][pc * 8];
      if (rr < nr)
        cp_async16(dst, Q + static_cast<size_t>(row_g0 + rr) * ldq + h * HD + pc * 8);
      else
        *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
    for (int i = tid; i < kAttnChunk * CPR; i += 128) {
      const int rr = i / CPR, pc = i - rr * CPR;
      const int key = kb + rr;
      void* dk = &sm.k[rr][pc * 8];
      void* dv = &sm.v[rr][pc * 8];
      if (key < ke) {
        const size_t off = kvbase + static_cast<size_t>(key) * HD + pc * 8;
        cp_async16(dk, KC + off);
        cp_async16(dv, VC + off);
      } else {
        *reinterpret_cast<uint4*>(dk) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(dv) = make_uint4(0, 0, 0, 0);
      }
    }
    cp_async_commit();
    cp_async_wait_all();
    __syncthreads();

    // ---- per warp: 32 keys x 16 rows ----
    const int wk0 = warp * 32;  // first key of this warp, relative to kb
    float o[HD / 8][4];
#pragma unroll
    for (int dn = 0; dn < HD / 8; ++dn) o[dn][0] = o[dn][1] = o[dn][2] = o[dn][3] = 0.f;
    float mA = -INFINITY, mB = -INFINITY, lA = 0.f, lB = 0.f;
    if (kb + wk0 < ke) {
      float s[4][4];
#pragma unroll
      for (int j = 0; j < 4; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
      for (int ks = 0; ks < HD / 16; ks += 2) {
        uint32_t qa0[4], qa1[4];
        ldmatrix_x4(qa0, &sm.q[lane & 15][ks * 16 + (lane >> 4) * 8]);
        ldmatrix_x4(qa1, &sm.q[lane & 15][(ks + 1) * 16 + (lane >> 4) * 8]);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          uint32_t kb4[4];
          const int mi = lane >> 3;
          ldmatrix_x4(kb4, &sm.k[wk0 + 8 * j + (lane & 7)][(ks + (mi >> 1)) * 16 + (mi & 1) * 8]);
          mma_f16_16816(s[j], qa0, kb4[0], kb4[1]);
          mma_f16_16816(s[j], qa1, kb4[2], kb4[3]);
        }
      }
      // mask + scale (log2 domain)
      const int posA = pos0 + g, posB = pos0 + g + 8;
      const bool rowA = g < nr, rowB = g + 8 < nr;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = kb + wk0 + 8 * j + 2 * cq + (e & 1);
          const bool top = e < 2;
          const bool valid = key < ke && (top ? (rowA && key <= posA) : (rowB && key <= posB));
          s[j][e] = valid ? s[j][e] * a.scale_log2 : -INFINITY;
        }
        mA = fmaxf(mA, fmaxf(s[j][0], s[j][1]));
        mB = fmaxf(mB, fmaxf(s[j][2], s[j][3]));
      }
      mA = fmaxf(mA, __shfl_xor_sync(0xffffffffu, mA, 1));
      mA = fmaxf(mA, __shfl_xor_sync(0xffffffffu, mA, 2));
      mB = fmaxf(mB, __shfl_xor_sync(0xffffffffu, mB, 1));
      mB = fmaxf(mB, __shfl_xor_sync(0xffffffffu, mB, 2));
      const float uA = (mA == -INFINITY) ? 0.f : mA;
      const float uB = (mB == -INFINITY) ? 0.f : mB;
      uint32_t pa[2][4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float p0 = exp2f(s[j][0] - uA), p1 = exp2f(s[j][1] - uA);
        const float p2 = exp2f(s[j][2] - uB), p3 = exp2f(s[j][3] - uB);
        lA += p0 + p1;
        lB += p2 + p3;
        pa[j >> 1][(j & 1) * 2 + 0] = pack_f16x2(p0, p1);
        pa[j >> 1][(j & 1) * 2 + 1] = pack_f16x2(p2, p3);
      }
      lA += __shfl_xor_sync(0xffffffffu, lA, 1);
      lA += __shfl_xor_sync(0xffffffffu, lA, 2);
      lB += __shfl_xor_sync(0xffffffffu, lB, 1);
      lB += __shfl_xor_sync(0xffffffffu, lB, 2);
      // O = P V: A fragments of P for keys 16kk..16kk+15 are the S accumulators
      // of n-tiles 2kk, 2kk+1 (a0: row g keys 2c.., a1: row g+8, a2/a3: +8 keys).
#pragma unroll
      for (int kk = 0; kk < 2; ++kk) {
        const uint32_t af[4] = {pa[kk][0], pa[kk][1], pa[kk][2], pa[kk][3]};
#pragma unroll
        for (int dn = 0; dn < HD / 8; dn += 2) {
          uint32_t vb[4];
          const int mi = lane >> 3;
          ldmatrix_x4_trans(vb, &sm.v[wk0 + 16 * kk + (mi & 1) * 8 + (lane & 7)][(dn + (mi >> 1)) * 8]);
          mma_f16_16816(o[dn], af, vb[0], vb[1]);
          mma_f16_16816(o[dn + 1], af, vb[2], vb[3]);
        }
      }
    }
    __syncthreads();  // every warp is done reading K/V before the merge area overwrites K
#pragma unroll
    for (int dn = 0; dn < HD / 8; ++dn) {
      const int d0 = dn * 8 + 2 * cq;
      co[warp][g][d0] = o[dn][0];
      co[warp][g][d0 + 1] = o[dn][1];
      co[warp][g + 8][d0] = o[dn][2];
      co[warp][g + 8][d0 + 1] = o[dn][3];
    }
    if (cq == 0) {
      sm.m[warp][g] = mA;
      sm.m[warp][g + 8] = mB;
      sm.l[warp][g] = lA;
      sm.l[warp][g + 8] = lB;
    }
    __syncthreads();
    {
      const int row = tid >> 3, part = tid & 7;
      constexpr int DPT = HD / 8;
      if (row < nr) {
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < 4; ++w) M = fmaxf(M, sm.m[w][row]);
        const size_t pidx = (static_cast<size_t>(row_g0 + row) * a.H + h) * a.nch_max + c;
        float* dst = a.part_o + pidx * HD + part * DPT;
        if (M == -INFINITY) {
#pragma unroll
          for (int dd = 0; dd < DPT; ++dd) dst[dd] = 0.f;
          if (part == 0) a.part_ml[pidx] = make_float2(-INFINITY, 0.f);
        } else {
          float f[4], l = 0.f;
#pragma unroll
          for (int w = 0; w < 4; ++w) {
            f[w] = exp2f(sm.m[w][row] - M);
            l += f[w] * sm.l[w][row];
          }
#pragma unroll
          for (int dd = 0; dd < DPT; ++dd) {
            const int d = part * DPT + dd;
            dst[dd] = ((f[0] * co[0][row][d] + f[1] * co[1][row][d]) + f[2] * co[2][row][d]) +
                      f[3] * co[3][row][d];
          }
          if (part == 0) a.part_ml[pidx] = make_float2(M, l);
        }
      }
    }
    __syncthreads();
  }
}

// fp32 (and generic) path: one warp per row, online softmax over the chunk.
template <typename Act, int HD>
__global__ void __launch_bounds__(128) attn_chunk_simt_kernel(const AttnArgs a) {
  __shared__ int pre[kMaxQTilesSmem + 1];
  pdl_launch_dependents();
  pdl_wait();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int total = attn_item_prefix(a, pre);
  const int group = a.H / a.Hkv;
  const int ldq = a.H * HD;
  constexpr int DPL = HD / 32;
  const Act* Q = static_cast<const Act*>(a.q);
  const Act* KC = static_cast<const Act*>(a.k_cache);
  const Act* VC = static_cast<const Act*>(a.v_cache);
  for (int item = blockIdx.x; item < total; item += gridDim.x) {
    const int qi = attn_find_qtile(pre, a.n_qtiles, item);
    const int local = item - pre[qi];
    const int c = local / a.H, h = local - c * a.H;
    const int2 qt = a.qtiles[qi];
    const int b = qt.x, r0 = qt.y;
    const int nr = min(kQTile, a.seq_nrows[b] - r0);
    const int start = a.seq_start[b];
    const int row_g0 = a.seq_row0[b] + r0;
    const int kb = c * kAttnChunk;
    const int kvh = h / group;
    const size_t kvbase = ((static_cast<size_t>(b) * a.Hkv + kvh) * a.max_seq) * HD;
    for (int i = warp; i < nr; i += 4) {
      const int pos = start + r0 + i;
      int kend = min(kb + kAttnChunk, pos + 1);
      if (kend > a.max_seq) {
        if (lane == 0) atomicOr(a.err, DERR_CAPACITY);
        kend = a.max_seq;
      }
      float q[DPL], o[DPL];
#pragma unroll
      for (int u = 0; u < DPL; ++u) {
        q[u] = ld_act(Q, static_cast<size_t>(row_g0 + i) * ldq + h * HD + lane + 32 * u);
        o[u] = 0.f;
      }
      float m = -INFINITY, l = 0.f;
      for (int key = kb; key < kend; ++key) {
        const size_t off = kvbase + static_cast<size_t>(key) * HD;
        float dot = 0.f;
#pragma unroll
        for (int u = 0; u < DPL; ++u) dot += q[u] * ld_act(KC, off + lane + 32 * u);
        const float s = warp_sum(dot) * a.scale_log2;
        const float mn = fmaxf(m, s);
        const float corr = exp2f(m - mn);  // m = -inf on the first key: corr = 0
        const float p = exp2f(s - mn);
        l = l * corr + p;
#pragma unroll
        for (int u = 0; u < DPL; ++u) o[u] = o[u] * corr + p * ld_act(VC, off + lane + 32 * u);
        m = mn;
      }
      const size_t pidx = (static_cast<size_t>(row_g0 + i) * a.H + h) * a.nch_max + c;
#pragma unroll
      for (int u = 0; u < DPL; ++u) a.part_o[pidx * HD + lane + 32 * u] = o[u];
      if (lane == 0) a.part_ml[pidx] = (kend > kb) ? make_float2(m, l) : make_float2(-INFINITY, 0.f);
    }
  }
}

// Merge of a row's chunk partials 0..pos/128 in chunk order; out = O / l.
template <typename Act>
__global__ void attn_combine_kernel(const AttnArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.x / a.H, h = blockIdx.x - (blockIdx.x / a.H) * a.H;
  if (t >= a.T) return;
  const int nch = min(a.pos[t] / kAttnChunk + 1, a.nch_max);
  const size_t base = (static_cast<size_t>(t) * a.H + h) * a.nch_max;
  float M = -INFINITY;
  for (int c = 0; c < nch; ++c) M = fmaxf(M, a.part_ml[base + c].x);
  for (int d = threadIdx.x; d < a.hd; d += blockDim.x) {
    float acc = 0.f, l = 0.f;
    for (int c = 0; c < nch; ++c) {
      const float2 ml = a.part_ml[base + c];
      const float f = exp2f(ml.x - M);
      l += f * ml.y;
      acc += f * a.part_o[(base + c) * a.hd + d];
    }
    st_gin(static_cast<Act*>(a.out), static_cast<size_t>(t) * a.H * a.hd + h * a.hd + d, a.plane_out,
           acc / l);
  }
}

// ---- launchers ----------------------------------------------------------------------

size_t attention_smem_bytes(int act_bf16, int hd) {
  if (!act_bf16) return 0;
  return hd == 64 ? sizeof(AttnSmemF16<64>) : sizeof(AttnSmemF16<128>);
}

cudaError_t attention_set_attributes() {
  cudaError_t e = cudaFuncSetAttribute(attn_chunk_mma_kernel<64>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(sizeof(AttnSmemF16<64>)));
  if (e != cudaSuccess) return e;
  for (const void* k : {reinterpret_cast<const void*>(attn_chunk_mma_kernel<64>),
                        reinterpret_cast<const void*>(attn_chunk_mma_kernel<128>)}) {
    e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout,
                             static_cast<int>(cudaSharedmemCarveoutMaxShared));
    if (e != cudaSuccess) return e;
  }
  return cudaFuncSetAttribute(attn_chunk_mma_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(sizeof(AttnSmemF16<128>)));
}

static void attn_cfg(cudaLaunchConfig_t& cfg, cudaLaunchAttribute* attr, dim3 grid, dim3 block,
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

cudaError_t launch_attention(const AttnArgs& a, int act_bf16, int grid, cudaStream_t s, bool pdl) {
  if (a.n_qtiles > kMaxQTilesSmem) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  if (act_bf16) {
    attn_cfg(cfg, attr, dim3(grid), dim3(128), attention_smem_bytes(1, a.hd), s, pdl);
    if (a.hd == 64) return cudaLaunchKernelEx(&cfg, attn_chunk_mma_kernel<64>, a);
    if (a.hd == 128) return cudaLaunchKernelEx(&cfg, attn_chunk_mma_kernel<128>, a);
    return cudaErrorInvalidValue;
  }
  attn_cfg(cfg, attr, dim3(grid), dim3(128), 0, s, pdl);
  if (a.hd == 64) return cudaLaunchKernelEx(&cfg, attn_chunk_simt_kernel<float, 64>, a);
  if (a.hd == 128) return cudaLaunchKernelEx(&cfg, attn_chunk_simt_kernel<float, 128>, a);
  return cudaErrorInvalidValue;
}

cudaError_t launch_attn_combine(const AttnArgs& a, int act_bf16, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  attn_cfg(cfg, attr, dim3(a.T * a.H), dim3(a.hd), 0, s, pdl);
  if (act_bf16) return cudaLaunchKernelEx(&cfg, attn_combine_kernel<__nv_bfloat16>, a);
  return cudaLaunchKernelEx(&cfg, attn_combine_kernel<float>, a);
}

}  // namespace cllm
