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

#include <type_traits>

#include "act.cuh"
#include "attn_item.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace cllm {

constexpr int kMaxQTilesSmem = 2048;

template <int HD>
struct AttnSmemF16 {
  AttnTileSmem<HD> t;
  int pre[kMaxQTilesSmem + 1];
};

struct CtaSync {
  __device__ void operator()() const { __syncthreads(); }
};

template <int HD>
__global__ void __launch_bounds__(128) attn_chunk_mma_kernel(const AttnArgs a) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  AttnSmemF16<HD>& sm = *reinterpret_cast<AttnSmemF16<HD>*>(smem_raw);
  pdl_launch_dependents();
  pdl_wait();
  const int total = attn_item_prefix(a, sm.pre, threadIdx.x, CtaSync{});
  for (int item = blockIdx.x; item < total; item += gridDim.x) {
    int qi, h;
    attn_mma_item<HD>(a, item, sm.pre, sm.t, threadIdx.x, CtaSync{}, qi, h, false);
  }
}

// The same items with Q, K and V tiles loaded by TMA from tensor maps (the
// persistent kernel's tile path; per-thread cp.async copies reach only a
// fraction of an SM's load bandwidth).
template <int HD>
constexpr size_t attn_tma_smem_bytes() {
  return 1024 + (sizeof(AttnTileSmemTma<HD>) + 15) / 16 * 16 + sizeof(int) * (kMaxQTilesSmem + 1);
}

template <int HD>
__global__ void __launch_bounds__(128) attn_chunk_tma_kernel(const __grid_constant__ AttnMaps m,
                                                             const AttnArgs a, int kv_row0) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base =
      reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  AttnTileSmemTma<HD>& t = *reinterpret_cast<AttnTileSmemTma<HD>*>(base);
  int* pre = reinterpret_cast<int*>(base + (sizeof(AttnTileSmemTma<HD>) + 15) / 16 * 16);
  pdl_launch_dependents();
  pdl_wait();
  const int total = attn_item_prefix(a, pre, threadIdx.x, CtaSync{});
  const AttnTma tma{&m.k, &m.v, &m.q, kv_row0};
  for (int item = blockIdx.x; item < total; item += gridDim.x) {
    int qi, h;
    attn_mma_item<HD>(a, item, pre, t, threadIdx.x, CtaSync{}, qi, h, GlobalMeta{a}, false, &tma);
  }
}

// fp32 (and generic) path: one warp per row, online softmax over the chunk.
template <typename Act, int HD>
__global__ void __launch_bounds__(128) attn_chunk_simt_kernel(const AttnArgs a) {
  __shared__ int pre[kMaxQTilesSmem + 1];
  pdl_launch_dependents();
  pdl_wait();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int total = attn_item_prefix(a, pre, threadIdx.x, CtaSync{}, 1);
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

// Merge of a row's partials (per chunk range) in order; out = O / l
// (fmaf accumulation in chunk order, as in the persistent kernel's merge).
// One (row, head) per hd/4 threads, 4 consecutive dims per thread (vector
// loads and stores); per element the same sums in the same order as a
// per-element loop.
template <typename Act>
__global__ void __launch_bounds__(128) attn_combine_kernel(const AttnArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  // the tensor-core path leaves one partial per range of kAttnRange chunks,
  // the fp32 path one per chunk
  constexpr int R = std::is_same<Act, float>::value ? 1 : kAttnRange;
  const int tpp = a.hd / 4;  // threads per (row, head)
  const int pair = blockIdx.x * (blockDim.x / tpp) + threadIdx.x / tpp;
  if (pair >= a.T * a.H) return;
  const int t = pair / a.H, h = pair - t * a.H;
  const int d = (threadIdx.x % tpp) * 4;
  const int nch = (min(a.pos[t] / kAttnChunk + 1, a.nch_max) + R - 1) / R;
  const size_t base = (static_cast<size_t>(t) * a.H + h) * a.nch_max;
  float M = -INFINITY;
  for (int c = 0; c < nch; ++c) M = fmaxf(M, a.part_ml[base + c].x);
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  float l = 0.f;
  for (int c = 0; c < nch; ++c) {
    const float2 ml = a.part_ml[base + c];
    const float f = exp2f(ml.x - M);
    l = fmaf(f, ml.y, l);
    const float4 o = *reinterpret_cast<const float4*>(a.part_o + (base + c) * a.hd + d);
    acc.x = fmaf(f, o.x, acc.x);
    acc.y = fmaf(f, o.y, acc.y);
    acc.z = fmaf(f, o.z, acc.z);
    acc.w = fmaf(f, o.w, acc.w);
  }
  st_gin4(static_cast<Act*>(a.out), static_cast<size_t>(t) * a.H * a.hd + h * a.hd + d, a.plane_out,
          make_float4(acc.x / l, acc.y / l, acc.z / l, acc.w / l));
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
  e = cudaFuncSetAttribute(attn_chunk_mma_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(sizeof(AttnSmemF16<128>)));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(attn_chunk_tma_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(attn_tma_smem_bytes<64>()));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_chunk_tma_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(attn_tma_smem_bytes<128>()));
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

cudaError_t launch_attention_tma(const AttnArgs& a, const AttnMaps& m, int kv_row0, int grid,
                                 cudaStream_t s, bool pdl) {
  if (a.n_qtiles > kMaxQTilesSmem) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  if (a.hd == 64) {
    attn_cfg(cfg, attr, dim3(grid), dim3(128), attn_tma_smem_bytes<64>(), s, pdl);
    return cudaLaunchKernelEx(&cfg, attn_chunk_tma_kernel<64>, m, a, kv_row0);
  }
  if (a.hd == 128) {
    attn_cfg(cfg, attr, dim3(grid), dim3(128), attn_tma_smem_bytes<128>(), s, pdl);
    return cudaLaunchKernelEx(&cfg, attn_chunk_tma_kernel<128>, m, a, kv_row0);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_attn_combine(const AttnArgs& a, int act_bf16, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  const int per_block = 128 / (a.hd / 4);  // (row, head) pairs per 128-thread block
  attn_cfg(cfg, attr, dim3((a.T * a.H + per_block - 1) / per_block), dim3(128), 0, s, pdl);
  if (act_bf16) return cudaLaunchKernelEx(&cfg, attn_combine_kernel<__nv_bfloat16>, a);
  return cudaLaunchKernelEx(&cfg, attn_combine_kernel<float>, a);
}

}  // namespace cllm
