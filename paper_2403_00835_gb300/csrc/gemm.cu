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

#define CLLM_EPI_GROUPS 1  // kernels of this unit may run two epilogue groups
#include "act.cuh"
#include "epilogue.cuh"
#include "gemm_roles.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace cllm {

// ---------------------------------------------------------------------------------
// tcgen05 kernel (bf16): one GEMM per launch
// ---------------------------------------------------------------------------------

// One CTA per SM with as many stages as fit: the weight stream is
// latency-bound by the bytes in flight per SM (~45 GB/s per SM at ~1.8 us
// loaded DRAM latency needs > 80 KB in flight).
template <int BNMAX>
using SoloCfg = TcCfg<BNMAX, BNMAX <= 32 ? 8 : (BNMAX <= 64 ? 6 : (BNMAX <= 128 ? 4 : 2))>;

constexpr int kSoloRedSlots = 2;  // split-K partial blocks staged per reduction round

// Epilogue groups: at 256 token columns one accumulator fills tensor memory,
// so the MMAs of a CTA's next unit wait for the whole epilogue of the last
// one (16 chunks); a second group of 4 warps halves that wait.
template <int KIND, int BNMAX>
constexpr int solo_groups() { return BNMAX == 256 ? 2 : 1; }

constexpr size_t kSoloGroupBytes = (sizeof(EpiSmem) + 15) / 16 * 16 + kSoloRedSlots * kRedSlotBytes;

template <int BNMAX>
constexpr size_t solo_smem_bytes() {
  using Cfg = SoloCfg<BNMAX>;
  constexpr int groups = BNMAX == 256 ? 2 : 1;  // room for two groups at 256 columns
  return 1024 + static_cast<size_t>(Cfg::STAGES) * Cfg::STAGE_BYTES + groups * kSoloGroupBytes + 16 +
         tc_bar_bytes(Cfg::STAGES) + 16;
}
constexpr size_t kSmemLimit = 227 * 1024 - 256;  // minus static shared memory
static_assert(solo_smem_bytes<32>() <= kSmemLimit && solo_smem_bytes<64>() <= kSmemLimit &&
                  solo_smem_bytes<128>() <= kSmemLimit && solo_smem_bytes<256>() <= kSmemLimit,
              "per-GEMM kernel shared memory over the 227 KB limit");

template <int KIND, int BNMAX>
__global__ void __launch_bounds__(64 + 128 * solo_groups<KIND, BNMAX>(), 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap mA0, const __grid_constant__ CUtensorMap mA1,
                   const __grid_constant__ CUtensorMap mA2, const __grid_constant__ CUtensorMap mB,
                   const GemmArgs g, const EpiArgs e) {
  using Cfg = SoloCfg<BNMAX>;
  constexpr int NG = solo_groups<KIND, BNMAX>();
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base =
      reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // [ring][per group: EpiSmem, staging slots][barriers][shared flags, 16 bytes]
  uint8_t* groups = base + Cfg::STAGES * Cfg::STAGE_BYTES;
  uint8_t* bars = groups + (BNMAX == 256 ? 2 : 1) * kSoloGroupBytes;
  int* jflag = reinterpret_cast<int*>(bars + tc_bar_bytes(Cfg::STAGES));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mA0);
    tma_prefetch_desc(&mA1);
    tma_prefetch_desc(&mA2);
    tma_prefetch_desc(&mB);
  }
  TcPipe P = tc_pipe_init<Cfg, NG>(base, bars);
  P.red_slots = kSoloRedSlots;
  P.jflag = jflag;
  // Every CTA of this grid is resident (one per SM): let the next kernel in
  // the stream start its independent prologue now.
  pdl_launch_dependents();
  int c0, c1;
  cta_range(g, blockIdx.x, c0, c1);
  if (warp == 0) {
    if (lane == 0) {
      int idx = 0, issued = 0;
      tc_produce<KIND, Cfg>(P, idx, issued, g, &mA0, &mA1, &mA2, &mB, c0, c1, PdlDep{});
      tc_produce_drain<Cfg>(P, issued);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int idx = 0, acc = 0;
      uint32_t accph = 0;
      tc_mma<Cfg>(P, idx, acc, accph, g, c0, c1);
      tc_mma_drain(P);
    }
  } else {
    pdl_wait();
    const int gi = (warp - 2) / 4;  // epilogue group
    uint8_t* mine = groups + gi * kSoloGroupBytes;
    EpiSmem& es = *reinterpret_cast<EpiSmem*>(mine);
    TcPipe Pg = P;
    Pg.red = reinterpret_cast<float*>(mine + (sizeof(EpiSmem) + 15) / 16 * 16);
    int acc = 0;
    uint32_t accph = 0;
    tc_epilogue<KIND, Cfg, NG>(Pg, acc, accph, g, e, c0, c1, blockIdx.x, es);
  }
  tc_pipe_release<Cfg>(P);
  if (threadIdx.x == 0 && *P.abort) atomicOr(g.err, DERR_TIMEOUT);
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
  if (r == 0) es.prepared = 0;
  __syncthreads();
  epi_apply<KIND, float>(e, mt, t0, acc, r, es);
  if (KIND == EPI_ARGMAX) epi_argmax_finish(e, r, es);
}

// ---------------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------------

int gemm_tc_stages(int bn_max) {
  switch (bn_max) {
    case 32: return SoloCfg<32>::STAGES;
    case 64: return SoloCfg<64>::STAGES;
    case 128: return SoloCfg<128>::STAGES;
    default: return SoloCfg<256>::STAGES;
  }
}

size_t gemm_tc_smem_bytes(int bn_max) {
  switch (bn_max) {
    case 32: return solo_smem_bytes<32>();
    case 64: return solo_smem_bytes<64>();
    case 128: return solo_smem_bytes<128>();
    default: return solo_smem_bytes<256>();
  }
}

template <int KIND, int BN>
static cudaError_t set_attr_one() {
  cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<KIND, BN>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(solo_smem_bytes<BN>()));
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
  fill_launch(cfg, attr, dim3(grid), dim3(64 + 128 * solo_groups<KIND, BN>()), solo_smem_bytes<BN>(), s, pdl);
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
