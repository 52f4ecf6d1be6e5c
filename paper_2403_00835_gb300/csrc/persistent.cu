// Persistent per-iteration kernel: one Jacobi iteration (embed, every decoder
// layer's QKV GEMM / attention / O GEMM / gate-up GEMM / down GEMM, the LM
// head and the accept step) as one launch of one CTA per SM.
//
// Phases run in order from a table in global memory.  Phase p may start only
// when every CTA has finished phases 0..p-1: a grid barrier on a monotonic
// counter (each CTA's epilogue warps add 1 after each phase; waits are
// bounded and poll `counter >= p * gridDim`).  The TMA producer streams the
// next GEMM phase's weight tiles into the shared-memory ring before that
// barrier opens -- weights do not depend on the previous phase -- so HBM keeps
// streaming while a phase drains (split-K reductions, epilogues, attention).
// Work split, reductions and epilogues are those of the per-GEMM kernels
// (gemm_roles.cuh), so the results are bit-identical to that path.
#include "attn_item.cuh"
#include "gemm_roles.cuh"
#include "step_items.cuh"

namespace cllm {

namespace {

struct EpiGroupSync {
  __device__ void operator()() const { named_bar_sync(1, 128); }
};

__host__ __device__ constexpr size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

template <int BNMAX, int HD>
struct PersistCfg {
  static constexpr size_t ATTN_BYTES = align_up(sizeof(AttnTileSmemTma<HD>), 1024);
  // the GEMM epilogue's part of the union: EpiSmem, then split-K staging
  // blocks (at least 4; as many as fit beside the attention tile)
  static constexpr size_t EPI_BYTES = align_up(sizeof(EpiSmem), 16);
  static constexpr size_t EPI_MIN = EPI_BYTES + 4 * kRedSlotBytes;
  static constexpr size_t UNION = align_up(ATTN_BYTES > EPI_MIN ? ATTN_BYTES : EPI_MIN, 16);
  static constexpr int RED_SLOTS = static_cast<int>((UNION - EPI_BYTES) / kRedSlotBytes);
  // the attention work-item prefix and the iteration's metadata, outside the
  // union: computed at the first attention phase, kept for every layer
  static constexpr size_t PRE_BYTES = align_up(4 * (kMaxQTilesStep + 1), 16);
  static constexpr size_t META_BYTES = PRE_BYTES + align_up(sizeof(AttnMetaSmem), 16);
  static constexpr int STAGE_BYTES = kBM * kBK * 2 + 2 * BNMAX * kBK * 2;
  static constexpr size_t BUDGET = 227 * 1024 - 256;  // minus the kernel's static shared memory
  static constexpr size_t FIXED = 1024 + UNION + META_BYTES + tc_bar_bytes(8) + 64;
  static constexpr int FIT = static_cast<int>((BUDGET - FIXED) / STAGE_BYTES);
  static constexpr int STAGES = FIT > 8 ? 8 : FIT;
  using Cfg = TcCfg<BNMAX, STAGES>;
  static constexpr size_t SMEM = 1024 + static_cast<size_t>(STAGES) * STAGE_BYTES + UNION +
                                 META_BYTES + tc_bar_bytes(STAGES) + 64;
  static_assert(STAGES >= 2, "ring too small");
  static_assert(SMEM <= BUDGET, "shared memory over budget");
};

// The phase's arguments are copied into registers first: read through a
// reference into the phase table, every asm statement with a memory clobber
// (TMA issue, mbarrier operations) would force them to be reloaded.
template <class Cfg, class Dep>
__device__ bool produce_phase(const TcPipe& P, int& idx, int& issued, const PhaseDesc& ph,
                              const CUtensorMap* maps, int cta, const Dep& dep) {
  const GemmArgs g = ph.g;
  const int epi = ph.epi;
  const CUtensorMap* m0 = maps + ph.map_a0;
  const CUtensorMap* m1 = maps + ph.map_a1;
  const CUtensorMap* m2 = maps + ph.map_a2;
  const CUtensorMap* mb = maps + ph.map_b;
  int c0, c1;
  cta_range(g, cta, c0, c1);
  switch (epi) {
    case EPI_QKV: return tc_produce<EPI_QKV, Cfg>(P, idx, issued, g, m0, m1, m2, mb, c0, c1, dep);
    case EPI_GATEUP:
      return tc_produce<EPI_GATEUP, Cfg>(P, idx, issued, g, m0, m1, m2, mb, c0, c1, dep);
    case EPI_RESID:
      return tc_produce<EPI_RESID, Cfg>(P, idx, issued, g, m0, m1, m2, mb, c0, c1, dep);
    default: return tc_produce<EPI_ARGMAX, Cfg>(P, idx, issued, g, m0, m1, m2, mb, c0, c1, dep);
  }
}

template <class Cfg>
__device__ bool epilogue_phase(const TcPipe& P, int& acc, uint32_t& accph, const PhaseDesc& ph,
                               int cta, EpiSmem& es) {
  const GemmArgs g = ph.g;
  const EpiArgs e = ph.e;
  const int epi = ph.epi;
  int c0, c1;
  cta_range(g, cta, c0, c1);
  switch (epi) {
    case EPI_QKV: return tc_epilogue<EPI_QKV, Cfg>(P, acc, accph, g, e, c0, c1, cta, es);
    case EPI_GATEUP: return tc_epilogue<EPI_GATEUP, Cfg>(P, acc, accph, g, e, c0, c1, cta, es);
    case EPI_RESID: return tc_epilogue<EPI_RESID, Cfg>(P, acc, accph, g, e, c0, c1, cta, es);
    default: return tc_epilogue<EPI_ARGMAX, Cfg>(P, acc, accph, g, e, c0, c1, cta, es);
  }
}

// Arrivals the grid barrier must count before phase p starts: every CTA
// arrives once after each earlier phase.  (The hold hook asks for one more.)
__device__ __forceinline__ unsigned barrier_target(const StepArgs& A, int p, int G) {
  return static_cast<unsigned>(p) * static_cast<unsigned>(G) + (p == A.hold_phase ? 1u : 0u);
}

template <class Cfg>
__device__ bool mma_phase(const TcPipe& P, int& idx, int& acc, uint32_t& accph, const PhaseDesc& ph,
                          int cta, unsigned long long* prof, long long prof_stride,
                          unsigned long long* trace) {
  const GemmArgs g = ph.g;
  int c0, c1;
  cta_range(g, cta, c0, c1);
  return tc_mma<Cfg>(P, idx, acc, accph, g, c0, c1, prof, prof_stride, trace);
}

}  // namespace

template <int BNMAX, int HD>
__global__ void __launch_bounds__(192, 1)
    step_persistent_kernel(const __grid_constant__ StepParams PRM) {
  const StepArgs& A = PRM.a;
  using PC = PersistCfg<BNMAX, HD>;
  using Cfg = typename PC::Cfg;
  extern __shared__ uint8_t smem_raw[];
  __shared__ float s_red[4];
  __shared__ int s_act[4], s_com[4];
  __shared__ int s_flag;
  uint8_t* base =
      reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* uni = base + static_cast<size_t>(Cfg::STAGES) * Cfg::STAGE_BYTES;
  EpiSmem& es = *reinterpret_cast<EpiSmem*>(uni);
  AttnTileSmemTma<HD>& at = *reinterpret_cast<AttnTileSmemTma<HD>*>(uni);  // 1024-aligned
  int* pre = reinterpret_cast<int*>(uni + PC::UNION);
  AttnMetaSmem& meta = *reinterpret_cast<AttnMetaSmem*>(uni + PC::UNION + PC::PRE_BYTES);
  uint8_t* bars = uni + PC::UNION + PC::META_BYTES;
  TcPipe P = tc_pipe_init<Cfg>(base, bars);
  P.red = reinterpret_cast<float*>(uni + PC::EPI_BYTES);
  P.red_slots = PC::RED_SLOTS;
  const int G = gridDim.x, cta = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      int idx = 0, issued = 0;
      for (int p = 0; p < A.n_phases; ++p) {
        const PhaseDesc& ph = A.phases[p];
        if (ph.kind != PH_GEMM) continue;
        const GridDep dep{A.bar, barrier_target(A, p, G)};
        const size_t PG = static_cast<size_t>(A.n_phases) * G;
        unsigned long long* cs =
            A.cta_stamps != nullptr ? A.cta_stamps + static_cast<size_t>(p) * G + cta : nullptr;
        if (cs != nullptr) cs[6 * PG] = globaltimer_ns();
        const bool ok = produce_phase<Cfg>(P, idx, issued, ph, PRM.maps, cta, dep);
        if (cs != nullptr) cs[8 * PG] = globaltimer_ns();
        if (!ok) break;
      }
      tc_produce_drain<Cfg>(P, issued);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int idx = 0, acc = 0;
      uint32_t accph = 0;
      for (int p = 0; p < A.n_phases; ++p) {
        const PhaseDesc& ph = A.phases[p];
        if (ph.kind != PH_GEMM) continue;
        unsigned long long* prof = nullptr;
        unsigned long long* trace = nullptr;
        const long long PG = static_cast<long long>(A.n_phases) * G;
        if (A.cta_stamps != nullptr) {
          prof = A.cta_stamps + 10 * PG + static_cast<long long>(p) * G + cta;
          if (p == A.trace_phase)
            trace = A.cta_stamps + kCtaStampSlots * PG + static_cast<long long>(cta) * kTraceCap;
        }
        if (!mma_phase<Cfg>(P, idx, acc, accph, ph, cta, prof, PG, trace)) break;
        if (A.cta_stamps != nullptr)
          A.cta_stamps[(static_cast<size_t>(A.n_phases) + p) * G + cta] = globaltimer_ns();
      }
      tc_mma_drain(P);
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
      if (p > 0) {
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
        ok = epilogue_phase<Cfg>(P, acc, accph, ph, cta, es);
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
        for (int item = cta; item < total; item += G) {
          int qi, h;
          if (attn_mma_item<HD>(a, item, pre, at, r, sync, qi, h, md, true, &tma))
            continue;  // output written
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
        }
      }
    }
    if (A.stamps != nullptr && cta == 0 && r == 0) A.stamps[A.n_phases] = globaltimer_ns();
  }
  tc_pipe_release<Cfg>(P);
  if (threadIdx.x == 0 && *P.abort) atomicOr(A.err, DERR_TIMEOUT);
}

// ---- launch ----------------------------------------------------------------------------

size_t step_persistent_smem_bytes(int bn_max, int hd) {
  if (hd == 64) {
    switch (bn_max) {
      case 32: return PersistCfg<32, 64>::SMEM;
      case 64: return PersistCfg<64, 64>::SMEM;
      default: return PersistCfg<128, 64>::SMEM;
    }
  }
  switch (bn_max) {
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
  if ((e = set_one<32, 64>()) != cudaSuccess) return e;
  if ((e = set_one<64, 64>()) != cudaSuccess) return e;
  if ((e = set_one<128, 64>()) != cudaSuccess) return e;
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
  cfg.blockDim = dim3(192);
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
      case 32: return launch_one<32, 64>(a, grid, s, cooperative);
      case 64: return launch_one<64, 64>(a, grid, s, cooperative);
      case 128: return launch_one<128, 64>(a, grid, s, cooperative);
      default: return cudaErrorInvalidValue;
    }
  }
  if (hd == 128) {
    switch (bn_max) {
      case 32: return launch_one<32, 128>(a, grid, s, cooperative);
      case 64: return launch_one<64, 128>(a, grid, s, cooperative);
      case 128: return launch_one<128, 128>(a, grid, s, cooperative);
      default: return cudaErrorInvalidValue;
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace cllm
