// Allocation-free variant of the weight-streaming GEMM (cllm_gemm_bf16_noalloc).
//
// Some callers cannot call cudaMalloc: code running under a caching allocator
// that has reserved the device's memory for itself, or a latency-critical
// path where the implicit device synchronisation of cudaMalloc/cudaFree is
// not acceptable.  This entry point runs the same tcgen05/TMA GEMM kernel as
// the rest of the library, but every byte of scratch it needs (split-K
// partial tiles, arrival tickets, the device error word, and the epilogue's
// side outputs) lives in one file-scope device array of fixed size, so the
// call allocates nothing.  The caller still provides the inputs and output.
#include "../../include/cllm.h"
#include "internal.cuh"

using namespace cllm;

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(8) << 20;  // 8 MiB, held by each device until exit

// One array per device that loads the library.  In host code this name is
// only a stand-in: its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of the scratch array in the current device's current
// context.  It is looked up on every call (a host-side table lookup, cheap):
// an address cached per device would be stale after cudaDeviceReset or in a
// second driver context on the same device, and the kernel would then write
// its partial sums into memory it does not own.  The first call in a context
// also loads the library's device code there.
int scratch_address(void** out) {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return CLLM_ECUDA;
  *out = p;
  return CLLM_OK;
}

__global__ void fill_bf16_one(__nv_bfloat16* p, int n) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x)
    p[i] = __float2bfloat16(1.f);
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

}  // namespace

extern "C" int cllm_gemm_bf16_noalloc(const void* W, const void* X, float* Y, int M, int K, int T,
                                      int x_rows, void* cuda_stream) {
  if (!W || !X || !Y || M < 128 || M % 128 || K < 8 || K % 8 || T < 1) return CLLM_EINVAL;
  if (x_rows < round_up(T, 16) || (T > 256 && x_rows < 256)) return CLLM_EINVAL;
  if ((reinterpret_cast<uintptr_t>(W) | reinterpret_cast<uintptr_t>(X) |
       reinterpret_cast<uintptr_t>(Y)) & 15u)
    return CLLM_EINVAL;
  // the call synchronises its stream and reads the error word back, which a
  // stream capture cannot hold: refuse before touching the stream
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(static_cast<cudaStream_t>(cuda_stream), &cap) != cudaSuccess)
    return CLLM_ECUDA;
  if (cap != cudaStreamCaptureStatusNone) return CLLM_EUNSUPPORTED;
  int dev = 0;
  cudaDeviceProp prop;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaGetDeviceProperties(&prop, dev) != cudaSuccess)
    return CLLM_ECUDA;
  if (prop.major != 10 || prop.minor != 3) return CLLM_EUNSUPPORTED;
  const int mtiles = M / kBM;
  const Part p = plan_gemm(mtiles, K, T, prop.multiProcessorCount);
  const int ldt = round_up(T, 16);
  // scratch layout inside the static array
  const size_t off_part = 0;
  const size_t sz_part = align256(static_cast<size_t>(mtiles) * p.maxc * p.bn * kBM * 4);
  const size_t off_tick = off_part + sz_part;
  const size_t sz_tick = align256(static_cast<size_t>(mtiles) * 4);
  const size_t off_err = off_tick + sz_tick;
  const size_t off_ssq = off_err + 256;
  const size_t sz_ssq = align256(static_cast<size_t>(mtiles) * ldt * 4);
  const size_t off_xg = off_ssq + sz_ssq;
  const size_t sz_xg = align256(static_cast<size_t>(2) * T * M * 2);
  const size_t off_one = off_xg + sz_xg;
  const size_t total = off_one + align256(static_cast<size_t>(M) * 2);
  if (total > kNoAllocScratchBytes) return CLLM_ECAPACITY;

  void* base = nullptr;
  int rc = scratch_address(&base);
  if (rc != CLLM_OK) return rc;
  char* sb = static_cast<char*>(base);
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  if (gemm_tc_set_attributes() != cudaSuccess) return CLLM_ECUDA;
  GemmMaps maps{};
  if (!make_map(&maps.a0, W, K, M, kBM) || !make_map(&maps.b, X, K, 2 * x_rows, p.bn))
    return CLLM_EINVAL;
  maps.a1 = maps.a2 = maps.a0;
  // the array keeps the previous call's contents: tickets and the error word
  // must start at zero
  if (cudaMemsetAsync(sb + off_tick, 0, sz_tick, s) != cudaSuccess ||
      cudaMemsetAsync(sb + off_err, 0, 256, s) != cudaSuccess)
    return CLLM_ECUDA;
  fill_bf16_one<<<ceil_div(M, 256), 256, 0, s>>>(reinterpret_cast<__nv_bfloat16*>(sb + off_one), M);
  if (cudaGetLastError() != cudaSuccess) return CLLM_ECUDA;

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
  g.l2_ahead = kL2AheadDefault;  // as the allocating GEMM entry points
  g.pre_stages = 1 << 20;
  g.partial = reinterpret_cast<float*>(sb + off_part);
  g.tickets = reinterpret_cast<int*>(sb + off_tick);
  g.err = reinterpret_cast<int*>(sb + off_err);
  EpiArgs e{};
  e.T = T;
  e.ldt = ldt;
  e.x = Y;
  e.xg = sb + off_xg;
  e.gnext = sb + off_one;
  e.plane_x = static_cast<size_t>(T) * M;
  e.ssq_out = reinterpret_cast<float*>(sb + off_ssq);
  e.d = M;
  e.err = g.err;
  if (launch_gemm_tc(EPI_RESID, p.bn_max, maps, g, e, p.grid, s, false) != cudaSuccess)
    return CLLM_ECUDA;
  int herr = 0;
  if (cudaMemcpyAsync(&herr, g.err, sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return CLLM_ECUDA;
  if (herr) return (herr & DERR_TIMEOUT) ? CLLM_ETIMEOUT : CLLM_EDEVICE;
  return CLLM_OK;
}
