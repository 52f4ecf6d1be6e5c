// Per-iteration kernels around the block forward:
//   embed       - token rows of the block (or of a prefill) -> fp32 residual
//                 stream, first RMSNorm input and per-tile sums of squares,
//                 plus each row's position and sequence index
//   accept      - the fixed-point test of Alg. 3: longest prefix of the block
//                 reproduced by the predictions, commit (advance the committed
//                 length; the K/V already sit in the cache), new head, refill
//   decode_init - reset a decode to the prefill state, draw the first guesses
// Guesses come from a counter-based splitmix64 stream (Vigna): the
// ((b<<40 | iteration<<16 | slot) + 1)-th output for key `seed`.
#include "act.cuh"
#include "internal.cuh"
#include "ptx.cuh"
#include "step_items.cuh"

namespace cllm {

struct StepSync {
  __device__ void operator()() const { __syncthreads(); }
};

template <typename Act>
__global__ void __launch_bounds__(128) embed_kernel(const EmbedArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ float red[4];
  embed_unit<Act>(a, blockIdx.x, blockIdx.y, threadIdx.x, red, StepSync{});
}

__global__ void __launch_bounds__(128) accept_kernel(const AcceptArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ int s_act[4], s_com[4];
  accept_body(a, threadIdx.x, s_act, s_com, StepSync{});
}

__global__ void __launch_bounds__(128) decode_init_kernel(const AcceptArgs a) {
  const int tid = threadIdx.x;
  for (int b = tid; b < a.B; b += blockDim.x) {
    a.L[b] = a.plen[b];
    a.committed[b] = 0;
    a.iters[b] = 0;
    a.done[b] = 0;
    if (a.width != nullptr) a.width[b] = a.n;
    int* y = a.block + b * a.n;
    y[0] = a.head[b];
    for (int k = 1; k < a.n; ++k) y[k] = draw_guess(a, b, 0, k);
    if (a.acc_hist != nullptr) {
      a.win_end[b] = 0;
      a.win_cnt[b] = 0;
      for (int k = 0; k < a.n; ++k) a.st_pos[static_cast<size_t>(b) * a.n + k] = -1;
    }
  }
  if (a.acc_hist != nullptr) {
    for (int i = tid; i <= a.n; i += blockDim.x) {
      a.acc_hist[i] = 0;
      a.win_hist[i] = 0;
    }
    if (tid < 2) a.totals[tid] = 0;
  }
  for (size_t i = tid; i < static_cast<size_t>(a.B) * a.max_new; i += blockDim.x) a.out[i] = -1;
  if (tid == 0) {
    a.status[0] = a.B;
    a.status[1] = 0;
  }
}

__global__ void set_head_kernel(int* block, const int* head, int B, int n, int V, int* err) {
  const int b = threadIdx.x;
  if (b < B) {
    const int h = head[b];
    if (h < 0 || h >= V) atomicOr(err, DERR_TOKEN);
    block[b * n] = h;
  }
}

template <typename Act>
__global__ void gather_rows_kernel(const Act* xg_src, const float* ssq_src, Act* xg_dst,
                                   float* ssq_dst, const int* rows, int d, int ldt_src,
                                   int ldt_dst, size_t plane_src, size_t plane_dst) {
  const int b = blockIdx.x;
  const int row = rows[b];
  for (int m = threadIdx.x; m < d; m += blockDim.x) {
    xg_dst[static_cast<size_t>(b) * d + m] = xg_src[static_cast<size_t>(row) * d + m];
    if (plane_dst)
      xg_dst[plane_dst + static_cast<size_t>(b) * d + m] =
          xg_src[plane_src + static_cast<size_t>(row) * d + m];
  }
  for (int i = threadIdx.x; i < d / 128; i += blockDim.x)
    ssq_dst[static_cast<size_t>(i) * ldt_dst + b] = ssq_src[static_cast<size_t>(i) * ldt_src + row];
}

// ---- launchers ----------------------------------------------------------------------

static void small_cfg(cudaLaunchConfig_t& cfg, cudaLaunchAttribute* attr, dim3 grid, dim3 block,
                      cudaStream_t s, bool pdl) {
  cfg = cudaLaunchConfig_t{};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
}

cudaError_t launch_embed(const EmbedArgs& a, int act_bf16, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  small_cfg(cfg, attr, dim3(a.T, a.d / 128), dim3(128), s, pdl);
  if (act_bf16) return cudaLaunchKernelEx(&cfg, embed_kernel<__nv_bfloat16>, a);
  return cudaLaunchKernelEx(&cfg, embed_kernel<float>, a);
}

cudaError_t launch_accept(const AcceptArgs& a, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg;
  cudaLaunchAttribute attr[1];
  small_cfg(cfg, attr, dim3(1), dim3(128), s, pdl);
  return cudaLaunchKernelEx(&cfg, accept_kernel, a);
}

cudaError_t launch_decode_init(const AcceptArgs& a, cudaStream_t s) {
  decode_init_kernel<<<1, 128, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_set_head(int* block, const int* head, int B, int n, int V, int* err,
                            cudaStream_t s) {
  set_head_kernel<<<1, 128, 0, s>>>(block, head, B, n, V, err);
  return cudaGetLastError();
}

cudaError_t launch_gather_rows(const void* xg_src, const float* ssq_src, void* xg_dst,
                               float* ssq_dst, const int* rows, int B, int d, int ldt_src,
                               int ldt_dst, size_t plane_src, size_t plane_dst, int act_bf16,
                               cudaStream_t s) {
  if (act_bf16)
    gather_rows_kernel<__nv_bfloat16><<<B, 256, 0, s>>>(
        static_cast<const __nv_bfloat16*>(xg_src), ssq_src, static_cast<__nv_bfloat16*>(xg_dst),
        ssq_dst, rows, d, ldt_src, ldt_dst, plane_src, plane_dst);
  else
    gather_rows_kernel<float><<<B, 256, 0, s>>>(static_cast<const float*>(xg_src), ssq_src,
                                                static_cast<float*>(xg_dst), ssq_dst, rows, d,
                                                ldt_src, ldt_dst, 0, 0);
  return cudaGetLastError();
}

}  // namespace cllm
