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

namespace cllm {

__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t i) {
  uint64_t z = seed + i * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ int draw_guess(const AcceptArgs& a, int b, int step, int slot) {
  const uint64_t ctr = (static_cast<uint64_t>(b) << 40) | (static_cast<uint64_t>(step) << 16) |
                       static_cast<uint64_t>(slot);
  const uint64_t r = splitmix64_at(a.seed, ctr + 1) >> 32;
  if (a.guess_mode == 1) {
    const int len = a.plen[b];
    return a.prompts[static_cast<size_t>(b) * a.prompt_ld + ((r * static_cast<uint64_t>(len)) >> 32)];
  }
  return static_cast<int>((r * static_cast<uint64_t>(a.V)) >> 32);
}

template <typename Act>
__global__ void __launch_bounds__(128) embed_kernel(const EmbedArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.x, grp = blockIdx.y, i = threadIdx.x;
  const int m = grp * 128 + i;
  int tok, pos, b;
  if (a.block != nullptr) {
    b = t / a.n;
    const int k = t - b * a.n;
    tok = a.block[b * a.n + k];
    pos = a.L[b] + k;
  } else {
    tok = a.tok_in[t];
    pos = a.pos_in[t];
    b = a.bidx_in[t];
  }
  if (tok < 0 || tok >= a.V) {
    if (i == 0 && grp == 0) atomicOr(a.err, DERR_TOKEN);
    tok = 0;
  }
  const float e = ld_act(static_cast<const Act*>(a.emb), static_cast<size_t>(tok) * a.d + m);
  const size_t o = static_cast<size_t>(t) * a.d + m;
  a.x[o] = e;
  st_gin(static_cast<Act*>(a.xg), o, a.plane, e * ld_act(static_cast<const Act*>(a.gain), m));
  __shared__ float red[4];
  const float s = warp_sum(e * e);
  if ((i & 31) == 0) red[i >> 5] = s;
  __syncthreads();
  if (i == 0) a.ssq[static_cast<size_t>(grp) * a.ldt + t] = ((red[0] + red[1]) + red[2]) + red[3];
  if (grp == 0 && i == 0) {
    if (pos < 0 || pos >= a.max_seq) atomicOr(a.err, DERR_CAPACITY);
    a.pos[t] = pos;
    a.bidx[t] = b;
  }
  if (a.block != nullptr && t == 0 && grp == 0) {
    for (int bb = i; bb < a.B; bb += blockDim.x) {
      a.seq_start[bb] = a.L[bb];
      a.seq_row0[bb] = bb * a.n;
      a.seq_nrows[bb] = a.n;
    }
  }
}

__global__ void __launch_bounds__(128) accept_kernel(const AcceptArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const int b = threadIdx.x;
  int active = 0, committed_now = 0;
  if (b < a.B) {
    const int n = a.n;
    const int* P = a.pred + b * n;
    int* y = a.block + b * n;
    if (!(a.decode && a.done[b])) {
      int acc = 1;
      while (acc < n && y[acc] == P[acc - 1]) ++acc;
      if (a.decode) {
        bool stop = false;
        if (a.eos >= 0) {
          for (int k = 0; k < acc; ++k)
            if (y[k] == a.eos) {
              acc = k + 1;
              stop = true;
              break;
            }
        }
        const int room = a.max_new - a.committed[b];
        if (acc > room) acc = room;
        int* out = a.out + static_cast<size_t>(b) * a.max_new + a.committed[b];
        for (int k = 0; k < acc; ++k) out[k] = y[k];
        a.committed[b] += acc;
        a.iters[b] += 1;
        if (stop || a.committed[b] >= a.max_new) a.done[b] = 1;
        active = a.done[b] ? 0 : 1;
        committed_now = acc;
      }
      a.accepted[b] = acc;
      a.L[b] += acc;
      a.head[b] = P[acc - 1];
      if (a.decode) {
        // next block: the predictions from the new head on, then fresh guesses
        const int keep = n - acc + 1;
        const int step = a.iters[b];
        for (int k = 0; k < n; ++k) y[k] = (k < keep) ? P[acc - 1 + k] : draw_guess(a, b, step, k);
      }
    }
  }
  __shared__ int s_act[4], s_com[4];
  int wa = active, wc = committed_now;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    wa += __shfl_xor_sync(0xffffffffu, wa, o);
    wc += __shfl_xor_sync(0xffffffffu, wc, o);
  }
  if ((b & 31) == 0) {
    s_act[b >> 5] = wa;
    s_com[b >> 5] = wc;
  }
  __syncthreads();
  if (b == 0) {
    a.status[0] = s_act[0] + s_act[1] + s_act[2] + s_act[3];
    a.status[1] = s_com[0] + s_com[1] + s_com[2] + s_com[3];
  }
}

__global__ void __launch_bounds__(128) decode_init_kernel(const AcceptArgs a) {
  const int tid = threadIdx.x;
  for (int b = tid; b < a.B; b += blockDim.x) {
    a.L[b] = a.plen[b];
    a.committed[b] = 0;
    a.iters[b] = 0;
    a.done[b] = 0;
    int* y = a.block + b * a.n;
    y[0] = a.head[b];
    for (int k = 1; k < a.n; ++k) y[k] = draw_guess(a, b, 0, k);
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
