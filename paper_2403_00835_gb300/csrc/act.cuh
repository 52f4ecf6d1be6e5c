// Element-type helpers: activations and weights are fp32 (CLLM_F32) or bf16.
#pragma once
#include <cuda_bf16.h>
#include <stdint.h>

namespace cllm {

__device__ __forceinline__ float ld_act(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ld_act(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void st_act(float* p, size_t i, float v) { p[i] = v; }
__device__ __forceinline__ void st_act(__nv_bfloat16* p, size_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

}  // namespace cllm
