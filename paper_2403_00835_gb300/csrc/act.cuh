// Element-type helpers: activations and weights are fp32 (CLLM_F32) or bf16.
#pragma once
#include <cuda_bf16.h>
#include <cuda_fp16.h>
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

__device__ __forceinline__ float ld_act(const __half* p, size_t i) { return __half2float(p[i]); }
__device__ __forceinline__ void st_act(__half* p, size_t i, float v) { p[i] = __float2half_rn(v); }

// GEMM activation inputs.  fp32 engine: one fp32 plane.  bf16 engine: the
// value is carried as two bf16 planes, hi = bf16(v) and lo = bf16(v - hi),
// `plane` elements apart; the weight GEMM multiplies both (exact bf16
// weights times a 16-bit-mantissa activation) into one fp32 accumulator.
__device__ __forceinline__ void st_gin(float* p, size_t i, size_t, float v) { p[i] = v; }
__device__ __forceinline__ void st_gin(__nv_bfloat16* p, size_t i, size_t plane, float v) {
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  p[i] = hi;
  p[i + plane] = __float2bfloat16_rn(v - __bfloat162float(hi));
}
// Four consecutive elements (i a multiple of 4): one vector store per plane.
__device__ __forceinline__ void st_gin4(float* p, size_t i, size_t, float4 v) {
  *reinterpret_cast<float4*>(p + i) = v;
}
__device__ __forceinline__ void st_gin4(__nv_bfloat16* p, size_t i, size_t plane, float4 v) {
  const float x[4] = {v.x, v.y, v.z, v.w};
  __nv_bfloat16 hi[4], lo[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    hi[k] = __float2bfloat16_rn(x[k]);
    lo[k] = __float2bfloat16_rn(x[k] - __bfloat162float(hi[k]));
  }
  uint2 h, l;
  h.x = static_cast<uint32_t>(__bfloat16_as_ushort(hi[0])) | (static_cast<uint32_t>(__bfloat16_as_ushort(hi[1])) << 16);
  h.y = static_cast<uint32_t>(__bfloat16_as_ushort(hi[2])) | (static_cast<uint32_t>(__bfloat16_as_ushort(hi[3])) << 16);
  l.x = static_cast<uint32_t>(__bfloat16_as_ushort(lo[0])) | (static_cast<uint32_t>(__bfloat16_as_ushort(lo[1])) << 16);
  l.y = static_cast<uint32_t>(__bfloat16_as_ushort(lo[2])) | (static_cast<uint32_t>(__bfloat16_as_ushort(lo[3])) << 16);
  *reinterpret_cast<uint2*>(p + i) = h;
  *reinterpret_cast<uint2*>(p + i + plane) = l;
}
__device__ __forceinline__ float ld_gin(const float* p, size_t i, size_t) { return p[i]; }
__device__ __forceinline__ float ld_gin(const __nv_bfloat16* p, size_t i, size_t plane) {
  return __bfloat162float(p[i]) + __bfloat162float(p[i + plane]);
}

// Element type of attention operands (Q, the K/V cache): fp32 in the fp32
// engine; fp16 (10-bit mantissa) in the bf16 engine.
template <typename Act>
struct AttnType {
  using T = Act;
};
template <>
struct AttnType<__nv_bfloat16> {
  using T = __half;
};

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
