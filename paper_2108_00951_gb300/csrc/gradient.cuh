// gradient.cuh — loading four consecutive gradient values (fp32, or bf16 bit
// patterns widened exactly: the 16 stored bits become the high half of the
// fp32 word).
#pragma once

#include "common.cuh"

namespace efs {

template <typename GT>
struct GradVec;

template <>
struct GradVec<float> {
  float4 v;
  __device__ __forceinline__ void load(const float* p) { v = ld_stream_f4(p); }
  __device__ __forceinline__ float operator[](int j) const {
    return j == 0 ? v.x : j == 1 ? v.y : j == 2 ? v.z : v.w;
  }
};

template <>
struct GradVec<uint16_t> {
  uint2 v;
  __device__ __forceinline__ void load(const uint16_t* p) { v = ld_stream_u2(p); }
  __device__ __forceinline__ float operator[](int j) const {
    const uint32_t w = (j < 2) ? v.x : v.y;
    return bf16_bits_to_f32((j & 1) ? (w >> 16) : (w & 0xffffu));
  }
};

__device__ __forceinline__ float grad_scalar(const float* g, uint64_t i) { return g[i]; }
__device__ __forceinline__ float grad_scalar(const uint16_t* g, uint64_t i) {
  return bf16_bits_to_f32(g[i]);
}

}  // namespace efs
