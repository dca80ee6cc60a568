// Element conversions shared by the SpMM kernels. bf16 travels as its 16-bit
// pattern (uint16_t): widening is exact, narrowing rounds to nearest even.
#pragma once

#include <cuda_bf16.h>
#include <cstdint>

namespace bsr {

__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }

template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ uint16_t from_f32<uint16_t>(float v) {
    return __bfloat16_as_ushort(__float2bfloat16_rn(v));
}

}  // namespace bsr
