// Helpers shared by the row-streaming kernels (edit-decide and the full
// denoising update): exp2, bf16/fp32 loads and 16-byte vector unpacking.
#pragma once
#include <cstdint>
#include <cuda_bf16.h>
#include "ptx_sm103.cuh"

namespace mbe {
namespace rows {

constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <typename T>
__device__ __forceinline__ float to_f32(T x);
template <>
__device__ __forceinline__ float to_f32<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

// Unpacks one 16-byte vector into floats.
template <typename T>
struct Vec;
template <>
struct Vec<float> {
  static constexpr int N = 4;
  __device__ __forceinline__ static void unpack(const uint4& v, float (&x)[4]) {
    x[0] = __uint_as_float(v.x); x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z); x[3] = __uint_as_float(v.w);
  }
};
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;
  __device__ __forceinline__ static void unpack(const uint4& v, float (&x)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      x[2 * k] = __uint_as_float(w[k] << 16);
      x[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
    }
  }
};

// Maximum of a vector's elements (3-input max instructions).
__device__ __forceinline__ float vec_max(const float (&x)[8]) {
  return fmax3(fmax3(x[0], x[1], x[2]), fmax3(x[3], x[4], x[5]), fmaxf(x[6], x[7]));
}
__device__ __forceinline__ float vec_max(const float (&x)[4]) { return fmax3(x[0], x[1], fmaxf(x[2], x[3])); }

// Lowest k with x[k] == v (v is one of the elements).
template <int N>
__device__ __forceinline__ int first_index(const float (&x)[N], float v) {
  int i = N - 1;
#pragma unroll
  for (int k = N - 2; k >= 0; --k)
    if (x[k] == v) i = k;
  return i;
}

}  // namespace rows
}  // namespace mbe
