// Helpers shared by the row-reducing kernels (edit-decide, the full denoising
// update and the fused LM head): exp2, bf16/fp32 loads, 16-byte vector
// unpacking, and the online (max, sum, entropy sum, argmax) state.
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

// Online state of a softmax row: the running maximum m with its lowest index,
// s = sum of e = 2^u and t = sum of e*u over the elements seen, u = (l - m) log2(e).
// ln(s) - ln2 * t / s is the entropy and 1 / s the largest probability.
struct Stats {
  float m;   // running maximum
  float s;   // sum of e = 2^u, u = (l - m) log2(e)
  float t;   // sum of e * u
  int idx;   // lowest index attaining m; -1 while empty
};

__device__ __forceinline__ void rebase(Stats& a, float m_new) {
  // re-expresses (s, t) relative to a larger maximum
  const float d = (a.m - m_new) * kLog2e;  // <= 0
  const float f = ex2(d);
  a.t = f * (a.t + d * a.s);
  a.s *= f;
  a.m = m_new;
}

__device__ __forceinline__ void absorb(Stats& a, float x, int col) {
  if (a.idx < 0) {
    a.m = x;
    a.idx = col;
    a.s = 1.f;
    a.t = 0.f;
    return;
  }
  if (x > a.m) {
    rebase(a, x);
    a.idx = col;
  }
  const float u = (x - a.m) * kLog2e;
  const float e = ex2(u);
  a.s += e;
  a.t = fmaf(e, u, a.t);
}

// Combines two partial states (the lowest index wins on equal maxima).
__device__ __forceinline__ void merge(Stats& a, Stats b) {
  if (b.idx < 0) return;
  if (a.idx < 0) {
    a = b;
    return;
  }
  if (b.m > a.m) {
    rebase(a, b.m);
    a.idx = b.idx;
  } else if (b.m < a.m) {
    rebase(b, a.m);
  } else {
    a.idx = min(a.idx, b.idx);
  }
  a.s += b.s;
  a.t += b.t;
}

__device__ __forceinline__ Stats shfl_xor(const Stats& t, int mask) {
  return Stats{__shfl_xor_sync(0xffffffffu, t.m, mask), __shfl_xor_sync(0xffffffffu, t.s, mask),
               __shfl_xor_sync(0xffffffffu, t.t, mask), __shfl_xor_sync(0xffffffffu, t.idx, mask)};
}

}  // namespace rows
}  // namespace mbe
