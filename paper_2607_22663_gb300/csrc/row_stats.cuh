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

// NaN-propagating maxima: NaN if an input is NaN, else the largest input.
__device__ __forceinline__ float fmax3_nan(float a, float b, float c) {
  float r;
  asm("max.NaN.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

// Maximum of a vector's elements (3-input max instructions); NaN if any
// element is NaN, so that one value tells whether the vector is usable.
__device__ __forceinline__ float vec_max(const float (&x)[8]) {
  return fmax3_nan(fmax3_nan(x[0], x[1], x[2]), fmax3_nan(x[3], x[4], x[5]), fmax_nan(x[6], x[7]));
}
__device__ __forceinline__ float vec_max(const float (&x)[4]) {
  return fmax3_nan(x[0], x[1], fmax_nan(x[2], x[3]));
}

// A row has a softmax only if none of its logits is NaN or +inf and one is
// finite; -inf logits are tokens of probability 0. A value that is NaN or +inf
// (a vector maximum, say) makes the row unusable.
__device__ __forceinline__ bool unusable(float x) { return !(x < __int_as_float(0x7f800000)); }
__device__ __forceinline__ float nan_f32() { return __int_as_float(0x7fc00000); }

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
// Empty state: m = -inf, s = t = 0, idx = -1. A row without a softmax (see
// unusable) sets s to NaN, which every later step keeps (absorb, rebase and
// merge only add to or scale s), so the final s tells the row apart.
struct Stats {
  float m;   // running maximum
  float s;   // sum of e = 2^u, u = (l - m) log2(e)
  float t;   // sum of e * u
  int idx;   // lowest index attaining m; -1 while no element above -inf was seen
};

// u is clamped here so that a -inf logit adds e * u = 0 * kMinU = 0 to t
// (2^kMinU is 0 in fp32).
constexpr float kMinU = -1.0e4f;

// Reference maximum for the exponentials: 0 while the state is empty, so that
// -inf logits give 2^-inf = 0 rather than 2^NaN.
__device__ __forceinline__ float ref_max(const Stats& a) { return a.idx < 0 ? 0.f : a.m; }

__device__ __forceinline__ void rebase(Stats& a, float m_new) {
  // re-expresses (s, t) relative to a larger maximum (a is not empty)
  const float d = (a.m - m_new) * kLog2e;  // <= 0
  const float f = ex2(d);
  a.t = f * (a.t + d * a.s);
  a.s *= f;
  a.m = m_new;
}

// Makes lm (with index li) the running maximum if it is larger; an empty state
// keeps its s and t (0, or NaN).
__device__ __forceinline__ void raise_max(Stats& a, float lm, int li) {
  if (lm > a.m) {
    if (a.idx < 0)
      a.m = lm;
    else
      rebase(a, lm);
    a.idx = li;
  }
}

__device__ __forceinline__ void absorb(Stats& a, float x, int col) {
  if (unusable(x)) {
    a.s = nan_f32();
    return;
  }
  raise_max(a, x, col);
  const float u = fmaxf((x - ref_max(a)) * kLog2e, kMinU);
  const float e = ex2(u);
  a.s += e;
  a.t = fmaf(e, u, a.t);
}

// Combines two partial states (the lowest index wins on equal maxima). An
// empty side contributes its s (0, or NaN) and nothing else.
__device__ __forceinline__ void merge(Stats& a, Stats b) {
  if (b.idx < 0) {
    a.s += b.s;
    return;
  }
  if (a.idx < 0) {
    const float z = a.s;
    a = b;
    a.s += z;
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

// True if the reduced state of a whole row gives no decision: a NaN or +inf
// logit (s is NaN) or every logit -inf (no maximum).
__device__ __forceinline__ bool undecidable(const Stats& a) { return a.idx < 0 || !(a.s > 0.f); }

__device__ __forceinline__ Stats shfl_xor(const Stats& t, int mask) {
  return Stats{__shfl_xor_sync(0xffffffffu, t.m, mask), __shfl_xor_sync(0xffffffffu, t.s, mask),
               __shfl_xor_sync(0xffffffffu, t.t, mask), __shfl_xor_sync(0xffffffffu, t.idx, mask)};
}

}  // namespace rows
}  // namespace mbe
