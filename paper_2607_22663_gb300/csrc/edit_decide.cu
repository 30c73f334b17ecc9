// Edit-decide: the T2T update of Eq. 2 fused into one pass over the logits.
//
// One CTA owns one row. Each thread streams 16-byte vectors of the row and keeps
// an online (max, sum of exp(l - max), argmax) triple; triples are merged with
// warp shuffles and then across warps through shared memory. Thread 0 turns the
// row's triple into the confidence c = 1 / sum_v exp(l_v - l_max) and applies
// the threshold-and-replace rule. The logits are read exactly once, so the
// kernel is bound by HBM bandwidth.
#include <cuda_bf16.h>
#include "common.cuh"
#include "row_stats.cuh"

namespace mbe {

MBE_DEFINE_ERROR_WORD(edit_decide_take_error)

namespace {

using namespace rows;

// Online (max, sum, argmax) state of a row. Empty: m = -inf, s = 0, idx = -1.
// A NaN or +inf logit makes s NaN, which every later step keeps (s is only
// scaled and added to), so the row's final s tells that it has no softmax.
struct Triple {
  float m;  // running maximum
  float s;  // sum of exp(l - m)
  int idx;  // lowest index attaining m; -1 while no element above -inf was seen
};

// Makes lm (index li) the running maximum if it is larger (an empty state has
// m = -inf: its s, 0 or NaN, is scaled by ex2(-inf) = 0 and stays 0 or NaN).
__device__ __forceinline__ void raise_max(Triple& t, float lm, int li) {
  if (lm > t.m) {
    t.s *= ex2((t.m - lm) * kLog2e);
    t.m = lm;
    t.idx = li;
  }
}

// Exponent reference: 0 while empty, so that -inf logits give ex2(-inf) = 0.
__device__ __forceinline__ float ref_max(const Triple& t) { return t.idx < 0 ? 0.f : t.m; }

// An empty side contributes its s (0, or NaN) and nothing else.
__device__ __forceinline__ void merge(Triple& a, const Triple& b) {
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
    a.s = a.s * ex2((a.m - b.m) * kLog2e) + b.s;
    a.m = b.m;
    a.idx = b.idx;
  } else if (b.m < a.m) {
    a.s += b.s * ex2((b.m - a.m) * kLog2e);
  } else {
    a.s += b.s;
    a.idx = min(a.idx, b.idx);
  }
}

__device__ __forceinline__ Triple shfl_xor(const Triple& t, int mask) {
  Triple o;
  o.m = __shfl_xor_sync(0xffffffffu, t.m, mask);
  o.s = __shfl_xor_sync(0xffffffffu, t.s, mask);
  o.idx = __shfl_xor_sync(0xffffffffu, t.idx, mask);
  return o;
}

template <typename T>
__device__ __forceinline__ void absorb_vector(Triple& t, const uint4& v, int col0) {
  constexpr int N = Vec<T>::N;
  float x[N];
  Vec<T>::unpack(v, x);
  const float lm = vec_max(x);  // NaN if some element is NaN
  if (unusable(lm)) {
    t.s = nan_f32();
    return;
  }
  if (lm > t.m) raise_max(t, lm, col0 + first_index(x, lm));
  const float mr = ref_max(t);
  float acc = 0.f;
#pragma unroll
  for (int k = 0; k < N; ++k) acc += ex2((x[k] - mr) * kLog2e);
  t.s += acc;
}

template <typename T, int kThreads>
__global__ void __launch_bounds__(kThreads) edit_decide_kernel(const T* __restrict__ logits, int64_t row_stride,
                                                               int vocab, bool vec_ok,
                                                               const int32_t* __restrict__ committed,
                                                               const float* __restrict__ tau_per_row, float tau,
                                                               const uint8_t* __restrict__ editable,
                                                               int32_t* new_tokens, uint8_t* __restrict__ edit_mask,
                                                               float* __restrict__ confidence,
                                                               int32_t* __restrict__ argmax_out) {
  constexpr int N = Vec<T>::N;
  constexpr int kUnroll = 4;
  const int row = blockIdx.x;
  const T* rp = logits + static_cast<int64_t>(row) * row_stride;
  Triple t{__int_as_float(0xff800000u), 0.f, -1};  // empty: m = -inf
  int scalar_from = 0;
  if (vec_ok) {
    const uint4* vp = reinterpret_cast<const uint4*>(rp);
    const int nvec = vocab / N;
    int v = threadIdx.x;
    for (; v + (kUnroll - 1) * kThreads < nvec; v += kUnroll * kThreads) {
      uint4 buf[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) buf[u] = __ldcs(vp + v + u * kThreads);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) absorb_vector<T>(t, buf[u], (v + u * kThreads) * N);
    }
    for (; v < nvec; v += kThreads) absorb_vector<T>(t, __ldcs(vp + v), v * N);
    scalar_from = nvec * N;
  }
  for (int c = scalar_from + threadIdx.x; c < vocab; c += kThreads) {
    const float x = to_f32<T>(rp[c]);
    if (unusable(x)) {
      t.s = nan_f32();
    } else {
      raise_max(t, x, c);
      t.s += ex2((x - ref_max(t)) * kLog2e);
    }
  }
  // warp merge
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    Triple o = shfl_xor(t, off);
    merge(t, o);
  }
  __shared__ Triple warp_part[kThreads / 32];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (lane == 0) warp_part[warp] = t;
  __syncthreads();
  if (warp == 0) {
    Triple a = lane < kThreads / 32 ? warp_part[lane] : Triple{__int_as_float(0xff800000u), 0.f, -1};
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      Triple o = shfl_xor(a, off);
      merge(a, o);
    }
    if (lane == 0) {
      const int32_t x = committed[row];
      if (a.idx < 0 || !(a.s > 0.f)) {
        // no softmax (a NaN or +inf logit, or every logit -inf): no decision
        atomicOr(&g_error_word, MBE_DEVERR_NONFINITE);
        new_tokens[row] = x;
        edit_mask[row] = 0;
        confidence[row] = nan_f32();
        if (argmax_out) argmax_out[row] = -1;
        return;
      }
      const float c = 1.0f / a.s;
      const float tr = tau_per_row ? tau_per_row[row] : tau;
      const bool can = editable ? (editable[row] != 0) : true;
      const bool ed = can && (a.idx != x) && (c > tr);
      new_tokens[row] = ed ? a.idx : x;
      edit_mask[row] = ed ? 1 : 0;
      confidence[row] = c;
      if (argmax_out) argmax_out[row] = a.idx;
    }
  }
}

template <typename T>
mbe_status launch(const void* logits, int64_t row_stride, int32_t rows, int32_t vocab, const int32_t* committed,
                  const float* tpr, float tau, const uint8_t* editable, int32_t* new_tokens, uint8_t* edit_mask,
                  float* confidence, int32_t* argmax_out, cudaStream_t stream) {
  const T* lp = static_cast<const T*>(logits);
  const bool vec_ok = aligned16(logits) && ((row_stride * static_cast<int64_t>(sizeof(T))) % 16 == 0);
  // rows of 256 KB and more: 512 threads (32 vectors each); 8-256 KB: 256 threads,
  // so that shorter rows still stream at least a few vectors per thread and eight
  // CTAs per SM overlap one another's final reductions
  const int64_t row_bytes = static_cast<int64_t>(vocab) * sizeof(T);
  if (row_bytes >= 256 * 1024) {
    edit_decide_kernel<T, 512><<<rows, 512, 0, stream>>>(lp, row_stride, vocab, vec_ok, committed, tpr, tau, editable,
                                                         new_tokens, edit_mask, confidence, argmax_out);
  } else if (row_bytes >= 8 * 1024) {
    edit_decide_kernel<T, 256><<<rows, 256, 0, stream>>>(lp, row_stride, vocab, vec_ok, committed, tpr, tau, editable,
                                                         new_tokens, edit_mask, confidence, argmax_out);
  } else {
    edit_decide_kernel<T, 64><<<rows, 64, 0, stream>>>(lp, row_stride, vocab, vec_ok, committed, tpr, tau, editable,
                                                       new_tokens, edit_mask, confidence, argmax_out);
  }
  return launch_status();
}

}  // namespace
}  // namespace mbe

extern "C" mbe_status mbe_edit_decide(const void* logits, mbe_dtype dtype, int64_t row_stride, int32_t rows,
                                      int32_t vocab, const int32_t* committed, const float* tau_per_row_or_null,
                                      float tau, const uint8_t* editable_or_null, int32_t* new_tokens,
                                      uint8_t* edit_mask, float* confidence, int32_t* argmax_or_null,
                                      cudaStream_t stream) {
  if (rows < 0 || vocab < 1 || row_stride < vocab) return MBE_ERR_INVALID_ARG;
  if (dtype != MBE_F32 && dtype != MBE_BF16) return MBE_ERR_INVALID_ARG;
  if (rows == 0) return MBE_OK;
  if (!logits || !committed || !new_tokens || !edit_mask || !confidence) return MBE_ERR_INVALID_ARG;
  if (dtype == MBE_F32)
    return mbe::launch<float>(logits, row_stride, rows, vocab, committed, tau_per_row_or_null, tau, editable_or_null,
                              new_tokens, edit_mask, confidence, argmax_or_null, stream);
  return mbe::launch<__nv_bfloat16>(logits, row_stride, rows, vocab, committed, tau_per_row_or_null, tau,
                                    editable_or_null, new_tokens, edit_mask, confidence, argmax_or_null, stream);
}
