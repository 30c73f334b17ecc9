// Full threshold update of a decoding step and tail-entropy block selection.
//
//  denoise_row_kernel    one CTA per row: a single HBM pass over the logits with
//                        an online (max, sum e, sum e*u, argmax) state, where
//                        e = 2^u and u = (l - max) * log2(e); it yields the
//                        confidence c = 1/sum e, the entropy
//                        H = ln(sum e) - ln2 * (sum e*u) / (sum e), and the
//                        row-local part of Eq. 2 (Gamma_t by omega_mask for
//                        masked rows, Delta_t by omega_edit for visible rows).
//  denoise_block_kernel  one CTA per sequence, one warp per block: the forced
//                        unmasking of Sec. 2.3 (a block whose masked rows all
//                        stay below omega_mask unmasks its most confident one),
//                        changed-block flags and per-sequence change counts.
//  tail_entropy_kernel   one CTA per sequence: Eq. 6 scores of the candidate
//                        blocks (mean of the ceil(rho B) largest entropies,
//                        rank-based selection) and the Eq. 7 argmax.
#include <cuda_bf16.h>
#include <cmath>
#include "common.cuh"
#include "row_stats.cuh"

namespace mbe {

MBE_DEFINE_ERROR_WORD(denoise_take_error)

namespace {

using namespace rows;

template <typename T>
__device__ __forceinline__ void absorb_vector(Stats& a, const uint4& v, int col0) {
  constexpr int N = Vec<T>::N;
  float x[N];
  Vec<T>::unpack(v, x);
  const float lm = vec_max(x);  // NaN if some element is NaN
  if (unusable(lm)) {
    a.s = nan_f32();
    return;
  }
  if (lm > a.m) raise_max(a, lm, col0 + first_index(x, lm));  // rare after the first vectors
  // u = l log2e - m log2e (clamped below, so that -inf logits add 0 to t) and
  // e = 2^u, two elements per packed FMA / add
  const float mr = ref_max(a);
  const float2 L = make_float2(kLog2e, kLog2e);
  const float2 ms = make_float2(-mr * kLog2e, -mr * kLog2e);
  float2 s = make_float2(0.f, 0.f), t = make_float2(0.f, 0.f);
#pragma unroll
  for (int k = 0; k < N; k += 2) {
    float2 u = ffma2(make_float2(x[k], x[k + 1]), L, ms);
    u.x = fmaxf(u.x, kMinU);
    u.y = fmaxf(u.y, kMinU);
    const float2 e = make_float2(ex2(u.x), ex2(u.y));
    s = fadd2(s, e);
    t = ffma2(e, u, t);
  }
  a.s += s.x + s.y;
  a.t += t.x + t.y;
}

struct RowArgs {
  int64_t row_stride;
  int vocab;
  bool vec_ok;
  const int32_t* tokens;
  int32_t mask_id;
  float omega_mask, omega_edit;
  const uint8_t* editable;
  int32_t* new_tokens;
  uint8_t* kind;
  float* confidence;
  int32_t* argmax;
  float* entropy;
};

template <typename T, int kThreads>
__global__ void __launch_bounds__(kThreads) denoise_row_kernel(const T* __restrict__ logits, const RowArgs a) {
  constexpr int N = Vec<T>::N;
  constexpr int kUnroll = 4;
  const int row = blockIdx.x;
  const T* rp = logits + static_cast<int64_t>(row) * a.row_stride;
  Stats st{__int_as_float(0xff800000u), 0.f, 0.f, -1};  // empty: m = -inf
  int scalar_from = 0;
  if (a.vec_ok) {
    const uint4* vp = reinterpret_cast<const uint4*>(rp);
    const int nvec = a.vocab / N;
    int v = threadIdx.x;
    for (; v + (kUnroll - 1) * kThreads < nvec; v += kUnroll * kThreads) {
      uint4 buf[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) buf[u] = __ldcs(vp + v + u * kThreads);
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) absorb_vector<T>(st, buf[u], (v + u * kThreads) * N);
    }
    for (; v < nvec; v += kThreads) absorb_vector<T>(st, __ldcs(vp + v), v * N);
    scalar_from = nvec * N;
  }
  for (int c = scalar_from + threadIdx.x; c < a.vocab; c += kThreads) absorb(st, to_f32<T>(rp[c]), c);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) merge(st, shfl_xor(st, off));
  __shared__ Stats part[kThreads / 32];
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (lane == 0) part[warp] = st;
  __syncthreads();
  if (warp != 0) return;
  Stats b = lane < kThreads / 32 ? part[lane] : Stats{0.f, 0.f, 0.f, -1};
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) merge(b, shfl_xor(b, off));
  if (lane != 0) return;
  const int32_t cur = a.tokens[row];
  if (undecidable(b)) {
    // no softmax (a NaN or +inf logit, or every logit -inf): the token stays,
    // and the row is never the forced one of its block (argmax -1)
    atomicOr(&g_error_word, MBE_DEVERR_NONFINITE);
    a.new_tokens[row] = cur;
    a.kind[row] = 0;
    a.confidence[row] = nan_f32();
    a.argmax[row] = -1;
    if (a.entropy) a.entropy[row] = nan_f32();
    return;
  }
  const float c = 1.0f / b.s;
  uint8_t k = 0;
  if (cur == a.mask_id) {
    if (c > a.omega_mask) k = 1;
  } else if ((a.editable == nullptr || a.editable[row] != 0) && b.idx != cur && c > a.omega_edit) {
    k = 3;
  }
  a.new_tokens[row] = k ? b.idx : cur;
  a.kind[row] = k;
  a.confidence[row] = c;
  a.argmax[row] = b.idx;
  if (a.entropy) a.entropy[row] = logf(b.s) - 0.6931471805599453f * b.t / b.s;
}

// One CTA per sequence; warp w handles blocks w, w + nwarps, ...
__global__ void __launch_bounds__(256) denoise_block_kernel(const int32_t* __restrict__ cu_rows, int total_rows,
                                                            int block_size, int max_blocks,
                                                            const int32_t* __restrict__ tokens, int32_t mask_id,
                                                            const float* __restrict__ confidence,
                                                            const int32_t* __restrict__ argmax, int32_t* new_tokens,
                                                            uint8_t* kind, uint8_t* block_changed,
                                                            int32_t* seq_changes) {
  const int s = blockIdx.x;
  const int r0 = cu_rows[s], r1 = cu_rows[s + 1];
  __shared__ int s_changes;
  if (threadIdx.x == 0) s_changes = 0;
  __syncthreads();
  const bool ok = r0 >= 0 && r1 >= r0 && r1 <= total_rows;
  if (!ok && threadIdx.x == 0) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
  const int nblocks = ok ? (r1 - r0 + block_size - 1) / block_size : 0;
  if (block_changed && nblocks > max_blocks && threadIdx.x == 0) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32, nwarps = blockDim.x / 32;
  for (int b = warp; b < nblocks; b += nwarps) {
    const int b0 = r0 + b * block_size, b1 = min(b0 + block_size, r1);
    bool any_masked = false, any_unmasked = false;
    float best_c = -1.f;
    int best_r = 0x7FFFFFFF;
    for (int r = b0 + lane; r < b1; r += 32) {
      if (tokens[r] != mask_id) continue;
      any_masked = true;
      if (kind[r] == 1) any_unmasked = true;
      if (argmax[r] < 0) continue;  // a row without a softmax is never forced
      const float c = confidence[r];
      if (c > best_c || (c == best_c && r < best_r)) {
        best_c = c;
        best_r = r;
      }
    }
    any_masked = __any_sync(0xffffffffu, any_masked);
    any_unmasked = __any_sync(0xffffffffu, any_unmasked);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float oc = __shfl_xor_sync(0xffffffffu, best_c, off);
      const int orr = __shfl_xor_sync(0xffffffffu, best_r, off);
      if (oc > best_c || (oc == best_c && orr < best_r)) {
        best_c = oc;
        best_r = orr;
      }
    }
    // best_r stays 0x7FFFFFFF when no masked row of the block has a softmax
    if (any_masked && !any_unmasked && best_r != 0x7FFFFFFF && lane == 0) {
      kind[best_r] = 2;
      new_tokens[best_r] = argmax[best_r];
    }
    __syncwarp();
    int changes = 0;
    for (int r = b0 + lane; r < b1; r += 32) changes += new_tokens[r] != tokens[r];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) changes += __shfl_xor_sync(0xffffffffu, changes, off);
    if (lane == 0) {
      if (block_changed && b < max_blocks) block_changed[static_cast<int64_t>(s) * max_blocks + b] = changes > 0;
      atomicAdd(&s_changes, changes);
    }
  }
  if (block_changed)
    for (int b = nblocks + threadIdx.x; b < max_blocks; b += blockDim.x)
      block_changed[static_cast<int64_t>(s) * max_blocks + b] = 0;
  __syncthreads();
  if (threadIdx.x == 0 && seq_changes) seq_changes[s] = s_changes;
}

// One CTA per sequence. Candidate slots are the last min(n_valid, k_max - 1)
// of n_hist; element i of a block is in its top-k iff fewer than k elements
// are larger (or equal with a lower index).
__global__ void __launch_bounds__(256) tail_entropy_kernel(const float* __restrict__ block_entropy,
                                                           const int32_t* __restrict__ n_valid, int n_hist,
                                                           int block_size, int top, int k_max, float* scores,
                                                           int32_t* best_slot, int32_t* window_blocks) {
  const int s = blockIdx.x;
  extern __shared__ float sh[];  // block_size floats
  __shared__ float s_sum;
  int nv = min(n_valid[s], n_hist);
  nv = max(nv, 0);
  const int ncand = min(nv, k_max - 1);
  int best = -1;
  float best_score = 0.f;
  for (int slot = 0; slot < n_hist; ++slot) {
    const bool cand = slot >= n_hist - ncand;
    if (!cand) {
      if (scores && threadIdx.x == 0) scores[static_cast<int64_t>(s) * n_hist + slot] = __int_as_float(0x7fc00000);
      continue;
    }
    const float* e = block_entropy + (static_cast<int64_t>(s) * n_hist + slot) * block_size;
    for (int i = threadIdx.x; i < block_size; i += blockDim.x) sh[i] = e[i];
    if (threadIdx.x == 0) s_sum = 0.f;
    __syncthreads();
    float part = 0.f;
    for (int i = threadIdx.x; i < block_size; i += blockDim.x) {
      const float xi = sh[i];
      int rank = 0;
      for (int j = 0; j < block_size; ++j) {
        const float xj = sh[j];
        rank += (xj > xi) || (xj == xi && j < i);
      }
      if (rank < top) part += xi;
    }
    atomicAdd(&s_sum, part);
    __syncthreads();
    const float sc = s_sum / top;
    if (best < 0 || sc > best_score) {
      best = slot;
      best_score = sc;
    }
    if (scores && threadIdx.x == 0) scores[static_cast<int64_t>(s) * n_hist + slot] = sc;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    best_slot[s] = best;
    window_blocks[s] = best < 0 ? 1 : n_hist - best + 1;
  }
}

template <typename T>
mbe_status launch_rows(const void* logits, int32_t rows, const RowArgs& a, cudaStream_t stream) {
  const T* lp = static_cast<const T*>(logits);
  // as in edit-decide: 512 threads from 256 KB rows, 256 threads for 8-256 KB rows
  const int64_t row_bytes = static_cast<int64_t>(a.vocab) * sizeof(T);
  if (row_bytes >= 256 * 1024)
    denoise_row_kernel<T, 512><<<rows, 512, 0, stream>>>(lp, a);
  else if (row_bytes >= 8 * 1024)
    denoise_row_kernel<T, 256><<<rows, 256, 0, stream>>>(lp, a);
  else
    denoise_row_kernel<T, 64><<<rows, 64, 0, stream>>>(lp, a);
  return launch_status("denoise_row_kernel launch");
}

}  // namespace
}  // namespace mbe

extern "C" mbe_status mbe_denoise_update(const void* logits, mbe_dtype dtype, int64_t row_stride, int32_t vocab,
                                         const int32_t* cu_rows, int32_t num_seqs, int32_t total_rows,
                                         int32_t block_size, int32_t max_blocks_per_seq, const int32_t* tokens,
                                         int32_t mask_id, float omega_mask, float omega_edit,
                                         const uint8_t* editable_or_null, int32_t* new_tokens, uint8_t* update_kind,
                                         float* confidence, int32_t* argmax, float* entropy_or_null,
                                         uint8_t* block_changed_or_null, int32_t* seq_changes_or_null,
                                         cudaStream_t stream) {
  using namespace mbe;
  if (num_seqs < 0 || total_rows < 0 || vocab < 1 || row_stride < vocab || block_size < 1) return MBE_ERR_INVALID_ARG;
  if (dtype != MBE_F32 && dtype != MBE_BF16) return MBE_ERR_INVALID_ARG;
  if (block_changed_or_null && max_blocks_per_seq < 1) return MBE_ERR_INVALID_ARG;
  if (num_seqs == 0 || total_rows == 0) return MBE_OK;
  if (!logits || !cu_rows || !tokens || !new_tokens || !update_kind || !confidence || !argmax)
    return MBE_ERR_INVALID_ARG;
  if (new_tokens == tokens) return MBE_ERR_INVALID_ARG;  // the block pass compares old and new tokens
  if (num_seqs > 0x7FFFFFFF / 2) return MBE_ERR_UNSUPPORTED;
  RowArgs a;
  a.row_stride = row_stride;
  a.vocab = vocab;
  a.vec_ok = aligned16(logits) &&
             ((row_stride * static_cast<int64_t>(dtype == MBE_F32 ? 4 : 2)) % 16 == 0);
  a.tokens = tokens;
  a.mask_id = mask_id;
  a.omega_mask = omega_mask;
  a.omega_edit = omega_edit;
  a.editable = editable_or_null;
  a.new_tokens = new_tokens;
  a.kind = update_kind;
  a.confidence = confidence;
  a.argmax = argmax;
  a.entropy = entropy_or_null;
  const mbe_status st = dtype == MBE_F32 ? launch_rows<float>(logits, total_rows, a, stream)
                                         : launch_rows<__nv_bfloat16>(logits, total_rows, a, stream);
  if (st != MBE_OK) return st;
  denoise_block_kernel<<<num_seqs, 256, 0, stream>>>(cu_rows, total_rows, block_size, max_blocks_per_seq, tokens,
                                                     mask_id, confidence, argmax, new_tokens, update_kind,
                                                     block_changed_or_null, seq_changes_or_null);
  return launch_status("denoise_block_kernel launch");
}

extern "C" mbe_status mbe_tail_entropy_select(const float* block_entropy, const int32_t* n_valid, int32_t num_seqs,
                                              int32_t n_hist, int32_t block_size, float rho, int32_t k_max,
                                              float* scores_or_null, int32_t* best_slot, int32_t* window_blocks,
                                              cudaStream_t stream) {
  using namespace mbe;
  if (num_seqs < 0 || n_hist < 1 || block_size < 1 || k_max < 1 || !(rho > 0.f) || rho > 1.f)
    return MBE_ERR_INVALID_ARG;
  if (block_size > 12 * 1024) return MBE_ERR_UNSUPPORTED;  // one block's entropies live in shared memory
  if (num_seqs == 0) return MBE_OK;
  if (!block_entropy || !n_valid || !best_slot || !window_blocks) return MBE_ERR_INVALID_ARG;
  const int top = static_cast<int>(std::ceil(static_cast<double>(rho) * block_size));
  tail_entropy_kernel<<<num_seqs, 256, block_size * sizeof(float), stream>>>(
      block_entropy, n_valid, n_hist, block_size, top, k_max, scores_or_null, best_slot, window_blocks);
  return launch_status("tail_entropy_kernel launch");
}
