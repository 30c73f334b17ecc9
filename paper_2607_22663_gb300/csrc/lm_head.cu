// LM-head projection fused with the edit decision of Eq. 2.
//
// logits[r, v] = sum_k hidden[r, k] * weight[v, k] are computed on the
// tensor cores (tcgen05, bf16 operands, fp32 accumulators in TMEM) and folded,
// tile by tile, into an online per-row state (max, sum of exp, entropy sum,
// argmax); the [rows, vocab] logits never reach HBM.
//
// lm_head_kernel (persistent, one CTA per SM, 256 threads):
//   warp 0      TMA producer: 128x64 hidden and 256x64 weight tiles into a
//               4-stage shared-memory ring (128-byte swizzle).
//   warp 1      MMA issuer: D[128x256] += A * B^T, 4 MMAs of K = 16 per
//               stage, into one of two 256-column TMEM accumulators.
//   warps 4-7   epilogue: thread = accumulator row = TMEM lane; reads its
//               row 32 columns at a time and updates the row state, so the
//               epilogue of one tile overlaps the MMAs of the next.
// A work unit is (128-row block, vocabulary chunk of 1..8 tiles of 256
// columns, chosen so every SM gets at least ~16 units); units go chunk-major so
// the CTAs running at the same time share a weight chunk in L2.
// Each unit writes one partial state per row. lm_head_decide_kernel merges a
// row's partial states and applies the threshold-and-replace rule.
#include <cuda_bf16.h>
#include <algorithm>
#include <mutex>
#include "common.cuh"
#include "ptx_sm103.cuh"
#include "row_stats.cuh"
#include "tma_host.cuh"

namespace mbe {

MBE_DEFINE_ERROR_WORD(lm_head_take_error)

namespace lmh {

using namespace rows;

constexpr int kBM = 128, kBN = 256, kBK = 64;
constexpr int kStages = 4;
constexpr int kMaxTilesPerUnit = 8;  // up to 2048 vocabulary columns per work unit
constexpr int kUnitsPerSm = 16;      // fewer tiles per unit until every SM gets this many units
constexpr int kThreads = 256;
constexpr uint32_t kABytes = kBM * kBK * 2;  // 16 KB
constexpr uint32_t kBBytes = kBN * kBK * 2;  // 32 KB
constexpr uint32_t kStageBytes = kABytes + kBBytes;
constexpr uint32_t kSmemBytes = kStages * kStageBytes + 1024;  // + 1024-byte alignment slack
constexpr uint32_t kTmemCols = 2 * kBN;
constexpr float kMaskedLogit = -1.0e30f;  // columns past the vocabulary (finite: e * u stays 0)

struct Partial {
  float m, s, t;
  int idx;
};

struct Params {
  int rows, vocab, d;
  int tpu;  // tiles per unit
  int n_m, n_chunks, n_units, n_kb;
  Partial* part;  // [rows, n_chunks]
  uint64_t wait_ns;  // limit of the ordinary mbarrier waits
};

struct Bars {
  uint64_t full[kStages], empty[kStages], acc_full[2], acc_empty[2], mma_done;
};

// Folds 32 consecutive logits (columns col0..col0+31) into the row state.
__device__ __forceinline__ void absorb32(Stats& a, const float (&x)[32], int col0) {
  float cm = fmax3(x[0], x[1], x[2]);
#pragma unroll
  for (int k = 3; k < 31; k += 2) cm = fmax3(cm, x[k], x[k + 1]);
  cm = fmaxf(cm, x[31]);
  // a NaN logit is skipped by the maximum but gives e = NaN below, and a +inf
  // one becomes the maximum with u = NaN for itself: s turns NaN either way
  if (cm > a.m) raise_max(a, cm, col0 + first_index(x, cm));
  const float mr = ref_max(a);
  const float2 L = make_float2(kLog2e, kLog2e);
  const float2 ms = make_float2(-mr * kLog2e, -mr * kLog2e);
  float2 s = make_float2(0.f, 0.f), t = make_float2(0.f, 0.f);
#pragma unroll
  for (int k = 0; k < 32; k += 2) {
    const float2 u = ffma2(make_float2(x[k], x[k + 1]), L, ms);
    const float2 e = make_float2(ex2(u.x), ex2(u.y));
    s = fadd2(s, e);
    t = ffma2(e, u, t);
  }
  a.s += s.x + s.y;
  a.t += t.x + t.y;
}

__global__ void __launch_bounds__(kThreads, 1)
    lm_head_kernel(const __grid_constant__ CUtensorMap tm_h, const __grid_constant__ CUtensorMap tm_w,
                   const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) Bars bars;
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  volatile int* abort_flag = &abort_s;
  const uint64_t wait_ns = p.wait_ns;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  auto bar = [](uint64_t& b) { return smem_u32(&b); };

  if (tid == 0) {
    abort_s = 0;
    for (int i = 0; i < kStages; ++i) {
      mbar_init(bar(bars.full[i]), 1);
      mbar_init(bar(bars.empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(bars.acc_full[i]), 1);
      mbar_init(bar(bars.acc_empty[i]), 4);  // one arrive per epilogue warp
    }
    mbar_init(bar(bars.mma_done), 1);
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), kTmemCols);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  // tiles of a chunk: columns [chunk * tpu * 256, ...) up to the vocabulary end
  auto tiles_of = [&](int chunk) { return min(p.tpu, (p.vocab + kBN - 1) / kBN - chunk * p.tpu); };

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tm_h);
      tma_prefetch_desc(&tm_w);
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
        const int chunk = u / p.n_m, mt = u - chunk * p.n_m;
        const int nt_count = tiles_of(chunk);
        for (int t = 0; t < nt_count && ok; ++t) {
          const int nt = chunk * p.tpu + t;
          for (int kb = 0; kb < p.n_kb; ++kb, ++it) {
            const uint32_t s = it % kStages;
            if (it >= kStages && !mbar_wait(bar(bars.empty[s]), ((it / kStages) - 1) & 1, abort_flag, wait_ns)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(bar(bars.full[s]), kStageBytes);
            const uint32_t dst = sbase + s * kStageBytes;
            tma_load_2d(dst, &tm_h, bar(bars.full[s]), kb * kBK, mt * kBM);
            tma_load_2d(dst + kABytes, &tm_w, bar(bars.full[s]), kb * kBK, nt * kBN);
          }
        }
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
      }
      // The copies already issued land before the CTA can exit, also when another
      // role aborted after this loop ended (they return at once otherwise).
      const int zero = 0;
      for (uint32_t n = (it >= kStages ? it - kStages : 0); n < it; ++n)
        mbar_wait(bar(bars.full[n % kStages]), (n / kStages) & 1, &zero);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, kBN, false, false);
      uint32_t it = 0, tile = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
        const int chunk = u / p.n_m;
        const int nt_count = tiles_of(chunk);
        for (int t = 0; t < nt_count && ok; ++t, ++tile) {
          const uint32_t acc = tile & 1;
          if (tile >= 2 && !mbar_wait(bar(bars.acc_empty[acc]), ((tile >> 1) - 1) & 1, abort_flag, wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem + acc * kBN;
          for (int kb = 0; kb < p.n_kb; ++kb, ++it) {
            const uint32_t s = it % kStages;
            if (!mbar_wait(bar(bars.full[s]), (it / kStages) & 1, abort_flag, wait_ns)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a = sbase + s * kStageBytes, b = a + kABytes;
            const uint64_t ad = sdesc_sw128(a, 16, 1024), bd = sdesc_sw128(b, 16, 1024);
#pragma unroll
            for (int k = 0; k < kBK / 16; ++k)
              umma_ss(d_tmem, desc_add(ad, (k * 32) >> 4), desc_add(bd, (k * 32) >> 4), idesc, (kb | k) != 0);
            umma_commit(bar(bars.empty[s]));
          }
          if (!ok) break;
          umma_commit(bar(bars.acc_full[acc]));
        }
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
      }
      // every MMA this thread issued must finish before TMEM is released
      const int zero = 0;
      umma_commit(bar(bars.mma_done));
      mbar_wait(bar(bars.mma_done), 0, &zero);
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3;
    const int r = quad * 32 + lane;
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    uint32_t tile = 0;
    bool ok = true;
    for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
      const int chunk = u / p.n_m, mt = u - chunk * p.n_m;
      const int nt_count = tiles_of(chunk);
      Stats st{__int_as_float(0xff800000u), 0.f, 0.f, -1};
      for (int t = 0; t < nt_count; ++t, ++tile) {
        const uint32_t acc = tile & 1;
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.acc_full[acc]), (tile >> 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
        tc_fence_after();
        const int col0 = (chunk * p.tpu + t) * kBN;
#pragma unroll 1
        for (int c = 0; c < kBN / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(t_lane + acc * kBN + c * 32, v);
          const int cb = col0 + c * 32;
          if (cb >= p.vocab) continue;  // whole chunk past the vocabulary
          float x[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) x[j] = cb + j < p.vocab ? __uint_as_float(v[j]) : kMaskedLogit;
          absorb32(st, x, cb);
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.acc_empty[acc]));
      }
      if (!ok) break;
      const int row = mt * kBM + r;
      if (row < p.rows) p.part[static_cast<int64_t>(row) * p.n_chunks + chunk] = Partial{st.m, st.s, st.t, st.idx};
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// One warp per row: merges the row's partial states, then Eq. 2.
__global__ void __launch_bounds__(256) lm_head_decide_kernel(const Partial* __restrict__ part, int rows,
                                                             int n_chunks, const int32_t* __restrict__ committed,
                                                             const float* __restrict__ tau_per_row, float tau,
                                                             const uint8_t* __restrict__ editable,
                                                             int32_t* __restrict__ new_tokens,
                                                             uint8_t* __restrict__ edit_mask,
                                                             float* __restrict__ confidence,
                                                             int32_t* __restrict__ argmax_out,
                                                             float* __restrict__ entropy) {
  const int row = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  Stats st{__int_as_float(0xff800000u), 0.f, 0.f, -1};
  for (int c = lane; c < n_chunks; c += 32) {
    const Partial q = part[static_cast<int64_t>(row) * n_chunks + c];
    merge(st, Stats{q.m, q.s, q.t, q.idx});
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) merge(st, shfl_xor(st, off));
  if (lane != 0) return;
  const int32_t cur = committed[row];
  if (undecidable(st)) {
    // no softmax (the projection produced a NaN or +inf logit): no decision
    atomicOr(&g_error_word, MBE_DEVERR_NONFINITE);
    new_tokens[row] = cur;
    edit_mask[row] = 0;
    confidence[row] = nan_f32();
    if (argmax_out) argmax_out[row] = -1;
    if (entropy) entropy[row] = nan_f32();
    return;
  }
  const float c = 1.0f / st.s;
  const float tr = tau_per_row ? tau_per_row[row] : tau;
  const bool ed = (editable == nullptr || editable[row] != 0) && st.idx != cur && c > tr;
  new_tokens[row] = ed ? st.idx : cur;
  edit_mask[row] = ed ? 1 : 0;
  confidence[row] = c;
  if (argmax_out) argmax_out[row] = st.idx;
  if (entropy) entropy[row] = logf(st.s) - 0.6931471805599453f * st.t / st.s;
}

int tiles_per_unit(int rows, int vocab, int num_sms) {
  const int64_t tiles = static_cast<int64_t>((rows + kBM - 1) / kBM) * ((vocab + kBN - 1) / kBN);
  const int64_t t = tiles / (static_cast<int64_t>(kUnitsPerSm) * num_sms);
  return static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(kMaxTilesPerUnit, t)));
}

int num_chunks(int vocab, int tpu) {
  const int tiles = (vocab + kBN - 1) / kBN;
  return (tiles + tpu - 1) / tpu;
}

struct DeviceState {
  int num_sms = 0;
  bool attr_set = false;
};

DeviceState* device_state(int dev) {
  static DeviceState st[64];
  static std::mutex mu;
  if (dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  DeviceState& d = st[dev];
  if (d.num_sms == 0 && cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    d.num_sms = 0;
  if (d.num_sms > 0 && !d.attr_set) {
    if (cudaFuncSetAttribute(lm_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) ==
        cudaSuccess)
      d.attr_set = true;
  }
  return &d;
}

}  // namespace lmh
}  // namespace mbe

extern "C" size_t mbe_lm_head_workspace_size(int32_t rows, int32_t vocab) {
  if (rows <= 0 || vocab <= 0) return 0;
  // sized for one tile per unit, the finest split the kernel uses
  return static_cast<size_t>(rows) * mbe::lmh::num_chunks(vocab, 1) * sizeof(mbe::lmh::Partial);
}

extern "C" mbe_status mbe_lm_head_edit_decide(const void* hidden, const void* weight, int32_t rows, int32_t vocab,
                                              int32_t hidden_dim, const int32_t* committed,
                                              const float* tau_per_row_or_null, float tau,
                                              const uint8_t* editable_or_null, int32_t* new_tokens,
                                              uint8_t* edit_mask, float* confidence, int32_t* argmax_or_null,
                                              float* entropy_or_null, void* workspace, size_t workspace_bytes,
                                              cudaStream_t stream) {
  using namespace mbe;
  using namespace mbe::lmh;
  if (rows < 0 || vocab < 1 || hidden_dim < 8 || hidden_dim % 8 != 0) return MBE_ERR_INVALID_ARG;
  if (rows == 0) return MBE_OK;
  if (!hidden || !weight || !committed || !new_tokens || !edit_mask || !confidence || !workspace)
    return MBE_ERR_INVALID_ARG;
  if (!aligned16(hidden) || !aligned16(weight) || !aligned16(workspace)) return MBE_ERR_INVALID_ARG;
  if (vocab > (1 << 30) || rows > (1 << 30)) return MBE_ERR_UNSUPPORTED;
  if (workspace_bytes < mbe_lm_head_workspace_size(rows, vocab)) return MBE_ERR_WORKSPACE;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    record_cuda_error(e, "cudaGetDevice");
    return MBE_ERR_CUDA;
  }
  DeviceState* ds = device_state(dev);
  if (!ds || ds->num_sms <= 0 || !ds->attr_set) {
    record_cuda_error(cudaGetLastError(), "lm_head device setup");
    return MBE_ERR_CUDA;
  }
  CUtensorMap th, tw;
  {
    const cuuint64_t dims[2] = {(cuuint64_t)hidden_dim, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)hidden_dim * 2};
    const cuuint32_t box[2] = {kBK, kBM};
    if (!encode_bf16_sw128(&th, hidden, 2, dims, strides, box)) return MBE_ERR_CUDA;
  }
  {
    const cuuint64_t dims[2] = {(cuuint64_t)hidden_dim, (cuuint64_t)vocab};
    const cuuint64_t strides[1] = {(cuuint64_t)hidden_dim * 2};
    const cuuint32_t box[2] = {kBK, kBN};
    if (!encode_bf16_sw128(&tw, weight, 2, dims, strides, box)) return MBE_ERR_CUDA;
  }
  Params p;
  p.rows = rows;
  p.vocab = vocab;
  p.d = hidden_dim;
  p.n_m = (rows + kBM - 1) / kBM;
  p.tpu = tiles_per_unit(rows, vocab, ds->num_sms);
  p.n_chunks = num_chunks(vocab, p.tpu);
  p.n_units = p.n_m * p.n_chunks;
  p.n_kb = (hidden_dim + kBK - 1) / kBK;
  p.part = static_cast<Partial*>(workspace);
  p.wait_ns = wait_limit_ns();
  const int grid = std::min(p.n_units, ds->num_sms);
  lm_head_kernel<<<grid, kThreads, kSmemBytes, stream>>>(th, tw, p);
  mbe_status st = launch_status("lm_head_kernel");
  if (st != MBE_OK) return st;
  lm_head_decide_kernel<<<(rows + 7) / 8, 256, 0, stream>>>(p.part, rows, p.n_chunks, committed,
                                                             tau_per_row_or_null, tau, editable_or_null, new_tokens,
                                                             edit_mask, confidence, argmax_or_null, entropy_or_null);
  return launch_status("lm_head_decide_kernel");
}
