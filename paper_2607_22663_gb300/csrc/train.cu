// Multi-Block Edit SFT attention support (Sec. 3): the cross-block attention
// mask and the backward of attention under a block mask. The forward under the
// mask is mbe_block_mask_attention (attention.cu).
//
// sft_mask_kernel: one CTA per (mask row, sequence); thread w builds 32-bit
// word w of the row from the link rules, so a row of nb blocks costs nb bits.
//
// bwd_prep_kernel: delta = rowsum(dO o O) per (token, head), dQ zeroed, the
// work counter armed.
// bwd_kernel (persistent, one CTA per SM, 384 threads): a work unit is
// (sequence, KV head g, 128-key tile); K and V stay in shared memory while the
// unit walks the 128-row query tiles (packed rows token * G + head of the heads
// of g) that see any of its key blocks. Per query tile i:
//   warp 0      TMA: Q_i and dO_i into a 2-stage ring (K, V once per unit);
//               the tile's column data (lse, delta, which query blocks see
//               each key block of the unit) into shared memory
//   warp 1      MMA: S^T = K Q_i^T (SS, into TMEM); dP^T = V dO_i^T once the
//               dQ of tile i-1 has left TMEM; then dV += P^T dO_i (TS, P^T
//               from TMEM), dK += dS^T Q_i and dQ_i = dS K (SS, dS from
//               shared memory). S^T of tile i+1 follows dQ_i at once, so it
//               runs while the compute warps read dQ_i out.
//   warps 4-11  two warps per TMEM lane quadrant, splitting columns 0-63 /
//               64-127; thread = key row: P^T = exp(S^T * scale - lse),
//               masked, back to TMEM as bf16 over the warp's own S^T columns;
//               dS^T = P^T o (dP^T - delta) into shared memory as a [key][query
//               row] tile (K-major for dK, MN-major for dQ); then thread =
//               query row: dQ_i * scale into the stage Q_i and dO_i came in,
//               as 32 x 32 fp32 boxes that TMA adds into dQ in L2; at the
//               unit's end, thread = key row: dK * scale and dV stored (fp32).
// TMEM: dK, dV, S^T/P^T and dP^T/dQ, 128 columns each.
#include <cuda_bf16.h>
#include <algorithm>
#include <cmath>
#include <mutex>
#include "common.cuh"
#include "ptx_sm103.cuh"
#include "tma_host.cuh"

namespace mbe {

MBE_DEFINE_ERROR_WORD(train_take_error)

namespace {

// Does block q attend to block k? Blocks: prompt [0, Np), noisy n_i = Np + i,
// clean c_j = Np + N + j (i, j < N).
__device__ __forceinline__ bool sft_link(int q, int k, int Np, int N, int K) {
  if (k < Np) return true;    // the prompt is visible to every block
  if (q < Np) return false;   // prompt blocks see only the prompt
  const bool q_noisy = q < Np + N, k_noisy = k < Np + N;
  const int qi = q_noisy ? q - Np : q - Np - N;
  const int ki = k_noisy ? k - Np : k - Np - N;
  if (q_noisy) {
    if (k_noisy) return ki == qi;                    // NN: its own block
    return ki < qi || (ki > qi && ki <= qi + K - 1);  // NC and NF
  }
  if (k_noisy) return ki >= qi - K + 1 && ki <= qi - 1;  // CN
  return ki == qi || ki <= qi - K;                        // CC without the implicated links
}

__global__ void __launch_bounds__(128) sft_mask_kernel(const int32_t* __restrict__ n_prompt_blocks,
                                                       const int32_t* __restrict__ n_blocks, int K, int mask_rows,
                                                       int mask_words, uint32_t* __restrict__ mask) {
  const int q = blockIdx.x, s = blockIdx.y;
  const int Np = n_prompt_blocks[s], N = n_blocks[s];
  const int64_t nb = static_cast<int64_t>(Np) + 2ll * N;
  const bool ok = Np >= 0 && N >= 0 && nb <= mask_rows;
  if (!ok && q == 0 && threadIdx.x == 0) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
  uint32_t* row = mask + (static_cast<int64_t>(s) * mask_rows + q) * mask_words;
  for (int w = threadIdx.x; w < mask_words; w += blockDim.x) {
    uint32_t word = 0;
    if (ok && q < nb) {
      for (int b = 0; b < 32; ++b) {
        const int k = 32 * w + b;
        if (k < nb && sft_link(q, k, Np, N, K)) word |= 1u << b;
      }
    }
    row[w] = word;
  }
}

}  // namespace

namespace bwd {

constexpr int kD = 128;                      // head size of the backward
constexpr int kTile = 128;                   // keys per key tile = packed rows per query tile
constexpr int kThreads = 384;                // 4 role warps + 8 compute warps (two per TMEM lane quadrant)
constexpr int kMaxQWords = 16;               // query-tile bitmask of a unit (<= 512 query tiles)
constexpr int kMaxKeyBlocks = 16;            // key blocks of a 128-key tile (block size >= 8)
constexpr uint32_t kHalf = 128 * 128;        // a 64-column half of a 128-row bf16 tile (16 KB)
constexpr uint32_t kTileBytes = 2 * kHalf;   // 32 KB
constexpr uint32_t kStageBytes = 2 * kTileBytes;  // Q_i and dO_i, then the fp32 dQ_i of the same tile
constexpr uint32_t kBoxBytes = 32 * 128;     // a dQ box: 32 rows x 32 fp32 (one 128-byte row each)
constexpr uint32_t kK = 0, kV = kTileBytes, kStage = 2 * kTileBytes, kDS = kStage + 2 * kStageBytes;
constexpr uint32_t kSmemBytes = kDS + kTileBytes + 1024;  // + 1024-byte alignment slack
constexpr uint32_t kTmDK = 0, kTmDV = 128, kTmS = 256, kTmDP = 384, kTmCols = 512;
constexpr float kLog2e = 1.4426950408889634f;

struct Params {
  const int32_t* seq_len;
  const int32_t* cu;
  const uint32_t* mask;
  const float* lse;
  const float* delta;
  const int32_t* unit_start;  // [batch + 1]: first work unit of each sequence
  int* counter;               // [0] work queue, [1] plan blocks done, [2] work units planned
  int* unit_nq;               // [max_units]: visible query tiles of each unit
  int* unit_order;            // [max_units]: units by descending visible query tiles
  uint32_t* unit_bits;        // [max_units][kMaxQWords]: the visible query tiles
  int max_units;
  float* dk;
  float* dv;
  int mask_rows, mask_words, block_log2;
  int batch, total_tokens, Hq, Hkv, G, lgG;
  float scale, scale_log2;
};

struct Unit {
  int32_t seq, g, kt, len, cu;
};

struct Bars {
  uint64_t u_full[2], u_empty[2], q_full[2], q_empty[2], kv_full, kv_empty, col_full, col_empty, s_full, dp_full,
      p_full, dq_full, dq_empty, acc_full, acc_empty, mma_done;
};

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ bool mask_bit(const Params& p, int seq, int qb, int kb) {
  if (qb < 0 || qb >= p.mask_rows || kb < 0 || (kb >> 5) >= p.mask_words) return false;
  return (p.mask[(static_cast<int64_t>(seq) * p.mask_rows + qb) * p.mask_words + (kb >> 5)] >> (kb & 31)) & 1u;
}

// Does any query block of query tile i see a key block of key tile kt?
__device__ __forceinline__ bool qtile_visible(const Params& p, const Unit& u, int i) {
  const int q0 = (i * kTile) >> p.lgG, q1 = min(u.len, ((i + 1) * kTile) >> p.lgG) - 1;
  const int k0 = u.kt * kTile, k1 = min(u.len, k0 + kTile) - 1;
  if (q1 < q0 || k1 < k0) return false;
  for (int qb = q0 >> p.block_log2; qb <= (q1 >> p.block_log2); ++qb)
    for (int kb = k0 >> p.block_log2; kb <= (k1 >> p.block_log2); ++kb)
      if (mask_bit(p, u.seq, qb, kb)) return true;
  return false;
}

__device__ __forceinline__ int next_bit(const volatile uint32_t* bits, int i) {
  for (int b = i + 1; b < kMaxQWords * 32;) {
    const uint32_t w = bits[b >> 5] >> (b & 31);
    if (w) return b + __ffs(w) - 1;
    b = (b & ~31) + 32;
  }
  return -1;
}

// Work unit u: (sequence, KV head, key tile), key tiles fastest.
__device__ __forceinline__ Unit decode_unit(const Params& p, int u) {
  int lo = 0, hi = p.batch - 1;  // the sequence whose unit range holds u
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.unit_start[mid] <= u) lo = mid; else hi = mid - 1;
  }
  const int len = p.seq_len[lo];
  const int tiles = max((len + kTile - 1) / kTile, 1);
  const int r = u - p.unit_start[lo];
  return Unit{lo, r / tiles, r % tiles, len, p.cu[lo]};
}

// First and (capped) last query block of query tile i.
__device__ __forceinline__ int qblock0(const Params& p, int i) { return ((i * kTile) >> p.lgG) >> p.block_log2; }
__device__ __forceinline__ int qblock_count(const Params& p, const Unit& u, int i) {
  const int last = min(u.len - 1, ((i + 1) * kTile - 1) >> p.lgG) >> p.block_log2;
  return min(32, last - qblock0(p, i) + 1);
}

__global__ void __launch_bounds__(kThreads, 1)
    bwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_do,
               const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v,
               const __grid_constant__ CUtensorMap tm_dq, const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) Bars bars;
  __shared__ Unit ring[2];
  __shared__ uint32_t ring_bits[2][kMaxQWords];
  // column data of the current query tile, written by the producer warp
  __shared__ __align__(16) float col_lse[kTile];    // lse in log2 units; +inf past the sequence (P = 0)
  __shared__ __align__(16) float col_delta[kTile];  // rowsum(dO o O)
  __shared__ uint32_t col_kvis[kMaxKeyBlocks];      // per key block of the unit: bit b = query block qb0 + b sees it
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  volatile int* abort_flag = &abort_s;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  auto bar = [](uint64_t& b) { return smem_u32(&b); };
  const int n_units = p.counter[2];

  if (tid == 0) {
    abort_s = 0;
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(bars.u_full[i]), 1);
      mbar_init(bar(bars.u_empty[i]), 9);  // MMA issuer + 8 compute warps
      mbar_init(bar(bars.q_full[i]), 1);
      mbar_init(bar(bars.q_empty[i]), 8);  // each compute warp once its dQ boxes have been read
    }
    mbar_init(bar(bars.kv_full), 1);
    mbar_init(bar(bars.kv_empty), 1);
    mbar_init(bar(bars.col_full), 1);
    mbar_init(bar(bars.col_empty), 8);
    mbar_init(bar(bars.s_full), 1);
    mbar_init(bar(bars.dp_full), 1);
    mbar_init(bar(bars.p_full), 8);
    mbar_init(bar(bars.dq_full), 1);
    mbar_init(bar(bars.dq_empty), 8);
    mbar_init(bar(bars.acc_full), 1);
    mbar_init(bar(bars.acc_empty), 8);
    mbar_init(bar(bars.mma_done), 1);
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), kTmCols);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    constexpr unsigned kAll = 0xffffffffu;
    if (lane == 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_do);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
    }
    uint32_t u_it = 0, kv_loads = 0, q_loads = 0, cols = 0;
    bool ok = true;
    for (;;) {
      int uidx = 0;
      if (lane == 0) uidx = atomicAdd(p.counter, 1);
      uidx = __shfl_sync(kAll, uidx, 0);
      const bool done = uidx >= n_units;
      const int slot = u_it & 1;
      if (u_it >= 2) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.u_empty[slot]), ((u_it >> 1) - 1) & 1, abort_flag));
        if (!ok) break;
      }
      Unit un{-1, 0, 0, 0, 0};
      if (!done) {
        // units in the planned order: most visible query tiles first
        const int u = p.unit_order[uidx];
        un = decode_unit(p, u);
        if (lane < kMaxQWords) ring_bits[slot][lane] = p.unit_bits[static_cast<int64_t>(u) * kMaxQWords + lane];
      }
      __syncwarp();
      if (lane == 0) {
        ring[slot] = un;
        mbar_arrive(bar(bars.u_full[slot]));
      }
      __syncwarp();
      ++u_it;
      if (done) break;
      const volatile uint32_t* bits = ring_bits[slot];
      int n_q = 0;
      for (int w = 0; w < kMaxQWords; ++w) n_q += __popc(bits[w]);
      if (n_q == 0) continue;
      if (kv_loads >= 1) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.kv_empty), (kv_loads - 1) & 1, abort_flag));
        if (!ok) break;
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(bar(bars.kv_full), 2 * kTileBytes);
        for (int h = 0; h < 2; ++h) {
          tma_load_3d(sbase + kK + h * kHalf, &tm_k, bar(bars.kv_full), h * 64, un.g, un.cu + un.kt * kTile);
          tma_load_3d(sbase + kV + h * kHalf, &tm_v, bar(bars.kv_full), h * 64, un.g, un.cu + un.kt * kTile);
        }
      }
      ++kv_loads;
      const int kb_first = (un.kt * kTile) >> p.block_log2;
      const int kb_last = (min(un.len, (un.kt + 1) * kTile) - 1) >> p.block_log2;
      for (int i = next_bit(bits, -1); i >= 0 && ok; i = next_bit(bits, i)) {
        const uint32_t st = q_loads & 1;
        if (q_loads >= 2) {
          ok = __all_sync(kAll, mbar_wait(bar(bars.q_empty[st]), ((q_loads >> 1) - 1) & 1, abort_flag));
          if (!ok) break;
        }
        if (lane == 0) {
          const uint32_t qa = sbase + kStage + st * kStageBytes;
          mbar_arrive_expect_tx(bar(bars.q_full[st]), kStageBytes);
          const int tok = un.cu + ((i * kTile) >> p.lgG);
          for (int h = 0; h < 2; ++h) {
            tma_load_3d(qa + h * kHalf, &tm_q, bar(bars.q_full[st]), h * 64, un.g * p.G, tok);
            tma_load_3d(qa + kTileBytes + h * kHalf, &tm_do, bar(bars.q_full[st]), h * 64, un.g * p.G, tok);
          }
        }
        ++q_loads;
        // column data of tile i, fetched before waiting for the compute warps to
        // finish with the previous tile's
        float lse_r[4], dl_r[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int R = i * kTile + lane + 32 * e;
          const int tok = R >> p.lgG, head = un.g * p.G + (R & (p.G - 1));
          const bool qv = tok < un.len;
          const int64_t row = (static_cast<int64_t>(un.cu) + tok) * p.Hq + head;
          lse_r[e] = qv ? p.lse[row] * kLog2e : __int_as_float(0x7f800000);
          dl_r[e] = qv ? p.delta[row] : 0.f;
        }
        const int qb0 = qblock0(p, i), nqb = qblock_count(p, un, i);
        uint32_t kvis = 0;
        if (lane < kMaxKeyBlocks && kb_first + lane <= kb_last)
          for (int b = 0; b < nqb; ++b)
            if (mask_bit(p, un.seq, qb0 + b, kb_first + lane)) kvis |= 1u << b;
        if (cols >= 1) {
          ok = __all_sync(kAll, mbar_wait(bar(bars.col_empty), (cols - 1) & 1, abort_flag));
          if (!ok) break;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          col_lse[lane + 32 * e] = lse_r[e];
          col_delta[lane + 32 * e] = dl_r[e];
        }
        if (lane < kMaxKeyBlocks) col_kvis[lane] = kvis;
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.col_full));
        ++cols;
      }
      if (!ok) break;
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
      // let the copies already issued land before the CTA can exit
      const int zero = 0;
      if (kv_loads >= 1) mbar_wait(bar(bars.kv_full), (kv_loads - 1) & 1, &zero);
      for (uint32_t n = (q_loads >= 2 ? q_loads - 2 : 0); n < q_loads; ++n)
        mbar_wait(bar(bars.q_full[n & 1]), (n >> 1) & 1, &zero);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_kk = idesc_bf16_f32(kTile, kTile, false, false);  // S^T, dP^T
      constexpr uint32_t idesc_tb = idesc_bf16_f32(kTile, kD, false, true);      // dV, dK: MN-major B
      constexpr uint32_t idesc_dq = idesc_bf16_f32(kTile, kD, true, true);       // dQ: MN-major A and B
      uint32_t u_it = 0, units = 0, tiles = 0;
      bool ok = true;
      for (;;) {
        const int slot = u_it & 1;
        if (!mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag)) { ok = false; break; }
        const Unit un = ring[slot];
        int n_q = 0;
        for (int w = 0; w < kMaxQWords; ++w) n_q += __popc(ring_bits[slot][w]);
        mbar_arrive(bar(bars.u_empty[slot]));
        ++u_it;
        if (un.seq < 0) break;
        if (n_q == 0) continue;
        if (!mbar_wait(bar(bars.kv_full), units & 1, abort_flag)) { ok = false; break; }
        for (int j = 0; j < n_q; ++j, ++tiles) {
          const uint32_t st = tiles & 1;
          if (!mbar_wait(bar(bars.q_full[st]), (tiles >> 1) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
          const uint32_t qa = sbase + kStage + st * kStageBytes, da = qa + kTileBytes;
          // S^T = K Q_i^T over the previous tile's P^T (read by MMAs issued before)
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint32_t off = h * kHalf + k * 32;
              umma_ss(tmem + kTmS, sdesc_sw128(sbase + kK + off, 16, 1024), sdesc_sw128(qa + off, 16, 1024), idesc_kk,
                      (h | k) ? 1u : 0u);
            }
          umma_commit(bar(bars.s_full));
          // dP^T = V dO_i^T, once the previous tile's dQ has been read out of the region
          if (tiles >= 1 && !mbar_wait(bar(bars.dq_empty), (tiles - 1) & 1, abort_flag)) { ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int h = 0; h < 2; ++h)
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const uint32_t off = h * kHalf + k * 32;
              umma_ss(tmem + kTmDP, sdesc_sw128(sbase + kV + off, 16, 1024), sdesc_sw128(da + off, 16, 1024),
                      idesc_kk, (h | k) ? 1u : 0u);
            }
          umma_commit(bar(bars.dp_full));
          if (!mbar_wait(bar(bars.p_full), tiles & 1, abort_flag)) { ok = false; break; }
          if (j == 0 && units >= 1 && !mbar_wait(bar(bars.acc_empty), (units - 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk) {
            const uint32_t acc = (j > 0 || kk > 0) ? 1u : 0u;
            // P^T of query columns 64 h .. 64 h + 63 sits packed at S region columns 64 h .. 64 h + 31
            umma_ts(tmem + kTmDV, tmem + kTmS + (kk >> 2) * 64 + (kk & 3) * 8,
                    sdesc_sw128(da + kk * 16 * 128, kHalf, 1024), idesc_tb, acc);
            // dS^T from shared memory: [key][query row] is K-major for A = dS^T
            umma_ss(tmem + kTmDK, sdesc_sw128(sbase + kDS + (kk >> 2) * kHalf + (kk & 3) * 32, 16, 1024),
                    sdesc_sw128(qa + kk * 16 * 128, kHalf, 1024), idesc_tb, acc);
          }
          // dQ_i = dS K (the same tile as MN-major A) into the dP region
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk)
            umma_ss(tmem + kTmDP, sdesc_sw128(sbase + kDS + kk * 16 * 128, kHalf, 1024),
                    sdesc_sw128(sbase + kK + kk * 16 * 128, kHalf, 1024), idesc_dq, kk > 0 ? 1u : 0u);
          umma_commit(bar(bars.dq_full));
        }
        if (!ok) break;
        umma_commit(bar(bars.acc_full));
        umma_commit(bar(bars.kv_empty));
        ++units;
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
      }
      const int zero = 0;
      umma_commit(bar(bars.mma_done));
      mbar_wait(bar(bars.mma_done), 0, &zero);
    }
  } else if (warp >= 4) {
    // ---------------------------------------------------------------- compute warps
    const int quad = warp & 3;
    const int hf = (warp - 4) >> 2;  // the pair of warps of a quadrant splits columns 0-63 / 64-127
    const int r = quad * 32 + lane;  // TMEM lane: key row, or query row for dQ
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const int sh = p.lgG + p.block_log2;  // packed row -> query block
    uint32_t u_it = 0, units = 0, tiles = 0;
    bool ok = true;
    for (;;) {
      const int slot = u_it & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag));
      if (!ok) break;
      const Unit un = ring[slot];
      const volatile uint32_t* bits = ring_bits[slot];
      ++u_it;
      auto release = [&]() {
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.u_empty[slot]));
      };
      if (un.seq < 0) {
        release();
        break;
      }
      int n_q = 0;
      for (int w = 0; w < kMaxQWords; ++w) n_q += __popc(bits[w]);
      const int key = un.kt * kTile + r;
      const bool key_ok = key < un.len;
      const int64_t kv_row = (static_cast<int64_t>(un.cu) + key) * p.Hkv + un.g;
      if (n_q == 0) {  // no query sees these keys: zero gradients (dK by one half, dV by the other)
        release();
        float* dst = (hf == 0 ? p.dk : p.dv) + kv_row * kD;
        if (key_ok)
          for (int d = 0; d < kD; d += 4) *reinterpret_cast<float4*>(dst + d) = make_float4(0.f, 0.f, 0.f, 0.f);
        continue;
      }
      const int kb_rel = (key >> p.block_log2) - ((un.kt * kTile) >> p.block_log2);
      for (int i = next_bit(bits, -1); i >= 0; i = next_bit(bits, i), ++tiles) {
        const uint32_t st = tiles & 1;
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.col_full), tiles & 1, abort_flag));
        if (!ok) break;
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.s_full), tiles & 1, abort_flag));
        if (!ok) break;
        tc_fence_after();
        const int qb0 = qblock0(p, i), nqb = qblock_count(p, un, i);
        const uint32_t all = nqb >= 32 ? 0xFFFFFFFFu : ((1u << nqb) - 1u);
        // query blocks of this tile that see this key row's block
        const uint32_t qvis = key_ok ? (col_kvis[kb_rel] & all) : 0u;
        // TMEM loads are warp-wide: the warp skips them only if no lane needs them
        const bool any_vis = __any_sync(0xffffffffu, qvis != 0u);
        const bool every = __all_sync(0xffffffffu, qvis == all);
        // P^T of this warp's 64 columns, packed to bf16 pairs
        uint32_t pw[32];
        if (!any_vis) {
#pragma unroll
          for (int m = 0; m < 32; ++m) pw[m] = 0u;
        } else {
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            uint32_t sv[32];
            tmem_ld32(t_lane + kTmS + 64 * hf + 32 * c, sv);
#pragma unroll
            for (int jj = 0; jj < 32; jj += 4) {
              const int col = 64 * hf + 32 * c + jj;
              const float4 l4 = *reinterpret_cast<const float4*>(&col_lse[col]);
              float x[4] = {fmaf(__uint_as_float(sv[jj]), p.scale_log2, -l4.x),
                            fmaf(__uint_as_float(sv[jj + 1]), p.scale_log2, -l4.y),
                            fmaf(__uint_as_float(sv[jj + 2]), p.scale_log2, -l4.z),
                            fmaf(__uint_as_float(sv[jj + 3]), p.scale_log2, -l4.w)};
              if (!every) {
#pragma unroll
                for (int e = 0; e < 4; ++e)
                  if (!((qvis >> (((i * kTile + col + e) >> sh) - qb0)) & 1u)) x[e] = __int_as_float(0xff800000);
              }
              pw[16 * c + jj / 2] = pack_bf16x2(ex2f(x[0]), ex2f(x[1]));
              pw[16 * c + jj / 2 + 1] = pack_bf16x2(ex2f(x[2]), ex2f(x[3]));
            }
          }
        }
        // P^T over S^T columns this warp has already read: 64 hf .. 64 hf + 31
        tmem_st32(t_lane + kTmS + 64 * hf, pw);
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.dp_full), tiles & 1, abort_flag));
        if (!ok) break;
        tc_fence_after();
        // dS^T = P^T o (dP^T - delta) into shared memory: row r of a [key][query row] tile
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          uint32_t dsw[16];
          if (!any_vis) {
#pragma unroll
            for (int m = 0; m < 16; ++m) dsw[m] = 0u;
          } else {
            uint32_t dv[32];
            tmem_ld32(t_lane + kTmDP + 64 * hf + 32 * c, dv);
#pragma unroll
            for (int jj = 0; jj < 32; jj += 4) {
              const int col = 64 * hf + 32 * c + jj;
              const float4 d4 = *reinterpret_cast<const float4*>(&col_delta[col]);
              const uint32_t pa = pw[16 * c + jj / 2], pb = pw[16 * c + jj / 2 + 1];
              dsw[jj / 2] = pack_bf16x2(__uint_as_float(pa << 16) * (__uint_as_float(dv[jj]) - d4.x),
                                        __uint_as_float(pa & 0xFFFF0000u) * (__uint_as_float(dv[jj + 1]) - d4.y));
              dsw[jj / 2 + 1] = pack_bf16x2(__uint_as_float(pb << 16) * (__uint_as_float(dv[jj + 2]) - d4.z),
                                            __uint_as_float(pb & 0xFFFF0000u) * (__uint_as_float(dv[jj + 3]) - d4.w));
            }
          }
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int chunk = (c * 4 + q) ^ (r & 7);
            *reinterpret_cast<uint4*>(smem + kDS + hf * kHalf + r * 128 + chunk * 16) =
                make_uint4(dsw[4 * q], dsw[4 * q + 1], dsw[4 * q + 2], dsw[4 * q + 3]);
          }
        }
        tmem_st_wait();
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(bar(bars.p_full));
          mbar_arrive(bar(bars.col_empty));
        }
        // dQ_i: thread = query row r of the tile, this warp's half of the head dimension
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.dq_full), tiles & 1, abort_flag));
        if (!ok) break;
        tc_fence_after();
        uint32_t o0[32], o1[32];
        tmem_ld32(t_lane + kTmDP + 64 * hf, o0);
        tmem_ld32(t_lane + kTmDP + 64 * hf + 32, o1);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.dq_empty));
        // The tile's MMAs are done with Q_i and dO_i: their stage takes dQ_i * scale as
        // two boxes of this warp (32 rows x 32 fp32, 128-byte swizzle) that TMA adds into dQ.
        // Rows past the sequence are exact zeros (P = 0 there).
        const uint32_t box = kStage + st * kStageBytes + (quad * 4 + hf * 2) * kBoxBytes;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const uint32_t at = lane * 128 + ((q ^ (lane & 7)) * 16);
          *reinterpret_cast<float4*>(smem + box + at) =
              make_float4(__uint_as_float(o0[4 * q]) * p.scale, __uint_as_float(o0[4 * q + 1]) * p.scale,
                          __uint_as_float(o0[4 * q + 2]) * p.scale, __uint_as_float(o0[4 * q + 3]) * p.scale);
          *reinterpret_cast<float4*>(smem + box + kBoxBytes + at) =
              make_float4(__uint_as_float(o1[4 * q]) * p.scale, __uint_as_float(o1[4 * q + 1]) * p.scale,
                          __uint_as_float(o1[4 * q + 2]) * p.scale, __uint_as_float(o1[4 * q + 3]) * p.scale);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          const int tok = un.cu + ((i * kTile + quad * 32) >> p.lgG);
          tma_reduce_add_3d(&tm_dq, sbase + box, 64 * hf, un.g * p.G, tok);
          tma_reduce_add_3d(&tm_dq, sbase + box + kBoxBytes, 64 * hf + 32, un.g * p.G, tok);
          bulk_commit_group();
          bulk_wait_group_read0();  // the stage may be refilled once TMA has read the boxes
          mbar_arrive(bar(bars.q_empty[st]));
        }
        __syncwarp();
      }
      if (!ok) break;
      release();
      // dK (first half of the pair) and dV (second half) of the unit's keys: thread = key row
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.acc_full), units & 1, abort_flag));
      if (!ok) break;
      tc_fence_after();
      {
        const uint32_t src = hf == 0 ? kTmDK : kTmDV;
        const float mul = hf == 0 ? p.scale : 1.f;
        float* dst = (hf == 0 ? p.dk : p.dv) + kv_row * kD;
#pragma unroll 1
        for (int c4 = 0; c4 < kD / 32; ++c4) {
          uint32_t a[32];
          tmem_ld32(t_lane + src + 32 * c4, a);
          if (key_ok)
#pragma unroll
            for (int e = 0; e < 32; e += 4)
              *reinterpret_cast<float4*>(dst + 32 * c4 + e) =
                  make_float4(__uint_as_float(a[e]) * mul, __uint_as_float(a[e + 1]) * mul,
                              __uint_as_float(a[e + 2]) * mul, __uint_as_float(a[e + 3]) * mul);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(bars.acc_empty));
      ++units;
    }
    if (lane == 0) bulk_wait_group0();  // every dQ addition of this warp done before the CTA exits
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
    }
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmCols);
  }
}

// The backward's work list: one warp per unit finds the query tiles that see
// its key tile; the last block to finish orders the units by descending count
// (a counting sort), so the persistent kernel takes the longest units first.
__global__ void __launch_bounds__(256) bwd_plan_kernel(const Params p) {
  constexpr int kBins = kMaxQWords * 32 + 1;
  __shared__ int hist[kBins];
  __shared__ int last_s;
  const int lane = threadIdx.x & 31;
  const int n_all = p.unit_start[p.batch];
  const int n_units = min(n_all, min(p.max_units, static_cast<int>(gridDim.x) * 8));
  const int u = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (u < n_units) {
    const Unit un = decode_unit(p, u);
    const int n_qt = ((un.len << p.lgG) + kTile - 1) / kTile;
    int n_q = 0;
    for (int w = 0; w < kMaxQWords; ++w) {
      const int i = 32 * w + lane;
      const uint32_t word = __ballot_sync(0xffffffffu, i < n_qt && qtile_visible(p, un, i));
      if (lane == 0) p.unit_bits[static_cast<int64_t>(u) * kMaxQWords + w] = word;
      n_q += __popc(word);
    }
    if (lane == 0) p.unit_nq[u] = n_q;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    last_s = atomicAdd(&p.counter[1], 1) == static_cast<int>(gridDim.x) - 1;
  }
  __syncthreads();
  if (!last_s) return;
  __threadfence();
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) hist[b] = 0;
  __syncthreads();
  for (int v = threadIdx.x; v < n_units; v += blockDim.x) atomicAdd(&hist[__ldcg(&p.unit_nq[v])], 1);
  __syncthreads();
  if (threadIdx.x < 32) {
    // exclusive prefix over the bins taken from the top: lane l owns 17 bins
    constexpr int kPer = (kBins + 31) / 32;
    int sum = 0;
    for (int j = lane * kPer; j < min(kBins, (lane + 1) * kPer); ++j) sum += hist[kBins - 1 - j];
    int incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, off);
      if (lane >= off) incl += y;
    }
    int acc = incl - sum;
    for (int j = lane * kPer; j < min(kBins, (lane + 1) * kPer); ++j) {
      const int c = hist[kBins - 1 - j];
      hist[kBins - 1 - j] = acc;
      acc += c;
    }
  }
  __syncthreads();
  for (int v = threadIdx.x; v < n_units; v += blockDim.x) p.unit_order[atomicAdd(&hist[__ldcg(&p.unit_nq[v])], 1)] = v;
  if (threadIdx.x == 0) {
    p.counter[2] = n_units;
    if (n_units < n_all) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
  }
}

// delta = rowsum(dO o O) per (token, head) (one warp per row), dQ zeroed, unit
// offsets and the work counters set up by block 0.
__global__ void __launch_bounds__(256) bwd_prep_kernel(const __nv_bfloat16* __restrict__ out,
                                                       const __nv_bfloat16* __restrict__ dout, int64_t rows,
                                                       float* __restrict__ delta, float* __restrict__ dq,
                                                       const int32_t* __restrict__ seq_len, int batch, int Hkv,
                                                       int32_t* unit_start, int* counter) {
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (blockDim.x / 32);
  for (int64_t row = static_cast<int64_t>(blockIdx.x) * (blockDim.x / 32) + threadIdx.x / 32; row < rows;
       row += warps) {
    const uint2 a = reinterpret_cast<const uint2*>(out + row * kD)[lane];
    const uint2 b = reinterpret_cast<const uint2*>(dout + row * kD)[lane];
    const float2 a0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&a.x));
    const float2 a1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&a.y));
    const float2 b0 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&b.x));
    const float2 b1 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&b.y));
    float s = a0.x * b0.x + a0.y * b0.y + a1.x * b1.x + a1.y * b1.y;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) delta[row] = s;
    reinterpret_cast<float4*>(dq + row * kD)[lane] = make_float4(0.f, 0.f, 0.f, 0.f);
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    int acc = 0;
    for (int s = 0; s < batch; ++s) {
      unit_start[s] = acc;
      const int len = seq_len[s];
      acc += len > 0 ? Hkv * ((len + kTile - 1) / kTile) : 0;
    }
    unit_start[batch] = acc;
    counter[0] = 0;
    counter[1] = 0;
  }
}

// Workspace: work counters and unit offsets, delta, then the work-unit plan
// (sized for at most num_q_heads KV heads).
struct WsLayout {
  size_t delta, nq, order, bits, total;
  int64_t max_units;
};

inline WsLayout ws_layout(int64_t batch, int64_t total_tokens, int64_t num_q_heads) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  WsLayout L;
  L.max_units = std::min<int64_t>(num_q_heads * ((total_tokens + kTile - 1) / kTile + batch), 1 << 30);
  L.delta = up(16 + static_cast<size_t>(batch + 1) * sizeof(int32_t));
  L.nq = up(L.delta + static_cast<size_t>(total_tokens) * num_q_heads * sizeof(float));
  L.order = up(L.nq + static_cast<size_t>(L.max_units) * sizeof(int32_t));
  L.bits = up(L.order + static_cast<size_t>(L.max_units) * sizeof(int32_t));
  L.total = L.bits + static_cast<size_t>(L.max_units) * kMaxQWords * sizeof(uint32_t);
  return L;
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
  if (d.num_sms > 0 && !d.attr_set &&
      cudaFuncSetAttribute(bwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) == cudaSuccess)
    d.attr_set = true;
  return &d;
}

}  // namespace bwd
}  // namespace mbe

extern "C" size_t mbe_block_mask_attention_bwd_workspace_size(int32_t batch, int32_t total_tokens,
                                                              int32_t num_q_heads) {
  if (batch < 0 || total_tokens < 0 || num_q_heads < 1) return 0;
  return mbe::bwd::ws_layout(batch, total_tokens, num_q_heads).total;
}

extern "C" mbe_status mbe_block_mask_attention_bwd(const void* q, const void* k, const void* v, const void* out,
                                                   const void* dout, const float* lse, const int32_t* seq_len,
                                                   const int32_t* cu_seqlens, const uint32_t* mask, int32_t mask_rows,
                                                   int32_t mask_words, int32_t batch, int32_t total_tokens,
                                                   int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                                   int32_t block_size, int32_t max_seq_len, float softmax_scale,
                                                   float* dq, float* dk, float* dv, void* workspace,
                                                   size_t workspace_bytes, cudaStream_t stream) {
  using namespace mbe;
  using namespace mbe::bwd;
  if (batch < 0 || total_tokens < 0 || num_q_heads < 1 || num_kv_heads < 1 || num_q_heads % num_kv_heads != 0 ||
      block_size < 8 || (block_size & (block_size - 1)) != 0 || mask_rows < 1 || mask_words < 1 ||
      static_cast<int64_t>(mask_words) * 32 < mask_rows || max_seq_len < 0 || !(softmax_scale >= 0.f))
    return MBE_ERR_INVALID_ARG;
  if (head_dim != kD) return MBE_ERR_UNSUPPORTED;
  const int G = num_q_heads / num_kv_heads;
  if (G > 32 || 32 % G != 0) return MBE_ERR_UNSUPPORTED;  // a warp's 32 query rows are whole tokens
  if (static_cast<int64_t>(max_seq_len) * G > static_cast<int64_t>(kMaxQWords) * 32 * kTile) return MBE_ERR_UNSUPPORTED;
  if ((max_seq_len + block_size - 1) / block_size > mask_rows) return MBE_ERR_INVALID_ARG;
  if (batch == 0 || total_tokens == 0) return MBE_OK;
  if (!q || !k || !v || !out || !dout || !lse || !seq_len || !cu_seqlens || !mask || !dq || !dk || !dv)
    return MBE_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out) || !aligned16(dout) || !aligned16(dq) ||
      !aligned16(dk) || !aligned16(dv))
    return MBE_ERR_INVALID_ARG;
  if (!workspace || workspace_bytes < mbe_block_mask_attention_bwd_workspace_size(batch, total_tokens, num_q_heads) ||
      !aligned16(workspace))
    return MBE_ERR_WORKSPACE;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    record_cuda_error(e, "cudaGetDevice");
    return MBE_ERR_CUDA;
  }
  DeviceState* ds = device_state(dev);
  if (!ds || ds->num_sms <= 0 || !ds->attr_set) {
    record_cuda_error(cudaGetLastError(), "block-mask backward setup");
    return MBE_ERR_CUDA;
  }
  CUtensorMap tq, tdo, tk, tv;
  {
    const cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)num_q_heads, (cuuint64_t)total_tokens};
    const cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)num_q_heads * kD * 2};
    const cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)(kTile / G)};
    if (!encode_bf16_sw128(&tq, q, 3, dims, strides, box) || !encode_bf16_sw128(&tdo, dout, 3, dims, strides, box))
      return MBE_ERR_CUDA;
  }
  {
    const cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)num_kv_heads, (cuuint64_t)total_tokens};
    const cuuint64_t strides[2] = {(cuuint64_t)kD * 2, (cuuint64_t)num_kv_heads * kD * 2};
    const cuuint32_t box[3] = {64, 1, (cuuint32_t)kTile};
    if (!encode_bf16_sw128(&tk, k, 3, dims, strides, box) || !encode_bf16_sw128(&tv, v, 3, dims, strides, box))
      return MBE_ERR_CUDA;
  }
  CUtensorMap tdq;  // fp32 dQ, added into by 32-row x 32-column boxes
  {
    const cuuint64_t dims[3] = {(cuuint64_t)kD, (cuuint64_t)num_q_heads, (cuuint64_t)total_tokens};
    const cuuint64_t strides[2] = {(cuuint64_t)kD * 4, (cuuint64_t)num_q_heads * kD * 4};
    const cuuint32_t box[3] = {32, (cuuint32_t)G, (cuuint32_t)(32 / G)};
    if (!encode_f32_sw128(&tdq, dq, 3, dims, strides, box)) return MBE_ERR_CUDA;
  }
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const WsLayout L = ws_layout(batch, total_tokens, num_q_heads);
  int* counter = reinterpret_cast<int*>(ws);
  int32_t* unit_start = reinterpret_cast<int32_t*>(ws + 16);
  float* delta = reinterpret_cast<float*>(ws + L.delta);
  const int64_t rows = static_cast<int64_t>(total_tokens) * num_q_heads;
  const int64_t prep_blocks = std::min<int64_t>((rows + 7) / 8, 8ll * ds->num_sms);
  bwd_prep_kernel<<<static_cast<unsigned>(std::max<int64_t>(prep_blocks, 1)), 256, 0, stream>>>(
      static_cast<const __nv_bfloat16*>(out), static_cast<const __nv_bfloat16*>(dout), rows, delta, dq, seq_len, batch,
      num_kv_heads, unit_start, counter);
  mbe_status st = launch_status("bwd_prep_kernel");
  if (st != MBE_OK) return st;
  Params p;
  p.seq_len = seq_len;
  p.cu = cu_seqlens;
  p.mask = mask;
  p.lse = lse;
  p.delta = delta;
  p.unit_start = unit_start;
  p.counter = counter;
  p.unit_nq = reinterpret_cast<int*>(ws + L.nq);
  p.unit_order = reinterpret_cast<int*>(ws + L.order);
  p.unit_bits = reinterpret_cast<uint32_t*>(ws + L.bits);
  p.max_units = static_cast<int>(L.max_units);
  p.dk = dk;
  p.dv = dv;
  p.mask_rows = mask_rows;
  p.mask_words = mask_words;
  p.block_log2 = 0;
  while ((1 << p.block_log2) < block_size) ++p.block_log2;
  p.batch = batch;
  p.total_tokens = total_tokens;
  p.Hq = num_q_heads;
  p.Hkv = num_kv_heads;
  p.G = G;
  p.lgG = 0;
  while ((1 << p.lgG) < G) ++p.lgG;
  p.scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt(static_cast<float>(kD));
  p.scale_log2 = p.scale * kLog2e;
  const int64_t launch_units =
      std::min<int64_t>(L.max_units, static_cast<int64_t>(num_kv_heads) * batch * ((max_seq_len + kTile - 1) / kTile));
  bwd_plan_kernel<<<static_cast<unsigned>(std::max<int64_t>((launch_units + 7) / 8, 1)), 256, 0, stream>>>(p);
  st = launch_status("bwd_plan_kernel");
  if (st != MBE_OK) return st;
  bwd_kernel<<<ds->num_sms, kThreads, kSmemBytes, stream>>>(tq, tdo, tk, tv, tdq, p);
  return launch_status("bwd_kernel");
}

extern "C" mbe_status mbe_sft_block_mask(const int32_t* n_prompt_blocks, const int32_t* n_blocks, int32_t K,
                                         int32_t batch, int32_t mask_rows, int32_t mask_words, uint32_t* mask,
                                         cudaStream_t stream) {
  using namespace mbe;
  if (K < 1 || batch < 0 || mask_rows < 1 || mask_words < 1 || static_cast<int64_t>(mask_words) * 32 < mask_rows)
    return MBE_ERR_INVALID_ARG;
  if (batch == 0) return MBE_OK;
  if (!n_prompt_blocks || !n_blocks || !mask) return MBE_ERR_INVALID_ARG;
  if (batch > 65535) return MBE_ERR_UNSUPPORTED;
  sft_mask_kernel<<<dim3(static_cast<unsigned>(mask_rows), static_cast<unsigned>(batch)), 128, 0, stream>>>(
      n_prompt_blocks, n_blocks, K, mask_rows, mask_words, mask);
  return launch_status("sft_mask_kernel");
}
