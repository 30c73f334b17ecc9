// Multi-Block Edit SFT attention support (Sec. 3): the cross-block attention
// mask and the backward of attention under a block mask. The forward under the
// mask is mbe_block_mask_attention (attention.cu).
//
// sft_mask_kernel: one CTA per (mask row, sequence); thread w builds 32-bit
// word w of the row from the link rules, so a row of nb blocks costs nb bits.
//
// bwd_prep_kernel: delta = rowsum(dO o O) per (token, head); the unit offsets
// of both work lists. bwd_plan_kernel (once per list): each unit's visible
// tiles of the other kind, and the units ordered longest first.
//
// dkdv_kernel (persistent, one CTA per SM, 384 threads): a work unit is
// (sequence, KV head g, 128-key tile); K and V stay in shared memory while the
// unit walks the 128-row query tiles (packed rows token * G + head of the heads
// of g) that see any of its key blocks. Per query tile t:
//   warp 0      TMA: Q_t and dO_t into a 2-stage ring (K, V once per unit);
//               the tile's column data (lse, delta, which query blocks see
//               each key block of the unit) into shared memory
//   warp 1      MMA: S^T = K Q_t^T and dP^T = V dO_t^T (SS, into TMEM), then
//               dV += P^T dO_t and dK += dS^T Q_t (TS: P^T and dS^T from
//               TMEM). S^T of tile t + 1 is issued as soon as the
//               compute warps have read S^T of tile t, so it runs under their
//               elementwise work.
//   warps 4-11  two warps per TMEM lane quadrant, splitting columns 0-63 /
//               64-127; thread = key row: P^T = exp(S^T * scale - lse),
//               masked; dS^T = P^T o (dP^T - delta); both as bf16 over the
//               warp's dP^T columns (A of dV and dK); at the unit's end dK *
//               scale and dV stored (fp32).
// dq_kernel (same shape): a work unit is (sequence, KV head g, 128-row query
// tile); Q and dO stay in shared memory while the unit walks the visible key
// tiles (K and V in a 2-stage ring). MMA: S = Q K_j^T into one of two TMEM
// buffers, dP = dO V_j^T, dQ += dS K_j (TS: dS from TMEM, over the S buffer);
// thread = query row: P = exp(S * scale - lse), dS = P o (dP - delta); at the
// unit's end dQ * scale stored. dQ needs no reduction across CTAs.
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
constexpr int kMaxWords = 16;                // tile bitmask of a unit (<= 512 tiles)
constexpr int kMaxKeyBlocks = 16;            // key blocks of a 128-key tile (block size >= 8)
constexpr uint32_t kHalf = 128 * 128;        // a 64-column half of a 128-row bf16 tile (16 KB)
constexpr uint32_t kTileBytes = 2 * kHalf;   // 32 KB
// shared memory of both kernels: two tiles held for the whole unit, a 3-stage
// ring of the streamed tile the step's first MMA reads (Q, or K) and a 2-stage
// ring of the other streamed tile (dO, or V)
constexpr uint32_t kFix0 = 0, kFix1 = kTileBytes, kRingA = 2 * kTileBytes, kRingB = kRingA + 3 * kTileBytes;
constexpr uint32_t kSmemBytes = kRingB + 2 * kTileBytes + 1024;  // + 1024-byte alignment slack
constexpr float kLog2e = 1.4426950408889634f;

// Work units of one kind: (sequence, KV head g, tile t), t fastest.
struct Plan {
  const int32_t* unit_start;  // [batch + 1]: first unit of each sequence
  int* counter;               // [0] work queue, [1] plan blocks done, [2] units planned
  int* nq;                    // [max_units]: visible tiles of the other kind per unit
  int* order;                 // [max_units]: units by descending nq
  uint32_t* bits;             // [max_units][kMaxWords]: the visible tiles
};

struct Params {
  const int32_t* seq_len;
  const int32_t* cu;
  const uint32_t* mask;
  const float* lse;
  const float* delta;
  Plan kv;  // key-tile units: dK, dV (dkdv_kernel)
  Plan qt;  // query-tile units: dQ (dq_kernel)
  int max_units;
  float* dq;
  float* dk;
  float* dv;
  int mask_rows, mask_words, block_log2;
  int batch, total_tokens, Hq, Hkv, G, lgG;
  float scale, scale_log2;
  uint64_t wait_ns;  // limit of the ordinary mbarrier waits
};

struct Unit {
  int32_t seq, g, t, len, cu;
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

__device__ __forceinline__ int key_tiles(int len) { return (len + kTile - 1) / kTile; }
__device__ __forceinline__ int query_tiles(const Params& p, int len) { return ((len << p.lgG) + kTile - 1) / kTile; }

// Does any query block of query tile i see a key block of key tile kt?
__device__ __forceinline__ bool pair_visible(const Params& p, int seq, int len, int i, int kt) {
  const int q0 = (i * kTile) >> p.lgG, q1 = min(len, ((i + 1) * kTile) >> p.lgG) - 1;
  const int k0 = kt * kTile, k1 = min(len, k0 + kTile) - 1;
  if (q1 < q0 || k1 < k0) return false;
  for (int qb = q0 >> p.block_log2; qb <= (q1 >> p.block_log2); ++qb)
    for (int kb = k0 >> p.block_log2; kb <= (k1 >> p.block_log2); ++kb)
      if (mask_bit(p, seq, qb, kb)) return true;
  return false;
}

__device__ __forceinline__ int next_bit(const volatile uint32_t* bits, int i) {
  for (int b = i + 1; b < kMaxWords * 32;) {
    const uint32_t w = bits[b >> 5] >> (b & 31);
    if (w) return b + __ffs(w) - 1;
    b = (b & ~31) + 32;
  }
  return -1;
}

// Work unit u of a plan; kKeys: units are key tiles, else query tiles.
template <bool kKeys>
__device__ __forceinline__ Unit decode_unit(const Params& p, const Plan& pl, int u) {
  int lo = 0, hi = p.batch - 1;  // the sequence whose unit range holds u
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (pl.unit_start[mid] <= u) lo = mid; else hi = mid - 1;
  }
  const int len = p.seq_len[lo];
  const int tiles = max(kKeys ? key_tiles(len) : query_tiles(p, len), 1);
  const int r = u - pl.unit_start[lo];
  return Unit{lo, r / tiles, r % tiles, len, p.cu[lo]};
}

// First and (capped) count of the query blocks of query tile i.
__device__ __forceinline__ int qblock0(const Params& p, int i) { return ((i * kTile) >> p.lgG) >> p.block_log2; }
__device__ __forceinline__ int qblock_count(const Params& p, const Unit& u, int i) {
  const int last = min(u.len - 1, ((i + 1) * kTile - 1) >> p.lgG) >> p.block_log2;
  return min(32, last - qblock0(p, i) + 1);
}

// Fetches the next unit of a plan's queue into ring slot `slot` (whole warp).
template <bool kKeys>
__device__ __forceinline__ Unit fetch_unit(const Params& p, const Plan& pl, int n_units, int lane, Unit* ring,
                                           uint32_t (*ring_bits)[kMaxWords], int slot, bool& done) {
  int uidx = 0;
  if (lane == 0) uidx = atomicAdd(pl.counter, 1);
  uidx = __shfl_sync(0xffffffffu, uidx, 0);
  done = uidx >= n_units;
  Unit un{-1, 0, 0, 0, 0};
  if (!done) {
    const int u = pl.order[uidx];  // longest units first
    un = decode_unit<kKeys>(p, pl, u);
    if (lane < kMaxWords) ring_bits[slot][lane] = pl.bits[static_cast<int64_t>(u) * kMaxWords + lane];
  }
  __syncwarp();
  if (lane == 0) ring[slot] = un;
  return un;
}

__device__ __forceinline__ int popc_bits(const volatile uint32_t* bits) {
  int n = 0;
  for (int w = 0; w < kMaxWords; ++w) n += __popc(bits[w]);
  return n;
}

// ============================================================================
// dkdv_kernel (key-tile units). TMEM: dK, dV, S^T, dP^T / P^T (128 columns each).
// ============================================================================
constexpr uint32_t kTmDK = 0, kTmDV = 128, kTmS = 256, kTmDP = 384, kTmCols = 512;

struct KvBars {
  uint64_t u_full[2], u_empty[2], q_full[3], q_empty[3], do_full[2], do_empty[2], kv_full, kv_empty, col_full,
      col_empty, s_full, pt_full, dp_full, ds_full, acc_full, acc_empty, mma_done;
};

__global__ void __launch_bounds__(kThreads, 1)
    dkdv_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_do,
                const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v, const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) KvBars bars;
  __shared__ Unit ring[2];
  __shared__ uint32_t ring_bits[2][kMaxWords];
  // column data of the current query tile, written by the producer warp
  __shared__ __align__(16) float col_nlse[kTile];    // -lse in log2 units; -inf past the sequence (P = 0)
  __shared__ __align__(16) float col_ndelta[kTile];  // -rowsum(dO o O)
  __shared__ uint32_t col_kvis[kMaxKeyBlocks];      // per key block of the unit: bit b = query block qb0 + b sees it
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  volatile int* abort_flag = &abort_s;
  const uint64_t wait_ns = p.wait_ns;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  auto bar = [](uint64_t& b) { return smem_u32(&b); };
  const int n_units = p.kv.counter[2];
  constexpr uint32_t kK = kFix0, kV = kFix1;

  if (tid == 0) {
    abort_s = 0;
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(bars.u_full[i]), 1);
      mbar_init(bar(bars.u_empty[i]), 9);  // MMA issuer + 8 compute warps
      mbar_init(bar(bars.do_full[i]), 1);
      mbar_init(bar(bars.do_empty[i]), 1);
    }
    for (int i = 0; i < 3; ++i) {
      mbar_init(bar(bars.q_full[i]), 1);
      mbar_init(bar(bars.q_empty[i]), 1);
    }
    mbar_init(bar(bars.kv_full), 1);
    mbar_init(bar(bars.kv_empty), 1);
    mbar_init(bar(bars.col_full), 1);
    mbar_init(bar(bars.col_empty), 8);
    mbar_init(bar(bars.s_full), 1);
    mbar_init(bar(bars.pt_full), 8);
    mbar_init(bar(bars.dp_full), 1);
    mbar_init(bar(bars.ds_full), 8);
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
    uint32_t u_it = 0, kv_loads = 0, q_loads = 0, do_loads = 0, cols = 0;
    bool ok = true;
    for (;;) {
      const int slot = u_it & 1;
      if (u_it >= 2) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.u_empty[slot]), ((u_it >> 1) - 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
      }
      bool done;
      const Unit un = fetch_unit<true>(p, p.kv, n_units, lane, ring, ring_bits, slot, done);
      if (lane == 0) mbar_arrive(bar(bars.u_full[slot]));
      ++u_it;
      if (done) break;
      const volatile uint32_t* bits = ring_bits[slot];
      if (popc_bits(bits) == 0) continue;
      if (kv_loads >= 1) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.kv_empty), (kv_loads - 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(bar(bars.kv_full), 2 * kTileBytes);
        for (int h = 0; h < 2; ++h) {
          tma_load_3d(sbase + kK + h * kHalf, &tm_k, bar(bars.kv_full), h * 64, un.g, un.cu + un.t * kTile);
          tma_load_3d(sbase + kV + h * kHalf, &tm_v, bar(bars.kv_full), h * 64, un.g, un.cu + un.t * kTile);
        }
      }
      ++kv_loads;
      const int kb_first = (un.t * kTile) >> p.block_log2;
      const int kb_last = (min(un.len, (un.t + 1) * kTile) - 1) >> p.block_log2;
      for (int i = next_bit(bits, -1); i >= 0 && ok; i = next_bit(bits, i)) {
        const int tok = un.cu + ((i * kTile) >> p.lgG);
        const uint32_t sq = q_loads % 3, sd = do_loads & 1;
        if (q_loads >= 3) {
          ok = __all_sync(kAll, mbar_wait(bar(bars.q_empty[sq]), ((q_loads / 3) - 1) & 1, abort_flag, wait_ns));
          if (!ok) break;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(bar(bars.q_full[sq]), kTileBytes);
          for (int h = 0; h < 2; ++h)
            tma_load_3d(sbase + kRingA + sq * kTileBytes + h * kHalf, &tm_q, bar(bars.q_full[sq]), h * 64,
                        un.g * p.G, tok);
        }
        ++q_loads;
        if (do_loads >= 2) {
          ok = __all_sync(kAll, mbar_wait(bar(bars.do_empty[sd]), ((do_loads >> 1) - 1) & 1, abort_flag, wait_ns));
          if (!ok) break;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(bar(bars.do_full[sd]), kTileBytes);
          for (int h = 0; h < 2; ++h)
            tma_load_3d(sbase + kRingB + sd * kTileBytes + h * kHalf, &tm_do, bar(bars.do_full[sd]), h * 64,
                        un.g * p.G, tok);
        }
        ++do_loads;
        // column data of tile i, fetched before waiting for the compute warps to
        // finish with the previous tile's
        float lse_r[4], dl_r[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int R = i * kTile + lane + 32 * e;
          const int tok = R >> p.lgG, head = un.g * p.G + (R & (p.G - 1));
          const bool qv = tok < un.len;
          const int64_t row = (static_cast<int64_t>(un.cu) + tok) * p.Hq + head;
          lse_r[e] = qv ? -p.lse[row] * kLog2e : __int_as_float(0xff800000);
          dl_r[e] = qv ? -p.delta[row] : 0.f;
        }
        const int qb0 = qblock0(p, i), nqb = qblock_count(p, un, i);
        uint32_t kvis = 0;
        if (lane < kMaxKeyBlocks && kb_first + lane <= kb_last)
          for (int b = 0; b < nqb; ++b)
            if (mask_bit(p, un.seq, qb0 + b, kb_first + lane)) kvis |= 1u << b;
        if (cols >= 1) {
          ok = __all_sync(kAll, mbar_wait(bar(bars.col_empty), (cols - 1) & 1, abort_flag, wait_ns));
          if (!ok) break;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          col_nlse[lane + 32 * e] = lse_r[e];
          col_ndelta[lane + 32 * e] = dl_r[e];
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
    }
    // The copies already issued land before the CTA can exit, also when another
    // role aborted after this loop ended (they return at once otherwise).
    if (lane == 0) {
      const int zero = 0;
      if (kv_loads >= 1) mbar_wait(bar(bars.kv_full), (kv_loads - 1) & 1, &zero);
      for (uint32_t n = (q_loads >= 3 ? q_loads - 3 : 0); n < q_loads; ++n)
        mbar_wait(bar(bars.q_full[n % 3]), (n / 3) & 1, &zero);
      for (uint32_t n = (do_loads >= 2 ? do_loads - 2 : 0); n < do_loads; ++n)
        mbar_wait(bar(bars.do_full[n & 1]), (n >> 1) & 1, &zero);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_kk = idesc_bf16_f32(kTile, kTile, false, false);  // S^T, dP^T
      constexpr uint32_t idesc_tb = idesc_bf16_f32(kTile, kD, false, true);      // dV, dK: MN-major B
      uint32_t u_it = 0, units = 0, tiles = 0;
      bool ok = true;
      // S^T = K Q_t^T into the S region (issued after dV of tile t - 1, the last reader there)
      auto issue_s = [&](uint32_t t) {
        if (!mbar_wait(bar(bars.q_full[t % 3]), (t / 3) & 1, abort_flag, wait_ns)) return false;
        tc_fence_after();
        const uint32_t qa = sbase + kRingA + (t % 3) * kTileBytes;
        const uint64_t kd = sdesc_sw128(sbase + kK, 16, 1024), qd = sdesc_sw128(qa, 16, 1024);
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint32_t off16 = (h * kHalf + k * 32) >> 4;
            umma_ss(tmem + kTmS, desc_add(kd, off16), desc_add(qd, off16), idesc_kk, (h | k) ? 1u : 0u);
          }
        umma_commit(bar(bars.s_full));
        return true;
      };
      // dP^T = V dO_t^T into the dP region (issued after dK of tile t - 1, the last reader there)
      auto issue_dp = [&](uint32_t t) {
        if (!mbar_wait(bar(bars.do_full[t & 1]), (t >> 1) & 1, abort_flag, wait_ns)) return false;
        tc_fence_after();
        const uint32_t da = sbase + kRingB + (t & 1) * kTileBytes;
        const uint64_t vd = sdesc_sw128(sbase + kV, 16, 1024), dd = sdesc_sw128(da, 16, 1024);
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint32_t off16 = (h * kHalf + k * 32) >> 4;
            umma_ss(tmem + kTmDP, desc_add(vd, off16), desc_add(dd, off16), idesc_kk, (h | k) ? 1u : 0u);
          }
        umma_commit(bar(bars.dp_full));
        return true;
      };
      for (;;) {
        const int slot = u_it & 1;
        if (!mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag, wait_ns)) { ok = false; break; }
        const Unit un = ring[slot];
        const int n_q = popc_bits(ring_bits[slot]);
        mbar_arrive(bar(bars.u_empty[slot]));
        ++u_it;
        if (un.seq < 0) break;
        if (n_q == 0) continue;
        if (!mbar_wait(bar(bars.kv_full), units & 1, abort_flag, wait_ns)) { ok = false; break; }
        if (!issue_s(tiles) || !issue_dp(tiles)) { ok = false; break; }
        for (int j = 0; j < n_q; ++j) {
          const uint32_t t = tiles + j;
          const uint32_t qa = sbase + kRingA + (t % 3) * kTileBytes, da = sbase + kRingB + (t & 1) * kTileBytes;
          // dV as soon as P^T is in TMEM (over S^T), then the next tile's S^T; both run
          // while the compute warps form dS^T
          if (!mbar_wait(bar(bars.pt_full), t & 1, abort_flag, wait_ns)) { ok = false; break; }
          if (j == 0 && units >= 1 && !mbar_wait(bar(bars.acc_empty), (units - 1) & 1, abort_flag, wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t dod = sdesc_sw128(da, kHalf, 1024);
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk)
            // P^T of query columns 64 h .. 64 h + 63 sits packed at S region columns 64 h .. 64 h + 31
            umma_ts(tmem + kTmDV, tmem + kTmS + (kk >> 2) * 64 + (kk & 3) * 8, desc_add(dod, (kk * 16 * 128) >> 4),
                    idesc_tb, (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit(bar(bars.do_empty[t & 1]));
          if (j + 1 < n_q && !issue_s(t + 1)) { ok = false; break; }
          // dK once dS^T is in TMEM (over dP^T), then the next tile's dP^T
          if (!mbar_wait(bar(bars.ds_full), t & 1, abort_flag, wait_ns)) { ok = false; break; }
          tc_fence_after();
          const uint64_t qtd = sdesc_sw128(qa, kHalf, 1024);
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk)
            umma_ts(tmem + kTmDK, tmem + kTmDP + (kk >> 2) * 64 + (kk & 3) * 8, desc_add(qtd, (kk * 16 * 128) >> 4),
                    idesc_tb, (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit(bar(bars.q_empty[t % 3]));
          if (j + 1 < n_q && !issue_dp(t + 1)) { ok = false; break; }
        }
        if (!ok) break;
        tiles += n_q;
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
    const int r = quad * 32 + lane;  // TMEM lane = key row
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const int sh = p.lgG + p.block_log2;  // packed row -> query block
    uint32_t u_it = 0, units = 0, tiles = 0;
    bool ok = true;
    for (;;) {
      const int slot = u_it & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag, wait_ns));
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
      const int n_q = popc_bits(bits);
      const int key = un.t * kTile + r;
      const bool key_ok = key < un.len;
      const int64_t kv_row = (static_cast<int64_t>(un.cu) + key) * p.Hkv + un.g;
      if (n_q == 0) {  // no query sees these keys: zero gradients (dK by one half, dV by the other)
        release();
        float* dst = (hf == 0 ? p.dk : p.dv) + kv_row * kD;
        if (key_ok)
          for (int d = 0; d < kD; d += 4) *reinterpret_cast<float4*>(dst + d) = make_float4(0.f, 0.f, 0.f, 0.f);
        continue;
      }
      const int kb_rel = (key >> p.block_log2) - ((un.t * kTile) >> p.block_log2);
      for (int i = next_bit(bits, -1); i >= 0; i = next_bit(bits, i), ++tiles) {
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.col_full), tiles & 1, abort_flag, wait_ns));
        if (!ok) break;
        const int qb0 = qblock0(p, i), nqb = qblock_count(p, un, i);
        const uint32_t all = nqb >= 32 ? 0xFFFFFFFFu : ((1u << nqb) - 1u);
        // query blocks of this tile that see this key row's block
        const uint32_t qvis = key_ok ? (col_kvis[kb_rel] & all) : 0u;
        // TMEM loads are warp-wide: the warp skips them only if no lane needs them
        const bool any_vis = __any_sync(0xffffffffu, qvis != 0u);
        const bool every = __all_sync(0xffffffffu, qvis == all);
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.s_full), tiles & 1, abort_flag, wait_ns));
        if (!ok) break;
        tc_fence_after();
        uint32_t sv[64];
        if (any_vis) tmem_ld64(t_lane + kTmS + 64 * hf, sv);
        // P^T of this warp's 64 columns, packed to bf16 pairs; a query block spans at
        // least 8 packed rows, so visibility is decided per group of 8 columns
        uint32_t pw[32];
        if (!any_vis) {
#pragma unroll
          for (int m = 0; m < 32; ++m) pw[m] = 0u;
        } else {
          const float2 sc2 = make_float2(p.scale_log2, p.scale_log2);
#pragma unroll
          for (int g8 = 0; g8 < 8; ++g8) {
            const int col = 64 * hf + 8 * g8;
            const float4 la = *reinterpret_cast<const float4*>(&col_nlse[col]);
            const float4 lb = *reinterpret_cast<const float4*>(&col_nlse[col + 4]);
            const float* sg = reinterpret_cast<const float*>(sv) + 8 * g8;
            const float2 x0 = ffma2(make_float2(sg[0], sg[1]), sc2, make_float2(la.x, la.y));
            const float2 x1 = ffma2(make_float2(sg[2], sg[3]), sc2, make_float2(la.z, la.w));
            const float2 x2 = ffma2(make_float2(sg[4], sg[5]), sc2, make_float2(lb.x, lb.y));
            const float2 x3 = ffma2(make_float2(sg[6], sg[7]), sc2, make_float2(lb.z, lb.w));
            const uint32_t keep =
                (every || ((qvis >> (((i * kTile + col) >> sh) - qb0)) & 1u)) ? 0xFFFFFFFFu : 0u;
            pw[4 * g8] = pack_bf16x2(ex2f(x0.x), ex2f(x0.y)) & keep;
            pw[4 * g8 + 1] = pack_bf16x2(ex2f(x1.x), ex2f(x1.y)) & keep;
            pw[4 * g8 + 2] = pack_bf16x2(ex2f(x2.x), ex2f(x2.y)) & keep;
            pw[4 * g8 + 3] = pack_bf16x2(ex2f(x3.x), ex2f(x3.y)) & keep;
          }
        }
        // P^T over the S^T columns this warp has read (A of dV)
        tmem_st32(t_lane + kTmS + 64 * hf, pw);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.pt_full));
        // dP^T of this tile
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.dp_full), tiles & 1, abort_flag, wait_ns));
        if (!ok) break;
        tc_fence_after();
        // dS^T = P^T o (dP^T - delta), packed to bf16 pairs
        uint32_t dsa[32];
        uint32_t dvv[64];
        if (any_vis) tmem_ld64(t_lane + kTmDP + 64 * hf, dvv);
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          uint32_t* dsw = dsa + 16 * c;
          if (!any_vis) {
#pragma unroll
            for (int m = 0; m < 16; ++m) dsw[m] = 0u;
          } else {
            const uint32_t* dv = dvv + 32 * c;
#pragma unroll
            for (int jj = 0; jj < 32; jj += 4) {
              const int col = 64 * hf + 32 * c + jj;
              const float4 d4 = *reinterpret_cast<const float4*>(&col_ndelta[col]);
              const uint32_t pa = pw[16 * c + jj / 2], pb = pw[16 * c + jj / 2 + 1];
              const float2 t0 = fadd2(make_float2(__uint_as_float(dv[jj]), __uint_as_float(dv[jj + 1])),
                                      make_float2(d4.x, d4.y));
              const float2 t1 = fadd2(make_float2(__uint_as_float(dv[jj + 2]), __uint_as_float(dv[jj + 3])),
                                      make_float2(d4.z, d4.w));
              const float2 s0 = fmul2(make_float2(__uint_as_float(pa << 16), __uint_as_float(pa & 0xFFFF0000u)), t0);
              const float2 s1 = fmul2(make_float2(__uint_as_float(pb << 16), __uint_as_float(pb & 0xFFFF0000u)), t1);
              dsw[jj / 2] = pack_bf16x2(s0.x, s0.y);
              dsw[jj / 2 + 1] = pack_bf16x2(s1.x, s1.y);
            }
          }
        }
        // dS^T over the dP^T columns this warp has read (A of dK)
        tmem_st32(t_lane + kTmDP + 64 * hf, dsa);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(bar(bars.ds_full));
          mbar_arrive(bar(bars.col_empty));
        }
      }
      if (!ok) break;
      release();
      // dK (first half of the pair) and dV (second half) of the unit's keys: thread = key row
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.acc_full), units & 1, abort_flag, wait_ns));
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

// ============================================================================
// dq_kernel (query-tile units): dQ_i = scale sum over visible key tiles j of
// dS_ij K_j, accumulated in TMEM and stored once. TMEM: S (two buffers), dP, dQ.
// ============================================================================
constexpr uint32_t kTmQS = 0, kTmQDP = 256, kTmQDQ = 384;

struct QBars {
  uint64_t u_full[2], u_empty[2], qd_full, qd_empty, k_full[3], k_empty[3], v_full[2], v_empty[2], s_full[2],
      dp_full, dp_free, ds_full, acc_full, acc_empty, mma_done;
};

__global__ void __launch_bounds__(kThreads, 1)
    dq_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_do,
              const __grid_constant__ CUtensorMap tm_k, const __grid_constant__ CUtensorMap tm_v, const Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) QBars bars;
  __shared__ Unit ring[2];
  __shared__ uint32_t ring_bits[2][kMaxWords];
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  volatile int* abort_flag = &abort_s;
  const uint64_t wait_ns = p.wait_ns;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  auto bar = [](uint64_t& b) { return smem_u32(&b); };
  const int n_units = p.qt.counter[2];
  constexpr uint32_t kQ = kFix0, kDO = kFix1;

  if (tid == 0) {
    abort_s = 0;
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(bars.u_full[i]), 1);
      mbar_init(bar(bars.u_empty[i]), 9);  // MMA issuer + 8 compute warps
      mbar_init(bar(bars.v_full[i]), 1);
      mbar_init(bar(bars.v_empty[i]), 1);
      mbar_init(bar(bars.s_full[i]), 1);
    }
    for (int i = 0; i < 3; ++i) {
      mbar_init(bar(bars.k_full[i]), 1);
      mbar_init(bar(bars.k_empty[i]), 1);
    }
    mbar_init(bar(bars.qd_full), 1);
    mbar_init(bar(bars.qd_empty), 1);
    mbar_init(bar(bars.dp_full), 1);
    mbar_init(bar(bars.dp_free), 8);
    mbar_init(bar(bars.ds_full), 8);
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
    uint32_t u_it = 0, qd_loads = 0, k_loads = 0, v_loads = 0;
    bool ok = true;
    for (;;) {
      const int slot = u_it & 1;
      if (u_it >= 2) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.u_empty[slot]), ((u_it >> 1) - 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
      }
      bool done;
      const Unit un = fetch_unit<false>(p, p.qt, n_units, lane, ring, ring_bits, slot, done);
      if (lane == 0) mbar_arrive(bar(bars.u_full[slot]));
      ++u_it;
      if (done) break;
      const volatile uint32_t* bits = ring_bits[slot];
      if (popc_bits(bits) == 0) continue;
      if (qd_loads >= 1) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.qd_empty), (qd_loads - 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
      }
      if (lane == 0) {
        mbar_arrive_expect_tx(bar(bars.qd_full), 2 * kTileBytes);
        const int tok = un.cu + ((un.t * kTile) >> p.lgG);
        for (int h = 0; h < 2; ++h) {
          tma_load_3d(sbase + kQ + h * kHalf, &tm_q, bar(bars.qd_full), h * 64, un.g * p.G, tok);
          tma_load_3d(sbase + kDO + h * kHalf, &tm_do, bar(bars.qd_full), h * 64, un.g * p.G, tok);
        }
      }
      ++qd_loads;
      for (int j = next_bit(bits, -1); j >= 0 && ok; j = next_bit(bits, j)) {
        const uint32_t sk = k_loads % 3, sv = v_loads & 1;
        if (k_loads >= 3) {
          ok = __all_sync(kAll, mbar_wait(bar(bars.k_empty[sk]), ((k_loads / 3) - 1) & 1, abort_flag, wait_ns));
          if (!ok) break;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(bar(bars.k_full[sk]), kTileBytes);
          for (int h = 0; h < 2; ++h)
            tma_load_3d(sbase + kRingA + sk * kTileBytes + h * kHalf, &tm_k, bar(bars.k_full[sk]), h * 64, un.g,
                        un.cu + j * kTile);
        }
        ++k_loads;
        if (v_loads >= 2) {
          ok = __all_sync(kAll, mbar_wait(bar(bars.v_empty[sv]), ((v_loads >> 1) - 1) & 1, abort_flag, wait_ns));
          if (!ok) break;
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(bar(bars.v_full[sv]), kTileBytes);
          for (int h = 0; h < 2; ++h)
            tma_load_3d(sbase + kRingB + sv * kTileBytes + h * kHalf, &tm_v, bar(bars.v_full[sv]), h * 64, un.g,
                        un.cu + j * kTile);
        }
        ++v_loads;
      }
      if (!ok) break;
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
    }
    // The copies already issued land before the CTA can exit (see dkdv_kernel).
    if (lane == 0) {
      const int zero = 0;
      if (qd_loads >= 1) mbar_wait(bar(bars.qd_full), (qd_loads - 1) & 1, &zero);
      for (uint32_t n = (k_loads >= 3 ? k_loads - 3 : 0); n < k_loads; ++n)
        mbar_wait(bar(bars.k_full[n % 3]), (n / 3) & 1, &zero);
      for (uint32_t n = (v_loads >= 2 ? v_loads - 2 : 0); n < v_loads; ++n)
        mbar_wait(bar(bars.v_full[n & 1]), (n >> 1) & 1, &zero);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_kk = idesc_bf16_f32(kTile, kTile, false, false);  // S, dP
      constexpr uint32_t idesc_dq = idesc_bf16_f32(kTile, kD, false, true);      // dQ: dS from TMEM, MN-major K
      uint32_t u_it = 0, units = 0, tiles = 0;
      bool ok = true;
      // S = Q K_t^T into S buffer t & 1 (issued after dQ of tile t - 2, which read dS there)
      auto issue_s = [&](uint32_t t) {
        const uint32_t b = t & 1;
        if (!mbar_wait(bar(bars.k_full[t % 3]), (t / 3) & 1, abort_flag, wait_ns)) return false;
        tc_fence_after();
        const uint32_t ka = sbase + kRingA + (t % 3) * kTileBytes;
        const uint64_t qd = sdesc_sw128(sbase + kQ, 16, 1024), kd = sdesc_sw128(ka, 16, 1024);
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint32_t off16 = (h * kHalf + k * 32) >> 4;
            umma_ss(tmem + kTmQS + 128 * b, desc_add(qd, off16), desc_add(kd, off16), idesc_kk, (h | k) ? 1u : 0u);
          }
        umma_commit(bar(bars.s_full[b]));
        return true;
      };
      // dP = dO V_t^T once the compute warps have read dP of tile t - 1
      auto issue_dp = [&](uint32_t t) {
        if (t >= 1 && !mbar_wait(bar(bars.dp_free), (t - 1) & 1, abort_flag, wait_ns)) return false;
        if (!mbar_wait(bar(bars.v_full[t & 1]), (t >> 1) & 1, abort_flag, wait_ns)) return false;
        tc_fence_after();
        const uint32_t va = sbase + kRingB + (t & 1) * kTileBytes;
        const uint64_t dod = sdesc_sw128(sbase + kDO, 16, 1024), vd = sdesc_sw128(va, 16, 1024);
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const uint32_t off16 = (h * kHalf + k * 32) >> 4;
            umma_ss(tmem + kTmQDP, desc_add(dod, off16), desc_add(vd, off16), idesc_kk, (h | k) ? 1u : 0u);
          }
        umma_commit(bar(bars.dp_full));
        umma_commit(bar(bars.v_empty[t & 1]));
        return true;
      };
      for (;;) {
        const int slot = u_it & 1;
        if (!mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag, wait_ns)) { ok = false; break; }
        const Unit un = ring[slot];
        const int n_k = popc_bits(ring_bits[slot]);
        mbar_arrive(bar(bars.u_empty[slot]));
        ++u_it;
        if (un.seq < 0) break;
        if (n_k == 0) continue;
        if (!mbar_wait(bar(bars.qd_full), units & 1, abort_flag, wait_ns)) { ok = false; break; }
        // S two tiles ahead: it runs while the compute warps form dS of the tile before
        if (!issue_s(tiles) || !issue_dp(tiles) || (n_k >= 2 && !issue_s(tiles + 1))) { ok = false; break; }
        for (int j = 0; j < n_k; ++j) {
          const uint32_t t = tiles + j;
          if (!mbar_wait(bar(bars.ds_full), t & 1, abort_flag, wait_ns)) { ok = false; break; }
          // the next tile's dP first: the compute warps wait for it, and its region was
          // read before ds_full
          if (j + 1 < n_k && !issue_dp(t + 1)) { ok = false; break; }
          if (j == 0 && units >= 1 && !mbar_wait(bar(bars.acc_empty), (units - 1) & 1, abort_flag, wait_ns)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t ka = sbase + kRingA + (t % 3) * kTileBytes;
          // dQ += dS K_t: dS of key columns 64 h .. 64 h + 63 sits packed at S buffer columns
          // 64 h .. 64 h + 31 (A from TMEM); K_t [key][d] is an MN-major B
          const uint64_t ktd = sdesc_sw128(ka, kHalf, 1024);
#pragma unroll
          for (int kk = 0; kk < kTile / 16; ++kk)
            umma_ts(tmem + kTmQDQ, tmem + kTmQS + 128 * (t & 1) + (kk >> 2) * 64 + (kk & 3) * 8,
                    desc_add(ktd, (kk * 16 * 128) >> 4), idesc_dq, (j > 0 || kk > 0) ? 1u : 0u);
          umma_commit(bar(bars.k_empty[t % 3]));
          if (j + 2 < n_k && !issue_s(t + 2)) { ok = false; break; }
        }
        if (!ok) break;
        tiles += n_k;
        umma_commit(bar(bars.acc_full));
        umma_commit(bar(bars.qd_empty));
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
    const int hf = (warp - 4) >> 2;  // the pair of warps of a quadrant splits key columns 0-63 / 64-127
    const int r = quad * 32 + lane;  // TMEM lane = query row of the tile
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const int kb_per_tile = max(1, kTile >> p.block_log2);  // key blocks of a key tile (<= 16, one mask word)
    const uint32_t tile_mask = (1u << kb_per_tile) - 1u;
    uint32_t u_it = 0, units = 0, tiles = 0;
    bool ok = true;
    for (;;) {
      const int slot = u_it & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag, wait_ns));
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
      const int n_k = popc_bits(bits);
      // this thread's query row: packed row R of the sequence = token * G + head in group
      const int R = un.t * kTile + r;
      const int tok = R >> p.lgG, head = un.g * p.G + (R & (p.G - 1));
      const bool qv = tok < un.len;
      float* dst = p.dq + ((static_cast<int64_t>(un.cu) + tok) * p.Hq + head) * kD + 64 * hf;
      if (n_k == 0) {  // no key is visible to these rows: dQ = 0
        release();
        if (qv)
          for (int d = 0; d < 64; d += 4) *reinterpret_cast<float4*>(dst + d) = make_float4(0.f, 0.f, 0.f, 0.f);
        continue;
      }
      const int64_t row = (static_cast<int64_t>(un.cu) + tok) * p.Hq + head;
      const float lse2 = qv ? p.lse[row] * kLog2e : __int_as_float(0x7f800000);  // +inf: P = 0
      const float dl = qv ? p.delta[row] : 0.f;
      const int qb = tok >> p.block_log2;
      const bool qb_ok = qv && qb < p.mask_rows;
      const uint32_t* mrow = p.mask + (static_cast<int64_t>(un.seq) * p.mask_rows + (qb_ok ? qb : 0)) * p.mask_words;
      for (int j = next_bit(bits, -1); j >= 0; j = next_bit(bits, j), ++tiles) {
        const uint32_t b = tiles & 1;
        // this row's visible key blocks of key tile j (one mask word holds them all)
        const int kb0 = (j * kTile) >> p.block_log2;
        const uint32_t word = (qb_ok && (kb0 >> 5) < p.mask_words) ? mrow[kb0 >> 5] : 0u;
        const uint32_t kbits = (word >> (kb0 & 31)) & tile_mask;
        const int n_vis = min(kTile, un.len - j * kTile);
        const bool any_vis = __any_sync(0xffffffffu, kbits != 0u);
        const bool every = __all_sync(0xffffffffu, !qv || (kbits == tile_mask && n_vis == kTile));
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.s_full[b]), (tiles >> 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
        tc_fence_after();
        uint32_t sv[64];
        if (any_vis) tmem_ld64(t_lane + kTmQS + 128 * b + 64 * hf, sv);
        // P of this warp's 64 key columns, packed to bf16 pairs; a key block spans at
        // least 8 columns, so visibility is decided per group of 8
        uint32_t pw[32];
        if (!any_vis) {
#pragma unroll
          for (int m = 0; m < 32; ++m) pw[m] = 0u;
        } else {
          const float2 sc2 = make_float2(p.scale_log2, p.scale_log2), nl2 = make_float2(-lse2, -lse2);
#pragma unroll
          for (int g8 = 0; g8 < 8; ++g8) {
            const int c0 = 64 * hf + 8 * g8;
            const float* sg = reinterpret_cast<const float*>(sv) + 8 * g8;
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 x = ffma2(make_float2(sg[2 * e], sg[2 * e + 1]), sc2, nl2);
              w[e] = pack_bf16x2(ex2f(x.x), ex2f(x.y));
            }
            if (!every) {
              const uint32_t keep = ((kbits >> (c0 >> p.block_log2)) & 1u) ? 0xFFFFFFFFu : 0u;
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                // keys past the sequence end share the last key block's bit
                const int c = c0 + 2 * e;
                const uint32_t tail = c >= n_vis ? 0u : (c + 1 >= n_vis ? 0x0000FFFFu : 0xFFFFFFFFu);
                w[e] &= keep & tail;
              }
            }
#pragma unroll
            for (int e = 0; e < 4; ++e) pw[4 * g8 + e] = w[e];
          }
        }
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.dp_full), tiles & 1, abort_flag, wait_ns));
        if (!ok) break;
        tc_fence_after();
        uint32_t dsa[32];
        if (!any_vis) {
#pragma unroll
          for (int m = 0; m < 32; ++m) dsa[m] = 0u;
        } else {
          uint32_t dv[64];
          tmem_ld64(t_lane + kTmQDP + 64 * hf, dv);
          const float2 nd2 = make_float2(-dl, -dl);
#pragma unroll
          for (int jj = 0; jj < 64; jj += 2) {
            const uint32_t pk = pw[jj / 2];
            const float2 t = fadd2(make_float2(__uint_as_float(dv[jj]), __uint_as_float(dv[jj + 1])), nd2);
            const float2 s2 = fmul2(make_float2(__uint_as_float(pk << 16), __uint_as_float(pk & 0xFFFF0000u)), t);
            dsa[jj / 2] = pack_bf16x2(s2.x, s2.y);
          }
        }
        // dS over the S columns this warp has read (A of dQ)
        tmem_st32(t_lane + kTmQS + 128 * b + 64 * hf, dsa);
        tmem_st_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(bar(bars.dp_free));
          mbar_arrive(bar(bars.ds_full));
        }
      }
      if (!ok) break;
      release();
      // dQ * scale of this row, this warp's half of the head dimension
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.acc_full), units & 1, abort_flag, wait_ns));
      if (!ok) break;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        uint32_t a[32];
        tmem_ld32(t_lane + kTmQDQ + 64 * hf + 32 * c, a);
        if (qv)
#pragma unroll
          for (int e = 0; e < 32; e += 4)
            *reinterpret_cast<float4*>(dst + 32 * c + e) =
                make_float4(__uint_as_float(a[e]) * p.scale, __uint_as_float(a[e + 1]) * p.scale,
                            __uint_as_float(a[e + 2]) * p.scale, __uint_as_float(a[e + 3]) * p.scale);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(bars.acc_empty));
      ++units;
    }
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

// The work lists of both kernels: one warp per unit finds the tiles of the
// other kind that it meets under the mask; the last block to finish orders
// the units by descending count (a counting sort), so the persistent kernels
// take the longest units first.
template <bool kKeys>
__global__ void __launch_bounds__(256) bwd_plan_kernel(const Params p) {
  constexpr int kBins = kMaxWords * 32 + 1;
  __shared__ int hist[kBins];
  __shared__ int last_s;
  const Plan& pl = kKeys ? p.kv : p.qt;
  const int lane = threadIdx.x & 31;
  const int n_all = pl.unit_start[p.batch];
  const int n_units = min(n_all, min(p.max_units, static_cast<int>(gridDim.x) * 8));
  const int u = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (u < n_units) {
    const Unit un = decode_unit<kKeys>(p, pl, u);
    const int n_other = kKeys ? query_tiles(p, un.len) : key_tiles(un.len);
    int n = 0;
    for (int w = 0; w < kMaxWords; ++w) {
      const int o = 32 * w + lane;
      const bool vis = o < n_other && (kKeys ? pair_visible(p, un.seq, un.len, o, un.t)
                                             : pair_visible(p, un.seq, un.len, un.t, o));
      const uint32_t word = __ballot_sync(0xffffffffu, vis);
      if (lane == 0) pl.bits[static_cast<int64_t>(u) * kMaxWords + w] = word;
      n += __popc(word);
    }
    if (lane == 0) pl.nq[u] = n;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    last_s = atomicAdd(&pl.counter[1], 1) == static_cast<int>(gridDim.x) - 1;
  }
  __syncthreads();
  if (!last_s) return;
  __threadfence();
  for (int b = threadIdx.x; b < kBins; b += blockDim.x) hist[b] = 0;
  __syncthreads();
  for (int v = threadIdx.x; v < n_units; v += blockDim.x) atomicAdd(&hist[__ldcg(&pl.nq[v])], 1);
  __syncthreads();
  if (threadIdx.x < 32) {
    // exclusive prefix over the bins taken from the top: lane l owns kPer bins
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
  for (int v = threadIdx.x; v < n_units; v += blockDim.x) pl.order[atomicAdd(&hist[__ldcg(&pl.nq[v])], 1)] = v;
  if (threadIdx.x == 0) {
    pl.counter[2] = n_units;
    if (n_units < n_all) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
  }
}

// delta = rowsum(dO o O) per (token, head) (one warp per row); the unit
// offsets of both plans and their counters set up by block 0.
__global__ void __launch_bounds__(256) bwd_prep_kernel(const __nv_bfloat16* __restrict__ out,
                                                       const __nv_bfloat16* __restrict__ dout, int64_t rows,
                                                       float* __restrict__ delta, const int32_t* __restrict__ seq_len,
                                                       int batch, int Hkv, int lgG, int32_t* kv_start, int32_t* q_start,
                                                       int* kv_counter, int* q_counter) {
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
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    int kv = 0, qt = 0;
    for (int s = 0; s < batch; ++s) {
      kv_start[s] = kv;
      q_start[s] = qt;
      const int len = seq_len[s];
      if (len > 0) {
        kv += Hkv * ((len + kTile - 1) / kTile);
        qt += Hkv * static_cast<int>(((static_cast<int64_t>(len) << lgG) + kTile - 1) / kTile);
      }
    }
    kv_start[batch] = kv;
    q_start[batch] = qt;
    for (int i = 0; i < 4; ++i) kv_counter[i] = q_counter[i] = 0;
  }
}

// Workspace: work counters and unit offsets of both plans, delta, then each
// plan's units (sized for at most num_q_heads KV heads).
struct WsLayout {
  size_t starts, delta, plan[2][3], total;
  int64_t max_units;
};

inline WsLayout ws_layout(int64_t batch, int64_t total_tokens, int64_t num_q_heads) {
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  WsLayout L;
  L.max_units = std::min<int64_t>(num_q_heads * ((total_tokens + kTile - 1) / kTile + batch), 1 << 30);
  L.starts = 64;  // after two sets of 4 counters
  L.delta = up(L.starts + 2 * static_cast<size_t>(batch + 1) * sizeof(int32_t));
  size_t at = up(L.delta + static_cast<size_t>(total_tokens) * num_q_heads * sizeof(float));
  for (int k = 0; k < 2; ++k) {
    L.plan[k][0] = at;  // nq
    L.plan[k][1] = at = up(at + static_cast<size_t>(L.max_units) * sizeof(int32_t));  // order
    L.plan[k][2] = at = up(at + static_cast<size_t>(L.max_units) * sizeof(int32_t));  // bits
    at = up(at + static_cast<size_t>(L.max_units) * kMaxWords * sizeof(uint32_t));
  }
  L.total = at;
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
      cudaFuncSetAttribute(dkdv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) == cudaSuccess &&
      cudaFuncSetAttribute(dq_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) == cudaSuccess)
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
  if (static_cast<int64_t>(max_seq_len) * G > static_cast<int64_t>(kMaxWords) * 32 * kTile) return MBE_ERR_UNSUPPORTED;
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
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const WsLayout L = ws_layout(batch, total_tokens, num_q_heads);
  int* kv_counter = reinterpret_cast<int*>(ws);
  int* q_counter = reinterpret_cast<int*>(ws + 16);
  int32_t* kv_start = reinterpret_cast<int32_t*>(ws + L.starts);
  int32_t* q_start = kv_start + (batch + 1);
  float* delta = reinterpret_cast<float*>(ws + L.delta);
  int lgG = 0;
  while ((1 << lgG) < G) ++lgG;
  const int64_t rows = static_cast<int64_t>(total_tokens) * num_q_heads;
  const int64_t prep_blocks = std::min<int64_t>((rows + 7) / 8, 8ll * ds->num_sms);
  bwd_prep_kernel<<<static_cast<unsigned>(std::max<int64_t>(prep_blocks, 1)), 256, 0, stream>>>(
      static_cast<const __nv_bfloat16*>(out), static_cast<const __nv_bfloat16*>(dout), rows, delta, seq_len, batch,
      num_kv_heads, lgG, kv_start, q_start, kv_counter, q_counter);
  mbe_status st = launch_status("bwd_prep_kernel");
  if (st != MBE_OK) return st;
  Params p;
  p.seq_len = seq_len;
  p.cu = cu_seqlens;
  p.mask = mask;
  p.lse = lse;
  p.delta = delta;
  p.kv = Plan{kv_start, kv_counter, reinterpret_cast<int*>(ws + L.plan[0][0]), reinterpret_cast<int*>(ws + L.plan[0][1]),
              reinterpret_cast<uint32_t*>(ws + L.plan[0][2])};
  p.qt = Plan{q_start, q_counter, reinterpret_cast<int*>(ws + L.plan[1][0]), reinterpret_cast<int*>(ws + L.plan[1][1]),
              reinterpret_cast<uint32_t*>(ws + L.plan[1][2])};
  p.max_units = static_cast<int>(L.max_units);
  p.dq = dq;
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
  p.lgG = lgG;
  p.scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt(static_cast<float>(kD));
  p.scale_log2 = p.scale * kLog2e;
  p.wait_ns = wait_limit_ns();
  // warps the plans launch: every unit of sequences no longer than max_seq_len
  const int64_t per_seq_kv = (static_cast<int64_t>(max_seq_len) + kTile - 1) / kTile;
  const int64_t per_seq_q = ((static_cast<int64_t>(max_seq_len) << lgG) + kTile - 1) / kTile;
  const int64_t kv_units = std::min<int64_t>(L.max_units, static_cast<int64_t>(num_kv_heads) * batch * per_seq_kv);
  const int64_t q_units = std::min<int64_t>(L.max_units, static_cast<int64_t>(num_kv_heads) * batch * per_seq_q);
  bwd_plan_kernel<true><<<static_cast<unsigned>(std::max<int64_t>((kv_units + 7) / 8, 1)), 256, 0, stream>>>(p);
  st = launch_status("bwd_plan_kernel");
  if (st != MBE_OK) return st;
  bwd_plan_kernel<false><<<static_cast<unsigned>(std::max<int64_t>((q_units + 7) / 8, 1)), 256, 0, stream>>>(p);
  st = launch_status("bwd_plan_kernel");
  if (st != MBE_OK) return st;
  dkdv_kernel<<<ds->num_sms, kThreads, kSmemBytes, stream>>>(tq, tdo, tk, tv, p);
  st = launch_status("dkdv_kernel");
  if (st != MBE_OK) return st;
  dq_kernel<<<ds->num_sms, kThreads, kSmemBytes, stream>>>(tq, tdo, tk, tv, p);
  return launch_status("dq_kernel");
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
