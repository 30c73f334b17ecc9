// Window attention of an MBE editing pass (Eq. 5; Sec. 2.2; Sec. 4.3) on sm_103a.
//
// Three launches on the caller's stream, all sized from host-known bounds so
// the sequence can be captured in a CUDA graph (shapes are device data):
//
//  1. attn_schedule_kernel (1 CTA): reads prefix_len/window_len/mask_mode,
//     cuts every (sequence, KV head, 256-row query slab) into work units of
//     key tiles, splits long units so that there are a few units per SM, and
//     orders them by descending cost (counting sort) for longest-first
//     dynamic scheduling.
//  2. attn_kernel (persistent, one CTA per SM, 12 warps):
//       warp 0      TMA producer: Q slab once per unit, then K/V tiles of 128
//                   keys into a ring of K and V tiles (paged prefix via a 4-D tensor
//                   map with the page id as a coordinate; window via 3-D)
//       warp 1      MMA issuer: S_i = Q_i K^T (SS form) and O_i += P_i V
//                   (TS form, P read from TMEM), tcgen05, accumulators in TMEM
//       warps 4-11  two softmax warpgroups, one per 128-row query tile: TMEM
//                   load of S, exp2 against the running max (the row max is
//                   taken first only where the max may have moved by 2^8),
//                   P written back to TMEM as bf16, lazy rescaling of O, epilogue.
//                   A unit with a single query tile ("split unit") gives the
//                   even key tiles to chain 0 and the odd ones to chain 1, both
//                   on the same rows; warpgroup 0 merges the two (m, l, O) in
//                   TMEM before its epilogue.
//     GQA: the G query heads sharing a KV head are packed into the rows of a
//     tile (row = token * G + head), so every K/V tile feeds 256 query rows.
//     The mask is applied per row as a visible-column count: every prefix key
//     is visible; window keys are visible up to W (bidirectional) or up to
//     the end of the query's own block (block-causal), and tiles past the
//     unit's last visible key are never loaded.
//  3. attn_merge_kernel: combines split-KV partial results by their
//     log-sum-exp.
#include <cmath>
#include <cuda.h>
#include <cuda_bf16.h>
#include <algorithm>
#include <mutex>
#include "common.cuh"
#include "ptx_sm103.cuh"
#include "tma_host.cuh"

namespace mbe {

MBE_DEFINE_ERROR_WORD(attention_take_error)

namespace attn {

constexpr int kTileKeys = 128;      // keys per K/V tile
constexpr int kTileRows = 128;      // packed query rows per tile (= TMEM lanes)
constexpr int kUnitRows = 256;      // packed query rows per work unit (two tiles)
constexpr int kThreads = 384;       // 12 warps
constexpr int kMergeThreads = 256;  // 8 rows per merge CTA
constexpr int kMaskTileWords = 16;   // block-mask mode: visible-tile bitmask of a unit (<= 512 key tiles)
constexpr int kMinChunk = 8;        // fewest key tiles in a split piece
constexpr int kSplitFactor = 4;     // most pieces per SM when splitting (bounds the workspace)
constexpr int kMaxGroupedSlabs = 8; // slabs of one (sequence, KV head) kept adjacent in the work list
constexpr float kUnitStartTiles = 2.f;  // start-up cost of a work unit, in key tiles (scheduler estimate)
constexpr int kBuckets = 1024;      // counting-sort buckets for unit cost
constexpr float kRescaleLog2 = 8.0f;  // rescale O only when the max grows by > 2^8
constexpr float kSpeculateSum = 128.f; // a tile's row sum below 2^7 proves no value reached 2^8
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemS = 256;    // S/P of tile i at columns 256 + 128 i; O_i at i * D

struct WorkUnit {
  int32_t seq, kv_head, row0, tile_begin, tile_end, slot, prefix, window_mode;  // window_mode = W | mode << 30
};
struct MergeGroup {
  int32_t seq, kv_head, row0, n_splits, slot_base, window, pad0, pad1;
};
// Plan signature: the call parameters that fix the workspace layout and the
// meaning of the work list. A run compares it with its own before using units.
constexpr int kSigWords = 9;
constexpr int32_t kPlanMagic = 0x4D424531;  // "MBE1"
struct PlanSig {
  int32_t w[kSigWords];
};
__host__ __device__ inline PlanSig make_sig(int batch, int total_tokens, int G, int Hkv, int D, int block_size,
                                            int max_window, int max_prefix) {
  return PlanSig{{kPlanMagic, batch, total_tokens, G, Hkv, D, block_size, max_window, max_prefix}};
}
__device__ inline bool sig_equal(const volatile int32_t* a, const PlanSig& b) {
  bool eq = true;
#pragma unroll
  for (int i = 0; i < kSigWords; ++i) eq &= (a[i] == b.w[i]);
  return eq;
}

struct Header {
  int32_t counter, n_units, n_groups;
  int32_t sig[kSigWords];
  int32_t pad[64 - 3 - kSigWords];
};
static_assert(sizeof(Header) == 256, "header size");

struct Layout {
  size_t units_tmp, units, groups, part_o, part_lse, total;
  int64_t max_units, max_groups, max_slots;
};

inline Layout make_layout(int batch, int Hq, int Hkv, int D, int max_window, int max_prefix, int num_sms) {
  const int64_t G = Hq / Hkv;
  const int64_t slabs = (static_cast<int64_t>(max_window) * G + kUnitRows - 1) / kUnitRows;
  const int64_t n_groups_all = static_cast<int64_t>(batch) * Hkv * slabs;
  const int64_t t_max = (max_prefix + kTileKeys - 1) / kTileKeys + (max_window + kTileKeys - 1) / kTileKeys;
  const int64_t total_max = std::max<int64_t>(n_groups_all * t_max, 1);
  Layout L;
  L.max_units = std::min<int64_t>(n_groups_all + static_cast<int64_t>(kSplitFactor) * num_sms, total_max) + 1;
  L.max_groups = std::min<int64_t>(static_cast<int64_t>(kSplitFactor) * num_sms, total_max / kMinChunk) + 1;
  L.max_slots = std::min<int64_t>(2ll * kSplitFactor * num_sms, 2 * total_max / kMinChunk) + 1;
  auto up = [](size_t x) { return (x + 255) & ~size_t(255); };
  size_t off = up(sizeof(Header));
  L.units_tmp = off; off = up(off + sizeof(WorkUnit) * L.max_units);
  L.units = off;     off = up(off + sizeof(WorkUnit) * L.max_units);
  L.groups = off;    off = up(off + sizeof(MergeGroup) * L.max_groups);
  L.part_o = off;    off = up(off + sizeof(float) * L.max_slots * kUnitRows * D);
  L.part_lse = off;  off = up(off + sizeof(float) * L.max_slots * kUnitRows);
  L.total = off;
  return L;
}

// ------------------------------------------------------------------ scheduler
struct SchedParams {
  const int32_t* prefix_len;  // null: no prefix (block-mask mode)
  const int32_t* window_len;
  const uint8_t* mask_mode;   // null: every sequence in block-mask mode
  const int32_t* cu_window;
  int batch, G, Hkv, block_size, max_window, max_prefix, num_sms, total_tokens;
  bool block_mask;
  PlanSig sig;
  Header* hdr;
  WorkUnit* units_tmp;
  WorkUnit* units;
  MergeGroup* groups;
  int64_t max_units, max_groups, max_slots;
};

// Key tiles (prefix, then window) that packed query rows [row0, row0 + 256) need.
// (block-mask mode: every window tile; the kernel skips the invisible ones)
__device__ __forceinline__ int slab_tiles(int P, int W, int mode, int row0, int G, int B) {
  const int nP = (P + kTileKeys - 1) / kTileKeys;
  int lim = W;
  if (mode == MBE_BLOCK_CAUSAL) {
    const int qmax = min(W, (row0 + kUnitRows) / G) - 1;
    lim = min(W, (qmax / B + 1) * B);
  }
  return nP + (lim + kTileKeys - 1) / kTileKeys;
}

__device__ __forceinline__ int seq_prefix(const SchedParams& p, int s) { return p.prefix_len ? p.prefix_len[s] : 0; }
__device__ __forceinline__ int seq_mode(const SchedParams& p, int s) {
  return p.mask_mode ? p.mask_mode[s] : MBE_BLOCK_MASK;
}

// A sequence is scheduled only if its lengths are within the declared bounds
// and its window rows [cu, cu + W) lie inside the q/out tensors.
__device__ __forceinline__ bool seq_ok(const SchedParams& p, int s, int P, int W, int mode) {
  if (W < 0 || W > p.max_window || P < 0 || P > p.max_prefix || mode > 2) return false;
  if ((mode == MBE_BLOCK_MASK) != p.block_mask) return false;
  const int cu = p.cu_window[s];
  return cu >= 0 && static_cast<int64_t>(cu) + W <= p.total_tokens;
}

__device__ __forceinline__ int cost_bucket(int cost, int chunk) {
  // 32-bit arithmetic while (cost - 1) * kBuckets fits (costs below 2^21 tiles)
  const int b = cost < (1 << 21) ? ((cost - 1) * kBuckets) / chunk
                                 : static_cast<int>((static_cast<int64_t>(cost - 1) * kBuckets) / chunk);
  return min(max(b, 0), kBuckets - 1);
}

// floor(k * T / n) for 0 <= k <= n <= T: 32-bit while k * T fits
__device__ __forceinline__ int split_point(int k, int T, int n) {
  return T < 46341 ? (k * T) / n : static_cast<int>((static_cast<int64_t>(k) * T) / n);
}

__global__ void __launch_bounds__(1024) attn_schedule_kernel(const SchedParams p) {
  __shared__ int s_total, s_nunits, s_ngroups, s_nslots, s_bad, s_tmin, s_tmax, s_nslab, s_sigma;
  __shared__ int hist[kBuckets];
  __shared__ int warp_sums[32];
  const int tid = threadIdx.x;
  if (tid == 0) {
    s_total = 0; s_nunits = 0; s_ngroups = 0; s_nslots = 0; s_bad = 0;
    s_tmin = 0x7FFFFFFF; s_tmax = 0; s_nslab = 0; s_sigma = 0;
  }
  for (int b = tid; b < kBuckets; b += blockDim.x) hist[b] = 0;
  __syncthreads();
  // pass 1: validate and count key tiles and slabs; the shortest and longest slab
  int local = 0, bad = 0, nslab = 0, tmin = 0x7FFFFFFF, tmax = 0;
  for (int s = tid; s < p.batch; s += blockDim.x) {
    const int P = seq_prefix(p, s), W = p.window_len[s], mode = seq_mode(p, s);
    if (!seq_ok(p, s, P, W, mode)) { bad = 1; continue; }
    const int slabs = (W * p.G + kUnitRows - 1) / kUnitRows;
    for (int sl = 0; sl < slabs; ++sl) {
      const int T = slab_tiles(P, W, mode, sl * kUnitRows, p.G, p.block_size);
      local += T * p.Hkv;
      tmin = min(tmin, T);
      tmax = max(tmax, T);
    }
    nslab += slabs * p.Hkv;
  }
  // one shared-memory atomic per warp (all 1024 threads on one address serialise)
  local = __reduce_add_sync(0xffffffffu, local);
  nslab = __reduce_add_sync(0xffffffffu, nslab);
  tmin = __reduce_min_sync(0xffffffffu, tmin);
  tmax = __reduce_max_sync(0xffffffffu, tmax);
  bad = __reduce_or_sync(0xffffffffu, bad);
  if ((tid & 31) == 0) {
    atomicAdd(&s_total, local);
    atomicAdd(&s_nslab, nslab);
    atomicMin(&s_tmin, tmin);
    atomicMax(&s_tmax, tmax);
    if (bad) atomicOr(&s_bad, 1);
  }
  __syncthreads();
  // Piece length: for each candidate (about 1..kSplitFactor pieces per SM)
  // count the units it makes and estimate the makespan as
  //   ceil(units / SMs) * (mean piece length + per-unit start-up cost),
  // keeping the longest pieces among equal estimates (fewer split-KV partials).
  __shared__ int s_units[kSplitFactor];
  if (tid < kSplitFactor) s_units[tid] = 0;
  __syncthreads();
  int cand[kSplitFactor];
#pragma unroll
  for (int k = 0; k < kSplitFactor; ++k) {
    const int target = (k + 1) * p.num_sms;  // ceil(s_total / target) without overflow
    cand[k] = max(kMinChunk, s_total / target + (s_total % target != 0 ? 1 : 0));
  }
  {
    int cnt[kSplitFactor] = {};
    for (int s = tid; s < p.batch; s += blockDim.x) {
      const int P = seq_prefix(p, s), W = p.window_len[s], mode = seq_mode(p, s);
      if (!seq_ok(p, s, P, W, mode)) continue;
      const int slabs = (W * p.G + kUnitRows - 1) / kUnitRows;
      for (int sl = 0; sl < slabs; ++sl) {
        const int T = slab_tiles(P, W, mode, sl * kUnitRows, p.G, p.block_size);
#pragma unroll
        for (int k = 0; k < kSplitFactor; ++k) cnt[k] += p.Hkv * ((T + cand[k] - 1) / cand[k]);
      }
    }
#pragma unroll
    for (int k = 0; k < kSplitFactor; ++k) {
      cnt[k] = __reduce_add_sync(0xffffffffu, cnt[k]);
      if ((tid & 31) == 0) atomicAdd(&s_units[k], cnt[k]);
    }
  }
  __syncthreads();
  int chunk = cand[0];
  float best = 3.4e38f;
  {
#pragma unroll
    for (int k = 0; k < kSplitFactor; ++k) {
      const int U = max(1, s_units[k]);
      const int waves = (U + p.num_sms - 1) / p.num_sms;
      const float est = waves * (static_cast<float>(s_total) / U + kUnitStartTiles);
      if (est < best * 0.98f) {  // a finer split must win clearly
        best = est;
        chunk = cand[k];
      }
    }
  }
  // Slabs of one length T (few long sequences of one shape): cutting the
  // concatenated key tiles of all slabs at multiples of total / SMs gives every
  // SM the same number of tiles in at most ceil(share / T) + 1 pieces, where equal
  // pieces per slab leave a fraction of a wave.
  const int T_uni = s_tmax;
  const bool stream_k = [&] {
    if (s_tmin != s_tmax || s_nslab < 1 || s_total < 2 * kMinChunk * p.num_sms) return false;
    const float share = static_cast<float>(s_total) / p.num_sms;
    const float est = ceilf(share) + (ceilf(share / T_uni) + 1.f) * kUnitStartTiles;
    return est < best * 0.98f;
  }();
  if (stream_k) chunk = min(T_uni, (s_total + p.num_sms - 1) / p.num_sms);  // the longest piece
  // pass 2: emit units (unsorted) and merge groups. The units of piece k of all
  // slabs of one (sequence, KV head) are emitted together (a "piece"): they
  // read the same K/V tiles, and the sort keeps them adjacent so that they run
  // at the same time and share those tiles in L2. The first unit of a piece
  // carries the piece's unit count and cost bucket in kv_head bits 16-19 / 20-29.
  bool overflow = false;
  auto emit_piece = [&](const WorkUnit* u, int count, int cost) {
    const int base = atomicAdd(&s_nunits, count);
    if (base + count > p.max_units) {
      overflow = true;
      return;
    }
    const int b = cost_bucket(cost, chunk);
    for (int i = 0; i < count; ++i) {
      WorkUnit w = u[i];
      if (i == 0) w.kv_head |= (count << 16) | (b << 20);
      p.units_tmp[base + i] = w;
    }
    atomicAdd(&hist[b], count);
  };
  // one thread per (sequence, KV head, slab group), so that few long sequences
  // still spread their pieces over many threads; a sequence with at most
  // kMaxGroupedSlabs slabs forms one group, longer ones one group per slab
  const int max_slabs = (p.max_window * p.G + kUnitRows - 1) / kUnitRows;
  const int groups_per_sg = max_slabs > kMaxGroupedSlabs ? max_slabs : 1;
  for (int64_t it = tid; it < static_cast<int64_t>(p.batch) * p.Hkv * groups_per_sg; it += blockDim.x) {
    const int sg = static_cast<int>(it / groups_per_sg);
    const int grp = static_cast<int>(it - static_cast<int64_t>(sg) * groups_per_sg);
    const int s = sg / p.Hkv, g = sg - s * p.Hkv;
    const int P = seq_prefix(p, s), W = p.window_len[s], mode = seq_mode(p, s);
    if (!seq_ok(p, s, P, W, mode)) continue;
    const int slabs = (W * p.G + kUnitRows - 1) / kUnitRows;
    if (stream_k) {
      if (grp > 0) continue;
      // slab sigma covers tiles [sigma T, sigma T + T) of the concatenation; SM share i
      // ends at b_i = floor(i total / SMs); a slab is cut at every b_i strictly inside it
      const int64_t total = s_total, S = p.num_sms;
      const int sigma0 = atomicAdd(&s_sigma, slabs);
      for (int sl = 0; sl < slabs; ++sl) {
        const int64_t lo = static_cast<int64_t>(sigma0 + sl) * T_uni, hi = lo + T_uni;
        const int64_t i_lo = ((lo + 1) * S + total - 1) / total;  // first i with b_i > lo
        const int64_t i_hi = (hi * S + total - 1) / total - 1;    // last i with b_i < hi
        const int n = static_cast<int>(i_hi >= i_lo ? i_hi - i_lo + 2 : 1);
        int slot0 = -1;
        if (n > 1) {
          const int gi = atomicAdd(&s_ngroups, 1);
          slot0 = atomicAdd(&s_nslots, n);
          if (gi < p.max_groups && slot0 + n <= p.max_slots)
            p.groups[gi] = MergeGroup{s, g, sl * kUnitRows, n, slot0, W, 0, 0};
          else
            overflow = true;
        }
        int64_t cut = lo;
        for (int k = 0; k < n; ++k) {
          const int64_t next = k + 1 < n ? ((i_lo + k) * total) / S : hi;
          const WorkUnit u{s, g, sl * kUnitRows, static_cast<int>(cut - lo), static_cast<int>(next - lo),
                           n > 1 ? slot0 + k : -1, P, W | (mode << 30)};
          emit_piece(&u, 1, static_cast<int>(next - cut));
          cut = next;
        }
      }
      continue;
    }
    const int ng = slabs <= kMaxGroupedSlabs ? slabs : 1;  // slabs per piece
    if (grp * ng >= slabs) continue;
    {
      for (int s0 = grp * ng; s0 < min(slabs, (grp + 1) * ng); s0 += ng) {
        const int cnt = min(ng, slabs - s0);
        int T[kMaxGroupedSlabs], n[kMaxGroupedSlabs], slot0[kMaxGroupedSlabs];
        int nmax = 0;
        for (int i = 0; i < cnt; ++i) {
          const int sl = s0 + i;
          T[i] = slab_tiles(P, W, mode, sl * kUnitRows, p.G, p.block_size);
          n[i] = (T[i] + chunk - 1) / chunk;
          nmax = max(nmax, n[i]);
          slot0[i] = -1;
          if (n[i] > 1) {
            const int gi = atomicAdd(&s_ngroups, 1);
            slot0[i] = atomicAdd(&s_nslots, n[i]);
            if (gi < p.max_groups && slot0[i] + n[i] <= p.max_slots) {
              p.groups[gi] = MergeGroup{s, g, sl * kUnitRows, n[i], slot0[i], W, 0, 0};
            } else {
              overflow = true;
            }
          }
        }
        for (int k = 0; k < nmax; ++k) {
          WorkUnit u[kMaxGroupedSlabs];
          int c = 0, cost = 1;
          for (int i = 0; i < cnt; ++i) {
            if (k >= n[i]) continue;
            const int tb = split_point(k, T[i], n[i]);
            const int te = split_point(k + 1, T[i], n[i]);
            u[c++] = WorkUnit{s, g, (s0 + i) * kUnitRows, tb, te, n[i] > 1 ? slot0[i] + k : -1, P, W | (mode << 30)};
            cost = max(cost, te - tb);
          }
          if (c > 0) emit_piece(u, c, cost);
        }
      }
    }
  }
  if (overflow) atomicOr(&s_bad, 2);
  __syncthreads();
  // exclusive scan of the histogram in descending-cost order
  {
    const int lane = tid & 31, warp = tid >> 5;
    const int b = kBuckets - 1 - tid;  // blockDim.x == kBuckets
    int v = hist[b];
    int x = v;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, off);
      if (lane >= off) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = warp_sums[lane];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, w, off);
        if (lane >= off) w += y;
      }
      warp_sums[lane] = w;
    }
    __syncthreads();
    const int excl = x - v + (warp > 0 ? warp_sums[warp - 1] : 0);
    __syncthreads();
    hist[b] = excl;
  }
  __syncthreads();
  const bool ok = (s_bad & 2) == 0;
  const int n_units = ok ? s_nunits : 0;
  for (int u = tid; u < n_units; u += blockDim.x) {
    const WorkUnit head = p.units_tmp[u];
    const int c = (head.kv_head >> 16) & 0xF;
    if (c == 0) continue;  // not the first unit of a piece
    const int pos = atomicAdd(&hist[(head.kv_head >> 20) & (kBuckets - 1)], c);
    for (int i = 0; i < c; ++i) {
      WorkUnit w = p.units_tmp[u + i];
      w.kv_head &= 0xFFFF;
      p.units[pos + i] = w;
    }
  }
  __syncthreads();
  if (tid == 0) {
    p.hdr->counter = 0;
    p.hdr->n_units = n_units;
    for (int i = 0; i < kSigWords; ++i) p.hdr->sig[i] = p.sig.w[i];
    p.hdr->n_groups = ok ? s_ngroups : 0;
    if (s_bad & 1) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
    if (s_bad & 2) atomicOr(&g_error_word, MBE_DEVERR_CAPACITY);
  }
}

// ------------------------------------------------------------------ main kernel
struct AttnParams {
  PlanSig sig;
  int batch, total_tokens;
  const int32_t* block_table;
  const int32_t* cu_window;
  __nv_bfloat16* out;
  float* lse;
  Header* hdr;
  const WorkUnit* units;
  float* part_o;
  float* part_lse;
  int max_pages, num_pages, Hq, G, block_size, page_size, box_rows, loads_per_tile;
  float scale_log2;
  // block-mask mode: bit kb of word kb / 32 of row qb of sequence s (mask + (s * mask_rows + qb) * mask_words)
  // is set iff query block qb attends to key block kb; block_log2 = log2(block_size)
  const uint32_t* mask;
  int mask_rows, mask_words, block_log2;
  uint64_t wait_ns;  // limit of the ordinary mbarrier waits
};

// Block-mask mode: does any query block of packed rows [row0, row0 + 256) see a
// key block of window tile t? W is the sequence length.
__device__ __forceinline__ bool tile_visible(const AttnParams& p, int seq, int row0, int W, int t) {
  const int q0 = row0 / p.G, q1 = min(W, (row0 + kUnitRows) / p.G) - 1;
  const int k0 = t * kTileKeys, k1 = min(W, k0 + kTileKeys) - 1;
  if (q1 < q0 || k1 < k0) return false;
  const int qb0 = q0 >> p.block_log2, qb1 = q1 >> p.block_log2;
  const int kb0 = k0 >> p.block_log2, kb1 = k1 >> p.block_log2;
  const uint32_t* m = p.mask + static_cast<int64_t>(seq) * p.mask_rows * p.mask_words;
  for (int qb = qb0; qb <= qb1 && qb < p.mask_rows; ++qb)
    for (int kb = kb0; kb <= kb1; ++kb)
      if (kb / 32 < p.mask_words && ((m[static_cast<int64_t>(qb) * p.mask_words + kb / 32] >> (kb % 32)) & 1u)) return true;
  return false;
}

// Next set bit after t in a unit's visible-tile bitmask (-1 if none).
__device__ __forceinline__ int next_tile(const volatile uint32_t* bits, int t) {
  for (int b = t + 1; b < kMaskTileWords * 32;) {
    const uint32_t w = bits[b >> 5] >> (b & 31);
    if (w) return b + __ffs(w) - 1;
    b = (b & ~31) + 32;
  }
  return -1;
}

// Shared memory: two Q tiles, then a ring of kSlots K-or-V tiles. Items are
// loaded in the order K(0), V(0), K(1), V(1), ...; K(t) is released once the
// QK products of tile t are done and V(t) once its PV products are done, so up
// to kSlots tile loads can be in flight.
template <int D>
struct Smem {
  static constexpr int kHalves = D / 64;
  static constexpr int kHalfBytes = 128 * 128;             // 128 rows x 128 B
  static constexpr int kQTile = kTileRows * D * 2;
  static constexpr int kItem = kTileKeys * D * 2;          // one K or one V tile
  static constexpr int kSlots = D == 128 ? 5 : 8;
  static constexpr int kQ = 0;
  static constexpr int kRing = 2 * kQTile;
  static constexpr int kUsed = kRing + kSlots * kItem;
  // at least 114 KB so that one CTA (and its 512 TMEM columns) owns the SM
  static constexpr int kBytes = (kUsed > 120 * 1024 ? kUsed : 120 * 1024) + 1024;
};
constexpr int kMaxSlots = 8;

__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float neg_inf() { return __int_as_float(0xff800000u); }

struct Bars {
  uint64_t q_full, q_empty, mma_done;
  uint64_t full[kMaxSlots], empty[kMaxSlots];
  uint64_t s_full[2], p_full[2], o_full[2], o_empty[2];
  uint64_t u_full[2], u_empty[2];
  uint64_t x_full, x_empty;  // split units: (m, l) of chain 1 handed to warpgroup 0
};

template <int D, bool kMask>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kw,
                const __grid_constant__ CUtensorMap tm_vw, const __grid_constant__ CUtensorMap tm_kc,
                const __grid_constant__ CUtensorMap tm_vc, const AttnParams p) {
  using S = Smem<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) Bars bars;
  __shared__ WorkUnit unit_ring[2];
  // block-mask mode: visible key tiles of each ring unit (bit t - tile_begin)
  __shared__ uint32_t unit_tiles[kMask ? 2 : 1][kMask ? kMaskTileWords : 1];
  __shared__ uint32_t tmem_base_s;
  __shared__ int abort_s;
  __shared__ float2 xchg[kTileRows];  // split units: running max and sum of chain 1, per row
  volatile int* abort_flag = &abort_s;
  const uint64_t wait_ns = p.wait_ns;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t sbase = smem_u32(smem);
  auto bar = [](uint64_t& b) { return smem_u32(&b); };

  if (tid == 0) {
    abort_s = 0;
    mbar_init(bar(bars.q_full), 1);
    mbar_init(bar(bars.q_empty), 1);
    mbar_init(bar(bars.mma_done), 1);
    for (int i = 0; i < S::kSlots; ++i) {
      mbar_init(bar(bars.full[i]), 1);
      mbar_init(bar(bars.empty[i]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(bar(bars.s_full[i]), 1);
      mbar_init(bar(bars.p_full[i]), 4);
      mbar_init(bar(bars.o_full[i]), 1);
      mbar_init(bar(bars.o_empty[i]), 4);
      mbar_init(bar(bars.u_full[i]), 1);
      mbar_init(bar(bars.u_empty[i]), 9);
    }
    mbar_init(bar(bars.x_full), 4);
    mbar_init(bar(bars.x_empty), 4);
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(&tmem_base_s), kTmemCols);
    tmem_relinquish();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base_s;
  // a work list planned for other parameters (or never planned) is not used
  const bool plan_ok = sig_equal(p.hdr->sig, p.sig);
  if (!plan_ok && blockIdx.x == 0 && tid == 0) atomicOr(&g_error_word, MBE_DEVERR_PLAN);
  const int n_units = plan_ok ? p.hdr->n_units : 0;

  if (warp == 0) {
    // ---------------------------------------------------------------- producer
    // The whole warp runs the loop (lane 0 issues the copies and barrier ops);
    // the lanes fetch 32 block-table entries at a time for the page lookups.
    if (lane == 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_kw);
      tma_prefetch_desc(&tm_vw);
      tma_prefetch_desc(&tm_kc);
      tma_prefetch_desc(&tm_vc);
    }
    constexpr unsigned kAll = 0xffffffffu;
    uint32_t item = 0, u_it = 0, q_loads = 0;
    bool ok = true;
    auto slot_of = [](uint32_t n) { return n % S::kSlots; };
    for (;;) {
      int uidx = 0;
      if (lane == 0) uidx = atomicAdd(&p.hdr->counter, 1);
      uidx = __shfl_sync(kAll, uidx, 0);
      const bool done = uidx >= n_units;
      const int uslot = u_it & 1;
      if (u_it >= 2) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.u_empty[uslot]), ((u_it >> 1) - 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
      }
      WorkUnit wu;
      if (done) {
        wu.seq = -1;
      } else {
        wu = p.units[uidx];
        const int W = wu.window_mode & 0x3FFFFFFF;
        const bool sane = wu.seq >= 0 && wu.seq < p.batch && wu.kv_head >= 0 && wu.tile_begin >= 0 &&
                          wu.tile_end > wu.tile_begin && W > 0 &&
                          (!kMask || wu.tile_end - wu.tile_begin <= kMaskTileWords * 32);
        const int cu = sane ? p.cu_window[wu.seq] : -1;
        if (!sane || cu < 0 || static_cast<int64_t>(cu) + W > p.total_tokens) {
          if (lane == 0) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
          continue;  // skip this unit; every role only ever sees published units
        }
      }
      if constexpr (kMask) {
        if (!done) {
          // visible key tiles of this unit (relative to tile_begin); an empty set keeps
          // its first tile (fully masked) so that every role still sees one tile
          const int n_rel = wu.tile_end - wu.tile_begin;
          const int W = wu.window_mode & 0x3FFFFFFF;
          bool any = false;
          for (int w = 0; w < kMaskTileWords; ++w) {
            const int rel = 32 * w + lane;
            const bool vis = rel < n_rel && tile_visible(p, wu.seq, wu.row0, W, wu.tile_begin + rel);
            const uint32_t word = __ballot_sync(kAll, vis);
            any |= word != 0;
            if (lane == 0) unit_tiles[uslot][w] = word;
          }
          if (!any && lane == 0) unit_tiles[uslot][0] = 1u;
        }
      }
      if (lane == 0) {
        unit_ring[uslot] = wu;
        mbar_arrive(bar(bars.u_full[uslot]));
      }
      __syncwarp();
      ++u_it;
      if (done) break;
      const int W = wu.window_mode & 0x3FFFFFFF;
      const int n_qt = (W * p.G - wu.row0) > kTileRows ? 2 : 1;
      const int cu = p.cu_window[wu.seq];
      if (q_loads >= 1) {
        ok = __all_sync(kAll, mbar_wait(bar(bars.q_empty), (q_loads - 1) & 1, abort_flag, wait_ns));
        if (!ok) break;
      }
      // the boxes of a load are issued by as many lanes at once (lane = box), each
      // completing on the same barrier, whose byte count lane 0 sets first
      if (lane == 0) mbar_arrive_expect_tx(bar(bars.q_full), n_qt * S::kQTile);
      __syncwarp();
      if (lane < n_qt * S::kHalves) {
        const int qt = lane / S::kHalves, h = lane % S::kHalves;
        tma_load_3d(sbase + S::kQ + qt * S::kQTile + h * S::kHalfBytes, &tm_q, bar(bars.q_full), h * 64,
                    wu.kv_head * p.G, cu + (wu.row0 + qt * kTileRows) / p.G);
      }
      ++q_loads;
      const int P = wu.prefix;
      const int nP = (P + kTileKeys - 1) / kTileKeys;
      const int64_t bt_row = static_cast<int64_t>(wu.seq) * p.max_pages;
      // Page ids: lane L holds the physical page of logical pages pg_base + L
      // (pg_lo) and pg_base + 32 + L (pg_hi); one coalesced block-table read
      // serves 32 pages.
      auto fetch_page = [&](int lpage) {
        int pg = p.num_pages;  // out of range: TMA fills zeros
        if (lpage >= 0 && static_cast<int64_t>(lpage) * p.page_size < P) {
          pg = p.block_table[bt_row + lpage];
          if (pg < 0 || pg >= p.num_pages) {
            atomicOr(&g_error_word, MBE_DEVERR_PAGE);
            pg = p.num_pages;
          }
        }
        return pg;
      };
      int pg_base = -(1 << 30), pg_lo = 0, pg_hi = 0;
      auto page_of = [&](int lp) {  // per-lane lp in [pg_base, pg_base + 64)
        const int lo = __shfl_sync(kAll, pg_lo, (lp - pg_base) & 31);
        const int hi = __shfl_sync(kAll, pg_hi, (lp - pg_base) & 31);
        return lp < pg_base + 32 ? lo : hi;
      };
      auto ensure_window = [&](int lp) {  // makes lp the current page window's anchor if needed
        if (lp < pg_base || lp >= pg_base + 64) {
          pg_base = lp;
          pg_lo = fetch_page(pg_base + lane);
          pg_hi = fetch_page(pg_base + 32 + lane);
        } else if (lp >= pg_base + 32) {
          pg_base += 32;
          pg_lo = pg_hi;
          pg_hi = fetch_page(pg_base + 32 + lane);
        }
      };
      // block-mask mode walks the unit's visible tiles, the other modes every tile
      const volatile uint32_t* tbits = unit_tiles[kMask ? uslot : 0];
      auto advance = [&](int t) {
        if (!kMask) return t + 1;
        const int r = next_tile(tbits, t - wu.tile_begin);
        return r < 0 ? wu.tile_end : wu.tile_begin + r;
      };
      for (int t = kMask ? advance(wu.tile_begin - 1) : wu.tile_begin; t < wu.tile_end && ok; t = advance(t)) {
        if (t < nP) ensure_window((t * kTileKeys) / p.page_size);
        for (int kv = 0; kv < 2; ++kv, ++item) {
          const uint32_t sl = slot_of(item), use = item / S::kSlots;
          if (use >= 1) {
            ok = __all_sync(kAll, mbar_wait(bar(bars.empty[sl]), (use - 1) & 1, abort_flag, wait_ns));
            if (!ok) break;
          }
          const uint32_t dst = sbase + S::kRing + sl * S::kItem;
          const uint32_t fb = bar(bars.full[sl]);
          if (lane == 0) mbar_arrive_expect_tx(fb, S::kItem);
          __syncwarp();
          if (t < nP) {
            // lane = box: page box l = lane / halves, column half h = lane % halves
            // (at most 16 boxes: 128 keys over pages of 8 or more, two halves)
            const CUtensorMap* tm = kv ? &tm_vc : &tm_kc;
            const int l = lane / S::kHalves, h = lane % S::kHalves;
            const int key0 = t * kTileKeys + min(l, p.loads_per_tile - 1) * p.box_rows;
            const int page = page_of(key0 / p.page_size);
            if (l < p.loads_per_tile)
              tma_load_4d(dst + h * S::kHalfBytes + l * p.box_rows * 128, tm, fb, h * 64, key0 % p.page_size,
                          wu.kv_head, page);
          } else if (lane < S::kHalves) {
            const int tok = cu + (t - nP) * kTileKeys;
            tma_load_3d(dst + lane * S::kHalfBytes, kv ? &tm_vw : &tm_kw, fb, lane * 64, wu.kv_head, tok);
          }
        }
      }
      if (!ok) break;
    }
    if (!ok && lane == 0) {
      *abort_flag = 1;
      atomicOr(&g_error_word, MBE_DEVERR_TIMEOUT);
    }
    // The copies already issued land before the CTA can exit, also when another
    // role aborted after this loop ended (without an abort they have all been
    // consumed, and these waits return at once).
    if (lane == 0) {
      const int zero = 0;
      for (uint32_t n = (item >= S::kSlots ? item - S::kSlots : 0); n < item; ++n)
        mbar_wait(bar(bars.full[slot_of(n)]), (n / S::kSlots) & 1, &zero);
      if (q_loads >= 1) mbar_wait(bar(bars.q_full), (q_loads - 1) & 1, &zero);
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(128, 128, false, false);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(128, D, false, true);
      uint32_t kv_it = 0, u_it = 0, q_it = 0;
      uint32_t p_cnt[2] = {0, 0}, o_cnt[2] = {0, 0};
      bool ok = true;
      auto item_addr = [&](uint32_t n) { return sbase + S::kRing + (n % S::kSlots) * S::kItem; };
      auto wait_item = [&](uint32_t n) { return mbar_wait(bar(bars.full[n % S::kSlots]), (n / S::kSlots) & 1, abort_flag, wait_ns); };
      auto release_item = [&](uint32_t n) { umma_commit(bar(bars.empty[n % S::kSlots])); };
      // S of chain i = Q tile qt times K (qt = i, or 0 for both chains of a split unit)
      // descriptors of a tile: one built per operand, the K steps by constant adds
      auto issue_qk = [&](int i, uint32_t ka, int qt) {
        const uint64_t qd = sdesc_sw128(sbase + S::kQ + qt * S::kQTile, 16, 1024), kd = sdesc_sw128(ka, 16, 1024);
#pragma unroll
        for (int h = 0; h < S::kHalves; ++h)
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_ss(tmem + kTmemS + 128 * i, desc_add(qd, (h * S::kHalfBytes + k * 32) >> 4),
                    desc_add(kd, (h * S::kHalfBytes + k * 32) >> 4), idesc_qk, (h | k) ? 1u : 0u);
      };
      auto issue_pv = [&](int i, uint32_t va, bool acc) {
        const uint64_t vd = sdesc_sw128(va, S::kHalfBytes, 1024);
#pragma unroll
        for (int kk = 0; kk < kTileKeys / 16; ++kk)
          umma_ts(tmem + i * D, tmem + kTmemS + 128 * i + kk * 8, desc_add(vd, (kk * 16 * 128) >> 4), idesc_pv,
                  (acc || kk > 0) ? 1u : 0u);
      };
      for (;;) {
        const int slot = u_it & 1;
        if (!mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag, wait_ns)) { ok = false; break; }
        const WorkUnit wu = unit_ring[slot];
        int n_t = wu.tile_end - wu.tile_begin;
        if constexpr (kMask) {
          n_t = 0;
          for (int w = 0; w < kMaskTileWords; ++w) n_t += __popc(unit_tiles[slot][w]);
        }
        mbar_arrive(bar(bars.u_empty[slot]));
        ++u_it;
        if (wu.seq < 0) break;
        const int W = wu.window_mode & 0x3FFFFFFF;
        const int n_qt = (W * p.G - wu.row0) > kTileRows ? 2 : 1;
        if (!mbar_wait(bar(bars.q_full), q_it & 1, abort_flag, wait_ns)) { ok = false; break; }
        ++q_it;
        // items of tile ki: K = 2 ki, V = 2 ki + 1
        if (n_qt == 1 && n_t >= 2) {
          // Split unit (one query tile, two or more key tiles): chain c takes the key
          // tiles j = c, c + 2, ..., both against query tile 0, so that the two chains
          // overlap as they do for two query tiles; the epilogue merges them.
          for (int c = 0; c < 2 && ok; ++c) {
            if (!wait_item(2 * (kv_it + c))) { ok = false; break; }
            tc_fence_after();
            issue_qk(c, item_addr(2 * (kv_it + c)), 0);
            umma_commit(bar(bars.s_full[c]));
            release_item(2 * (kv_it + c));
          }
          if (!ok) break;
          if (n_t == 2) umma_commit(bar(bars.q_empty));
          for (int j0 = 0; j0 < n_t && ok; j0 += 2) {
#pragma unroll
            for (int c = 0; c < 2; ++c) {  // chain c as a constant: no indexed counters
              const int j = j0 + c;
              if (j >= n_t || !ok) break;
              const uint32_t ki = kv_it + j;
              if (!wait_item(2 * ki + 1)) { ok = false; break; }
              if (!mbar_wait(bar(bars.p_full[c]), p_cnt[c] & 1, abort_flag, wait_ns)) { ok = false; break; }
              ++p_cnt[c];
              if (j < 2 && o_cnt[c] > 0 && !mbar_wait(bar(bars.o_empty[c]), (o_cnt[c] - 1) & 1, abort_flag, wait_ns)) {
                ok = false;
                break;
              }
              tc_fence_after();
              issue_pv(c, item_addr(2 * ki + 1), j >= 2);
              if (j + 2 >= n_t) umma_commit(bar(bars.o_full[c]));  // the chain's last tile
              release_item(2 * ki + 1);
              if (j + 2 < n_t) {
                const uint32_t kn = 2 * (ki + 2);
                if (!wait_item(kn)) { ok = false; break; }
                tc_fence_after();
                issue_qk(c, item_addr(kn), 0);
                umma_commit(bar(bars.s_full[c]));
                release_item(kn);
                if (j + 3 == n_t) umma_commit(bar(bars.q_empty));  // the unit's last QK
              }
            }
          }
          if (!ok) break;
          kv_it += n_t;
          ++o_cnt[0];
          ++o_cnt[1];
          continue;
        }
        if (!wait_item(2 * kv_it)) { ok = false; break; }
        tc_fence_after();
        for (int i = 0; i < n_qt; ++i) {
          issue_qk(i, item_addr(2 * kv_it), i);
          umma_commit(bar(bars.s_full[i]));
        }
        release_item(2 * kv_it);
        if (n_t == 1) umma_commit(bar(bars.q_empty));
        for (int j = 0; j < n_t && ok; ++j) {
          const uint32_t ki = kv_it + j;
          if (!wait_item(2 * ki + 1)) { ok = false; break; }
          for (int i = 0; i < n_qt; ++i) {
            if (!mbar_wait(bar(bars.p_full[i]), p_cnt[i] & 1, abort_flag, wait_ns)) { ok = false; break; }
            ++p_cnt[i];
            if (j == 0 && o_cnt[i] > 0 && !mbar_wait(bar(bars.o_empty[i]), (o_cnt[i] - 1) & 1, abort_flag, wait_ns)) {
              ok = false;
              break;
            }
            tc_fence_after();
            issue_pv(i, item_addr(2 * ki + 1), j > 0);
            if (j == n_t - 1) umma_commit(bar(bars.o_full[i]));
            if (i == n_qt - 1) release_item(2 * ki + 1);
            if (j + 1 < n_t) {
              const uint32_t kn = 2 * (ki + 1);
              if (i == 0) {
                if (!wait_item(kn)) { ok = false; break; }
                tc_fence_after();
              }
              issue_qk(i, item_addr(kn), i);
              umma_commit(bar(bars.s_full[i]));
              if (i == n_qt - 1) {
                release_item(kn);
                if (j + 2 == n_t) umma_commit(bar(bars.q_empty));
              }
            }
          }
        }
        if (!ok) break;
        kv_it += n_t;
        for (int i = 0; i < n_qt; ++i) ++o_cnt[i];
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
    // ---------------------------------------------------------------- softmax + epilogue
    const int wg = (warp - 4) >> 2;           // query tile 0 or 1
    const int quad = warp & 3;                // TMEM lane quadrant of this warp
    const int r = quad * 32 + lane;           // row within the tile
    const uint32_t t_lane = tmem + (static_cast<uint32_t>(quad * 32) << 16);
    const uint32_t tS = t_lane + kTmemS + 128 * wg;
    const uint32_t tO = t_lane + wg * D;
    uint32_t u_it = 0, s_cnt = 0, o_cnt = 0, kv_it = 0, x_cnt = 0;
    bool ok = true;
    for (;;) {
      const int slot = u_it & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.u_full[slot]), (u_it >> 1) & 1, abort_flag, wait_ns));
      if (!ok) break;
      const WorkUnit wu = unit_ring[slot];
      // block-mask mode keeps the ring slot (and its tile bitmask) until its tiles are done
      auto release_unit = [&]() {
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.u_empty[slot]));
      };
      if (!kMask) release_unit();
      ++u_it;
      if (wu.seq < 0) {
        if (kMask) release_unit();
        break;
      }
      const int W = wu.window_mode & 0x3FFFFFFF;
      const int mode = static_cast<int>(static_cast<uint32_t>(wu.window_mode) >> 30);
      const int n_qt = (W * p.G - wu.row0) > kTileRows ? 2 : 1;
      int n_t = wu.tile_end - wu.tile_begin;
      const volatile uint32_t* tbits = unit_tiles[kMask ? slot : 0];
      if constexpr (kMask) {
        n_t = 0;
        for (int w = 0; w < kMaskTileWords; ++w) n_t += __popc(tbits[w]);
      }
      const int P = wu.prefix;
      const int nP = (P + kTileKeys - 1) / kTileKeys;
      // split unit: both warpgroups work on query tile 0, warpgroup c on key tiles c, c + 2, ...
      const bool split = n_qt == 1 && n_t >= 2;
      if (wg >= n_qt && !split) {
        kv_it += n_t;
        if (kMask) release_unit();
        continue;
      }
      const int R = wu.row0 + kTileRows * (split ? 0 : wg) + r;
      const int qi = R / p.G, hh = R - qi * p.G;
      const bool valid = qi < W;
      const int lim = (mode == MBE_BLOCK_CAUSAL) ? min(W, (qi / p.block_size + 1) * p.block_size) : W;
      // block-mask mode: this row's mask row (query block of token qi)
      const uint32_t* mrow = nullptr;
      int kbpt = 1;
      uint32_t all_bits = 1u;
      if constexpr (kMask) {
        const int qb = min(qi, W - 1) >> p.block_log2;
        mrow = p.mask + (static_cast<int64_t>(wu.seq) * p.mask_rows + min(qb, p.mask_rows - 1)) * p.mask_words;
        kbpt = max(1, kTileKeys >> p.block_log2);
        all_bits = kbpt >= 32 ? 0xFFFFFFFFu : ((1u << kbpt) - 1u);
      }
      float m = neg_inf(), l = 0.f;
      int t = wu.tile_begin - 1;
      for (int j = 0; j < n_t; ++j) {
        if constexpr (kMask) {
          const int rnext = next_tile(tbits, t - wu.tile_begin);
          t = wu.tile_begin + max(rnext, 0);
        } else {
          t = wu.tile_begin + j;
        }
        if (split && (j & 1) != wg) continue;
        const uint32_t ki = kv_it + j;
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.s_full[wg]), s_cnt & 1, abort_flag, wait_ns));
        if (!ok) break;
        ++s_cnt;
        tc_fence_after();
        const int n_vis = t < nP ? min(kTileKeys, P - t * kTileKeys) : max(0, min(kTileKeys, lim - (t - nP) * kTileKeys));
        // block-mask mode: bit c >> block_log2 of nib tells whether column c's key block is visible
        uint32_t nib = 0xFFFFFFFFu;
        if constexpr (kMask) {
          const int kb0 = ((t - nP) * kTileKeys) >> p.block_log2;
          const uint32_t word = (kb0 >> 5) < p.mask_words ? mrow[kb0 >> 5] : 0u;
          nib = (word >> (kb0 & 31)) & all_bits;
        }
        auto visible = [&](int k) { return k < n_vis && (!kMask || ((nib >> (k >> p.block_log2)) & 1u)); };
        // The whole S row (128 fp32) comes from TMEM in one load; P is packed to
        // bf16 in place (entry k <- columns 2k, 2k+1) and stored as 64 columns
        // over the start of the same TMEM region.
        const bool all_vis = __all_sync(0xffffffffu, n_vis == kTileKeys && (!kMask || nib == all_bits));
        bool full = all_vis;
        uint32_t v[128];
        tmem_ld128(tS, v);
        // block-mask mode: invisible columns (other key blocks, past the sequence)
        // become -inf and the tile takes the packed path (exp2(-inf) = 0); cm holds
        // this row's visible columns so that S read again is masked the same way
        uint32_t cm[4] = {0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu, 0xFFFFFFFFu};
        auto mask_invisible = [&]() {
#pragma unroll
          for (int k = 0; k < 128; ++k)
            if (!((cm[k >> 5] >> (k & 31)) & 1u)) v[k] = 0xFF800000u;
        };
        if constexpr (kMask) {
          if (!all_vis) {
#pragma unroll
            for (int w = 0; w < 4; ++w) {
              uint32_t bits;
              if (p.block_log2 >= 5) {
                bits = ((nib >> ((32 * w) >> p.block_log2)) & 1u) ? 0xFFFFFFFFu : 0u;
              } else {  // 8- or 16-token blocks: 32 / B blocks per word
                const int per = 32 >> p.block_log2, base = (32 * w) >> p.block_log2;
                const uint32_t run = (1u << (1 << p.block_log2)) - 1u;
                bits = 0u;
                for (int b = 0; b < per; ++b)
                  if ((nib >> (base + b)) & 1u) bits |= run << (b << p.block_log2);
              }
              const int lo = 32 * w;
              bits &= n_vis >= lo + 32 ? 0xFFFFFFFFu : (n_vis <= lo ? 0u : ((1u << (n_vis - lo)) - 1u));
              cm[w] = bits;
            }
            mask_invisible();
            full = true;
          }
        }
        // exponentials of a fully visible tile against the reference max: P (bf16
        // pairs) replaces the first half of v, (l0, l1) are its row sums
        auto exp_full = [&](float neg_mu, float& l0, float& l1) {
          const float2 sl2 = make_float2(p.scale_log2, p.scale_log2), nm2 = make_float2(neg_mu, neg_mu);
          float2 la = make_float2(0.f, 0.f), lb = make_float2(0.f, 0.f);
#pragma unroll
          for (int k = 0; k < 64; ++k) {
            const float2 x = ffma2(make_float2(__uint_as_float(v[2 * k]), __uint_as_float(v[2 * k + 1])), sl2, nm2);
            const float2 e = make_float2(ex2f(x.x), ex2f(x.y));
            if (k & 1) lb = fadd2(lb, e); else la = fadd2(la, e);
            v[k] = pack_bf16x2(e.x, e.y);
          }
          const float2 ls = fadd2(la, lb);
          l0 = ls.x;
          l1 = ls.y;
        };
        // Lazy rescaling: the reference max m only moves when the tile's max
        // exceeds it by more than 2^8; P, l and O then all use the new m. A fully
        // visible tile with a finite m first takes its exponentials against m as it
        // stands: if no row's sum exceeds 2^7, no value reached 2^8, m would not move
        // and P is final (the values the max-first order gives). Otherwise S is read
        // again and the row max decides, as for every other tile.
        float l0 = 0.f, l1 = 0.f, alpha = 1.f;
        bool rescale = false, done = false;
        if (full && __all_sync(0xffffffffu, m != neg_inf())) {
          exp_full(-m, l0, l1);
          done = !__any_sync(0xffffffffu, !(l0 + l1 <= kSpeculateSum));
          if (!done) {
            tmem_ld128(tS, v);
            if (kMask && !all_vis) mask_invisible();
          }
        }
        if (!done) {
          float mx = neg_inf();
          if (full) {
            // eight independent accumulators: the maximum does not depend on the order,
            // and short dependency chains keep the softmax latency down
            float acc[8];
#pragma unroll
            for (int a = 0; a < 8; ++a) acc[a] = neg_inf();
#pragma unroll
            for (int k = 0; k < 128; k += 16)
#pragma unroll
              for (int a = 0; a < 8; ++a)
                acc[a] = fmax3(acc[a], __uint_as_float(v[k + 2 * a]), __uint_as_float(v[k + 2 * a + 1]));
            mx = fmaxf(fmax3(acc[0], acc[1], acc[2]), fmax3(acc[3], fmax3(acc[4], acc[5], acc[6]), acc[7]));
          } else {
#pragma unroll
            for (int k = 0; k < 128; ++k)
              if (visible(k)) mx = fmaxf(mx, __uint_as_float(v[k]));
          }
          const float m_new = fmaxf(m, mx * p.scale_log2);
          rescale = __any_sync(0xffffffffu, m_new > m + kRescaleLog2);
          if (rescale) {
            alpha = (m_new == neg_inf()) ? 1.f : ex2f(m - m_new);
            m = m_new;
          }
          const float neg_mu = (m == neg_inf()) ? 0.f : -m;
          if (full) {
            exp_full(neg_mu, l0, l1);
          } else {
#pragma unroll
            for (int k = 0; k < 64; ++k) {
              const float p0 = visible(2 * k) ? ex2f(fmaf(__uint_as_float(v[2 * k]), p.scale_log2, neg_mu)) : 0.f;
              const float p1 = visible(2 * k + 1) ? ex2f(fmaf(__uint_as_float(v[2 * k + 1]), p.scale_log2, neg_mu)) : 0.f;
              l0 += p0;
              l1 += p1;
              v[k] = pack_bf16x2(p0, p1);
            }
          }
        }
        tmem_st64(tS, v);
        l = l * alpha + (l0 + l1);
        if (rescale && j >= (split ? 2 : 1)) {
          // O holds PV of this chain's earlier tiles (complete: s_full of this tile
          // was committed after them)
#pragma unroll 1
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o[32];
            tmem_ld32(tO + 32 * c, o);
#pragma unroll
            for (int k = 0; k < 32; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * alpha);
            tmem_st32(tO + 32 * c, o);
          }
        }
        tmem_st_wait();
        // Rows past the end of the last prefix tile (stale cache rows) or of the
        // last window tile (whatever follows the window in k_win / v_win, even
        // NaN) are masked in S but still enter P V as 0 * V: zero them in V.
        const int v0 = (t == nP - 1) ? P % kTileKeys : (t - nP == (W - 1) / kTileKeys ? W % kTileKeys : 0);
        if ((split || wg == 0) && v0 != 0) {
          const uint32_t nv = 2 * ki + 1;  // the V item of this tile
          ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.full[nv % S::kSlots]), (nv / S::kSlots) & 1, abort_flag, wait_ns));
          if (!ok) break;
          uint8_t* vt = smem + S::kRing + (nv % S::kSlots) * S::kItem;
          const int per_row = S::kHalves * 8;  // 16-byte chunks per key row
          for (int idx = r; idx < (kTileKeys - v0) * per_row; idx += kTileRows) {
            const int row = v0 + idx / per_row, rem = idx % per_row;
            *reinterpret_cast<uint4*>(vt + (rem / 8) * S::kHalfBytes + row * 128 + (rem % 8) * 16) =
                make_uint4(0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.p_full[wg]));
      }
      if (!ok) break;
      kv_it += n_t;
      if (kMask) release_unit();
      // epilogue: O_i is complete once o_full fires
      ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.o_full[wg]), o_cnt & 1, abort_flag, wait_ns));
      if (!ok) break;
      ++o_cnt;
      tc_fence_after();
      if (split && wg == 1) {
        // chain 1 of a split unit hands its running max and sum to warpgroup 0, which
        // reads O_1 from TMEM (same lanes), merges and releases both O buffers
        if (x_cnt > 0) {
          ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.x_empty), (x_cnt - 1) & 1, abort_flag, wait_ns));
          if (!ok) break;
        }
        ++x_cnt;
        xchg[r] = make_float2(m, l);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.x_full));
        continue;
      }
      if (split) {
        ok = __all_sync(0xffffffffu, mbar_wait(bar(bars.x_full), x_cnt & 1, abort_flag, wait_ns));
        if (!ok) break;
        ++x_cnt;
        tc_fence_after();  // O_1 is complete: warpgroup 1 saw its o_full before x_full
        const float2 c1 = xchg[r];
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(bars.x_empty));
        const float mm = fmaxf(m, c1.x);
        const float a0 = (m == neg_inf()) ? 0.f : ex2f(m - mm);
        const float a1 = (c1.x == neg_inf()) ? 0.f : ex2f(c1.x - mm);
        l = l * a0 + c1.y * a1;
        m = mm;
        // O_0 <- a0 O_0 + a1 O_1 in TMEM; the epilogue below then reads O_0 only
#pragma unroll 1
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o0[32], o1[32];
          tmem_ld32(tO + 32 * c, o0);
          tmem_ld32(t_lane + D + 32 * c, o1);
#pragma unroll
          for (int k = 0; k < 32; ++k)
            o0[k] = __float_as_uint(fmaf(__uint_as_float(o0[k]), a0, __uint_as_float(o1[k]) * a1));
          tmem_st32(tO + 32 * c, o0);
        }
        tmem_st_wait();
      }
      const float inv_l = l > 0.f ? 1.f / l : 0.f;
      const float lse2 = l > 0.f ? m + __log2f(l) : neg_inf();
      if (wu.slot < 0) {
        const int cu = p.cu_window[wu.seq];
        __nv_bfloat16* orow =
            p.out + (static_cast<int64_t>(cu + qi) * p.Hq + wu.kv_head * p.G + hh) * D;
        // O / l as bf16, 32 columns per TMEM load, with 32-byte stores: the row is
        // 32-byte aligned and each store fills one sector
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + 32 * c, o);
          if (valid) {
            uint32_t w[16];
#pragma unroll
            for (int k = 0; k < 16; ++k)
              w[k] = pack_bf16x2(__uint_as_float(o[2 * k]) * inv_l, __uint_as_float(o[2 * k + 1]) * inv_l);
#pragma unroll
            for (int v = 0; v < 2; ++v)
              st_global_v8(orow + 32 * c + 16 * v, w[8 * v], w[8 * v + 1], w[8 * v + 2], w[8 * v + 3], w[8 * v + 4],
                           w[8 * v + 5], w[8 * v + 6], w[8 * v + 7]);
          }
        }
        if (valid && p.lse) p.lse[static_cast<int64_t>(cu + qi) * p.Hq + wu.kv_head * p.G + hh] = lse2 * 0.6931471805599453f;
      } else {
        // split piece: fp32 O / l and the log2-sum-exp, merged afterwards
        const int prow = kTileRows * wg + r;
        float* po = p.part_o + (static_cast<int64_t>(wu.slot) * kUnitRows + prow) * D;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + 32 * c, o);
          if (valid) {
#pragma unroll
            for (int v = 0; v < 4; ++v) {
              uint32_t w[8];
#pragma unroll
              for (int k = 0; k < 8; ++k) w[k] = __float_as_uint(__uint_as_float(o[8 * v + k]) * inv_l);
              st_global_v8(po + 32 * c + 8 * v, w[0], w[1], w[2], w[3], w[4], w[5], w[6], w[7]);
            }
          }
        }
        if (valid) p.part_lse[static_cast<int64_t>(wu.slot) * kUnitRows + prow] = lse2;
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(bar(bars.o_empty[wg]));
        if (split) mbar_arrive(bar(bars.o_empty[1]));
      }
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

// ------------------------------------------------------------------ split merge
struct MergeParams {
  PlanSig sig;
  int batch, total_tokens;
  Header* hdr;
  const MergeGroup* groups;
  const float* part_o;
  const float* part_lse;
  const int32_t* cu_window;
  __nv_bfloat16* out;
  float* lse;
  int Hq, G;
};

// One warp per block of kMergeRows packed query rows of a split group: lane l
// holds D/32 consecutive output columns of every row, so every partial row is
// read as one coalesced 4 D-byte line; the loads of all rows of the block and of
// kMergeBatch splits are issued before any is used, so that groups with few
// splits still keep several lines per warp in flight.
constexpr int kMergeRows = 4;
constexpr int kMergeBatch = 2;

template <int D>
__device__ __forceinline__ void merge_rows_warp(const MergeParams& p, const MergeGroup& grp, int r0, int lane) {
  constexpr int kPer = D / 32;  // 4 for D = 128, 2 for D = 64
  const int cu = p.cu_window[grp.seq];
  if (cu < 0 || static_cast<int64_t>(cu) + grp.window > p.total_tokens) return;
  bool live[kMergeRows];
  int64_t orow[kMergeRows];
  bool any = false;
#pragma unroll
  for (int rr = 0; rr < kMergeRows; ++rr) {
    const int R = grp.row0 + r0 + rr;
    const int qi = R / p.G, hh = R - qi * p.G;
    live[rr] = qi < grp.window;
    any |= live[rr];
    orow[rr] = static_cast<int64_t>(cu + qi) * p.Hq + grp.kv_head * p.G + hh;
  }
  if (!any) return;
  // partial row r of split k: lse at (slot_base + k) * kUnitRows + r, O at that row * D
  const int64_t base = static_cast<int64_t>(grp.slot_base) * kUnitRows + r0;
  const int n = grp.n_splits;
  // Online merge: the running maximum M of the splits' log-sum-exps rescales
  // what has been summed so far when it grows (one pass over the partials).
  float M[kMergeRows], wsum[kMergeRows], acc[kMergeRows][kPer];
#pragma unroll
  for (int rr = 0; rr < kMergeRows; ++rr) {
    M[rr] = neg_inf();
    wsum[rr] = 0.f;
#pragma unroll
    for (int d = 0; d < kPer; ++d) acc[rr][d] = 0.f;
  }
  for (int k0 = 0; k0 < n; k0 += kMergeBatch) {
    float lk[kMergeRows][kMergeBatch], v[kMergeRows][kMergeBatch][kPer];
#pragma unroll
    for (int u = 0; u < kMergeBatch; ++u) {
      const int k = k0 + u;
#pragma unroll
      for (int rr = 0; rr < kMergeRows; ++rr) {
        lk[rr][u] = neg_inf();
#pragma unroll
        for (int d = 0; d < kPer; ++d) v[rr][u][d] = 0.f;
        if (k < n && live[rr]) {
          const int64_t row = base + static_cast<int64_t>(k) * kUnitRows + rr;
          lk[rr][u] = p.part_lse[row];
          const float* src = p.part_o + row * D + lane * kPer;
          if constexpr (kPer == 4) {
            const float4 x = *reinterpret_cast<const float4*>(src);
            v[rr][u][0] = x.x; v[rr][u][1] = x.y; v[rr][u][2] = x.z; v[rr][u][3] = x.w;
          } else {
            const float2 x = *reinterpret_cast<const float2*>(src);
            v[rr][u][0] = x.x; v[rr][u][1] = x.y;
          }
        }
      }
    }
#pragma unroll
    for (int rr = 0; rr < kMergeRows; ++rr) {
      float mb = lk[rr][0];
#pragma unroll
      for (int u = 1; u < kMergeBatch; ++u) mb = fmaxf(mb, lk[rr][u]);
      if (mb > M[rr]) {
        const float c = (M[rr] == neg_inf()) ? 0.f : ex2f(M[rr] - mb);
        wsum[rr] *= c;
#pragma unroll
        for (int d = 0; d < kPer; ++d) acc[rr][d] *= c;
        M[rr] = mb;
      }
#pragma unroll
      for (int u = 0; u < kMergeBatch; ++u) {
        const float w = (lk[rr][u] == neg_inf()) ? 0.f : ex2f(lk[rr][u] - M[rr]);
        wsum[rr] += w;
#pragma unroll
        for (int d = 0; d < kPer; ++d) acc[rr][d] += w * v[rr][u][d];
      }
    }
  }
#pragma unroll
  for (int rr = 0; rr < kMergeRows; ++rr) {
    if (!live[rr]) continue;
    const float inv = wsum[rr] > 0.f ? 1.f / wsum[rr] : 0.f;
    __nv_bfloat16* dst = p.out + orow[rr] * D + lane * kPer;
    if constexpr (kPer == 4)
      *reinterpret_cast<uint2*>(dst) = make_uint2(pack_bf16x2(acc[rr][0] * inv, acc[rr][1] * inv),
                                                  pack_bf16x2(acc[rr][2] * inv, acc[rr][3] * inv));
    else
      *reinterpret_cast<uint32_t*>(dst) = pack_bf16x2(acc[rr][0] * inv, acc[rr][1] * inv);
    if (p.lse && lane == 0)
      p.lse[orow[rr]] = (wsum[rr] > 0.f ? M[rr] + __log2f(wsum[rr]) : neg_inf()) * 0.6931471805599453f;
  }
}

// Grid-stride over (split group, block of kMergeRows rows) items, one warp per item.
template <int D>
__global__ void __launch_bounds__(kMergeThreads, 2) attn_merge_kernel(const MergeParams p) {
  // the attention kernel has finished: re-arm the work counter so that the same
  // plan can serve the next run
  if (blockIdx.x == 0 && threadIdx.x == 0) p.hdr->counter = 0;
  // one thread reads the header (a plan with no split groups leaves at once)
  __shared__ int s_groups;
  if (threadIdx.x == 0) s_groups = sig_equal(p.hdr->sig, p.sig) ? p.hdr->n_groups : 0;
  __syncthreads();
  if (s_groups <= 0) return;
  constexpr int kBlocks = kUnitRows / kMergeRows;
  const int64_t n_items = static_cast<int64_t>(s_groups) * kBlocks;
  const int lane = threadIdx.x & 31;
  const int64_t warps = static_cast<int64_t>(gridDim.x) * (kMergeThreads / 32);
  for (int64_t it = static_cast<int64_t>(blockIdx.x) * (kMergeThreads / 32) + threadIdx.x / 32; it < n_items;
       it += warps) {
    const MergeGroup grp = p.groups[it / kBlocks];
    if (grp.seq < 0 || grp.seq >= p.batch) continue;
    merge_rows_warp<D>(p, grp, static_cast<int>(it % kBlocks) * kMergeRows, lane);
  }
}

// ------------------------------------------------------------------ host side
struct DeviceInfo {
  int num_sms = 0;
  bool attr_set[4] = {false, false, false, false};
};

DeviceInfo* device_info(int dev) {
  static DeviceInfo info[64];
  static std::mutex mu;
  if (dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  DeviceInfo& d = info[dev];
  if (d.num_sms == 0) {
    if (cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) d.num_sms = 0;
  }
  return &d;
}

template <int D, bool kMask>
bool ensure_smem_attr(DeviceInfo* di) {
  const int idx = (D == 128 ? 1 : 0) + (kMask ? 2 : 0);
  if (!di->attr_set[idx]) {
    if (cudaFuncSetAttribute(attn_kernel<D, kMask>, cudaFuncAttributeMaxDynamicSharedMemorySize, Smem<D>::kBytes) !=
        cudaSuccess)
      return false;
    di->attr_set[idx] = true;
  }
  return true;
}

inline bool pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }

mbe_status check_shapes(int32_t batch, int32_t Hq, int32_t Hkv, int32_t D, int32_t max_window, int32_t max_prefix) {
  if (batch < 0 || Hq < 1 || Hkv < 1 || max_window < 0 || max_prefix < 0) return MBE_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return MBE_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return MBE_ERR_UNSUPPORTED;
  const int G = Hq / Hkv;
  if (!pow2(G) || G > kTileRows || Hkv > 0xFFFF) return MBE_ERR_UNSUPPORTED;
  if (max_window > (1 << 20) || max_prefix > (1 << 28)) return MBE_ERR_UNSUPPORTED;
  return MBE_OK;
}

// Block mask of the block-mask mode (null otherwise).
struct MaskArgs {
  const uint32_t* bits = nullptr;
  int rows = 0, words = 0;
};

template <int D, bool kMask>
mbe_status run(const void* q, const void* k_win, const void* v_win, const void* k_cache, const void* v_cache,
               int32_t num_pages, const int32_t* block_table, int32_t max_pages, const int32_t* prefix_len,
               const int32_t* window_len, const int32_t* cu_window, const uint8_t* mask_mode, int32_t batch,
               int32_t total_q_tokens, int32_t Hq, int32_t Hkv, int32_t block_size, int32_t page_size,
               int32_t max_window, int32_t max_prefix, float scale, void* out, float* lse, void* workspace,
               const Layout& L, DeviceInfo* di, bool with_plan, const MaskArgs& mask, cudaStream_t stream) {
  const int G = Hq / Hkv;
  CUtensorMap tq, tkw, tvw, tkc, tvc;
  {
    const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hq, (cuuint64_t)total_q_tokens};
    const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hq * D * 2};
    const cuuint32_t box[3] = {64, (cuuint32_t)G, (cuuint32_t)(kTileRows / G)};
    if (!encode_bf16_sw128(&tq, q, 3, dims, strides, box)) return MBE_ERR_CUDA;
  }
  {
    const cuuint64_t dims[3] = {(cuuint64_t)D, (cuuint64_t)Hkv, (cuuint64_t)total_q_tokens};
    const cuuint64_t strides[2] = {(cuuint64_t)D * 2, (cuuint64_t)Hkv * D * 2};
    const cuuint32_t box[3] = {64, 1, (cuuint32_t)kTileKeys};
    if (!encode_bf16_sw128(&tkw, k_win, 3, dims, strides, box) ||
        !encode_bf16_sw128(&tvw, v_win, 3, dims, strides, box))
      return MBE_ERR_CUDA;
  }
  const int box_rows = std::min(page_size, kTileKeys);
  {
    const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)page_size, (cuuint64_t)Hkv, (cuuint64_t)num_pages};
    const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)page_size * D * 2,
                                   (cuuint64_t)Hkv * page_size * D * 2};
    const cuuint32_t box[4] = {64, (cuuint32_t)box_rows, 1, 1};
    if (!encode_bf16_sw128(&tkc, k_cache, 4, dims, strides, box) ||
        !encode_bf16_sw128(&tvc, v_cache, 4, dims, strides, box))
      return MBE_ERR_CUDA;
  }
  if (!ensure_smem_attr<D, kMask>(di)) {
    record_cuda_error(cudaGetLastError(), "cudaFuncSetAttribute(attn_kernel)");
    return MBE_ERR_CUDA;
  }
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  Header* hdr = reinterpret_cast<Header*>(ws);
  const PlanSig sig = make_sig(batch, total_q_tokens, G, Hkv, D, block_size, max_window, max_prefix);
  SchedParams sp{prefix_len, window_len, mask_mode, cu_window, batch, G, Hkv, block_size, max_window, max_prefix,
                 di->num_sms, total_q_tokens, kMask, sig, hdr, reinterpret_cast<WorkUnit*>(ws + L.units_tmp),
                 reinterpret_cast<WorkUnit*>(ws + L.units), reinterpret_cast<MergeGroup*>(ws + L.groups), L.max_units,
                 L.max_groups, L.max_slots};
  if (with_plan) {
    attn_schedule_kernel<<<1, kBuckets, 0, stream>>>(sp);
    if (launch_status("attn_schedule_kernel launch") != MBE_OK) return MBE_ERR_CUDA;
  }
  AttnParams ap;
  ap.sig = sig;
  ap.batch = batch;
  ap.total_tokens = total_q_tokens;
  ap.block_table = block_table;
  ap.cu_window = cu_window;
  ap.out = static_cast<__nv_bfloat16*>(out);
  ap.lse = lse;
  ap.hdr = hdr;
  ap.units = reinterpret_cast<const WorkUnit*>(ws + L.units);
  ap.part_o = reinterpret_cast<float*>(ws + L.part_o);
  ap.part_lse = reinterpret_cast<float*>(ws + L.part_lse);
  ap.max_pages = max_pages;
  ap.num_pages = num_pages;
  ap.Hq = Hq;
  ap.G = G;
  ap.block_size = block_size;
  ap.page_size = page_size;
  ap.box_rows = box_rows;
  ap.loads_per_tile = kTileKeys / box_rows;
  ap.scale_log2 = scale * 1.4426950408889634f;
  ap.mask = mask.bits;
  ap.mask_rows = mask.rows;
  ap.mask_words = mask.words;
  ap.block_log2 = 0;
  while ((1 << ap.block_log2) < block_size) ++ap.block_log2;
  ap.wait_ns = wait_limit_ns();
  attn_kernel<D, kMask><<<di->num_sms, kThreads, Smem<D>::kBytes, stream>>>(tq, tkw, tvw, tkc, tvc, ap);
  if (launch_status("attn_kernel launch") != MBE_OK) return MBE_ERR_CUDA;
  MergeParams mp{sig, batch, total_q_tokens, hdr, reinterpret_cast<const MergeGroup*>(ws + L.groups), ap.part_o,
                 ap.part_lse, cu_window, ap.out, lse, Hq, G};
  const int64_t merge_grid = std::max<int64_t>(
      1, std::min<int64_t>(L.max_groups * (kUnitRows / kMergeRows / (kMergeThreads / 32)), 2 * di->num_sms));
  attn_merge_kernel<D><<<static_cast<unsigned>(merge_grid), kMergeThreads, 0, stream>>>(mp);
  if (launch_status("attn_merge_kernel launch") != MBE_OK) return MBE_ERR_CUDA;
  return MBE_OK;
}

}  // namespace attn
}  // namespace mbe

using namespace mbe;
using namespace mbe::attn;

extern "C" size_t mbe_window_attention_workspace_size(int32_t batch, int32_t num_q_heads, int32_t num_kv_heads,
                                                      int32_t head_dim, int32_t max_window, int32_t max_prefix) {
  if (check_shapes(batch, num_q_heads, num_kv_heads, head_dim, max_window, max_prefix) != MBE_OK) return 0;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  DeviceInfo* di = device_info(dev);
  if (!di || di->num_sms <= 0) return 0;
  return make_layout(batch, num_q_heads, num_kv_heads, head_dim, max_window, max_prefix, di->num_sms).total;
}

namespace {

struct Checked {
  Layout L;
  DeviceInfo* di;
  float scale;
};

// Host-side validation shared by the attention entry points; st == MBE_OK with
// nothing_to_do set means the call is a no-op.
mbe_status check_call(int32_t num_pages, int32_t max_pages_per_seq, int32_t batch, int32_t total_q_tokens,
                      int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim, int32_t block_size,
                      int32_t page_size, int32_t max_window, int32_t max_prefix, float softmax_scale,
                      void* workspace, size_t workspace_bytes, bool pointers_ok, bool& nothing_to_do, Checked& c) {
  nothing_to_do = false;
  mbe_status st = check_shapes(batch, num_q_heads, num_kv_heads, head_dim, max_window, max_prefix);
  if (st != MBE_OK) return st;
  if (block_size < 1 || total_q_tokens < 0 || num_pages < 1 || max_pages_per_seq < 1) return MBE_ERR_INVALID_ARG;
  if (!pow2(page_size) || page_size < 8) return MBE_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(max_pages_per_seq) * page_size < max_prefix) return MBE_ERR_INVALID_ARG;
  if (!(softmax_scale >= 0.f) || std::isinf(softmax_scale)) return MBE_ERR_INVALID_ARG;
  if (batch == 0 || total_q_tokens == 0 || max_window == 0) {
    nothing_to_do = true;
    return MBE_OK;
  }
  if (!pointers_ok) return MBE_ERR_INVALID_ARG;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return MBE_ERR_CUDA;
  c.di = device_info(dev);
  if (!c.di || c.di->num_sms <= 0) return MBE_ERR_CUDA;
  c.L = make_layout(batch, num_q_heads, num_kv_heads, head_dim, max_window, max_prefix, c.di->num_sms);
  if (!workspace || workspace_bytes < c.L.total || !aligned16(workspace)) return MBE_ERR_WORKSPACE;
  if (c.L.max_groups > 0x7FFFFFFF) return MBE_ERR_UNSUPPORTED;
  c.scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt(static_cast<float>(head_dim));
  return MBE_OK;
}

mbe_status attention_call(const void* q, const void* k_win, const void* v_win, const void* k_cache, const void* v_cache,
                          int32_t num_pages, const int32_t* block_table, int32_t max_pages_per_seq,
                          const int32_t* prefix_len, const int32_t* window_len, const int32_t* cu_window,
                          const uint8_t* mask_mode, int32_t batch, int32_t total_q_tokens, int32_t num_q_heads,
                          int32_t num_kv_heads, int32_t head_dim, int32_t block_size, int32_t page_size,
                          int32_t max_window, int32_t max_prefix, float softmax_scale, void* out, float* lse_or_null,
                          void* workspace, size_t workspace_bytes, bool with_plan, cudaStream_t stream) {
  bool noop = false;
  Checked c;
  const bool pointers_ok = q && k_win && v_win && k_cache && v_cache && block_table && prefix_len && window_len &&
                           cu_window && mask_mode && out && aligned16(q) && aligned16(k_win) && aligned16(v_win) &&
                           aligned16(k_cache) && aligned16(v_cache) && aligned16(out);
  mbe_status st = check_call(num_pages, max_pages_per_seq, batch, total_q_tokens, num_q_heads, num_kv_heads, head_dim,
                             block_size, page_size, max_window, max_prefix, softmax_scale, workspace, workspace_bytes,
                             pointers_ok, noop, c);
  if (st != MBE_OK || noop) return st;
  if (head_dim == 128)
    return run<128, false>(q, k_win, v_win, k_cache, v_cache, num_pages, block_table, max_pages_per_seq, prefix_len,
                    window_len, cu_window, mask_mode, batch, total_q_tokens, num_q_heads, num_kv_heads, block_size,
                    page_size, max_window, max_prefix, c.scale, out, lse_or_null, workspace, c.L, c.di, with_plan,
                    MaskArgs{}, stream);
  return run<64, false>(q, k_win, v_win, k_cache, v_cache, num_pages, block_table, max_pages_per_seq, prefix_len, window_len,
                 cu_window, mask_mode, batch, total_q_tokens, num_q_heads, num_kv_heads, block_size, page_size,
                 max_window, max_prefix, c.scale, out, lse_or_null, workspace, c.L, c.di, with_plan, MaskArgs{},
                 stream);
}

}  // namespace

extern "C" mbe_status mbe_window_attention(const void* q, const void* k_win, const void* v_win, const void* k_cache,
                                           const void* v_cache, int32_t num_pages, const int32_t* block_table,
                                           int32_t max_pages_per_seq, const int32_t* prefix_len,
                                           const int32_t* window_len, const int32_t* cu_window,
                                           const uint8_t* mask_mode, int32_t batch, int32_t total_q_tokens,
                                           int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                           int32_t block_size, int32_t page_size, int32_t max_window,
                                           int32_t max_prefix, float softmax_scale, void* out, float* lse_or_null,
                                           void* workspace, size_t workspace_bytes, cudaStream_t stream) {
  return attention_call(q, k_win, v_win, k_cache, v_cache, num_pages, block_table, max_pages_per_seq, prefix_len,
                        window_len, cu_window, mask_mode, batch, total_q_tokens, num_q_heads, num_kv_heads, head_dim,
                        block_size, page_size, max_window, max_prefix, softmax_scale, out, lse_or_null, workspace,
                        workspace_bytes, true, stream);
}

extern "C" mbe_status mbe_window_attention_plan(const int32_t* prefix_len, const int32_t* window_len,
                                                const int32_t* cu_window, const uint8_t* mask_mode, int32_t batch,
                                                int32_t total_q_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                                int32_t head_dim, int32_t block_size, int32_t max_window,
                                                int32_t max_prefix, void* workspace, size_t workspace_bytes,
                                                cudaStream_t stream) {
  bool noop = false;
  Checked c;
  // page geometry does not enter the plan: pass a page size and table width that always validate
  const bool pointers_ok = prefix_len && window_len && cu_window && mask_mode;
  mbe_status st = check_call(1, max_prefix > 0 ? max_prefix : 1, batch, total_q_tokens, num_q_heads, num_kv_heads,
                             head_dim, block_size, 8, max_window, max_prefix, 0.f, workspace, workspace_bytes,
                             pointers_ok, noop, c);
  if (st != MBE_OK || noop) return st;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const PlanSig sig = make_sig(batch, total_q_tokens, num_q_heads / num_kv_heads, num_kv_heads, head_dim, block_size,
                               max_window, max_prefix);
  SchedParams sp{prefix_len, window_len, mask_mode, cu_window, batch, num_q_heads / num_kv_heads, num_kv_heads,
                 block_size, max_window, max_prefix, c.di->num_sms, total_q_tokens, false, sig, reinterpret_cast<Header*>(ws),
                 reinterpret_cast<WorkUnit*>(ws + c.L.units_tmp), reinterpret_cast<WorkUnit*>(ws + c.L.units),
                 reinterpret_cast<MergeGroup*>(ws + c.L.groups), c.L.max_units, c.L.max_groups, c.L.max_slots};
  attn_schedule_kernel<<<1, kBuckets, 0, stream>>>(sp);
  return launch_status("attn_schedule_kernel launch");
}

extern "C" mbe_status mbe_window_attention_run(const void* q, const void* k_win, const void* v_win,
                                               const void* k_cache, const void* v_cache, int32_t num_pages,
                                               const int32_t* block_table, int32_t max_pages_per_seq,
                                               const int32_t* prefix_len, const int32_t* window_len,
                                               const int32_t* cu_window, const uint8_t* mask_mode, int32_t batch,
                                               int32_t total_q_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                               int32_t head_dim, int32_t block_size, int32_t page_size,
                                               int32_t max_window, int32_t max_prefix, float softmax_scale, void* out,
                                               float* lse_or_null, void* workspace, size_t workspace_bytes,
                                               cudaStream_t stream) {
  return attention_call(q, k_win, v_win, k_cache, v_cache, num_pages, block_table, max_pages_per_seq, prefix_len,
                        window_len, cu_window, mask_mode, batch, total_q_tokens, num_q_heads, num_kv_heads, head_dim,
                        block_size, page_size, max_window, max_prefix, softmax_scale, out, lse_or_null, workspace,
                        workspace_bytes, false, stream);
}

extern "C" mbe_status mbe_window_attention_plan_stats(const void* workspace, size_t workspace_bytes, int32_t* n_units,
                                                      int32_t* n_split_groups, cudaStream_t stream) {
  if (!workspace || workspace_bytes < sizeof(Header) || !n_units || !n_split_groups) return MBE_ERR_INVALID_ARG;
  int32_t h[3] = {0, 0, 0};
  if (cudaMemcpyAsync(h, workspace, sizeof(h), cudaMemcpyDeviceToHost, stream) != cudaSuccess ||
      cudaStreamSynchronize(stream) != cudaSuccess) {
    record_cuda_error(cudaGetLastError(), "mbe_window_attention_plan_stats");
    return MBE_ERR_CUDA;
  }
  *n_units = h[1];
  *n_split_groups = h[2];
  return MBE_OK;
}

// ------------------------------------------------------------------ no-allocation variant
// Scratch for mbe_window_attention_noalloc: a fixed device array that every
// GPU loading this library holds until the process exits. Host code must not
// pass the symbol itself to a kernel (on the host it is only a stand-in); the
// device address is looked up once per device with cudaGetSymbolAddress.
namespace mbe {
namespace attn {
constexpr size_t kNoAllocScratchBytes = size_t(64) << 20;  // 64 MiB
}  // namespace attn
}  // namespace mbe

static __device__ __align__(256) uint8_t g_noalloc_scratch[mbe::attn::kNoAllocScratchBytes];

namespace {

// Device address of g_noalloc_scratch on device `dev` (looked up on the first
// call made with that device current), or nullptr if the lookup failed.
void* noalloc_scratch(int dev) {
  static void* addr[64] = {};
  static std::mutex mu;
  if (dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess) return nullptr;
    addr[dev] = p;
  }
  return addr[dev];
}

}  // namespace

extern "C" mbe_status mbe_window_attention_noalloc(const void* q, const void* k_win, const void* v_win,
                                                   const void* k_cache, const void* v_cache, int32_t num_pages,
                                                   const int32_t* block_table, int32_t max_pages_per_seq,
                                                   const int32_t* prefix_len, const int32_t* window_len,
                                                   const int32_t* cu_window, const uint8_t* mask_mode, int32_t batch,
                                                   int32_t total_q_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                                   int32_t head_dim, int32_t block_size, int32_t page_size,
                                                   int32_t max_window, int32_t max_prefix, float softmax_scale,
                                                   void* out, float* lse_or_null, cudaStream_t stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return MBE_ERR_CUDA;
  void* scratch = noalloc_scratch(dev);
  if (scratch == nullptr) return MBE_ERR_CUDA;
  // The regular entry point checks the bounds against the scratch size and
  // returns MBE_ERR_WORKSPACE, launching nothing, when they need more.
  return mbe_window_attention(q, k_win, v_win, k_cache, v_cache, num_pages, block_table, max_pages_per_seq,
                              prefix_len, window_len, cu_window, mask_mode, batch, total_q_tokens, num_q_heads,
                              num_kv_heads, head_dim, block_size, page_size, max_window, max_prefix, softmax_scale,
                              out, lse_or_null, scratch, mbe::attn::kNoAllocScratchBytes, stream);
}

extern "C" mbe_status mbe_block_mask_attention(const void* q, const void* k, const void* v, const int32_t* seq_len,
                                               const int32_t* cu_seqlens, const uint32_t* mask, int32_t mask_rows,
                                               int32_t mask_words, int32_t batch, int32_t total_tokens,
                                               int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                               int32_t block_size, int32_t max_seq_len, float softmax_scale,
                                               void* out, float* lse_or_null, void* workspace,
                                               size_t workspace_bytes, cudaStream_t stream) {
  if (block_size < 8 || (block_size & (block_size - 1)) != 0 || mask_rows < 1 || mask_words < 1 ||
      static_cast<int64_t>(mask_words) * 32 < mask_rows || max_seq_len < 0)
    return MBE_ERR_INVALID_ARG;
  if (max_seq_len > kMaskTileWords * 32 * kTileKeys) return MBE_ERR_UNSUPPORTED;
  if ((max_seq_len + block_size - 1) / block_size > mask_rows) return MBE_ERR_INVALID_ARG;
  bool noop = false;
  Checked c;
  const bool pointers_ok = q && k && v && seq_len && cu_seqlens && mask && out && aligned16(q) && aligned16(k) &&
                           aligned16(v) && aligned16(out);
  mbe_status st = check_call(1, 1, batch, total_tokens, num_q_heads, num_kv_heads, head_dim, block_size, kTileKeys,
                             max_seq_len, 0, softmax_scale, workspace, workspace_bytes, pointers_ok, noop, c);
  if (st != MBE_OK || noop) return st;
  const MaskArgs ma{mask, mask_rows, mask_words};
  // the sequence is the window; the (unused) paged-cache maps point at k / v
  if (head_dim == 128)
    return run<128, true>(q, k, v, k, v, 1, nullptr, 1, nullptr, seq_len, cu_seqlens, nullptr, batch, total_tokens,
                          num_q_heads, num_kv_heads, block_size, kTileKeys, max_seq_len, 0, c.scale, out, lse_or_null,
                          workspace, c.L, c.di, true, ma, stream);
  return run<64, true>(q, k, v, k, v, 1, nullptr, 1, nullptr, seq_len, cu_seqlens, nullptr, batch, total_tokens,
                       num_q_heads, num_kv_heads, block_size, kTileKeys, max_seq_len, 0, c.scale, out, lse_or_null,
                       workspace, c.L, c.di, true, ma, stream);
}
