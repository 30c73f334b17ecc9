// Targeted refresh (Sec. 4.3) and the device-side editing-pass loop.
//
// refresh_plan_kernel turns the changed-block flags of a pass into a ragged
// batch of one-block attention problems (one per changed window block, prefix
// P + b*B, bidirectional inside the block), which the attention and KV-write
// kernels consume unchanged: no host round trip, so the whole pass can be
// captured in a CUDA graph. gather_rows_kernel compacts per-row inputs for that
// batch. The pass loop wraps a captured pass in a conditional WHILE graph node
// whose condition a one-CTA kernel sets from the per-sequence change counts
// (Sec. 4.1: stop when a pass changes no token, or after N_MBE passes).
#include "common.cuh"

namespace mbe {

MBE_DEFINE_ERROR_WORD(refresh_take_error)

namespace {

constexpr int kScanThreads = 1024;
constexpr int kTableThreads = 256;

// Window length of entry e = s * max_blocks + b, or 0 if block b of s did not
// change (or lies past the window). Sets *bad for an invalid window length.
__device__ __forceinline__ int entry_len(const uint8_t* __restrict__ changed, const int32_t* __restrict__ window_len,
                                         int e, int max_blocks, int block_size, int max_window, bool* bad) {
  const int s = e / max_blocks, b = e - s * max_blocks;
  const int W = window_len[s];
  if (W < 0 || W > max_window || W > max_blocks * block_size) {
    *bad = true;
    return 0;
  }
  const int start = b * block_size;
  if (!changed[e] || start >= W) return 0;
  return min(block_size, W - start);
}

// CTA 0 scans the entry lengths and writes the per-entry descriptors and the
// row map; the other CTAs copy block-table rows (the only part whose size
// scales with the page count).
__global__ void __launch_bounds__(kScanThreads) refresh_plan_kernel(
    const uint8_t* __restrict__ changed, int max_blocks, const int32_t* __restrict__ prefix_len,
    const int32_t* __restrict__ window_len, const int32_t* __restrict__ cu_window,
    const int32_t* __restrict__ block_table, int max_pages, int batch, int block_size, int max_window, int total_rows,
    int32_t* __restrict__ r_prefix_len, int32_t* __restrict__ r_window_len, int32_t* __restrict__ r_cu_window,
    uint8_t* __restrict__ r_mask_mode, int32_t* __restrict__ r_block_table, int32_t* __restrict__ r_src_row,
    int32_t* __restrict__ r_count) {
  const int E = batch * max_blocks;
  if (blockIdx.x > 0) {
    // block tables: entry e gets its sequence's row if it changed, -1 otherwise
    const int64_t total = static_cast<int64_t>(E) * max_pages;
    const int64_t stride = static_cast<int64_t>(gridDim.x - 1) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x - 1) * blockDim.x + threadIdx.x; i < total; i += stride) {
      const int e = static_cast<int>(i / max_pages), p = static_cast<int>(i - static_cast<int64_t>(e) * max_pages);
      bool bad = false;
      const int len = entry_len(changed, window_len, e, max_blocks, block_size, max_window, &bad);
      r_block_table[i] = len > 0 ? block_table[static_cast<int64_t>(e / max_blocks) * max_pages + p] : -1;
    }
    return;
  }
  __shared__ int warp_sums[kScanThreads / 32];
  __shared__ int chunk_total;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  bool bad = false, over = false;
  int carry = 0, entries = 0;
  for (int base = 0; base < E; base += kScanThreads) {
    const int e = base + threadIdx.x;
    const int len = e < E ? entry_len(changed, window_len, e, max_blocks, block_size, max_window, &bad) : 0;
    // block-wide inclusive scan of len: warp shuffles, then the warp totals
    int x = len;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = lane < kScanThreads / 32 ? warp_sums[lane] : 0;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      if (lane < kScanThreads / 32) warp_sums[lane] = w;
      if (lane == kScanThreads / 32 - 1) chunk_total = w;
    }
    __syncthreads();
    const int start = carry + x - len + (warp > 0 ? warp_sums[warp - 1] : 0);
    entries += __syncthreads_count(len > 0);
    if (e < E) {
      const int s = e / max_blocks, b = e - s * max_blocks;
      r_cu_window[e] = start;
      r_prefix_len[e] = len > 0 ? prefix_len[s] + b * block_size : 0;
      r_window_len[e] = len;
      r_mask_mode[e] = MBE_MULTI_BLOCK_BIDIRECTIONAL;
      const int src0 = len > 0 ? cu_window[s] + b * block_size : 0;
      for (int i = 0; i < len; ++i) {
        if (start + i < total_rows)
          r_src_row[start + i] = src0 + i;
        else
          over = true;
      }
    }
    carry += chunk_total;
    __syncthreads();  // warp_sums / chunk_total are rewritten by the next chunk
  }
  for (int k = carry + threadIdx.x; k < total_rows; k += blockDim.x) r_src_row[k] = -1;
  const bool any_bad = __syncthreads_or(bad), any_over = __syncthreads_or(over);
  if (threadIdx.x == 0) {
    r_cu_window[E] = carry;
    r_count[0] = entries;
    r_count[1] = carry;
    if (any_bad) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
    if (any_over) atomicOr(&g_error_word, MBE_DEVERR_CAPACITY);
  }
}

// dst row k = src row map[k]; zeros where map[k] < 0; zeros and a device flag
// where map[k] >= src_rows; rows from *rows_used on (if given) untouched. V is
// the copy width (16, 4 or 1 bytes).
template <typename V>
__global__ void __launch_bounds__(256) gather_rows_kernel(const V* __restrict__ src, int64_t src_rows,
                                                          int64_t row_elems, const int32_t* __restrict__ map,
                                                          int64_t rows, const int32_t* __restrict__ rows_used,
                                                          V* __restrict__ dst) {
  if (rows_used) rows = min(rows, static_cast<int64_t>(max(*rows_used, 0)));
  const int64_t total = rows * row_elems;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += stride) {
    const int64_t k = i / row_elems, c = i - k * row_elems;
    const int32_t r = map[k];
    V v{};
    if (r >= 0 && r < src_rows)
      v = src[r * row_elems + c];
    else if (r >= src_rows && c == 0)
      atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
    dst[i] = v;
  }
}

// The same for up to MBE_GATHER_MAX tensors sharing one row map, 16-byte
// chunks: chunk c of a destination row belongs to tensor t where
// off[t] <= c < off[t + 1] (off[t] = chunks per row of the tensors before t).
struct GatherSet {
  const uint4* src[MBE_GATHER_MAX];
  uint4* dst[MBE_GATHER_MAX];
  int64_t elems[MBE_GATHER_MAX];     // 16-byte chunks per row of tensor t
  int64_t off[MBE_GATHER_MAX + 1];
  int n;
};

__global__ void __launch_bounds__(256) gather_rows_multi_kernel(const GatherSet g, int64_t src_rows,
                                                                const int32_t* __restrict__ map, int64_t rows,
                                                                const int32_t* __restrict__ rows_used) {
  if (rows_used) rows = min(rows, static_cast<int64_t>(max(*rows_used, 0)));
  const int64_t per_row = g.off[g.n];
  const int64_t total = rows * per_row;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += stride) {
    const int64_t k = i / per_row, c = i - k * per_row;
    int t = 0;
#pragma unroll
    for (int u = 1; u < MBE_GATHER_MAX; ++u) t += (u < g.n && c >= g.off[u]) ? 1 : 0;
    const int64_t cc = c - g.off[t];
    const int32_t r = map[k];
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (r >= 0 && r < src_rows)
      v = g.src[t][r * g.elems[t] + cc];
    else if (r >= src_rows && c == 0)
      atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
    g.dst[t][k * g.elems[t] + cc] = v;
  }
}

// The per-layer row work of the refresh in one launch: refresh row k (k <
// *rows_used) is copied from source row src_row[k] of q / k_win / v_win into
// the compact q_out / k_out / v_out, and its K and V go into the paged cache at
// its refresh-layout position: entry e (the largest e with r_cu[e] <= k) row
// i = k - r_cu[e] sits at r_prefix[e] + i of block-table row e. One CTA per row
// at a time (grid-stride); chunks are 16 bytes.
__global__ void __launch_bounds__(256) refresh_rows_kernel(
    const uint4* __restrict__ q, const uint4* __restrict__ kw, const uint4* __restrict__ vw, int64_t src_rows,
    const int32_t* __restrict__ src_row, const int32_t* __restrict__ rows_used, int64_t rows,
    const int32_t* __restrict__ r_prefix, const int32_t* __restrict__ r_cu, const int32_t* __restrict__ r_bt,
    int E, int max_pages, uint4* __restrict__ k_cache, uint4* __restrict__ v_cache, int num_pages, int page_size,
    int q_chunks, int kv_chunks, int chunks_per_head, int Hkv, uint4* __restrict__ q_out, uint4* __restrict__ k_out,
    uint4* __restrict__ v_out) {
  __shared__ int64_t s_dst;  // cache offset (in chunks) of head 0 of this row's slot; -1: no cache write
  if (rows_used) rows = min(rows, static_cast<int64_t>(max(*rows_used, 0)));
  const int per_row = q_chunks + 2 * kv_chunks;
  for (int64_t k = blockIdx.x; k < rows; k += gridDim.x) {
    const int32_t r = src_row[k];
    const bool have = r >= 0 && r < src_rows;
    if (threadIdx.x == 0) {
      int64_t dst = -1;
      if (r >= src_rows) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
      if (have && E > 0) {
        int lo = 0, hi = E - 1;  // the largest e with r_cu[e] <= k
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (r_cu[mid] <= k) lo = mid; else hi = mid - 1;
        }
        const int64_t pos = static_cast<int64_t>(r_prefix[lo]) + (k - r_cu[lo]);
        const int64_t lp = pos / page_size;
        const int page = (lp >= 0 && lp < max_pages) ? r_bt[static_cast<int64_t>(lo) * max_pages + lp] : -2;
        if (k < r_cu[lo] || k >= r_cu[lo + 1] || lp < 0 || lp >= max_pages) {
          // a row outside every entry (row count and layout disagree) or past its block-table row
          atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
        } else if (page < 0 || page >= num_pages) {
          atomicOr(&g_error_word, MBE_DEVERR_PAGE);
        } else {
          dst = (static_cast<int64_t>(page) * Hkv * page_size + pos % page_size) * chunks_per_head;
        }
      }
      s_dst = dst;
    }
    __syncthreads();
    const int64_t dst = s_dst;
    for (int c = threadIdx.x; c < per_row; c += blockDim.x) {
      uint4 x = make_uint4(0u, 0u, 0u, 0u);
      if (c < q_chunks) {
        if (have) x = q[static_cast<int64_t>(r) * q_chunks + c];
        q_out[k * q_chunks + c] = x;
        continue;
      }
      const int kv = (c - q_chunks) >= kv_chunks ? 1 : 0;
      const int cc = c - q_chunks - kv * kv_chunks;
      if (have) x = (kv ? vw : kw)[static_cast<int64_t>(r) * kv_chunks + cc];
      (kv ? v_out : k_out)[k * kv_chunks + cc] = x;
      if (dst >= 0) {
        // head g of the slot: pages are [Hkv, page_size, D]
        const int g = cc / chunks_per_head, w = cc - g * chunks_per_head;
        (kv ? v_cache : k_cache)[dst + static_cast<int64_t>(g) * page_size * chunks_per_head + w] = x;
      }
    }
    __syncthreads();  // s_dst is rewritten for the next row
  }
}

// Ends a pass: counts it and keeps the loop going while some sequence changed
// a token and fewer than max_passes passes have run.
__global__ void __launch_bounds__(256) pass_loop_condition_kernel(cudaGraphConditionalHandle handle,
                                                                  const int32_t* __restrict__ seq_changes,
                                                                  int num_seqs, int32_t* passes_done,
                                                                  int max_passes) {
  bool changed = false;
  for (int s = threadIdx.x; s < num_seqs; s += blockDim.x) changed |= seq_changes[s] != 0;
  const bool any = __syncthreads_or(changed);
  if (threadIdx.x == 0) {
    const int done = *passes_done + 1;
    *passes_done = done;
    cudaGraphSetConditional(handle, (any && done < max_passes) ? 1u : 0u);
  }
}

int sm_count() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) !=
                                               cudaSuccess)
    return 0;
  return n;
}

}  // namespace
}  // namespace mbe

extern "C" mbe_status mbe_refresh_plan(const uint8_t* block_changed, int32_t max_blocks_per_seq,
                                       const int32_t* prefix_len, const int32_t* window_len,
                                       const int32_t* cu_window, const int32_t* block_table,
                                       int32_t max_pages_per_seq, int32_t batch, int32_t block_size,
                                       int32_t max_window, int32_t total_rows, int32_t* r_prefix_len,
                                       int32_t* r_window_len, int32_t* r_cu_window, uint8_t* r_mask_mode,
                                       int32_t* r_block_table, int32_t* r_src_row, int32_t* r_count,
                                       cudaStream_t stream) {
  using namespace mbe;
  if (batch < 0 || max_blocks_per_seq < 1 || max_pages_per_seq < 1 || block_size < 1 || max_window < 0 ||
      total_rows < 0)
    return MBE_ERR_INVALID_ARG;
  if (static_cast<int64_t>(batch) * max_blocks_per_seq > (1 << 24) ||
      static_cast<int64_t>(max_blocks_per_seq) * block_size > (1 << 30))
    return MBE_ERR_UNSUPPORTED;
  if (!r_cu_window || !r_count || (total_rows > 0 && !r_src_row)) return MBE_ERR_INVALID_ARG;
  if (batch > 0 && (!block_changed || !prefix_len || !window_len || !cu_window || !block_table || !r_prefix_len ||
                    !r_window_len || !r_mask_mode || !r_block_table))
    return MBE_ERR_INVALID_ARG;
  const int sms = sm_count();
  if (sms == 0) {
    record_cuda_error(cudaGetLastError(), "cudaDeviceGetAttribute");
    return MBE_ERR_CUDA;
  }
  const int64_t table = static_cast<int64_t>(batch) * max_blocks_per_seq * max_pages_per_seq;
  int64_t table_ctas = (table + 8 * kTableThreads - 1) / (8 * kTableThreads);
  if (table_ctas > 2 * sms) table_ctas = 2 * sms;
  refresh_plan_kernel<<<static_cast<unsigned>(1 + table_ctas), kScanThreads, 0, stream>>>(
      block_changed, max_blocks_per_seq, prefix_len, window_len, cu_window, block_table, max_pages_per_seq, batch,
      block_size, max_window, total_rows, r_prefix_len, r_window_len, r_cu_window, r_mask_mode, r_block_table,
      r_src_row, r_count);
  return launch_status("refresh_plan_kernel");
}

extern "C" mbe_status mbe_gather_rows(const void* src, int64_t src_rows, int64_t row_bytes, const int32_t* src_row,
                                      int64_t rows, const int32_t* rows_used_or_null, void* dst,
                                      cudaStream_t stream) {
  using namespace mbe;
  if (src_rows < 0 || row_bytes < 1 || rows < 0) return MBE_ERR_INVALID_ARG;
  if (rows == 0) return MBE_OK;
  if (!src_row || !dst || (src_rows > 0 && !src)) return MBE_ERR_INVALID_ARG;
  const int sms = sm_count();
  if (sms == 0) {
    record_cuda_error(cudaGetLastError(), "cudaDeviceGetAttribute");
    return MBE_ERR_CUDA;
  }
  const uintptr_t a = reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst);
  const int width = (row_bytes % 16 == 0 && a % 16 == 0) ? 16 : (row_bytes % 4 == 0 && a % 4 == 0) ? 4 : 1;
  const int64_t elems = rows * (row_bytes / width);
  int64_t ctas = (elems + 255) / 256;
  if (ctas > 4 * sms) ctas = 4 * sms;
  const unsigned g = static_cast<unsigned>(ctas);
  if (width == 16)
    gather_rows_kernel<uint4><<<g, 256, 0, stream>>>(static_cast<const uint4*>(src), src_rows, row_bytes / 16,
                                                     src_row, rows, rows_used_or_null, static_cast<uint4*>(dst));
  else if (width == 4)
    gather_rows_kernel<uint32_t><<<g, 256, 0, stream>>>(static_cast<const uint32_t*>(src), src_rows, row_bytes / 4,
                                                        src_row, rows, rows_used_or_null,
                                                        static_cast<uint32_t*>(dst));
  else
    gather_rows_kernel<uint8_t><<<g, 256, 0, stream>>>(static_cast<const uint8_t*>(src), src_rows, row_bytes,
                                                       src_row, rows, rows_used_or_null, static_cast<uint8_t*>(dst));
  return launch_status("gather_rows_kernel");
}

extern "C" mbe_status mbe_gather_rows_multi(int32_t n_tensors, const void* const* srcs, const int64_t* row_bytes,
                                            void* const* dsts, int64_t src_rows, const int32_t* src_row,
                                            int64_t rows, const int32_t* rows_used_or_null, cudaStream_t stream) {
  using namespace mbe;
  if (n_tensors < 1 || n_tensors > MBE_GATHER_MAX || !srcs || !row_bytes || !dsts || src_rows < 0 || rows < 0)
    return MBE_ERR_INVALID_ARG;
  bool vec = true;
  for (int t = 0; t < n_tensors; ++t) {
    if (row_bytes[t] < 1 || !dsts[t] || (src_rows > 0 && !srcs[t])) return MBE_ERR_INVALID_ARG;
    const uintptr_t a = reinterpret_cast<uintptr_t>(srcs[t]) | reinterpret_cast<uintptr_t>(dsts[t]);
    vec &= row_bytes[t] % 16 == 0 && a % 16 == 0;
  }
  if (rows == 0) return MBE_OK;
  if (!src_row) return MBE_ERR_INVALID_ARG;
  if (!vec) {  // rows that are not whole 16-byte chunks: one copy per tensor
    for (int t = 0; t < n_tensors; ++t) {
      const mbe_status st =
          mbe_gather_rows(srcs[t], src_rows, row_bytes[t], src_row, rows, rows_used_or_null, dsts[t], stream);
      if (st != MBE_OK) return st;
    }
    return MBE_OK;
  }
  GatherSet g{};
  g.n = n_tensors;
  g.off[0] = 0;
  for (int t = 0; t < n_tensors; ++t) {
    g.src[t] = static_cast<const uint4*>(srcs[t]);
    g.dst[t] = static_cast<uint4*>(dsts[t]);
    g.elems[t] = row_bytes[t] / 16;
    g.off[t + 1] = g.off[t] + g.elems[t];
  }
  for (int t = n_tensors; t < MBE_GATHER_MAX; ++t) g.off[t + 1] = g.off[t];
  const int sms = sm_count();
  if (sms == 0) {
    record_cuda_error(cudaGetLastError(), "cudaDeviceGetAttribute");
    return MBE_ERR_CUDA;
  }
  int64_t ctas = (rows * g.off[n_tensors] + 255) / 256;
  if (ctas > 4 * sms) ctas = 4 * sms;
  gather_rows_multi_kernel<<<static_cast<unsigned>(ctas), 256, 0, stream>>>(g, src_rows, src_row, rows,
                                                                             rows_used_or_null);
  return launch_status("gather_rows_multi_kernel");
}

extern "C" mbe_status mbe_refresh_gather_write(
    const void* q, const void* k_win, const void* v_win, int64_t src_rows, int32_t num_q_heads,
    int32_t num_kv_heads, int32_t head_dim, const int32_t* src_row, const int32_t* rows_used_or_null, int64_t rows,
    const int32_t* r_prefix_len, const int32_t* r_cu_window, const int32_t* r_block_table, int32_t num_entries,
    int32_t max_pages_per_seq, void* k_cache, void* v_cache, int32_t num_pages, int32_t page_size, void* q_out,
    void* k_out, void* v_out, cudaStream_t stream) {
  using namespace mbe;
  if (src_rows < 0 || rows < 0 || num_q_heads < 1 || num_kv_heads < 1 || head_dim < 8 || head_dim % 8 != 0 ||
      num_entries < 0 || max_pages_per_seq < 1 || num_pages < 1 || page_size < 1)
    return MBE_ERR_INVALID_ARG;
  if (rows == 0) return MBE_OK;
  if (!src_row || !q_out || !k_out || !v_out || !k_cache || !v_cache || (src_rows > 0 && (!q || !k_win || !v_win)) ||
      (num_entries > 0 && (!r_prefix_len || !r_cu_window || !r_block_table)))
    return MBE_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_win) || !aligned16(v_win) || !aligned16(k_cache) || !aligned16(v_cache) ||
      !aligned16(q_out) || !aligned16(k_out) || !aligned16(v_out))
    return MBE_ERR_INVALID_ARG;
  const int sms = sm_count();
  if (sms == 0) {
    record_cuda_error(cudaGetLastError(), "cudaDeviceGetAttribute");
    return MBE_ERR_CUDA;
  }
  const int chunks_per_head = head_dim / 8;
  int64_t ctas = rows;
  if (ctas > 8 * sms) ctas = 8 * sms;
  refresh_rows_kernel<<<static_cast<unsigned>(ctas), 256, 0, stream>>>(
      static_cast<const uint4*>(q), static_cast<const uint4*>(k_win), static_cast<const uint4*>(v_win), src_rows,
      src_row, rows_used_or_null, rows, r_prefix_len, r_cu_window, r_block_table, num_entries, max_pages_per_seq,
      static_cast<uint4*>(k_cache), static_cast<uint4*>(v_cache), num_pages, page_size,
      num_q_heads * chunks_per_head, num_kv_heads * chunks_per_head, chunks_per_head, num_kv_heads,
      static_cast<uint4*>(q_out), static_cast<uint4*>(k_out), static_cast<uint4*>(v_out));
  return launch_status("refresh_rows_kernel");
}

struct mbe_pass_loop {
  cudaGraph_t graph = nullptr;
  cudaGraph_t body = nullptr;  // owned by graph (the WHILE node's body)
  cudaGraphExec_t exec = nullptr;
  cudaGraphConditionalHandle handle{};
  cudaStream_t stream = nullptr;
  int32_t* passes_done = nullptr;
  int32_t max_passes = 0;
  bool capturing = false;
  bool has_condition = false;
};

namespace {
mbe_status cuda_fail(cudaError_t e, const char* where) {
  mbe::record_cuda_error(e, where);
  return MBE_ERR_CUDA;
}
}  // namespace

extern "C" mbe_status mbe_pass_loop_begin(int32_t max_passes, int32_t* passes_done, cudaStream_t stream,
                                          mbe_pass_loop** loop_out) {
  if (!loop_out) return MBE_ERR_INVALID_ARG;
  *loop_out = nullptr;
  if (max_passes < 1 || !passes_done || stream == nullptr) return MBE_ERR_INVALID_ARG;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  cudaError_t e = cudaStreamIsCapturing(stream, &cs);
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamIsCapturing");
  if (cs != cudaStreamCaptureStatusNone) return MBE_ERR_INVALID_ARG;
  auto* L = new mbe_pass_loop;
  L->stream = stream;
  L->passes_done = passes_done;
  L->max_passes = max_passes;
  const char* where = "cudaGraphCreate";
  e = cudaGraphCreate(&L->graph, 0);
  cudaGraphNode_t reset = nullptr, loop = nullptr;
  if (e == cudaSuccess) {
    where = "cudaGraphAddMemsetNode";
    cudaMemsetParams mp = {};
    mp.dst = passes_done;
    mp.elementSize = sizeof(int32_t);
    mp.width = 1;
    mp.height = 1;
    mp.pitch = sizeof(int32_t);
    mp.value = 0;
    e = cudaGraphAddMemsetNode(&reset, L->graph, nullptr, 0, &mp);
  }
  if (e == cudaSuccess) {
    where = "cudaGraphConditionalHandleCreate";
    e = cudaGraphConditionalHandleCreate(&L->handle, L->graph, 1u, cudaGraphCondAssignDefault);
  }
  if (e == cudaSuccess) {
    where = "cudaGraphAddNode(conditional)";
    cudaGraphNodeParams np = {};
    np.type = cudaGraphNodeTypeConditional;
    np.conditional.handle = L->handle;
    np.conditional.type = cudaGraphCondTypeWhile;
    np.conditional.size = 1;
    e = cudaGraphAddNode(&loop, L->graph, &reset, nullptr, 1, &np);
    if (e == cudaSuccess) L->body = np.conditional.phGraph_out[0];
  }
  if (e == cudaSuccess) {
    where = "cudaStreamBeginCaptureToGraph";
    e = cudaStreamBeginCaptureToGraph(stream, L->body, nullptr, nullptr, 0, cudaStreamCaptureModeRelaxed);
  }
  if (e != cudaSuccess) {
    if (L->graph) cudaGraphDestroy(L->graph);
    delete L;
    return cuda_fail(e, where);
  }
  L->capturing = true;
  *loop_out = L;
  return MBE_OK;
}

extern "C" mbe_status mbe_pass_loop_until_stable(mbe_pass_loop* loop, const int32_t* seq_changes, int32_t num_seqs,
                                                 cudaStream_t stream) {
  if (!loop || !loop->capturing || stream != loop->stream || loop->has_condition || num_seqs < 0 ||
      (num_seqs > 0 && !seq_changes))
    return MBE_ERR_INVALID_ARG;
  mbe::pass_loop_condition_kernel<<<1, 256, 0, stream>>>(loop->handle, seq_changes, num_seqs, loop->passes_done,
                                                          loop->max_passes);
  const mbe_status st = mbe::launch_status("pass_loop_condition_kernel");
  if (st == MBE_OK) loop->has_condition = true;
  return st;
}

extern "C" mbe_status mbe_pass_loop_end(mbe_pass_loop* loop, cudaStream_t stream) {
  if (!loop || !loop->capturing || stream != loop->stream) return MBE_ERR_INVALID_ARG;
  cudaGraph_t captured = nullptr;
  cudaError_t e = cudaStreamEndCapture(stream, &captured);
  loop->capturing = false;
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamEndCapture");
  // without the condition kernel the WHILE body would never clear its condition
  if (!loop->has_condition) return MBE_ERR_INVALID_ARG;
  e = cudaGraphInstantiate(&loop->exec, loop->graph, 0);
  if (e != cudaSuccess) {
    loop->exec = nullptr;
    return cuda_fail(e, "cudaGraphInstantiate");
  }
  return MBE_OK;
}

extern "C" mbe_status mbe_pass_loop_launch(mbe_pass_loop* loop, cudaStream_t stream) {
  if (!loop || !loop->exec) return MBE_ERR_INVALID_ARG;
  const cudaError_t e = cudaGraphLaunch(loop->exec, stream);
  return e == cudaSuccess ? MBE_OK : cuda_fail(e, "cudaGraphLaunch");
}

extern "C" void mbe_pass_loop_destroy(mbe_pass_loop* loop) {
  if (!loop) return;
  if (loop->capturing) {
    cudaGraph_t g = nullptr;
    cudaStreamEndCapture(loop->stream, &g);
  }
  if (loop->exec) cudaGraphExecDestroy(loop->exec);
  if (loop->graph) cudaGraphDestroy(loop->graph);
  delete loop;
}
