// KV window write: the cache refresh of Sec. 4.3, as a coalesced page scatter.
//
// Grid (chunks, batch): every thread moves one 16-byte chunk of one window
// token's K and V for one KV head into its page slot. Consecutive threads cover
// consecutive chunks of a head row, so both the window read and the cache write
// are 16-byte vectorised and coalesced within each (token, head) row.
#include "common.cuh"

namespace mbe {

MBE_DEFINE_ERROR_WORD(kv_write_take_error)

namespace {

__global__ void __launch_bounds__(256) kv_window_write_kernel(
    const uint4* __restrict__ k_win, const uint4* __restrict__ v_win, uint4* __restrict__ k_cache,
    uint4* __restrict__ v_cache, int num_pages, const int32_t* __restrict__ block_table, int max_pages,
    const int32_t* __restrict__ prefix_len, const int32_t* __restrict__ window_len,
    const int32_t* __restrict__ cu_window, const uint8_t* __restrict__ block_mask, int max_blocks, int Hkv,
    int chunks_per_head, int block_size, int page_size, int max_window) {
  const int s = blockIdx.y;
  const int P = prefix_len[s], W = window_len[s], t0 = cu_window[s];
  if (W < 0 || W > max_window || P < 0) {
    if (blockIdx.x == 0 && threadIdx.x == 0) atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
    return;
  }
  const int chunks_per_token = Hkv * chunks_per_head;
  const int64_t total = static_cast<int64_t>(W) * chunks_per_token;
  for (int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; idx < total;
       idx += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(idx / chunks_per_token);
    const int rem = static_cast<int>(idx % chunks_per_token);
    const int g = rem / chunks_per_head, c = rem % chunks_per_head;
    if (block_mask) {
      const int b = i / block_size;
      if (b >= max_blocks || block_mask[static_cast<int64_t>(s) * max_blocks + b] == 0) continue;
    }
    const int pos = P + i;
    const int lp = pos / page_size;
    if (lp >= max_pages) {
      atomicOr(&g_error_word, MBE_DEVERR_LENGTH);
      continue;
    }
    const int page = block_table[static_cast<int64_t>(s) * max_pages + lp];
    if (page < 0 || page >= num_pages) {
      atomicOr(&g_error_word, MBE_DEVERR_PAGE);
      continue;
    }
    const int64_t dst = ((static_cast<int64_t>(page) * Hkv + g) * page_size + pos % page_size) * chunks_per_head + c;
    const int64_t src = (static_cast<int64_t>(t0 + i) * Hkv + g) * chunks_per_head + c;
    k_cache[dst] = k_win[src];
    v_cache[dst] = v_win[src];
  }
}

}  // namespace
}  // namespace mbe

extern "C" mbe_status mbe_kv_window_write(const void* k_win, const void* v_win, void* k_cache, void* v_cache,
                                          int32_t num_pages, const int32_t* block_table, int32_t max_pages_per_seq,
                                          const int32_t* prefix_len, const int32_t* window_len,
                                          const int32_t* cu_window, const uint8_t* block_write_mask_or_null,
                                          int32_t max_blocks_per_seq, int32_t batch, int32_t max_window,
                                          int32_t num_kv_heads, int32_t head_dim, int32_t block_size,
                                          int32_t page_size, cudaStream_t stream) {
  using namespace mbe;
  if (batch < 0 || max_window < 0 || num_kv_heads < 1 || head_dim < 8 || head_dim % 8 != 0 || block_size < 1 ||
      page_size < 1 || num_pages < 1 || max_pages_per_seq < 1)
    return MBE_ERR_INVALID_ARG;
  if (batch == 0 || max_window == 0) return MBE_OK;
  if (!k_win || !v_win || !k_cache || !v_cache || !block_table || !prefix_len || !window_len || !cu_window)
    return MBE_ERR_INVALID_ARG;
  if (!aligned16(k_win) || !aligned16(v_win) || !aligned16(k_cache) || !aligned16(v_cache))
    return MBE_ERR_INVALID_ARG;
  if (block_write_mask_or_null && max_blocks_per_seq < (max_window + block_size - 1) / block_size)
    return MBE_ERR_INVALID_ARG;
  if (batch > 65535) return MBE_ERR_UNSUPPORTED;
  const int chunks_per_head = head_dim / 8;
  const int64_t chunks = static_cast<int64_t>(max_window) * num_kv_heads * chunks_per_head;
  int64_t gx = (chunks + 255) / 256;
  if (gx > 4096) gx = 4096;
  dim3 grid(static_cast<unsigned>(gx), static_cast<unsigned>(batch));
  kv_window_write_kernel<<<grid, 256, 0, stream>>>(
      static_cast<const uint4*>(k_win), static_cast<const uint4*>(v_win), static_cast<uint4*>(k_cache),
      static_cast<uint4*>(v_cache), num_pages, block_table, max_pages_per_seq, prefix_len, window_len, cu_window,
      block_write_mask_or_null, max_blocks_per_seq, num_kv_heads, chunks_per_head, block_size, page_size, max_window);
  return launch_status();
}
