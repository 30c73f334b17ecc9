// Multi-Block Edit SFT attention support (Sec. 3): the cross-block attention
// mask. The forward under the mask is mbe_block_mask_attention (attention.cu).
//
// sft_mask_kernel: one CTA per (mask row, sequence); thread w builds 32-bit
// word w of the row from the link rules, so a row of nb blocks costs nb bits.
#include "common.cuh"

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
}  // namespace mbe

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
