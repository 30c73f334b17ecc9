/*
 * mbe.h -- C ABI of the GB300 (sm_103a) library for the data-parallel hot path
 * of Multi-Block Editing (MBE) for block-diffusion language models
 * (arXiv 2607.22663).
 *
 * One editing pass of MBE (Sec. 4.1, Eq. 5) reopens a window of k already
 * decoded blocks, runs the model over the window with full attention inside
 * it while reading the committed prefix from the KV cache, and applies the
 * token-to-token (T2T) edit rule of Eq. 2 to the window's historical part.
 * Blocks that changed are recomputed under standard (block-causal) attention
 * and their KV written back (Sec. 4.3, cache control). This library provides
 * the three data-parallel steps of that pass:
 *
 *   mbe_window_attention   attention of the window queries over the paged
 *                          prefix plus the window (Eq. 5; Sec. 2.2)
 *   mbe_edit_decide        argmax / confidence / threshold-and-replace (Eq. 2)
 *   mbe_kv_window_write    scatter of window K/V into the paged cache (Sec. 4.3)
 *
 * and, around them, the full decoding-step update (mbe_denoise_update: Eq. 2
 * with forced unmasking, entropies, changed blocks), the tail-entropy
 * window choice (mbe_tail_entropy_select: Eqs. 6-7), the targeted refresh of
 * the changed blocks (mbe_refresh_plan, mbe_gather_rows: Sec. 4.3), a
 * device-side loop over editing passes (mbe_pass_loop_*: Sec. 4.1), the
 * LM-head projection fused with the edit decision (mbe_lm_head_edit_decide)
 * and the cross-block training attention of Multi-Block Edit SFT, forward
 * and backward (mbe_sft_block_mask, mbe_block_mask_attention[_bwd]: Sec. 3).
 *
 * Conventions shared by every entry point
 *   - All pointers are DEVICE pointers unless stated otherwise; the caller
 *     owns every buffer. The library never allocates device memory (the
 *     CUDA graph that mbe_pass_loop_end instantiates aside).
 *   - Every call validates its host-visible arguments synchronously and returns
 *     a status; on any status other than MBE_OK nothing was launched.
 *   - Work is enqueued asynchronously on `stream`. Conditions that only the
 *     device can see (a length above the declared maximum, a page id outside
 *     the cache, a bounded wait that ran out) set a device error word and the
 *     affected work is skipped; mbe_get_device_error() reports and clears it.
 *   - bf16 tensors are IEEE bfloat16 bit patterns, row-major, densely packed in
 *     the stated shapes; every base pointer must be 16-byte aligned.
 *   - Window tokens of all sequences are packed back to back ("ragged"):
 *     sequence s owns rows cu_window[s] .. cu_window[s] + window_len[s] - 1.
 *   - Query head h reads KV head h / (num_q_heads / num_kv_heads) (grouped-
 *     query attention with contiguous groups).
 */
#ifndef MBE_H
#define MBE_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MBE_OK = 0,
  MBE_ERR_INVALID_ARG = 1,   /* bad host-visible argument (null, shape, alignment) */
  MBE_ERR_UNSUPPORTED = 2,   /* valid but not implemented (e.g. head_dim 96) */
  MBE_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed */
  MBE_ERR_TIMEOUT = 4,       /* a bounded device wait expired (device error word) */
  MBE_ERR_WORKSPACE = 5,     /* workspace missing or smaller than required */
  MBE_ERR_DEVICE_CHECK = 6   /* a device-side argument check failed (device error word) */
} mbe_status;

/* Attention mask of the window part (Sec. 2.2 and Eq. 5). */
typedef enum {
  MBE_BLOCK_CAUSAL = 0,               /* window query i sees window key j iff floor(j/B) <= floor(i/B) */
  MBE_MULTI_BLOCK_BIDIRECTIONAL = 1,  /* every window query sees every window key (full attention in W_j) */
  MBE_BLOCK_MASK = 2                  /* an explicit block-level mask (mbe_block_mask_attention only) */
} mbe_mask_mode;

typedef enum { MBE_F32 = 0, MBE_BF16 = 1 } mbe_dtype;

/* Bits of the device error word (see mbe_get_device_error). */
#define MBE_DEVERR_TIMEOUT 0x1u       /* a bounded wait in a kernel expired */
#define MBE_DEVERR_LENGTH 0x2u        /* prefix_len/window_len/mask_mode outside the declared range */
#define MBE_DEVERR_PAGE 0x4u          /* a block_table entry outside [0, num_pages) */
#define MBE_DEVERR_CAPACITY 0x8u      /* work list larger than the workspace was sized for */
#define MBE_DEVERR_PLAN 0x10u         /* mbe_window_attention_run found no plan for its parameters in the workspace */
#define MBE_DEVERR_NONFINITE 0x20u    /* a logit row had no softmax (NaN / +inf logit, or every logit -inf) */

/*
 * mbe_window_attention -- attention of one editing (or standard) pass.
 * Paper: Eq. 5 (window W_j = [j* B, (j+1) B) with full attention inside the
 * window), Sec. 2.2 (block j conditions on the committed prefix; blocks are
 * decoded left to right), Sec. 4.3 (the editing pass reads cached history and
 * writes no KV).
 *
 * For sequence s (P = prefix_len[s], W = window_len[s]) and window query i,
 * query head h, KV head g = h / (num_q_heads / num_kv_heads):
 *   out[cu_window[s] + i, h, :] = sum_j softmax_j(scale * q . k_j) v_j
 * over the visible keys j: all P prefix keys (cache positions 0..P-1, read
 * through block_table), and the window keys permitted by mask_mode[s].
 *
 *   q          bf16 [total_q_tokens, num_q_heads, head_dim]
 *   k_win,v_win bf16 [total_q_tokens, num_kv_heads, head_dim]: K/V of this pass's
 *              window tokens (never written to the cache by this call)
 *   k_cache,v_cache bf16 [num_pages, num_kv_heads, page_size, head_dim]
 *   block_table int32 [batch, max_pages_per_seq]: physical page of logical page
 *              p of sequence s; entries past ceil(P/page_size) are not read.
 *              An entry outside [0, num_pages) reads zeros and sets
 *              MBE_DEVERR_PAGE.
 *   prefix_len, window_len int32 [batch]; cu_window int32 [batch + 1] with
 *              cu_window[0] = 0, cu_window[s+1] = cu_window[s] + window_len[s],
 *              cu_window[batch] <= total_q_tokens (rows past it are not
 *              attended to, and those of out are not written).
 *   mask_mode  uint8 [batch], values of mbe_mask_mode (per sequence, so mixed
 *              standard and editing passes run in one launch).
 *   max_window, max_prefix  host upper bounds of window_len[] and prefix_len[]
 *              (they size the workspace; a larger device value sets
 *              MBE_DEVERR_LENGTH and that sequence is skipped).
 *   softmax_scale  0 means 1/sqrt(head_dim).
 *   out        bf16 [total_q_tokens, num_q_heads, head_dim]
 *   lse_or_null fp32 [total_q_tokens, num_q_heads]: natural-log sum of exp of
 *              the scaled scores, or NULL.
 *   workspace  device scratch of at least mbe_window_attention_workspace_size()
 *              bytes (work list and split-KV partials); not shared between
 *              concurrent calls.
 * Supported: head_dim in {64, 128}; num_q_heads / num_kv_heads a power of two
 * <= 128; page_size a power of two >= 8; block_size >= 1. Rows of k_win/v_win
 * outside every window, and cache rows past a prefix, may hold any bits (NaN
 * included): they never reach out.
 * Errors: MBE_ERR_INVALID_ARG, MBE_ERR_UNSUPPORTED, MBE_ERR_WORKSPACE,
 * MBE_ERR_CUDA (launch failure).
 */
mbe_status mbe_window_attention(const void* q, const void* k_win, const void* v_win, const void* k_cache,
                                const void* v_cache, int32_t num_pages, const int32_t* block_table,
                                int32_t max_pages_per_seq, const int32_t* prefix_len, const int32_t* window_len,
                                const int32_t* cu_window, const uint8_t* mask_mode, int32_t batch,
                                int32_t total_q_tokens, int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                int32_t block_size, int32_t page_size, int32_t max_window, int32_t max_prefix,
                                float softmax_scale, void* out, float* lse_or_null, void* workspace,
                                size_t workspace_bytes, cudaStream_t stream);

/*
 * mbe_window_attention_plan / mbe_window_attention_run -- the same attention as
 * mbe_window_attention, split so that one work list serves many calls.
 * Paper: Sec. 4.3 (an editing pass runs every layer over the same window
 * shapes); Eq. 5 and Sec. 2.2 as for mbe_window_attention.
 *
 * mbe_window_attention = plan + run. The plan (a device-side work list built
 * from prefix_len, window_len, cu_window, mask_mode and the bounds) is written
 * into `workspace`; every later run with the same workspace, the same
 * per-sequence lengths and modes, the same batch, heads, head_dim, block_size
 * and bounds reuses it, so the layers of one pass pay for one plan. Q/K/V,
 * cache, block table, scale and outputs may differ between runs. Runs that
 * share a workspace must be ordered on the GPU (one stream). Arguments,
 * layouts and errors are those of mbe_window_attention. The plan records the
 * parameters that fix its layout (batch, total_q_tokens, heads, head_dim,
 * block_size, max_window, max_prefix); a run whose parameters differ, or a
 * workspace holding no plan, computes nothing and sets MBE_DEVERR_PLAN. A run
 * whose cu_window places a planned window outside q/out skips it and sets
 * MBE_DEVERR_LENGTH. Changing the device-side lengths or modes without a new
 * plan is not detected and gives wrong (but in-bounds) results.
 */
mbe_status mbe_window_attention_plan(const int32_t* prefix_len, const int32_t* window_len, const int32_t* cu_window,
                                     const uint8_t* mask_mode, int32_t batch, int32_t total_q_tokens,
                                     int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim, int32_t block_size,
                                     int32_t max_window, int32_t max_prefix, void* workspace, size_t workspace_bytes,
                                     cudaStream_t stream);
mbe_status mbe_window_attention_run(const void* q, const void* k_win, const void* v_win, const void* k_cache,
                                    const void* v_cache, int32_t num_pages, const int32_t* block_table,
                                    int32_t max_pages_per_seq, const int32_t* prefix_len, const int32_t* window_len,
                                    const int32_t* cu_window, const uint8_t* mask_mode, int32_t batch,
                                    int32_t total_q_tokens, int32_t num_q_heads, int32_t num_kv_heads,
                                    int32_t head_dim, int32_t block_size, int32_t page_size, int32_t max_window,
                                    int32_t max_prefix, float softmax_scale, void* out, float* lse_or_null,
                                    void* workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * mbe_window_attention_plan_stats -- what the plan held in `workspace` (by
 * mbe_window_attention or mbe_window_attention_plan) contains: the number of
 * work units and the number of query slabs whose keys were cut into split-KV
 * pieces (merged afterwards by log-sum-exp). Paper: Sec. 4.3 (mixed-shape
 * forwards; here one device-side work list serves every shape). Synchronises
 * `stream`, then copies 12 bytes of the workspace to the host.
 * Errors: MBE_ERR_INVALID_ARG (null pointer, workspace smaller than 256 B),
 * MBE_ERR_CUDA.
 */
mbe_status mbe_window_attention_plan_stats(const void* workspace, size_t workspace_bytes, int32_t* n_units,
                                           int32_t* n_split_groups, cudaStream_t stream);

/*
 * mbe_window_attention_noalloc -- mbe_window_attention for callers that cannot
 * allocate device memory. The paper has no counterpart: this is an interface
 * convenience of this library, not a step of the method.
 *
 * Some callers cannot call cudaMalloc: code that runs inside a host framework
 * which owns every byte of device memory through its own pool and only hands
 * out input and output buffers, and code on a latency-critical path that must
 * not risk the device-wide synchronisation cudaMalloc/cudaFree may cause. This
 * entry point takes the same arguments as mbe_window_attention except the
 * workspace, and uses instead a static device array of 64 MiB that lives in
 * the library (every GPU that loads libmbe holds those 64 MiB until the
 * process exits). It allocates nothing.
 *
 *   - Shapes whose workspace (mbe_window_attention_workspace_size) exceeds
 *     64 MiB are rejected with MBE_ERR_WORKSPACE before anything is launched.
 *   - The first call on a device, with that device current, looks up the
 *     array's device address (cudaGetSymbolAddress) and keeps it for the rest
 *     of the process; make that first call before any stream capture on that
 *     device. A cudaDeviceReset (or any other teardown of the device's primary
 *     context) invalidates the kept address: do not call this entry point on
 *     that device after such a reset.
 *   - All calls on a device share the one array and each call overwrites what
 *     the previous call left there. Calls whose kernels overlap on the GPU
 *     (for example on two streams without ordering between them) race and give
 *     wrong results: order them on one stream or with events.
 * Errors: as mbe_window_attention, plus MBE_ERR_CUDA if the address lookup fails.
 */
mbe_status mbe_window_attention_noalloc(const void* q, const void* k_win, const void* v_win, const void* k_cache,
                                        const void* v_cache, int32_t num_pages, const int32_t* block_table,
                                        int32_t max_pages_per_seq, const int32_t* prefix_len,
                                        const int32_t* window_len, const int32_t* cu_window,
                                        const uint8_t* mask_mode, int32_t batch, int32_t total_q_tokens,
                                        int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                        int32_t block_size, int32_t page_size, int32_t max_window,
                                        int32_t max_prefix, float softmax_scale, void* out, float* lse_or_null,
                                        cudaStream_t stream);

/* Bytes of device workspace mbe_window_attention needs for these bounds on the
 * current device (depends on its SM count). Returns 0 for invalid arguments. */
size_t mbe_window_attention_workspace_size(int32_t batch, int32_t num_q_heads, int32_t num_kv_heads,
                                           int32_t head_dim, int32_t max_window, int32_t max_prefix);

/*
 * mbe_edit_decide -- the T2T update of Eq. 2 for every row of a pass.
 * Paper: Eq. 2 (Delta_t: a visible token is overwritten by the highest-
 * probability prediction when the prediction differs and its confidence
 * exceeds omega_edit); Sec. 4.1 (edits only in the window's historical part).
 *
 * For row r of logits l[r, 0..vocab-1]:
 *   argmax[r]     = x_hat = argmax_v l[r, v], the lowest index among ties
 *   confidence[r] = c = softmax(l[r])[x_hat] = 1 / sum_v exp(l[r, v] - l[r, x_hat])   (fp32)
 *   edit_mask[r]  = editable[r] && x_hat != committed[r] && c > tau_r
 *   new_tokens[r] = edit_mask[r] ? x_hat : committed[r]
 * with tau_r = tau_per_row[r] if given, else tau.
 *
 *   logits     [rows, row_stride] of `dtype`, the first `vocab` entries of each
 *              row used. A -inf logit is a token of probability 0 (a vocabulary
 *              mask). A row with a NaN or +inf logit, or with every logit -inf,
 *              has no softmax: it keeps its token (edit_mask 0), gets argmax -1
 *              and confidence NaN, and the call sets MBE_DEVERR_NONFINITE.
 *   committed  int32 [rows]; new_tokens may alias committed
 *   editable_or_null uint8 [rows] (NULL: every row editable)
 *   new_tokens int32 [rows], edit_mask uint8 [rows], confidence fp32 [rows],
 *   argmax_or_null int32 [rows]
 * Errors: MBE_ERR_INVALID_ARG (null pointer, vocab < 1, row_stride < vocab),
 * MBE_ERR_CUDA.
 */
mbe_status mbe_edit_decide(const void* logits, mbe_dtype dtype, int64_t row_stride, int32_t rows, int32_t vocab,
                           const int32_t* committed, const float* tau_per_row_or_null, float tau,
                           const uint8_t* editable_or_null, int32_t* new_tokens, uint8_t* edit_mask,
                           float* confidence, int32_t* argmax_or_null, cudaStream_t stream);

/*
 * mbe_denoise_update -- the full update of Eq. 2 for one forward of block
 * diffusion (standard step or editing pass), with the forced unmasking of
 * Sec. 2.3, the prediction entropy, and the changed-block record of Sec. 4.3.
 * Paper: Eq. 2 (Gamma_t = masked positions with c > omega_mask, unmasked to
 * x_hat; Delta_t = visible positions with x_hat != x and c > omega_edit,
 * overwritten by x_hat); Sec. 2.3 (if Gamma_t is empty while masks remain, the
 * most confident masked position is unmasked); Eq. 4 / Eq. 6 (entropy of the
 * prediction); Sec. 4.1 / 4.3 (stop when no token changes; refresh only the
 * blocks that changed).
 *
 * Rows are ragged by sequence: sequence s owns rows cu_rows[s] ..
 * cu_rows[s+1]-1 (device array, cu_rows[num_seqs] = total_rows); block b of
 * sequence s is its rows b*block_size .. (b+1)*block_size-1. Per row r with
 * current token x = tokens[r], x_hat and c as in mbe_edit_decide:
 *   update_kind[r] = 1 if x == mask_id and c > omega_mask            (Gamma_t)
 *                    2 if x == mask_id, forced (see below)
 *                    3 if x != mask_id, editable, x_hat != x, c > omega_edit (Delta_t)
 *                    0 otherwise;  new_tokens[r] = kind ? x_hat : x
 * A block with masked rows of which none is in Gamma_t unmasks its most
 * confident masked row (lowest row on equal fp32 confidence). Logit rows
 * without a softmax are handled as in mbe_edit_decide (token kept, kind 0,
 * argmax -1, confidence and entropy NaN, MBE_DEVERR_NONFINITE) and are never
 * the forced row: a block whose masked rows all lack one unmasks none.
 *   entropy_or_null[r] = -sum_v p_v ln p_v (fp32)
 *   block_changed_or_null[s * max_blocks_per_seq + b] = 1 iff some row of block
 *     b changed token (0 for blocks past the sequence's rows); it is the
 *     block_write_mask of mbe_kv_window_write for the refresh.
 *   seq_changes_or_null[s] = number of rows of s whose token changed.
 * logits: [total_rows, row_stride] of `dtype` (first `vocab` entries used);
 * tokens, new_tokens, argmax: int32 [total_rows] (new_tokens must not alias
 * tokens); update_kind uint8, confidence fp32 [total_rows]; editable_or_null
 * uint8 [total_rows] (NULL: all rows). A cu_rows range outside [0, total_rows]
 * or more than max_blocks_per_seq blocks set MBE_DEVERR_LENGTH.
 * Errors: MBE_ERR_INVALID_ARG, MBE_ERR_CUDA.
 */
mbe_status mbe_denoise_update(const void* logits, mbe_dtype dtype, int64_t row_stride, int32_t vocab,
                              const int32_t* cu_rows, int32_t num_seqs, int32_t total_rows, int32_t block_size,
                              int32_t max_blocks_per_seq, const int32_t* tokens, int32_t mask_id, float omega_mask,
                              float omega_edit, const uint8_t* editable_or_null, int32_t* new_tokens,
                              uint8_t* update_kind, float* confidence, int32_t* argmax, float* entropy_or_null,
                              uint8_t* block_changed_or_null, int32_t* seq_changes_or_null, cudaStream_t stream);

/*
 * mbe_tail_entropy_select -- tail-entropy choice of the editing window start.
 * Paper: Eq. 6 (S_rho(i) = mean of the ceil(rho B) largest final standard-scope
 * entropies of block i), Eq. 7 (j* = argmax of S_rho over the candidate blocks
 * C_j = {max(0, j - K_max + 1) <= i < j}), Eq. 5 (window W_j = [j* B, (j+1) B)).
 *
 *   block_entropy fp32 [num_seqs, n_hist, block_size]: the entropies (e.g. from
 *     mbe_denoise_update) of each sequence's last n_hist blocks, oldest first;
 *     slot n_hist-1 is block j-1.
 *   n_valid int32 [num_seqs]: how many of those slots hold blocks (<= n_hist).
 *   Candidates are the last min(n_valid, k_max - 1) slots.
 *   best_slot int32 [num_seqs]: the candidate with the largest score (the
 *     oldest on equal fp32 scores), -1 if there is none (j = 0);
 *   window_blocks int32 [num_seqs]: n_hist - best_slot + 1 (1 without candidate),
 *     the number of blocks of W_j including the current block j;
 *   scores_or_null fp32 [num_seqs, n_hist]: S_rho of each candidate, NaN elsewhere.
 * ceil(rho * block_size) is evaluated in double precision from the float rho.
 * The paper maintains the running argmax with a monotonic deque over
 * consecutive blocks; here each call evaluates its <= k_max - 1 candidates.
 * Errors: MBE_ERR_INVALID_ARG (rho outside (0, 1], k_max < 1, ...),
 * MBE_ERR_UNSUPPORTED (block_size > 12288), MBE_ERR_CUDA.
 */
mbe_status mbe_tail_entropy_select(const float* block_entropy, const int32_t* n_valid, int32_t num_seqs,
                                   int32_t n_hist, int32_t block_size, float rho, int32_t k_max, float* scores_or_null,
                                   int32_t* best_slot, int32_t* window_blocks, cudaStream_t stream);

/*
 * mbe_kv_window_write -- refresh of the cache with the window's K/V.
 * Paper: Sec. 4.1 (modified blocks are recomputed under standard attention to
 * refresh their KV cache) and Sec. 4.3 (cache control: only the changed blocks
 * are written back, after editing converges).
 *
 * For sequence s and window token i (P = prefix_len[s]), every KV head g:
 *   cache[block_table[s][(P+i)/page_size], g, (P+i) % page_size, :] = win[cu_window[s]+i, g, :]
 * for K and V. With block_write_mask_or_null ([batch, max_blocks_per_seq]
 * uint8), window block b = i / block_size is written only where the mask is
 * non-zero. A page id outside [0, num_pages) is skipped and sets
 * MBE_DEVERR_PAGE; a window longer than max_window sets MBE_DEVERR_LENGTH.
 *   k_win, v_win bf16 [total tokens, num_kv_heads, head_dim]
 *   k_cache, v_cache bf16 [num_pages, num_kv_heads, page_size, head_dim]
 * head_dim must be a multiple of 8.
 */
mbe_status mbe_kv_window_write(const void* k_win, const void* v_win, void* k_cache, void* v_cache,
                               int32_t num_pages, const int32_t* block_table, int32_t max_pages_per_seq,
                               const int32_t* prefix_len, const int32_t* window_len, const int32_t* cu_window,
                               const uint8_t* block_write_mask_or_null, int32_t max_blocks_per_seq, int32_t batch,
                               int32_t max_window, int32_t num_kv_heads, int32_t head_dim, int32_t block_size,
                               int32_t page_size, cudaStream_t stream);

/*
 * mbe_sft_block_mask -- the cross-block attention mask of Multi-Block Edit SFT.
 * Paper: Sec. 3 ("Cross-block attention mask"): standard block SFT links
 * noisy-to-noisy (NN), noisy-to-clean-prefix (NC) and clean-to-clean (CC);
 * MBE adds noisy-sees-forward (NF) links from noisy block i to clean blocks
 * i+1 .. i+K-1 and clean-sees-noisy (CN) links, and removes the CC links a
 * noisy block could use to reach its own clean block; prompt tokens are their
 * own category. The paper defers the exact construction to a supplement that
 * is not available; this follows the reading below. Sequence s is laid out as
 * [n_prompt_blocks[s] prompt blocks | N = n_blocks[s] noisy blocks n_i |
 * N clean blocks c_j]; bit k of row q is set iff block q attends to block k:
 *   prompt -> prompt;  n_i -> prompt, n_i, c_j (j < i), c_j (i < j <= i+K-1);
 *   c_j -> prompt, c_j, c_k (k <= j-K), n_i (j-K+1 <= i <= j-1).
 * K = 1 gives the standard block-diffusion SFT mask. mask uint32 [batch,
 * mask_rows, mask_words] as mbe_block_mask_attention reads it; rows past the
 * sequence's blocks are zero. A sequence with more than mask_rows blocks gets
 * zero rows and sets MBE_DEVERR_LENGTH.
 * Errors: MBE_ERR_INVALID_ARG (K < 1, mask_words * 32 < mask_rows, null
 * pointers), MBE_ERR_UNSUPPORTED (batch > 65535), MBE_ERR_CUDA.
 */
mbe_status mbe_sft_block_mask(const int32_t* n_prompt_blocks, const int32_t* n_blocks, int32_t K, int32_t batch,
                              int32_t mask_rows, int32_t mask_words, uint32_t* mask, cudaStream_t stream);

/*
 * mbe_block_mask_attention -- attention of whole training sequences under a
 * block-level mask, the forward of Multi-Block Edit SFT's cross-block attention
 * (Sec. 3, "Cross-block attention mask"; build the mask with mbe_sft_block_mask).
 * Sequence s owns tokens cu_seqlens[s] .. cu_seqlens[s] + seq_len[s] - 1 of
 *   q bf16 [total_tokens, num_q_heads, head_dim], k, v bf16 [total_tokens, num_kv_heads, head_dim];
 * query token i (block i / block_size) attends to key token j iff bit
 * (j / block_size) % 32 of word (j / block_size) / 32 of mask row i / block_size is set:
 *   mask uint32 [batch, mask_rows, mask_words] (mask_rows >= ceil(max_seq_len /
 *   block_size), mask_words * 32 >= mask_rows).
 * out bf16 [total_tokens, num_q_heads, head_dim]; lse_or_null fp32 [total_tokens,
 * num_q_heads] (natural-log sum of exp of the scaled scores; -inf and a zero
 * output row for a token that sees no key). softmax_scale 0 means
 * 1/sqrt(head_dim). Key tiles of 128 keys that no row of a 256-row work unit
 * sees are skipped. block_size must be a power of two >= 8 and max_seq_len <=
 * 65536; workspace as for mbe_window_attention_workspace_size(batch,
 * num_q_heads, num_kv_heads, head_dim, max_seq_len, 0). Rows of q, k and v
 * after cu_seqlens[batch] may hold any bits (NaN included): they never reach
 * out.
 * Errors as mbe_window_attention.
 */
mbe_status mbe_block_mask_attention(const void* q, const void* k, const void* v, const int32_t* seq_len,
                                    const int32_t* cu_seqlens, const uint32_t* mask, int32_t mask_rows,
                                    int32_t mask_words, int32_t batch, int32_t total_tokens, int32_t num_q_heads,
                                    int32_t num_kv_heads, int32_t head_dim, int32_t block_size, int32_t max_seq_len,
                                    float softmax_scale, void* out, float* lse_or_null, void* workspace,
                                    size_t workspace_bytes, cudaStream_t stream);

/*
 * mbe_block_mask_attention_bwd -- gradients of mbe_block_mask_attention (the
 * backward of Multi-Block Edit SFT's cross-block attention, Sec. 3).
 * With P the attention probabilities under the mask (recomputed from q, k and
 * the forward's lse), dO = dout and delta_i = dO_i . O_i:
 *   dV = P^T dO,  dS = P o (dO V^T - delta),  dQ = scale dS K,  dK = scale dS^T Q
 * summed over the query heads that share a KV head. Inputs as in
 * mbe_block_mask_attention plus out (its bf16 output), dout bf16 [total_tokens,
 * num_q_heads, head_dim] and lse fp32 [total_tokens, num_q_heads] (its natural-
 * log output). Outputs (fp32, overwritten): dq [total_tokens, num_q_heads,
 * head_dim], dk, dv [total_tokens, num_kv_heads, head_dim]. P and dS are
 * rounded to bf16 before their products (tensor cores), as in the forward's P.
 * workspace: mbe_block_mask_attention_bwd_workspace_size(batch, total_tokens,
 * num_q_heads) bytes, 16-byte aligned. head_dim must be 128; num_q_heads /
 * num_kv_heads must divide 32; max_seq_len * that ratio <= 65536. Rows past
 * cu_seqlens[batch] are not written; where total_tokens exceeds
 * cu_seqlens[batch], those rows of q, k, v, out and dout must hold finite
 * values (the last tiles of the last sequence read them, and masked products
 * still multiply them by zero).
 * Errors: MBE_ERR_INVALID_ARG, MBE_ERR_UNSUPPORTED, MBE_ERR_WORKSPACE,
 * MBE_ERR_CUDA; a bounded wait that expires sets MBE_DEVERR_TIMEOUT.
 */
size_t mbe_block_mask_attention_bwd_workspace_size(int32_t batch, int32_t total_tokens, int32_t num_q_heads);
mbe_status mbe_block_mask_attention_bwd(const void* q, const void* k, const void* v, const void* out,
                                        const void* dout, const float* lse, const int32_t* seq_len,
                                        const int32_t* cu_seqlens, const uint32_t* mask, int32_t mask_rows,
                                        int32_t mask_words, int32_t batch, int32_t total_tokens, int32_t num_q_heads,
                                        int32_t num_kv_heads, int32_t head_dim, int32_t block_size,
                                        int32_t max_seq_len, float softmax_scale, float* dq, float* dk, float* dv,
                                        void* workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * mbe_lm_head_edit_decide -- the LM-head projection fused with the edit
 * decision, so that the [rows, vocab] logits never reach memory.
 * Paper: Eq. 2 (T2T set Delta_t: x_hat = argmax of the prediction, c its
 * probability; replace where x_hat != x and c > omega_edit) on the logits
 * l[r, v] = sum_k hidden[r, k] * weight[v, k] of the window rows (Sec. 4.1),
 * and the prediction entropy of Eqs. 4 and 6.
 *   hidden  bf16 [rows, hidden_dim]   final hidden states of the window rows
 *   weight  bf16 [vocab, hidden_dim]  LM head, one row per token id
 *   committed, tau_per_row_or_null, tau, editable_or_null, new_tokens,
 *   edit_mask, confidence, argmax_or_null: as in mbe_edit_decide
 *   entropy_or_null fp32 [rows]: -sum_v p_v ln p_v
 *   workspace: device buffer of at least mbe_lm_head_workspace_size(rows,
 *     vocab) bytes, 16-byte aligned (per-row partial states of the vocabulary
 *     chunks: 16 bytes per row and 256 tokens at most).
 * The logits are accumulated in fp32 on the tensor cores (bf16 products), so
 * they differ from exact dot products by fp32 rounding of the running sums;
 * decisions are taken on those fp32 values. A row whose logits include NaN or
 * +inf (from non-finite hidden or weight values) gets no decision, as in
 * mbe_edit_decide (MBE_DEVERR_NONFINITE). hidden_dim must be a multiple of 8
 * and hidden / weight 16-byte aligned.
 * Errors: MBE_ERR_INVALID_ARG, MBE_ERR_WORKSPACE, MBE_ERR_UNSUPPORTED
 * (rows or vocab above 2^30), MBE_ERR_CUDA; a bounded wait that expires sets
 * MBE_DEVERR_TIMEOUT.
 */
size_t mbe_lm_head_workspace_size(int32_t rows, int32_t vocab);
mbe_status mbe_lm_head_edit_decide(const void* hidden, const void* weight, int32_t rows, int32_t vocab,
                                   int32_t hidden_dim, const int32_t* committed, const float* tau_per_row_or_null,
                                   float tau, const uint8_t* editable_or_null, int32_t* new_tokens,
                                   uint8_t* edit_mask, float* confidence, int32_t* argmax_or_null,
                                   float* entropy_or_null, void* workspace, size_t workspace_bytes,
                                   cudaStream_t stream);

/*
 * mbe_refresh_plan -- lays out the targeted refresh of the blocks that changed.
 * Paper: Sec. 4.3 (after an editing pass, only the blocks whose tokens changed
 * are recomputed under standard attention and their KV written back) with the
 * block-causal conditioning of Sec. 2.2 and Eq. 5's window W_j.
 *
 * Recomputing window block b of sequence s under standard attention means its
 * queries see the cached prefix, the window blocks before b as they stand in
 * the cache (write the changed blocks first, with mbe_kv_window_write on this
 * layout), and all of block b. That is one attention problem per changed
 * block: prefix P_s + b*B and a one-block bidirectional window. This writes
 * those problems as a ragged batch of E = batch * max_blocks_per_seq entries,
 * entry e = s * max_blocks_per_seq + b, empty unless block b of s changed:
 *   r_prefix_len int32 [E]   P_s + b*B for a changed block, else 0
 *   r_window_len int32 [E]   min(B, W_s - b*B) for a changed block inside the
 *                            window, else 0
 *   r_cu_window int32 [E+1]  exclusive prefix sum of r_window_len
 *   r_mask_mode uint8 [E]    MBE_MULTI_BLOCK_BIDIRECTIONAL
 *   r_block_table int32 [E, max_pages_per_seq]  block_table row s, or -1
 *   r_src_row int32 [total_rows]  window row (index into the pass's rows,
 *                            cu_window) of refresh row k < r_cu_window[E];
 *                            -1 for the rest (see mbe_gather_rows)
 *   r_count int32 [2]        {changed entries, refresh rows}
 * Pass the result to mbe_window_attention / mbe_kv_window_write with batch E,
 * max_window B and max_prefix >= max_s(P_s + B * floor((W_s - 1) / B)) (the
 * start of the last block; max_s(P_s + W_s) - 1 always suffices; the block
 * tables must cover it, as they do P_s + W_s for the write); total_rows = rows of the
 * pass (cu_window[batch]) always suffices. Inputs: block_changed uint8
 * [batch, max_blocks_per_seq] (as written by mbe_denoise_update), prefix_len,
 * window_len int32 [batch], cu_window int32 [batch+1], block_table int32
 * [batch, max_pages_per_seq]. Everything stays on the device, so the call can
 * be captured in a CUDA graph. Device checks: a window longer than max_window
 * or than max_blocks_per_seq * B is treated as unchanged and sets
 * MBE_DEVERR_LENGTH; more refresh rows than total_rows sets MBE_DEVERR_CAPACITY.
 * Errors: MBE_ERR_INVALID_ARG (null pointers, negative sizes),
 * MBE_ERR_UNSUPPORTED (more than 2^24 entries), MBE_ERR_CUDA.
 */
mbe_status mbe_refresh_plan(const uint8_t* block_changed, int32_t max_blocks_per_seq, const int32_t* prefix_len,
                            const int32_t* window_len, const int32_t* cu_window, const int32_t* block_table,
                            int32_t max_pages_per_seq, int32_t batch, int32_t block_size, int32_t max_window,
                            int32_t total_rows, int32_t* r_prefix_len, int32_t* r_window_len, int32_t* r_cu_window,
                            uint8_t* r_mask_mode, int32_t* r_block_table, int32_t* r_src_row, int32_t* r_count,
                            cudaStream_t stream);

/*
 * mbe_gather_rows -- dst[k] = src[src_row[k]] for rows of row_bytes bytes
 * (k < rows): the compaction of per-row inputs (token ids, hidden states,
 * Q/K/V) for the refresh batch of mbe_refresh_plan. A negative src_row[k]
 * gives a zero row; src_row[k] >= src_rows gives a zero row and sets
 * MBE_DEVERR_LENGTH. rows_used_or_null (device int32, e.g. &r_count[1] of
 * mbe_refresh_plan) limits the copy to rows k < min(rows, *rows_used): the rows
 * after it are left as they are, so a refresh batch only costs its changed rows.
 * src and dst are device buffers that must not overlap; 16-byte rows and
 * alignment give vectorised copies.
 * Errors: MBE_ERR_INVALID_ARG, MBE_ERR_CUDA.
 */
mbe_status mbe_gather_rows(const void* src, int64_t src_rows, int64_t row_bytes, const int32_t* src_row,
                           int64_t rows, const int32_t* rows_used_or_null, void* dst, cudaStream_t stream);

/*
 * mbe_gather_rows_multi -- mbe_gather_rows for n_tensors (1..MBE_GATHER_MAX)
 * tensors that share one row map, in one launch: dsts[t][k] =
 * srcs[t][src_row[k]] for rows of row_bytes[t] bytes, with the zero rows, the
 * MBE_DEVERR_LENGTH flag and the rows_used_or_null limit of mbe_gather_rows.
 * This is how the refresh batch of Sec. 4.3 compacts a layer's Q, K and V
 * together. srcs, row_bytes and dsts are host arrays of n_tensors entries;
 * the buffers they point to are device buffers with src_rows source rows and
 * at least `rows` destination rows, none overlapping. When every row is a
 * whole number of 16-byte chunks and every buffer is 16-byte aligned the copy
 * is one kernel launch; otherwise it is one mbe_gather_rows per tensor.
 * Errors: MBE_ERR_INVALID_ARG (n_tensors out of range, null pointers,
 * negative sizes), MBE_ERR_CUDA.
 */
#define MBE_GATHER_MAX 4
mbe_status mbe_gather_rows_multi(int32_t n_tensors, const void* const* srcs, const int64_t* row_bytes,
                                 void* const* dsts, int64_t src_rows, const int32_t* src_row, int64_t rows,
                                 const int32_t* rows_used_or_null, cudaStream_t stream);

/*
 * mbe_refresh_gather_write -- the per-layer row work of the targeted refresh
 * (Sec. 4.3: the changed blocks are recomputed under standard attention and
 * their KV written back) in one launch. For refresh row k < min(rows,
 * *rows_used_or_null) of the layout written by mbe_refresh_plan it copies
 * source row src_row[k] of q [src_rows, num_q_heads, head_dim], k_win and
 * v_win [src_rows, num_kv_heads, head_dim] (bf16) into row k of q_out, k_out
 * and v_out, and writes that K and V row into k_cache / v_cache
 * [num_pages, num_kv_heads, page_size, head_dim] at the row's refresh-layout
 * position: row k belongs to entry e, the largest e < num_entries with
 * r_cu_window[e] <= k, and goes to position r_prefix_len[e] + k -
 * r_cu_window[e] through block-table row e (r_block_table [num_entries,
 * max_pages_per_seq]). The result equals mbe_gather_rows_multi of the three
 * tensors followed by mbe_kv_window_write of k_out / v_out on the refresh
 * layout. Rows with src_row[k] < 0 become zero rows and write no cache slot;
 * src_row[k] >= src_rows gives a zero row and MBE_DEVERR_LENGTH; a row outside
 * every entry (k >= r_cu_window[num_entries]) or a position past the
 * block-table row sets MBE_DEVERR_LENGTH and a page id outside [0, num_pages)
 * MBE_DEVERR_PAGE (those rows write no cache slot). Rows from
 * *rows_used_or_null on are left as they are. All buffers are device memory,
 * 16-byte aligned, none overlapping.
 * Errors: MBE_ERR_INVALID_ARG (null or misaligned pointers, bad sizes),
 * MBE_ERR_CUDA.
 */
mbe_status mbe_refresh_gather_write(const void* q, const void* k_win, const void* v_win, int64_t src_rows,
                                    int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                    const int32_t* src_row, const int32_t* rows_used_or_null, int64_t rows,
                                    const int32_t* r_prefix_len, const int32_t* r_cu_window,
                                    const int32_t* r_block_table, int32_t num_entries, int32_t max_pages_per_seq,
                                    void* k_cache, void* v_cache, int32_t num_pages, int32_t page_size,
                                    void* q_out, void* k_out, void* v_out, cudaStream_t stream);

/*
 * Editing-pass loop on the device. Paper: Sec. 4.1 (the window is edited by
 * repeated passes until a pass changes no token or N_MBE passes have run) and
 * Sec. 4.3 (one graph serves every shape of the pass).
 *
 * mbe_pass_loop_begin creates a CUDA graph made of a reset of *passes_done
 * and a conditional WHILE node, and starts capturing `stream` (not the legacy
 * default stream) into the node's body in relaxed capture mode: everything
 * enqueued on `stream` until mbe_pass_loop_end is one pass. The body must
 * end with mbe_pass_loop_until_stable, which counts the pass in *passes_done
 * (device int32) and runs another pass only if some seq_changes[s] != 0 (as
 * written by mbe_denoise_update in the same pass) and fewer than max_passes
 * passes ran. mbe_pass_loop_end instantiates the graph; mbe_pass_loop_launch
 * runs all passes with one launch and no host synchronisation. Buffers used in
 * the body must outlive the loop. mbe_pass_loop_destroy releases everything
 * (it also ends a capture still open).
 * Errors: MBE_ERR_INVALID_ARG (max_passes < 1, null pointers, a stream already
 * capturing or the default stream, until_stable missing or repeated, another
 * stream), MBE_ERR_CUDA (capture or instantiation failed; see
 * mbe_last_error_string).
 */
typedef struct mbe_pass_loop mbe_pass_loop;
mbe_status mbe_pass_loop_begin(int32_t max_passes, int32_t* passes_done, cudaStream_t stream,
                               mbe_pass_loop** loop_out);
mbe_status mbe_pass_loop_until_stable(mbe_pass_loop* loop, const int32_t* seq_changes, int32_t num_seqs,
                                      cudaStream_t stream);
mbe_status mbe_pass_loop_end(mbe_pass_loop* loop, cudaStream_t stream);
mbe_status mbe_pass_loop_launch(mbe_pass_loop* loop, cudaStream_t stream);
void mbe_pass_loop_destroy(mbe_pass_loop* loop);

/* Synchronises `stream`, then reads and clears the device error word of the
 * current device. Returns MBE_OK if it was clear, MBE_ERR_TIMEOUT if the
 * timeout bit was set, else MBE_ERR_DEVICE_CHECK; *flags_or_null receives the
 * MBE_DEVERR_* bits. */
mbe_status mbe_get_device_error(cudaStream_t stream, uint32_t* flags_or_null);

/* Default wall-clock limit of one bounded device wait: 1 s. */
#define MBE_DEFAULT_WAIT_LIMIT_NS 1000000000ull

/*
 * mbe_set_wait_limit_ns -- failure-detection hook (no counterpart in the
 * paper). Sets the wall-clock limit, in nanoseconds, of each bounded wait
 * (an mbarrier phase wait inside the attention, LM-head and attention-
 * backward kernels) of every kernel launched after the call, from any host
 * thread, and returns the previous limit. The default is
 * MBE_DEFAULT_WAIT_LIMIT_NS. A kernel whose wait runs out sets
 * MBE_DEVERR_TIMEOUT, lets the copies and tensor-core operations it already
 * issued finish, releases its tensor memory and returns, so the context stays
 * usable; the outputs of that call are incomplete. With a limit of 0 every
 * wait that is not complete at its first try runs out, which lets a test drive
 * that path without any fault. The waits of the abort path itself always keep
 * the default limit. Lowering the limit is meant for tests only.
 */
uint64_t mbe_set_wait_limit_ns(uint64_t limit_ns);

/* Host-thread-local description of the last CUDA runtime failure the library
 * saw (the call site, the error name and message); useful after MBE_ERR_CUDA. */
const char* mbe_last_error_string(void);

/* Static description of a status code. */
const char* mbe_status_string(mbe_status status);

/* Library version: major * 10000 + minor * 100 + patch. */
int32_t mbe_version(void);

#ifdef __cplusplus
}
#endif
#endif /* MBE_H */
