/*
 * mbe_oracle.c -- plain, slow, obviously-correct CPU oracle for the hot path
 * of Multi-Block Editing (MBE): the editing pass's window attention, the T2T
 * edit decision, and the KV window write.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing on the product path may call this code:
 * only the tests, the smoke check and the benchmark's CPU-baseline leg use it.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * Arithmetic: inputs are bf16 (or fp32) values widened exactly to double;
 * every sum, exponential and division is done in double precision. Masks are
 * built explicitly as boolean arrays before any score is computed.
 *
 * Citations are to the paper (arXiv 2607.22663, "Multi-Block Editing"):
 *   Sec. 2.2   block diffusion: block j spans [jB,(j+1)B) and conditions on
 *              the committed prefix.
 *   Eq. 2      T2T edit set: a visible token is overwritten by the argmax
 *              prediction iff prediction != token and confidence > omega_edit.
 *   Eq. 5      editing window W_j = [j* B, (j+1) B) with full attention inside
 *              the window (Sec. 4.1 "Inference algorithm").
 *   Sec. 4.3   cache control: the editing pass reads the cached history and
 *              writes no KV; changed blocks are later recomputed under standard
 *              (block-causal) attention and their KV written back.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_OK 0
#define ORC_BAD_ARG 1
#define ORC_BAD_PAGE 2
#define ORC_UNDECIDABLE 3 /* completed; some rows had no softmax (see row_softmax) */
#define ORC_NOMEM 4

/* bf16 bit pattern -> exact double */
static double bf16_to_double(uint16_t b) {
  uint32_t u = ((uint32_t)b) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

/* logit v of row r: dtype 0 float32, 1 bf16 bits, 2 float64 */
static double load_logit(const void* logits, int32_t dtype, int64_t idx) {
  if (dtype == 0) return (double)((const float*)logits)[idx];
  if (dtype == 1) return bf16_to_double(((const uint16_t*)logits)[idx]);
  return ((const double*)logits)[idx];
}

/*
 * Softmax statistics of logit row `off` (vocab entries): the maximum m, its
 * lowest index x_hat and S = sum_v exp(l_v - m). The row has a softmax only if
 * none of its logits is NaN or +inf and at least one is finite; a -inf logit
 * is a token of probability 0 (a vocabulary mask). Returns 0, with x_hat = -1,
 * for a row without a softmax: Eq. 2 cannot decide on it ("undecidable").
 */
static int row_softmax(const void* logits, int32_t dtype, int64_t off, int32_t vocab, double* m_out,
                       int32_t* xh_out, double* s_out) {
  double m = -INFINITY;
  int32_t xh = -1;
  for (int32_t v = 0; v < vocab; ++v) {
    const double x = load_logit(logits, dtype, off + v);
    if (isnan(x) || x == INFINITY) {
      *xh_out = -1;
      return 0;
    }
    if (x > m) {
      m = x;
      xh = v;
    }
  }
  *xh_out = xh;
  if (xh < 0) return 0; /* every logit is -inf */
  double ssum = 0.0;
  for (int32_t v = 0; v < vocab; ++v) ssum += exp(load_logit(logits, dtype, off + v) - m);
  *m_out = m;
  *s_out = ssum;
  return 1;
}

int oracle_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/*
 * Window attention of one editing (or standard) pass, Eq. 5 and Sec. 2.2.
 *
 * For sequence s with committed prefix length P = prefix_len[s] and window
 * length W = window_len[s], the key sequence is the P cached prefix tokens
 * (read from the paged cache through block_table) followed by the W window
 * tokens of this pass (k_win/v_win rows cu_window[s] .. cu_window[s]+W-1).
 *
 * Visibility of key j to window query i (both window-local for the window):
 *   prefix key                          : always visible
 *   window key, multi_block_bidirectional (mode 1): visible  (full attention
 *                                          inside W_j, Eq. 5)
 *   window key, block_causal (mode 0)   : visible iff floor(j/B) <= floor(i/B)
 *                                          (a block sees earlier blocks and
 *                                          itself, Sec. 2.2)
 * Query head h reads kv head h / (Hq/Hkv).
 *
 * out[t, h, :] = sum_j softmax_j(scale * q.k_j) v_j over visible j  (double)
 * lse[t, h]    = log sum_j exp(scale * q.k_j)                       (double)
 *
 * If n_units >= 0, only the (unit_seq[u], unit_qhead[u]) pairs are computed
 * (all window rows of that pair); otherwise every (seq, head) is computed.
 */
int oracle_window_attention(const uint16_t* q, const uint16_t* k_win, const uint16_t* v_win,
                            const uint16_t* k_cache, const uint16_t* v_cache, const int32_t* block_table,
                            int32_t max_pages_per_seq, const int32_t* prefix_len, const int32_t* window_len,
                            const int32_t* cu_window, const uint8_t* mask_mode, int32_t batch, int32_t Hq,
                            int32_t Hkv, int32_t D, int32_t block_size, int32_t page_size, int32_t num_pages,
                            double scale, int32_t n_units, const int32_t* unit_seq, const int32_t* unit_qhead,
                            double* out, double* lse) {
  if (batch < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || D <= 0 || block_size <= 0 || page_size <= 0)
    return ORC_BAD_ARG;
  const int64_t total = n_units >= 0 ? n_units : (int64_t)batch * Hq;
  const int32_t group = Hq / Hkv;
  int status = ORC_OK;

#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t u = 0; u < total; ++u) {
    int32_t s, h;
    if (n_units >= 0) {
      s = unit_seq[u];
      h = unit_qhead[u];
    } else {
      s = (int32_t)(u / Hq);
      h = (int32_t)(u % Hq);
    }
    if (s < 0 || s >= batch || h < 0 || h >= Hq) {
#pragma omp atomic write
      status = ORC_BAD_ARG;
      continue;
    }
    const int32_t P = prefix_len[s], W = window_len[s], t0 = cu_window[s];
    const int32_t g = h / group;
    const int32_t nk = P + W;
    if (W == 0) continue;
    if (P < 0 || W < 0 || (P + page_size - 1) / page_size > max_pages_per_seq) {
#pragma omp atomic write
      status = ORC_BAD_ARG;
      continue;
    }
    /* key and value rows (pointers into the inputs), logical order */
    const uint16_t** krow = (const uint16_t**)malloc(sizeof(uint16_t*) * (size_t)(nk > 0 ? nk : 1));
    const uint16_t** vrow = (const uint16_t**)malloc(sizeof(uint16_t*) * (size_t)(nk > 0 ? nk : 1));
    unsigned char* mask = (unsigned char*)malloc((size_t)W * (size_t)(nk > 0 ? nk : 1));
    double* z = (double*)malloc(sizeof(double) * (size_t)(nk > 0 ? nk : 1));
    if (!krow || !vrow || !mask || !z) {
      free(krow); free(vrow); free(mask); free(z);
#pragma omp atomic write
      status = ORC_NOMEM;
      continue;
    }
    int bad = 0;
    for (int32_t j = 0; j < P; ++j) {
      const int32_t page = block_table[(int64_t)s * max_pages_per_seq + j / page_size];
      if (page < 0 || page >= num_pages) { bad = 1; break; }
      const int64_t off = (((int64_t)page * Hkv + g) * page_size + (j % page_size)) * D;
      krow[j] = k_cache + off;
      vrow[j] = v_cache + off;
    }
    for (int32_t j = 0; j < W; ++j) {
      const int64_t off = ((int64_t)(t0 + j) * Hkv + g) * D;
      krow[P + j] = k_win + off;
      vrow[P + j] = v_win + off;
    }
    if (bad) {
      free(krow); free(vrow); free(mask); free(z);
#pragma omp atomic write
      status = ORC_BAD_PAGE;
      continue;
    }
    /* explicit boolean mask M[i][j] */
    for (int32_t i = 0; i < W; ++i) {
      for (int32_t j = 0; j < nk; ++j) {
        unsigned char vis;
        if (j < P) {
          vis = 1;
        } else if (mask_mode[s] == 1) {
          vis = 1;
        } else {
          const int32_t w = j - P;
          vis = (w / block_size) <= (i / block_size);
        }
        mask[(int64_t)i * nk + j] = vis;
      }
    }
    for (int32_t i = 0; i < W; ++i) {
      const uint16_t* qi = q + ((int64_t)(t0 + i) * Hq + h) * D;
      double m = -INFINITY;
      for (int32_t j = 0; j < nk; ++j) {
        if (!mask[(int64_t)i * nk + j]) continue;
        double dot = 0.0;
        for (int32_t d = 0; d < D; ++d) dot += bf16_to_double(qi[d]) * bf16_to_double(krow[j][d]);
        z[j] = scale * dot;
        if (z[j] > m) m = z[j];
      }
      double zsum = 0.0;
      for (int32_t j = 0; j < nk; ++j)
        if (mask[(int64_t)i * nk + j]) zsum += exp(z[j] - m);
      double* oi = out + ((int64_t)(t0 + i) * Hq + h) * D;
      for (int32_t d = 0; d < D; ++d) oi[d] = 0.0;
      for (int32_t j = 0; j < nk; ++j) {
        if (!mask[(int64_t)i * nk + j]) continue;
        const double p = exp(z[j] - m) / zsum;
        for (int32_t d = 0; d < D; ++d) oi[d] += p * bf16_to_double(vrow[j][d]);
      }
      if (lse) lse[(int64_t)(t0 + i) * Hq + h] = m + log(zsum);
    }
    free(krow); free(vrow); free(mask); free(z);
  }
  return status;
}

/*
 * T2T edit decision of Eq. 2 for the rows of one editing pass.
 *
 * For row r with logits l[r, 0..V-1]:
 *   x_hat = argmax_v l[r, v]      (ties: the lowest index)
 *   c     = p(x_hat) = exp(l[x_hat]) / sum_v exp(l[v]) = 1 / sum_v exp(l[v] - l[x_hat])
 *   edit  = editable[r] && x_hat != committed[r] && c > tau_r
 *   new   = edit ? x_hat : committed[r]
 * tau_r is tau_per_row[r] when given, else tau. The comparison c > tau_r is
 * taken on c rounded to float, the precision of tau. editable == NULL means
 * every row is editable (the caller restricts edits to the historical part of
 * the window, Sec. 4.1). A row without a softmax (a NaN or +inf logit, or
 * every logit -inf; see row_softmax) keeps its token: edit 0, x_hat -1, c NaN,
 * and the call returns ORC_UNDECIDABLE after finishing every row.
 * dtype 0: float32 logits, 1: bf16 logits, 2: float64 logits (the LM-head
 * projection of oracle_lm_head_logits). If n_sel >= 0 only rows
 * sel_rows[0..n_sel-1] are computed; outputs are indexed by row.
 */
int oracle_edit_decide(const void* logits, int32_t dtype, int64_t row_stride, int32_t rows, int32_t vocab,
                       const int32_t* committed, const float* tau_per_row, float tau, const uint8_t* editable,
                       int32_t n_sel, const int32_t* sel_rows, int32_t* new_tokens, uint8_t* edit_mask,
                       double* confidence, int32_t* argmax_out) {
  if (rows < 0 || vocab <= 0 || dtype < 0 || dtype > 2 || row_stride < vocab) return ORC_BAD_ARG;
  const int64_t total = n_sel >= 0 ? n_sel : rows;
  int bad_arg = 0, undecidable = 0;
#pragma omp parallel for schedule(static)
  for (int64_t u = 0; u < total; ++u) {
    const int32_t r = n_sel >= 0 ? sel_rows[u] : (int32_t)u;
    if (r < 0 || r >= rows) {
#pragma omp atomic write
      bad_arg = 1;
      continue;
    }
    double m = 0.0, ssum = 0.0;
    int32_t xh = -1;
    if (!row_softmax(logits, dtype, (int64_t)r * row_stride, vocab, &m, &xh, &ssum)) {
#pragma omp atomic write
      undecidable = 1;
      if (new_tokens) new_tokens[r] = committed[r];
      if (edit_mask) edit_mask[r] = 0;
      if (confidence) confidence[r] = NAN;
      if (argmax_out) argmax_out[r] = -1;
      continue;
    }
    const double c = 1.0 / ssum;
    const float tr = tau_per_row ? tau_per_row[r] : tau;
    const int ed = (editable == NULL || editable[r] != 0) && xh != committed[r] && ((float)c > tr);
    if (new_tokens) new_tokens[r] = ed ? xh : committed[r];
    if (edit_mask) edit_mask[r] = (uint8_t)ed;
    if (confidence) confidence[r] = c;
    if (argmax_out) argmax_out[r] = xh;
  }
  if (bad_arg) return ORC_BAD_ARG;
  return undecidable ? ORC_UNDECIDABLE : ORC_OK;
}

/*
 * KV window write (Sec. 4.3 targeted refresh): the K/V of window token i of
 * sequence s is stored at logical cache position P + i, i.e. in page
 * block_table[s][(P+i) / page_size], slot (P+i) % page_size, for every kv head.
 * If block_write_mask is given ([batch, max_blocks_per_seq] bytes), window
 * block b = i / block_size is written only where block_write_mask[s][b] != 0
 * (only the blocks whose tokens changed are refreshed).
 */
int oracle_kv_window_write(const uint16_t* k_win, const uint16_t* v_win, uint16_t* k_cache, uint16_t* v_cache,
                           const int32_t* block_table, int32_t max_pages_per_seq, const int32_t* prefix_len,
                           const int32_t* window_len, const int32_t* cu_window, const uint8_t* block_write_mask,
                           int32_t max_blocks_per_seq, int32_t batch, int32_t Hkv, int32_t D, int32_t block_size,
                           int32_t page_size, int32_t num_pages) {
  if (batch < 0 || Hkv <= 0 || D <= 0 || block_size <= 0 || page_size <= 0) return ORC_BAD_ARG;
  for (int32_t s = 0; s < batch; ++s) {
    const int32_t P = prefix_len[s], W = window_len[s], t0 = cu_window[s];
    for (int32_t i = 0; i < W; ++i) {
      if (block_write_mask && !block_write_mask[(int64_t)s * max_blocks_per_seq + i / block_size]) continue;
      const int32_t pos = P + i;
      if (pos / page_size >= max_pages_per_seq) return ORC_BAD_ARG;
      const int32_t page = block_table[(int64_t)s * max_pages_per_seq + pos / page_size];
      if (page < 0 || page >= num_pages) return ORC_BAD_PAGE;
      for (int32_t g = 0; g < Hkv; ++g) {
        const int64_t dst = (((int64_t)page * Hkv + g) * page_size + pos % page_size) * D;
        const int64_t src = ((int64_t)(t0 + i) * Hkv + g) * D;
        for (int32_t d = 0; d < D; ++d) {
          k_cache[dst + d] = k_win[src + d];
          v_cache[dst + d] = v_win[src + d];
        }
      }
    }
  }
  return ORC_OK;
}

/*
 * Full threshold update of a decoding step (Eq. 2 with the forced unmasking
 * rule of Sec. 2.3), plus the per-row entropy H = -sum_v p_v log p_v of the
 * prediction (the quantity behind Eq. 4, PPL = exp(H), and Eq. 6).
 *
 * Rows are ragged: sequence s owns rows cu_rows[s] .. cu_rows[s+1]-1; window
 * block b of sequence s holds its rows b*block_size .. (b+1)*block_size-1.
 * For row r with current token x = tokens[r], argmax x_hat and confidence c
 * (as in oracle_edit_decide):
 *   masked (x == mask_id):  unmask to x_hat if c > omega_mask       (Gamma_t, kind 1)
 *   visible:                replace by x_hat if editable[r], x_hat != x and
 *                           c > omega_edit                          (Delta_t, kind 3)
 * Then, per block: if the block has masked rows and none of them was unmasked,
 * its masked row of highest confidence (lowest row on equal confidence) is
 * unmasked anyway (kind 2). Confidence comparisons use c rounded to float.
 * A row without a softmax (see row_softmax) keeps its token (kind 0) with
 * x_hat -1 and c, H NaN; it is never the forced row, so a block whose masked
 * rows all lack a softmax unmasks none. The call then returns ORC_UNDECIDABLE
 * after finishing every row and block.
 * block_changed[s][b] = 1 iff some row of block b got a new token (new != x);
 * seq_changes[s] = number of rows of s whose token changed.
 */
int oracle_denoise_update(const void* logits, int32_t dtype, int64_t row_stride, int32_t vocab,
                          const int32_t* cu_rows, int32_t num_seqs, int32_t block_size, int32_t max_blocks,
                          const int32_t* tokens, int32_t mask_id, float omega_mask, float omega_edit,
                          const uint8_t* editable, int32_t* new_tokens, uint8_t* kind, double* confidence,
                          int32_t* argmax_out, double* entropy, uint8_t* block_changed, int32_t* seq_changes) {
  if (num_seqs < 0 || vocab <= 0 || block_size <= 0 || dtype < 0 || dtype > 2 || row_stride < vocab)
    return ORC_BAD_ARG;
  const int32_t rows = num_seqs > 0 ? cu_rows[num_seqs] : 0;
  int undecidable = 0;
#pragma omp parallel for schedule(static)
  for (int32_t r = 0; r < rows; ++r) {
    const int64_t off = (int64_t)r * row_stride;
    double m = 0.0, ssum = 0.0;
    int32_t xh = -1;
    if (!row_softmax(logits, dtype, off, vocab, &m, &xh, &ssum)) {
#pragma omp atomic write
      undecidable = 1;
      confidence[r] = NAN;
      argmax_out[r] = -1;
      if (entropy) entropy[r] = NAN;
      kind[r] = 0;
      new_tokens[r] = tokens[r];
      continue;
    }
    double h = 0.0;
    for (int32_t v = 0; v < vocab; ++v) {
      const double pv = exp(load_logit(logits, dtype, off + v) - m) / ssum;
      if (pv > 0.0) h -= pv * log(pv);
    }
    const double c = 1.0 / ssum;
    confidence[r] = c;
    argmax_out[r] = xh;
    if (entropy) entropy[r] = h;
    const int32_t cur = tokens[r];
    uint8_t k = 0;
    if (cur == mask_id) {
      if ((float)c > omega_mask) k = 1;
    } else if ((editable == NULL || editable[r] != 0) && xh != cur && (float)c > omega_edit) {
      k = 3;
    }
    kind[r] = k;
    new_tokens[r] = k ? xh : cur;
  }
  for (int32_t s = 0; s < num_seqs; ++s) {
    const int32_t r0 = cu_rows[s], r1 = cu_rows[s + 1];
    const int32_t nblocks = (r1 - r0 + block_size - 1) / block_size;
    if (nblocks > max_blocks && block_changed) return ORC_BAD_ARG;
    int32_t changes = 0;
    for (int32_t b = 0; b < nblocks; ++b) {
      const int32_t b0 = r0 + b * block_size, b1 = (b0 + block_size < r1) ? b0 + block_size : r1;
      int any_masked = 0, any_unmasked = 0, best = -1;
      float best_c = 0.f;
      for (int32_t r = b0; r < b1; ++r) {
        if (tokens[r] != mask_id) continue;
        any_masked = 1;
        if (kind[r] == 1) any_unmasked = 1;
        if (argmax_out[r] < 0) continue; /* no softmax: never forced */
        if (best < 0 || (float)confidence[r] > best_c) {
          best = r;
          best_c = (float)confidence[r];
        }
      }
      if (any_masked && !any_unmasked && best >= 0) {
        kind[best] = 2;
        new_tokens[best] = argmax_out[best];
      }
      int changed = 0;
      for (int32_t r = b0; r < b1; ++r)
        if (new_tokens[r] != tokens[r]) {
          changed = 1;
          ++changes;
        }
      if (block_changed) block_changed[(int64_t)s * max_blocks + b] = (uint8_t)changed;
    }
    if (block_changed)
      for (int32_t b = nblocks; b < max_blocks; ++b) block_changed[(int64_t)s * max_blocks + b] = 0;
    if (seq_changes) seq_changes[s] = changes;
  }
  return undecidable ? ORC_UNDECIDABLE : ORC_OK;
}

static int cmp_desc(const void* a, const void* b) {
  const double x = *(const double*)a, y = *(const double*)b;
  return (x < y) - (x > y);
}

/*
 * Tail-entropy block selection, Eqs. 6-7. For each sequence s the caller keeps
 * the final standard-scope entropies of its last n_hist blocks in
 * block_entropy[s][0..n_hist-1][0..block_size-1], oldest block first (slot
 * n_hist-1 is block j-1); n_valid[s] <= n_hist of them exist. The candidates
 * of Eq. 7 are the last min(n_valid[s], k_max - 1) slots. For each candidate
 *   S_rho(i) = mean of the ceil(rho * block_size) largest entropies of block i
 * (Eq. 6); best_slot[s] is the candidate of largest score (the oldest one on
 * equal scores) and window_blocks[s] = n_hist - best_slot[s] + 1 is the number
 * of blocks of the editing window W_j = [j* B, (j+1) B) of Eq. 5. Sequences
 * without candidates get best_slot -1 and window_blocks 1. scores (optional)
 * receives S_rho for every candidate slot (NaN elsewhere).
 */
int oracle_tail_entropy_select(const float* block_entropy, const int32_t* n_valid, int32_t num_seqs, int32_t n_hist,
                               int32_t block_size, double rho, int32_t k_max, double* scores, int32_t* best_slot,
                               int32_t* window_blocks) {
  if (num_seqs < 0 || n_hist < 1 || block_size < 1 || k_max < 1 || !(rho > 0.0) || rho > 1.0) return ORC_BAD_ARG;
  const int32_t top = (int32_t)ceil(rho * block_size);
  double* buf = (double*)malloc(sizeof(double) * (size_t)block_size);
  if (!buf) return ORC_NOMEM;
  for (int32_t s = 0; s < num_seqs; ++s) {
    int32_t nv = n_valid[s] < n_hist ? n_valid[s] : n_hist;
    if (nv < 0) nv = 0;
    const int32_t ncand = nv < k_max - 1 ? nv : k_max - 1;
    int32_t best = -1;
    double best_score = -INFINITY;
    for (int32_t slot = 0; slot < n_hist; ++slot) {
      const int cand = slot >= n_hist - ncand;
      if (scores) scores[(int64_t)s * n_hist + slot] = NAN;
      if (!cand) continue;
      for (int32_t r = 0; r < block_size; ++r)
        buf[r] = (double)block_entropy[((int64_t)s * n_hist + slot) * block_size + r];
      qsort(buf, (size_t)block_size, sizeof(double), cmp_desc);
      double sum = 0.0;
      for (int32_t r = 0; r < top; ++r) sum += buf[r];
      const double sc = sum / top;
      if (scores) scores[(int64_t)s * n_hist + slot] = sc;
      if (best < 0 || (float)sc > (float)best_score) {
        best = slot;
        best_score = sc;
      }
    }
    best_slot[s] = best;
    window_blocks[s] = best < 0 ? 1 : n_hist - best + 1;
  }
  free(buf);
  return ORC_OK;
}

/*
 * Targeted refresh of the blocks that changed (Sec. 4.3 with the block-causal
 * conditioning of Sec. 2.2). Recomputing window block b of sequence s under
 * standard attention means that its queries see the cached prefix, the window
 * blocks before b as they stand in the cache (the changed ones are written
 * there first), and all of block b itself. That is one attention problem per
 * changed block: prefix P_s + b*B, a one-block window in bidirectional mode.
 * This lays those problems out as a ragged batch of E = batch * max_blocks
 * entries, entry e = s * max_blocks + b, empty unless block b of s changed:
 *   r_prefix_len[e] = P_s + b*B and r_window_len[e] = min(B, W_s - b*B)
 *                     for a changed block inside the window; 0 and 0 otherwise
 *   r_cu_window[e]  = sum of r_window_len[0..e-1]  (E + 1 values)
 *   r_mask_mode[e]  = 1 (bidirectional)
 *   r_block_table[e][:] = block_table[s][:] for a changed block, -1 otherwise
 *   r_src_row[k]    = cu_window[s] + b*B + i for refresh row k = r_cu_window[e] + i,
 *                     and -1 for k from r_cu_window[E] up to total_rows
 *   r_count[0] = changed entries, r_count[1] = r_cu_window[E]
 * A window longer than max_blocks * B, or more refresh rows than total_rows,
 * is an argument error.
 */
int oracle_refresh_plan(const uint8_t* block_changed, int32_t max_blocks, const int32_t* prefix_len,
                        const int32_t* window_len, const int32_t* cu_window, const int32_t* block_table,
                        int32_t max_pages_per_seq, int32_t batch, int32_t block_size, int32_t total_rows,
                        int32_t* r_prefix_len, int32_t* r_window_len, int32_t* r_cu_window, uint8_t* r_mask_mode,
                        int32_t* r_block_table, int32_t* r_src_row, int32_t* r_count) {
  if (batch < 0 || max_blocks < 1 || block_size < 1 || total_rows < 0 || max_pages_per_seq < 0) return ORC_BAD_ARG;
  for (int32_t s = 0; s < batch; ++s)
    if (window_len[s] < 0 || window_len[s] > max_blocks * block_size) return ORC_BAD_ARG;
  int32_t rows = 0, entries = 0;
  for (int32_t s = 0; s < batch; ++s) {
    for (int32_t b = 0; b < max_blocks; ++b) {
      const int64_t e = (int64_t)s * max_blocks + b;
      const int32_t start = b * block_size;
      const int changed = block_changed[e] != 0 && start < window_len[s];
      int32_t len = 0;
      if (changed) {
        len = window_len[s] - start;
        if (len > block_size) len = block_size;
      }
      r_cu_window[e] = rows;
      r_prefix_len[e] = changed ? prefix_len[s] + start : 0;
      r_window_len[e] = len;
      r_mask_mode[e] = 1;
      for (int32_t p = 0; p < max_pages_per_seq; ++p)
        r_block_table[e * max_pages_per_seq + p] = changed ? block_table[(int64_t)s * max_pages_per_seq + p] : -1;
      for (int32_t i = 0; i < len; ++i) {
        if (rows >= total_rows) return ORC_BAD_ARG;
        r_src_row[rows++] = cu_window[s] + start + i;
      }
      entries += changed;
    }
  }
  r_cu_window[(int64_t)batch * max_blocks] = rows;
  for (int32_t k = rows; k < total_rows; ++k) r_src_row[k] = -1;
  r_count[0] = entries;
  r_count[1] = rows;
  return ORC_OK;
}

/*
 * LM-head projection of the final hidden states (the logits the T2T rule of
 * Eq. 2 reads): l[r, v] = sum_k hidden[r, k] * weight[v, k] over k = 0..d-1,
 * bf16 inputs widened exactly to double, products and sums in double in
 * ascending k. If n_sel >= 0 only rows sel_rows[0..n_sel-1] are computed and
 * out holds them in that order ([n_sel, vocab]); else out is [rows, vocab].
 */
int oracle_lm_head_logits(const uint16_t* hidden, const uint16_t* weight, int32_t rows, int32_t vocab, int32_t d,
                          int32_t n_sel, const int32_t* sel_rows, double* out) {
  if (rows < 0 || vocab <= 0 || d <= 0) return ORC_BAD_ARG;
  const int64_t total = n_sel >= 0 ? n_sel : rows;
  for (int64_t u = 0; u < total; ++u) {
    const int32_t r = n_sel >= 0 ? sel_rows[u] : (int32_t)u;
    if (r < 0 || r >= rows) return ORC_BAD_ARG;
  }
  double* hrow = (double*)malloc(sizeof(double) * (size_t)d * (size_t)(total > 0 ? total : 1));
  if (!hrow) return ORC_NOMEM;
  for (int64_t u = 0; u < total; ++u) {
    const int32_t r = n_sel >= 0 ? sel_rows[u] : (int32_t)u;
    for (int32_t k = 0; k < d; ++k) hrow[u * d + k] = bf16_to_double(hidden[(int64_t)r * d + k]);
  }
#pragma omp parallel for schedule(static)
  for (int32_t v = 0; v < vocab; ++v) {
    double* wrow = (double*)malloc(sizeof(double) * (size_t)d);
    if (!wrow) continue;
    for (int32_t k = 0; k < d; ++k) wrow[k] = bf16_to_double(weight[(int64_t)v * d + k]);
    for (int64_t u = 0; u < total; ++u) {
      double acc = 0.0;
      for (int32_t k = 0; k < d; ++k) acc += hrow[u * d + k] * wrow[k];
      out[u * vocab + v] = acc;
    }
    free(wrow);
  }
  free(hrow);
  return ORC_OK;
}

/*
 * Cross-block attention mask of Multi-Block Edit SFT (Sec. 3, "Cross-block
 * attention mask"), at block granularity. The training sequence is
 * [prompt blocks 0..Np-1 | noisy blocks n_0..n_{N-1} | clean blocks c_0..c_{N-1}],
 * block b = Np + i for n_i and Np + N + j for c_j. Links (reading of the paper;
 * its supplement with the exact construction is not available):
 *   prompt -> prompt (all prompt blocks; prompt tokens are their own category)
 *   n_i -> prompt, n_i (NN), c_j for j < i (NC), c_j for i < j <= i+K-1 (NF)
 *   c_j -> prompt, c_j, c_k for k <= j-K (CC whose target is not reachable by
 *          a noisy block that sees c_j), n_i for j-K+1 <= i <= j-1 (CN)
 * With K = 1 this is the standard block-diffusion SFT mask (NN, NC, block-causal
 * CC). mask: nb = Np + 2N rows of words_per_row 32-bit words; bit k of row q is
 * set iff block q attends to block k.
 */
int oracle_sft_block_mask(int32_t n_prompt_blocks, int32_t n_blocks, int32_t K, int32_t words_per_row,
                          uint32_t* mask) {
  const int32_t Np = n_prompt_blocks, N = n_blocks, nb = Np + 2 * N;
  if (Np < 0 || N < 0 || K < 1 || words_per_row * 32 < nb) return ORC_BAD_ARG;
  memset(mask, 0, sizeof(uint32_t) * (size_t)nb * (size_t)words_per_row);
#define ORC_SET(q, k) (mask[(int64_t)(q) * words_per_row + (k) / 32] |= 1u << ((k) % 32))
  for (int32_t q = 0; q < nb; ++q)
    for (int32_t p = 0; p < Np; ++p) ORC_SET(q, p);
  for (int32_t i = 0; i < N; ++i) {
    const int32_t q = Np + i;
    ORC_SET(q, q);
    for (int32_t j = 0; j < N; ++j)
      if (j < i || (j > i && j <= i + K - 1)) ORC_SET(q, Np + N + j);
  }
  for (int32_t j = 0; j < N; ++j) {
    const int32_t q = Np + N + j;
    ORC_SET(q, q);
    for (int32_t k = 0; k <= j - K; ++k) ORC_SET(q, Np + N + k);
    for (int32_t i = j - K + 1; i <= j - 1; ++i)
      if (i >= 0) ORC_SET(q, Np + i);
  }
#undef ORC_SET
  return ORC_OK;
}

static int mask_bit(const uint32_t* mask, int32_t words_per_row, int32_t qb, int32_t kb) {
  return (mask[(int64_t)qb * words_per_row + kb / 32] >> (kb % 32)) & 1u;
}

/*
 * Attention of one training sequence under a block mask: query token i (block
 * i / B) attends to key token j iff bit (i / B, j / B) of the mask is set.
 * q [T, Hq, D], k/v [T, Hkv, D] bf16; query head h uses KV head h / (Hq/Hkv).
 * out [T, Hq, D] and lse [T, Hq] (natural log) in double; a row that sees no
 * key gets out = 0 and lse = -inf.
 */
int oracle_block_mask_attention(const uint16_t* q, const uint16_t* k, const uint16_t* v, int32_t T, int32_t Hq,
                                int32_t Hkv, int32_t D, int32_t B, const uint32_t* mask, int32_t words_per_row,
                                double scale, double* out, double* lse) {
  if (T < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || D <= 0 || B <= 0) return ORC_BAD_ARG;
  const int32_t G = Hq / Hkv;
  int status = ORC_OK;
#pragma omp parallel for schedule(dynamic)
  for (int64_t ih = 0; ih < (int64_t)T * Hq; ++ih) {
    const int32_t i = (int32_t)(ih / Hq), h = (int32_t)(ih % Hq), g = h / G;
    double* z = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1));
    if (!z) {
#pragma omp atomic write
      status = ORC_NOMEM;
      continue;
    }
    double m = -INFINITY;
    for (int32_t j = 0; j < T; ++j) {
      if (!mask_bit(mask, words_per_row, i / B, j / B)) {
        z[j] = -INFINITY;
        continue;
      }
      double s = 0.0;
      for (int32_t d = 0; d < D; ++d)
        s += bf16_to_double(q[((int64_t)i * Hq + h) * D + d]) * bf16_to_double(k[((int64_t)j * Hkv + g) * D + d]);
      z[j] = s * scale;
      if (z[j] > m) m = z[j];
    }
    double* o = out + ((int64_t)i * Hq + h) * D;
    for (int32_t d = 0; d < D; ++d) o[d] = 0.0;
    if (m == -INFINITY) {
      lse[(int64_t)i * Hq + h] = -INFINITY;
      free(z);
      continue;
    }
    double zs = 0.0;
    for (int32_t j = 0; j < T; ++j) {
      if (z[j] == -INFINITY) continue;
      const double p = exp(z[j] - m);
      zs += p;
      for (int32_t d = 0; d < D; ++d) o[d] += p * bf16_to_double(v[((int64_t)j * Hkv + g) * D + d]);
    }
    for (int32_t d = 0; d < D; ++d) o[d] /= zs;
    lse[(int64_t)i * Hq + h] = m + log(zs);
    free(z);
  }
  return status;
}

/*
 * Gradients of the block-masked attention above for an upstream gradient dO
 * (bf16 [T, Hq, D]), from the definitions, in double: with P the attention
 * probabilities (recomputed from q, k and the mask),
 *   dV_g = sum over the G heads of g of P^T dO
 *   dP   = dO V^T,  delta_i = sum_j P_ij dP_ij  (= dO_i . O_i)
 *   dS   = P o (dP - delta)
 *   dQ   = scale * dS K,  dK_g = scale * sum over the heads of g of dS^T Q
 * dq [T, Hq, D], dk / dv [T, Hkv, D] are written (overwritten) in double.
 */
int oracle_block_mask_attention_bwd(const uint16_t* q, const uint16_t* k, const uint16_t* v, const uint16_t* dout,
                                    int32_t T, int32_t Hq, int32_t Hkv, int32_t D, int32_t B, const uint32_t* mask,
                                    int32_t words_per_row, double scale, double* dq, double* dk, double* dv) {
  if (T < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || D <= 0 || B <= 0) return ORC_BAD_ARG;
  const int32_t G = Hq / Hkv;
  memset(dk, 0, sizeof(double) * (size_t)T * Hkv * D);
  memset(dv, 0, sizeof(double) * (size_t)T * Hkv * D);
  memset(dq, 0, sizeof(double) * (size_t)T * Hq * D);
  int status = ORC_OK;
  /* one KV head at a time so that dK / dV accumulate without races */
  for (int32_t g = 0; g < Hkv; ++g) {
    for (int32_t hh = 0; hh < G; ++hh) {
      const int32_t h = g * G + hh;
      double* P = (double*)malloc(sizeof(double) * (size_t)T * (size_t)(T > 0 ? T : 1));
      double* dS = (double*)malloc(sizeof(double) * (size_t)T * (size_t)(T > 0 ? T : 1));
      if (!P || !dS) {
        free(P);
        free(dS);
        return ORC_NOMEM;
      }
#pragma omp parallel for schedule(dynamic)
      for (int32_t i = 0; i < T; ++i) {
        double* Pi = P + (int64_t)i * T;
        double m = -INFINITY;
        for (int32_t j = 0; j < T; ++j) {
          if (!mask_bit(mask, words_per_row, i / B, j / B)) {
            Pi[j] = -INFINITY;
            continue;
          }
          double s = 0.0;
          for (int32_t d = 0; d < D; ++d)
            s += bf16_to_double(q[((int64_t)i * Hq + h) * D + d]) * bf16_to_double(k[((int64_t)j * Hkv + g) * D + d]);
          Pi[j] = s * scale;
          if (Pi[j] > m) m = Pi[j];
        }
        double zs = 0.0;
        for (int32_t j = 0; j < T; ++j) {
          Pi[j] = (m == -INFINITY || Pi[j] == -INFINITY) ? 0.0 : exp(Pi[j] - m);
          zs += Pi[j];
        }
        for (int32_t j = 0; j < T; ++j) Pi[j] = zs > 0.0 ? Pi[j] / zs : 0.0;
        /* dP_ij = dO_i . V_j; delta_i = sum_j P_ij dP_ij */
        double* dSi = dS + (int64_t)i * T;
        double delta = 0.0;
        for (int32_t j = 0; j < T; ++j) {
          double dp = 0.0;
          if (Pi[j] != 0.0)
            for (int32_t d = 0; d < D; ++d)
              dp += bf16_to_double(dout[((int64_t)i * Hq + h) * D + d]) * bf16_to_double(v[((int64_t)j * Hkv + g) * D + d]);
          dSi[j] = dp;
          delta += Pi[j] * dp;
        }
        for (int32_t j = 0; j < T; ++j) dSi[j] = Pi[j] * (dSi[j] - delta);
        /* dQ_i = scale * sum_j dS_ij K_j */
        for (int32_t d = 0; d < D; ++d) {
          double acc = 0.0;
          for (int32_t j = 0; j < T; ++j)
            if (dSi[j] != 0.0) acc += dSi[j] * bf16_to_double(k[((int64_t)j * Hkv + g) * D + d]);
          dq[((int64_t)i * Hq + h) * D + d] = scale * acc;
        }
      }
      /* dV_j += sum_i P_ij dO_i ; dK_j += scale * sum_i dS_ij Q_i */
#pragma omp parallel for schedule(static)
      for (int32_t j = 0; j < T; ++j) {
        for (int32_t d = 0; d < D; ++d) {
          double av = 0.0, ak = 0.0;
          for (int32_t i = 0; i < T; ++i) {
            const double p = P[(int64_t)i * T + j], ds = dS[(int64_t)i * T + j];
            if (p != 0.0) av += p * bf16_to_double(dout[((int64_t)i * Hq + h) * D + d]);
            if (ds != 0.0) ak += ds * bf16_to_double(q[((int64_t)i * Hq + h) * D + d]);
          }
          dv[((int64_t)j * Hkv + g) * D + d] += av;
          dk[((int64_t)j * Hkv + g) * D + d] += scale * ak;
        }
      }
      free(P);
      free(dS);
    }
  }
  return status;
}
