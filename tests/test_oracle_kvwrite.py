"""Pins of the KV window write oracle (Sec. 4.3 targeted refresh). CPU only."""
import numpy as np
import torch

import oracle
from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, BLOCK_CAUSAL, AttnProblem, attention_problem, bf16_bits
from tests._util import dense_keys, oracle_attention


def _write(prob, mask=None):
    return oracle.kv_window_write(bf16_bits(prob.k_win), bf16_bits(prob.v_win), bf16_bits(prob.k_cache),
                                  bf16_bits(prob.v_cache), prob.block_table.numpy(), prob.prefix_len.numpy(),
                                  prob.window_len.numpy(), prob.cu_window.numpy(), prob.block_size,
                                  block_write_mask=mask)


def test_window_lands_at_logical_positions_and_nothing_else_changes():
    prob = attention_problem([37, 64, 0], [32, 48, 16], [BIDIRECTIONAL] * 3, 4, 2, 16, 16, 16, seed=3, spare_pages=5)
    kc0, vc0 = bf16_bits(prob.k_cache), bf16_bits(prob.v_cache)
    kc, vc = _write(prob)
    touched = np.zeros(kc.shape[:3], dtype=bool)
    kw, vw = bf16_bits(prob.k_win), bf16_bits(prob.v_win)
    for s in range(prob.batch):
        P, W, t0 = prob.prefix_host[s], prob.window_host[s], int(prob.cu_window[s])
        for i in range(W):
            pos = P + i
            page = int(prob.block_table[s, pos // 16])
            np.testing.assert_array_equal(kc[page, :, pos % 16], kw[t0 + i])
            np.testing.assert_array_equal(vc[page, :, pos % 16], vw[t0 + i])
            touched[page, :, pos % 16] = True
    np.testing.assert_array_equal(kc[~touched], kc0[~touched])
    np.testing.assert_array_equal(vc[~touched], vc0[~touched])


def test_block_write_mask_writes_only_changed_blocks():
    B = 16
    prob = attention_problem([20, 48], [48, 32], [BLOCK_CAUSAL] * 2, 2, 1, 8, B, 8, seed=4)
    mask = np.array([[1, 0, 1], [0, 1, 0]], dtype=np.uint8)
    kc0 = bf16_bits(prob.k_cache)
    kc, _ = _write(prob, mask)
    kw = bf16_bits(prob.k_win)
    for s in range(2):
        P, W, t0 = prob.prefix_host[s], prob.window_host[s], int(prob.cu_window[s])
        for i in range(W):
            pos = P + i
            page = int(prob.block_table[s, pos // 8])
            if mask[s, i // B]:
                np.testing.assert_array_equal(kc[page, :, pos % 8], kw[t0 + i])
            else:
                np.testing.assert_array_equal(kc[page, :, pos % 8], kc0[page, :, pos % 8])


def test_written_window_serves_as_prefix_of_the_next_pass():
    """After refreshing block b's KV, a standard pass of the next block with
    prefix P+W equals the same pass with block b supplied as a window: the
    cache write and the paged read agree on logical positions."""
    B, P = 16, 40
    first = attention_problem([P], [B], [BLOCK_CAUSAL], 4, 2, 16, B, 8, seed=6, reserve_tokens=[2 * B])
    kc, vc = _write(first)
    nxt = attention_problem([P + B], [B], [BLOCK_CAUSAL], 4, 2, 16, B, 8, seed=7)
    view = lambda a: torch.from_numpy(a.astype(np.int16)).view(torch.bfloat16)
    after = AttnProblem(**{**nxt.__dict__, "k_cache": view(kc), "v_cache": view(vc),
                           "block_table": first.block_table})
    out_a, _ = oracle_attention(after)
    # same keys, with block b given explicitly as part of a 2-block window
    two = AttnProblem(q=torch.cat([first.q, nxt.q]), k_win=torch.cat([first.k_win, nxt.k_win]),
                      v_win=torch.cat([first.v_win, nxt.v_win]), k_cache=first.k_cache, v_cache=first.v_cache,
                      block_table=first.block_table, prefix_len=torch.tensor([P], dtype=torch.int32),
                      window_len=torch.tensor([2 * B], dtype=torch.int32),
                      cu_window=torch.tensor([0, 2 * B], dtype=torch.int32),
                      mask_mode=torch.tensor([BLOCK_CAUSAL], dtype=torch.uint8), block_size=B, page_size=8,
                      prefix_host=[P], window_host=[2 * B], mode_host=[BLOCK_CAUSAL])
    out_two, _ = oracle_attention(two)
    np.testing.assert_allclose(out_a, out_two[B:], rtol=0, atol=1e-12)
