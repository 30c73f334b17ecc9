"""Pins of the targeted-refresh layout oracle (Sec. 4.3 with the block-causal
conditioning of Sec. 2.2). CPU only.

The refresh recomputes only the window blocks that changed. The oracle lays
that out as one attention problem per changed block (prefix P + b*B, a
one-block bidirectional window). These tests pin the layout by a worked
example and tie the composite (refresh write + refresh attention) to the
block-causal window attention of the whole window, which the attention oracle
computes independently.
"""
import numpy as np
import pytest

import oracle
from paper_2607_22663_gb300.workloads import BLOCK_CAUSAL, BIDIRECTIONAL, attention_problem, bf16_bits


def test_hand_worked_layout():
    # Two sequences, B = 32: s0 has P = 10, W = 64 (blocks 0, 1; block 1
    # changed); s1 has P = 0, W = 40 (blocks 0 and a partial block 1 of 8
    # rows, both changed). cu_window = [0, 64, 104].
    #   entry (0,0): unchanged                    -> prefix 0,  window 0
    #   entry (0,1): rows 32..63 of s0            -> prefix 10 + 32 = 42, window 32
    #   entry (1,0): rows 64..95                  -> prefix 0,  window 32
    #   entry (1,1): rows 96..103 (partial block) -> prefix 32, window 8
    bt = np.arange(8, dtype=np.int32).reshape(2, 4)
    o = oracle.refresh_plan(np.array([[0, 1], [1, 1]]), [10, 0], [64, 40], [0, 64, 104], bt, 32)
    np.testing.assert_array_equal(o["prefix_len"], [0, 42, 0, 32])
    np.testing.assert_array_equal(o["window_len"], [0, 32, 32, 8])
    np.testing.assert_array_equal(o["cu_window"], [0, 0, 32, 64, 72])
    np.testing.assert_array_equal(o["mask_mode"], [1, 1, 1, 1])
    np.testing.assert_array_equal(o["block_table"], [[-1] * 4, [0, 1, 2, 3], [4, 5, 6, 7], [4, 5, 6, 7]])
    expect_rows = list(range(32, 64)) + list(range(64, 104)) + [-1] * 32
    np.testing.assert_array_equal(o["src_row"], expect_rows)
    np.testing.assert_array_equal(o["count"], [3, 72])


def test_no_change_gives_an_empty_batch():
    o = oracle.refresh_plan(np.zeros((3, 2), np.uint8), [5, 6, 7], [64, 32, 0], [0, 64, 96, 96],
                            np.zeros((3, 3), np.int32), 32)
    assert o["count"].tolist() == [0, 0]
    assert not o["window_len"].any() and not o["prefix_len"].any()
    assert (o["cu_window"] == 0).all() and (o["src_row"] == -1).all() and (o["block_table"] == -1).all()


def test_flags_past_the_window_are_ignored():
    # s0 has one block but its flag for block 2 is set; s1 is empty.
    o = oracle.refresh_plan(np.array([[1, 0, 1], [1, 1, 1]]), [0, 4], [20, 0], [0, 20, 20],
                            np.zeros((2, 1), np.int32), 32)
    np.testing.assert_array_equal(o["window_len"], [20, 0, 0, 0, 0, 0])
    assert o["count"].tolist() == [1, 20]


def test_window_longer_than_the_flags_is_an_error():
    with pytest.raises(RuntimeError):
        oracle.refresh_plan(np.ones((1, 1), np.uint8), [0], [40], [0, 40], np.zeros((1, 2), np.int32), 32)


def _refresh(prob, changed, k_src, v_src, k_cache, v_cache):
    """Refresh through the oracle: plan, write the changed blocks' K/V into the
    cache, attend each changed block. Returns (plan, out rows, cache after)."""
    q, kw, vw = bf16_bits(prob.q), bf16_bits(k_src), bf16_bits(v_src)
    plan = oracle.refresh_plan(changed, prob.prefix_len.numpy(), prob.window_len.numpy(), prob.cu_window.numpy(),
                               prob.block_table.numpy(), prob.block_size)
    rows = plan["src_row"][:plan["count"][1]]
    kc, vc = oracle.kv_window_write(kw[rows], vw[rows], k_cache, v_cache, plan["block_table"], plan["prefix_len"],
                                    plan["window_len"], plan["cu_window"], prob.block_size)
    out, _ = oracle.window_attention(q[rows], kw[rows], vw[rows], kc, vc, plan["block_table"], plan["prefix_len"],
                                     plan["window_len"], plan["cu_window"], plan["mask_mode"], prob.block_size,
                                     prob.page_size)
    return plan, out, (kc, vc)


def test_refresh_of_every_block_is_the_block_causal_window():
    # Sec. 2.2: with every block changed, recomputing the blocks one by one over
    # the refreshed cache is block-causal attention over the whole window.
    B = 16
    prob = attention_problem([37, 0, 80], [48, 40, 16], [BIDIRECTIONAL] * 3, 4, 2, 32, B, 16, seed=11)
    changed = np.ones((3, 3), np.uint8)
    plan, out_r, _ = _refresh(prob, changed, prob.k_win, prob.v_win, bf16_bits(prob.k_cache), bf16_bits(prob.v_cache))
    rows = plan["src_row"][:plan["count"][1]]
    assert sorted(rows.tolist()) == list(range(int(prob.cu_window[-1])))
    causal = oracle.window_attention(bf16_bits(prob.q), bf16_bits(prob.k_win), bf16_bits(prob.v_win),
                                     bf16_bits(prob.k_cache), bf16_bits(prob.v_cache), prob.block_table.numpy(),
                                     prob.prefix_len.numpy(), prob.window_len.numpy(), prob.cu_window.numpy(),
                                     np.full(3, BLOCK_CAUSAL, np.uint8), B, 16)[0]
    np.testing.assert_allclose(out_r, causal[rows], rtol=0, atol=1e-12)


def test_refresh_of_some_blocks_sees_the_cached_unchanged_blocks():
    # Unchanged blocks keep the K/V already in the cache (written when they were
    # committed); changed blocks get fresh K/V. Each changed block must equal
    # block-causal attention over a window whose unchanged blocks carry the
    # cached K/V and whose changed blocks carry the fresh K/V.
    B = 16
    prob = attention_problem([21, 64, 5], [48, 64, 33], [BIDIRECTIONAL] * 3, 6, 3, 32, B, 8, seed=12)
    old = attention_problem([21, 64, 5], [48, 64, 33], [BIDIRECTIONAL] * 3, 6, 3, 32, B, 8, seed=13)
    changed = np.array([[0, 1, 1, 0, 0], [1, 0, 1, 0, 0], [0, 0, 1, 0, 0]], np.uint8)
    # the cache as the earlier decoding left it: prefix plus the committed (old) window K/V
    kc0, vc0 = oracle.kv_window_write(bf16_bits(old.k_win), bf16_bits(old.v_win), bf16_bits(prob.k_cache),
                                      bf16_bits(prob.v_cache), prob.block_table.numpy(), prob.prefix_len.numpy(),
                                      prob.window_len.numpy(), prob.cu_window.numpy(), B)
    plan, out_r, (kc1, vc1) = _refresh(prob, changed, prob.k_win, prob.v_win, kc0, vc0)
    rows = plan["src_row"][:plan["count"][1]]
    assert plan["count"].tolist() == [5, len(rows)]
    # the window as the refresh sees it: fresh rows for changed blocks, cached rows elsewhere
    use_new = np.zeros(int(prob.cu_window[-1]), bool)
    use_new[rows] = True
    kmix = np.where(use_new[:, None, None], bf16_bits(prob.k_win), bf16_bits(old.k_win))
    vmix = np.where(use_new[:, None, None], bf16_bits(prob.v_win), bf16_bits(old.v_win))
    causal = oracle.window_attention(bf16_bits(prob.q), kmix, vmix, kc0, vc0, prob.block_table.numpy(),
                                     prob.prefix_len.numpy(), prob.window_len.numpy(), prob.cu_window.numpy(),
                                     np.full(3, BLOCK_CAUSAL, np.uint8), B, 8)[0]
    np.testing.assert_allclose(out_r, causal[rows], rtol=0, atol=1e-12)
    # and the cache after the refresh holds exactly that mixed window
    kc2, vc2 = oracle.kv_window_write(kmix, vmix, kc0, vc0, prob.block_table.numpy(), prob.prefix_len.numpy(),
                                      prob.window_len.numpy(), prob.cu_window.numpy(), B)
    np.testing.assert_array_equal(kc1, kc2)
    np.testing.assert_array_equal(vc1, vc2)
