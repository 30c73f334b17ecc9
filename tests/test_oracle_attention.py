"""Pins of the attention oracle (Eq. 5, Sec. 2.2) against library routines,
closed forms and invariants. CPU only."""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, BLOCK_CAUSAL, AttnProblem, attention_problem, bf16_bits
from tests._util import dense_keys, np_logsumexp, oracle_attention

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _sdpa_reference(prob, s, h, mask=None, scale=None):
    """torch float64 scaled_dot_product_attention over the densely gathered keys."""
    G = prob.num_q_heads // prob.num_kv_heads
    K, V = dense_keys(prob, s, h // G)
    t0 = int(prob.cu_window[s])
    W = prob.window_host[s]
    q = prob.q[t0:t0 + W, h].double()
    scale = scale if scale is not None else 1.0 / math.sqrt(prob.head_dim)
    o = F.scaled_dot_product_attention(q[None, None], K[None, None], V[None, None],
                                       attn_mask=None if mask is None else mask[None, None], scale=scale)[0, 0]
    scores = (q @ K.T) * scale
    if mask is not None:
        scores = scores.masked_fill(~mask, float("-inf"))
    return o, torch.from_numpy(np_logsumexp(scores.numpy(), axis=1))


def _paper_mask(P, W, mode, B):
    """Visibility from Eq. 5 / Sec. 2.2 written with torch broadcasting."""
    i = torch.arange(W)[:, None]
    j = torch.arange(P + W)[None, :]
    if mode == BIDIRECTIONAL:
        return torch.ones(W, P + W, dtype=torch.bool)
    return (j < P) | (((j - P).clamp(min=0) // B) <= (i // B))


CASES = [
    # prefix, window, modes, Hq, Hkv, D, B, page
    ([64], [64], [BIDIRECTIONAL], 4, 1, 64, 32, 32),
    ([0, 37, 96], [32, 64, 96], [BLOCK_CAUSAL, BIDIRECTIONAL, BLOCK_CAUSAL], 4, 2, 16, 32, 16),
    ([130, 5], [48, 20], [BLOCK_CAUSAL, BLOCK_CAUSAL], 8, 2, 8, 16, 8),
    ([300], [24], [BIDIRECTIONAL], 2, 2, 32, 8, 64),
]


@pytest.mark.parametrize("case", CASES)
def test_oracle_matches_sdpa_with_explicit_mask(case):
    prefix, window, modes, Hq, Hkv, D, B, ps = case
    prob = attention_problem(prefix, window, modes, Hq, Hkv, D, B, ps, seed=11)
    out, lse = oracle_attention(prob)
    for s in range(prob.batch):
        t0 = int(prob.cu_window[s])
        W = window[s]
        mask = _paper_mask(prefix[s], W, modes[s], B)
        for h in range(Hq):
            ref, ref_lse = _sdpa_reference(prob, s, h, mask)
            np.testing.assert_allclose(out[t0:t0 + W, h], ref.numpy(), rtol=0, atol=1e-12)
            np.testing.assert_allclose(lse[t0:t0 + W, h], ref_lse.numpy(), rtol=0, atol=1e-12)


def test_one_block_window_is_standard_block_diffusion_pass():
    """W = B: block-causal and bidirectional both reduce to plain (mask-free)
    attention over prefix + the block (Sec. 2.2 standard pass)."""
    prob = attention_problem([96, 40], [32, 32], [BLOCK_CAUSAL, BLOCK_CAUSAL], 4, 1, 32, 32, 16, seed=5)
    out_c, _ = oracle_attention(prob)
    prob_b = AttnProblem(**{**prob.__dict__, "mask_mode": torch.tensor([1, 1], dtype=torch.uint8),
                            "mode_host": [1, 1]})
    out_b, _ = oracle_attention(prob_b)
    np.testing.assert_array_equal(out_c, out_b)
    for s in range(2):
        t0 = int(prob.cu_window[s])
        for h in range(4):
            ref, _ = _sdpa_reference(prob, s, h, mask=None)
            np.testing.assert_allclose(out_c[t0:t0 + 32, h], ref.numpy(), rtol=0, atol=1e-12)


def test_block_size_one_is_causal_attention():
    """B = 1 (Sec. 2.2 with one-token blocks): each window query sees the prefix
    and the window keys up to itself. Without a prefix that is torch's own causal
    attention (is_causal); with one, the window part of the mask is a lower triangle."""
    W, D = 24, 32
    prob = attention_problem([0], [W], [BLOCK_CAUSAL], 4, 2, D, 1, 8, seed=41)
    out, lse = oracle_attention(prob)
    for h in range(4):
        K, V = dense_keys(prob, 0, h // 2)
        q = prob.q[:W, h].double()
        ref = F.scaled_dot_product_attention(q[None, None], K[None, None], V[None, None], is_causal=True,
                                             scale=1.0 / math.sqrt(D))[0, 0]
        np.testing.assert_allclose(out[:W, h], ref.numpy(), rtol=0, atol=1e-12)
    P = 37
    prob = attention_problem([P], [W], [BLOCK_CAUSAL], 4, 2, D, 1, 8, seed=42)
    out, lse = oracle_attention(prob)
    mask = torch.cat([torch.ones(W, P, dtype=torch.bool), torch.ones(W, W, dtype=torch.bool).tril()], dim=1)
    for h in range(4):
        ref, ref_lse = _sdpa_reference(prob, 0, h, mask)
        np.testing.assert_allclose(out[:W, h], ref.numpy(), rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[:W, h], ref_lse.numpy(), rtol=0, atol=1e-12)


def test_block_at_least_as_long_as_the_window_is_bidirectional():
    """B >= W: the whole window is one block, so block-causal and bidirectional
    attention (Eq. 5) coincide exactly."""
    for B in (64, 128):
        prob = attention_problem([70], [64], [BLOCK_CAUSAL], 4, 1, 32, B, 16, seed=43)
        out_c, lse_c = oracle_attention(prob)
        prob_b = AttnProblem(**{**prob.__dict__, "mask_mode": torch.tensor([BIDIRECTIONAL], dtype=torch.uint8),
                                "mode_host": [BIDIRECTIONAL]})
        out_b, lse_b = oracle_attention(prob_b)
        np.testing.assert_array_equal(out_c, out_b)
        np.testing.assert_array_equal(lse_c, lse_b)


def test_block_causal_equals_sequential_single_block_passes():
    """k blocks in block-causal mode == decoding them one block at a time, each
    pass seeing the prefix plus the earlier window blocks as cached history."""
    B, k, P, D = 16, 3, 40, 32
    prob = attention_problem([P], [k * B], [BLOCK_CAUSAL], 4, 2, D, B, 8, seed=21)
    out, lse = oracle_attention(prob)
    for b in range(k):
        # build a one-block problem whose prefix = original prefix + window blocks < b
        Pb = P + b * B
        ps = prob.page_size
        npages = (Pb + ps - 1) // ps
        kc = torch.zeros(npages, 2, ps, D, dtype=torch.bfloat16)
        vc = torch.zeros_like(kc)
        Kd0, Vd0 = dense_keys(prob, 0, 0)
        Kd1, Vd1 = dense_keys(prob, 0, 1)
        for pos in range(Pb):
            kc[pos // ps, 0, pos % ps] = Kd0[pos].to(torch.bfloat16)
            vc[pos // ps, 0, pos % ps] = Vd0[pos].to(torch.bfloat16)
            kc[pos // ps, 1, pos % ps] = Kd1[pos].to(torch.bfloat16)
            vc[pos // ps, 1, pos % ps] = Vd1[pos].to(torch.bfloat16)
        rows = slice(b * B, (b + 1) * B)
        sub = AttnProblem(q=prob.q[rows].clone(), k_win=prob.k_win[rows].clone(), v_win=prob.v_win[rows].clone(),
                          k_cache=kc, v_cache=vc, block_table=torch.arange(npages, dtype=torch.int32)[None],
                          prefix_len=torch.tensor([Pb], dtype=torch.int32),
                          window_len=torch.tensor([B], dtype=torch.int32),
                          cu_window=torch.tensor([0, B], dtype=torch.int32),
                          mask_mode=torch.tensor([BLOCK_CAUSAL], dtype=torch.uint8), block_size=B, page_size=ps,
                          prefix_host=[Pb], window_host=[B], mode_host=[BLOCK_CAUSAL])
        o_b, l_b = oracle_attention(sub)
        np.testing.assert_allclose(out[rows], o_b, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[rows], l_b, rtol=0, atol=1e-12)


def test_probability_probe_rows_sum_to_one_and_masked_are_zero():
    """With V = identity over key positions (D >= #keys), the output row IS the
    attention probability row: entries sum to 1 and masked keys get exactly 0."""
    B, P, W, D = 8, 20, 24, 64
    prob = attention_problem([P], [W], [BLOCK_CAUSAL], 2, 1, D, B, 8, seed=3)
    eye = torch.eye(D, dtype=torch.bfloat16)
    Kd, _ = dense_keys(prob, 0, 0)
    vc = torch.zeros_like(prob.v_cache)
    for pos in range(P):
        vc[prob.block_table[0, pos // 8], 0, pos % 8] = eye[pos]
    vw = torch.zeros_like(prob.v_win)
    for j in range(W):
        vw[j, 0] = eye[P + j]
    probe = AttnProblem(**{**prob.__dict__, "v_cache": vc, "v_win": vw})
    out, _ = oracle_attention(probe)
    mask = _paper_mask(P, W, BLOCK_CAUSAL, B)
    for h in range(2):
        pr = out[:, h, :P + W]
        np.testing.assert_allclose(pr.sum(axis=1), 1.0, atol=1e-13)
        assert (pr[~mask.numpy()] == 0).all()
        assert (pr[mask.numpy()] > 0).all()
        assert (out[:, h, P + W:] == 0).all()


def test_bidirectional_invariant_to_permuting_window_keys():
    B = 16
    prob = attention_problem([50, 17], [48, 32], [BIDIRECTIONAL, BIDIRECTIONAL], 4, 2, 32, B, 16, seed=8)
    out, _ = oracle_attention(prob)
    g = torch.Generator().manual_seed(1)
    kw, vw = prob.k_win.clone(), prob.v_win.clone()
    for s in range(2):
        t0, W = int(prob.cu_window[s]), prob.window_host[s]
        perm = torch.randperm(W, generator=g) + t0
        kw[t0:t0 + W] = prob.k_win[perm]
        vw[t0:t0 + W] = prob.v_win[perm]
    out2, _ = oracle_attention(AttnProblem(**{**prob.__dict__, "k_win": kw, "v_win": vw}))
    np.testing.assert_allclose(out, out2, rtol=0, atol=1e-12)
    # block-causal is NOT invariant: the pin distinguishes the two modes
    pc = AttnProblem(**{**prob.__dict__, "mask_mode": torch.tensor([0, 0], dtype=torch.uint8), "mode_host": [0, 0]})
    oc1, _ = oracle_attention(pc)
    oc2, _ = oracle_attention(AttnProblem(**{**pc.__dict__, "k_win": kw, "v_win": vw}))
    assert np.abs(oc1 - oc2).max() > 1e-3


def test_invariant_to_physical_page_permutation():
    prob = attention_problem([77, 130], [32, 32], [BIDIRECTIONAL, BLOCK_CAUSAL], 4, 2, 16, 16, 8, seed=9,
                             shuffle_pages=False)
    out, lse = oracle_attention(prob)
    g = torch.Generator().manual_seed(2)
    perm = torch.randperm(prob.num_pages, generator=g)  # new position of old page i: perm[i]
    kc = torch.empty_like(prob.k_cache)
    vc = torch.empty_like(prob.v_cache)
    kc[perm] = prob.k_cache
    vc[perm] = prob.v_cache
    bt = prob.block_table.clone()
    valid = bt >= 0
    bt[valid] = perm[bt[valid].long()].to(torch.int32)
    out2, lse2 = oracle_attention(AttnProblem(**{**prob.__dict__, "k_cache": kc, "v_cache": vc, "block_table": bt}))
    np.testing.assert_array_equal(out, out2)
    np.testing.assert_array_equal(lse, lse2)


def test_gqa_equals_replicated_kv_heads():
    prob = attention_problem([45], [32], [BLOCK_CAUSAL], 8, 2, 16, 16, 16, seed=4)
    out, _ = oracle_attention(prob)
    rep = lambda t: t.repeat_interleave(4, dim=1)
    prob_r = AttnProblem(**{**prob.__dict__, "k_win": rep(prob.k_win), "v_win": rep(prob.v_win),
                            "k_cache": rep(prob.k_cache), "v_cache": rep(prob.v_cache)})
    out_r, _ = oracle_attention(prob_r)
    np.testing.assert_array_equal(out, out_r)


@pytest.mark.parametrize("mode", [BIDIRECTIONAL, BLOCK_CAUSAL])
def test_split_invariance_prefix_and_window_merge_by_lse(mode):
    """Attention over prefix + window equals the log-sum-exp merge of attention
    over the prefix alone and over the window alone (the identity split-KV
    merging relies on). With P = W the prefix-only part is the oracle itself,
    run with no prefix on a window made of the prefix rows (bidirectional)."""
    P = W = 48
    prob = attention_problem([P], [W], [mode], 4, 2, 16, 16, 16, seed=21)
    full, full_lse = oracle_attention(prob)
    no_prefix = {"prefix_len": torch.tensor([0], dtype=torch.int32), "prefix_host": [0]}
    ow, lw = oracle_attention(AttnProblem(**{**prob.__dict__, **no_prefix}))
    pos = torch.arange(P)
    pages = prob.block_table[0][pos // prob.page_size].long()
    kp = prob.k_cache[pages, :, pos % prob.page_size]          # [P, Hkv, D], rows in logical order
    vp = prob.v_cache[pages, :, pos % prob.page_size]
    op, lp = oracle_attention(AttnProblem(**{**prob.__dict__, **no_prefix, "k_win": kp, "v_win": vp,
                                             "mask_mode": torch.tensor([BIDIRECTIONAL], dtype=torch.uint8),
                                             "mode_host": [BIDIRECTIONAL]}))
    m = np.maximum(lp, lw)
    wp, ww = np.exp(lp - m), np.exp(lw - m)
    merged = (wp[..., None] * op + ww[..., None] * ow) / (wp + ww)[..., None]
    np.testing.assert_allclose(full, merged, rtol=0, atol=1e-12)
    np.testing.assert_allclose(full_lse, m + np.log(wp + ww), rtol=0, atol=1e-12)


def test_units_subset_matches_full():
    prob = attention_problem([60, 33], [32, 64], [BIDIRECTIONAL, BLOCK_CAUSAL], 4, 2, 16, 32, 16, seed=12)
    out, lse = oracle_attention(prob)
    sub, sub_lse = oracle_attention(prob, units=[(1, 3), (0, 0)])
    t1 = int(prob.cu_window[1])
    np.testing.assert_array_equal(sub[t1:t1 + 64, 3], out[t1:t1 + 64, 3])
    np.testing.assert_array_equal(sub[0:32, 0], out[0:32, 0])
    assert np.isnan(sub[0:32, 1]).all()


def test_golden_closed_forms():
    spec = json.load(open(os.path.join(GOLDEN, "attention_closed_forms.json")))
    bf = lambda x: torch.tensor(x, dtype=torch.bfloat16)
    q = bf(spec["q"])[:, None, :]            # [2, 1, 2]
    kw = bf(spec["window_k"])[:, None, :]
    vw = bf(spec["window_v"])[:, None, :]
    kc = bf(spec["prefix_k"]).reshape(1, 1, 1, 2)
    vc = bf(spec["prefix_v"]).reshape(1, 1, 1, 2)
    for case in spec["cases"]:
        prob = AttnProblem(q=q, k_win=kw, v_win=vw, k_cache=kc, v_cache=vc,
                           block_table=torch.zeros(1, 1, dtype=torch.int32),
                           prefix_len=torch.tensor([1], dtype=torch.int32),
                           window_len=torch.tensor([2], dtype=torch.int32),
                           cu_window=torch.tensor([0, 2], dtype=torch.int32),
                           mask_mode=torch.tensor([case["mode"]], dtype=torch.uint8),
                           block_size=case["block_size"], page_size=1, prefix_host=[1], window_host=[2],
                           mode_host=[case["mode"]])
        out, _ = oracle_attention(prob, scale=1.0)
        expected = np.array([[eval(e, {"math": math}) for e in row] for row in case["expected"]])
        np.testing.assert_allclose(out[:, 0, :], expected, rtol=0, atol=1e-14, err_msg=case["name"])


def test_bad_page_id_is_reported():
    import oracle
    prob = attention_problem([40], [16], [BIDIRECTIONAL], 2, 1, 8, 16, 8, seed=1)
    bt = prob.block_table.clone()
    bt[0, 1] = prob.num_pages + 3
    with pytest.raises(RuntimeError, match="page"):
        oracle_attention(AttnProblem(**{**prob.__dict__, "block_table": bt}))
