"""Parity of the CUDA window attention (mbe_window_attention) with the fp64
oracle, called through the C ABI. Tolerance: max abs error 1e-2 on bf16
outputs (plus an LSE check)."""
import numpy as np
import pytest
import torch

from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300 import workloads as wl
from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, BLOCK_CAUSAL, AttnProblem, attention_problem
from tests._gpu import compare_attention, run_attention, subproblem

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _sample(n, k, seed):
    g = torch.Generator().manual_seed(seed)
    return sorted(torch.randperm(n, generator=g)[:k].tolist())


def test_tiny_workload_full():
    w = wl.tiny(DEV)
    prob = w["attn"][0]
    out, lse = run_attention(prob)
    compare_attention(prob, out, lse)


def test_batch8_workload_full():
    prob = wl.batch8(DEV)["attn"][0]
    out, lse = run_attention(prob)
    compare_attention(prob, out, lse)


RAGGED = [
    # prefix, window, modes, Hq, Hkv, D, B, page
    ([0, 37, 300, 129], [32, 96, 64, 160], [BLOCK_CAUSAL, BIDIRECTIONAL, BLOCK_CAUSAL, BIDIRECTIONAL], 16, 4, 128, 32, 32),
    ([200, 1000], [64, 32], [BIDIRECTIONAL, BLOCK_CAUSAL], 8, 8, 128, 32, 16),       # G = 1
    ([513, 64], [48, 16], [BLOCK_CAUSAL, BIDIRECTIONAL], 32, 4, 128, 16, 256),        # G = 8, page 256
    ([255, 700, 1], [64, 128, 8], [BIDIRECTIONAL, BLOCK_CAUSAL, BIDIRECTIONAL], 8, 2, 64, 32, 64),   # D = 64
    ([130, 90], [40, 24], [BLOCK_CAUSAL, BLOCK_CAUSAL], 4, 2, 128, 8, 8),            # page 8, odd windows
    ([4000], [256], [BLOCK_CAUSAL], 16, 4, 128, 32, 128),                          # 4 query slabs
    # the other group sizes GQA packing allows: a 128-row tile holds 128 / G tokens
    ([2100, 45], [96, 64], [BLOCK_CAUSAL, BIDIRECTIONAL], 8, 4, 128, 32, 32),       # G = 2
    ([1500, 300], [32, 72], [BIDIRECTIONAL, BLOCK_CAUSAL], 32, 2, 128, 32, 32),     # G = 16
    ([800], [64], [BLOCK_CAUSAL], 32, 1, 128, 16, 64),                             # G = 32: 4 tokens per tile
    ([257, 30], [24, 40], [BLOCK_CAUSAL, BIDIRECTIONAL], 128, 1, 64, 8, 16),        # G = 128: 1 token per tile
    # block sizes: 1 (block-causal is then causal), 48 (not a power of two), 128 > W
    ([150], [40], [BLOCK_CAUSAL], 16, 4, 128, 1, 32),
    ([500, 61], [96, 144], [BLOCK_CAUSAL, BLOCK_CAUSAL], 16, 4, 128, 48, 32),
    ([700], [64], [BLOCK_CAUSAL], 16, 4, 128, 128, 64),
]


@pytest.mark.parametrize("case", RAGGED)
def test_ragged_shapes(case):
    prefix, window, modes, Hq, Hkv, D, B, ps = case
    prob = attention_problem(prefix, window, modes, Hq, Hkv, D, B, ps, seed=31, device=DEV, spare_pages=3)
    out, lse = run_attention(prob)
    compare_attention(prob, out, lse)


def test_sharp_attention_outputs_order_one():
    """Q scaled x6 so softmax rows concentrate and outputs are O(1); the bar is
    the bound derived from bf16 rounding of P and of the output."""
    prob = attention_problem([300, 77], [64, 96], [BIDIRECTIONAL, BLOCK_CAUSAL], 16, 4, 128, 32, 32, seed=5,
                             device=DEV, q_scale=6.0)
    out, lse = run_attention(prob)
    err, rel = compare_attention(prob, out, lse, derived_bound=True)
    assert out.float().abs().max().item() > 1.0


def test_scores_rising_across_key_tiles_rescale_every_tile():
    """Every query is aligned with one direction and the prefix keys grow along
    it, so each key tile's scores exceed the previous tile's by about 20 (log2
    units): the exponentials taken against the running maximum overflow their
    2^7 check on every tile, the kernel falls back to the max-first order and
    rescales O each time. The result must still match the oracle."""
    P, W, D = 1000, 64, 128
    prob = attention_problem([P], [W], [BIDIRECTIONAL], 8, 2, D, 32, 64, seed=17)
    g = torch.Generator().manual_seed(17)
    u = torch.randn(D, generator=g)
    u /= u.norm()
    q = (8.0 * u).expand_as(prob.q).to(torch.bfloat16)
    kc = prob.k_cache.clone()
    for j in range(P):
        page = int(prob.block_table[0, j // prob.page_size])
        kc[page, :, j % prob.page_size] = (20.0 * j / 128.0 * u).to(torch.bfloat16)
    steep = AttnProblem(**{**prob.__dict__, "q": q, "k_cache": kc})
    out, lse = run_attention(steep.to(DEV))
    compare_attention(steep, out, lse)
    # the softmax is concentrated on the last prefix keys: lse grows with the last score
    assert lse.float().min().item() > 100.0


def test_probability_probe_on_gpu_output():
    """V = one-hot key positions: the GPU output row is the probability row;
    masked keys must get exactly 0 and rows must sum to 1."""
    B, P, W, D = 16, 40, 48, 128
    prob = attention_problem([P], [W], [BLOCK_CAUSAL], 4, 1, D, B, 8, seed=3, device=DEV)
    eye = torch.eye(D, dtype=torch.bfloat16, device=DEV)
    vc = torch.zeros_like(prob.v_cache)
    for pos in range(P):
        vc[int(prob.block_table[0, pos // 8]), 0, pos % 8] = eye[pos]
    vw = torch.zeros_like(prob.v_win)
    vw[:, 0] = eye[P:P + W]
    probe = AttnProblem(**{**prob.__dict__, "v_cache": vc, "v_win": vw})
    out, _ = run_attention(probe)
    pr = out.float().cpu()[:, :, :P + W]
    i = torch.arange(W)[:, None]
    j = torch.arange(P + W)[None, :]
    vis = (j < P) | (((j - P).clamp(min=0) // B) <= (i // B))
    for h in range(4):
        assert torch.all(pr[:, h][~vis] == 0)
        assert torch.allclose(pr[:, h].sum(dim=1), torch.ones(W), atol=1e-2)
    assert torch.all(out.float().cpu()[:, :, P + W:] == 0)


def test_page_permutation_is_bit_exact():
    prob = attention_problem([500, 260], [64, 64], [BIDIRECTIONAL, BLOCK_CAUSAL], 16, 4, 128, 32, 32, seed=9,
                             device=DEV, shuffle_pages=False)
    out, lse = run_attention(prob)
    perm = torch.randperm(prob.num_pages, generator=torch.Generator().manual_seed(4)).to(DEV)
    kc = torch.empty_like(prob.k_cache)
    vc = torch.empty_like(prob.v_cache)
    kc[perm] = prob.k_cache
    vc[perm] = prob.v_cache
    bt = prob.block_table.clone()
    valid = bt >= 0
    bt[valid] = perm[bt[valid].long()].to(torch.int32)
    out2, lse2 = run_attention(AttnProblem(**{**prob.__dict__, "k_cache": kc, "v_cache": vc, "block_table": bt}))
    assert torch.equal(out, out2) and torch.equal(lse, lse2)


def test_stale_cache_rows_past_prefix_do_not_leak():
    """Positions of the last prefix page beyond P hold NaN: the output must not see them."""
    prob = attention_problem([45, 300], [32, 64], [BIDIRECTIONAL, BIDIRECTIONAL], 8, 2, 128, 32, 32, seed=12,
                             device=DEV)
    ref, ref_lse = run_attention(prob)
    kc, vc = prob.k_cache.clone(), prob.v_cache.clone()
    for s, P in enumerate(prob.prefix_host):
        last = (P - 1) // 32
        page = int(prob.block_table[s, last])
        kc[page, :, P % 32:] = float("nan")
        vc[page, :, P % 32:] = float("nan")
    out, lse = run_attention(AttnProblem(**{**prob.__dict__, "k_cache": kc, "v_cache": vc}))
    assert torch.isfinite(out.float()).all()
    assert torch.equal(out, ref) and torch.equal(lse, ref_lse)


@pytest.mark.parametrize("mode", [BIDIRECTIONAL, BLOCK_CAUSAL])
def test_rows_past_the_last_window_do_not_leak(mode):
    """q / k_win / v_win rows after cu_window[batch] hold NaN: the last key tile
    reads them, and neither out nor lse may see them."""
    prob = attention_problem([45, 300], [32, 72], [mode, mode], 8, 2, 128, 32, 32, seed=14, device=DEV)
    ref, ref_lse = run_attention(prob)
    T = int(prob.cu_window[-1])

    def pad(x):
        return torch.cat([x, torch.full((200,) + tuple(x.shape[1:]), float("nan"), dtype=x.dtype, device=DEV)])
    out, lse = run_attention(AttnProblem(**{**prob.__dict__, "q": pad(prob.q), "k_win": pad(prob.k_win),
                                            "v_win": pad(prob.v_win)}))
    assert torch.isfinite(out[:T].float()).all()
    assert torch.equal(out[:T], ref) and torch.equal(lse[:T], ref_lse)


def test_empty_windows_and_zero_prefix():
    prob = attention_problem([100, 0, 64, 0], [0, 32, 0, 64], [BIDIRECTIONAL, BLOCK_CAUSAL, BIDIRECTIONAL,
                                                               BIDIRECTIONAL], 8, 2, 128, 32, 32, seed=2, device=DEV)
    out, lse = run_attention(prob)
    compare_attention(prob, out, lse)


def test_gqa_equals_replicated_kv_heads():
    prob = attention_problem([333], [64], [BLOCK_CAUSAL], 16, 4, 128, 32, 32, seed=6, device=DEV)
    out, _ = run_attention(prob)
    rep = lambda t: t.repeat_interleave(4, dim=1).contiguous()
    prob_r = AttnProblem(**{**prob.__dict__, "k_win": rep(prob.k_win), "v_win": rep(prob.v_win),
                            "k_cache": rep(prob.k_cache), "v_cache": rep(prob.v_cache)})
    out_r, _ = run_attention(prob_r)
    assert (out.float() - out_r.float()).abs().max().item() <= 1e-2


def _planned_run(prob, q_scale_note=None):
    """Plan into an explicit workspace, report the plan's split groups, then run."""
    args = (prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, prob.block_table, prob.prefix_len,
            prob.window_len, prob.cu_window, prob.mask_mode)
    kw = dict(block_size=prob.block_size, max_window=prob.max_window, max_prefix=prob.max_prefix)
    need = mbe.window_attention_workspace_size(prob.batch, prob.num_q_heads, prob.num_kv_heads, prob.head_dim,
                                               prob.max_window, prob.max_prefix)
    ws = torch.empty(need, dtype=torch.uint8, device=DEV)
    mbe.window_attention_plan(prob.prefix_len, prob.window_len, prob.cu_window, prob.mask_mode,
                              total_q_tokens=prob.total_tokens, num_q_heads=prob.num_q_heads,
                              num_kv_heads=prob.num_kv_heads, head_dim=prob.head_dim, workspace=ws, **kw)
    n_units, n_groups = mbe.window_attention_plan_stats(ws)
    out, lse = mbe.window_attention_run(*args, return_lse=True, workspace=ws, **kw)
    assert mbe.get_device_error() == (0, 0)
    return out, lse, n_units, n_groups


def test_split_kv_matches_oracle_and_unsplit():
    """Few long sequences force split-KV pieces and the LSE merge; each compared
    (sequence, head) pair is held to the bar relative to its output RMS."""
    prob = attention_problem([20000, 9000], [64, 64], [BIDIRECTIONAL, BLOCK_CAUSAL], 32, 8, 128, 32, 64, seed=13,
                             device=DEV)
    out, lse, n_units, n_groups = _planned_run(prob)
    assert n_groups > 0 and n_units > 2 * 8
    ref, ref_lse = run_attention(prob)
    assert torch.equal(out, ref) and torch.equal(lse, ref_lse)
    compare_attention(prob, out, lse, heads=[0, 5, 17, 31])


def test_split_kv_sharpened_outputs_order_one():
    """Queries sharpened x6 over prefixes of 20k-24k keys: the plan cuts the keys
    into split-KV pieces merged by log-sum-exp, and the outputs are O(1), so the
    worst-case bar u sum_j p_j |v_j| + u |o| (sum_j p_j |v_j| from the oracle on
    |V|) pins the weight of every piece in the merge."""
    prob = attention_problem([24000, 20000], [64, 64], [BIDIRECTIONAL, BLOCK_CAUSAL], 32, 8, 128, 32, 64, seed=19,
                             device=DEV, q_scale=6.0)
    out, lse, n_units, n_groups = _planned_run(prob)
    assert n_groups > 0
    compare_attention(prob, out, lse, heads=[0, 9, 22, 31], derived_bound=True)
    assert out.float().abs().max().item() > 1.0


def test_bad_page_id_sets_flag_without_fault():
    prob = attention_problem([200], [32], [BIDIRECTIONAL], 4, 1, 128, 32, 32, seed=1, device=DEV)
    bt = prob.block_table.clone()
    bt[0, 2] = prob.num_pages + 50
    mbe.window_attention(prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, bt, prob.prefix_len,
                         prob.window_len, prob.cu_window, prob.mask_mode, block_size=32, max_window=32,
                         max_prefix=200)
    st, flags = mbe.get_device_error()
    assert st == 6
    assert flags & mbe.DEVERR_PAGE
    assert mbe.get_device_error() == (0, 0)


def test_length_above_declared_max_sets_flag():
    prob = attention_problem([64], [64], [BIDIRECTIONAL], 4, 1, 128, 32, 32, seed=1, device=DEV)
    mbe.window_attention(prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, prob.block_table,
                         prob.prefix_len, prob.window_len, prob.cu_window, prob.mask_mode, block_size=32,
                         max_window=32, max_prefix=64)
    st, flags = mbe.get_device_error()
    assert st == 6 and flags & mbe.DEVERR_LENGTH


def test_varlen64_workload_sampled():
    w = wl.varlen64(DEV, vocab=1024)
    prob = w["attn"][0]
    out, lse = run_attention(prob)
    seqs = _sample(prob.batch, 12, 0)
    compare_attention(prob, out, lse, seqs=seqs)


def test_long32k_workload_sampled():
    w = wl.long32k(DEV)
    for prob in w["attn"]:
        out, lse = run_attention(prob)
        compare_attention(prob, out, lse, seqs=[0, 3], heads=[0, 9, 30])


def test_stream_k_pieces_of_one_query_tile_slabs():
    """Slabs of one length with a single query tile each (W G = 128 rows): the
    plan cuts their concatenated key tiles at multiples of total / SMs, so split
    pieces of units that run both TMEM chains on one query tile are merged by
    log-sum-exp. Checked against the oracle on sampled sequences; the plan must
    hold split groups."""
    prob = wl.attention_problem([16384] * 8, [32] * 8, [wl.BIDIRECTIONAL] * 8, 32, 8, 128, 32, 32, seed=61,
                                device=DEV)
    out, lse = run_attention(prob)
    need = mbe.window_attention_workspace_size(prob.batch, 32, 8, 128, prob.max_window, prob.max_prefix)
    ws = torch.empty(need, dtype=torch.uint8, device=DEV)
    mbe.window_attention_plan(prob.prefix_len, prob.window_len, prob.cu_window, prob.mask_mode,
                              total_q_tokens=prob.total_tokens, num_q_heads=32, num_kv_heads=8, head_dim=128,
                              block_size=32, max_window=prob.max_window, max_prefix=prob.max_prefix, workspace=ws)
    n_units, n_groups = mbe.window_attention_plan_stats(ws)
    assert n_groups > 0 and n_units > prob.batch * 8
    compare_attention(prob, out, lse, seqs=[0, 5], heads=[0, 13, 31])


def test_serving128_full_size_sampled():
    """Full per-layer shapes of the serving mix (2 of its 24 layers)."""
    w = wl.serving128(DEV, layers=2, vocab=8)
    for li, prob in enumerate(w["attn"]):
        out, lse = run_attention(prob)
        seqs = _sample(prob.batch, 6, li)
        # include the longest and the shortest prefix
        seqs = sorted(set(seqs) | {int(np.argmax(prob.prefix_host)), int(np.argmin(prob.prefix_host))})
        compare_attention(prob, out, lse, seqs=seqs, heads=[0, 7, 13, 31])


def test_plan_once_run_many_layers_equals_per_call():
    """One plan serves several layers (different Q/K/V and caches, same
    lengths); every run matches a full call bit for bit, and repeated runs on
    the same plan give identical results."""
    w = wl.serving128(DEV, layers=3, batch=16, vocab=8)
    a0 = w["attn"][0]
    kw = dict(block_size=a0.block_size, max_window=a0.max_window, max_prefix=a0.max_prefix)
    need = mbe.window_attention_workspace_size(a0.batch, a0.num_q_heads, a0.num_kv_heads, a0.head_dim,
                                               a0.max_window, a0.max_prefix)
    ws = torch.empty(need, dtype=torch.uint8, device=DEV)
    mbe.window_attention_plan(a0.prefix_len, a0.window_len, a0.cu_window, a0.mask_mode, total_q_tokens=a0.total_tokens,
                              num_q_heads=a0.num_q_heads, num_kv_heads=a0.num_kv_heads, head_dim=a0.head_dim,
                              workspace=ws, **kw)
    for rep in range(2):
        for a in w["attn"]:
            args = (a.q, a.k_win, a.v_win, a.k_cache, a.v_cache, a.block_table, a.prefix_len, a.window_len,
                    a.cu_window, a.mask_mode)
            ref, ref_lse = mbe.window_attention(*args, return_lse=True, **kw)
            out, lse = mbe.window_attention_run(*args, return_lse=True, workspace=ws, **kw)
            assert torch.equal(out, ref) and torch.equal(lse, ref_lse)
    assert mbe.get_device_error() == (0, 0)


def test_run_without_matching_plan_sets_flag_and_writes_nothing():
    """A run whose bounds differ from the plan's (a different workspace layout),
    or a run on a workspace that holds no plan, must compute nothing and set
    MBE_DEVERR_PLAN instead of reading the workspace as a work list."""
    prob = attention_problem([300, 200], [64, 64], [BIDIRECTIONAL, BIDIRECTIONAL], 8, 2, 128, 32, 32, seed=3,
                             device=DEV)
    args = (prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, prob.block_table, prob.prefix_len,
            prob.window_len, prob.cu_window, prob.mask_mode)
    need = mbe.window_attention_workspace_size(2, 8, 2, 128, 128, 300)
    ws = torch.zeros(need, dtype=torch.uint8, device=DEV)
    mbe.window_attention_plan(prob.prefix_len, prob.window_len, prob.cu_window, prob.mask_mode,
                              total_q_tokens=prob.total_tokens, num_q_heads=8, num_kv_heads=2, head_dim=128,
                              block_size=32, max_window=64, max_prefix=300, workspace=ws)
    out = torch.full_like(prob.q, 7.0)
    mbe.window_attention_run(*args, block_size=32, max_window=128, max_prefix=300, out=out, workspace=ws)
    st, flags = mbe.get_device_error()
    assert st == 6 and flags & mbe.DEVERR_PLAN
    assert torch.all(out == 7.0)
    fresh = torch.zeros(need, dtype=torch.uint8, device=DEV)
    mbe.window_attention_run(*args, block_size=32, max_window=64, max_prefix=300, out=out, workspace=fresh)
    st, flags = mbe.get_device_error()
    assert st == 6 and flags & mbe.DEVERR_PLAN
    assert torch.all(out == 7.0)
    # the matching run on the planned workspace works
    ref = mbe.window_attention(*args, block_size=32, max_window=64, max_prefix=300)
    mbe.window_attention_run(*args, block_size=32, max_window=64, max_prefix=300, out=out, workspace=ws)
    assert torch.equal(out, ref)
    assert mbe.get_device_error() == (0, 0)
