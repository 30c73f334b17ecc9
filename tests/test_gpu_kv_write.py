"""Parity of the CUDA KV window write (mbe_kv_window_write) with the oracle:
bit-exact over the whole cache (pages outside the window keep their contents)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300 import workloads as wl
from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, BLOCK_CAUSAL, AttnProblem, attention_problem, bf16_bits
from tests._gpu import compare_attention, run_attention

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _gpu_write(prob, mask=None):
    kc, vc = prob.k_cache.clone(), prob.v_cache.clone()
    mbe.kv_window_write(prob.k_win, prob.v_win, kc, vc, prob.block_table, prob.prefix_len, prob.window_len,
                        prob.cu_window, block_size=prob.block_size, max_window=max(prob.max_window, 1),
                        block_write_mask=mask)
    st, flags = mbe.get_device_error()
    return kc, vc, st, flags


def _oracle_write(prob, mask=None):
    return oracle.kv_window_write(bf16_bits(prob.k_win), bf16_bits(prob.v_win), bf16_bits(prob.k_cache),
                                  bf16_bits(prob.v_cache), prob.block_table.cpu().numpy(),
                                  prob.prefix_len.cpu().numpy(), prob.window_len.cpu().numpy(),
                                  prob.cu_window.cpu().numpy(), prob.block_size,
                                  block_write_mask=None if mask is None else mask.cpu().numpy())


@pytest.mark.parametrize("page", [8, 32, 64, 256])
def test_matches_oracle_bit_exact(page):
    prob = attention_problem([37, 0, 1000, 64], [64, 32, 96, 1], [BIDIRECTIONAL] * 4, 16, 4, 128, 32, page,
                             seed=page, device=DEV, spare_pages=7)
    kc, vc, st, _ = _gpu_write(prob)
    assert st == 0
    kr, vr = _oracle_write(prob)
    assert np.array_equal(bf16_bits(kc), kr) and np.array_equal(bf16_bits(vc), vr)


def test_block_write_mask():
    prob = attention_problem([40, 96], [96, 64], [BIDIRECTIONAL] * 2, 8, 2, 64, 32, 16, seed=3, device=DEV)
    mask = torch.tensor([[1, 0, 1], [0, 1, 0]], dtype=torch.uint8, device=DEV)
    kc, vc, st, _ = _gpu_write(prob, mask)
    assert st == 0
    kr, vr = _oracle_write(prob, mask)
    assert np.array_equal(bf16_bits(kc), kr) and np.array_equal(bf16_bits(vc), vr)


def test_long32k_write_then_attend():
    """The long-context workload: the window of an editing pass is written at
    positions [P, P+W) (bit-exact against the oracle), then a standard pass over
    the next block (block-causal, prefix P+W) reads the written keys from the
    cache and matches the oracle on that cache."""
    w = wl.long32k(DEV, windows=(64, 128))   # the cache reserves room for 128 window tokens
    prob = w["attn"][0]
    kc, vc, st, _ = _gpu_write(prob)
    assert st == 0
    kr, vr = _oracle_write(prob)
    assert np.array_equal(bf16_bits(kc), kr) and np.array_equal(bf16_bits(vc), vr)
    g = torch.Generator(device=DEV).manual_seed(44)
    B, n = 32, prob.batch
    rnd = lambda *shape: torch.randn(*shape, generator=g, device=DEV).to(torch.bfloat16)
    nxt = AttnProblem(q=rnd(n * B, 32, 128), k_win=rnd(n * B, 8, 128), v_win=rnd(n * B, 8, 128), k_cache=kc,
                      v_cache=vc, block_table=prob.block_table, prefix_len=prob.prefix_len + prob.window_len,
                      window_len=torch.full((n,), B, dtype=torch.int32, device=DEV),
                      cu_window=torch.arange(0, n * B + 1, B, dtype=torch.int32, device=DEV),
                      mask_mode=torch.full((n,), BLOCK_CAUSAL, dtype=torch.uint8, device=DEV), block_size=B,
                      page_size=prob.page_size, prefix_host=[p + 64 for p in prob.prefix_host], window_host=[B] * n,
                      mode_host=[BLOCK_CAUSAL] * n)
    out, lse = run_attention(nxt)
    compare_attention(nxt, out, lse, seqs=[0, 3], heads=[0, 13, 31])
    # the written rows matter: the same pass over the cache before the write differs
    stale = AttnProblem(**{**nxt.__dict__, "k_cache": prob.k_cache, "v_cache": prob.v_cache})
    out_stale, _ = run_attention(stale)
    assert not torch.equal(out_stale, out)


def test_bad_page_flagged_and_skipped():
    prob = attention_problem([10], [32], [BIDIRECTIONAL], 4, 1, 128, 32, 32, seed=1, device=DEV)
    bt = prob.block_table.clone()
    bt[0, 1] = -7
    kc, vc = prob.k_cache.clone(), prob.v_cache.clone()
    mbe.kv_window_write(prob.k_win, prob.v_win, kc, vc, bt, prob.prefix_len, prob.window_len, prob.cu_window,
                        block_size=32, max_window=32)
    st, flags = mbe.get_device_error()
    assert st == 6 and flags & mbe.DEVERR_PAGE
