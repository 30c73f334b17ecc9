"""Failure detection of the bounded device waits, without a GPU fault.

Every mbarrier wait in the tcgen05 kernels (window attention, fused LM head,
attention backward) is bounded. mbe_set_wait_limit_ns(0) turns each wait
that is not already complete into an expired one, so the kernels take their
abort path: they record MBE_DEVERR_TIMEOUT, let the copies and MMAs they
issued finish, release their tensor memory and return. The tests check the
status the host reads, then restore the limit and check that the next call in
the same process computes the right result (no held tensor memory, no stuck
barrier or work counter)."""
import numpy as np
import pytest
import torch

from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, BLOCK_CAUSAL, attention_problem, sft_problem
from tests._gpu import compare_attention, run_attention

pytestmark = pytest.mark.gpu
DEV = "cuda"


class _ZeroWaitLimit:
    def __enter__(self):
        self.prev = mbe.set_wait_limit_ns(0)
        return self

    def __exit__(self, *exc):
        mbe.set_wait_limit_ns(self.prev)
        return False


def _expect_timeout():
    st, flags = mbe.get_device_error()
    assert st == 4, (st, flags)   # MBE_ERR_TIMEOUT
    assert flags & mbe.DEVERR_TIMEOUT


def test_default_limit_is_one_second():
    prev = mbe.set_wait_limit_ns(mbe.DEFAULT_WAIT_LIMIT_NS)
    assert prev == mbe.DEFAULT_WAIT_LIMIT_NS
    assert mbe.set_wait_limit_ns(prev) == mbe.DEFAULT_WAIT_LIMIT_NS


def test_attention_wait_expiry_reports_timeout_and_recovers():
    prob = attention_problem([3000, 1200, 64, 20000], [64, 128, 32, 64],
                             [BIDIRECTIONAL, BLOCK_CAUSAL, BIDIRECTIONAL, BIDIRECTIONAL], 16, 4, 128, 32, 64, seed=41,
                             device=DEV)
    args = (prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, prob.block_table, prob.prefix_len,
            prob.window_len, prob.cu_window, prob.mask_mode)
    kw = dict(block_size=prob.block_size, max_window=prob.max_window, max_prefix=prob.max_prefix)
    with _ZeroWaitLimit():
        for _ in range(3):
            mbe.window_attention(*args, **kw)
            _expect_timeout()
    out, lse = run_attention(prob)
    compare_attention(prob, out, lse, heads=[0, 5, 10, 15])
    assert mbe.get_device_error() == (0, 0)


def test_lm_head_wait_expiry_reports_timeout_and_recovers():
    g = torch.Generator(device=DEV).manual_seed(3)
    R, V, d = 512, 8192, 512
    h = torch.randn(R, d, generator=g, device=DEV).to(torch.bfloat16)
    w = (torch.randn(V, d, generator=g, device=DEV) * d ** -0.5).to(torch.bfloat16)
    committed = torch.randint(0, V, (R,), generator=g, device=DEV, dtype=torch.int32)
    ref = mbe.lm_head_edit_decide(h, w, committed, tau=0.0, want_entropy=True)
    assert mbe.get_device_error() == (0, 0)
    with _ZeroWaitLimit():
        for _ in range(2):
            mbe.lm_head_edit_decide(h, w, committed, tau=0.0, want_entropy=True)
            _expect_timeout()
    res = mbe.lm_head_edit_decide(h, w, committed, tau=0.0, want_entropy=True)
    assert mbe.get_device_error() == (0, 0)
    for a, b in zip(res, ref):
        assert torch.equal(a, b)


def test_attention_backward_wait_expiry_reports_timeout_and_recovers():
    prob = sft_problem([1, 0], [6, 3], 8, 2, 128, 32, seed=7, trim=[0, 7])
    mask = mbe.sft_block_mask(prob.n_prompt_blocks.to(DEV), prob.n_blocks.to(DEV), 2, prob.mask_rows)
    d = {k: getattr(prob, k).to(DEV) for k in ("q", "k", "v", "dout", "seq_len", "cu_seqlens")}
    kw = dict(block_size=prob.block_size, max_seq_len=prob.max_seq_len)
    out, lse = mbe.block_mask_attention(d["q"], d["k"], d["v"], d["seq_len"], d["cu_seqlens"], mask, return_lse=True,
                                        **kw)

    def bwd():
        return mbe.block_mask_attention_bwd(d["q"], d["k"], d["v"], out, d["dout"], lse, d["seq_len"],
                                            d["cu_seqlens"], mask, **kw)
    ref = bwd()
    assert mbe.get_device_error() == (0, 0)
    with _ZeroWaitLimit():
        for _ in range(2):
            bwd()
            _expect_timeout()
        # the forward under a block mask runs the same attention kernel
        mbe.block_mask_attention(d["q"], d["k"], d["v"], d["seq_len"], d["cu_seqlens"], mask, **kw)
        _expect_timeout()
    again = bwd()
    assert mbe.get_device_error() == (0, 0)
    for a, b in zip(again, ref):
        assert torch.equal(a, b)
    out2, lse2 = mbe.block_mask_attention(d["q"], d["k"], d["v"], d["seq_len"], d["cu_seqlens"], mask,
                                          return_lse=True, **kw)
    assert torch.equal(out2, out) and torch.equal(lse2, lse)
    assert mbe.get_device_error() == (0, 0)
