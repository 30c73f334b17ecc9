"""mbe_window_attention_noalloc, the attention entry point for callers that
cannot allocate device memory (a framework that owns all device memory in its
own pool, or a latency-critical path that must not risk the synchronisation of
cudaMalloc/cudaFree). It keeps its scratch in a static 64 MiB device array of
the library instead of a caller workspace; its results must match the regular
entry point's, call after call, since each call reuses and overwrites the same
array. This file is collected last on purpose."""
import ctypes

import pytest
import torch

from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, BLOCK_CAUSAL, attention_problem
from tests._gpu import ATTN_ATOL

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _problem():
    # a 4000-token prefix makes the scheduler split work, so partial results
    # and the merge go through the static array too
    return attention_problem([4000, 700, 3000, 64], [64, 96, 32, 64],
                             [BIDIRECTIONAL, BLOCK_CAUSAL, BIDIRECTIONAL, BLOCK_CAUSAL], 16, 4, 128, 32, 32,
                             seed=77, device=DEV)


def test_noalloc_matches_regular_entry_point_on_two_calls():
    prob = _problem()
    kw = dict(block_size=prob.block_size, max_window=prob.max_window, max_prefix=prob.max_prefix)
    args = (prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, prob.block_table, prob.prefix_len,
            prob.window_len, prob.cu_window, prob.mask_mode)
    ref, ref_lse = mbe.window_attention(*args, return_lse=True, **kw)
    assert mbe.window_attention_workspace_size(prob.batch, prob.num_q_heads, prob.num_kv_heads, prob.head_dim,
                                               prob.max_window, prob.max_prefix) <= 64 << 20
    for _ in range(2):
        out = torch.full_like(prob.q, float("nan"))
        lse = torch.full_like(ref_lse, float("nan"))
        mbe.window_attention_noalloc(*args, out=out, lse=lse, **kw)
        torch.cuda.synchronize()
        assert torch.isfinite(out.float()).all()
        assert (out.float() - ref.float()).abs().max().item() <= ATTN_ATOL
        assert (lse - ref_lse).abs().max().item() <= 1e-3
    st, flags = mbe.get_device_error()
    assert st == 0, (st, flags)


def test_noalloc_rejects_shapes_beyond_the_static_scratch():
    prob = _problem()
    out = torch.empty_like(prob.q)
    L = mbe.lib()
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    # bounds that would need far more than 64 MiB of scratch: rejected before any launch
    st = L.mbe_window_attention_noalloc(P(prob.q), P(prob.k_win), P(prob.v_win), P(prob.k_cache), P(prob.v_cache),
                                        prob.num_pages, P(prob.block_table), 1 << 16, P(prob.prefix_len),
                                        P(prob.window_len), P(prob.cu_window), P(prob.mask_mode), 4096,
                                        prob.total_tokens, 16, 4, 128, 32, 32, 4096, 1 << 20, 0.0, P(out), None,
                                        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 5  # MBE_ERR_WORKSPACE
    assert mbe.get_device_error() == (0, 0)
