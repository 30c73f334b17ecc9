"""The binding's argument checks. The C ABI takes plain pointers and trusts the
lengths it is given, so each wrapper holds every array to the shape those
lengths imply and every tensor to the call's device. A malformed argument must
raise in Python before anything is launched (the device error word stays
clear)."""
import pytest
import torch

from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, BLOCK_CAUSAL, attention_problem, edit_problem, sft_problem

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _attn():
    prob = attention_problem([64, 96], [64, 32], [BIDIRECTIONAL, BLOCK_CAUSAL], 8, 2, 128, 32, 32, seed=3,
                             device=DEV)
    args = [prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, prob.block_table, prob.prefix_len,
            prob.window_len, prob.cu_window, prob.mask_mode]
    kw = dict(block_size=32, max_window=64, max_prefix=96)
    return prob, args, kw


def _nothing_launched():
    torch.cuda.synchronize()
    assert mbe.get_device_error() == (0, 0)


@pytest.mark.parametrize("index,bad", [
    (6, lambda t: t[:-1]),                     # prefix_len one short of the batch
    (7, lambda t: torch.cat([t, t[:1]])),      # window_len one too long
    (8, lambda t: t[:-1]),                     # cu_window without its last entry
    (9, lambda t: t[:1]),                      # mask_mode of one sequence
    (1, lambda t: t[:-1]),                     # k_win one row short of q
    (4, lambda t: t[:, :1]),                   # v_cache with fewer KV heads than k_cache
    (6, lambda t: t.cpu()),                    # prefix_len on the host
])
def test_window_attention_rejects_malformed_arrays(index, bad):
    _, args, kw = _attn()
    args[index] = bad(args[index]).contiguous()
    with pytest.raises((ValueError, TypeError)):
        mbe.window_attention(*args, **kw)
    _nothing_launched()


def test_window_attention_rejects_malformed_outputs():
    prob, args, kw = _attn()
    T, Hq, D = prob.q.shape
    with pytest.raises(ValueError):
        mbe.window_attention(*args, out=torch.empty((T - 1, Hq, D), dtype=torch.bfloat16, device=DEV), **kw)
    with pytest.raises(ValueError):
        mbe.window_attention(*args, lse=torch.empty((T, Hq - 1), dtype=torch.float32, device=DEV), **kw)
    with pytest.raises(TypeError):
        mbe.window_attention(*args, lse=torch.empty((T, Hq), dtype=torch.float16, device=DEV), **kw)
    with pytest.raises(ValueError):
        mbe.window_attention_noalloc(*args, out=torch.empty((T, Hq, D - 8), dtype=torch.bfloat16, device=DEV), **kw)
    with pytest.raises(ValueError):
        ws = torch.empty(16, dtype=torch.uint8, device=DEV)
        mbe.window_attention_plan(prob.prefix_len, prob.window_len, prob.cu_window[:-1].contiguous(), prob.mask_mode,
                                  total_q_tokens=T, num_q_heads=Hq, num_kv_heads=2, head_dim=D, workspace=ws, **kw)
    _nothing_launched()


def test_edit_decide_rejects_malformed_arrays():
    p = edit_problem(64, 1000, torch.float32, seed=2, device=DEV)
    R = p.logits.shape[0]
    with pytest.raises(ValueError):
        mbe.edit_decide(p.logits, p.committed[:-1].contiguous())
    with pytest.raises(ValueError):
        mbe.edit_decide(p.logits, p.committed, tau_per_row=torch.zeros(R + 1, device=DEV))
    with pytest.raises(ValueError):
        mbe.edit_decide(p.logits, p.committed, editable=torch.ones(R - 1, dtype=torch.uint8, device=DEV))
    with pytest.raises(TypeError):
        mbe.edit_decide(p.logits, p.committed, new_tokens=torch.empty(R, dtype=torch.int64, device=DEV))
    with pytest.raises(ValueError):
        mbe.edit_decide(p.logits, p.committed, confidence=torch.empty(R // 2, dtype=torch.float32, device=DEV))
    _nothing_launched()


def test_kv_window_write_rejects_malformed_arrays():
    prob, _, _ = _attn()
    base = dict(block_size=32, max_window=64)
    a = [prob.k_win, prob.v_win, prob.k_cache.clone(), prob.v_cache.clone(), prob.block_table, prob.prefix_len,
         prob.window_len, prob.cu_window]
    for index, bad in ((6, lambda t: t[:-1]), (7, lambda t: t[:-1]), (1, lambda t: t[:-1])):
        b = list(a)
        b[index] = bad(b[index]).contiguous()
        with pytest.raises(ValueError):
            mbe.kv_window_write(*b, **base)
    with pytest.raises(ValueError):
        mbe.kv_window_write(*a, block_write_mask=torch.ones((1, 2), dtype=torch.uint8, device=DEV), **base)
    _nothing_launched()


def test_block_mask_attention_rejects_malformed_arrays():
    prob = sft_problem([1], [2], 4, 1, 128, 32, seed=1, device=DEV)
    mask = mbe.sft_block_mask(prob.n_prompt_blocks, prob.n_blocks, 2, prob.mask_rows)
    torch.cuda.synchronize()
    kw = dict(block_size=32, max_seq_len=prob.max_seq_len)
    with pytest.raises(ValueError):
        mbe.block_mask_attention(prob.q, prob.k, prob.v, prob.seq_len, prob.cu_seqlens[:-1].contiguous(), mask, **kw)
    with pytest.raises(ValueError):
        mbe.block_mask_attention(prob.q, prob.k[:-1].contiguous(), prob.v, prob.seq_len, prob.cu_seqlens, mask, **kw)
    T, Hq, D = prob.q.shape
    lse = torch.zeros((T, Hq), dtype=torch.float32, device=DEV)
    with pytest.raises(ValueError):
        mbe.block_mask_attention_bwd(prob.q, prob.k, prob.v, prob.q, prob.dout, lse, prob.seq_len, prob.cu_seqlens,
                                     mask, dq=torch.empty((T, Hq, D - 1), dtype=torch.float32, device=DEV), **kw)
    _nothing_launched()
