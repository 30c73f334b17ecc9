"""Parity of the Multi-Block Edit SFT attention (Sec. 3): the cross-block mask
builder (bit-exact) and attention under a block mask (max abs error <= 1e-2
on the bf16 output and 2e-3 relative on the LSE, as the window attention),
through the C ABI against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300.workloads import bf16_bits, sft_problem
from tests._gpu import ATTN_ATOL

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _gpu_mask(prob, K):
    return mbe.sft_block_mask(prob.n_prompt_blocks.to(DEV), prob.n_blocks.to(DEV), K, prob.mask_rows)


@pytest.mark.parametrize("K", [1, 2, 3, 5])
def test_mask_builder_matches_oracle(K):
    Np, N = [0, 1, 3, 2], [1, 4, 9, 40]
    prob = sft_problem(Np, N, 2, 1, 64, 32, seed=K)
    m = _gpu_mask(prob, K).cpu().numpy().view(np.uint32)
    for s in range(len(N)):
        ref = oracle.sft_block_mask(Np[s], N[s], K, words_per_row=m.shape[2])
        nb = Np[s] + 2 * N[s]
        np.testing.assert_array_equal(m[s, :nb], ref)
        assert not m[s, nb:].any()
    assert mbe.get_device_error() == (0, 0)


def _run(prob, mask, **kw):
    d = {k: getattr(prob, k).to(DEV) for k in ("q", "k", "v", "seq_len", "cu_seqlens")}
    out, lse = mbe.block_mask_attention(d["q"], d["k"], d["v"], d["seq_len"], d["cu_seqlens"], mask,
                                        block_size=prob.block_size, max_seq_len=prob.max_seq_len, return_lse=True,
                                        **kw)
    torch.cuda.synchronize()
    assert mbe.get_device_error() == (0, 0)
    return out.float().cpu().numpy(), lse.cpu().numpy()


def _check(prob, mask_np, out, lse):
    cu = prob.cu_seqlens.tolist()
    worst = 0.0
    for s in range(len(prob.seq_host)):
        a, b = cu[s], cu[s + 1]
        ref, lref = oracle.block_mask_attention(bf16_bits(prob.q[a:b]), bf16_bits(prob.k[a:b]), bf16_bits(prob.v[a:b]),
                                                prob.block_size, mask_np[s])
        err = np.abs(out[a:b] - ref).max()
        worst = max(worst, err)
        fin = np.isfinite(lref)
        np.testing.assert_allclose(lse[a:b][fin], lref[fin], rtol=2e-3, atol=2e-3)
        assert np.isneginf(lse[a:b][~fin]).all() and not out[a:b][~fin].any()
    assert worst <= ATTN_ATOL, worst
    return worst


@pytest.mark.parametrize("D,G,B,K", [(128, 4, 32, 3), (64, 2, 32, 2), (128, 1, 16, 4), (128, 8, 64, 1)])
def test_forward_matches_oracle(D, G, B, K):
    Np, N = [1, 0, 2], [6, 3, 8]
    prob = sft_problem(Np, N, 2 * G, 2, D, B, seed=D + G + B, trim=[0, 5, B - 1])
    mask = _gpu_mask(prob, K)
    out, lse = _run(prob, mask)
    _check(prob, mask.cpu().numpy().view(np.uint32), out, lse)


def test_forward_with_a_hand_mask_and_an_empty_row():
    # block 1 sees nothing: its rows must come out as zeros with lse = -inf;
    # block 2 sees only block 0 (a tile two tiles away from it)
    B = 32
    prob = sft_problem([0], [4], 4, 1, 128, B, seed=9)  # 8 blocks, 256 tokens
    nb = 8
    bits = np.zeros((1, nb, 1), np.uint32)
    for qb in range(nb):
        bits[0, qb, 0] = (1 << (qb + 1)) - 1       # block-causal ...
    bits[0, 1, 0] = 0                                # ... but block 1 sees nothing
    bits[0, 2, 0] = 1                                # and block 2 only block 0
    mask = torch.from_numpy(bits.view(np.int32)).to(DEV)
    out, lse = _run(prob, mask)
    _check(prob, bits, out, lse)
    assert np.isneginf(lse[32:64]).all()


def test_longer_sequences_with_split_pieces():
    # few long sequences: the scheduler splits the key range; the merge combines pieces
    prob = sft_problem([2, 1], [40, 25], 8, 2, 128, 32, seed=11)  # 2624 and 1632 tokens
    mask = _gpu_mask(prob, 3)
    out, lse = _run(prob, mask)
    _check(prob, mask.cpu().numpy().view(np.uint32), out, lse)


def test_argument_errors():
    prob = sft_problem([1], [2], 4, 1, 128, 32, seed=1)
    mask = _gpu_mask(prob, 2)
    d = {k: getattr(prob, k).to(DEV) for k in ("q", "k", "v", "seq_len", "cu_seqlens")}
    with pytest.raises(mbe.MbeError):      # block size not a power of two
        mbe.block_mask_attention(d["q"], d["k"], d["v"], d["seq_len"], d["cu_seqlens"], mask, block_size=24,
                                 max_seq_len=prob.max_seq_len)
    with pytest.raises(mbe.MbeError):      # mask rows fewer than the sequence's blocks
        mbe.block_mask_attention(d["q"], d["k"], d["v"], d["seq_len"], d["cu_seqlens"], mask[:, :2].contiguous(),
                                 block_size=32, max_seq_len=prob.max_seq_len)
