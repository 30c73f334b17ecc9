"""Parity of the Multi-Block Edit SFT attention (Sec. 3): the cross-block mask
builder (bit-exact), attention under a block mask (max abs error <= 1e-2 on
the bf16 output and 2e-3 relative on the LSE, as the window attention) and its
gradients, through the C ABI against the oracle.

Gradient bar, per element (twice the bound, plus 1e-5 of the largest
reference value for fp32 accumulation and exp2): P and dS are rounded to bf16
(unit roundoff u = 2^-8) before their tensor-core products, so dV is off by at
most u |P|^T |dO|, dK by scale u |dS|^T |Q| and dQ by scale u |dS| |K|; delta
is formed from the bf16 forward output, |O_bf16 - O| <= u |O|, which moves dS
by at most P u sum_d |dO||O| and adds scale (P u sum_d |dO||O|)^T |Q| to dK and
the same against |K| to dQ. Every gradient also stays within 1e-2 relative in
the Frobenius norm."""
import dataclasses

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


def test_forward_rows_after_the_last_sequence_do_not_leak():
    """q / k / v rows after cu_seqlens[batch] hold NaN: the last key tile of the
    last sequence reads them, and the output must not see them."""
    prob = sft_problem([1, 0], [3, 4], 8, 2, 128, 32, seed=13, trim=[0, 9])
    mask = _gpu_mask(prob, 2)
    ref, ref_lse = _run(prob, mask)
    T = int(prob.cu_seqlens[-1])
    pad = lambda x: torch.cat([x, torch.full((100,) + tuple(x.shape[1:]), float("nan"), dtype=x.dtype)])
    padded = dataclasses.replace(prob, q=pad(prob.q), k=pad(prob.k), v=pad(prob.v))
    out, lse = _run(padded, mask)
    assert np.isfinite(out[:T]).all()
    np.testing.assert_array_equal(out[:T], ref)
    np.testing.assert_array_equal(lse[:T], ref_lse)
    _check(prob, mask.cpu().numpy().view(np.uint32), out[:T], lse[:T])


def test_forward_rising_scores_under_a_partial_mask():
    """Keys grow along the queries' direction, so every key tile's scores exceed
    the running maximum by about 2^20 and the kernel falls back from the
    speculated exponentials to the max-first order; the mask hides every odd key
    block, so those tiles are partially visible and the fallback (which reads S
    again) must keep the hidden columns, which hold the larger scores, out."""
    B = 32
    prob = sft_problem([0], [16], 4, 1, 128, B, seed=23)  # 32 blocks, 1024 tokens
    T = prob.seq_host[0]
    nb = T // B
    g = torch.Generator().manual_seed(23)
    u = torch.randn(128, generator=g)
    u /= u.norm()
    q = (8.0 * u).expand_as(prob.q).to(torch.bfloat16).contiguous()
    k = torch.stack([20.0 * j / 128.0 * u for j in range(T)])[:, None, :].expand_as(prob.k)
    steep = dataclasses.replace(prob, q=q, k=k.to(torch.bfloat16).contiguous())
    bits = np.zeros((1, nb, 1), np.uint32)
    bits[0, :, 0] = sum(1 << kb for kb in range(0, nb, 2))  # even key blocks only
    mask = torch.from_numpy(bits.view(np.int32)).to(DEV)
    out, lse = _run(steep, mask)
    _check(steep, bits, out, lse)


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


def _torch_probs(q, k, v, do, tmask, scale):
    """float64 P and dS of one sequence (GQA by repeating KV heads): [Hq, T, T]."""
    G = q.shape[1] // k.shape[1]
    qd = q.double().permute(1, 0, 2)
    kd = k.double().repeat_interleave(G, dim=1).permute(1, 0, 2)
    vd = v.double().repeat_interleave(G, dim=1).permute(1, 0, 2)
    dod = do.double().permute(1, 0, 2)
    s = (qd @ kd.transpose(1, 2)) * scale
    s = s.masked_fill(~torch.from_numpy(tmask)[None], float("-inf"))
    P = torch.nan_to_num(torch.softmax(s, dim=-1), nan=0.0)
    dP = dod @ vd.transpose(1, 2)
    delta = (P * dP).sum(-1, keepdim=True)
    return P, P * (dP - delta)


def _bwd_bounds(q, k, out_gpu, do, P, dS, scale):
    """Per-element bars (module docstring): bf16 rounding of P and dS before their
    products, the bf16 forward output in delta, fp32 accumulation."""
    u = 2.0 ** -8
    G = q.shape[1] // k.shape[1]
    Hkv = k.shape[1]
    qd, kd = q.double().abs().permute(1, 0, 2), k.double().abs().repeat_interleave(G, dim=1).permute(1, 0, 2)
    dod, od = do.double().abs().permute(1, 0, 2), torch.from_numpy(out_gpu).double().abs().permute(1, 0, 2)
    e = u * (dod * od).sum(-1, keepdim=True)                      # delta error per query row
    Pe = P * e                                                     # dS error from delta
    b_dv = u * (P.transpose(1, 2) @ dod)                           # [Hq, T, D]
    b_dk = scale * ((u * dS.abs() + Pe).transpose(1, 2) @ qd)
    b_dq = scale * ((u * dS.abs() + Pe) @ kd)
    fold = lambda b: b.reshape(Hkv, G, *b.shape[1:]).sum(1).permute(1, 0, 2).numpy()
    return b_dq.permute(1, 0, 2).numpy(), fold(b_dk), fold(b_dv)


def _check_bwd(prob, mask_bits, out_gpu, grads):
    cu = prob.cu_seqlens.tolist()
    D = prob.q.shape[2]
    scale = D ** -0.5
    nb = mask_bits.shape[1]
    for s in range(len(prob.seq_host)):
        a, b = cu[s], cu[s + 1]
        if a == b:
            continue
        q, k, v, do = prob.q[a:b], prob.k[a:b], prob.v[a:b], prob.dout[a:b]
        ref = oracle.block_mask_attention_bwd(bf16_bits(q), bf16_bits(k), bf16_bits(v), bf16_bits(do),
                                              prob.block_size, mask_bits[s])
        t = np.arange(b - a) // prob.block_size
        blk = oracle.mask_bits_to_dense(mask_bits[s], nb)
        P, dS = _torch_probs(q, k, v, do, blk[t[:, None], t[None, :]], scale)
        bounds = _bwd_bounds(q, k, out_gpu[a:b], do, P, dS, scale)
        for name, g, r, bd in zip(("dq", "dk", "dv"), (x[a:b] for x in grads), ref, bounds):
            err = np.abs(g - r)
            tol = 2 * bd + 1e-5 * max(np.abs(r).max(), 1e-30)
            assert (err <= tol).all(), (name, s, float(err.max()), float((err / tol).max()))
            rel = np.linalg.norm(g - r) / max(np.linalg.norm(r), 1e-30)
            assert rel < 1e-2, (name, s, rel)


def _fwd_bwd(prob, mask):
    d = {k: getattr(prob, k).to(DEV) for k in ("q", "k", "v", "dout", "seq_len", "cu_seqlens")}
    out, lse = mbe.block_mask_attention(d["q"], d["k"], d["v"], d["seq_len"], d["cu_seqlens"], mask,
                                        block_size=prob.block_size, max_seq_len=prob.max_seq_len, return_lse=True)
    grads = mbe.block_mask_attention_bwd(d["q"], d["k"], d["v"], out, d["dout"], lse, d["seq_len"],
                                         d["cu_seqlens"], mask, block_size=prob.block_size,
                                         max_seq_len=prob.max_seq_len)
    torch.cuda.synchronize()
    assert mbe.get_device_error() == (0, 0)
    return out.float().cpu().numpy(), [g.cpu().numpy() for g in grads]


@pytest.mark.parametrize("G,B,K,Np,N,trim", [(4, 32, 3, [1, 0], [6, 3], [0, 7]), (1, 16, 2, [2], [5], [3]),
                                             (8, 64, 1, [1], [3], [0]), (2, 32, 4, [1, 3], [9, 4], [31, 0]),
                                             (4, 8, 2, [1], [9], [5]), (16, 32, 2, [1], [3], [9]),
                                             (32, 16, 3, [1, 2], [2, 3], [0, 4])])
def test_backward_matches_oracle(G, B, K, Np, N, trim):
    prob = sft_problem(Np, N, 2 * G, 2, 128, B, seed=100 + G + B + K, trim=trim)
    mask = _gpu_mask(prob, K)
    out, grads = _fwd_bwd(prob, mask)
    _check_bwd(prob, mask.cpu().numpy().view(np.uint32), out, grads)


def test_backward_with_unseen_keys_and_blind_rows():
    # block 1 sees nothing (dQ = 0 there); key block 3 is seen by nobody (dK = dV = 0 there)
    B = 32
    prob = sft_problem([0], [4], 4, 1, 128, B, seed=12)
    nb = 8
    bits = np.zeros((1, nb, 1), np.uint32)
    for qb in range(nb):
        bits[0, qb, 0] = ((1 << (qb + 1)) - 1) & ~(1 << 3)
    bits[0, 1, 0] = 0
    mask = torch.from_numpy(bits.view(np.int32)).to(DEV)
    out, grads = _fwd_bwd(prob, mask)
    _check_bwd(prob, bits, out, grads)
    assert not grads[0][32:64].any()
    assert not grads[1][96:128].any() and not grads[2][96:128].any()


def test_backward_long_sequence():
    # many query tiles per key tile and several key tiles per sequence
    prob = sft_problem([2], [30], 8, 2, 128, 32, seed=13)  # 1984 tokens
    mask = _gpu_mask(prob, 3)
    out, grads = _fwd_bwd(prob, mask)
    _check_bwd(prob, mask.cpu().numpy().view(np.uint32), out, grads)


def test_backward_argument_errors():
    # 64 query heads per KV head: a warp's 32 query rows would not be whole tokens
    prob = sft_problem([1], [2], 64, 1, 128, 32, seed=5)
    mask = _gpu_mask(prob, 2)
    d = {k: getattr(prob, k).to(DEV) for k in ("q", "k", "v", "dout", "seq_len", "cu_seqlens")}
    lse = torch.zeros(d["q"].shape[:2], dtype=torch.float32, device=DEV)
    with pytest.raises(mbe.MbeError):
        mbe.block_mask_attention_bwd(d["q"], d["k"], d["v"], d["q"], d["dout"], lse, d["seq_len"], d["cu_seqlens"],
                                     mask, block_size=32, max_seq_len=prob.max_seq_len)


def test_backward_with_an_empty_sequence_in_the_batch():
    # the middle sequence has no tokens: no work units, nothing written for it
    prob = sft_problem([1, 0, 2], [3, 0, 4], 8, 2, 128, 32, seed=21, trim=[5, 0, 0])
    mask = _gpu_mask(prob, 2)
    out, grads = _fwd_bwd(prob, mask)
    _check_bwd(prob, mask.cpu().numpy().view(np.uint32), out, grads)
