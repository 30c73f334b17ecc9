"""Pins of the oracle's cross-block SFT mask (Sec. 3) and of attention under a
block mask, forward and gradients. CPU only."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300.workloads import bf16_bits
from tests._util import np_logsumexp


def _dense(Np, N, K):
    return oracle.mask_bits_to_dense(oracle.sft_block_mask(Np, N, K), Np + 2 * N)


def test_k1_is_the_standard_block_diffusion_sft_mask():
    # categories: prompt, noisy n_i, clean c_j; standard links NN (own block),
    # NC (strictly earlier clean blocks), CC (block-causal), prompt visible to all
    Np, N = 2, 5
    nb = Np + 2 * N
    kind = np.array(["p"] * Np + ["n"] * N + ["c"] * N)
    idx = np.array(list(range(Np)) + list(range(N)) + list(range(N)))
    q_kind, k_kind = kind[:, None], kind[None, :]
    q_i, k_i = idx[:, None], idx[None, :]
    ref = (k_kind == "p") \
        | ((q_kind == "n") & (k_kind == "n") & (q_i == k_i)) \
        | ((q_kind == "n") & (k_kind == "c") & (k_i < q_i)) \
        | ((q_kind == "c") & (k_kind == "c") & (k_i <= q_i))
    ref[:Np] = False
    ref[:Np, :Np] = True
    np.testing.assert_array_equal(_dense(Np, N, 1), ref)
    assert ref.shape == (nb, nb)


def test_hand_worked_mask_k3():
    # 1 prompt block, N = 4, K = 3: blocks 0 | n0..n3 = 1..4 | c0..c3 = 5..8
    rows = {0: [0], 1: [0, 1, 6, 7], 2: [0, 2, 5, 7, 8], 3: [0, 3, 5, 6, 8], 4: [0, 4, 5, 6, 7],
            5: [0, 5], 6: [0, 1, 6], 7: [0, 1, 2, 7], 8: [0, 2, 3, 5, 8]}
    m = _dense(1, 4, 3)
    for r, cols in rows.items():
        assert sorted(np.nonzero(m[r])[0].tolist()) == cols, r


@pytest.mark.parametrize("K", [2, 3, 5])
def test_no_noisy_block_reaches_its_clean_target_in_two_hops(K):
    # the stated purpose of removing the implicated CC links
    Np, N = 1, 9
    m = _dense(Np, N, K).astype(np.int64)
    two = m @ m
    for i in range(N):
        n_i, c_i = Np + i, Np + N + i
        assert m[n_i, c_i] == 0 and two[n_i, c_i] == 0
        # and it does see the next K-1 clean blocks (NF)
        for j in range(i + 1, min(i + K, N)):
            assert m[n_i, Np + N + j] == 1


def _rand(shape, g, scale=1.0):
    return (torch.randn(shape, generator=g) * scale).to(torch.bfloat16)


def _token_mask(mask_bits, nb, T, B):
    blk = oracle.mask_bits_to_dense(mask_bits, nb)
    t = np.arange(T) // B
    return blk[t[:, None], t[None, :]]


def _torch_attention(q, k, v, tmask, scale):
    """float64 masked attention with torch (GQA by repeating KV heads)."""
    T, Hq, D = q.shape
    G = Hq // k.shape[1]
    qd = q.double().permute(1, 0, 2)
    kd = k.double().repeat_interleave(G, dim=1).permute(1, 0, 2)
    vd = v.double().repeat_interleave(G, dim=1).permute(1, 0, 2)
    s = qd @ kd.transpose(1, 2) * scale
    s = s.masked_fill(~torch.from_numpy(tmask)[None], float("-inf"))
    p = torch.softmax(s, dim=-1)
    p = torch.nan_to_num(p, nan=0.0)
    return (p @ vd).permute(1, 0, 2), s


def test_forward_matches_torch_float64():
    g = torch.Generator().manual_seed(1)
    B, Np, N, K = 8, 1, 3, 2
    nb = Np + 2 * N
    T = nb * B - 3   # a ragged last block
    q, k, v = _rand((T, 4, 16), g), _rand((T, 2, 16), g), _rand((T, 2, 16), g)
    mb = oracle.sft_block_mask(Np, N, K)
    out, lse = oracle.block_mask_attention(bf16_bits(q), bf16_bits(k), bf16_bits(v), B, mb)
    ref, s = _torch_attention(q, k, v, _token_mask(mb, nb, T, B), 0.25)
    np.testing.assert_allclose(out, ref.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, np_logsumexp(s.numpy(), axis=-1).T, rtol=0, atol=1e-12)


def test_forward_with_a_block_causal_mask_is_the_window_oracle():
    # an independent oracle function: a block-causal window with no prefix
    from paper_2607_22663_gb300.workloads import BLOCK_CAUSAL, attention_problem
    B = 16
    prob = attention_problem([0], [80], [BLOCK_CAUSAL], 4, 2, 32, B, 16, seed=3)
    nb = 5
    mask = np.zeros((nb, 1), np.uint32)
    for qb in range(nb):
        mask[qb, 0] = (1 << (qb + 1)) - 1
    out, _ = oracle.block_mask_attention(bf16_bits(prob.q), bf16_bits(prob.k_win), bf16_bits(prob.v_win), B, mask)
    ref, _ = oracle.window_attention(bf16_bits(prob.q), bf16_bits(prob.k_win), bf16_bits(prob.v_win),
                                     bf16_bits(prob.k_cache), bf16_bits(prob.v_cache), prob.block_table.numpy(),
                                     prob.prefix_len.numpy(), prob.window_len.numpy(), prob.cu_window.numpy(),
                                     prob.mask_mode.numpy(), B, 16)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_gradients_match_torch_autograd_float64():
    g = torch.Generator().manual_seed(2)
    B, Np, N, K = 8, 1, 3, 3
    nb = Np + 2 * N
    T = nb * B
    q, k, v, do = _rand((T, 4, 16), g), _rand((T, 2, 16), g), _rand((T, 2, 16), g), _rand((T, 4, 16), g)
    mb = oracle.sft_block_mask(Np, N, K)
    dq, dk, dv = oracle.block_mask_attention_bwd(bf16_bits(q), bf16_bits(k), bf16_bits(v), bf16_bits(do), B, mb)
    qd, kd, vd = (t.double().requires_grad_() for t in (q, k, v))
    out, _ = _torch_attention(qd, kd, vd, _token_mask(mb, nb, T, B), 0.25)
    out.backward(do.double())
    np.testing.assert_allclose(dq, qd.grad.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(dk, kd.grad.numpy(), rtol=0, atol=1e-12)
    np.testing.assert_allclose(dv, vd.grad.numpy(), rtol=0, atol=1e-12)


def test_gradients_by_finite_differences():
    # central differences of L = sum(dO * O) in float64, for a few entries of q, k, v
    g = torch.Generator().manual_seed(4)
    B = 4
    T, Hq, Hkv, D = 12, 2, 1, 8
    q, k, v, do = _rand((T, Hq, D), g), _rand((T, Hkv, D), g), _rand((T, Hkv, D), g), _rand((T, Hq, D), g)
    mb = oracle.sft_block_mask(1, 1, 1)  # 3 blocks: prompt, n_0, c_0
    dq, dk, dv = oracle.block_mask_attention_bwd(bf16_bits(q), bf16_bits(k), bf16_bits(v), bf16_bits(do), B, mb)
    tmask = _token_mask(mb, 3, T, B)

    def loss(qx, kx, vx):
        o, _ = _torch_attention(qx, kx, vx, tmask, D ** -0.5)
        return float((o * do.double()).sum())

    eps = 1e-6
    for name, grad, idx in (("q", dq, (5, 1, 3)), ("k", dk, (2, 0, 7)), ("v", dv, (9, 0, 0)), ("k", dk, (10, 0, 1))):
        base = {"q": q.double(), "k": k.double(), "v": v.double()}
        plus = {n: t.clone() for n, t in base.items()}
        minus = {n: t.clone() for n, t in base.items()}
        plus[name][idx] += eps
        minus[name][idx] -= eps
        fd = (loss(plus["q"], plus["k"], plus["v"]) - loss(minus["q"], minus["k"], minus["v"])) / (2 * eps)
        assert abs(fd - grad[idx]) < 1e-7, (name, idx, fd, grad[idx])
