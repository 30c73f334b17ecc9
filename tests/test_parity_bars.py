"""The attention bars of tests/_bars.py have power where the absolute 1e-2
bound has none: on the CPU, with split pieces computed exactly from their
definition (and pinned to the oracle through the log-sum-exp merge identity
that split-KV merging relies on), a merge that drops a piece's output, drops a
whole piece, or weights pieces equally fails the bar, while a model of the
kernel's own rounding (bf16 P against a lazily raised maximum, fp32 sums,
bf16 output) passes it. The random-walk scale that the oracle yields on
doubled scores and squared values is pinned to its definition. No GPU."""
import numpy as np
import pytest
import torch

from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, AttnProblem, attention_problem
from tests._bars import HOEFFDING, U_BF16, derived_bar, excess, sigma_walk, walk_bar
from tests._util import dense_keys, oracle_attention, oracle_walk_scale, to_bf16_round

LOG2E = 1.4426950408889634


def _pieces(q, K, V, scale, cuts):
    """(o_k, lse_k) of attention restricted to keys [cuts[k], cuts[k+1])."""
    s = (q @ K.T) * scale
    outs, lses = [], []
    for a, b in zip(cuts[:-1], cuts[1:]):
        st = s[:, a:b]
        m = st.max(1, keepdims=True)
        p = np.exp(st - m)
        l = p.sum(1, keepdims=True)
        outs.append(p @ V[a:b] / l)
        lses.append((m + np.log(l))[:, 0])
    return outs, np.array(lses)


def _merge(outs, lses, mistake=None):
    M = lses.max(0)
    w = np.exp(lses - M)
    outs = [o.copy() for o in outs]
    if mistake == "drop_output":       # piece 1's O lost, its LSE kept
        outs[1][:] = 0.0
    elif mistake == "equal_weights":
        w = np.ones_like(w)
    elif mistake == "drop_piece":      # piece 1 lost entirely
        w[1] = 0.0
    return sum(w[k][:, None] * outs[k] for k in range(len(outs))) / w.sum(0)[:, None]


def _kernel_model(q, K, V, scale, cuts):
    """The kernel's arithmetic per piece: 128-key tiles, p = 2^(s - m) with m
    raised only when a tile's maximum exceeds it by more than 2^8, p rounded to
    bf16 for P V, row sums of the unrounded p; pieces merged by log-sum-exp;
    output rounded to bf16."""
    s = (q @ K.T) * scale * LOG2E
    outs, lses = [], []
    for a, b in zip(cuts[:-1], cuts[1:]):
        W = q.shape[0]
        m = np.full(W, -np.inf)
        l = np.zeros(W)
        O = np.zeros((W, V.shape[1]))
        for t0 in range(a, b, 128):
            st = s[:, t0:min(b, t0 + 128)]
            mx = st.max(1)
            raise_m = (m == -np.inf) | (mx > m + 8.0)
            m_new = np.where(raise_m, np.maximum(m, mx), m)
            alpha = np.where(m == -np.inf, 0.0, np.exp2(m - m_new))
            O *= alpha[:, None]
            l *= alpha
            m = m_new
            p = np.exp2(st - m[:, None]).astype(np.float32).astype(np.float64)
            l += p.sum(1)
            O += to_bf16_round(p) @ V[t0:t0 + st.shape[1]]
        outs.append(O / l[:, None])
        lses.append(m / LOG2E + np.log(l))
    return to_bf16_round(_merge(outs, np.array(lses)))


@pytest.mark.parametrize("q_scale", [1.0, 6.0])
def test_merge_mistakes_fail_the_bars_and_kernel_rounding_passes(q_scale):
    P, W, D = 12000, 64, 128
    prob = attention_problem([P], [W], [BIDIRECTIONAL], 1, 1, D, 32, 64, seed=23, q_scale=q_scale)
    o_full, _ = oracle_attention(prob)
    K, V = [x.numpy() for x in dense_keys(prob, 0, 0)]
    q = prob.q[:, 0].double().numpy()
    scale = D ** -0.5
    cuts = [0, 3000, 6000, 9000, P, P + W]            # four prefix pieces and the window
    outs, lses = _pieces(q, K, V, scale, cuts)
    ref = o_full[:, 0]
    # the exact pieces merge to the oracle's output: they are pinned to it
    np.testing.assert_allclose(_merge(outs, lses), ref, rtol=0, atol=1e-12)
    if q_scale == 1.0:
        bar = walk_bar(ref, oracle_walk_scale(prob)[:, 0])
    else:
        absv = AttnProblem(**{**prob.__dict__, "v_cache": prob.v_cache.abs(), "v_win": prob.v_win.abs()})
        spv = oracle_attention(absv)[0][:, 0]
        bar = derived_bar(ref, spv, P + W)
    assert excess(np.abs(to_bf16_round(_merge(outs, lses)) - ref), bar) <= 1.0
    assert excess(np.abs(_kernel_model(q, K, V, scale, cuts) - ref), bar) <= 1.0
    for mistake in ("drop_output", "equal_weights", "drop_piece"):
        err = np.abs(to_bf16_round(_merge(outs, lses, mistake)) - ref)
        assert excess(err, bar) > 20.0, mistake
        if q_scale == 1.0:
            # outputs of size ~1/sqrt(n): the absolute 1e-2 bound sees the same
            # mistake at least ten times less clearly (or not at all)
            assert excess(err, bar) > 10.0 * err.max() / 1e-2, mistake


def test_walk_scale_from_oracle_equals_its_definition():
    """sigma^2 = sum_j P_j^2 v_jd^2 over the visible keys, from the oracle run on
    doubled scores and squared values, equals the sum written out with the
    probabilities of the scores (block-causal mask, paged prefix, two heads)."""
    from paper_2607_22663_gb300.workloads import BLOCK_CAUSAL
    prob = attention_problem([300], [64], [BLOCK_CAUSAL], 2, 1, 64, 32, 32, seed=29)
    sig = oracle_walk_scale(prob)
    K, V = [x.numpy() for x in dense_keys(prob, 0, 0)]
    P, W = 300, 64
    i = np.arange(W)[:, None]
    j = np.arange(P + W)[None, :]
    vis = (j < P) | ((j - P) // 32 <= i // 32)
    v2 = to_bf16_round(V ** 2)          # the squared values the oracle receives (bf16)
    for h in range(2):
        s_ = (prob.q[:, h].double().numpy() @ K.T) / 8.0
        s_ = np.where(vis, s_, -np.inf)
        p = np.exp(s_ - s_.max(1, keepdims=True))
        p /= p.sum(1, keepdims=True)
        np.testing.assert_allclose(sig[:, h], np.sqrt((p ** 2) @ v2), rtol=1e-10)


def test_walk_bar_scale():
    """The walk part of the bar is 6.54 u sigma (Hoeffding at 1e-9 per element);
    the rounding part follows |o| with u = 2^-8."""
    o, sg = np.full((4, 8), 0.5), np.full((4, 8), 0.25)
    assert abs(HOEFFDING - 6.5447) < 1e-3
    np.testing.assert_allclose(walk_bar(o, sg), U_BF16 * 0.5 + HOEFFDING * U_BF16 * 0.25 + 1e-5)
