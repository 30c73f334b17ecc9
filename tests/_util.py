"""Helpers shared by the tests: dense re-gathering of paged K/V (independent of
both the oracle and the CUDA path) and bf16 conversions."""
import numpy as np
import torch

from paper_2607_22663_gb300.workloads import bf16_bits


def dense_keys(prob, s, g):
    """Logical key/value rows [P+W, D] (float64) of sequence s, kv head g, gathered
    with torch indexing from the paged cache and the window tensors."""
    P, W = prob.prefix_host[s], prob.window_host[s]
    ps = prob.page_size
    pos = torch.arange(P)
    pages = prob.block_table[s].cpu()[pos // ps].long()
    kp = prob.k_cache.cpu()[pages, g, pos % ps].double()
    vp = prob.v_cache.cpu()[pages, g, pos % ps].double()
    t0 = int(prob.cu_window.cpu()[s])
    kw = prob.k_win.cpu()[t0:t0 + W, g].double()
    vw = prob.v_win.cpu()[t0:t0 + W, g].double()
    return torch.cat([kp, kw]), torch.cat([vp, vw])


def np_logsumexp(s, axis=-1):
    """log(sum(exp(s))) along an axis in float64, shifted by the row maximum; rows
    that are all -inf give -inf. numpy rather than torch.logsumexp: torch's CPU
    kernel returned values up to 3e-10 off in some rows on the first call of a
    process (about one process in thirty), while the scores it was given were exact."""
    s = np.asarray(s, dtype=np.float64)
    m = np.max(s, axis=axis, keepdims=True)
    m_safe = np.where(np.isfinite(m), m, 0.0)
    with np.errstate(divide="ignore"):
        out = np.log(np.sum(np.exp(s - m_safe), axis=axis, keepdims=True)) + m_safe
    return np.squeeze(out, axis=axis)


def oracle_attention(prob, units=None, scale=None):
    import oracle
    return oracle.window_attention(bf16_bits(prob.q), bf16_bits(prob.k_win), bf16_bits(prob.v_win),
                                   bf16_bits(prob.k_cache), bf16_bits(prob.v_cache),
                                   prob.block_table.cpu().numpy(), prob.prefix_len.cpu().numpy(),
                                   prob.window_len.cpu().numpy(), prob.cu_window.cpu().numpy(),
                                   prob.mask_mode.cpu().numpy(), prob.block_size, prob.page_size, scale=scale,
                                   units=units)


def to_bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float64 values to the nearest bf16 (ties to even), returned as float64."""
    return torch.from_numpy(np.ascontiguousarray(x)).to(torch.bfloat16).double().numpy()


def oracle_walk_scale(prob, units=None, scale=None):
    """sqrt(sum_j P_j^2 v_jd^2) per output element [T, Hq, D] (tests/_bars.py):
    the oracle on the scores for lse, and on doubled scores with the values
    squared (rounded to bf16) for the weighted sum of v^2."""
    import math

    from paper_2607_22663_gb300.workloads import AttnProblem
    from tests._bars import sigma_walk
    sc = scale if scale is not None else 1.0 / math.sqrt(prob.head_dim)
    _, lse = oracle_attention(prob, units=units, scale=sc)
    sq = lambda t: (t.float() ** 2).to(torch.bfloat16)
    prob2 = AttnProblem(**{**prob.__dict__, "v_cache": sq(prob.v_cache), "v_win": sq(prob.v_win)})
    out2, lse2 = oracle_attention(prob2, units=units, scale=2.0 * sc)
    return sigma_walk(lse, lse2, out2)
