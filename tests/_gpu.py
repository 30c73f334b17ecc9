"""GPU-test helpers: run the CUDA path through the binding, carve sampled
sequences out of a large problem for the oracle, and compare."""
import numpy as np
import torch

from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300.workloads import AttnProblem, bf16_bits
from paper_2607_22663_gb300.workloads import extract_sequences as subproblem

ATTN_ATOL = 1e-2      # max abs error of bf16 attention outputs vs the fp64 oracle
CONF_RTOL = 1e-5      # relative error of fp32 confidences vs the fp64 oracle
TIE_EPS = 1e-6        # decisions within this margin (top-2 gap, |c - tau|) are exempt


def run_attention(prob: AttnProblem, softmax_scale=0.0):
    out, lse = mbe.window_attention(prob.q, prob.k_win, prob.v_win, prob.k_cache, prob.v_cache, prob.block_table,
                                    prob.prefix_len, prob.window_len, prob.cu_window, prob.mask_mode,
                                    block_size=prob.block_size, max_window=max(prob.max_window, 1),
                                    max_prefix=prob.max_prefix, softmax_scale=softmax_scale, return_lse=True)
    st, flags = mbe.get_device_error()
    assert st == 0, (st, flags)
    return out, lse


def oracle_attention(prob: AttnProblem, units=None, scale=None):
    import oracle
    return oracle.window_attention(bf16_bits(prob.q), bf16_bits(prob.k_win), bf16_bits(prob.v_win),
                                   bf16_bits(prob.k_cache), bf16_bits(prob.v_cache), prob.block_table.cpu().numpy(),
                                   prob.prefix_len.cpu().numpy(), prob.window_len.cpu().numpy(),
                                   prob.cu_window.cpu().numpy(), prob.mask_mode.cpu().numpy(), prob.block_size,
                                   prob.page_size, scale=scale, units=units)


def compare_attention(prob: AttnProblem, out_gpu, lse_gpu, seqs=None, heads=None, scale=None, derived_bound=False):
    """Compare GPU outputs of the listed (sequence, q-head) pairs with the oracle.

    Default bar: max abs error <= ATTN_ATOL. With derived_bound, each element
    must instead satisfy |err| <= u * (max|v| + |o_ref|) + 1e-4, u = 2^-8 the
    bf16 unit roundoff: the probabilities are rounded to bf16 before the PV
    product (error <= u * sum_j p_j |v_j| <= u * max|v|) and the output is
    rounded to bf16 (error <= u * |o|); fp32 accumulation adds < 1e-4. This is
    the bar for inputs sharpened so that outputs are O(1).
    Returns (max abs error, max abs error / output RMS)."""
    seqs = list(range(prob.batch)) if seqs is None else list(seqs)
    Hq = prob.num_q_heads
    heads = list(range(Hq)) if heads is None else list(heads)
    sub = subproblem(prob, seqs)
    units = [(i, h) for i in range(len(seqs)) for h in heads]
    o_ref, l_ref = oracle_attention(sub, units=units, scale=scale)
    cu_all = prob.cu_window.cpu()
    worst, worst_rel = 0.0, 0.0
    for i, s in enumerate(seqs):
        W = prob.window_host[s]
        if W == 0:
            continue
        t0, u0 = int(cu_all[s]), int(sub.cu_window[i])
        g = out_gpu[t0:t0 + W][:, heads].float().cpu().numpy()
        r = o_ref[u0:u0 + W][:, heads]
        err = np.abs(g - r).max()
        rms = np.sqrt((r ** 2).mean()) + 1e-30
        if derived_bound:
            vmax = max(prob.v_cache.float().abs().max().item(), prob.v_win.float().abs().max().item())
            bound = 2.0 ** -8 * (vmax + np.abs(r)) + 1e-4
            assert (np.abs(g - r) <= bound).all(), f"error above the derived bf16 bound (max err {err})"
        worst, worst_rel = max(worst, err), max(worst_rel, err / rms)
        if lse_gpu is not None:
            lg = lse_gpu[t0:t0 + W][:, heads].cpu().numpy()
            lr = l_ref[u0:u0 + W][:, heads]
            np.testing.assert_allclose(lg, lr, rtol=0, atol=2e-3 * max(1.0, np.abs(lr).max()))
    if not derived_bound:
        assert worst <= ATTN_ATOL, f"max abs error {worst} > {ATTN_ATOL} (rel to rms {worst_rel})"
    return worst, worst_rel


def compare_edit(res_gpu, res_ref, logits64, tau_rows, rows=None):
    """Bit-exact argmax; confidence within CONF_RTOL; edit/new exact except at
    near-ties (top-2 margin < TIE_EPS) or near-threshold rows (|c - tau| < TIE_EPS)."""
    new_g, mask_g, conf_g, am_g = [t.cpu().numpy() for t in res_gpu]
    rows = np.arange(len(new_g)) if rows is None else np.asarray(rows)
    am_r = res_ref["argmax"][rows]
    conf_r = res_ref["confidence"][rows]
    if logits64.shape[1] >= 2:
        top2 = torch.topk(logits64, 2, dim=1).values
        margin = (top2[:, 0] - top2[:, 1]).numpy()
    else:
        margin = np.full(logits64.shape[0], np.inf)
    near_tie = margin < TIE_EPS
    near_tau = np.abs(conf_r - tau_rows) < TIE_EPS
    exempt = near_tie | near_tau
    ok_am = (am_g[rows] == am_r) | near_tie
    assert ok_am.all(), f"argmax mismatch at rows {rows[~ok_am][:10]}"
    rel = np.abs(conf_g[rows] - conf_r) / conf_r
    assert rel.max() <= CONF_RTOL, f"confidence rel err {rel.max()}"
    bad = ((mask_g[rows] != res_ref["edit_mask"][rows]) | (new_g[rows] != res_ref["new_tokens"][rows])) & ~exempt
    assert not bad.any(), f"edit mismatch at rows {rows[bad][:10]}"
    return rel.max(), int(exempt.sum())
