"""Parity of mbe_lm_head_edit_decide (LM-head projection fused with the edit
decision of Eq. 2) with the oracle, through the C ABI.

The oracle forms the logits in float64 from the same bf16 inputs; the kernel
accumulates them in fp32 on the tensor cores: a running fp32 sum updated once
per 16-deep MMA step. Every update rounds by at most 2^-23 of a partial sum
bounded by A_v = sum_k |h_k w_vk| (2^-23 also covers truncating accumulation),
so |l_gpu - l_ref| <= eps_v = (ceil(d/16) + 1) * 2^-23 * A_v. From this bound:
  - argmax: the GPU's choice is within 2 eps of the row maximum, and equal to
    the oracle's wherever the top-2 margin exceeds 2 eps;
  - confidence: |ln c_gpu - ln c_ref| <= 2 eps, plus the 1e-5 relative error of
    the fp32 softmax sums;
  - entropy: dH/dl_v = -p_v (ln p_v + H), so |dH| <= 2 H eps, plus the 5e-4
    of the fp32 entropy evaluation;
  - decisions: bit-exact except rows with an ambiguous argmax or a confidence
    within the confidence bar of the threshold.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300.workloads import bf16_bits

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _problem(R, V, d, seed, peak_frac=0.5, argmax_frac=0.3, device="cpu"):
    g = torch.Generator(device=device).manual_seed(seed)
    h = torch.randn(R, d, generator=g, device=device)
    w = torch.randn(V, d, generator=g, device=device) * (2.0 / math.sqrt(d))
    # plant confident predictions: W[v_r] gains a component along H[r]
    n_peak = int(peak_frac * R)
    rows = torch.randperm(R, generator=g, device=device)[:n_peak]
    toks = torch.randint(0, V, (n_peak,), generator=g, device=device)
    alpha = 4.0 + 8.0 * torch.rand(n_peak, generator=g, device=device)
    w.index_add_(0, toks, h[rows] * (alpha / (h[rows] ** 2).sum(1)).unsqueeze(1))
    committed = torch.randint(0, V, (R,), generator=g, device=device, dtype=torch.int32)
    return h.to(torch.bfloat16), w.to(torch.bfloat16), committed, argmax_frac


def _bounds(h, w, rows):
    """eps_v of the module docstring for the given rows: [len(rows), V]."""
    d = h.shape[1]
    idx = torch.as_tensor(np.asarray(rows), device=h.device).long()
    A = (h[idx].double().abs() @ w.double().abs().T).cpu()
    return (math.ceil(d / 16) + 1) * 2.0 ** -23 * A.numpy()


def _check(h, w, committed, tau, res, rows=None, editable=None):
    R, V = h.shape[0], w.shape[0]
    rows = np.arange(R) if rows is None else np.asarray(rows)
    logits = oracle.lm_head_logits(bf16_bits(h.cpu()), bf16_bits(w.cpu()), rows=rows)
    eps = _bounds(h, w, rows).max(axis=1)
    new_g, mask_g, conf_g, am_g, ent_g = [None if t is None else t.cpu().numpy()[rows] for t in res]
    ref = oracle.edit_decide(logits, committed.cpu().numpy()[rows], tau=tau,
                             editable=None if editable is None else editable.cpu().numpy()[rows])
    den = oracle.denoise_update(logits, committed.cpu().numpy()[rows], [0, len(rows)], 32, -1, 0.5, 0.0)
    top2 = np.sort(logits, axis=1)[:, -2:]
    margin = top2[:, 1] - top2[:, 0]
    lmax = top2[:, 1]
    # argmax: valid within 2 eps everywhere, exact where the margin is clear
    picked = logits[np.arange(len(rows)), am_g]
    assert (picked >= lmax - 2 * eps).all()
    clear = margin > 2 * eps
    assert (am_g[clear] == ref["argmax"][clear]).all()
    # confidence and entropy within the derived bars
    c_bar = np.expm1(2 * eps) + 1e-5
    assert (np.abs(np.log(conf_g) - np.log(ref["confidence"])) <= c_bar).all()
    if ent_g is not None:
        assert (np.abs(ent_g - den["entropy"]) <= 5e-4 + 2 * den["entropy"] * eps).all()
    # decisions exact away from ambiguous argmaxes and near-threshold confidences
    near = np.abs(ref["confidence"] - tau) <= c_bar * ref["confidence"]
    exempt = ~clear | near
    ok = (new_g == ref["new_tokens"]) & (mask_g == ref["edit_mask"])
    assert (ok | exempt).all(), np.nonzero(~(ok | exempt))[0][:10]
    if len(rows) >= 100:
        assert exempt.mean() < 0.05, f"too many exempt rows: {exempt.mean()}"
    return ref, exempt


@pytest.mark.parametrize("R,V,d", [(300, 5000, 512), (1, 100, 200), (129, 2304, 64), (257, 4097, 136)])
def test_matches_oracle_ragged(R, V, d):
    h, w, committed, _ = _problem(R, V, d, seed=R + V + d)
    hd, wd, cd = h.to(DEV), w.to(DEV), committed.to(DEV)
    # committed = the oracle argmax on a third of the rows (no edit there)
    logits = oracle.lm_head_logits(bf16_bits(h), bf16_bits(w))
    keep = np.arange(R) % 3 == 0
    cd[torch.from_numpy(keep).to(DEV)] = torch.from_numpy(logits.argmax(1)[keep].astype(np.int32)).to(DEV)
    confs = torch.softmax(torch.from_numpy(logits), 1).max(1).values
    for tau in (0.0, float(confs.median()), 1.5):
        res = mbe.lm_head_edit_decide(hd, wd, cd, tau=tau, want_entropy=True)
        torch.cuda.synchronize()
        ref, _ = _check(h, w, cd, tau, res)
        if tau > 1.0:
            assert not res[1].any() and torch.equal(res[0], cd)
    assert mbe.get_device_error() == (0, 0)


def test_tau_per_row_and_editable():
    R, V, d = 200, 3000, 256
    h, w, committed, _ = _problem(R, V, d, seed=5)
    hd, wd, cd = h.to(DEV), w.to(DEV), committed.to(DEV)
    g = torch.Generator().manual_seed(6)
    tpr = (torch.rand(R, generator=g) * 0.9).to(DEV)
    editable = (torch.arange(R) % 4 != 1).to(torch.uint8).to(DEV)
    res = mbe.lm_head_edit_decide(hd, wd, cd, tau_per_row=tpr, editable=editable)
    torch.cuda.synchronize()
    rows = np.arange(R)
    logits = oracle.lm_head_logits(bf16_bits(h), bf16_bits(w))
    ref = oracle.edit_decide(logits, cd.cpu().numpy(), tau_per_row=tpr.cpu().numpy(), editable=editable.cpu().numpy())
    eps = _bounds(h, w, rows).max(axis=1)
    top2 = np.sort(logits, axis=1)[:, -2:]
    exempt = (top2[:, 1] - top2[:, 0] <= 2 * eps) | \
        (np.abs(ref["confidence"] - tpr.cpu().numpy()) <= (np.expm1(2 * eps) + 1e-5) * ref["confidence"])
    ok = (res[0].cpu().numpy() == ref["new_tokens"]) & (res[1].cpu().numpy() == ref["edit_mask"])
    assert (ok | exempt).all()
    assert not res[1].cpu().numpy()[np.arange(R) % 4 == 1].any()


def test_full_size_sampled_rows():
    # the serving projection: 8192 window rows, 131072-token vocabulary, hidden 4096
    R, V, d = 8192, 131072, 4096
    h, w, committed, _ = _problem(R, V, d, seed=7, device=DEV)
    res = mbe.lm_head_edit_decide(h, w, committed, tau=0.5, want_entropy=True)
    torch.cuda.synchronize()
    assert mbe.get_device_error() == (0, 0)
    rows = [0, 127, 128, 4095, 5000, 8063, 8190, 8191]
    _check(h, w, committed, 0.5, res, rows=rows)


def test_argument_errors():
    h, w, c, _ = _problem(4, 64, 64, seed=8)
    hd, wd, cd = h.to(DEV), w.to(DEV), c.to(DEV)
    with pytest.raises(mbe.MbeError):
        mbe.lm_head_edit_decide(hd, wd, cd, workspace=torch.empty(16, dtype=torch.uint8, device=DEV))
    with pytest.raises(mbe.MbeError):     # hidden_dim not a multiple of 8
        mbe.lm_head_edit_decide(hd[:, :60].contiguous(), wd[:, :60].contiguous(), cd)
    # zero rows: nothing to do
    out = mbe.lm_head_edit_decide(hd[:0], wd, cd[:0])
    assert out[0].numel() == 0


def test_non_finite_hidden_row_gets_no_decision():
    """A hidden row holding NaN (or +inf) makes every logit of its row NaN: that
    row keeps its token with argmax -1 and confidence / entropy NaN, and
    MBE_DEVERR_NONFINITE is raised. Each row's logits depend on its own hidden
    row only, so every other row is bit-identical to the run without it."""
    R, V, d = 160, 3000, 256
    h, w, committed, _ = _problem(R, V, d, seed=9)
    hd, wd, cd = h.to(DEV), w.to(DEV), committed.to(DEV)
    ref = mbe.lm_head_edit_decide(hd, wd, cd, tau=0.0, want_entropy=True)
    assert mbe.get_device_error() == (0, 0)
    hb = hd.clone()
    hb[5, 17] = float("nan")
    hb[130, :] = float("inf")
    res = mbe.lm_head_edit_decide(hb, wd, cd, tau=0.0, want_entropy=True)
    st, flags = mbe.get_device_error()
    assert st == 6 and flags == mbe.DEVERR_NONFINITE
    bad = [5, 130]
    new, mask, conf, am, ent = res
    assert (am[bad] == -1).all() and torch.equal(new[bad], cd[bad]) and not mask[bad].any()
    assert torch.isnan(conf[bad]).all() and torch.isnan(ent[bad]).all()
    good = torch.tensor([r for r in range(R) if r not in bad], device=DEV)
    for a, b in zip(res, ref):
        assert torch.equal(a[good], b[good])
