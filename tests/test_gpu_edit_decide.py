"""Parity of the CUDA edit-decide (mbe_edit_decide) with the fp64 oracle,
through the C ABI. Bar: argmax bit-exact, confidence rel. error <= 1e-5,
edit_mask/new_tokens bit-exact except at rows whose top-2 logit margin is
below 1e-6 or whose confidence is within 1e-6 of tau."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300 import workloads as wl
from paper_2607_22663_gb300.workloads import bf16_bits, edit_problem
from tests._gpu import compare_edit

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _oracle(logits_cpu, committed, tau=0.0, tau_per_row=None, editable=None, rows=None):
    if logits_cpu.dtype == torch.bfloat16:
        return oracle.edit_decide(bf16_bits(logits_cpu), committed.cpu().numpy(), tau=tau,
                                  tau_per_row=None if tau_per_row is None else tau_per_row.cpu().numpy(),
                                  editable=None if editable is None else editable.cpu().numpy(), rows=rows,
                                  is_bf16=True)
    return oracle.edit_decide(logits_cpu.numpy(), committed.cpu().numpy(), tau=tau,
                              tau_per_row=None if tau_per_row is None else tau_per_row.cpu().numpy(),
                              editable=None if editable is None else editable.cpu().numpy(), rows=rows)


def _check(prob, tau=None, tau_per_row=None, editable=None, rows=None):
    tau = prob.tau if tau is None else tau
    res = mbe.edit_decide(prob.logits, prob.committed, tau=tau, tau_per_row=tau_per_row, editable=editable)
    torch.cuda.synchronize()
    lc = prob.logits.cpu()
    ref = _oracle(lc, prob.committed, tau=tau, tau_per_row=tau_per_row, editable=editable, rows=rows)
    sel = np.arange(lc.shape[0]) if rows is None else np.asarray(rows)
    tau_rows = (tau_per_row.cpu().numpy()[sel] if tau_per_row is not None else np.full(len(sel), tau))
    return compare_edit(res, ref, lc[sel].double(), tau_rows, rows=sel), res, ref


def _median_conf(prob):
    res = mbe.edit_decide(prob.logits, prob.committed, tau=0.0)
    return float(res[2].median().item())


@pytest.mark.parametrize("name", ["tiny", "batch8"])
def test_workload_full(name):
    w = wl.WORKLOADS[name](DEV)
    prob = w["edit"]
    for tau in (prob.tau, 0.0, _median_conf(prob), 1.5):
        (rel, exempt), res, ref = _check(prob, tau=tau)
    # at tau = 0 (the paper's omega_edit) every differing row edits
    (_, _), res, ref = _check(prob, tau=0.0)
    assert res[1].sum().item() == int((ref["argmax"] != prob.committed.cpu().numpy()).sum())


def test_varlen64_per_row_tau_full():
    w = wl.varlen64(DEV)
    prob = w["edit"]
    _check(prob, tau_per_row=prob.tau_per_row)
    # a tau that splits the rows, so the threshold really decides
    (_, _), res, _ = _check(prob, tau=_median_conf(prob))
    assert 0 < res[1].sum().item() < prob.logits.shape[0]


def test_serving128_full_size_sampled():
    prob = wl.serving128(DEV, layers=1)["edit"]
    rows = sorted(torch.randperm(prob.logits.shape[0], generator=torch.Generator().manual_seed(0))[:768].tolist())
    editable = wl.editable_historical([64] * 128, 32, DEV)
    for tau in (0.9, 0.0, _median_conf(prob)):
        _check(prob, tau=tau, editable=editable, rows=rows)


def test_sharp_peaks_edit_at_high_tau():
    prob = edit_problem(256, 32768, torch.bfloat16, seed=4, device=DEV, peak_frac=1.0, peak_lo=40.0, peak_hi=40.0)
    (_, _), res, ref = _check(prob, tau=0.9)
    assert res[1].float().mean().item() > 0.9


@pytest.mark.parametrize("vocab,dtype", [(1000, torch.float32), (1003, torch.bfloat16), (7, torch.float32),
                                         (131073, torch.bfloat16), (1, torch.float32)])
def test_ragged_vocab_and_tails(vocab, dtype):
    prob = edit_problem(37, vocab, dtype, seed=vocab, device=DEV, peak_frac=0.5, peak_lo=1.0, peak_hi=6.0)
    _check(prob, tau=0.0)
    _check(prob, tau=_median_conf(prob))


def test_strided_rows_unaligned_path():
    base = edit_problem(64, 1003, torch.float32, seed=3, device=DEV)
    big = torch.zeros(64, 1010, dtype=torch.float32, device=DEV)
    big[:, :1003] = base.logits
    view = big[:, :1003]
    res = mbe.edit_decide(view, base.committed, tau=0.0)
    ref = _oracle(base.logits.cpu(), base.committed, tau=0.0)
    compare_edit(res, ref, base.logits.cpu().double(), np.zeros(64))


def test_exact_ties_pick_lowest_index():
    logits = torch.zeros(8, 4096, dtype=torch.bfloat16, device=DEV)
    for r in range(8):
        logits[r, [100 + r, 3000 - r, 4095]] = 5.0
    committed = torch.full((8,), 4095, dtype=torch.int32, device=DEV)
    new, mask, conf, am = mbe.edit_decide(logits, committed, tau=0.0)
    assert am.cpu().tolist() == [100 + r for r in range(8)]
    assert mask.all().item()


def test_uniform_rows_confidence_one_over_v():
    logits = torch.full((4, 50000), 0.25, dtype=torch.float32, device=DEV)
    committed = torch.zeros(4, dtype=torch.int32, device=DEV)
    new, mask, conf, am = mbe.edit_decide(logits, committed, tau=0.0)
    assert (am == 0).all().item() and not mask.any().item()
    assert torch.allclose(conf.double(), torch.full((4,), 1 / 50000, dtype=torch.float64, device=DEV), rtol=1e-5)


def test_new_tokens_may_alias_committed():
    prob = edit_problem(128, 4096, torch.bfloat16, seed=9, device=DEV)
    ref = mbe.edit_decide(prob.logits, prob.committed.clone(), tau=0.0)
    c = prob.committed.clone()
    mbe.edit_decide(prob.logits, c, tau=0.0, new_tokens=c)
    assert torch.equal(c, ref[0])


@pytest.mark.parametrize("dtype,vocab", [(torch.float32, 1000), (torch.bfloat16, 32768), (torch.bfloat16, 37)])
def test_rows_without_softmax_and_vocabulary_masks(dtype, vocab):
    """Rows with a NaN or +inf logit, or with every logit -inf, get no decision:
    the token stays, argmax is -1, confidence NaN, and the call raises
    MBE_DEVERR_NONFINITE. -inf logits beside finite ones are tokens of
    probability 0, also where they fill whole 16-byte vectors at the start of a
    thread's stride or the scalar tail. Every other row matches the oracle."""
    R = 40
    g = torch.Generator().manual_seed(vocab)
    logits = torch.randn(R, vocab, generator=g) * 2.0
    logits[torch.arange(R), torch.randint(0, vocab, (R,), generator=g)] += 5.0
    committed = torch.randint(0, vocab, (R,), generator=g, dtype=torch.int64).to(torch.int32)
    logits[3, vocab // 2] = float("nan")
    logits[7, vocab - 1] = float("inf")
    logits[11, :] = float("-inf")
    logits[13, 0] = float("nan")
    logits[13, 1:] = float("-inf")
    logits[17, : min(vocab - 1, 4096)] = float("-inf")       # leading vectors of every thread
    logits[19, :-1] = float("-inf")                           # only the last entry (scalar tail if ragged) is finite
    logits[21] = logits[21].masked_fill(torch.rand(vocab, generator=g) < 0.3, float("-inf"))
    lc = logits.to(dtype)
    res = mbe.edit_decide(lc.to(DEV), committed.to(DEV), tau=0.0)
    st, flags = mbe.get_device_error()
    assert st == 6 and flags == mbe.DEVERR_NONFINITE
    ref = _oracle(lc, committed, tau=0.0)
    assert ref["undecidable"]
    new_g, mask_g, conf_g, am_g = [t.cpu().numpy() for t in res]
    bad = np.array([3, 7, 11, 13])
    assert (ref["argmax"][bad] == -1).all()
    np.testing.assert_array_equal(am_g[bad], -1)
    np.testing.assert_array_equal(new_g[bad], committed.numpy()[bad])
    assert not mask_g[bad].any() and np.isnan(conf_g[bad]).all()
    good = np.array([r for r in range(R) if r not in bad])
    compare_edit(res, ref, lc[good].double(), np.zeros(len(good)), rows=good)
    assert am_g[19] == vocab - 1 and conf_g[19] == 1.0
    assert mbe.get_device_error() == (0, 0)
