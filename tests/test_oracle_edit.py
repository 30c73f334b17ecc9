"""Pins of the edit-decide oracle (Eq. 2 T2T rule) against library routines,
closed forms and invariants. CPU only."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300.workloads import bf16_bits, edit_problem

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _torch_reference(logits64, committed, tau_rows, editable=None):
    p = torch.softmax(logits64, dim=1)
    am = torch.argmax(logits64, dim=1)          # first maximal index on ties
    c = p.gather(1, am[:, None])[:, 0]
    ed = (am != committed) & (c.float() > tau_rows)
    if editable is not None:
        ed &= editable.bool()
    new = torch.where(ed, am, committed)
    return am, c, ed, new


@pytest.mark.parametrize("rows,vocab,dtype", [(64, 1024, torch.float32), (40, 777, torch.bfloat16),
                                              (8, 32768, torch.bfloat16)])
def test_oracle_matches_torch_softmax_argmax(rows, vocab, dtype):
    prob = edit_problem(rows, vocab, dtype, seed=7, peak_frac=0.6, peak_lo=2.0, peak_hi=10.0)
    # thresholds spread around the median confidence so that about half the
    # candidate rows edit (a rule that ignored tau would fail)
    c_med = torch.softmax(prob.logits.double(), dim=1).max(dim=1).values.median().item()
    taus = torch.rand(rows, generator=torch.Generator().manual_seed(3)) * 2 * c_med
    editable = (torch.arange(rows) % 3 != 0).to(torch.uint8)
    if dtype == torch.bfloat16:
        res = oracle.edit_decide(bf16_bits(prob.logits), prob.committed.numpy(), tau_per_row=taus.numpy(),
                                 editable=editable.numpy(), is_bf16=True)
    else:
        res = oracle.edit_decide(prob.logits.numpy(), prob.committed.numpy(), tau_per_row=taus.numpy(),
                                 editable=editable.numpy())
    am, c, ed, new = _torch_reference(prob.logits.double(), prob.committed.long(), taus, editable)
    np.testing.assert_array_equal(res["argmax"], am.numpy())
    np.testing.assert_allclose(res["confidence"], c.numpy(), rtol=1e-13)
    np.testing.assert_array_equal(res["edit_mask"], ed.numpy().astype(np.uint8))
    np.testing.assert_array_equal(res["new_tokens"], new.numpy())
    assert res["edit_mask"].any() and not res["edit_mask"].all()


def test_golden_closed_forms():
    spec = json.load(open(os.path.join(GOLDEN, "edit_decide_closed_forms.json")))
    for case in spec["cases"]:
        logits = np.array([case["logits"]], dtype=np.float32)
        expected_c = eval(case["conf_expr"], {"math": math})
        for chk in case["checks"]:
            res = oracle.edit_decide(logits, np.array([case["committed"]]), tau=chk["tau"])
            assert res["argmax"][0] == case["argmax"], case["name"]
            # float32 logits (ln 3 is rounded), so allow a few float32 ulps of the logit
            assert abs(res["confidence"][0] - expected_c) < 1e-6, case["name"]
            assert res["edit_mask"][0] == chk["edit"], (case["name"], chk)
            assert res["new_tokens"][0] == chk["new"], (case["name"], chk)


def test_uniform_rows_give_one_over_v_and_index_zero():
    for V in (1, 2, 5, 1000):
        logits = np.full((3, V), -2.25, dtype=np.float32)
        res = oracle.edit_decide(logits, np.array([0, 1, V - 1]), tau=0.0)
        assert (res["argmax"] == 0).all()
        np.testing.assert_allclose(res["confidence"], 1.0 / V, rtol=1e-15)


def test_tau_above_one_changes_nothing():
    prob = edit_problem(128, 512, torch.float32, seed=1, peak_frac=1.0, peak_lo=30.0, peak_hi=40.0)
    res = oracle.edit_decide(prob.logits.numpy(), prob.committed.numpy(), tau=1.5)
    assert not res["edit_mask"].any()
    np.testing.assert_array_equal(res["new_tokens"], prob.committed.numpy())
    # the same rows at tau 0 do edit wherever argmax != committed: the pin has power
    res0 = oracle.edit_decide(prob.logits.numpy(), prob.committed.numpy(), tau=0.0)
    assert res0["edit_mask"].sum() > 100


def test_committed_equal_argmax_is_fixed_point():
    prob = edit_problem(64, 300, torch.float32, seed=2, peak_frac=0.5, peak_lo=3.0, peak_hi=6.0)
    am = prob.logits.argmax(dim=1).to(torch.int32).numpy()
    res = oracle.edit_decide(prob.logits.numpy(), am, tau=-1.0)
    assert not res["edit_mask"].any()
    np.testing.assert_array_equal(res["new_tokens"], am)


def test_tau_zero_edits_exactly_where_prediction_differs():
    prob = edit_problem(200, 64, torch.float32, seed=3)
    res = oracle.edit_decide(prob.logits.numpy(), prob.committed.numpy(), tau=0.0)
    np.testing.assert_array_equal(res["edit_mask"].astype(bool), res["argmax"] != prob.committed.numpy())


def test_confidence_bounds():
    prob = edit_problem(300, 97, torch.float32, seed=4, sd=5.0, peak_frac=0.3, peak_lo=0.0, peak_hi=50.0)
    res = oracle.edit_decide(prob.logits.numpy(), prob.committed.numpy(), tau=0.5)
    c = res["confidence"]
    assert (c >= 1.0 / 97 - 1e-15).all() and (c <= 1.0).all()


def test_bf16_path_equals_float_path_on_rounded_values():
    prob = edit_problem(32, 1000, torch.bfloat16, seed=6)
    rb = oracle.edit_decide(bf16_bits(prob.logits), prob.committed.numpy(), tau=0.2, is_bf16=True)
    rf = oracle.edit_decide(prob.logits.float().numpy(), prob.committed.numpy(), tau=0.2)
    for k in rb:
        np.testing.assert_array_equal(rb[k], rf[k])


def test_row_subset_matches_full():
    prob = edit_problem(16, 50, torch.float32, seed=8)
    full = oracle.edit_decide(prob.logits.numpy(), prob.committed.numpy(), tau=0.1)
    sub = oracle.edit_decide(prob.logits.numpy(), prob.committed.numpy(), tau=0.1, rows=[3, 9])
    for r in (3, 9):
        assert sub["argmax"][r] == full["argmax"][r]
        assert sub["confidence"][r] == full["confidence"][r]
    assert not full["undecidable"] and not sub["undecidable"]


@pytest.mark.parametrize("bad", ["nan", "posinf", "all_neginf"])
def test_row_without_softmax_keeps_its_token(bad):
    """Eq. 2 needs the softmax of the row. A row with a NaN or +inf logit, or
    with every logit -inf, has none: its token stays (no edit, even at tau < 0),
    its argmax is -1 and its confidence NaN, and every other row is decided as
    if that row were absent."""
    prob = edit_problem(12, 40, torch.float32, seed=9, peak_frac=1.0, peak_lo=30.0, peak_hi=40.0)
    logits = prob.logits.numpy().copy()
    committed = (prob.logits.argmax(dim=1).numpy() + 1) % 40   # every decidable row edits at tau < 0
    if bad == "nan":
        logits[5, 17] = np.nan
    elif bad == "posinf":
        logits[5, 3] = np.inf
    else:
        logits[5, :] = -np.inf
    res = oracle.edit_decide(logits, committed, tau=-1.0)
    assert res["undecidable"]
    assert res["new_tokens"][5] == committed[5] and res["edit_mask"][5] == 0
    assert res["argmax"][5] == -1 and np.isnan(res["confidence"][5])
    others = np.array([r for r in range(12) if r != 5])
    ref = oracle.edit_decide(logits[others], committed[others], tau=-1.0)
    assert not ref["undecidable"]
    for k in ("new_tokens", "edit_mask", "confidence", "argmax"):
        np.testing.assert_array_equal(res[k][others], ref[k])
    assert ref["edit_mask"].all()


def test_neginf_logits_are_tokens_of_probability_zero():
    """A -inf logit beside finite ones (a vocabulary mask) is a token of
    probability 0: argmax and confidence equal torch's softmax over the finite
    entries, i.e. the same row with those tokens removed."""
    prob = edit_problem(20, 300, torch.float32, seed=10, peak_frac=0.5, peak_lo=1.0, peak_hi=6.0)
    logits = prob.logits.numpy().copy()
    g = np.random.default_rng(0)
    hidden = g.random(logits.shape) < 0.3
    hidden[:, 0] = True                       # the first token of every row is masked
    logits[hidden] = -np.inf
    res = oracle.edit_decide(logits, prob.committed.numpy(), tau=0.0)
    assert not res["undecidable"]
    p = torch.softmax(torch.from_numpy(logits).double(), dim=1)
    np.testing.assert_array_equal(res["argmax"], p.argmax(dim=1).numpy())
    np.testing.assert_allclose(res["confidence"], p.max(dim=1).values.numpy(), rtol=1e-13)
    for r in range(3):
        keep = np.flatnonzero(~hidden[r])
        red = oracle.edit_decide(logits[r:r + 1, keep], np.array([0]), tau=0.0)
        assert keep[red["argmax"][0]] == res["argmax"][r]
        np.testing.assert_allclose(red["confidence"][0], res["confidence"][r], rtol=1e-14)
