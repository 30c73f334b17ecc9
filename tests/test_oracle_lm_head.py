"""Pins of the oracle's LM-head projection (the logits the T2T rule of Eq. 2
reads) and of its float64 path through the edit decision. CPU only."""
import numpy as np
import torch

import oracle
from paper_2607_22663_gb300.workloads import bf16_bits


def _bf16(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(shape, generator=g) * scale).to(torch.bfloat16)


def test_logits_match_a_float64_matmul():
    h, w = _bf16((9, 200), 1, 0.3), _bf16((77, 200), 2, 0.3)
    got = oracle.lm_head_logits(bf16_bits(h), bf16_bits(w))
    ref = h.double().numpy() @ w.double().numpy().T
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_one_hot_hidden_rows_select_weight_columns_exactly():
    d, V = 24, 50
    w = _bf16((V, d), 3)
    h = torch.zeros(d, d, dtype=torch.bfloat16)
    h[torch.arange(d), torch.arange(d)] = 1.0      # row k picks hidden unit k (the last one included)
    got = oracle.lm_head_logits(bf16_bits(h), bf16_bits(w))
    np.testing.assert_array_equal(got, w.double().numpy().T)
    # scaling a one-hot row by 2 doubles the logits (exact in bf16 and double)
    h2 = h * 2
    np.testing.assert_array_equal(oracle.lm_head_logits(bf16_bits(h2), bf16_bits(w)), 2 * w.double().numpy().T)


def test_selected_rows_equal_the_full_projection():
    h, w = _bf16((12, 64), 4), _bf16((33, 64), 5)
    full = oracle.lm_head_logits(bf16_bits(h), bf16_bits(w))
    rows = [11, 0, 5, 5]
    np.testing.assert_array_equal(oracle.lm_head_logits(bf16_bits(h), bf16_bits(w), rows=rows), full[rows])


def test_float64_logits_through_the_edit_rule():
    # Eq. 2 on float64 logits: argmax, c = max softmax probability, strict threshold
    h, w = _bf16((40, 128), 6, 0.5), _bf16((300, 128), 7, 0.5)
    logits = oracle.lm_head_logits(bf16_bits(h), bf16_bits(w))
    committed = np.arange(40, dtype=np.int32) % 300
    res = oracle.edit_decide(logits, committed, tau=0.0)
    p = torch.softmax(torch.from_numpy(logits), dim=1)
    np.testing.assert_array_equal(res["argmax"], p.argmax(dim=1).numpy())
    np.testing.assert_allclose(res["confidence"], p.max(dim=1).values.numpy(), rtol=1e-13)
    np.testing.assert_array_equal(res["edit_mask"], (res["argmax"] != committed).astype(np.uint8))
    # the entropy of the same logits through the full update
    den = oracle.denoise_update(logits, committed, [0, 40], 8, -1, 0.5, 0.0)
    ref_h = torch.distributions.Categorical(logits=torch.from_numpy(logits)).entropy().numpy()
    np.testing.assert_allclose(den["entropy"], ref_h, rtol=1e-12, atol=1e-12)
