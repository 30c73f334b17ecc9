"""Pins of the full Eq. 2 update (Gamma_t, forced unmasking, Delta_t), of the
per-row entropy and of the tail-entropy block selection (Eqs. 6-7). CPU only."""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300.workloads import bf16_bits, edit_problem

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_golden_closed_forms():
    spec = json.load(open(os.path.join(GOLDEN, "denoise_closed_forms.json")))
    logits = np.array(spec["logits"], dtype=np.float32)
    for case in spec["cases"]:
        res = oracle.denoise_update(logits, spec["tokens"], [0, 4], spec["block_size"], spec["mask_id"],
                                    case["omega_mask"], case["omega_edit"])
        assert res["new_tokens"].tolist() == case["new_tokens"], case["name"]
        assert res["kind"].tolist() == case["kind"], case["name"]
        assert res["block_changed"][0].tolist() == case["block_changed"], case["name"]
        assert res["seq_changes"][0] == case["seq_changes"], case["name"]
        expected_h = [eval(e, {"math": math}) for e in spec["entropy_expr"]]
        np.testing.assert_allclose(res["entropy"], expected_h, rtol=0, atol=1e-6)


@pytest.mark.parametrize("V", [1, 2, 7, 1000, 32768])
def test_uniform_rows_have_ppl_equal_to_vocabulary(V):
    """Sec. 3: a uniform distribution over n tokens has PPL = exp(H) = n."""
    logits = np.full((3, V), 0.75, dtype=np.float32)
    res = oracle.denoise_update(logits, [1, 1, 1], [0, 3], 4, -1, 0.5, 0.0)
    np.testing.assert_allclose(np.exp(res["entropy"]), V, rtol=1e-10)  # n terms summed in double


def test_entropy_matches_torch_categorical():
    prob = edit_problem(50, 3000, torch.bfloat16, seed=5, peak_frac=0.5, peak_lo=1.0, peak_hi=9.0)
    res = oracle.denoise_update(bf16_bits(prob.logits), prob.committed.numpy(), [0, 50], 32, -1, 0.5, 0.0,
                                is_bf16=True)
    ref = torch.distributions.Categorical(logits=prob.logits.double()).entropy().numpy()
    np.testing.assert_allclose(res["entropy"], ref, rtol=1e-11, atol=1e-12)


def _random_step(rows, vocab, seed, mask_frac, mask_id):
    g = torch.Generator().manual_seed(seed)
    logits = (torch.randn(rows, vocab, generator=g) * 2.0)
    hot = torch.randint(0, vocab, (rows,), generator=g)
    logits[torch.arange(rows), hot] += 6.0 * torch.rand(rows, generator=g)
    tokens = torch.randint(0, vocab, (rows,), generator=g, dtype=torch.int64).to(torch.int32)
    masked = torch.rand(rows, generator=g) < mask_frac
    tokens[masked] = mask_id
    return logits.numpy().astype(np.float32), tokens.numpy()


def test_rules_against_definitions_on_random_rows():
    mask_id, B = 511, 16
    cu = np.array([0, 40, 40, 77, 120], dtype=np.int32)
    logits, tokens = _random_step(120, 512, 3, 0.6, mask_id)
    editable = (np.arange(120) % 5 != 0).astype(np.uint8)
    res = oracle.denoise_update(logits, tokens, cu, B, mask_id, 0.5, 0.1, editable=editable)
    ref = oracle.edit_decide(logits, tokens, tau=0.1, editable=editable)
    p = torch.softmax(torch.from_numpy(logits).double(), dim=1)
    am = p.argmax(dim=1).numpy()
    c = p.max(dim=1).values.numpy()
    np.testing.assert_array_equal(res["argmax"], am)
    np.testing.assert_allclose(res["confidence"], c, rtol=1e-13)
    for s in range(4):
        for b0 in range(cu[s], cu[s + 1], B):
            rows = np.arange(b0, min(b0 + B, cu[s + 1]))
            masked = rows[tokens[rows] == mask_id]
            gamma = masked[c[masked].astype(np.float32) > np.float32(0.5)]
            for r in rows:
                if tokens[r] != mask_id:   # Delta_t: same rule as the edit decision
                    assert res["new_tokens"][r] == ref["new_tokens"][r]
                    assert res["kind"][r] == (3 if ref["edit_mask"][r] else 0)
            if len(masked) and not len(gamma):
                forced = masked[np.argmax(c[masked].astype(np.float32))]
                assert res["kind"][forced] == 2 and res["new_tokens"][forced] == am[forced]
                assert (res["kind"][masked] != 1).all() and (res["kind"][masked] == 2).sum() == 1
            else:
                assert set(np.nonzero(res["kind"][masked] == 1)[0]) == set(np.nonzero(np.isin(masked, gamma))[0])
                assert (res["kind"][masked] != 2).all()
            changed = (res["new_tokens"][rows] != tokens[rows]).any()
            assert res["block_changed"][s, (b0 - cu[s]) // B] == changed
        assert res["seq_changes"][s] == (res["new_tokens"][cu[s]:cu[s + 1]] != tokens[cu[s]:cu[s + 1]]).sum()


def test_a_block_resolves_within_block_size_steps():
    """Sec. 2.3: forced unmasking guarantees that a fully masked block resolves
    within at most B steps, whatever the thresholds."""
    mask_id, B = 63, 16
    tokens = np.full(B, mask_id, dtype=np.int32)
    for step in range(B):
        logits, _ = _random_step(B, 64, 100 + step, 0.0, mask_id)
        logits[:, mask_id] = -30.0          # the model does not predict [MASK]
        res = oracle.denoise_update(logits, tokens, [0, B], B, mask_id, 0.999, 0.999)
        assert res["seq_changes"][0] >= 1 or (tokens != mask_id).all()
        tokens = res["new_tokens"]
        if (tokens != mask_id).all():
            break
    assert (tokens != mask_id).all() and step < B


def test_tail_entropy_hand_example():
    """Eq. 6 with B = 32, rho = 1/4: the mean of the 8 largest entropies."""
    B = 32
    e = np.zeros((1, 3, B), dtype=np.float32)
    e[0, 0] = np.arange(B, dtype=np.float32) / 32     # top 8: 24..31 -> mean 27.5/32
    e[0, 1] = 0.85                                     # flat block: 0.85
    e[0, 2] = 0.0
    e[0, 2, 5] = 6.0                                   # one spike: 6/8 = 0.75
    res = oracle.tail_entropy_select(e, [3], 0.25, 4)
    np.testing.assert_allclose(res["scores"][0], [27.5 / 32, 0.85, 0.75], rtol=1e-6)
    assert res["best_slot"][0] == 0 and res["window_blocks"][0] == 4   # j* = j-3: W_j spans 4 blocks
    # K_max = 3 leaves the last two blocks as candidates; a single history block -> only it
    res = oracle.tail_entropy_select(e, [3], 0.25, 3)
    assert res["best_slot"][0] == 1 and np.isnan(res["scores"][0, 0])
    res = oracle.tail_entropy_select(e, [1], 0.25, 4)
    assert res["best_slot"][0] == 2 and res["window_blocks"][0] == 2
    res = oracle.tail_entropy_select(e, [0], 0.25, 4)     # j = 0: no window (Eq. 5 needs j > 0)
    assert res["best_slot"][0] == -1 and res["window_blocks"][0] == 1


def test_tail_entropy_brute_force():
    g = np.random.default_rng(7)
    S, H, B = 20, 5, 24
    e = g.gamma(2.0, 0.5, size=(S, H, B)).astype(np.float32)
    nv = g.integers(0, H + 1, size=S).astype(np.int32)
    for rho in (0.1, 0.25, 1.0):
        for k_max in (2, 4, 6):
            res = oracle.tail_entropy_select(e, nv, rho, k_max)
            top = math.ceil(rho * B)
            for s in range(S):
                ncand = min(nv[s], k_max - 1)
                cands = list(range(H - ncand, H))
                sc = {i: np.sort(e[s, i].astype(np.float64))[::-1][:top].mean() for i in cands}
                for i in cands:
                    assert abs(res["scores"][s, i] - sc[i]) < 1e-12
                if cands:
                    best = max(cands, key=lambda i: (np.float32(sc[i]), -i))
                    assert res["best_slot"][s] == best
                else:
                    assert res["best_slot"][s] == -1


def test_forced_unmask_tie_takes_lowest_row():
    logits = np.tile(np.array([[0.0, 1.0, 0.0]], dtype=np.float32), (4, 1))
    res = oracle.denoise_update(logits, [7, 7, 7, 7], [0, 4], 4, 7, 0.9, 0.0)
    assert res["kind"].tolist() == [2, 0, 0, 0]
    assert res["new_tokens"].tolist() == [1, 7, 7, 7]


@pytest.mark.parametrize("bad", ["nan", "all_neginf"])
def test_block_whose_masked_rows_lack_a_softmax_unmasks_nothing(bad):
    """Forced unmasking (Sec. 2.3) picks the most confident masked row of a
    block; a row without a softmax has no confidence, so it is never picked,
    and a block whose masked rows all lack one unmasks none. Rows of the other
    blocks are decided as without them."""
    mask_id, B = 63, 8
    logits, tokens = _random_step(24, 64, 11, 0.0, mask_id)
    logits[:, mask_id] = -30.0                 # no row predicts [MASK]
    masked = [9, 12, 14]                       # block 1 (rows 8..15): only these rows are masked
    tokens[masked] = mask_id
    for r in masked:
        if bad == "nan":
            logits[r, 5] = np.nan
        else:
            logits[r, :] = -np.inf
    tokens[20] = mask_id                       # block 2: one masked row with a softmax
    res = oracle.denoise_update(logits, tokens, [0, 24], B, mask_id, 2.0, 2.0)
    assert res["undecidable"]
    for r in masked:
        assert res["kind"][r] == 0 and res["new_tokens"][r] == mask_id
        assert res["argmax"][r] == -1 and np.isnan(res["confidence"][r]) and np.isnan(res["entropy"][r])
    assert res["block_changed"][0, 1] == 0
    assert res["kind"][20] == 2                # forced in its own block (omega_mask 2 admits nothing)
    others = np.array([r for r in range(24) if r not in masked])
    np.testing.assert_array_equal(res["argmax"][others], np.argmax(logits[others], axis=1))


def test_forced_unmask_skips_rows_without_softmax():
    """A block with one masked row that has a softmax and others that do not
    force-unmasks that row, whatever the others' logits."""
    mask_id, B = 63, 8
    logits, tokens = _random_step(8, 64, 12, 0.0, mask_id)
    logits[:, mask_id] = -30.0
    tokens[[1, 2, 6]] = mask_id
    logits[1, :] = -np.inf
    logits[6, 0] = np.inf
    res = oracle.denoise_update(logits, tokens, [0, 8], B, mask_id, 2.0, 2.0)
    assert res["kind"].tolist() == [0, 0, 2, 0, 0, 0, 0, 0]
    assert res["new_tokens"][2] == np.argmax(logits[2])


def test_entropy_with_neginf_logits_equals_reduced_row():
    """-inf logits are tokens of probability 0: the entropy equals that of the
    row without them (torch's categorical entropy of the finite entries)."""
    logits, tokens = _random_step(6, 200, 13, 0.0, -1)
    hidden = np.random.default_rng(1).random(logits.shape) < 0.5
    logits[hidden] = -np.inf
    res = oracle.denoise_update(logits, tokens, [0, 6], 8, -1, 0.5, 0.0)
    assert not res["undecidable"]
    for r in range(6):
        keep = torch.from_numpy(logits[r, ~hidden[r]]).double()
        ref = torch.distributions.Categorical(logits=keep).entropy().item()
        np.testing.assert_allclose(res["entropy"][r], ref, rtol=1e-12)
