"""Parity of the targeted refresh (mbe_refresh_plan, mbe_gather_rows, then the
KV write and attention on that layout; Sec. 4.3) and of the device-side
editing-pass loop (mbe_pass_loop_*, Sec. 4.1) with the oracle, through the C
ABI. Layouts and caches are compared bit-exactly; attention outputs with the
attention bar (1e-2 absolute vs the fp64 oracle)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_22663_gb300 import mbe
from paper_2607_22663_gb300.workloads import BIDIRECTIONAL, attention_problem, bf16_bits
from tests._gpu import ATTN_ATOL

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _plan_case(batch, max_blocks, B, seed, max_pages=7, p_change=0.4):
    g = torch.Generator().manual_seed(seed)
    W = torch.randint(0, max_blocks * B + 1, (batch,), generator=g, dtype=torch.int32)
    W[::5] = 0
    P = torch.randint(0, 5000, (batch,), generator=g, dtype=torch.int32)
    cu = torch.zeros(batch + 1, dtype=torch.int32)
    cu[1:] = torch.cumsum(W, 0)
    changed = (torch.rand(batch, max_blocks, generator=g) < p_change).to(torch.uint8)
    bt = torch.randint(-1, 10000, (batch, max_pages), generator=g, dtype=torch.int32)
    return changed, P, W, cu, bt


def _gpu_plan(changed, P, W, cu, bt, B, max_window, total_rows=None):
    total = int(cu[-1]) if total_rows is None else total_rows
    out = mbe.refresh_plan(changed.to(DEV), P.to(DEV), W.to(DEV), cu.to(DEV), bt.to(DEV), block_size=B,
                           max_window=max_window, total_rows=total)
    return {k: v.cpu().numpy() for k, v in out.items()}


@pytest.mark.parametrize("batch,max_blocks,B,max_pages", [(6, 3, 32, 5), (300, 8, 16, 9), (1, 1, 32, 1),
                                                          (2000, 4, 32, 300)])
def test_refresh_plan_matches_oracle(batch, max_blocks, B, max_pages):
    changed, P, W, cu, bt = _plan_case(batch, max_blocks, B, seed=batch + B, max_pages=max_pages)
    got = _gpu_plan(changed, P, W, cu, bt, B, max_blocks * B)
    ref = oracle.refresh_plan(changed.numpy(), P.numpy(), W.numpy(), cu.numpy(), bt.numpy(), B)
    for k in ref:
        np.testing.assert_array_equal(got[k], ref[k], err_msg=k)
    assert mbe.get_device_error() == (0, 0)


def test_refresh_plan_without_changes_and_empty_batch():
    changed, P, W, cu, bt = _plan_case(9, 2, 32, seed=5, p_change=0.0)
    got = _gpu_plan(changed, P, W, cu, bt, 32, 64)
    assert got["count"].tolist() == [0, 0] and (got["src_row"] == -1).all() and (got["block_table"] == -1).all()
    z = torch.zeros(0, dtype=torch.int32)
    got = _gpu_plan(torch.zeros((0, 2), dtype=torch.uint8), z, z, torch.zeros(1, dtype=torch.int32),
                    torch.zeros((0, 3), dtype=torch.int32), 32, 64, total_rows=4)
    assert got["count"].tolist() == [0, 0] and got["cu_window"].tolist() == [0] and (got["src_row"] == -1).all()


def test_refresh_plan_device_checks():
    changed, P, W, cu, bt = _plan_case(4, 2, 32, seed=6, p_change=1.0)
    W[1] = 60
    cu[1:] = torch.cumsum(W, 0)
    # window 60 above the declared max_window 40: that sequence is treated as unchanged and flagged
    got = _gpu_plan(changed, P, W, cu, bt, 32, 40)
    assert got["window_len"][2:4].tolist() == [0, 0]
    st, flags = mbe.get_device_error()
    assert flags & mbe.DEVERR_LENGTH
    # fewer rows than the refresh needs: the rows that fit are written, the rest flagged
    got = _gpu_plan(changed, P, W, cu, bt, 32, 64, total_rows=10)
    assert got["src_row"].tolist() == oracle.refresh_plan(changed.numpy(), P.numpy(), W.numpy(), cu.numpy(),
                                                          bt.numpy(), 32)["src_row"][:10].tolist()
    st, flags = mbe.get_device_error()
    assert flags & mbe.DEVERR_CAPACITY


@pytest.mark.parametrize("shape,dtype", [((37, 4, 128), torch.bfloat16), ((50,), torch.int32),
                                         ((13, 3), torch.uint8)])
def test_gather_rows(shape, dtype):
    g = torch.Generator().manual_seed(7)
    src = torch.randint(0, 100, shape, generator=g).to(dtype)
    idx = torch.randint(-1, shape[0], (70,), generator=g, dtype=torch.int32)
    got = mbe.gather_rows(src.to(DEV), idx.to(DEV)).cpu()
    ref = torch.zeros((70,) + shape[1:], dtype=dtype)
    ok = idx >= 0
    ref[ok] = src[idx[ok].long()]
    assert torch.equal(got, ref)
    assert mbe.get_device_error() == (0, 0)
    idx[3] = shape[0] + 5
    got = mbe.gather_rows(src.to(DEV), idx.to(DEV)).cpu()
    assert not got[3].any()
    st, flags = mbe.get_device_error()
    assert flags == mbe.DEVERR_LENGTH
    # a device row count: rows from it on keep what the output held
    fill = torch.full((70,) + shape[1:], 9, dtype=dtype, device=DEV)
    n = torch.tensor([41], dtype=torch.int32, device=DEV)
    idx[3] = 0
    got = mbe.gather_rows(src.to(DEV), idx.to(DEV), out=fill, rows_used=n).cpu()
    ref[3] = src[0]
    assert torch.equal(got[:41], ref[:41]) and (got[41:] == 9).all()
    n.fill_(-3)
    got = mbe.gather_rows(src.to(DEV), idx.to(DEV), out=fill, rows_used=n).cpu()
    assert torch.equal(got[:41], ref[:41]) and (got[41:] == 9).all()
    assert mbe.get_device_error() == (0, 0)


def test_gather_rows_multi():
    """One launch for several tensors sharing a row map equals one gather per
    tensor; rows that are not whole 16-byte chunks take the per-tensor path."""
    g = torch.Generator().manual_seed(11)
    R, n = 45, 70
    idx = torch.randint(-1, R, (n,), generator=g, dtype=torch.int32)
    sets = [[torch.randn(R, 4, 128, generator=g).to(torch.bfloat16), torch.randn(R, 2, 128, generator=g).to(torch.bfloat16),
             torch.randn(R, 2, 64, generator=g).to(torch.bfloat16)],
            [torch.randint(0, 9, (R,), generator=g, dtype=torch.int32), torch.randn(R, 2, 128, generator=g).to(torch.bfloat16)],
            [torch.randint(0, 255, (R, 3), generator=g).to(torch.uint8)]]
    for srcs in sets:
        d_srcs = [x.to(DEV) for x in srcs]
        outs = [torch.full((n,) + x.shape[1:], 7, dtype=x.dtype, device=DEV) for x in srcs]
        mbe.gather_rows_multi(list(zip(d_srcs, outs)), idx.to(DEV))
        for x, o in zip(srcs, outs):
            ref = torch.zeros((n,) + x.shape[1:], dtype=x.dtype)
            ok = idx >= 0
            ref[ok] = x[idx[ok].long()]
            assert torch.equal(o.cpu(), ref)
        assert mbe.get_device_error() == (0, 0)
        # a device row count leaves the rows from it on untouched; an index past the
        # source gives a zero row and the length flag
        bad = idx.clone()
        bad[2] = R + 3
        cnt = torch.tensor([33], dtype=torch.int32, device=DEV)
        outs2 = [torch.full_like(o, 5) for o in outs]
        mbe.gather_rows_multi(list(zip(d_srcs, outs2)), bad.to(DEV), rows_used=cnt)
        for o, o2 in zip(outs, outs2):
            got = o2.cpu()
            assert not got[2].any() and torch.equal(got[3:33], o.cpu()[3:33]) and (got[33:] == 5).all()
        st, flags = mbe.get_device_error()
        assert flags == mbe.DEVERR_LENGTH
    with pytest.raises(ValueError):
        mbe.gather_rows_multi([], idx.to(DEV))


def _refresh_problem(seed):
    B = 32
    prefix, window = [100, 0, 2000, 517, 64], [64, 96, 33, 128, 32]
    prob = attention_problem(prefix, window, [BIDIRECTIONAL] * 5, 8, 2, 128, B, 64, seed=seed)
    old = attention_problem(prefix, window, [BIDIRECTIONAL] * 5, 8, 2, 128, B, 64, seed=seed + 1)
    g = torch.Generator().manual_seed(seed)
    changed = (torch.rand(5, 4, generator=g) < 0.5).to(torch.uint8)
    changed[0, 1] = 1
    return prob, old, changed, B


def _oracle_refresh(prob, old, changed, B):
    kc0, vc0 = oracle.kv_window_write(bf16_bits(old.k_win), bf16_bits(old.v_win), bf16_bits(prob.k_cache),
                                      bf16_bits(prob.v_cache), prob.block_table.numpy(), prob.prefix_len.numpy(),
                                      prob.window_len.numpy(), prob.cu_window.numpy(), B)
    plan = oracle.refresh_plan(changed.numpy(), prob.prefix_len.numpy(), prob.window_len.numpy(),
                               prob.cu_window.numpy(), prob.block_table.numpy(), B)
    rows = plan["src_row"][:plan["count"][1]]
    q, kw, vw = bf16_bits(prob.q)[rows], bf16_bits(prob.k_win)[rows], bf16_bits(prob.v_win)[rows]
    kc, vc = oracle.kv_window_write(kw, vw, kc0, vc0, plan["block_table"], plan["prefix_len"], plan["window_len"],
                                    plan["cu_window"], B)
    out, _ = oracle.window_attention(q, kw, vw, kc, vc, plan["block_table"], plan["prefix_len"], plan["window_len"],
                                     plan["cu_window"], plan["mask_mode"], B, prob.page_size)
    return rows, out, kc, vc


def _refresh_max_prefix(prob):
    # the last block of a window starts at B * floor((W - 1) / B)
    B = prob.block_size
    return max(p + B * ((w - 1) // B) for p, w in zip(prob.prefix_host, prob.window_host) if w > 0)


def _gpu_refresh(prob, old, changed, B, stream=None, bufs=None, fused=False):
    """The refresh on the GPU, every step through the library: write the cache
    as decoding left it, plan, gather Q/K/V of the changed rows, write them,
    attend (fused: the gather and the write in one mbe_refresh_gather_write).
    With `bufs` nothing is allocated (graph capture)."""
    d = prob.to(DEV) if bufs is None else bufs["prob"]
    T = int(prob.cu_window[-1])
    E = prob.batch * changed.shape[1]
    if bufs is None:
        bufs = {"prob": d, "old_k": old.k_win.to(DEV), "old_v": old.v_win.to(DEV), "changed": changed.to(DEV),
                # NaN rows: only the refresh rows are gathered, and the rows after
                # them (read in the last key tile) must never reach the output
                "plan": None, "q": torch.full_like(d.q, float("nan")), "k": torch.full_like(d.k_win, float("nan")),
                "v": torch.full_like(d.k_win, float("nan")), "out": torch.zeros_like(d.q),
                "ws": torch.empty(mbe.window_attention_workspace_size(E, 8, 2, 128, B, _refresh_max_prefix(prob)),
                                  dtype=torch.uint8, device=DEV)}
    mw = max(prob.window_host)
    mbe.kv_window_write(bufs["old_k"], bufs["old_v"], d.k_cache, d.v_cache, d.block_table, d.prefix_len, d.window_len,
                        d.cu_window, block_size=B, max_window=mw, stream=stream)
    plan = mbe.refresh_plan(bufs["changed"], d.prefix_len, d.window_len, d.cu_window, d.block_table, block_size=B,
                            max_window=mw, total_rows=T, out=bufs["plan"], stream=stream)
    bufs["plan"] = plan
    # only the refresh rows are gathered (Q, K and V in one launch); the rest of the
    # buffers are never read
    if fused:
        mbe.refresh_gather_write(d.q, d.k_win, d.v_win, plan, d.k_cache, d.v_cache,
                                 out=(bufs["q"], bufs["k"], bufs["v"]), stream=stream)
    else:
        mbe.gather_rows_multi([(d.q, bufs["q"]), (d.k_win, bufs["k"]), (d.v_win, bufs["v"])], plan["src_row"],
                              rows_used=plan["count"][1:], stream=stream)
        mbe.kv_window_write(bufs["k"], bufs["v"], d.k_cache, d.v_cache, plan["block_table"], plan["prefix_len"],
                            plan["window_len"], plan["cu_window"], block_size=B, max_window=B, stream=stream)
    mbe.window_attention(bufs["q"], bufs["k"], bufs["v"], d.k_cache, d.v_cache, plan["block_table"],
                         plan["prefix_len"], plan["window_len"], plan["cu_window"], plan["mask_mode"], block_size=B,
                         max_window=B, max_prefix=_refresh_max_prefix(prob), out=bufs["out"], workspace=bufs["ws"],
                         stream=stream)
    return bufs


def test_refresh_attention_and_cache_match_oracle():
    prob, old, changed, B = _refresh_problem(seed=21)
    bufs = _gpu_refresh(prob, old, changed, B)
    torch.cuda.synchronize()
    assert mbe.get_device_error() == (0, 0)
    rows, out_ref, kc_ref, vc_ref = _oracle_refresh(prob, old, changed, B)
    n = len(rows)
    assert bufs["plan"]["count"].cpu().tolist()[1] == n
    got = bufs["out"][:n].float().cpu().numpy()
    assert np.abs(got - out_ref).max() <= ATTN_ATOL
    np.testing.assert_array_equal(bf16_bits(bufs["prob"].k_cache.cpu()), kc_ref)
    np.testing.assert_array_equal(bf16_bits(bufs["prob"].v_cache.cpu()), vc_ref)
    # rows past the refresh rows are left as they were
    assert bufs["q"][n:].isnan().all() and bufs["v"][n:].isnan().all()


def test_refresh_gather_write_matches_oracle_and_separate_calls():
    """mbe_refresh_gather_write (gather + cache write in one launch) gives the
    same compact rows, cache and attention output as mbe_gather_rows_multi
    followed by mbe_kv_window_write, and matches the oracle."""
    prob, old, changed, B = _refresh_problem(seed=23)
    sep = _gpu_refresh(prob, old, changed, B)
    fus = _gpu_refresh(prob, old, changed, B, fused=True)
    torch.cuda.synchronize()
    assert mbe.get_device_error() == (0, 0)
    rows, out_ref, kc_ref, vc_ref = _oracle_refresh(prob, old, changed, B)
    n = len(rows)
    for key in ("q", "k", "v", "out"):
        assert torch.equal(fus[key][:n], sep[key][:n]), key
    assert fus["q"][n:].isnan().all() and fus["k"][n:].isnan().all() and fus["v"][n:].isnan().all()
    for cache in ("k_cache", "v_cache"):
        assert torch.equal(getattr(fus["prob"], cache), getattr(sep["prob"], cache))
    np.testing.assert_array_equal(bf16_bits(fus["prob"].k_cache.cpu()), kc_ref)
    np.testing.assert_array_equal(bf16_bits(fus["prob"].v_cache.cpu()), vc_ref)
    assert np.abs(fus["out"][:n].float().cpu().numpy() - out_ref).max() <= ATTN_ATOL


def test_refresh_gather_write_bad_page_flags_and_skips_like_separate_calls():
    """A changed block whose page id lies outside the cache: the fused call sets
    MBE_DEVERR_PAGE and skips those cache slots, as the KV write does, and both
    paths leave identical compact rows and caches."""
    prob, old, changed, B = _refresh_problem(seed=24)
    d = prob.to(DEV)
    bt = d.block_table.clone()
    bt[0, (prob.prefix_host[0] + B) // prob.page_size] = d.k_cache.shape[0] + 7   # block 1 of sequence 0
    changed[0, 1] = 1
    plan = mbe.refresh_plan(changed.to(DEV), d.prefix_len, d.window_len, d.cu_window, bt, block_size=B,
                            max_window=max(prob.window_host), total_rows=int(prob.cu_window[-1]))
    res = []
    for fused in (True, False):
        outs = tuple(torch.zeros_like(x) for x in (d.q, d.k_win, d.v_win))
        kc, vc = d.k_cache.clone(), d.v_cache.clone()
        if fused:
            mbe.refresh_gather_write(d.q, d.k_win, d.v_win, plan, kc, vc, out=outs)
        else:
            mbe.gather_rows_multi(list(zip((d.q, d.k_win, d.v_win), outs)), plan["src_row"],
                                  rows_used=plan["count"][1:])
            mbe.kv_window_write(outs[1], outs[2], kc, vc, plan["block_table"], plan["prefix_len"], plan["window_len"],
                                plan["cu_window"], block_size=B, max_window=B)
        st, flags = mbe.get_device_error()
        assert flags == mbe.DEVERR_PAGE, flags
        res.append(outs + (kc, vc))
    for a, b in zip(*res):
        assert torch.equal(a, b)
    assert not torch.equal(res[0][3], d.k_cache)   # the other changed blocks were written


def test_refresh_gather_write_row_outside_every_entry_writes_no_slot():
    """A row count larger than the layout (and a valid source row for the extra
    row): that row is compacted but writes no cache slot, and the call sets
    MBE_DEVERR_LENGTH; the caches equal those of the consistent call."""
    prob, old, changed, B = _refresh_problem(seed=25)
    d = prob.to(DEV)
    plan = mbe.refresh_plan(changed.to(DEV), d.prefix_len, d.window_len, d.cu_window, d.block_table, block_size=B,
                            max_window=max(prob.window_host), total_rows=int(prob.cu_window[-1]))
    n = int(plan["count"][1])
    assert n < plan["src_row"].numel()
    res = []
    for extra in (False, True):
        p2 = {k: v.clone() for k, v in plan.items()}
        if extra:
            p2["src_row"][n] = 0
            p2["count"][1] = n + 1
        outs = tuple(torch.zeros_like(x) for x in (d.q, d.k_win, d.v_win))
        kc, vc = d.k_cache.clone(), d.v_cache.clone()
        mbe.refresh_gather_write(d.q, d.k_win, d.v_win, p2, kc, vc, out=outs)
        st, flags = mbe.get_device_error()
        assert flags == (mbe.DEVERR_LENGTH if extra else 0), flags
        res.append((outs, kc, vc))
    assert torch.equal(res[0][1], res[1][1]) and torch.equal(res[0][2], res[1][2])
    assert torch.equal(res[1][0][0][n], d.q[0])   # the extra row itself is compacted


def test_refresh_in_a_captured_graph_matches_eager():
    prob, old, changed, B = _refresh_problem(seed=22)
    eager = _gpu_refresh(prob, old, changed, B)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    bufs = _gpu_refresh(prob, old, changed, B)     # allocates the buffers
    bufs["out"].zero_()
    torch.cuda.synchronize()
    passes = torch.zeros(1, dtype=torch.int32, device=DEV)
    no_change = torch.zeros(prob.batch, dtype=torch.int32, device=DEV)
    loop = mbe.PassLoop(3, passes, s)
    try:
        with torch.cuda.stream(s):
            _gpu_refresh(prob, old, changed, B, stream=s, bufs=bufs)
        loop.until_stable(no_change)
        loop.end()
        loop.launch()
        s.synchronize()
    finally:
        loop.close()
    assert passes.item() == 1
    assert torch.equal(bufs["out"], eager["out"])
    assert torch.equal(bufs["prob"].k_cache, eager["prob"].k_cache)
    assert mbe.get_device_error() == (0, 0)


def _loop_problem(lengths, vocab, seed, mask_frac):
    g = torch.Generator().manual_seed(seed)
    R = sum(lengths)
    logits = torch.randn(R, vocab, generator=g) * 2.0
    hot = torch.randint(0, vocab - 1, (R,), generator=g)
    logits[torch.arange(R), hot] += 7.0 * torch.rand(R, generator=g)
    mask_id = vocab - 1
    logits[:, mask_id] = -20.0
    tokens = torch.randint(0, vocab - 1, (R,), generator=g, dtype=torch.int64).to(torch.int32)
    tokens[torch.rand(R, generator=g) < mask_frac] = mask_id
    cu = torch.tensor([0] + list(np.cumsum(lengths)), dtype=torch.int32)
    return logits, tokens, cu, mask_id


def _oracle_passes(logits, tokens, cu, B, mask_id, om, oe, max_passes):
    tok = tokens.numpy().copy()
    passes = 0
    while True:
        r = oracle.denoise_update(logits.numpy(), tok, cu.numpy(), B, mask_id, om, oe)
        passes += 1
        tok = r["new_tokens"]
        if not r["seq_changes"].any() or passes >= max_passes:
            return tok, passes


@pytest.mark.parametrize("mask_frac,om,oe,max_passes", [(0.0, 0.9, 0.3, 5), (0.5, 0.8, 0.3, 5),
                                                        (0.5, 0.95, 0.3, 40), (0.5, 0.95, 0.3, 1), (0.0, 0.9, 1.5, 5)])
def test_pass_loop_stops_like_the_oracle(mask_frac, om, oe, max_passes):
    B = 16
    lengths = [48, 16, 0, 33]
    logits, tokens, cu, mask_id = _loop_problem(lengths, 500, seed=31, mask_frac=mask_frac)
    tok_ref, passes_ref = _oracle_passes(logits, tokens, cu, B, mask_id, om, oe, max_passes)
    R = tokens.shape[0]
    d_logits, d_tok, d_cu = logits.to(DEV), tokens.to(DEV), cu.to(DEV)
    ident = torch.arange(R, dtype=torch.int32, device=DEV)
    out = mbe.denoise_update(d_logits, d_tok, d_cu, block_size=B, mask_id=mask_id, omega_mask=om, omega_edit=oe,
                             max_blocks=3)
    torch.cuda.synchronize()
    passes = torch.zeros(1, dtype=torch.int32, device=DEV)
    s = torch.cuda.Stream()
    loop = mbe.PassLoop(max_passes, passes, s)
    try:
        mbe.denoise_update(d_logits, d_tok, d_cu, block_size=B, mask_id=mask_id, omega_mask=om, omega_edit=oe,
                           out=out, stream=s)
        # the pass's new tokens become the current tokens of the next pass
        mbe.gather_rows(out["new_tokens"], ident, out=d_tok, stream=s)
        loop.until_stable(out["seq_changes"])
        loop.end()
        for _ in range(2):     # a second launch starts again from the reset pass count
            d_tok.copy_(tokens.to(DEV))
            torch.cuda.synchronize()
            loop.launch()
            s.synchronize()
            assert passes.item() == passes_ref
            np.testing.assert_array_equal(d_tok.cpu().numpy(), tok_ref)
    finally:
        loop.close()
    assert mbe.get_device_error() == (0, 0)


def test_pass_loop_rejects_a_body_without_condition_and_bad_arguments():
    s = torch.cuda.Stream()
    passes = torch.zeros(1, dtype=torch.int32, device=DEV)
    loop = mbe.PassLoop(2, passes, s)
    with pytest.raises(mbe.MbeError):
        loop.end()          # no until_stable: the graph is not instantiated
    with pytest.raises(mbe.MbeError):
        loop.launch()
    loop.close()
    with pytest.raises(mbe.MbeError):
        mbe.PassLoop(0, passes, s)
    with pytest.raises(ValueError):
        mbe.PassLoop(2, passes, torch.cuda.default_stream())
    torch.cuda.synchronize()
