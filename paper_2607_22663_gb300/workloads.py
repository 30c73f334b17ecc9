"""Seeded synthetic inputs shaped like MBE block-diffusion decoding.

This module only draws random tensors and lays them out; it contains none of
the hot path's arithmetic (no attention, no softmax, no edit rule). Both the
CUDA path and the CPU oracle receive the same tensors from here.

The shapes follow the five workloads the library is measured on:

* ``tiny``      one sequence, block 32, prefix 64, bidirectional 2-block window,
                4/1 heads, head_dim 64, page 32; fp32 logits [64 x 1024]
                N(0, sd 2) with a +8 peak on half the rows; tau 0.9; seed 0.
* ``batch8``    8 sequences, prefix 1024, window 64, 16/4 heads, head_dim 128,
                page 32 with a shuffled page table; bf16 logits [512 x 32768],
                peaks U(2,10) on 60% of rows; tau 0.9; seed 2.
* ``varlen64``  64 sequences, window k~U{1..4} blocks of 32, prefix
                U[256,8192] rounded down to 32, half block-causal, half
                bidirectional (shuffled); bf16 logits [sum(W) x 65536] with
                peaks U(2,10) on 60% of rows; tau~U(0.7,0.95) per sequence; seed 3.
* ``long32k``   4 sequences, prefix 32768, windows 64/128/256 (three calls),
                32/8 heads, page 64 with a random page permutation; KV write of
                each window; seed 4.
* ``serving128`` 128 sequences, prefix U[512,16384] (not rounded), window 64,
                32/8 heads, page 32 (not stated by the workload; the size the
                other paged workloads use), 24 layers with independent Q/K/V and
                caches; bf16 logits [8192 x 131072] N(0, sd 2) with peaks
                U(0,12) on every row, committed = the row argmax on 80% of
                rows; tau 0.9; seed 5.

Q/K/V are N(0,1) rounded to bf16. "N(0,2)" is read as standard deviation 2.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List, Optional

import torch

BLOCK_CAUSAL = 0
BIDIRECTIONAL = 1


@dataclass
class AttnProblem:
    """One attention call: window Q/K/V plus a paged KV cache and metadata."""
    q: torch.Tensor            # bf16 [T, Hq, D]
    k_win: torch.Tensor        # bf16 [T, Hkv, D]
    v_win: torch.Tensor        # bf16 [T, Hkv, D]
    k_cache: torch.Tensor      # bf16 [num_pages, Hkv, page_size, D]
    v_cache: torch.Tensor      # bf16 [num_pages, Hkv, page_size, D]
    block_table: torch.Tensor  # int32 [batch, max_pages]
    prefix_len: torch.Tensor   # int32 [batch]
    window_len: torch.Tensor   # int32 [batch]
    cu_window: torch.Tensor    # int32 [batch + 1]
    mask_mode: torch.Tensor    # uint8 [batch]
    block_size: int
    page_size: int
    prefix_host: List[int] = field(default_factory=list)
    window_host: List[int] = field(default_factory=list)
    mode_host: List[int] = field(default_factory=list)

    @property
    def batch(self):
        return len(self.prefix_host)

    @property
    def num_q_heads(self):
        return self.q.shape[1]

    @property
    def num_kv_heads(self):
        return self.k_win.shape[1]

    @property
    def head_dim(self):
        return self.q.shape[2]

    @property
    def num_pages(self):
        return self.k_cache.shape[0]

    @property
    def total_tokens(self):
        return self.q.shape[0]

    @property
    def max_window(self):
        return max(self.window_host) if self.window_host else 0

    @property
    def max_prefix(self):
        return max(self.prefix_host) if self.prefix_host else 0

    def to(self, device):
        kw = {k: (v.to(device) if isinstance(v, torch.Tensor) else v) for k, v in self.__dict__.items()}
        return AttnProblem(**kw)


@dataclass
class EditProblem:
    """One edit-decide call over the logits of a pass."""
    logits: torch.Tensor        # fp32 or bf16 [R, V]
    committed: torch.Tensor     # int32 [R]
    tau: float
    tau_per_row: Optional[torch.Tensor] = None   # fp32 [R]
    editable: Optional[torch.Tensor] = None      # uint8 [R]

    def to(self, device):
        kw = {k: (v.to(device) if isinstance(v, torch.Tensor) else v) for k, v in self.__dict__.items()}
        return EditProblem(**kw)


def _gen(seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return g


def _randn_bf16(shape, g, device, chunk_elems=1 << 28):
    """N(0,1) rounded to bf16, generated in chunks to bound temporary memory."""
    out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    flat = out.view(-1)
    n = flat.numel()
    for s in range(0, n, chunk_elems):
        e = min(n, s + chunk_elems)
        flat[s:e] = torch.randn(e - s, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
    return out


def attention_problem(prefix, window, modes, num_q_heads, num_kv_heads, head_dim, block_size, page_size, seed,
                      device="cpu", shuffle_pages=True, spare_pages=0, reserve_tokens=None, q_scale=1.0,
                      g=None) -> AttnProblem:
    """Random problem with the given per-sequence prefix/window lengths and modes.

    Each sequence owns ceil((P + reserve)/page_size) pages (reserve defaults to
    its window length so the window can be written back); page ids are a random
    permutation when shuffle_pages. Unused table entries hold -1.
    """
    batch = len(prefix)
    assert len(window) == batch and len(modes) == batch
    g = g or _gen(seed, device)
    reserve = window if reserve_tokens is None else reserve_tokens
    pages_per = [(p + r + page_size - 1) // page_size for p, r in zip(prefix, reserve)]
    max_pages = max(1, max(pages_per) if pages_per else 1)
    num_pages = sum(pages_per) + spare_pages
    num_pages = max(num_pages, 1)
    if shuffle_pages:
        perm = torch.randperm(num_pages, generator=g, device=device).to(torch.int32)
    else:
        perm = torch.arange(num_pages, device=device, dtype=torch.int32)
    bt = torch.full((batch, max_pages), -1, dtype=torch.int32, device=device)
    off = 0
    for s, n in enumerate(pages_per):
        bt[s, :n] = perm[off:off + n]
        off += n
    T = sum(window)
    q = _randn_bf16((T, num_q_heads, head_dim), g, device)
    if q_scale != 1.0:
        q = (q.float() * q_scale).to(torch.bfloat16)
    k_win = _randn_bf16((T, num_kv_heads, head_dim), g, device)
    v_win = _randn_bf16((T, num_kv_heads, head_dim), g, device)
    k_cache = _randn_bf16((num_pages, num_kv_heads, page_size, head_dim), g, device)
    v_cache = _randn_bf16((num_pages, num_kv_heads, page_size, head_dim), g, device)
    cu = [0]
    for w in window:
        cu.append(cu[-1] + w)
    t32 = lambda x: torch.tensor(x, dtype=torch.int32, device=device)
    return AttnProblem(q=q, k_win=k_win, v_win=v_win, k_cache=k_cache, v_cache=v_cache, block_table=bt,
                       prefix_len=t32(prefix), window_len=t32(window), cu_window=t32(cu),
                       mask_mode=torch.tensor(modes, dtype=torch.uint8, device=device), block_size=block_size,
                       page_size=page_size, prefix_host=list(prefix), window_host=list(window),
                       mode_host=list(modes))


def edit_problem(rows, vocab, dtype, seed, device="cpu", sd=2.0, peak_frac=0.5, peak_lo=8.0, peak_hi=8.0, tau=0.9,
                 tau_per_row=None, committed_argmax_frac=0.0, g=None) -> EditProblem:
    """Logits N(0, sd) with a planted peak U(peak_lo, peak_hi) at a random token on
    a random `peak_frac` of rows; committed tokens uniform over the vocabulary,
    except a random `committed_argmax_frac` of rows whose committed token is the
    row's largest logit (torch.argmax of the generated row: an input recipe)."""
    g = g or _gen(seed, device)
    logits = torch.randn(rows, vocab, generator=g, device=device, dtype=torch.float32)
    logits.mul_(sd)
    n_peak = int(round(peak_frac * rows))
    prow = torch.randperm(rows, generator=g, device=device)[:n_peak]
    ptok = torch.randint(0, vocab, (n_peak,), generator=g, device=device)
    height = peak_lo + (peak_hi - peak_lo) * torch.rand(n_peak, generator=g, device=device)
    logits[prow, ptok] += height
    logits = logits.to(dtype)
    committed = torch.randint(0, vocab, (rows,), generator=g, device=device, dtype=torch.int64).to(torch.int32)
    if committed_argmax_frac > 0:
        n_am = int(round(committed_argmax_frac * rows))
        arow = torch.randperm(rows, generator=g, device=device)[:n_am]
        committed[arow] = torch.argmax(logits[arow].float(), dim=1).to(torch.int32)
    return EditProblem(logits=logits, committed=committed, tau=tau, tau_per_row=tau_per_row)


def editable_historical(window_host, block_size, device="cpu"):
    """Rows of the window's historical part [j* B, j B): every row except the
    last block of each window (Sec. 4.1: T2T edits only the historical part)."""
    out = []
    for w in window_host:
        last = max(0, w - block_size)
        out += [1] * last + [0] * (w - last)
    return torch.tensor(out, dtype=torch.uint8, device=device)


# ---------------------------------------------------------------- named workloads
def tiny(device="cpu"):
    g = _gen(0, device)
    attn = attention_problem([64], [64], [BIDIRECTIONAL], 4, 1, 64, 32, 32, 0, device, g=g)
    edit = edit_problem(64, 1024, torch.float32, 0, device, sd=2.0, peak_frac=0.5, peak_lo=8.0, peak_hi=8.0,
                        tau=0.9, g=g)
    return {"name": "tiny", "attn": [attn], "edit": edit, "layers": 1}


def batch8(device="cpu"):
    g = _gen(2, device)
    attn = attention_problem([1024] * 8, [64] * 8, [BIDIRECTIONAL] * 8, 16, 4, 128, 32, 32, 2, device, g=g)
    edit = edit_problem(512, 32768, torch.bfloat16, 2, device, sd=2.0, peak_frac=0.6, peak_lo=2.0, peak_hi=10.0,
                        tau=0.9, g=g)
    return {"name": "batch8", "attn": [attn], "edit": edit, "layers": 1}


def varlen64(device="cpu", vocab=65536):
    g = _gen(3, "cpu")
    k = torch.randint(1, 5, (64,), generator=g).tolist()
    window = [32 * x for x in k]
    prefix = [(int(x) // 32) * 32 for x in torch.randint(256, 8193, (64,), generator=g).tolist()]
    modes = [BLOCK_CAUSAL] * 32 + [BIDIRECTIONAL] * 32
    perm = torch.randperm(64, generator=g).tolist()
    modes = [modes[i] for i in perm]
    taus = (0.7 + 0.25 * torch.rand(64, generator=g)).tolist()
    gd = _gen(3, device)
    attn = attention_problem(prefix, window, modes, 16, 4, 128, 32, 32, 3, device, g=gd)
    rows = sum(window)
    tau_rows = torch.tensor([t for t, w in zip(taus, window) for _ in range(w)], dtype=torch.float32, device=device)
    edit = edit_problem(rows, vocab, torch.bfloat16, 3, device, sd=2.0, peak_frac=0.6, peak_lo=2.0, peak_hi=10.0,
                        tau=0.9, tau_per_row=tau_rows, g=gd)
    return {"name": "varlen64", "attn": [attn], "edit": edit, "layers": 1}


def long32k(device="cpu", windows=(64, 128, 256)):
    """One cache (prefix 32768, reserving room for the largest window) and one
    window per call size; each call is followed by the window's KV write."""
    gd = _gen(4, device)
    calls = []
    wmax = max(windows)
    base = attention_problem([32768] * 4, [wmax] * 4, [BIDIRECTIONAL] * 4, 32, 8, 128, 32, 64, 4, device, g=gd)
    for w in windows:
        T = 4 * w
        cu = torch.arange(0, T + 1, w, dtype=torch.int32, device=device)
        calls.append(AttnProblem(q=_randn_bf16((T, 32, 128), gd, device), k_win=_randn_bf16((T, 8, 128), gd, device),
                                 v_win=_randn_bf16((T, 8, 128), gd, device), k_cache=base.k_cache,
                                 v_cache=base.v_cache, block_table=base.block_table, prefix_len=base.prefix_len,
                                 window_len=torch.full((4,), w, dtype=torch.int32, device=device), cu_window=cu,
                                 mask_mode=base.mask_mode, block_size=32, page_size=64, prefix_host=[32768] * 4,
                                 window_host=[w] * 4, mode_host=[BIDIRECTIONAL] * 4))
    return {"name": "long32k", "attn": calls, "edit": None, "layers": 1}


def serving128(device="cpu", layers=24, vocab=131072, batch=128, page_size=32):
    g = _gen(5, "cpu")
    prefix = torch.randint(512, 16385, (batch,), generator=g).tolist()
    window = [64] * batch
    gd = _gen(5, device)
    first = attention_problem(prefix, window, [BIDIRECTIONAL] * batch, 32, 8, 128, 32, page_size, 5, device, g=gd)
    attn = [first]
    for _ in range(1, layers):
        attn.append(AttnProblem(q=_randn_bf16(first.q.shape, gd, device), k_win=_randn_bf16(first.k_win.shape, gd, device),
                                v_win=_randn_bf16(first.v_win.shape, gd, device),
                                k_cache=_randn_bf16(first.k_cache.shape, gd, device),
                                v_cache=_randn_bf16(first.v_cache.shape, gd, device), block_table=first.block_table,
                                prefix_len=first.prefix_len, window_len=first.window_len, cu_window=first.cu_window,
                                mask_mode=first.mask_mode, block_size=32, page_size=page_size,
                                prefix_host=first.prefix_host,
                                window_host=first.window_host, mode_host=first.mode_host))
    edit = edit_problem(batch * 64, vocab, torch.bfloat16, 5, device, sd=2.0, peak_frac=1.0, peak_lo=0.0,
                        peak_hi=12.0, tau=0.9, committed_argmax_frac=0.8, g=gd)
    return {"name": "serving128", "attn": attn, "edit": edit, "layers": layers}


WORKLOADS = {"tiny": tiny, "batch8": batch8, "varlen64": varlen64, "long32k": long32k, "serving128": serving128}


@dataclass
class SftProblem:
    """A packed batch of Multi-Block Edit SFT training sequences: sequence s is
    [prompt blocks | noisy blocks | clean blocks] of block_size tokens
    (its last block may be cut short by `trim`)."""
    q: torch.Tensor        # bf16 [T, Hq, D]
    k: torch.Tensor        # bf16 [T, Hkv, D]
    v: torch.Tensor        # bf16 [T, Hkv, D]
    dout: torch.Tensor     # bf16 [T, Hq, D], upstream gradient of the attention output
    seq_len: torch.Tensor  # int32 [batch]
    cu_seqlens: torch.Tensor  # int32 [batch + 1]
    n_prompt_blocks: torch.Tensor  # int32 [batch]
    n_blocks: torch.Tensor  # int32 [batch]
    block_size: int
    seq_host: list

    @property
    def max_seq_len(self):
        return max(self.seq_host) if self.seq_host else 0

    @property
    def mask_rows(self):
        return max(1, (self.max_seq_len + self.block_size - 1) // self.block_size)


def sft_problem(n_prompt_blocks, n_blocks, num_q_heads, num_kv_heads, head_dim, block_size, seed, device="cpu",
                trim=None, g=None) -> SftProblem:
    """Random N(0,1) bf16 q/k/v/dout for SFT sequences of (Np + 2N) blocks each,
    optionally shortened by trim[s] tokens (a ragged last block)."""
    g = g or _gen(seed, device)
    trim = trim or [0] * len(n_blocks)
    lens = [(p + 2 * n) * block_size - t for p, n, t in zip(n_prompt_blocks, n_blocks, trim)]
    T = sum(lens)
    cu = [0]
    for n in lens:
        cu.append(cu[-1] + n)
    t32 = lambda x: torch.tensor(x, dtype=torch.int32, device=device)
    return SftProblem(q=_randn_bf16((T, num_q_heads, head_dim), g, device),
                      k=_randn_bf16((T, num_kv_heads, head_dim), g, device),
                      v=_randn_bf16((T, num_kv_heads, head_dim), g, device),
                      dout=_randn_bf16((T, num_q_heads, head_dim), g, device), seq_len=t32(lens), cu_seqlens=t32(cu),
                      n_prompt_blocks=t32(list(n_prompt_blocks)), n_blocks=t32(list(n_blocks)),
                      block_size=block_size, seq_host=lens)


def extract_sequences(prob: AttnProblem, seqs):
    """The given sequences of `prob` as a standalone CPU problem (their pages
    copied into a compact cache, block table renumbered)."""
    ps = prob.page_size
    bt_all = prob.block_table.cpu()
    cu_all = prob.cu_window.cpu()
    pages, bts, qs, kws, vws = [], [], [], [], []
    prefix, window, modes, cu = [], [], [], [0]
    for s in seqs:
        P, W = prob.prefix_host[s], prob.window_host[s]
        n = (P + ps - 1) // ps
        ids = bt_all[s, :n].long()
        bts.append(list(range(len(pages), len(pages) + n)))
        pages += ids.tolist()
        t0 = int(cu_all[s])
        qs.append(prob.q[t0:t0 + W].cpu())
        kws.append(prob.k_win[t0:t0 + W].cpu())
        vws.append(prob.v_win[t0:t0 + W].cpu())
        prefix.append(P)
        window.append(W)
        modes.append(prob.mode_host[s])
        cu.append(cu[-1] + W)
    idx = torch.tensor(pages if pages else [0], dtype=torch.long, device=prob.k_cache.device)
    kc = prob.k_cache.index_select(0, idx).cpu()
    vc = prob.v_cache.index_select(0, idx).cpu()
    maxp = max(1, max(len(b) for b in bts))
    bt = torch.full((len(seqs), maxp), -1, dtype=torch.int32)
    for i, b in enumerate(bts):
        bt[i, :len(b)] = torch.tensor(b, dtype=torch.int32)
    t32 = lambda x: torch.tensor(x, dtype=torch.int32)
    return AttnProblem(q=torch.cat(qs), k_win=torch.cat(kws), v_win=torch.cat(vws), k_cache=kc, v_cache=vc,
                       block_table=bt, prefix_len=t32(prefix), window_len=t32(window), cu_window=t32(cu),
                       mask_mode=torch.tensor(modes, dtype=torch.uint8), block_size=prob.block_size,
                       page_size=ps, prefix_host=prefix, window_host=window, mode_host=modes)


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 tensor (for the oracle's C interface)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view("uint16")
