"""CPU oracle for the MBE editing-pass hot path (test infrastructure only).

This package is a plain, slow, double-precision restatement of what the hot
path computes, written from the paper (arXiv 2607.22663):

* ``window_attention``  -- Eq. 5 editing window with full attention inside the
  window, Sec. 2.2 block-causal conditioning, over a paged cached prefix.
* ``edit_decide``       -- the T2T edit set of Eq. 2 (argmax, confidence,
  threshold-and-replace).
* ``kv_window_write``   -- Sec. 4.3 targeted refresh: window K/V written to
  the paged cache at positions [P, P+W).
* ``denoise_update``    -- the full Eq. 2 step (M2T set Gamma_t with forced
  unmasking, T2T set Delta_t), per-row entropies, changed-block flags.
* ``tail_entropy_select`` -- Eqs. 6-7 tail-entropy scores and window start.
* ``refresh_plan``      -- Sec. 4.3 targeted refresh: one block-causal
  recompute problem per changed block, laid out as a ragged batch.
* ``lm_head_logits``    -- the LM-head projection whose rows the T2T rule
  reads (float64 logits for ``edit_decide`` / ``denoise_update``).
* ``sft_block_mask``, ``block_mask_attention``, ``block_mask_attention_bwd`` --
  the cross-block training mask of Multi-Block Edit SFT (Sec. 3) and attention
  (forward and gradients) under a block mask.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import it. It shares no code with the CUDA library and never
imports it. The arithmetic lives in ``mbe_oracle.c`` (compiled with gcc, no
fast-math); this module only marshals numpy arrays.

Parity status: every function is pinned by tests in ``tests/test_oracle_*.py``
against library routines (torch float64 SDPA / softmax), closed forms and
invariants; nothing here is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_SRC = _HERE / "mbe_oracle.c"
_BUILD = _HERE / "_build"
_LIB_PATH = _BUILD / "libmbe_oracle.so"
_lib = None

STATUS = {0: "ok", 1: "bad argument", 2: "page id out of range", 3: "rows without a softmax", 4: "out of memory"}
UNDECIDABLE = 3  # completed; some logit rows had no softmax (NaN / +inf, or every logit -inf)


def build(force: bool = False) -> Path:
    """Compile the oracle's C source into a shared library (gcc, OpenMP, -O2)."""
    _BUILD.mkdir(exist_ok=True)
    if force or not _LIB_PATH.exists() or _LIB_PATH.stat().st_mtime < _SRC.stat().st_mtime:
        tmp = _LIB_PATH.with_suffix(".so.tmp%d" % os.getpid())
        cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", str(tmp), str(_SRC), "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(str(_LIB_PATH))
        P = ctypes.c_void_p
        i32, i64, f32, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_double
        lib.oracle_num_threads.restype = ctypes.c_int
        lib.oracle_window_attention.restype = ctypes.c_int
        lib.oracle_window_attention.argtypes = [P, P, P, P, P, P, i32, P, P, P, P, i32, i32, i32, i32, i32, i32,
                                                i32, f64, i32, P, P, P, P]
        lib.oracle_edit_decide.restype = ctypes.c_int
        lib.oracle_edit_decide.argtypes = [P, i32, i64, i32, i32, P, P, f32, P, i32, P, P, P, P, P]
        lib.oracle_denoise_update.restype = ctypes.c_int
        lib.oracle_denoise_update.argtypes = [P, i32, i64, i32, P, i32, i32, i32, P, i32, f32, f32, P, P, P, P, P, P,
                                              P, P]
        lib.oracle_tail_entropy_select.restype = ctypes.c_int
        lib.oracle_tail_entropy_select.argtypes = [P, P, i32, i32, i32, f64, i32, P, P, P]
        lib.oracle_kv_window_write.restype = ctypes.c_int
        lib.oracle_kv_window_write.argtypes = [P, P, P, P, P, i32, P, P, P, P, i32, i32, i32, i32, i32, i32, i32]
        lib.oracle_lm_head_logits.restype = ctypes.c_int
        lib.oracle_lm_head_logits.argtypes = [P, P, i32, i32, i32, i32, P, P]
        lib.oracle_sft_block_mask.restype = ctypes.c_int
        lib.oracle_sft_block_mask.argtypes = [i32, i32, i32, i32, P]
        lib.oracle_block_mask_attention.restype = ctypes.c_int
        lib.oracle_block_mask_attention.argtypes = [P, P, P, i32, i32, i32, i32, i32, P, i32, f64, P, P]
        lib.oracle_block_mask_attention_bwd.restype = ctypes.c_int
        lib.oracle_block_mask_attention_bwd.argtypes = [P, P, P, P, i32, i32, i32, i32, i32, P, i32, f64, P, P, P]
        lib.oracle_refresh_plan.restype = ctypes.c_int
        lib.oracle_refresh_plan.argtypes = [P, i32, P, P, P, P, i32, i32, i32, i32, P, P, P, P, P, P, P]
        _lib = lib
    return _lib


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def _logit_dtype(logits, is_bf16):
    """0 float32, 1 bf16 bits (uint16, is_bf16), 2 float64."""
    if is_bf16:
        return 1
    return 2 if np.asarray(logits).dtype == np.float64 else 0


def _check(rc):
    if rc != 0:
        raise RuntimeError("oracle: " + STATUS.get(rc, str(rc)))


def window_attention(q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window,
                     mask_mode, block_size, page_size, scale=None, units=None):
    """Window attention (Eq. 5, Sec. 2.2) in float64.

    q: uint16 bf16 bits [T, Hq, D]; k_win/v_win: [T, Hkv, D];
    k_cache/v_cache: [num_pages, Hkv, page_size, D]; block_table: int32
    [batch, max_pages]; prefix_len/window_len: int32 [batch]; cu_window: int32
    [batch+1]; mask_mode: uint8 [batch] (0 block_causal, 1 bidirectional).
    units: optional list of (seq, q_head) pairs to compute (others stay NaN).
    Returns (out float64 [T, Hq, D], lse float64 [T, Hq]).
    """
    lib = _load()
    q = _c(q, np.uint16)
    T, Hq, D = q.shape
    Hkv = k_win.shape[1]
    num_pages = k_cache.shape[0]
    block_table = _c(block_table, np.int32)
    batch = block_table.shape[0]
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    out = np.full((T, Hq, D), np.nan, dtype=np.float64)
    lse = np.full((T, Hq), np.nan, dtype=np.float64)
    if units is None:
        n_units, us, uh = -1, None, None
    else:
        units = np.asarray(units, dtype=np.int32).reshape(-1, 2)
        n_units = units.shape[0]
        us, uh = np.ascontiguousarray(units[:, 0]), np.ascontiguousarray(units[:, 1])
    args = [_c(k_win, np.uint16), _c(v_win, np.uint16), _c(k_cache, np.uint16), _c(v_cache, np.uint16)]
    pl, wl, cu, mm = _c(prefix_len, np.int32), _c(window_len, np.int32), _c(cu_window, np.int32), _c(mask_mode, np.uint8)
    rc = lib.oracle_window_attention(_ptr(q), *[_ptr(a) for a in args], _ptr(block_table), block_table.shape[1],
                                     _ptr(pl), _ptr(wl), _ptr(cu), _ptr(mm), batch, Hq, Hkv, D, block_size,
                                     page_size, num_pages, float(scale), n_units, _ptr(us), _ptr(uh), _ptr(out),
                                     _ptr(lse))
    _check(rc)
    return out, lse


def edit_decide(logits, committed, tau=0.0, tau_per_row=None, editable=None, rows=None, is_bf16=False):
    """T2T edit decision of Eq. 2 in float64.

    logits: float32 [R, V], float64 [R, V] or uint16 bf16 bits [R, V] (set is_bf16).
    Returns dict of new_tokens int32, edit_mask uint8, confidence float64,
    argmax int32 (all [R]; rows not in `rows` are left as -1 / 0 / NaN) and
    "undecidable": True if some computed row had no softmax (a NaN or +inf
    logit, or every logit -inf); such a row keeps its token, with argmax -1 and
    confidence NaN.
    """
    lib = _load()
    logits = np.ascontiguousarray(logits)
    R, V = logits.shape
    committed = _c(committed, np.int32)
    tpr = _c(tau_per_row, np.float32)
    ed = _c(editable, np.uint8)
    new = np.full(R, -1, dtype=np.int32)
    mask = np.zeros(R, dtype=np.uint8)
    conf = np.full(R, np.nan, dtype=np.float64)
    am = np.full(R, -1, dtype=np.int32)
    sel = None if rows is None else np.ascontiguousarray(rows, dtype=np.int32)
    dtype = _logit_dtype(logits, is_bf16)
    if dtype == 0:
        logits = np.ascontiguousarray(logits, dtype=np.float32)
    rc = lib.oracle_edit_decide(_ptr(logits), dtype, V, R, V, _ptr(committed), _ptr(tpr), float(tau), _ptr(ed),
                                -1 if sel is None else sel.shape[0], _ptr(sel), _ptr(new), _ptr(mask), _ptr(conf),
                                _ptr(am))
    if rc != UNDECIDABLE:
        _check(rc)
    return {"new_tokens": new, "edit_mask": mask, "confidence": conf, "argmax": am, "undecidable": rc == UNDECIDABLE}


def denoise_update(logits, tokens, cu_rows, block_size, mask_id, omega_mask, omega_edit, editable=None,
                   max_blocks=None, is_bf16=False):
    """Full Eq. 2 update (Gamma_t, forced unmasking, Delta_t) with entropies,
    changed-block flags and per-sequence change counts, in float64.
    "undecidable" is True if some row had no softmax (it keeps its token, with
    argmax -1 and confidence / entropy NaN, and is never force-unmasked)."""
    lib = _load()
    dtype = _logit_dtype(logits, is_bf16)
    logits = np.ascontiguousarray(logits) if dtype else np.ascontiguousarray(logits, dtype=np.float32)
    R, V = logits.shape
    cu = _c(cu_rows, np.int32)
    ns = cu.shape[0] - 1
    if max_blocks is None:
        max_blocks = max([1] + [int((cu[s + 1] - cu[s] + block_size - 1) // block_size) for s in range(ns)])
    tokens = _c(tokens, np.int32)
    out = {"new_tokens": np.zeros(R, np.int32), "kind": np.zeros(R, np.uint8), "confidence": np.zeros(R),
           "argmax": np.zeros(R, np.int32), "entropy": np.zeros(R), "block_changed": np.zeros((ns, max_blocks), np.uint8),
           "seq_changes": np.zeros(ns, np.int32)}
    rc = lib.oracle_denoise_update(_ptr(logits), dtype, V, V, _ptr(cu), ns, block_size, max_blocks,
                                   _ptr(tokens), int(mask_id), float(omega_mask), float(omega_edit),
                                   _ptr(_c(editable, np.uint8)), _ptr(out["new_tokens"]), _ptr(out["kind"]),
                                   _ptr(out["confidence"]), _ptr(out["argmax"]), _ptr(out["entropy"]),
                                   _ptr(out["block_changed"]), _ptr(out["seq_changes"]))
    if rc != UNDECIDABLE:
        _check(rc)
    out["undecidable"] = rc == UNDECIDABLE
    return out


def tail_entropy_select(block_entropy, n_valid, rho, k_max):
    """Eqs. 6-7: tail-entropy scores of the candidate blocks and the chosen
    window start. block_entropy: float32 [S, n_hist, B]; n_valid: int32 [S]."""
    lib = _load()
    be = np.ascontiguousarray(block_entropy, dtype=np.float32)
    S, H, B = be.shape
    nv = _c(n_valid, np.int32)
    scores = np.zeros((S, H))
    best = np.zeros(S, np.int32)
    wb = np.zeros(S, np.int32)
    # rho as the float32 the library receives, so ceil(rho * B) uses the same value
    rc = lib.oracle_tail_entropy_select(_ptr(be), _ptr(nv), S, H, B, float(np.float32(rho)), int(k_max), _ptr(scores),
                                        _ptr(best),
                                        _ptr(wb))
    _check(rc)
    return {"scores": scores, "best_slot": best, "window_blocks": wb}


def kv_window_write(k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, block_size,
                    block_write_mask=None):
    """Targeted-refresh KV write (Sec. 4.3). Returns new (k_cache, v_cache) copies."""
    lib = _load()
    kc = np.array(k_cache, dtype=np.uint16, copy=True)
    vc = np.array(v_cache, dtype=np.uint16, copy=True)
    num_pages, Hkv, page_size, D = kc.shape
    bt = _c(block_table, np.int32)
    batch = bt.shape[0]
    bwm = _c(block_write_mask, np.uint8)
    maxb = 0 if bwm is None else bwm.shape[1]
    rc = lib.oracle_kv_window_write(_ptr(_c(k_win, np.uint16)), _ptr(_c(v_win, np.uint16)), _ptr(kc), _ptr(vc),
                                    _ptr(bt), bt.shape[1], _ptr(_c(prefix_len, np.int32)),
                                    _ptr(_c(window_len, np.int32)), _ptr(_c(cu_window, np.int32)), _ptr(bwm), maxb,
                                    batch, Hkv, D, block_size, page_size, num_pages)
    _check(rc)
    return kc, vc


def refresh_plan(block_changed, prefix_len, window_len, cu_window, block_table, block_size, total_rows=None):
    """Targeted refresh layout (Sec. 4.3): one entry per (sequence, window
    block), non-empty for the changed blocks. Returns a dict of numpy arrays
    prefix_len, window_len, cu_window, mask_mode, block_table, src_row, count."""
    lib = _load()
    bc = _c(block_changed, np.uint8)
    batch, max_blocks = bc.shape
    bt = _c(block_table, np.int32)
    cu = _c(cu_window, np.int32)
    if total_rows is None:
        total_rows = int(cu[batch]) if batch else 0
    E = batch * max_blocks
    out = {"prefix_len": np.zeros(E, np.int32), "window_len": np.zeros(E, np.int32),
           "cu_window": np.zeros(E + 1, np.int32), "mask_mode": np.zeros(E, np.uint8),
           "block_table": np.zeros((E, bt.shape[1]), np.int32), "src_row": np.zeros(total_rows, np.int32),
           "count": np.zeros(2, np.int32)}
    rc = lib.oracle_refresh_plan(_ptr(bc), max_blocks, _ptr(_c(prefix_len, np.int32)), _ptr(_c(window_len, np.int32)),
                                 _ptr(cu), _ptr(bt), bt.shape[1], batch, block_size, total_rows,
                                 _ptr(out["prefix_len"]), _ptr(out["window_len"]), _ptr(out["cu_window"]),
                                 _ptr(out["mask_mode"]), _ptr(out["block_table"]), _ptr(out["src_row"]),
                                 _ptr(out["count"]))
    _check(rc)
    return out


def lm_head_logits(hidden, weight, rows=None):
    """LM-head logits in float64 from bf16 bits: hidden uint16 [R, d], weight
    uint16 [V, d]. Returns [R, V] (or [len(rows), V] for the selected rows)."""
    lib = _load()
    h = _c(hidden, np.uint16)
    w = _c(weight, np.uint16)
    R, d = h.shape
    V = w.shape[0]
    assert w.shape[1] == d
    sel = None if rows is None else np.ascontiguousarray(rows, dtype=np.int32)
    n = R if sel is None else sel.shape[0]
    out = np.zeros((n, V), dtype=np.float64)
    rc = lib.oracle_lm_head_logits(_ptr(h), _ptr(w), R, V, d, -1 if sel is None else n, _ptr(sel), _ptr(out))
    _check(rc)
    return out


def sft_block_mask(n_prompt_blocks, n_blocks, K, words_per_row=None):
    """Cross-block SFT mask (Sec. 3) as uint32 bits [nb, words_per_row]."""
    lib = _load()
    nb = n_prompt_blocks + 2 * n_blocks
    wpr = words_per_row or max(1, (nb + 31) // 32)
    m = np.zeros((nb, wpr), dtype=np.uint32)
    _check(lib.oracle_sft_block_mask(n_prompt_blocks, n_blocks, K, wpr, _ptr(m)))
    return m


def mask_bits_to_dense(mask, nb):
    """Boolean [nb, nb] view of a uint32 bit mask."""
    m = np.asarray(mask, dtype=np.uint32)
    cols = np.arange(nb)
    return ((m[:, cols // 32] >> (cols % 32).astype(np.uint32)) & 1).astype(bool)[:nb]


def block_mask_attention(q, k, v, block_size, mask, scale=None):
    """Attention of one sequence under a block mask, float64 (out [T,Hq,D], lse [T,Hq])."""
    lib = _load()
    q, k, v = _c(q, np.uint16), _c(k, np.uint16), _c(v, np.uint16)
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    m = _c(mask, np.uint32)
    scale = 1.0 / np.sqrt(D) if scale is None else scale
    out = np.zeros((T, Hq, D))
    lse = np.zeros((T, Hq))
    _check(lib.oracle_block_mask_attention(_ptr(q), _ptr(k), _ptr(v), T, Hq, Hkv, D, block_size, _ptr(m), m.shape[1],
                                           float(scale), _ptr(out), _ptr(lse)))
    return out, lse


def block_mask_attention_bwd(q, k, v, dout, block_size, mask, scale=None):
    """Gradients (dq [T,Hq,D], dk, dv [T,Hkv,D]) of block-masked attention, float64."""
    lib = _load()
    q, k, v, do = _c(q, np.uint16), _c(k, np.uint16), _c(v, np.uint16), _c(dout, np.uint16)
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    m = _c(mask, np.uint32)
    scale = 1.0 / np.sqrt(D) if scale is None else scale
    dq = np.zeros((T, Hq, D))
    dk = np.zeros((T, Hkv, D))
    dv = np.zeros((T, Hkv, D))
    _check(lib.oracle_block_mask_attention_bwd(_ptr(q), _ptr(k), _ptr(v), _ptr(do), T, Hq, Hkv, D, block_size, _ptr(m),
                                               m.shape[1], float(scale), _ptr(dq), _ptr(dk), _ptr(dv)))
    return dq, dk, dv
