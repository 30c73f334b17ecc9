"""Python binding of libmbe (argument marshalling only).

Each function takes torch tensors, checks their dtype/device/layout, and calls
the C entry point of the same name in ``libmbe.so`` on the current CUDA stream.
All arithmetic runs in the library's CUDA kernels; there is no fallback: if the
library is missing or the call fails, an exception is raised.
"""
from __future__ import annotations

import ctypes
import re
from pathlib import Path
from typing import Optional

import torch

from . import build as _build

MBE_OK = 0
STATUS_NAMES = {0: "MBE_OK", 1: "MBE_ERR_INVALID_ARG", 2: "MBE_ERR_UNSUPPORTED", 3: "MBE_ERR_CUDA",
                4: "MBE_ERR_TIMEOUT", 5: "MBE_ERR_WORKSPACE", 6: "MBE_ERR_DEVICE_CHECK"}
DEVERR_TIMEOUT, DEVERR_LENGTH, DEVERR_PAGE, DEVERR_CAPACITY, DEVERR_PLAN = 0x1, 0x2, 0x4, 0x8, 0x10
DEVERR_NONFINITE = 0x20
DEFAULT_WAIT_LIMIT_NS = 1_000_000_000
BLOCK_CAUSAL, MULTI_BLOCK_BIDIRECTIONAL, BLOCK_MASK = 0, 1, 2
HEADER = _build.INCLUDE / "mbe.h"

_lib = None


class MbeError(RuntimeError):
    def __init__(self, fn, status):
        self.status = status
        detail = ""
        if status == 3:
            try:
                detail = "; " + lib().mbe_last_error_string().decode()
            except Exception:
                pass
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(status, status)} ({_status_string(status)}{detail})")


def _status_string(status):
    try:
        return lib().mbe_status_string(status).decode()
    except Exception:
        return "?"


def lib(build_if_missing: bool = True):
    """The loaded libmbe (ctypes.CDLL), building it in-tree if needed."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if build_if_missing:
        path = _build.build()
    if not Path(path).exists():
        raise RuntimeError(f"libmbe.so not found at {path}; run paper_2607_22663_gb300.build.build()")
    L = ctypes.CDLL(str(path))
    P, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    L.mbe_window_attention.restype = ctypes.c_int
    L.mbe_window_attention.argtypes = [P, P, P, P, P, i32, P, i32, P, P, P, P, i32, i32, i32, i32, i32, i32, i32, i32,
                                       i32, f32, P, P, P, sz, P]
    L.mbe_window_attention_run.restype = ctypes.c_int
    L.mbe_window_attention_run.argtypes = list(L.mbe_window_attention.argtypes)
    L.mbe_window_attention_plan.restype = ctypes.c_int
    L.mbe_window_attention_plan.argtypes = [P, P, P, P, i32, i32, i32, i32, i32, i32, i32, i32, P, sz, P]
    L.mbe_window_attention_noalloc.restype = ctypes.c_int
    L.mbe_window_attention_noalloc.argtypes = [P, P, P, P, P, i32, P, i32, P, P, P, P, i32, i32, i32, i32, i32, i32,
                                               i32, i32, i32, f32, P, P, P]
    L.mbe_window_attention_workspace_size.restype = sz
    L.mbe_window_attention_workspace_size.argtypes = [i32, i32, i32, i32, i32, i32]
    L.mbe_edit_decide.restype = ctypes.c_int
    L.mbe_edit_decide.argtypes = [P, ctypes.c_int, i64, i32, i32, P, P, f32, P, P, P, P, P, P]
    L.mbe_denoise_update.restype = ctypes.c_int
    L.mbe_denoise_update.argtypes = [P, ctypes.c_int, i64, i32, P, i32, i32, i32, i32, P, i32, f32, f32, P, P, P, P, P,
                                     P, P, P, P]
    L.mbe_tail_entropy_select.restype = ctypes.c_int
    L.mbe_tail_entropy_select.argtypes = [P, P, i32, i32, i32, f32, i32, P, P, P, P]
    L.mbe_kv_window_write.restype = ctypes.c_int
    L.mbe_kv_window_write.argtypes = [P, P, P, P, i32, P, i32, P, P, P, P, i32, i32, i32, i32, i32, i32, i32, P]
    L.mbe_lm_head_workspace_size.restype = sz
    L.mbe_lm_head_workspace_size.argtypes = [i32, i32]
    L.mbe_lm_head_edit_decide.restype = ctypes.c_int
    L.mbe_lm_head_edit_decide.argtypes = [P, P, i32, i32, i32, P, P, f32, P, P, P, P, P, P, P, sz, P]
    L.mbe_sft_block_mask.restype = ctypes.c_int
    L.mbe_sft_block_mask.argtypes = [P, P, i32, i32, i32, i32, P, P]
    L.mbe_block_mask_attention.restype = ctypes.c_int
    L.mbe_block_mask_attention.argtypes = [P, P, P, P, P, P, i32, i32, i32, i32, i32, i32, i32, i32, i32, f32, P, P, P,
                                           sz, P]
    L.mbe_block_mask_attention_bwd_workspace_size.restype = sz
    L.mbe_block_mask_attention_bwd_workspace_size.argtypes = [i32, i32, i32]
    L.mbe_block_mask_attention_bwd.restype = ctypes.c_int
    L.mbe_block_mask_attention_bwd.argtypes = [P, P, P, P, P, P, P, P, P, i32, i32, i32, i32, i32, i32, i32, i32, i32,
                                               f32, P, P, P, P, sz, P]
    L.mbe_refresh_plan.restype = ctypes.c_int
    L.mbe_refresh_plan.argtypes = [P, i32, P, P, P, P, i32, i32, i32, i32, i32, P, P, P, P, P, P, P, P]
    L.mbe_gather_rows.restype = ctypes.c_int
    L.mbe_gather_rows.argtypes = [P, i64, i64, P, i64, P, P, P]
    L.mbe_gather_rows_multi.restype = ctypes.c_int
    L.mbe_gather_rows_multi.argtypes = [i32, P, P, P, i64, P, i64, P, P]
    L.mbe_refresh_gather_write.restype = ctypes.c_int
    L.mbe_refresh_gather_write.argtypes = [P, P, P, i64, i32, i32, i32, P, P, i64, P, P, P, i32, i32, P, P, i32, i32,
                                           P, P, P, P]
    L.mbe_pass_loop_begin.restype = ctypes.c_int
    L.mbe_pass_loop_begin.argtypes = [i32, P, P, ctypes.POINTER(ctypes.c_void_p)]
    L.mbe_pass_loop_until_stable.restype = ctypes.c_int
    L.mbe_pass_loop_until_stable.argtypes = [P, P, i32, P]
    L.mbe_pass_loop_end.restype = ctypes.c_int
    L.mbe_pass_loop_end.argtypes = [P, P]
    L.mbe_pass_loop_launch.restype = ctypes.c_int
    L.mbe_pass_loop_launch.argtypes = [P, P]
    L.mbe_pass_loop_destroy.restype = None
    L.mbe_pass_loop_destroy.argtypes = [P]
    L.mbe_get_device_error.restype = ctypes.c_int
    L.mbe_get_device_error.argtypes = [P, ctypes.POINTER(ctypes.c_uint32)]
    L.mbe_status_string.restype = ctypes.c_char_p
    L.mbe_status_string.argtypes = [ctypes.c_int]
    L.mbe_last_error_string.restype = ctypes.c_char_p
    L.mbe_last_error_string.argtypes = []
    L.mbe_version.restype = i32
    L.mbe_version.argtypes = []
    L.mbe_set_wait_limit_ns.restype = ctypes.c_uint64
    L.mbe_set_wait_limit_ns.argtypes = [ctypes.c_uint64]
    L.mbe_window_attention_plan_stats.restype = ctypes.c_int
    L.mbe_window_attention_plan_stats.argtypes = [P, sz, ctypes.POINTER(i32), ctypes.POINTER(i32), P]
    _lib = L
    return L


def declared_symbols():
    """Function names declared in include/mbe.h."""
    text = HEADER.read_text()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(mbe_\w+)\s*\(", text, flags=re.M)))


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _need(t, name, dtype=None, cuda=True):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if cuda and not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _shape(t, name, shape):
    """The C ABI takes plain pointers and trusts the lengths it is given, so every
    array the call reads or writes is held to the shape those lengths imply."""
    if t is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")


def _same_device(dev, stream, **tensors):
    """Every tensor on `dev`, `dev` the current CUDA device (the library launches on
    the current device) and an explicit stream on `dev` too."""
    for name, t in tensors.items():
        if t is not None and t.device != dev:
            raise ValueError(f"{name} is on {t.device}, the call's tensors are on {dev}")
    if dev.index != torch.cuda.current_device():
        raise ValueError(f"the tensors are on {dev} but the current CUDA device is {torch.cuda.current_device()}")
    if stream is not None and stream.device != dev:
        raise ValueError(f"stream is on {stream.device}, the tensors on {dev}")


def _check(fn, st):
    if st != MBE_OK:
        raise MbeError(fn, st)


def window_attention_workspace_size(batch, num_q_heads, num_kv_heads, head_dim, max_window, max_prefix):
    return int(lib().mbe_window_attention_workspace_size(batch, num_q_heads, num_kv_heads, head_dim, max_window,
                                                         max_prefix))


def _attention_shapes(q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, mask_mode):
    """Shapes of a window-attention call (include/mbe.h): q [T, Hq, D], k_win and v_win
    [T, Hkv, D], caches [num_pages, Hkv, page_size, D], block_table [batch, max_pages],
    prefix_len / window_len / mask_mode [batch], cu_window [batch + 1]."""
    if q.dim() != 3 or k_cache.dim() != 4 or block_table.dim() != 2:
        raise ValueError("q must be [T, Hq, D], the caches [num_pages, Hkv, page_size, D], block_table [batch, pages]")
    T, Hq, D = q.shape
    num_pages, Hkv, page_size, _ = k_cache.shape
    _shape(k_cache, "k_cache", (num_pages, Hkv, page_size, D))
    _shape(v_cache, "v_cache", (num_pages, Hkv, page_size, D))
    _shape(k_win, "k_win", (T, Hkv, D))
    _shape(v_win, "v_win", (T, Hkv, D))
    batch, max_pages = block_table.shape
    for t, n in ((prefix_len, "prefix_len"), (window_len, "window_len"), (mask_mode, "mask_mode")):
        _shape(t, n, (batch,))
    _shape(cu_window, "cu_window", (batch + 1,))
    return T, Hq, D, num_pages, Hkv, page_size, batch, max_pages


def _attention(fn_name, q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, mask_mode, *,
               block_size, max_window, max_prefix, softmax_scale=0.0, out=None, lse=None, return_lse=False,
               workspace=None, stream=None):
    for t, n in ((q, "q"), (k_win, "k_win"), (v_win, "v_win"), (k_cache, "k_cache"), (v_cache, "v_cache")):
        _need(t, n, torch.bfloat16)
    for t, n in ((block_table, "block_table"), (prefix_len, "prefix_len"), (window_len, "window_len"),
                 (cu_window, "cu_window")):
        _need(t, n, torch.int32)
    _need(mask_mode, "mask_mode", torch.uint8)
    T, Hq, D, num_pages, Hkv, page_size, batch, max_pages = _attention_shapes(
        q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, mask_mode)
    if out is None:
        out = torch.empty_like(q)
    _need(out, "out", torch.bfloat16)
    _shape(out, "out", (T, Hq, D))
    if return_lse and lse is None:
        lse = torch.empty((T, Hq), dtype=torch.float32, device=q.device)
    if lse is not None:
        _need(lse, "lse", torch.float32)
        _shape(lse, "lse", (T, Hq))
    if workspace is not None:
        _need(workspace, "workspace", torch.uint8)
    _same_device(q.device, stream, k_win=k_win, v_win=v_win, k_cache=k_cache, v_cache=v_cache,
                 block_table=block_table, prefix_len=prefix_len, window_len=window_len, cu_window=cu_window,
                 mask_mode=mask_mode, out=out, lse=lse, workspace=workspace)
    need = window_attention_workspace_size(batch, Hq, Hkv, D, max_window, max_prefix)
    if workspace is None or workspace.numel() < need:
        if fn_name == "mbe_window_attention_run":
            raise ValueError("mbe_window_attention_run needs the workspace its plan was written into")
        workspace = torch.empty(max(need, 1), dtype=torch.uint8, device=q.device)
    st = getattr(lib(), fn_name)(_ptr(q), _ptr(k_win), _ptr(v_win), _ptr(k_cache), _ptr(v_cache), num_pages,
                                 _ptr(block_table), max_pages, _ptr(prefix_len), _ptr(window_len), _ptr(cu_window),
                                 _ptr(mask_mode), batch, T, Hq, Hkv, D, block_size, page_size, max_window,
                                 max_prefix, float(softmax_scale), _ptr(out), _ptr(lse), _ptr(workspace),
                                 workspace.numel(), _stream(stream))
    _check(fn_name, st)
    return (out, lse) if return_lse else out


def window_attention(q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, mask_mode,
                     **kw):
    """mbe_window_attention: see include/mbe.h. Returns out (and lse if requested)."""
    return _attention("mbe_window_attention", q, k_win, v_win, k_cache, v_cache, block_table, prefix_len,
                      window_len, cu_window, mask_mode, **kw)


def window_attention_plan(prefix_len, window_len, cu_window, mask_mode, *, total_q_tokens, num_q_heads, num_kv_heads,
                          head_dim, block_size, max_window, max_prefix, workspace, stream=None):
    """mbe_window_attention_plan: writes the work list for these lengths into `workspace`."""
    for t, n in ((prefix_len, "prefix_len"), (window_len, "window_len"), (cu_window, "cu_window")):
        _need(t, n, torch.int32)
    _need(mask_mode, "mask_mode", torch.uint8)
    _need(workspace, "workspace", torch.uint8)
    batch = prefix_len.shape[0]
    for t, n in ((prefix_len, "prefix_len"), (window_len, "window_len"), (mask_mode, "mask_mode")):
        _shape(t, n, (batch,))
    _shape(cu_window, "cu_window", (batch + 1,))
    _same_device(prefix_len.device, stream, window_len=window_len, cu_window=cu_window, mask_mode=mask_mode,
                 workspace=workspace)
    st = lib().mbe_window_attention_plan(_ptr(prefix_len), _ptr(window_len), _ptr(cu_window), _ptr(mask_mode), batch,
                                         total_q_tokens, num_q_heads, num_kv_heads, head_dim, block_size, max_window,
                                         max_prefix, _ptr(workspace), workspace.numel(), _stream(stream))
    _check("mbe_window_attention_plan", st)


def window_attention_run(q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, mask_mode,
                         **kw):
    """mbe_window_attention_run: the attention with the plan already in `workspace`."""
    return _attention("mbe_window_attention_run", q, k_win, v_win, k_cache, v_cache, block_table, prefix_len,
                      window_len, cu_window, mask_mode, **kw)


def window_attention_noalloc(q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window,
                             mask_mode, *, block_size, max_window, max_prefix, softmax_scale=0.0, out, lse=None,
                             stream=None):
    """mbe_window_attention_noalloc: the attention with the library's static
    64 MiB scratch instead of a workspace, for callers that must not allocate.
    `out` (and `lse`, if wanted) must be given: this call allocates nothing."""
    for t, n in ((q, "q"), (k_win, "k_win"), (v_win, "v_win"), (k_cache, "k_cache"), (v_cache, "v_cache"),
                 (out, "out")):
        _need(t, n, torch.bfloat16)
    for t, n in ((block_table, "block_table"), (prefix_len, "prefix_len"), (window_len, "window_len"),
                 (cu_window, "cu_window")):
        _need(t, n, torch.int32)
    _need(mask_mode, "mask_mode", torch.uint8)
    T, Hq, D, num_pages, Hkv, page_size, batch, max_pages = _attention_shapes(
        q, k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, mask_mode)
    _shape(out, "out", (T, Hq, D))
    if lse is not None:
        _need(lse, "lse", torch.float32)
        _shape(lse, "lse", (T, Hq))
    _same_device(q.device, stream, k_win=k_win, v_win=v_win, k_cache=k_cache, v_cache=v_cache,
                 block_table=block_table, prefix_len=prefix_len, window_len=window_len, cu_window=cu_window,
                 mask_mode=mask_mode, out=out, lse=lse)
    st = lib().mbe_window_attention_noalloc(_ptr(q), _ptr(k_win), _ptr(v_win), _ptr(k_cache), _ptr(v_cache),
                                            num_pages, _ptr(block_table), max_pages, _ptr(prefix_len),
                                            _ptr(window_len), _ptr(cu_window), _ptr(mask_mode), batch, T, Hq, Hkv,
                                            D, block_size, page_size, max_window, max_prefix, float(softmax_scale),
                                            _ptr(out), _ptr(lse), _stream(stream))
    _check("mbe_window_attention_noalloc", st)
    return out


def edit_decide(logits, committed, tau=0.0, tau_per_row=None, editable=None, *, new_tokens=None, edit_mask=None,
                confidence=None, argmax=None, want_argmax=True, stream=None):
    """mbe_edit_decide: see include/mbe.h. Returns (new_tokens, edit_mask, confidence, argmax)."""
    if logits.dim() != 2 or logits.stride(1) != 1:
        raise ValueError("logits must be [rows, vocab] with unit stride along the vocabulary")
    if not logits.is_cuda:
        raise ValueError("logits must be a CUDA tensor")
    dt = {torch.float32: 0, torch.bfloat16: 1}.get(logits.dtype)
    if dt is None:
        raise TypeError("logits must be float32 or bfloat16")
    R, V = logits.shape
    _need(committed, "committed", torch.int32)
    dev = logits.device
    new_tokens = torch.empty(R, dtype=torch.int32, device=dev) if new_tokens is None else new_tokens
    edit_mask = torch.empty(R, dtype=torch.uint8, device=dev) if edit_mask is None else edit_mask
    confidence = torch.empty(R, dtype=torch.float32, device=dev) if confidence is None else confidence
    if want_argmax and argmax is None:
        argmax = torch.empty(R, dtype=torch.int32, device=dev)
    for t, n, dtype in ((tau_per_row, "tau_per_row", torch.float32), (editable, "editable", torch.uint8),
                        (new_tokens, "new_tokens", torch.int32), (edit_mask, "edit_mask", torch.uint8),
                        (confidence, "confidence", torch.float32), (argmax, "argmax", torch.int32)):
        if t is not None:
            _need(t, n, dtype)
            _shape(t, n, (R,))
    _shape(committed, "committed", (R,))
    _same_device(dev, stream, committed=committed, tau_per_row=tau_per_row, editable=editable, new_tokens=new_tokens,
                 edit_mask=edit_mask, confidence=confidence, argmax=argmax)
    st = lib().mbe_edit_decide(_ptr(logits), dt, logits.stride(0), R, V, _ptr(committed), _ptr(tau_per_row),
                               float(tau), _ptr(editable), _ptr(new_tokens), _ptr(edit_mask), _ptr(confidence),
                               _ptr(argmax), _stream(stream))
    _check("mbe_edit_decide", st)
    return new_tokens, edit_mask, confidence, argmax


def denoise_update(logits, tokens, cu_rows, *, block_size, mask_id, omega_mask, omega_edit, editable=None,
                   max_blocks=None, want_entropy=True, want_blocks=True, out=None, stream=None):
    """mbe_denoise_update: see include/mbe.h. Returns a dict of device tensors.

    `out` (a dict as returned by an earlier call) reuses its buffers, so the
    call allocates nothing and can be captured in a CUDA graph; max_blocks is
    then taken from out["block_changed"]."""
    if logits.dim() != 2 or logits.stride(1) != 1 or not logits.is_cuda:
        raise ValueError("logits must be a CUDA [rows, vocab] tensor with unit stride along the vocabulary")
    dt = {torch.float32: 0, torch.bfloat16: 1}.get(logits.dtype)
    if dt is None:
        raise TypeError("logits must be float32 or bfloat16")
    R, V = logits.shape
    _need(tokens, "tokens", torch.int32)
    _need(cu_rows, "cu_rows", torch.int32)
    if editable is not None:
        _need(editable, "editable", torch.uint8)
        _shape(editable, "editable", (R,))
    _shape(tokens, "tokens", (R,))
    if cu_rows.dim() != 1 or cu_rows.numel() < 1:
        raise ValueError("cu_rows must be [sequences + 1]")
    ns = cu_rows.shape[0] - 1
    dev = logits.device
    _same_device(dev, stream, tokens=tokens, cu_rows=cu_rows, editable=editable)
    if out is not None:
        for k, dtype in (("new_tokens", torch.int32), ("kind", torch.uint8), ("confidence", torch.float32),
                         ("argmax", torch.int32)):
            _need(out[k], k, dtype)
            if out[k].numel() != R:
                raise ValueError(f"out[{k!r}] must hold {R} rows")
        if out.get("block_changed") is not None:
            _need(out["block_changed"], "block_changed", torch.uint8)
            max_blocks = out["block_changed"].shape[1]
            if out["block_changed"].shape[0] != ns or out.get("seq_changes") is None or \
                    out["seq_changes"].numel() != ns:
                raise ValueError("out['block_changed'] / out['seq_changes'] must cover every sequence")
            _need(out["seq_changes"], "seq_changes", torch.int32)
        if out.get("entropy") is not None:
            _need(out["entropy"], "entropy", torch.float32)
        max_blocks = max_blocks or 1
    else:
        if max_blocks is None:
            max_blocks = max(1, (int((cu_rows[1:] - cu_rows[:-1]).max().item()) + block_size - 1) // block_size) \
                if ns else 1
        out = {"new_tokens": torch.empty(R, dtype=torch.int32, device=dev),
               "kind": torch.empty(R, dtype=torch.uint8, device=dev),
               "confidence": torch.empty(R, dtype=torch.float32, device=dev),
               "argmax": torch.empty(R, dtype=torch.int32, device=dev),
               "entropy": torch.empty(R, dtype=torch.float32, device=dev) if want_entropy else None,
               "block_changed": torch.empty((ns, max_blocks), dtype=torch.uint8, device=dev) if want_blocks else None,
               "seq_changes": torch.empty(ns, dtype=torch.int32, device=dev) if want_blocks else None}
    _same_device(dev, stream, **{k: v for k, v in out.items() if v is not None})
    st = lib().mbe_denoise_update(_ptr(logits), dt, logits.stride(0), V, _ptr(cu_rows), ns, R, block_size, max_blocks,
                                  _ptr(tokens), int(mask_id), float(omega_mask), float(omega_edit), _ptr(editable),
                                  _ptr(out["new_tokens"]), _ptr(out["kind"]), _ptr(out["confidence"]),
                                  _ptr(out["argmax"]), _ptr(out.get("entropy")), _ptr(out.get("block_changed")),
                                  _ptr(out.get("seq_changes")), _stream(stream))
    _check("mbe_denoise_update", st)
    return out


def tail_entropy_select(block_entropy, n_valid, *, rho, k_max, want_scores=True, stream=None):
    """mbe_tail_entropy_select: see include/mbe.h. Returns (best_slot, window_blocks, scores)."""
    _need(block_entropy, "block_entropy", torch.float32)
    _need(n_valid, "n_valid", torch.int32)
    S, H, B = block_entropy.shape
    dev = block_entropy.device
    _shape(n_valid, "n_valid", (S,))
    _same_device(dev, stream, n_valid=n_valid)
    best = torch.empty(S, dtype=torch.int32, device=dev)
    wb = torch.empty(S, dtype=torch.int32, device=dev)
    scores = torch.empty((S, H), dtype=torch.float32, device=dev) if want_scores else None
    st = lib().mbe_tail_entropy_select(_ptr(block_entropy), _ptr(n_valid), S, H, B, float(rho), int(k_max),
                                       _ptr(scores), _ptr(best), _ptr(wb), _stream(stream))
    _check("mbe_tail_entropy_select", st)
    return best, wb, scores


def kv_window_write(k_win, v_win, k_cache, v_cache, block_table, prefix_len, window_len, cu_window, *, block_size,
                    max_window, block_write_mask=None, stream=None):
    """mbe_kv_window_write: see include/mbe.h. Writes k_cache/v_cache in place."""
    for t, n in ((k_win, "k_win"), (v_win, "v_win"), (k_cache, "k_cache"), (v_cache, "v_cache")):
        _need(t, n, torch.bfloat16)
    for t, n in ((block_table, "block_table"), (prefix_len, "prefix_len"), (window_len, "window_len"),
                 (cu_window, "cu_window")):
        _need(t, n, torch.int32)
    if k_cache.dim() != 4 or k_win.dim() != 3 or block_table.dim() != 2:
        raise ValueError("k_win must be [T, Hkv, D], the caches [num_pages, Hkv, page_size, D], block_table [batch, pages]")
    num_pages, Hkv, page_size, D = k_cache.shape
    _shape(v_cache, "v_cache", (num_pages, Hkv, page_size, D))
    _shape(k_win, "k_win", (k_win.shape[0], Hkv, D))
    _shape(v_win, "v_win", tuple(k_win.shape))
    batch, max_pages = block_table.shape
    _shape(prefix_len, "prefix_len", (batch,))
    _shape(window_len, "window_len", (batch,))
    _shape(cu_window, "cu_window", (batch + 1,))
    max_blocks = 0
    if block_write_mask is not None:
        _need(block_write_mask, "block_write_mask", torch.uint8)
        if block_write_mask.dim() != 2 or block_write_mask.shape[0] != batch:
            raise ValueError("block_write_mask must be [batch, blocks]")
        max_blocks = block_write_mask.shape[1]
    _same_device(k_win.device, stream, v_win=v_win, k_cache=k_cache, v_cache=v_cache, block_table=block_table,
                 prefix_len=prefix_len, window_len=window_len, cu_window=cu_window, block_write_mask=block_write_mask)
    st = lib().mbe_kv_window_write(_ptr(k_win), _ptr(v_win), _ptr(k_cache), _ptr(v_cache), num_pages,
                                   _ptr(block_table), max_pages, _ptr(prefix_len), _ptr(window_len), _ptr(cu_window),
                                   _ptr(block_write_mask), max_blocks, batch, max_window, Hkv, D, block_size,
                                   page_size, _stream(stream))
    _check("mbe_kv_window_write", st)


def lm_head_workspace_size(rows, vocab):
    return int(lib().mbe_lm_head_workspace_size(int(rows), int(vocab)))


def lm_head_edit_decide(hidden, weight, committed, tau=0.0, tau_per_row=None, editable=None, *, new_tokens=None,
                        edit_mask=None, confidence=None, argmax=None, entropy=None, want_argmax=True,
                        want_entropy=False, workspace=None, stream=None):
    """mbe_lm_head_edit_decide: see include/mbe.h. Returns (new_tokens,
    edit_mask, confidence, argmax, entropy) (argmax / entropy None unless wanted)."""
    _need(hidden, "hidden", torch.bfloat16)
    _need(weight, "weight", torch.bfloat16)
    _need(committed, "committed", torch.int32)
    if hidden.dim() != 2 or weight.dim() != 2 or hidden.shape[1] != weight.shape[1]:
        raise ValueError("hidden must be [rows, d] and weight [vocab, d]")
    R, d = hidden.shape
    V = weight.shape[0]
    if committed.numel() != R:
        raise ValueError("committed must hold one token per row")
    if tau_per_row is not None:
        _need(tau_per_row, "tau_per_row", torch.float32)
    if editable is not None:
        _need(editable, "editable", torch.uint8)
    dev = hidden.device
    new_tokens = torch.empty(R, dtype=torch.int32, device=dev) if new_tokens is None else new_tokens
    edit_mask = torch.empty(R, dtype=torch.uint8, device=dev) if edit_mask is None else edit_mask
    confidence = torch.empty(R, dtype=torch.float32, device=dev) if confidence is None else confidence
    if want_argmax and argmax is None:
        argmax = torch.empty(R, dtype=torch.int32, device=dev)
    if want_entropy and entropy is None:
        entropy = torch.empty(R, dtype=torch.float32, device=dev)
    for t, n, dtype in ((tau_per_row, "tau_per_row", torch.float32), (editable, "editable", torch.uint8),
                        (new_tokens, "new_tokens", torch.int32), (edit_mask, "edit_mask", torch.uint8),
                        (confidence, "confidence", torch.float32), (argmax, "argmax", torch.int32),
                        (entropy, "entropy", torch.float32)):
        if t is not None:
            _need(t, n, dtype)
            _shape(t, n, (R,))
    need = lm_head_workspace_size(R, V)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    _need(workspace, "workspace", torch.uint8)
    _same_device(dev, stream, weight=weight, committed=committed, tau_per_row=tau_per_row, editable=editable,
                 new_tokens=new_tokens, edit_mask=edit_mask, confidence=confidence, argmax=argmax, entropy=entropy,
                 workspace=workspace)
    st = lib().mbe_lm_head_edit_decide(_ptr(hidden), _ptr(weight), R, V, d, _ptr(committed), _ptr(tau_per_row),
                                       float(tau), _ptr(editable), _ptr(new_tokens), _ptr(edit_mask),
                                       _ptr(confidence), _ptr(argmax), _ptr(entropy), _ptr(workspace),
                                       workspace.numel(), _stream(stream))
    _check("mbe_lm_head_edit_decide", st)
    return new_tokens, edit_mask, confidence, argmax, entropy


def sft_block_mask(n_prompt_blocks, n_blocks, K, mask_rows, mask_words=None, out=None, stream=None):
    """mbe_sft_block_mask: see include/mbe.h. Returns uint32 bits as int32 [batch, mask_rows, mask_words]."""
    _need(n_prompt_blocks, "n_prompt_blocks", torch.int32)
    _need(n_blocks, "n_blocks", torch.int32)
    batch = n_blocks.numel()
    mask_words = mask_words or max(1, (mask_rows + 31) // 32)
    if out is None:
        out = torch.empty((batch, mask_rows, mask_words), dtype=torch.int32, device=n_blocks.device)
    _need(out, "out", torch.int32)
    _shape(n_prompt_blocks, "n_prompt_blocks", (batch,))
    _shape(out, "out", (batch, mask_rows, mask_words))
    _same_device(n_blocks.device, stream, n_prompt_blocks=n_prompt_blocks, out=out)
    st = lib().mbe_sft_block_mask(_ptr(n_prompt_blocks), _ptr(n_blocks), int(K), batch, mask_rows, mask_words,
                                  _ptr(out), _stream(stream))
    _check("mbe_sft_block_mask", st)
    return out


def _block_mask_shapes(q, k, v, seq_len, cu_seqlens, mask):
    """Shapes of a block-mask attention call (include/mbe.h): q [T, Hq, D], k and v
    [T, Hkv, D], mask [batch, mask_rows, mask_words], seq_len [batch], cu_seqlens
    [batch + 1]."""
    if q.dim() != 3 or k.dim() != 3 or mask.dim() != 3:
        raise ValueError("q must be [T, Hq, D], k and v [T, Hkv, D], mask [batch, rows, words]")
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    _shape(k, "k", (T, Hkv, D))
    _shape(v, "v", (T, Hkv, D))
    batch, mask_rows, mask_words = mask.shape
    _shape(seq_len, "seq_len", (batch,))
    _shape(cu_seqlens, "cu_seqlens", (batch + 1,))
    return T, Hq, D, Hkv, batch, mask_rows, mask_words


def block_mask_attention(q, k, v, seq_len, cu_seqlens, mask, *, block_size, max_seq_len, softmax_scale=0.0,
                         out=None, lse=None, return_lse=False, workspace=None, stream=None):
    """mbe_block_mask_attention: see include/mbe.h. mask: int32 (uint32 bits)
    [batch, mask_rows, mask_words]. Returns out (and lse if requested)."""
    for t, n in ((q, "q"), (k, "k"), (v, "v")):
        _need(t, n, torch.bfloat16)
    for t, n in ((seq_len, "seq_len"), (cu_seqlens, "cu_seqlens"), (mask, "mask")):
        _need(t, n, torch.int32)
    T, Hq, D, Hkv, batch, mask_rows, mask_words = _block_mask_shapes(q, k, v, seq_len, cu_seqlens, mask)
    if out is None:
        out = torch.empty_like(q)
    _need(out, "out", torch.bfloat16)
    _shape(out, "out", (T, Hq, D))
    if return_lse and lse is None:
        lse = torch.empty((T, Hq), dtype=torch.float32, device=q.device)
    if lse is not None:
        _need(lse, "lse", torch.float32)
        _shape(lse, "lse", (T, Hq))
    need = window_attention_workspace_size(batch, Hq, Hkv, D, max_seq_len, 0)
    if workspace is None:
        workspace = torch.empty(max(need, 1), dtype=torch.uint8, device=q.device)
    _need(workspace, "workspace", torch.uint8)
    _same_device(q.device, stream, k=k, v=v, seq_len=seq_len, cu_seqlens=cu_seqlens, mask=mask, out=out, lse=lse,
                 workspace=workspace)
    st = lib().mbe_block_mask_attention(_ptr(q), _ptr(k), _ptr(v), _ptr(seq_len), _ptr(cu_seqlens), _ptr(mask),
                                        mask_rows, mask_words, batch, T, Hq, Hkv, D, block_size, max_seq_len,
                                        float(softmax_scale), _ptr(out), _ptr(lse), _ptr(workspace), workspace.numel(),
                                        _stream(stream))
    _check("mbe_block_mask_attention", st)
    return (out, lse) if return_lse else out


def block_mask_attention_bwd(q, k, v, out, dout, lse, seq_len, cu_seqlens, mask, *, block_size, max_seq_len,
                             softmax_scale=0.0, dq=None, dk=None, dv=None, workspace=None, stream=None):
    """mbe_block_mask_attention_bwd: see include/mbe.h. Returns fp32 (dq, dk, dv)."""
    for t, n in ((q, "q"), (k, "k"), (v, "v"), (out, "out"), (dout, "dout")):
        _need(t, n, torch.bfloat16)
    _need(lse, "lse", torch.float32)
    for t, n in ((seq_len, "seq_len"), (cu_seqlens, "cu_seqlens"), (mask, "mask")):
        _need(t, n, torch.int32)
    T, Hq, D, Hkv, batch, mask_rows, mask_words = _block_mask_shapes(q, k, v, seq_len, cu_seqlens, mask)
    _shape(out, "out", (T, Hq, D))
    _shape(dout, "dout", (T, Hq, D))
    _shape(lse, "lse", (T, Hq))
    dev = q.device
    dq = torch.empty((T, Hq, D), dtype=torch.float32, device=dev) if dq is None else dq
    dk = torch.empty((T, Hkv, D), dtype=torch.float32, device=dev) if dk is None else dk
    dv = torch.empty((T, Hkv, D), dtype=torch.float32, device=dev) if dv is None else dv
    for t, n, shp in ((dq, "dq", (T, Hq, D)), (dk, "dk", (T, Hkv, D)), (dv, "dv", (T, Hkv, D))):
        _need(t, n, torch.float32)
        _shape(t, n, shp)
    need = int(lib().mbe_block_mask_attention_bwd_workspace_size(batch, T, Hq))
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    _need(workspace, "workspace", torch.uint8)
    _same_device(dev, stream, k=k, v=v, out=out, dout=dout, lse=lse, seq_len=seq_len, cu_seqlens=cu_seqlens,
                 mask=mask, dq=dq, dk=dk, dv=dv, workspace=workspace)
    st = lib().mbe_block_mask_attention_bwd(_ptr(q), _ptr(k), _ptr(v), _ptr(out), _ptr(dout), _ptr(lse),
                                            _ptr(seq_len), _ptr(cu_seqlens), _ptr(mask), mask_rows, mask_words, batch,
                                            T, Hq, Hkv, D, block_size, max_seq_len, float(softmax_scale), _ptr(dq),
                                            _ptr(dk), _ptr(dv), _ptr(workspace), workspace.numel(), _stream(stream))
    _check("mbe_block_mask_attention_bwd", st)
    return dq, dk, dv


def refresh_plan(block_changed, prefix_len, window_len, cu_window, block_table, *, block_size, max_window,
                 total_rows=None, out=None, stream=None):
    """mbe_refresh_plan: see include/mbe.h. Returns a dict of device tensors
    prefix_len, window_len, cu_window, mask_mode, block_table, src_row, count
    (reusing `out` when given, so that the call can be captured in a graph)."""
    _need(block_changed, "block_changed", torch.uint8)
    for t, n in ((prefix_len, "prefix_len"), (window_len, "window_len"), (cu_window, "cu_window"),
                 (block_table, "block_table")):
        _need(t, n, torch.int32)
    batch, max_blocks = block_changed.shape
    max_pages = block_table.shape[1]
    if block_table.shape[0] != batch or prefix_len.numel() != batch or window_len.numel() != batch or \
            cu_window.numel() != batch + 1:
        raise ValueError("block_changed, prefix_len, window_len, cu_window and block_table disagree on the batch")
    E = batch * max_blocks
    dev = block_changed.device
    if out is None:
        if total_rows is None:
            raise ValueError("total_rows (rows of the pass) is required when out is not given")
        out = {"prefix_len": torch.empty(E, dtype=torch.int32, device=dev),
               "window_len": torch.empty(E, dtype=torch.int32, device=dev),
               "cu_window": torch.empty(E + 1, dtype=torch.int32, device=dev),
               "mask_mode": torch.empty(E, dtype=torch.uint8, device=dev),
               "block_table": torch.empty((E, max_pages), dtype=torch.int32, device=dev),
               "src_row": torch.empty(int(total_rows), dtype=torch.int32, device=dev),
               "count": torch.empty(2, dtype=torch.int32, device=dev)}
    shapes = {"prefix_len": (E,), "window_len": (E,), "cu_window": (E + 1,), "mask_mode": (E,),
              "block_table": (E, max_pages), "count": (2,)}
    for k, shp in shapes.items():
        _need(out[k], k, torch.uint8 if k == "mask_mode" else torch.int32)
        if tuple(out[k].shape) != shp:
            raise ValueError(f"out[{k!r}] must have shape {shp}")
    _need(out["src_row"], "src_row", torch.int32)
    _same_device(dev, stream, prefix_len=prefix_len, window_len=window_len, cu_window=cu_window,
                 block_table=block_table, **{f"out_{k}": t for k, t in out.items()})
    st = lib().mbe_refresh_plan(_ptr(block_changed), max_blocks, _ptr(prefix_len), _ptr(window_len), _ptr(cu_window),
                                _ptr(block_table), max_pages, batch, block_size, max_window, out["src_row"].numel(),
                                _ptr(out["prefix_len"]), _ptr(out["window_len"]), _ptr(out["cu_window"]),
                                _ptr(out["mask_mode"]), _ptr(out["block_table"]), _ptr(out["src_row"]),
                                _ptr(out["count"]), _stream(stream))
    _check("mbe_refresh_plan", st)
    return out


def gather_rows(src, src_row, out=None, rows_used=None, stream=None):
    """mbe_gather_rows: out[k] = src[src_row[k]] (zero rows where src_row[k] < 0);
    with rows_used (a device int32 tensor, e.g. plan["count"][1:]) only rows
    k < rows_used[0] are written."""
    _need(src, "src", None)
    _need(src_row, "src_row", torch.int32)
    rows = src_row.numel()
    if out is None:
        out = torch.empty((rows,) + tuple(src.shape[1:]), dtype=src.dtype, device=src.device)
    _need(out, "out", src.dtype)
    if tuple(out.shape[1:]) != tuple(src.shape[1:]) or out.shape[0] != rows:
        raise ValueError("out must be [len(src_row)] + src.shape[1:]")
    row_bytes = (src[0].numel() if src.shape[0] else out[0].numel() if rows else 1) * src.element_size()
    if rows_used is not None:
        _need(rows_used, "rows_used", torch.int32)
    _same_device(src.device, stream, src_row=src_row, out=out, rows_used=rows_used)
    st = lib().mbe_gather_rows(_ptr(src), src.shape[0], row_bytes, _ptr(src_row), rows,
                               _ptr(rows_used) if rows_used is not None else None, _ptr(out), _stream(stream))
    _check("mbe_gather_rows", st)
    return out


def gather_rows_multi(pairs, src_row, rows_used=None, stream=None):
    """mbe_gather_rows_multi: out[k] = src[src_row[k]] for every (src, out) in
    `pairs` (at most 4 tensors with the same number of rows), one launch."""
    _need(src_row, "src_row", torch.int32)
    rows = src_row.numel()
    if not 1 <= len(pairs) <= 4:
        raise ValueError("gather_rows_multi takes 1 to 4 (src, out) pairs")
    src_rows = pairs[0][0].shape[0]
    srcs, dsts, nbytes = [], [], []
    for src, out in pairs:
        _need(src, "src", None)
        _need(out, "out", src.dtype)
        if src.shape[0] != src_rows:
            raise ValueError("every src must have the same number of rows")
        if tuple(out.shape[1:]) != tuple(src.shape[1:]) or out.shape[0] != rows:
            raise ValueError("out must be [len(src_row)] + src.shape[1:]")
        srcs.append(src.data_ptr())
        dsts.append(out.data_ptr())
        nbytes.append(max(1, (src[0].numel() if src_rows else out[0].numel() if rows else 1) * src.element_size()))
    if rows_used is not None:
        _need(rows_used, "rows_used", torch.int32)
    _same_device(src_row.device, stream, rows_used=rows_used,
                 **{f"{k}{i}": t for i, (a, b) in enumerate(pairs) for k, t in (("src", a), ("out", b))})
    n = len(pairs)
    c_src = (ctypes.c_void_p * n)(*srcs)
    c_dst = (ctypes.c_void_p * n)(*dsts)
    c_bytes = (ctypes.c_int64 * n)(*nbytes)
    st = lib().mbe_gather_rows_multi(n, c_src, c_bytes, c_dst, src_rows, _ptr(src_row), rows,
                                     _ptr(rows_used) if rows_used is not None else None, _stream(stream))
    _check("mbe_gather_rows_multi", st)
    return [out for _, out in pairs]


def refresh_gather_write(q, k_win, v_win, plan, k_cache, v_cache, *, out, stream=None):
    """mbe_refresh_gather_write: compacts the refresh rows of `plan` (as returned
    by refresh_plan) from q / k_win / v_win into out = (q_out, k_out, v_out) and
    writes their K/V into k_cache / v_cache at the refresh-layout positions."""
    q_out, k_out, v_out = out
    for t, n in ((q, "q"), (k_win, "k_win"), (v_win, "v_win"), (k_cache, "k_cache"), (v_cache, "v_cache"),
                 (q_out, "q_out"), (k_out, "k_out"), (v_out, "v_out")):
        _need(t, n, torch.bfloat16)
    if q.dim() != 3 or k_win.dim() != 3 or k_cache.dim() != 4:
        raise ValueError("q must be [rows, Hq, D], k_win and v_win [rows, Hkv, D], the caches [pages, Hkv, page, D]")
    src_rows, Hq, D = q.shape
    Hkv = k_win.shape[1]
    _shape(k_win, "k_win", (src_rows, Hkv, D))
    _shape(v_win, "v_win", (src_rows, Hkv, D))
    num_pages, _, page_size, _ = k_cache.shape
    _shape(k_cache, "k_cache", (num_pages, Hkv, page_size, D))
    _shape(v_cache, "v_cache", (num_pages, Hkv, page_size, D))
    rows = plan["src_row"].numel()
    if q_out.shape[0] < rows or k_out.shape[0] < rows or v_out.shape[0] < rows:
        raise ValueError("the outputs must hold every refresh row of the plan")
    if tuple(q_out.shape[1:]) != (Hq, D) or tuple(k_out.shape[1:]) != (Hkv, D) or tuple(v_out.shape[1:]) != (Hkv, D):
        raise ValueError("q_out must be [rows, Hq, D] and k_out, v_out [rows, Hkv, D]")
    E, max_pages = plan["block_table"].shape
    _same_device(q.device, stream, k_win=k_win, v_win=v_win, k_cache=k_cache, v_cache=v_cache, q_out=q_out,
                 k_out=k_out, v_out=v_out, **{f"plan_{k}": t for k, t in plan.items()})
    st = lib().mbe_refresh_gather_write(_ptr(q), _ptr(k_win), _ptr(v_win), src_rows, Hq, Hkv, D, _ptr(plan["src_row"]),
                                        _ptr(plan["count"][1:]), rows, _ptr(plan["prefix_len"]),
                                        _ptr(plan["cu_window"]), _ptr(plan["block_table"]), E, max_pages,
                                        _ptr(k_cache), _ptr(v_cache), num_pages, page_size, _ptr(q_out),
                                        _ptr(k_out), _ptr(v_out), _stream(stream))
    _check("mbe_refresh_gather_write", st)
    return out


class PassLoop:
    """mbe_pass_loop_*: see include/mbe.h. Usage::

        loop = PassLoop(max_passes, passes_done, stream)   # starts capturing `stream`
        with torch.cuda.stream(stream):
            ...one pass: library calls on `stream` with preallocated buffers...
        loop.until_stable(seq_changes)
        loop.end()
        loop.launch()          # all passes, one graph launch
        loop.close()
    """

    def __init__(self, max_passes, passes_done, stream):
        _need(passes_done, "passes_done", torch.int32)
        if stream is None or stream.cuda_stream == 0:
            raise ValueError("the pass loop needs a non-default stream")
        self.stream = stream
        self._h = ctypes.c_void_p(None)
        st = lib().mbe_pass_loop_begin(int(max_passes), _ptr(passes_done), _stream(stream), ctypes.byref(self._h))
        _check("mbe_pass_loop_begin", st)

    def until_stable(self, seq_changes):
        _need(seq_changes, "seq_changes", torch.int32)
        st = lib().mbe_pass_loop_until_stable(self._h, _ptr(seq_changes), seq_changes.numel(), _stream(self.stream))
        _check("mbe_pass_loop_until_stable", st)

    def end(self):
        _check("mbe_pass_loop_end", lib().mbe_pass_loop_end(self._h, _stream(self.stream)))

    def launch(self, stream=None):
        _check("mbe_pass_loop_launch", lib().mbe_pass_loop_launch(self._h, _stream(stream or self.stream)))

    def close(self):
        if self._h:
            lib().mbe_pass_loop_destroy(self._h)
            self._h = ctypes.c_void_p(None)

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def get_device_error(stream=None):
    """(status, flag bits) of the device error word; clears it."""
    flags = ctypes.c_uint32(0)
    st = lib().mbe_get_device_error(_stream(stream), ctypes.byref(flags))
    return st, flags.value


def set_wait_limit_ns(limit_ns: int) -> int:
    """Sets the limit of the kernels' bounded waits (mbe_set_wait_limit_ns);
    returns the previous limit."""
    return int(lib().mbe_set_wait_limit_ns(int(limit_ns)))


def window_attention_plan_stats(workspace, stream=None):
    """(work units, split-KV merge groups) of the plan held in `workspace`."""
    _need(workspace, "workspace", torch.uint8)
    n_units, n_groups = ctypes.c_int32(0), ctypes.c_int32(0)
    _check("mbe_window_attention_plan_stats",
           lib().mbe_window_attention_plan_stats(_ptr(workspace), workspace.numel(), ctypes.byref(n_units),
                                                 ctypes.byref(n_groups), _stream(stream)))
    return n_units.value, n_groups.value
