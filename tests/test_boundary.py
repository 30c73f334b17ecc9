"""The C-ABI library loads and exports every symbol include/mbe.h declares;
host-side argument checks return their status without touching the GPU."""
import ctypes
import re

import pytest

from paper_2607_22663_gb300 import mbe


def test_every_declared_symbol_is_exported():
    L = mbe.lib()
    names = mbe.declared_symbols()
    assert set(names) >= {"mbe_window_attention", "mbe_window_attention_workspace_size", "mbe_edit_decide",
                          "mbe_kv_window_write", "mbe_get_device_error", "mbe_status_string", "mbe_version"}
    for n in names:
        assert hasattr(L, n), n


def test_status_strings_and_version():
    L = mbe.lib()
    for code in range(7):
        assert L.mbe_status_string(code)
    assert L.mbe_status_string(99) == b"unknown status"
    assert L.mbe_version() >= 100


def test_header_enums_match_binding():
    text = mbe.HEADER.read_text()
    for name, val in (("MBE_OK", 0), ("MBE_ERR_INVALID_ARG", 1), ("MBE_ERR_UNSUPPORTED", 2), ("MBE_ERR_CUDA", 3),
                      ("MBE_ERR_TIMEOUT", 4), ("MBE_ERR_WORKSPACE", 5), ("MBE_ERR_DEVICE_CHECK", 6)):
        assert re.search(rf"\b{name}\s*=\s*{val}\b", text), name
        assert mbe.STATUS_NAMES[val] == name
    for name, val in (("MBE_DEVERR_TIMEOUT", mbe.DEVERR_TIMEOUT), ("MBE_DEVERR_LENGTH", mbe.DEVERR_LENGTH),
                      ("MBE_DEVERR_PAGE", mbe.DEVERR_PAGE), ("MBE_DEVERR_CAPACITY", mbe.DEVERR_CAPACITY),
                      ("MBE_DEVERR_PLAN", mbe.DEVERR_PLAN)):
        m = re.search(rf"#define {name} (0x[0-9a-fA-F]+)u", text)
        assert m and int(m.group(1), 16) == val, name


def _attn_args(**over):
    # a well-formed call except for what `over` changes; pointers are fake but
    # every rejected case returns before any pointer is used
    a = dict(q=16, k_win=16, v_win=16, k_cache=16, v_cache=16, num_pages=4, block_table=16, max_pages=4, prefix=16,
             window=16, cu=16, mode=16, batch=1, T=64, Hq=4, Hkv=1, D=128, B=32, ps=32, max_window=64, max_prefix=64,
             scale=0.0, out=16, lse=None, ws=None, ws_bytes=0)
    a.update(over)
    return a


def _call_attn(a):
    L = mbe.lib()
    P = lambda v: None if v is None else ctypes.c_void_p(v)
    return L.mbe_window_attention(P(a["q"]), P(a["k_win"]), P(a["v_win"]), P(a["k_cache"]), P(a["v_cache"]),
                                  a["num_pages"], P(a["block_table"]), a["max_pages"], P(a["prefix"]), P(a["window"]),
                                  P(a["cu"]), P(a["mode"]), a["batch"], a["T"], a["Hq"], a["Hkv"], a["D"], a["B"],
                                  a["ps"], a["max_window"], a["max_prefix"], a["scale"], P(a["out"]), P(a["lse"]),
                                  P(a["ws"]), a["ws_bytes"], None)


@pytest.mark.parametrize("over,status", [
    (dict(Hq=6, Hkv=4), 1),            # heads not divisible
    (dict(D=96), 2),                   # head_dim unsupported
    (dict(Hq=12, Hkv=4), 2),           # group of 3 heads: not a power of two
    (dict(ps=24), 2),                  # page size not a power of two
    (dict(ps=4), 2),                   # page size below 8
    (dict(B=0), 1),                    # block size
    (dict(max_pages=1), 1),            # block table too narrow for max_prefix
    (dict(scale=-1.0), 1),             # negative scale
    (dict(batch=-1), 1),
    (dict(q=None), 1),                 # null pointer
    (dict(q=8), 1),                    # misaligned pointer
])
def test_attention_host_validation(over, status):
    assert _call_attn(_attn_args(**over)) == status


def test_attention_empty_batch_is_noop():
    assert _call_attn(_attn_args(batch=0, q=None, out=None)) == 0
    assert _call_attn(_attn_args(T=0)) == 0


def test_edit_decide_host_validation():
    L = mbe.lib()
    f = L.mbe_edit_decide
    P = ctypes.c_void_p
    assert f(P(16), 1, 100, 4, 0, P(16), None, 0.0, None, P(16), P(16), P(16), None, None) == 1   # vocab 0
    assert f(P(16), 1, 10, 4, 100, P(16), None, 0.0, None, P(16), P(16), P(16), None, None) == 1  # stride < vocab
    assert f(P(16), 7, 100, 4, 100, P(16), None, 0.0, None, P(16), P(16), P(16), None, None) == 1  # bad dtype
    assert f(None, 1, 100, 4, 100, P(16), None, 0.0, None, P(16), P(16), P(16), None, None) == 1   # null logits
    assert f(None, 1, 100, 0, 100, None, None, 0.0, None, None, None, None, None, None) == 0       # zero rows


def test_kv_write_host_validation():
    L = mbe.lib()
    f = L.mbe_kv_window_write
    P = ctypes.c_void_p
    ok = dict(kw=16, vw=16, kc=16, vc=16, npg=4, bt=16, maxp=4, pre=16, win=16, cu=16, mask=None, maxb=0, batch=1,
              maxw=32, hkv=1, d=128, b=32, ps=32)

    def call(**o):
        a = {**ok, **o}
        g = lambda v: None if v is None else P(v)
        return f(g(a["kw"]), g(a["vw"]), g(a["kc"]), g(a["vc"]), a["npg"], g(a["bt"]), a["maxp"], g(a["pre"]),
                 g(a["win"]), g(a["cu"]), g(a["mask"]), a["maxb"], a["batch"], a["maxw"], a["hkv"], a["d"], a["b"],
                 a["ps"], None)
    assert call(d=12) == 1               # head_dim not a multiple of 8
    assert call(kc=None) == 1
    assert call(kw=24) == 1              # misaligned
    assert call(mask=16, maxb=0) == 1    # mask narrower than the window's blocks
    assert call(batch=0) == 0


def test_workspace_size_rejects_bad_shapes():
    L = mbe.lib()
    assert L.mbe_window_attention_workspace_size(1, 6, 4, 128, 64, 64) == 0
    assert L.mbe_window_attention_workspace_size(1, 4, 1, 96, 64, 64) == 0


def test_attention_plan_host_validation():
    L = mbe.lib()
    P = ctypes.c_void_p
    f = L.mbe_window_attention_plan
    # null length array; a zero batch is a no-op
    assert f(None, P(16), P(16), P(16), 1, 64, 4, 1, 128, 32, 64, 64, P(16), 1 << 20, None) == 1
    assert f(None, None, None, None, 0, 0, 4, 1, 128, 32, 64, 64, None, 0, None) == 0
    assert f(P(16), P(16), P(16), P(16), 1, 64, 6, 4, 128, 32, 64, 64, P(16), 1 << 20, None) == 1   # heads


def test_denoise_and_tail_entropy_host_validation():
    L = mbe.lib()
    P = ctypes.c_void_p
    d = L.mbe_denoise_update
    ok = [P(16), 1, 100, 100, P(16), 1, 8, 4, 2, P(16), 9, 0.5, 0.0, None, P(32), P(16), P(16), P(16), None, None, None,
          None]
    bad = list(ok); bad[3] = 0          # vocab 0
    assert d(*bad) == 1
    bad = list(ok); bad[14] = P(16)     # new_tokens aliases tokens
    assert d(*bad) == 1
    bad = list(ok); bad[9] = None       # null tokens
    assert d(*bad) == 1
    zero = list(ok); zero[5] = 0        # no sequences: nothing to do
    assert d(*zero) == 0
    t = L.mbe_tail_entropy_select
    assert t(P(16), P(16), 2, 3, 32, 0.0, 4, None, P(16), P(16), None) == 1     # rho 0
    assert t(P(16), P(16), 2, 3, 32, 1.5, 4, None, P(16), P(16), None) == 1     # rho > 1
    assert t(P(16), P(16), 2, 3, 32, 0.25, 0, None, P(16), P(16), None) == 1    # k_max 0
    assert t(P(16), P(16), 2, 3, 20000, 0.25, 4, None, P(16), P(16), None) == 2  # block too large
    assert t(None, None, 0, 3, 32, 0.25, 4, None, None, None, None) == 0
