import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built libmbe")


def pytest_collection_modifyitems(config, items):
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for it in items:
        if "gpu" in it.keywords:
            it.add_marker(skip)


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Attention parity, relative to each compared pair's output RMS."""
    try:
        from tests._gpu import ATTN_REPORT
    except Exception:
        return
    if not ATTN_REPORT:
        return
    terminalreporter.write_sep("-", "attention parity: worst |err| / output RMS, worst err / bar (tests/_bars.py)")
    for name, rel, bar in ATTN_REPORT:
        terminalreporter.write_line(f"{rel:8.4f}  {bar:6.3f}  {name}")
