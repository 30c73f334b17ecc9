"""GB300 (sm_103a) library for the hot path of Multi-Block Editing (MBE).

The compute runs in ``libmbe.so`` (CUDA kernels behind the C ABI declared in
``include/mbe.h``); ``paper_2607_22663_gb300.mbe`` is its thin Python binding.
"""
from .mbe import (BLOCK_CAUSAL, MULTI_BLOCK_BIDIRECTIONAL, MbeError, edit_decide, get_device_error,  # noqa: F401
                  kv_window_write, window_attention, window_attention_workspace_size)
