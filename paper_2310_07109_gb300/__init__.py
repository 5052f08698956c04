"""SparseCoder hot path on GB300 (sm_103a): Longformer-style sparse attention
fused with learned token pruning, behind the C ABI of include/sparsecoder.h.

The Python surface is a thin ctypes binding (``binding``); the arithmetic runs
in ``libsparsecoder.so`` (``csrc/``), built in-tree by ``build.build_library``.
"""
from .binding import (SC_KEEP_ABSOLUTE, SC_KEEP_RELATIVE, SC_KEEP_TOP_RATIO, TAIL_MAX_LEN,
                      SparseCoderError, layer_forward, load, new_workspace, stack_forward,
                      stack_launch_count, status_string, workspace_size, workspace_status)

__all__ = ["SC_KEEP_ABSOLUTE", "SC_KEEP_RELATIVE", "SC_KEEP_TOP_RATIO", "TAIL_MAX_LEN",
           "SparseCoderError", "layer_forward", "load", "new_workspace", "stack_forward",
           "stack_launch_count", "status_string", "workspace_size", "workspace_status"]
