"""SparseCoder hot path on GB300 (sm_103a): Longformer-style sparse attention
fused with learned token pruning, behind the C ABI of include/sparsecoder.h.

The Python surface is a thin ctypes binding (``binding``); the arithmetic runs
in ``libsparsecoder.so`` (``csrc/``), built in-tree by ``build.build_library``.
"""
from .binding import (ENCODER_WEIGHTS, SC_KEEP_ABSOLUTE, SC_KEEP_RELATIVE, SC_KEEP_TOP_RATIO,
                      TAIL_MAX_LEN, SparseCoderError, encoder_layer_forward,
                      encoder_workspace_size, layer_forward, layer_norm_forward, linear_forward,
                      load, new_encoder_workspace, new_host_outputs, new_stack_host_workspace,
                      new_workspace, stack_forward, stack_forward_host,
                      stack_host_workspace_size, stack_launch_count, status_string,
                      workspace_size, workspace_status)

__all__ = ["ENCODER_WEIGHTS", "SC_KEEP_ABSOLUTE", "SC_KEEP_RELATIVE", "SC_KEEP_TOP_RATIO",
           "TAIL_MAX_LEN", "SparseCoderError", "encoder_layer_forward", "encoder_workspace_size",
           "layer_forward", "layer_norm_forward", "linear_forward", "load",
           "new_encoder_workspace", "new_host_outputs", "new_stack_host_workspace",
           "new_workspace", "stack_forward", "stack_forward_host", "stack_host_workspace_size",
           "stack_launch_count",
           "status_string", "workspace_size", "workspace_status"]
