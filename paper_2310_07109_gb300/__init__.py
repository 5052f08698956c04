"""SparseCoder hot path on GB300 (sm_103a): Longformer-style sparse attention
fused with learned token pruning, behind the C ABI of include/sparsecoder.h.

The Python surface is a thin ctypes binding (``binding``); the arithmetic runs
in ``libsparsecoder.so`` (``csrc/``), built in-tree by ``build.build_library``.
"""
from .binding import (ENCODER_WEIGHTS, SC_ERR_CUDA, SC_ERR_INVALID_ARG, SC_ERR_TIMEOUT,
                      SC_ERR_UNSUPPORTED, SC_ERR_WORKSPACE, SC_KEEP_ABSOLUTE, SC_KEEP_RELATIVE,
                      SC_KEEP_TOP_RATIO, SC_OK, SC_ROWS_SINGLE_PASS, SC_ROWS_TWO_PASS,
                      SC_STACK_NO_TAIL, SC_STACK_PLAIN_LAUNCHES, TAIL_MAX_LEN, SparseCoderError,
                      debug_graph_counts, debug_stall_waits, encoder_layer_forward,
                      encoder_workspace_size,
                      layer_forward, layer_forward_noalloc, layer_noalloc_status,
                      layer_norm_forward, linear_forward, load, new_encoder_workspace,
                      new_host_outputs, new_stack_host_workspace, new_workspace,
                      select_rows_kernel, stack_forward,
                      stack_forward_host, stack_host_workspace_size, stack_launch_count,
                      status_string, workspace_size, workspace_status)

__all__ = ["ENCODER_WEIGHTS", "SC_ERR_CUDA", "SC_ERR_INVALID_ARG", "SC_ERR_TIMEOUT",
           "SC_ERR_UNSUPPORTED", "SC_ERR_WORKSPACE", "SC_KEEP_ABSOLUTE", "SC_KEEP_RELATIVE",
           "SC_KEEP_TOP_RATIO", "SC_OK", "SC_ROWS_SINGLE_PASS", "SC_ROWS_TWO_PASS", "SC_STACK_NO_TAIL", "SC_STACK_PLAIN_LAUNCHES", "TAIL_MAX_LEN", "SparseCoderError",
           "debug_graph_counts", "debug_stall_waits", "encoder_layer_forward", "encoder_workspace_size",
           "layer_forward", "layer_forward_noalloc", "layer_noalloc_status",
           "layer_norm_forward", "linear_forward", "load", "new_encoder_workspace",
           "new_host_outputs", "new_stack_host_workspace", "new_workspace", "select_rows_kernel",
           "stack_forward",
           "stack_forward_host", "stack_host_workspace_size", "stack_launch_count",
           "status_string", "workspace_size", "workspace_status"]
