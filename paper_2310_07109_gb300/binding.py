"""ctypes binding of ``libsparsecoder.so`` (include/sparsecoder.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  PyTorch provides device memory and the current stream.  There is no
CPU fallback: if the library cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

_lock = threading.Lock()
_lib = None

SC_HEAD_DIM = 64
SC_MAX_LEN = 4096
SC_MAX_GLOBAL = 16
SC_MAX_WINDOW = 512

SC_OK, SC_ERR_INVALID_ARG, SC_ERR_UNSUPPORTED, SC_ERR_CUDA, SC_ERR_TIMEOUT, SC_ERR_WORKSPACE = range(6)


class SparseCoderError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(msg)
        self.code = code


class LayerArgs(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("L", ctypes.c_int), ("H", ctypes.c_int), ("w", ctypes.c_int),
                ("Q", ctypes.c_void_p), ("K", ctypes.c_void_p), ("V", ctypes.c_void_p),
                ("len", ctypes.c_void_p), ("pos", ctypes.c_void_p),
                ("global_pos", ctypes.POINTER(ctypes.c_int32)), ("n_global", ctypes.c_int),
                ("alpha", ctypes.c_float), ("theta", ctypes.c_void_p),
                ("O", ctypes.c_void_p), ("scores", ctypes.c_void_p),
                ("pos_out", ctypes.c_void_p), ("len_out", ctypes.c_void_p),
                ("keep_rule", ctypes.c_int)]


class StackArgs(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("B", ctypes.c_int), ("L", ctypes.c_int),
                ("H", ctypes.c_int), ("w", ctypes.c_int),
                ("Q", ctypes.c_void_p), ("K", ctypes.c_void_p), ("V", ctypes.c_void_p),
                ("pad_mask", ctypes.c_void_p),
                ("global_pos", ctypes.POINTER(ctypes.c_int32)), ("n_global", ctypes.c_int),
                ("alpha", ctypes.POINTER(ctypes.c_float)),
                ("O", ctypes.c_void_p), ("scores", ctypes.c_void_p),
                ("pos", ctypes.c_void_p), ("len", ctypes.c_void_p), ("flags", ctypes.c_int),
                ("keep_rule", ctypes.c_int), ("O_last", ctypes.c_void_p)]


class EncoderArgs(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("L", ctypes.c_int), ("H", ctypes.c_int), ("w", ctypes.c_int),
                ("X", ctypes.c_void_p), ("len", ctypes.c_void_p), ("pos", ctypes.c_void_p),
                ("global_pos", ctypes.POINTER(ctypes.c_int32)), ("n_global", ctypes.c_int),
                ("keep_rule", ctypes.c_int), ("alpha", ctypes.c_float), ("theta", ctypes.c_void_p),
                ("W_qkv", ctypes.c_void_p), ("b_qkv", ctypes.c_void_p),
                ("W_o", ctypes.c_void_p), ("b_o", ctypes.c_void_p),
                ("ln1_gamma", ctypes.c_void_p), ("ln1_beta", ctypes.c_void_p),
                ("W_1", ctypes.c_void_p), ("b_1", ctypes.c_void_p),
                ("W_2", ctypes.c_void_p), ("b_2", ctypes.c_void_p),
                ("ln2_gamma", ctypes.c_void_p), ("ln2_beta", ctypes.c_void_p),
                ("Y", ctypes.c_void_p), ("O", ctypes.c_void_p), ("scores", ctypes.c_void_p),
                ("pos_out", ctypes.c_void_p), ("len_out", ctypes.c_void_p)]


class LinearArgs(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("L", ctypes.c_int), ("N", ctypes.c_int), ("K", ctypes.c_int),
                ("A", ctypes.c_void_p), ("rows", ctypes.c_void_p), ("gidx", ctypes.c_void_p),
                ("W", ctypes.c_void_p), ("bias", ctypes.c_void_p), ("gelu", ctypes.c_int),
                ("res", ctypes.c_void_p), ("res_gathered", ctypes.c_int),
                ("out", ctypes.c_void_p), ("out_f32", ctypes.c_int)]


SC_STACK_NO_TAIL = 1
SC_STACK_PLAIN_LAUNCHES = 2
# keep rules (sc_keep_rule): what a layer's value alpha means
SC_KEEP_RELATIVE = 0   # theta = alpha / n
SC_KEEP_ABSOLUTE = 1   # theta = alpha
SC_KEEP_TOP_RATIO = 2  # keep ceil(alpha n) tokens: the first and the best others
# sequences with at most this many current tokens finish in the cluster kernel
# (SC_TAIL_MAX_LEN of include/sparsecoder.h)
TAIL_MAX_LEN = 384

EXPORTED = ["sc_layer_forward", "sc_layer_forward_noalloc", "sc_stack_forward",
            "sc_stack_forward_profiled", "sc_stack_launch_count", "sc_stack_forward_host",
            "sc_stack_host_workspace_size", "sc_stack_host_launch_count",
            "sc_workspace_size", "sc_workspace_status", "sc_status_string", "sc_last_error",
            "sc_encoder_layer_forward", "sc_encoder_workspace_size", "sc_linear_forward",
            "sc_layer_norm_forward", "sc_layer_noalloc_status", "sc_debug_stall_waits",
            "sc_select_rows_kernel", "sc_debug_graph_counts"]


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = False):
    """Load the CUDA library (optionally building it first); raise if unavailable."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if build_if_missing and not os.path.exists(path):
            _build.build_library()
        if not os.path.exists(path):
            raise RuntimeError(
                "libsparsecoder.so is not built (run __graft_entry__.build() or "
                "python -m paper_2310_07109_gb300.build); there is no fallback path")
        lib = ctypes.CDLL(path)
        lib.sc_workspace_size.restype = ctypes.c_size_t
        lib.sc_workspace_size.argtypes = [ctypes.c_int] * 3
        lib.sc_layer_forward.restype = ctypes.c_int
        lib.sc_layer_forward.argtypes = [ctypes.POINTER(LayerArgs), ctypes.c_void_p,
                                         ctypes.c_size_t, ctypes.c_void_p]
        lib.sc_stack_forward.restype = ctypes.c_int
        lib.sc_stack_forward.argtypes = [ctypes.POINTER(StackArgs), ctypes.c_void_p,
                                         ctypes.c_size_t, ctypes.c_void_p]
        lib.sc_layer_forward_noalloc.restype = ctypes.c_int
        lib.sc_layer_forward_noalloc.argtypes = [ctypes.POINTER(LayerArgs), ctypes.c_void_p]
        lib.sc_layer_noalloc_status.restype = ctypes.c_int
        lib.sc_layer_noalloc_status.argtypes = [ctypes.c_void_p]
        lib.sc_debug_stall_waits.restype = None
        lib.sc_debug_stall_waits.argtypes = [ctypes.c_ulonglong]
        lib.sc_debug_graph_counts.restype = None
        lib.sc_debug_graph_counts.argtypes = [ctypes.POINTER(ctypes.c_ulonglong),
                                              ctypes.POINTER(ctypes.c_ulonglong)]
        lib.sc_select_rows_kernel.restype = ctypes.c_int
        lib.sc_select_rows_kernel.argtypes = [ctypes.c_int]
        lib.sc_stack_forward_profiled.restype = ctypes.c_int
        lib.sc_stack_forward_profiled.argtypes = [ctypes.POINTER(StackArgs), ctypes.c_void_p,
                                                  ctypes.c_size_t, ctypes.c_void_p,
                                                  ctypes.POINTER(ctypes.c_void_p), ctypes.c_int]
        lib.sc_stack_launch_count.restype = ctypes.c_int
        lib.sc_stack_launch_count.argtypes = [ctypes.POINTER(StackArgs),
                                              ctypes.POINTER(ctypes.c_int)]
        lib.sc_stack_host_workspace_size.restype = ctypes.c_size_t
        lib.sc_stack_host_workspace_size.argtypes = [ctypes.c_int] * 4
        lib.sc_stack_forward_host.restype = ctypes.c_int
        lib.sc_stack_forward_host.argtypes = [ctypes.POINTER(StackArgs), ctypes.c_void_p,
                                              ctypes.c_size_t, ctypes.c_void_p]
        lib.sc_stack_host_launch_count.restype = ctypes.c_int
        lib.sc_stack_host_launch_count.argtypes = [ctypes.POINTER(StackArgs),
                                                   ctypes.POINTER(ctypes.c_int)]
        lib.sc_workspace_status.restype = ctypes.c_int
        lib.sc_workspace_status.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
        lib.sc_status_string.restype = ctypes.c_char_p
        lib.sc_status_string.argtypes = [ctypes.c_int]
        lib.sc_last_error.restype = ctypes.c_char_p
        lib.sc_last_error.argtypes = []
        lib.sc_encoder_workspace_size.restype = ctypes.c_size_t
        lib.sc_encoder_workspace_size.argtypes = [ctypes.c_int] * 3
        lib.sc_encoder_layer_forward.restype = ctypes.c_int
        lib.sc_encoder_layer_forward.argtypes = [ctypes.POINTER(EncoderArgs), ctypes.c_void_p,
                                                 ctypes.c_size_t, ctypes.c_void_p]
        lib.sc_linear_forward.restype = ctypes.c_int
        lib.sc_linear_forward.argtypes = [ctypes.POINTER(LinearArgs), ctypes.c_void_p,
                                          ctypes.c_size_t, ctypes.c_void_p]
        lib.sc_layer_norm_forward.restype = ctypes.c_int
        lib.sc_layer_norm_forward.argtypes = [ctypes.c_int] * 3 + [ctypes.c_void_p] * 4 + [
            ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p]
        _lib = lib
        return lib


def status_string(code: int) -> str:
    return load().sc_status_string(int(code)).decode()


def _check(code: int):
    if code != SC_OK:
        msg = status_string(code)
        if code == SC_ERR_CUDA:
            msg += " (" + load().sc_last_error().decode() + ")"
        raise SparseCoderError(code, msg)


def workspace_size(B: int, L: int, H: int) -> int:
    return int(load().sc_workspace_size(int(B), int(L), int(H)))


def new_workspace(B: int, L: int, H: int, device=None) -> torch.Tensor:
    n = workspace_size(B, L, H)
    if n == 0:
        raise SparseCoderError(SC_ERR_INVALID_ARG, "invalid workspace sizes")
    ws = torch.zeros(n + 256, dtype=torch.uint8, device=device or "cuda")
    off = (-ws.data_ptr()) % 256
    return ws[off:off + n]


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream_handle(stream):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _int32_host(values):
    vals = [int(v) for v in values]
    arr = (ctypes.c_int32 * max(1, len(vals)))(*vals)
    return arr, len(vals)


def layer_forward(Q, K, V, length, pos, w, global_pos, alpha=0.0, theta=None, *, O=None,
                  scores=None, pos_out=None, len_out=None, workspace=None, stream=None,
                  keep_rule=SC_KEEP_RELATIVE):
    """One layer on current-order inputs (``sc_layer_forward``).

    Q, K, V: bf16 [B, L, H, 64] cuda tensors; length: int32 [B]; pos: int32 [B, L].
    keep_rule: an SC_KEEP_* value saying what ``alpha`` is.
    Returns (O, scores, pos_out, len_out).
    """
    B, L, H, D = Q.shape
    dev = Q.device
    O = O if O is not None else torch.empty((B, L, H, D), dtype=torch.bfloat16, device=dev)
    scores = scores if scores is not None else torch.empty((B, L), dtype=torch.float32, device=dev)
    pos_out = pos_out if pos_out is not None else torch.empty((B, L), dtype=torch.int32, device=dev)
    len_out = len_out if len_out is not None else torch.empty((B,), dtype=torch.int32, device=dev)
    ws = workspace if workspace is not None else new_workspace(B, L, H, dev)
    garr, ng = _int32_host(global_pos)
    a = LayerArgs(B, L, H, int(w), _ptr(Q), _ptr(K), _ptr(V), _ptr(length), _ptr(pos),
                  ctypes.cast(garr, ctypes.POINTER(ctypes.c_int32)), ng, float(alpha),
                  _ptr(theta), _ptr(O), _ptr(scores), _ptr(pos_out), _ptr(len_out),
                  int(keep_rule))
    _check(load().sc_layer_forward(ctypes.byref(a), _ptr(ws), ws.numel(), _stream_handle(stream)))
    return O, scores, pos_out, len_out


def layer_forward_noalloc(Q, K, V, length, pos, w, global_pos, alpha=0.0, theta=None, *, O,
                          scores, pos_out, len_out, stream=None, keep_rule=SC_KEEP_RELATIVE):
    """One layer through ``sc_layer_forward_noalloc``: no device memory is
    allocated, by this call or the library; every output tensor is passed in."""
    B, L, H, D = Q.shape
    garr, ng = _int32_host(global_pos)
    a = LayerArgs(B, L, H, int(w), _ptr(Q), _ptr(K), _ptr(V), _ptr(length), _ptr(pos),
                  ctypes.cast(garr, ctypes.POINTER(ctypes.c_int32)), ng, float(alpha),
                  _ptr(theta), _ptr(O), _ptr(scores), _ptr(pos_out), _ptr(len_out),
                  int(keep_rule))
    _check(load().sc_layer_forward_noalloc(ctypes.byref(a), _stream_handle(stream)))
    return O, scores, pos_out, len_out


def layer_noalloc_status(stream=None) -> int:
    """Synchronise and return (then clear) the status of the no-allocation calls."""
    return int(load().sc_layer_noalloc_status(_stream_handle(stream)))


SC_ROWS_SINGLE_PASS = 0
SC_ROWS_TWO_PASS = 1


def select_rows_kernel(which: int) -> None:
    """``sc_select_rows_kernel``: SC_ROWS_TWO_PASS (default) or SC_ROWS_SINGLE_PASS."""
    _check(load().sc_select_rows_kernel(int(which)))


def debug_stall_waits(ns: int) -> None:
    """Test hook (``sc_debug_stall_waits``): while ns > 0 every per-layer
    attention CTA waits on a barrier nothing completes for at most ns ns and
    aborts; 0 turns it off."""
    load().sc_debug_stall_waits(int(ns))


def debug_graph_counts():
    """Test hook (``sc_debug_graph_counts``): (stack calls recorded into a new
    graph, stack calls that launched a kept graph) since the library was loaded."""
    rec, reu = ctypes.c_ulonglong(0), ctypes.c_ulonglong(0)
    load().sc_debug_graph_counts(ctypes.byref(rec), ctypes.byref(reu))
    return int(rec.value), int(reu.value)


def _stack_flags(no_tail, plain_launches):
    return (SC_STACK_NO_TAIL if no_tail else 0) | (SC_STACK_PLAIN_LAUNCHES if plain_launches else 0)


def stack_forward(Q, K, V, pad_mask, global_pos, w, alpha, *, out=None, workspace=None,
                  stream=None, events=None, no_tail=False, keep_rule=SC_KEEP_RELATIVE,
                  o_last_only=False, plain_launches=False):
    """The pruned layer stack (``sc_stack_forward``).

    Q, K, V: bf16 [n_layers, B, L, H, 64] cuda tensors in original-position order;
    pad_mask: uint8 [B, L] cuda tensor or None; alpha: host sequence [n_layers],
    the value of the keep rule ``keep_rule`` (an SC_KEEP_* value) per layer.
    events: optional list of >= 3 + 3 * n_layers torch.cuda.Event(enable_timing=True)
    or None (nothing recorded at that point), recorded around the kernels on the
    launching stream (sc_stack_forward_profiled).
    no_tail: run every layer through the per-layer kernels (SC_STACK_NO_TAIL).
    plain_launches: launch the kernels directly even when not capturing
    (SC_STACK_PLAIN_LAUNCHES) instead of through the library's cached graph.
    o_last_only: write no O but the last layer's, to out["O_last"] [B, L, H, 64]
    (O = NULL in the arguments).
    Returns a dict with O (or O_last), scores, pos, len (device tensors).
    """
    nl, B, L, H, D = Q.shape
    dev = Q.device
    if out is None:
        out = {"scores": torch.empty((nl, B, L), dtype=torch.float32, device=dev),
               "pos": torch.empty((nl + 1, B, L), dtype=torch.int32, device=dev),
               "len": torch.empty((nl + 1, B), dtype=torch.int32, device=dev)}
        if o_last_only:
            out["O_last"] = torch.empty((B, L, H, D), dtype=torch.bfloat16, device=dev)
        else:
            out["O"] = torch.empty((nl, B, L, H, D), dtype=torch.bfloat16, device=dev)
    ws = workspace if workspace is not None else new_workspace(B, L, H, dev)
    garr, ng = _int32_host(global_pos)
    al = (ctypes.c_float * nl)(*[float(x) for x in alpha])
    a = StackArgs(nl, B, L, H, int(w), _ptr(Q), _ptr(K), _ptr(V), _ptr(pad_mask),
                  ctypes.cast(garr, ctypes.POINTER(ctypes.c_int32)), ng,
                  ctypes.cast(al, ctypes.POINTER(ctypes.c_float)),
                  _ptr(out.get("O")), _ptr(out["scores"]), _ptr(out["pos"]), _ptr(out["len"]),
                  _stack_flags(no_tail, plain_launches), int(keep_rule), _ptr(out.get("O_last")))
    if events is None:
        _check(load().sc_stack_forward(ctypes.byref(a), _ptr(ws), ws.numel(),
                                       _stream_handle(stream)))
    else:
        handles = (ctypes.c_void_p * len(events))(
            *[None if e is None else e.cuda_event for e in events])
        _check(load().sc_stack_forward_profiled(ctypes.byref(a), _ptr(ws), ws.numel(),
                                                _stream_handle(stream), handles, len(events)))
    return out


def stack_launch_count(n_layers, B, L, H, w, global_pos, has_pad_mask, no_tail=False,
                       host=False) -> int:
    """Kernels one ``stack_forward`` (``host``: ``stack_forward_host``) call launches for
    these sizes on the current device."""
    garr, ng = _int32_host(global_pos)
    # only whether pad_mask is NULL matters: a non-null marker is never dereferenced
    a = StackArgs(int(n_layers), int(B), int(L), int(H), int(w), None, None, None,
                  16 if has_pad_mask else None,
                  ctypes.cast(garr, ctypes.POINTER(ctypes.c_int32)), ng, None, None, None,
                  None, None, SC_STACK_NO_TAIL if no_tail else 0)
    cnt = ctypes.c_int(0)
    fn = load().sc_stack_host_launch_count if host else load().sc_stack_launch_count
    _check(fn(ctypes.byref(a), ctypes.byref(cnt)))
    return int(cnt.value)


def stack_host_workspace_size(n_layers, B, L, H) -> int:
    return int(load().sc_stack_host_workspace_size(int(n_layers), int(B), int(L), int(H)))


def new_stack_host_workspace(n_layers, B, L, H, device=None) -> torch.Tensor:
    n = stack_host_workspace_size(n_layers, B, L, H)
    if n == 0:
        raise SparseCoderError(SC_ERR_INVALID_ARG, "invalid workspace sizes")
    ws = torch.zeros(n + 256, dtype=torch.uint8, device=device or "cuda")
    off = (-ws.data_ptr()) % 256
    return ws[off:off + n]


def new_host_outputs(n_layers, B, L, H, o_last_only=False):
    """Page-locked host result tensors for ``stack_forward_host`` (``o_last_only``:
    the last layer's O alone, as "O_last")."""
    out = {"scores": torch.empty((n_layers, B, L), dtype=torch.float32, pin_memory=True),
           "pos": torch.empty((n_layers + 1, B, L), dtype=torch.int32, pin_memory=True),
           "len": torch.empty((n_layers + 1, B), dtype=torch.int32, pin_memory=True)}
    if o_last_only:
        out["O_last"] = torch.empty((B, L, H, 64), dtype=torch.bfloat16, pin_memory=True)
    else:
        out["O"] = torch.empty((n_layers, B, L, H, 64), dtype=torch.bfloat16, pin_memory=True)
    return out


def stack_forward_host(Q, K, V, pad_mask, global_pos, w, alpha, *, out=None, workspace=None,
                       stream=None, no_tail=False, keep_rule=SC_KEEP_RELATIVE,
                       plain_launches=False):
    """The pruned stack on host tensors (``sc_stack_forward_host``).

    Q, K, V: bf16 [n_layers, B, L, H, 64] page-locked CPU tensors (``pin_memory()``);
    pad_mask: uint8 [B, L] page-locked CPU tensor or None; the other arguments as for
    ``stack_forward``.  ``out``: page-locked result tensors (``new_host_outputs``);
    only the current slots of each layer (and all of ``len``) are written; with
    "O_last" in place of "O", only the last layer's O.
    The call is asynchronous on ``stream`` (default: torch's current stream of the
    current device): synchronise before reading ``out``.  The first call on newly
    page-locked buffers is slower (milliseconds) while the device maps their pages;
    reuse the buffers across calls.
    Returns the dict of host tensors O, scores, pos, len.
    """
    nl, B, L, H, D = Q.shape
    for name, t in (("Q", Q), ("K", K), ("V", V), ("pad_mask", pad_mask)):
        if t is not None and (t.device.type != "cpu" or not t.is_pinned()):
            raise SparseCoderError(SC_ERR_INVALID_ARG, name + " must be a page-locked CPU tensor")
    if out is None:
        out = new_host_outputs(nl, B, L, H)
    ws = workspace if workspace is not None else new_stack_host_workspace(nl, B, L, H)
    garr, ng = _int32_host(global_pos)
    al = (ctypes.c_float * nl)(*[float(x) for x in alpha])
    a = StackArgs(nl, B, L, H, int(w), _ptr(Q), _ptr(K), _ptr(V), _ptr(pad_mask),
                  ctypes.cast(garr, ctypes.POINTER(ctypes.c_int32)), ng,
                  ctypes.cast(al, ctypes.POINTER(ctypes.c_float)),
                  _ptr(out.get("O")), _ptr(out["scores"]), _ptr(out["pos"]), _ptr(out["len"]),
                  _stack_flags(no_tail, plain_launches), int(keep_rule), _ptr(out.get("O_last")))
    _check(load().sc_stack_forward_host(ctypes.byref(a), _ptr(ws), ws.numel(),
                                        _stream_handle(stream)))
    return out


def workspace_status(workspace, stream=None) -> int:
    """Synchronise and return (then clear) the workspace status code."""
    return int(load().sc_workspace_status(_ptr(workspace), workspace.numel(),
                                          _stream_handle(stream)))


# ---------------------------------------------------------------------------
# the encoder layer around the path
# ---------------------------------------------------------------------------
ENCODER_WEIGHTS = ("W_qkv", "b_qkv", "W_o", "b_o", "ln1_gamma", "ln1_beta", "W_1", "b_1",
                   "W_2", "b_2", "ln2_gamma", "ln2_beta")


def encoder_workspace_size(B, L, H) -> int:
    return int(load().sc_encoder_workspace_size(int(B), int(L), int(H)))


def new_encoder_workspace(B, L, H, device=None):
    n = encoder_workspace_size(B, L, H)
    if n == 0:
        raise SparseCoderError(SC_ERR_INVALID_ARG, "invalid encoder sizes")
    ws = torch.zeros(n + 256, dtype=torch.uint8, device=device or "cuda")
    off = (-ws.data_ptr()) % 256
    return ws[off:off + n]


def encoder_layer_forward(X, length, pos, w, global_pos, weights, alpha=0.0, theta=None, *,
                          keep_rule=SC_KEEP_RELATIVE, out=None, workspace=None, stream=None):
    """One encoder layer (``sc_encoder_layer_forward``): X bf16 [B, L, D] current order,
    length int32 [B], pos int32 [B, L]; ``weights`` maps ENCODER_WEIGHTS to cuda tensors
    (bf16 matrices [out, in], fp32 vectors).  Returns dict(Y, O, scores, pos_out, len_out)."""
    B, L, D = X.shape
    H = D // 64
    dev = X.device
    if out is None:
        out = {"Y": torch.empty((B, L, D), dtype=torch.bfloat16, device=dev),
               "O": torch.empty((B, L, D), dtype=torch.bfloat16, device=dev),
               "scores": torch.empty((B, L), dtype=torch.float32, device=dev),
               "pos_out": torch.empty((B, L), dtype=torch.int32, device=dev),
               "len_out": torch.empty((B,), dtype=torch.int32, device=dev)}
    ws = workspace if workspace is not None else new_encoder_workspace(B, L, H, dev)
    garr, ng = _int32_host(global_pos)
    a = EncoderArgs(B, L, H, int(w), _ptr(X), _ptr(length), _ptr(pos),
                    ctypes.cast(garr, ctypes.POINTER(ctypes.c_int32)), ng, int(keep_rule),
                    float(alpha), _ptr(theta), *[_ptr(weights[k]) for k in ENCODER_WEIGHTS],
                    _ptr(out["Y"]), _ptr(out["O"]), _ptr(out["scores"]), _ptr(out["pos_out"]),
                    _ptr(out["len_out"]))
    _check(load().sc_encoder_layer_forward(ctypes.byref(a), _ptr(ws), ws.numel(),
                                           _stream_handle(stream)))
    return out


def linear_forward(A, W, *, B, L, rows=None, gidx=None, bias=None, gelu=False, res=None,
                   res_gathered=False, out=None, out_f32=False, workspace=None, stream=None):
    """``sc_linear_forward``: A bf16 [B*L, K] (any leading shape), W bf16 [N, K]."""
    N, K = W.shape
    if out is None:
        out = torch.empty((B * L, N), dtype=torch.float32 if out_f32 else torch.bfloat16,
                          device=A.device)
    ws = workspace if workspace is not None else new_workspace(1, 1, 1, A.device)
    a = LinearArgs(int(B), int(L), int(N), int(K), _ptr(A), _ptr(rows), _ptr(gidx), _ptr(W),
                   _ptr(bias), int(bool(gelu)), _ptr(res), int(bool(res_gathered)), _ptr(out),
                   int(bool(out_f32)))
    _check(load().sc_linear_forward(ctypes.byref(a), _ptr(ws), ws.numel(), _stream_handle(stream)))
    return out


def layer_norm_forward(x, gamma, beta, *, B, L, rows=None, eps=1e-5, out=None, stream=None):
    """``sc_layer_norm_forward``: x fp32 [B*L, D] -> bf16."""
    D = x.shape[-1]
    if out is None:
        out = torch.empty((B * L, D), dtype=torch.bfloat16, device=x.device)
    _check(load().sc_layer_norm_forward(int(B), int(L), int(D), _ptr(rows), _ptr(x), _ptr(gamma),
                                        _ptr(beta), ctypes.c_float(eps), _ptr(out),
                                        _stream_handle(stream)))
    return out
