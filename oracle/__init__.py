"""Plain fp64 CPU oracle for SparseCoder's sparse attention + learned token pruning.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may use this module.  The CUDA library never
imports it, and it imports nothing from the CUDA package.

The arithmetic lives in ``sc_oracle.c`` (plain C, double precision, loops over
the paper's definitions).  This module only builds it with gcc when the shared
object is missing or older than the source, and marshals numpy arrays.

Functions
---------
layer(Q, K, V, is_global, w, theta)          one layer, every output
layer_sampled(Q, K, V, is_global, w, rows, cols)
                                             O rows / scores of chosen rows/cols
stack(Q, K, V, pad_mask, global_pos, w, alpha, keep_rule)
                                             the pruned layer stack (bf16 bits in)
top_count(rho, n), keep_top(scores, k)       the top-ratio keep rule

oracle.encoder: the rest of the encoder layer around the path (projections,
layer norms, GELU), float64 numpy.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sc_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

_dp = ctypes.POINTER(ctypes.c_double)
_ip = ctypes.POINTER(ctypes.c_int)
_u16p = ctypes.POINTER(ctypes.c_uint16)
_u8p = ctypes.POINTER(ctypes.c_uint8)


def build(force: bool = False) -> str:
    """Compile ``sc_oracle.c`` into ``liboracle.so`` next to it (gcc, -O2, no fast-math)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".%d.tmp" % os.getpid()
    cmd = ["gcc", "-O2", "-fPIC", "-shared", "-pthread", "-std=c11",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            lib.sco_layer.restype = ctypes.c_int
            lib.sco_layer.argtypes = [ctypes.c_int] * 4 + [_dp] * 3 + [
                _ip, ctypes.c_double, _dp, _dp, _ip, ctypes.c_int]
            lib.sco_layer_sampled.restype = ctypes.c_int
            lib.sco_layer_sampled.argtypes = [ctypes.c_int] * 4 + [_dp] * 3 + [
                _ip, _ip, ctypes.c_int, _dp, _ip, ctypes.c_int, _dp]
            lib.sco_stack.restype = ctypes.c_int
            lib.sco_stack.argtypes = [ctypes.c_int] * 6 + [_u16p] * 3 + [
                _u8p, _ip, ctypes.c_int, _dp, ctypes.c_int, _dp, _dp, _ip, _ip,
                ctypes.c_int]
            lib.sco_top_count.restype = ctypes.c_int
            lib.sco_top_count.argtypes = [ctypes.c_double, ctypes.c_int]
            lib.sco_keep_top.restype = ctypes.c_int
            lib.sco_keep_top.argtypes = [ctypes.c_int, _dp, ctypes.c_int, _ip]
            _lib = lib
    return _lib


def default_threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:  # pragma: no cover
        return max(1, os.cpu_count() or 1)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def layer(Q, K, V, is_global, w, theta, nthreads=None):
    """One layer on current-order inputs.

    Q, K, V: float64 [n, H, d]; is_global: [n] bool/int; theta: absolute threshold.
    Returns (O [n,H,d] float64, scores [n] float64, keep [n] bool).
    """
    Q, K, V = _c(Q, np.float64), _c(K, np.float64), _c(V, np.float64)
    n, H, d = Q.shape
    assert K.shape == Q.shape and V.shape == Q.shape
    g = _c(np.asarray(is_global).astype(np.int32), np.int32)
    O = np.zeros((n, H, d), np.float64)
    s = np.zeros(max(n, 1), np.float64)
    keep = np.zeros(max(n, 1), np.int32)
    lib = _load()
    r = lib.sco_layer(n, H, d, int(w), Q.ctypes.data_as(_dp), K.ctypes.data_as(_dp),
                      V.ctypes.data_as(_dp), g.ctypes.data_as(_ip), float(theta),
                      O.ctypes.data_as(_dp), s.ctypes.data_as(_dp),
                      keep.ctypes.data_as(_ip), int(nthreads or default_threads()))
    if r < 0:
        raise ValueError("oracle layer rejected its arguments")
    return O, s[:n], keep[:n].astype(bool)


# keep rules of the stack (the value per layer is alpha_l, theta_l or rho_l)
KEEP_RELATIVE = 0   # theta = alpha_l / n_l
KEEP_ABSOLUTE = 1   # theta = theta_l
KEEP_TOP_RATIO = 2  # k = ceil(rho_l n_l) tokens: the first and the k-1 best others


def top_count(rho, n):
    """k = ceil(rho * n) clamped to 1..n (0 for n = 0); rho is taken as the
    float32 value a caller of the library passes."""
    return int(_load().sco_top_count(float(np.float32(rho)), int(n)))


def keep_top(scores, k):
    """keep mask of the top-ratio rule for ``k`` kept tokens (token 0 always)."""
    s = _c(np.asarray(scores, dtype=np.float64).reshape(-1), np.float64)
    keep = np.zeros(max(len(s), 1), np.int32)
    if _load().sco_keep_top(len(s), s.ctypes.data_as(_dp), int(k), keep.ctypes.data_as(_ip)) < 0:
        raise ValueError("oracle keep_top rejected its arguments")
    return keep[:len(s)].astype(bool)


def layer_sampled(Q, K, V, is_global, w, rows=(), cols=()):
    """O rows for ``rows`` ([len(rows), H, d]) and scores for ``cols`` ([len(cols)])."""
    Q, K, V = _c(Q, np.float64), _c(K, np.float64), _c(V, np.float64)
    n, H, d = Q.shape
    g = _c(np.asarray(is_global).astype(np.int32), np.int32)
    rows = _c(np.asarray(rows, dtype=np.int32).reshape(-1), np.int32)
    cols = _c(np.asarray(cols, dtype=np.int32).reshape(-1), np.int32)
    O = np.zeros((max(len(rows), 1), H, d), np.float64)
    s = np.zeros(max(len(cols), 1), np.float64)
    lib = _load()
    r = lib.sco_layer_sampled(n, H, d, int(w), Q.ctypes.data_as(_dp),
                              K.ctypes.data_as(_dp), V.ctypes.data_as(_dp),
                              g.ctypes.data_as(_ip), rows.ctypes.data_as(_ip),
                              len(rows), O.ctypes.data_as(_dp),
                              cols.ctypes.data_as(_ip), len(cols),
                              s.ctypes.data_as(_dp))
    if r < 0:
        raise ValueError("oracle sampled layer rejected its arguments")
    return O[:len(rows)], s[:len(cols)]


def stack(Q, K, V, pad_mask, global_pos, w, alpha, want_O=True, nthreads=None,
          keep_rule=KEEP_RELATIVE):
    """The pruned layer stack.

    Q, K, V: bf16 bit patterns (uint16) [n_layers, B, L, H, d], original order.
    pad_mask: uint8/bool [B, L] (1 = real token) or None.
    global_pos: sorted original positions of the global tokens.
    alpha: [n_layers], the keep rule's value per layer: theta_l = alpha_l / n_l
    per sequence (KEEP_RELATIVE), theta_l = alpha_l (KEEP_ABSOLUTE), or the
    kept ratio rho_l = alpha_l (KEEP_TOP_RATIO; taken as float32, as the
    library receives it).
    Returns dict with O ([nl,B,L,H,d] float64 or None), scores ([nl,B,L]),
    pos ([nl+1,B,L] int32), len ([nl+1,B] int32).  Slots at or past the
    current length hold -1 (pos) / NaN (scores, O).
    """
    Q, K, V = _c(Q, np.uint16), _c(K, np.uint16), _c(V, np.uint16)
    nl, B, L, H, d = Q.shape
    assert K.shape == Q.shape and V.shape == Q.shape
    alpha = _c(np.asarray(alpha, dtype=np.float64).reshape(-1), np.float64)
    assert alpha.shape[0] == nl
    if keep_rule == KEEP_TOP_RATIO:
        alpha = alpha.astype(np.float32).astype(np.float64)
    gp = _c(np.asarray(global_pos, dtype=np.int32).reshape(-1), np.int32)
    mask = None if pad_mask is None else _c(np.asarray(pad_mask).astype(np.uint8), np.uint8)
    O = np.full((nl, B, L, H, d), np.nan) if want_O else None
    scores = np.full((nl, B, L), np.nan)
    pos = np.full((nl + 1, B, L), -1, np.int32)
    lens = np.zeros((nl + 1, B), np.int32)
    lib = _load()
    r = lib.sco_stack(nl, B, L, H, d, int(w), Q.ctypes.data_as(_u16p),
                      K.ctypes.data_as(_u16p), V.ctypes.data_as(_u16p),
                      None if mask is None else mask.ctypes.data_as(_u8p),
                      gp.ctypes.data_as(_ip), len(gp), alpha.ctypes.data_as(_dp),
                      int(keep_rule), None if O is None else O.ctypes.data_as(_dp),
                      scores.ctypes.data_as(_dp), pos.ctypes.data_as(_ip),
                      lens.ctypes.data_as(_ip), int(nthreads or default_threads()))
    if r < 0:
        raise ValueError("oracle stack rejected its arguments")
    return {"O": O, "scores": scores, "pos": pos, "len": lens}
