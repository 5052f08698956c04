"""The C ABI without a GPU: the library loads, exports every function that
include/sparsecoder.h declares, and rejects bad arguments on the host before
anything is launched (so these calls never reach the device)."""
import ctypes
import os
import re

import pytest

from paper_2310_07109_gb300 import binding as bd
from paper_2310_07109_gb300 import build as bld

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "sparsecoder.h")


@pytest.fixture(scope="module")
def lib():
    bld.build_library()
    return bd.load()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:size_t|int|void|const char\*)\s+(sc_\w+)\s*\(", text,
                                 re.M)))


def test_header_declares_the_documented_calls():
    names = declared_functions()
    assert set(bd.EXPORTED) <= set(names)
    assert "sc_layer_forward" in names and "sc_stack_forward" in names


def test_binding_constants_match_the_header():
    text = open(HEADER).read()
    defines = dict(re.findall(r"^#define\s+(SC_\w+)\s+(\d+)", text, re.M))
    assert int(defines["SC_TAIL_MAX_LEN"]) == bd.TAIL_MAX_LEN
    assert int(defines["SC_STACK_NO_TAIL"]) == bd.SC_STACK_NO_TAIL
    assert int(defines["SC_MAX_WINDOW"]) == bd.SC_MAX_WINDOW
    rules = dict(re.findall(r"^\s*(SC_KEEP_\w+)\s*=\s*(\d+)", text, re.M))
    assert {k: int(v) for k, v in rules.items()} == {
        "SC_KEEP_RELATIVE": bd.SC_KEEP_RELATIVE, "SC_KEEP_ABSOLUTE": bd.SC_KEEP_ABSOLUTE,
        "SC_KEEP_TOP_RATIO": bd.SC_KEEP_TOP_RATIO}


def test_every_declared_symbol_is_exported(lib):
    raw = ctypes.CDLL(bd.library_path())
    for name in declared_functions():
        assert hasattr(raw, name), name


def test_status_strings(lib):
    for code in range(6):
        assert bd.status_string(code).startswith("SC_")
    assert "unknown" in bd.status_string(99)


def test_workspace_size(lib):
    assert bd.workspace_size(2, 4096, 12) > 2 * 12 * 4096 * 8
    assert bd.workspace_size(0, 10, 1) == 0
    assert bd.workspace_size(1, 4097, 1) == 0
    assert bd.workspace_size(1, 1, 1) % 256 == 0


FAKE = 1 << 40  # host-side validation never dereferences device pointers


def _layer_args(**kw):
    g = (ctypes.c_int32 * 2)(0, 5)
    a = dict(B=1, L=256, H=12, w=64, Q=FAKE, K=FAKE, V=FAKE, len=FAKE, pos=FAKE,
             global_pos=ctypes.cast(g, ctypes.POINTER(ctypes.c_int32)), n_global=2, alpha=0.5,
             theta=None, O=FAKE, scores=FAKE, pos_out=FAKE + 4096, len_out=FAKE + 8192)
    a.update(kw)
    return bd.LayerArgs(**a), g


def _call_layer(lib, ws=FAKE, ws_bytes=1 << 30, **kw):
    a, keep = _layer_args(**kw)
    return lib.sc_layer_forward(ctypes.byref(a), ctypes.c_void_p(ws), ws_bytes, None)


def test_layer_rejects_bad_arguments(lib):
    assert lib.sc_layer_forward(None, None, 0, None) == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, Q=None) == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, B=0) == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, w=-1) == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, L=5000) == bd.SC_ERR_UNSUPPORTED
    assert _call_layer(lib, L=2048, w=513) == bd.SC_ERR_UNSUPPORTED
    assert _call_layer(lib, n_global=17) == bd.SC_ERR_UNSUPPORTED
    assert _call_layer(lib, Q=FAKE + 8) == bd.SC_ERR_INVALID_ARG        # not 16-byte aligned
    assert _call_layer(lib, pos_out=FAKE) == bd.SC_ERR_INVALID_ARG      # aliases pos
    assert _call_layer(lib, ws=None) == bd.SC_ERR_WORKSPACE
    assert _call_layer(lib, ws_bytes=16) == bd.SC_ERR_WORKSPACE
    assert _call_layer(lib, ws=FAKE + 128) == bd.SC_ERR_WORKSPACE       # not 256-byte aligned
    bad = (ctypes.c_int32 * 2)(5, 0)                                      # unsorted
    assert _call_layer(lib, global_pos=ctypes.cast(bad, ctypes.POINTER(ctypes.c_int32))) \
        == bd.SC_ERR_INVALID_ARG
    dup = (ctypes.c_int32 * 2)(3, 3)
    assert _call_layer(lib, global_pos=ctypes.cast(dup, ctypes.POINTER(ctypes.c_int32))) \
        == bd.SC_ERR_INVALID_ARG
    far = (ctypes.c_int32 * 2)(0, 256)                                    # outside [0, L)
    assert _call_layer(lib, global_pos=ctypes.cast(far, ctypes.POINTER(ctypes.c_int32))) \
        == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, keep_rule=3) == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, keep_rule=-1) == bd.SC_ERR_INVALID_ARG
    # the top-ratio rule takes no per-sequence thresholds and a finite ratio
    assert _call_layer(lib, keep_rule=bd.SC_KEEP_TOP_RATIO, theta=FAKE) == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, keep_rule=bd.SC_KEEP_TOP_RATIO, alpha=float("nan")) \
        == bd.SC_ERR_INVALID_ARG
    assert _call_layer(lib, keep_rule=bd.SC_KEEP_TOP_RATIO, alpha=float("inf")) \
        == bd.SC_ERR_INVALID_ARG


def test_stack_rejects_bad_arguments(lib):
    g = (ctypes.c_int32 * 1)(0)
    al = (ctypes.c_float * 12)(*([0.5] * 12))

    def call(**kw):
        a = dict(n_layers=12, B=2, L=1024, H=12, w=256, Q=FAKE, K=FAKE, V=FAKE, pad_mask=None,
                 global_pos=ctypes.cast(g, ctypes.POINTER(ctypes.c_int32)), n_global=1,
                 alpha=ctypes.cast(al, ctypes.POINTER(ctypes.c_float)), O=FAKE, scores=FAKE,
                 pos=FAKE, len=FAKE)
        a.update(kw)
        return lib.sc_stack_forward(ctypes.byref(bd.StackArgs(**a)), ctypes.c_void_p(FAKE),
                                    1 << 30, None)

    assert call(n_layers=0) == bd.SC_ERR_INVALID_ARG
    assert call(alpha=None) == bd.SC_ERR_INVALID_ARG
    assert call(scores=None) == bd.SC_ERR_INVALID_ARG
    assert call(V=FAKE + 2) == bd.SC_ERR_INVALID_ARG
    # O == NULL is a valid request (only the last layer's O, to O_last, or none);
    # a misaligned O_last is refused before anything runs
    assert call(O=None, O_last=FAKE + 2) == bd.SC_ERR_INVALID_ARG
    assert call(L=8192) == bd.SC_ERR_UNSUPPORTED
    assert call(w=513) == bd.SC_ERR_UNSUPPORTED
    assert call(flags=4) == bd.SC_ERR_INVALID_ARG   # bits 0 and 1 are the two flags
    assert call(keep_rule=7) == bd.SC_ERR_INVALID_ARG
    bad = (ctypes.c_float * 12)(*([0.5] * 11 + [float("nan")]))
    assert call(keep_rule=bd.SC_KEEP_TOP_RATIO,
                alpha=ctypes.cast(bad, ctypes.POINTER(ctypes.c_float))) == bd.SC_ERR_INVALID_ARG


def test_stack_host_rejects_bad_arguments(lib):
    """The host-buffer stack checks its sizes, its workspace and that every host
    range is page-locked memory mapped for the device before anything runs."""
    g = (ctypes.c_int32 * 1)(0)
    al = (ctypes.c_float * 2)(0.5, 0.5)
    nl, B, L, H = 2, 2, 256, 2
    n_qkv = nl * B * L * H * 64
    plain = {k: (ctypes.c_uint16 * n_qkv)() for k in ("Q", "K", "V", "O")}
    small = {"scores": (ctypes.c_float * (nl * B * L))(), "pos": (ctypes.c_int32 * ((nl + 1) * B * L))(),
             "len": (ctypes.c_int32 * ((nl + 1) * B))()}
    bufs = {k: ctypes.addressof(v) for k, v in {**plain, **small}.items()}
    need = bd.stack_host_workspace_size(nl, B, L, H)

    def call(ws_bytes=need, **kw):
        a = dict(n_layers=nl, B=B, L=L, H=H, w=64, pad_mask=None,
                 global_pos=ctypes.cast(g, ctypes.POINTER(ctypes.c_int32)), n_global=1,
                 alpha=ctypes.cast(al, ctypes.POINTER(ctypes.c_float)), **bufs)
        a.update(kw)
        return lib.sc_stack_forward_host(ctypes.byref(bd.StackArgs(**a)), ctypes.c_void_p(FAKE),
                                         ws_bytes, None)

    assert lib.sc_stack_forward_host(None, None, 0, None) == bd.SC_ERR_INVALID_ARG
    assert call(n_layers=0) == bd.SC_ERR_INVALID_ARG
    assert call(Q=None) == bd.SC_ERR_INVALID_ARG
    assert call(L=8192) == bd.SC_ERR_UNSUPPORTED
    assert call(flags=4) == bd.SC_ERR_INVALID_ARG   # bits 0 and 1 are the two flags
    assert call(ws_bytes=need - 256) == bd.SC_ERR_WORKSPACE
    # ordinary (pageable) host memory is refused: the kernels could not reach it
    assert call() == bd.SC_ERR_INVALID_ARG


def test_stack_host_workspace_size(lib):
    nl, B, L, H = 12, 2, 4096, 12
    base = bd.workspace_size(B, L, H)
    results = nl * B * L * (H * 64 * 2 + 4) + (nl + 1) * B * (L + 1) * 4
    n = bd.stack_host_workspace_size(nl, B, L, H)
    assert base + results <= n <= base + results + 5 * 256 and n % 256 == 0
    assert bd.stack_host_workspace_size(0, B, L, H) == 0
    assert bd.stack_host_workspace_size(nl, B, 4097, H) == 0


def test_launch_count_rejects_bad_arguments(lib):
    g = (ctypes.c_int32 * 1)(0)

    def count(fn, **kw):
        a = dict(n_layers=12, B=2, L=1024, H=12, w=256, Q=None, K=None, V=None, pad_mask=None,
                 global_pos=ctypes.cast(g, ctypes.POINTER(ctypes.c_int32)), n_global=1,
                 alpha=None, O=None, scores=None, pos=None, len=None)
        a.update(kw)
        c = ctypes.c_int(-1)
        return fn(ctypes.byref(bd.StackArgs(**a)), ctypes.byref(c))

    for fn in (lib.sc_stack_launch_count, lib.sc_stack_host_launch_count):
        assert count(n_layers=0, fn=fn) == bd.SC_ERR_INVALID_ARG
        assert count(flags=4, fn=fn) == bd.SC_ERR_INVALID_ARG
        assert count(L=8192, fn=fn) == bd.SC_ERR_UNSUPPORTED
        assert count(B=0, fn=fn) == bd.SC_ERR_INVALID_ARG
        assert fn(None, None) == bd.SC_ERR_INVALID_ARG


def test_encoder_calls_reject_bad_arguments(lib):
    assert lib.sc_encoder_layer_forward(None, None, 0, None) == bd.SC_ERR_INVALID_ARG
    a = bd.EncoderArgs()
    a.B, a.L, a.H, a.w = 1, 256, 11, 64          # odd head count: D not a multiple of 128
    assert lib.sc_encoder_layer_forward(ctypes.byref(a), ctypes.c_void_p(FAKE), 1 << 30,
                                        None) == bd.SC_ERR_UNSUPPORTED
    a.H = 12                                     # null pointers
    assert lib.sc_encoder_layer_forward(ctypes.byref(a), ctypes.c_void_p(FAKE), 1 << 30,
                                        None) == bd.SC_ERR_INVALID_ARG
    assert bd.encoder_workspace_size(2, 1024, 12) > bd.workspace_size(2, 1024, 12)
    assert bd.encoder_workspace_size(2, 1024, 11) == 0
    lin = bd.LinearArgs(1, 128, 100, 64, FAKE, None, None, FAKE, None, 0, None, 0, FAKE, 0)
    assert lib.sc_linear_forward(ctypes.byref(lin), ctypes.c_void_p(FAKE), 256,
                                 None) == bd.SC_ERR_INVALID_ARG   # N not a multiple of 128
    lin.N, lin.K = 128, 96
    assert lib.sc_linear_forward(ctypes.byref(lin), ctypes.c_void_p(FAKE), 256,
                                 None) == bd.SC_ERR_INVALID_ARG   # K not a multiple of 64
    lin.K = 64
    assert lib.sc_linear_forward(ctypes.byref(lin), ctypes.c_void_p(FAKE), 16,
                                 None) == bd.SC_ERR_WORKSPACE
    assert lib.sc_layer_norm_forward(1, 1, 100, None, ctypes.c_void_p(FAKE), ctypes.c_void_p(FAKE),
                                     ctypes.c_void_p(FAKE), ctypes.c_float(1e-5),
                                     ctypes.c_void_p(FAKE), None) == bd.SC_ERR_INVALID_ARG
