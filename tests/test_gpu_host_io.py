"""GPU parity of the stack with host inputs and results (sc_stack_forward_host).

The kernels read the surviving tokens' rows straight from page-locked host
memory and write back only the current slots of each layer.  Checked against
the fp64 oracle (kept lists exactly, O and scores within the stated
tolerances), against the device-memory entry point on the same inputs (the
same kernels on the same values: every defined result bit for bit), for the result
slots it must leave alone, and replayed from a CUDA graph.
"""
import numpy as np
import pytest
import torch

import workloads as wk
from parity_utils import bits_to_torch, check_stack, resample_stack, torch_bf16_to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    return sc


def _host_inputs(inp):
    qkv = [torch.from_numpy(np.ascontiguousarray(inp[k]).view(np.int16)).view(torch.bfloat16)
           .pin_memory() for k in ("Q", "K", "V")]
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).pin_memory()
    return qkv, mask


def _sentinel_outputs(sc, wl):
    out = sc.new_host_outputs(wl.n_layers, wl.B, wl.L, wl.H)
    out["O"].view(torch.int16).fill_(-1)          # bf16 NaN pattern 0xFFFF
    out["scores"].fill_(float("nan"))
    out["pos"].fill_(-7)
    out["len"].fill_(-7)
    return out


def _run_host(sc, wl, inp, no_tail=False, out=None):
    (Q, K, V), mask = _host_inputs(inp)
    out = out if out is not None else _sentinel_outputs(sc, wl)
    ws = sc.new_stack_host_workspace(wl.n_layers, wl.B, wl.L, wl.H)
    sc.stack_forward_host(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"], out=out,
                          workspace=ws, no_tail=no_tail, keep_rule=wl.keep_rule)
    assert sc.workspace_status(ws) == 0
    return out


def _run_device(sc, wl, inp, no_tail=False):
    Q, K, V = (bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V"))
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).cuda()
    ws = sc.new_workspace(wl.B, wl.L, wl.H)
    out = sc.stack_forward(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"], workspace=ws,
                           no_tail=no_tail, keep_rule=wl.keep_rule)
    assert sc.workspace_status(ws) == 0
    return {k: v.cpu() for k, v in out.items()}


def _numpy(out):
    return {"O": torch_bf16_to_f64(out["O"]), "scores": out["scores"].numpy(),
            "pos": out["pos"].numpy(), "len": out["len"].numpy()}


def _assert_same_defined_slots(wl, a, b, global_pos=None):
    """Every result the stack defines bit for bit, the global tokens' O rows
    included (their parts over key blocks are added in a fixed order)."""
    assert torch.equal(a["len"], b["len"])
    lens = a["len"].numpy()
    for l in range(wl.n_layers + 1):
        for s in range(wl.B):
            n = int(lens[l, s])
            assert torch.equal(a["pos"][l, s, :n], b["pos"][l, s, :n]), (l, s)
            if l < wl.n_layers and n:
                assert torch.equal(a["scores"][l, s, :n].view(torch.int32),
                                   b["scores"][l, s, :n].view(torch.int32)), (l, s)
                assert torch.equal(a["O"][l, s, :n].view(torch.int16),
                                   b["O"][l, s, :n].view(torch.int16)), (l, s)


def _assert_rest_untouched(wl, out):
    lens = out["len"].numpy()
    for l in range(wl.n_layers + 1):
        for s in range(wl.B):
            n = int(lens[l, s])
            assert (out["pos"][l, s, n:] == -7).all(), (l, s)
            if l < wl.n_layers:
                assert torch.isnan(out["scores"][l, s, n:]).all(), (l, s)
                assert (out["O"][l, s, n:].view(torch.int16) == -1).all(), (l, s)


HOST_STACKS = [
    # per-layer kernels, then the cluster kernel
    wk.Workload("host_12x700", n_layers=12, B=2, L=700, w=64, n_extra_global=3, seed=13),
    # padding removed before layer 0 (ragged lengths)
    wk.Workload("host_ragged_5x600", n_layers=5, B=3, L=600, w=128, ragged=(200, 600), seed=14),
    # short sequences: the cluster kernel only
    wk.Workload("host_short_6x300", n_layers=6, B=3, L=300, w=32, n_extra_global=1, seed=15),
]


@pytest.mark.parametrize("no_tail", [False, True], ids=["with_tail", "per_layer_only"])
@pytest.mark.parametrize("wl", HOST_STACKS, ids=[w.name for w in HOST_STACKS])
def test_host_stack_matches_oracle(sc, wl, no_tail):
    inp, res, _ = resample_stack(wl)
    out = _run_host(sc, wl, inp, no_tail)
    check_stack(wl, res, _numpy(out))
    _assert_rest_untouched(wl, out)


HOST_VS_DEVICE = [
    wk.Workload("host_dev_12x2048", n_layers=12, B=2, L=2048, w=256, n_extra_global=8, seed=16),
    wk.Workload("host_dev_top_ratio", n_layers=6, B=4, L=1024, w=64, n_extra_global=2,
                keep_rule=2, alpha_first=0.95, alpha_last=0.8, seed=17),
    wk.Workload("host_dev_wide", n_layers=3, B=2, L=1536, w=512, n_extra_global=2,
                alpha_first=0.2, alpha_last=0.6, seed=18),
    wk.Workload("host_dev_ragged_4096", n_layers=4, B=2, L=4096, w=256, ragged=(1000, 4096),
                seed=19),
]


@pytest.mark.parametrize("wl", HOST_VS_DEVICE, ids=[w.name for w in HOST_VS_DEVICE])
def test_host_stack_equals_device_stack(sc, wl):
    inp = wk.make_inputs(wl)
    host = _run_host(sc, wl, inp)
    dev = _run_device(sc, wl, inp)
    _assert_same_defined_slots(wl, host, dev, inp["global_pos"])
    _assert_rest_untouched(wl, host)


def test_host_stack_graph_replay(sc):
    """The host call captured once and replayed on new input values: the
    results follow the inputs (the graph reads the host buffers at replay)."""
    wl = wk.Workload("host_graph_12x1024", n_layers=12, B=2, L=1024, w=64, n_extra_global=2,
                     seed=20)
    inp_a = wk.make_inputs(wl)
    inp_b = wk.make_inputs(wk.Workload("host_graph_b", n_layers=12, B=2, L=1024, w=64,
                                       n_extra_global=2, seed=21))
    inp_b["global_pos"] = inp_a["global_pos"]   # captured with the graph, like alpha and w
    (Q, K, V), _ = _host_inputs(inp_a)
    out = _sentinel_outputs(sc, wl)
    ws = sc.new_stack_host_workspace(wl.n_layers, wl.B, wl.L, wl.H)
    stream = torch.cuda.Stream()
    # warm-up outside the capture (first-call configuration, lazy loading)
    with torch.cuda.stream(stream):
        sc.stack_forward_host(Q, K, V, None, inp_a["global_pos"], wl.w, inp_a["alpha"], out=out,
                              workspace=ws, stream=stream)
    stream.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        sc.stack_forward_host(Q, K, V, None, inp_a["global_pos"], wl.w, inp_a["alpha"], out=out,
                              workspace=ws, stream=stream)
    for inp in (inp_b, inp_a):
        for t, k in zip((Q, K, V), ("Q", "K", "V")):
            t.view(torch.int16).copy_(torch.from_numpy(inp[k].view(np.int16)))
        graph.replay()
        torch.cuda.synchronize()
        assert sc.workspace_status(ws) == 0
        expect = _run_device(sc, wl, inp)
        _assert_same_defined_slots(wl, {k: v.clone() for k, v in out.items()}, expect,
                                   inp["global_pos"])


def test_host_stack_refuses_pageable_memory(sc):
    wl = wk.Workload("host_pageable", n_layers=2, B=1, L=256, w=64, seed=22)
    inp = wk.make_inputs(wl)
    Q = torch.from_numpy(inp["Q"].view(np.int16)).view(torch.bfloat16)   # not page-locked
    (_, K, V), _ = _host_inputs(inp)
    with pytest.raises(sc.SparseCoderError):
        sc.stack_forward_host(Q, K, V, None, inp["global_pos"], wl.w, inp["alpha"])
    # the binding's check aside, the library refuses the range itself
    import ctypes
    from paper_2310_07109_gb300 import binding as bd
    out = sc.new_host_outputs(wl.n_layers, wl.B, wl.L, wl.H)
    ws = sc.new_stack_host_workspace(wl.n_layers, wl.B, wl.L, wl.H)
    g = (ctypes.c_int32 * 1)(0)
    al = (ctypes.c_float * 2)(*inp["alpha"])
    a = bd.StackArgs(wl.n_layers, wl.B, wl.L, wl.H, wl.w, Q.data_ptr(), K.data_ptr(),
                     V.data_ptr(), None, ctypes.cast(g, ctypes.POINTER(ctypes.c_int32)), 1,
                     ctypes.cast(al, ctypes.POINTER(ctypes.c_float)), out["O"].data_ptr(),
                     out["scores"].data_ptr(), out["pos"].data_ptr(), out["len"].data_ptr(), 0, 0)
    rc = sc.load().sc_stack_forward_host(ctypes.byref(a), ctypes.c_void_p(ws.data_ptr()),
                                         ws.numel(), None)
    assert rc == bd.SC_ERR_INVALID_ARG


@pytest.mark.parametrize("L,pad,no_tail", [(700, False, False), (700, True, False),
                                           (700, False, True), (300, False, False)])
def test_host_launch_count(sc, L, pad, no_tail):
    """The host-buffer call's plan: the device call's, plus the layer-0 gather
    (when the per-layer kernels run and no padding already forces it) and one
    export (beside the cluster kernel, which writes its own layers' results to
    the host buffers, or after the per-layer kernels)."""
    dev = sc.stack_launch_count(12, 2, L, 12, 64, [0, 5], pad, no_tail=no_tail)
    host = sc.stack_launch_count(12, 2, L, 12, 64, [0, 5], pad, no_tail=no_tail, host=True)
    per_layer = L > sc.TAIL_MAX_LEN or no_tail
    assert host == dev + (1 if per_layer and not pad else 0) + 1


def test_host_stack_last_layer_output_only(sc):
    """O = NULL with O_last: only the last layer's O comes back, equal bit for
    bit to that layer of the full call, and every other result unchanged."""
    wl = wk.Workload("host_o_last", n_layers=6, B=2, L=900, w=64, n_extra_global=3,
                     alpha_first=0.1, alpha_last=0.3, seed=23)
    inp = wk.make_inputs(wl)
    full = _run_host(sc, wl, inp)
    (Q, K, V), mask = _host_inputs(inp)
    out = sc.new_host_outputs(wl.n_layers, wl.B, wl.L, wl.H, o_last_only=True)
    out["O_last"].view(torch.int16).fill_(-1)
    ws = sc.new_stack_host_workspace(wl.n_layers, wl.B, wl.L, wl.H)
    sc.stack_forward_host(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"], out=out,
                          workspace=ws)
    assert sc.workspace_status(ws) == 0
    assert torch.equal(out["len"], full["len"])
    last = wl.n_layers - 1
    for s in range(wl.B):
        n = int(full["len"][last, s])
        assert torch.equal(out["O_last"][s, :n].view(torch.int16),
                           full["O"][last, s, :n].view(torch.int16)), s
        assert (out["O_last"][s, n:].view(torch.int16) == -1).all(), s
        for l in range(wl.n_layers):
            m = int(full["len"][l, s])
            assert torch.equal(out["scores"][l, s, :m], full["scores"][l, s, :m]), (l, s)
