"""Eager stack calls through the library's own CUDA graphs.

An eager sc_stack_forward / sc_stack_forward_host call whose plan has both the
per-layer kernels and the cluster kernel is recorded into a graph of the
library (the layer loop is a WHILE node whose condition the device sets) and
the instantiated graph is kept; a later call with the same arguments launches
the kept graph without recording.  Checked here: the graph route gives the
results of the plain-launch route (SC_STACK_PLAIN_LAUNCHES) bit for bit and the
oracle's; an identical call reuses the kept graph; a call that changes what
the host reads at enqueue (the alpha values, the global list, an output
address, the rows design) records a new graph and follows the change; more
argument sets than kept graphs replace the least recently used ones.
"""
import numpy as np
import pytest
import torch

import oracle
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


def _numpy(out):
    return {"O": torch_bf16_to_f64(out["O"]), "scores": out["scores"].cpu().numpy(),
            "pos": out["pos"].cpu().numpy(), "len": out["len"].cpu().numpy()}


def _outputs(wl, dev="cuda"):
    nl, B, L, H = wl.n_layers, wl.B, wl.L, wl.H
    out = {"O": torch.empty((nl, B, L, H, 64), dtype=torch.bfloat16, device=dev),
           "scores": torch.empty((nl, B, L), dtype=torch.float32, device=dev),
           "pos": torch.empty((nl + 1, B, L), dtype=torch.int32, device=dev),
           "len": torch.empty((nl + 1, B), dtype=torch.int32, device=dev)}
    out["O"].view(torch.int16).fill_(-1)
    out["scores"].fill_(float("nan"))
    out["pos"].fill_(-7)
    out["len"].fill_(-7)
    return out


def _same_defined_slots(wl, a, b):
    a = {k: v.cpu() for k, v in a.items()}
    b = {k: v.cpu() for k, v in b.items()}
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


def _counts_after(sc, fn):
    r0, u0 = sc.debug_graph_counts()
    fn()
    torch.cuda.synchronize()
    r1, u1 = sc.debug_graph_counts()
    return r1 - r0, u1 - u0


# per-layer kernels for the long sequence(s), then the cluster kernel
WL = wk.Workload("eager_graph_12x900", n_layers=12, B=2, L=900, w=64, n_extra_global=3, seed=61)


def test_graph_route_equals_plain_launches_and_oracle(sc):
    inp, res, _ = resample_stack(WL)
    t = {k: bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V")}
    ws = sc.new_workspace(WL.B, WL.L, WL.H)
    out_g, out_p = _outputs(WL), _outputs(WL)

    def call(out, plain=False):
        sc.stack_forward(t["Q"], t["K"], t["V"], None, inp["global_pos"], WL.w, inp["alpha"],
                         out=out, workspace=ws, plain_launches=plain)

    assert _counts_after(sc, lambda: call(out_g)) == (1, 0)     # recorded
    assert sc.workspace_status(ws) == 0
    check_stack(WL, res, _numpy(out_g))
    assert _counts_after(sc, lambda: call(out_p, plain=True)) == (0, 0)
    assert sc.workspace_status(ws) == 0
    _same_defined_slots(WL, out_g, out_p)
    # the same call again: the kept graph, on new values in the same tensors
    inp2, res2, _ = resample_stack(WL.with_(seed=WL.seed + 100),
                                   overrides={"global_pos": inp["global_pos"]})
    for k in ("Q", "K", "V"):
        t[k].copy_(bits_to_torch(inp2[k], "cuda"))
    assert _counts_after(sc, lambda: call(out_g)) == (0, 1)     # reused
    assert sc.workspace_status(ws) == 0
    check_stack(WL, res2, _numpy(out_g))


def test_changed_host_arguments_record_again(sc):
    inp, res, _ = resample_stack(WL.with_(seed=62))
    t = {k: bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V")}
    ws = sc.new_workspace(WL.B, WL.L, WL.H)
    out = _outputs(WL)

    def call(alpha, gpos, o=out):
        sc.stack_forward(t["Q"], t["K"], t["V"], None, gpos, WL.w, alpha, out=o, workspace=ws)

    assert _counts_after(sc, lambda: call(inp["alpha"], inp["global_pos"]))[0] == 1
    check_stack(WL, res, _numpy(out))
    # alpha = 0 keeps every token: a new graph, whose results follow the values
    zero = np.zeros(WL.n_layers)
    assert _counts_after(sc, lambda: call(zero, inp["global_pos"])) == (1, 0)
    res0 = oracle.stack(inp["Q"], inp["K"], inp["V"], None, inp["global_pos"], WL.w, zero)
    assert (out["len"].cpu().numpy() == WL.L).all()
    check_stack(WL, res0, _numpy(out))
    # another global list (kept tokens do not move: alpha = 0)
    g2 = [0, 7, 450]
    assert _counts_after(sc, lambda: call(zero, g2)) == (1, 0)
    res_g = oracle.stack(inp["Q"], inp["K"], inp["V"], None, g2, WL.w, zero)
    check_stack(WL, res_g, _numpy(out))
    # the first arguments again: their kept graph
    assert _counts_after(sc, lambda: call(inp["alpha"], inp["global_pos"])) == (0, 1)
    check_stack(WL, res, _numpy(out))
    # other output tensors: recorded again, written there
    out2 = _outputs(WL)
    assert _counts_after(sc, lambda: call(inp["alpha"], inp["global_pos"], out2)) == (1, 0)
    check_stack(WL, res, _numpy(out2))
    # the other rows design, read at enqueue: recorded again
    sc.select_rows_kernel(sc.SC_ROWS_SINGLE_PASS)
    try:
        assert _counts_after(sc, lambda: call(inp["alpha"], inp["global_pos"], out2)) == (1, 0)
    finally:
        sc.select_rows_kernel(sc.SC_ROWS_TWO_PASS)
    assert sc.workspace_status(ws) == 0
    check_stack(WL, res, _numpy(out2))


def test_plans_without_both_kinds_launch_directly(sc):
    """Only the cluster kernel (L <= TAIL_MAX_LEN), or only the per-layer
    kernels (SC_STACK_NO_TAIL): no graph is recorded."""
    for wl, no_tail in ((wk.Workload("eager_short", n_layers=4, B=2, L=256, w=32,
                                     n_extra_global=1, seed=63), False),
                        (WL.with_(n_layers=3, seed=64), True)):
        inp, res, _ = resample_stack(wl)
        t = {k: bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V")}
        ws = sc.new_workspace(wl.B, wl.L, wl.H)
        out = _outputs(wl)
        assert _counts_after(sc, lambda: sc.stack_forward(
            t["Q"], t["K"], t["V"], None, inp["global_pos"], wl.w, inp["alpha"], out=out,
            workspace=ws, no_tail=no_tail)) == (0, 0)
        assert sc.workspace_status(ws) == 0
        check_stack(wl, res, _numpy(out))


def test_host_call_graph_route(sc):
    """sc_stack_forward_host: the stack and the export of the per-layer results
    in one kept graph; equal to the plain launches and to the oracle."""
    inp, res, _ = resample_stack(WL.with_(seed=65))
    qkv = [torch.from_numpy(np.ascontiguousarray(inp[k]).view(np.int16)).view(torch.bfloat16)
           .pin_memory() for k in ("Q", "K", "V")]
    ws = sc.new_stack_host_workspace(WL.n_layers, WL.B, WL.L, WL.H)
    out_g = sc.new_host_outputs(WL.n_layers, WL.B, WL.L, WL.H)
    out_p = sc.new_host_outputs(WL.n_layers, WL.B, WL.L, WL.H)

    def call(out, plain=False):
        sc.stack_forward_host(*qkv, None, inp["global_pos"], WL.w, inp["alpha"], out=out,
                              workspace=ws, plain_launches=plain)

    assert _counts_after(sc, lambda: call(out_g)) == (1, 0)
    assert _counts_after(sc, lambda: call(out_g)) == (0, 1)
    assert _counts_after(sc, lambda: call(out_p, plain=True)) == (0, 0)
    assert sc.workspace_status(ws) == 0
    check_stack(WL, res, _numpy(out_g))
    _same_defined_slots(WL, out_g, out_p)


def test_graph_route_on_a_side_stream(sc):
    """The kept graph is launched on the caller's stream, after its earlier work."""
    inp, res, _ = resample_stack(WL.with_(seed=66))
    ws = sc.new_workspace(WL.B, WL.L, WL.H)
    out = _outputs(WL)
    stream = torch.cuda.Stream()
    t = {k: torch.zeros(inp[k].shape, dtype=torch.bfloat16, device="cuda")
         for k in ("Q", "K", "V")}
    src = {k: bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V")}
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        for _ in range(2):          # recorded, then kept
            for k in ("Q", "K", "V"):
                t[k].copy_(src[k])   # ordered before the call on the same stream
            sc.stack_forward(t["Q"], t["K"], t["V"], None, inp["global_pos"], WL.w,
                             inp["alpha"], out=out, workspace=ws, stream=stream)
            for v in t.values():
                v.zero_()
    stream.synchronize()
    assert sc.workspace_status(ws) == 0
    check_stack(WL, res, _numpy(out))


def test_more_argument_sets_than_kept_graphs(sc):
    """18 output sets cycled twice through the 16 kept graphs: the least
    recently used graphs are replaced (and destroyed while the stream may still
    run them), and every call's results are those of the first."""
    wl = wk.Workload("eager_lru", n_layers=3, B=2, L=500, w=64, n_extra_global=2, seed=67)
    inp, res, _ = resample_stack(wl)
    t = {k: bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V")}
    ws = sc.new_workspace(wl.B, wl.L, wl.H)
    outs = [_outputs(wl) for _ in range(18)]
    r0, _ = sc.debug_graph_counts()
    for _ in range(2):
        for o in outs:
            sc.stack_forward(t["Q"], t["K"], t["V"], None, inp["global_pos"], wl.w, inp["alpha"],
                             out=o, workspace=ws)
    torch.cuda.synchronize()
    r1, _ = sc.debug_graph_counts()
    assert r1 - r0 == 36          # LRU over 18 sets in a cycle: every call records
    assert sc.workspace_status(ws) == 0
    check_stack(wl, res, _numpy(outs[0]))
    for o in outs[1:]:
        _same_defined_slots(wl, outs[0], o)
