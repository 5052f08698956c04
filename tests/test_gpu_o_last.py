"""The stack with O = NULL: only the last layer's O is written, to O_last
(the scores that decide the kept tokens need no earlier O).  Checked bit for
bit against the same layer of a call that writes every layer's O, through the
per-layer kernels, the cluster kernel and the captured graph, and with no O
at all (O_last NULL as well)."""
import numpy as np
import pytest
import torch

import workloads as wk
from parity_utils import bits_to_torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    return sc


CASES = [
    # per-layer kernels for every layer (theta small), globals
    wk.Workload("olast_per_layer", n_layers=4, B=2, L=1200, w=128, n_extra_global=4,
                alpha_first=0.05, alpha_last=0.1, seed=41),
    # hand-over to the cluster kernel mid-stack
    wk.Workload("olast_handover", n_layers=8, B=3, L=1000, w=64, n_extra_global=2, seed=42),
    # the cluster kernel only
    wk.Workload("olast_cluster", n_layers=5, B=2, L=300, w=32, n_extra_global=1, seed=43),
]


def _inputs(wl):
    inp = wk.make_inputs(wl)
    t = {k: bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V")}
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).cuda()
    return inp, t, mask


def _same_last_layer(wl, full, part):
    assert torch.equal(full["len"], part["len"])
    last = wl.n_layers - 1
    lens = full["len"].cpu()
    for b in range(wl.B):
        for l in range(wl.n_layers):
            n = int(lens[l, b])
            assert torch.equal(full["scores"][l, b, :n], part["scores"][l, b, :n]), (l, b)
            m = int(lens[l + 1, b])
            assert torch.equal(full["pos"][l + 1, b, :m], part["pos"][l + 1, b, :m]), (l, b)
        n = int(lens[last, b])
        if "O_last" in part:
            assert torch.equal(part["O_last"][b, :n].view(torch.int16),
                               full["O"][last, b, :n].view(torch.int16)), b
            assert (part["O_last"][b, n:].view(torch.int16) == -1).all(), b


@pytest.mark.parametrize("no_tail", [False, True], ids=["with_tail", "per_layer_only"])
@pytest.mark.parametrize("wl", CASES, ids=[w.name for w in CASES])
def test_last_layer_output_only(sc, wl, no_tail):
    inp, t, mask = _inputs(wl)
    ws = sc.new_workspace(wl.B, wl.L, wl.H)
    full = sc.stack_forward(t["Q"], t["K"], t["V"], mask, inp["global_pos"], wl.w, inp["alpha"],
                            workspace=ws, no_tail=no_tail)
    out = {"O_last": torch.full((wl.B, wl.L, wl.H, 64), -1, dtype=torch.int16,
                                device="cuda").view(torch.bfloat16),
           "scores": torch.empty_like(full["scores"]), "pos": torch.empty_like(full["pos"]),
           "len": torch.empty_like(full["len"])}
    sc.stack_forward(t["Q"], t["K"], t["V"], mask, inp["global_pos"], wl.w, inp["alpha"],
                     out=out, workspace=ws, no_tail=no_tail)
    assert sc.workspace_status(ws) == 0
    _same_last_layer(wl, full, out)
    # no O at all
    none = {k: torch.empty_like(v) for k, v in out.items() if k != "O_last"}
    sc.stack_forward(t["Q"], t["K"], t["V"], mask, inp["global_pos"], wl.w, inp["alpha"],
                     out=none, workspace=ws, no_tail=no_tail)
    assert sc.workspace_status(ws) == 0
    _same_last_layer(wl, full, none)


def test_last_layer_output_only_graph(sc):
    """Captured in a CUDA graph (the per-layer kernels in the device-driven
    layer loop, where the last layer is known only on the device)."""
    wl = CASES[0]
    inp, t, mask = _inputs(wl)
    ws = sc.new_workspace(wl.B, wl.L, wl.H)
    full = sc.stack_forward(t["Q"], t["K"], t["V"], mask, inp["global_pos"], wl.w, inp["alpha"],
                            workspace=ws)
    torch.cuda.synchronize()
    out = {"O_last": torch.full((wl.B, wl.L, wl.H, 64), -1, dtype=torch.int16,
                                device="cuda").view(torch.bfloat16),
           "scores": torch.empty_like(full["scores"]), "pos": torch.empty_like(full["pos"]),
           "len": torch.empty_like(full["len"])}
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(g, stream=side):
            sc.stack_forward(t["Q"], t["K"], t["V"], mask, inp["global_pos"], wl.w,
                             inp["alpha"], out=out, workspace=ws)
    torch.cuda.current_stream().wait_stream(side)
    g.replay()
    torch.cuda.synchronize()
    assert sc.workspace_status(ws) == 0
    _same_last_layer(wl, full, out)
