"""The pruned stack captured into a CUDA graph and replayed.

Under capture the library runs the per-layer kernels inside a WHILE node whose
condition the device sets (the layer index lives in device memory), so a
replay does only the layers that some sequence still runs per layer.  Each
case replays the graph, compares with the fp64 oracle, then writes new inputs
into the same tensors and replays again (no state may leak between replays).
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


def _host(out):
    return {"O": torch_bf16_to_f64(out["O"]), "scores": out["scores"].cpu().numpy(),
            "pos": out["pos"].cpu().numpy(), "len": out["len"].cpu().numpy()}


def _capture(sc, wl, inp):
    dev = "cuda"
    t = {k: bits_to_torch(inp[k], dev) for k in ("Q", "K", "V")}
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).to(dev)
    ws = sc.new_workspace(wl.B, wl.L, wl.H, dev)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        out = sc.stack_forward(t["Q"], t["K"], t["V"], mask, inp["global_pos"], wl.w, inp["alpha"],
                               workspace=ws, keep_rule=wl.keep_rule)
        torch.cuda.synchronize()
        # eager result of the same call, then clobber the outputs
        eager = _host(out)
        for v in out.values():
            v.fill_(0 if v.dtype != torch.float32 else float("nan"))
        with torch.cuda.graph(graph, stream=side):
            sc.stack_forward(t["Q"], t["K"], t["V"], mask, inp["global_pos"], wl.w, inp["alpha"],
                             out=out, workspace=ws, keep_rule=wl.keep_rule)
    torch.cuda.current_stream().wait_stream(side)
    return graph, t, mask, out, ws, eager


def _replay_and_check(sc, wl, graph, t, out, ws, inp, res):
    for k in ("Q", "K", "V"):
        t[k].copy_(bits_to_torch(inp[k], "cuda"))
    graph.replay()
    torch.cuda.synchronize()
    assert sc.workspace_status(ws) == 0
    got = _host(out)
    check_stack(wl, res, got)
    return got


CASES = [
    wk.Workload("handover_1200", n_layers=5, B=2, L=1200, w=128, n_extra_global=6,
                salient_frac=0.08, salient_scale=4.0, alpha_first=0.5, alpha_last=1.0, seed=16),
    wk.Workload("small_12x700", n_layers=12, B=2, L=700, w=64, n_extra_global=3, seed=3),
    wk.Workload("all_tail_w64", n_layers=4, B=3, L=256, w=64, n_extra_global=4, ragged=(40, 256),
                seed=11),
    # the wide rows layout and the top-ratio rule inside the captured loop
    wk.Workload("wide_top_ratio_768", n_layers=3, B=2, L=768, w=400, n_extra_global=2,
                alpha_first=0.6, alpha_last=0.5, keep_rule=2, seed=23),
]


@pytest.mark.parametrize("wl", CASES, ids=[w.name for w in CASES])
def test_graph_replay_matches_oracle(sc, wl):
    inp, res, _ = resample_stack(wl)
    graph, t, mask, out, ws, eager = _capture(sc, wl, inp)
    got = _replay_and_check(sc, wl, graph, t, out, ws, inp, res)
    np.testing.assert_array_equal(got["len"], eager["len"])
    # new contents in the same input tensors (another seed; the global list and
    # padding that the graph holds stay), replayed again
    inp2, res2, _ = resample_stack(wl.with_(seed=wl.seed + 100),
                                   overrides={"global_pos": inp["global_pos"],
                                              "pad_mask": inp["pad_mask"]})
    _replay_and_check(sc, wl, graph, t, out, ws, inp2, res2)


def test_graph_replay_every_layer_per_layer(sc):
    """theta = 0 keeps all 500 tokens: the WHILE loop runs all three layers."""
    wl = wk.Workload("theta0_500", n_layers=3, B=2, L=500, w=64, n_extra_global=2,
                     alpha_first=0.0, alpha_last=0.0, seed=21)
    inp = wk.make_inputs(wl)
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], None, inp["global_pos"], wl.w, inp["alpha"])
    graph, t, mask, out, ws, _ = _capture(sc, wl, inp)
    got = _replay_and_check(sc, wl, graph, t, out, ws, inp, res)
    assert (got["len"] == 500).all()


def test_graph_replay_with_padding_holes(sc):
    wl = wk.Workload("holes_600", n_layers=4, B=2, L=600, w=64, n_extra_global=2, seed=22)
    inp = wk.make_inputs(wl)
    rng = np.random.default_rng(22)
    mask = (rng.random((wl.B, wl.L)) < 0.7).astype(np.uint8)
    mask[:, 0] = 1
    mask[:, inp["global_pos"]] = 1
    inp["pad_mask"] = mask
    # thresholds far from every score: keep everything, so no resampling is needed
    inp["alpha"] = np.zeros(wl.n_layers)
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], mask, inp["global_pos"], wl.w, inp["alpha"])
    graph, t, _, out, ws, _ = _capture(sc, wl, inp)
    _replay_and_check(sc, wl, graph, t, out, ws, inp, res)
