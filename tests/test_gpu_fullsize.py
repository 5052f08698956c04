"""Full-size workloads against the whole fp64 oracle stack.

Every workload at its full size (configs 2, 3, 4 and each point of the config-5
sweep with its theta = 0 control) is drawn with near-threshold resampling: any
token whose oracle score lies within 1e-4 / n of its layer's threshold gets its
Q/K rows redrawn until none does (Sec. "Token Pruning", Steps 2-3 decide on
exactly that comparison).  The whole stack is then compared with the oracle's,
layer by layer and sequence by sequence:
  - lengths and kept positions bit-exact;
  - every O row of every current token within max-abs 2e-2;
  - every score within 1e-5 absolute, and each layer's scores summing to 1.
Three routes run the same inputs: sc_stack_forward as captured in a CUDA graph
(the call the benchmark times), sc_stack_forward eagerly with every layer on the
per-layer kernels (SC_STACK_NO_TAIL), and sc_stack_forward_host on page-locked
host buffers (the benchmark's end-to-end call).
"""
import numpy as np
import pytest
import torch

import workloads as wk
from parity_utils import bits_to_torch, check_stack, resample_stack, stored_redraws

pytestmark = pytest.mark.gpu

FULL = [wk.CFG2, wk.CFG3, wk.CFG4, wk.cfg5(512), wk.cfg5(1024), wk.cfg5(2048), wk.cfg5(4096),
        wk.cfg5(512, control=True), wk.cfg5(1024, control=True), wk.cfg5(2048, control=True),
        wk.cfg5(4096, control=True)]


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    return sc


def _host(out):
    return {"O": out["O"].view(torch.int16).numpy().view(np.uint16),
            "scores": out["scores"].numpy(), "pos": out["pos"].numpy(),
            "len": out["len"].numpy()}


def _device_outputs(sc, wl, inp, graph):
    Q, K, V = (bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V"))
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).cuda()
    ws = sc.new_workspace(wl.B, wl.L, wl.H)
    if graph:
        stream = torch.cuda.Stream()
        stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(stream):
            out = sc.stack_forward(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"],
                                   workspace=ws, keep_rule=wl.keep_rule)   # first call: set-up
            torch.cuda.synchronize()
            for t in out.values():
                t.fill_(-1) if t.dtype != torch.bfloat16 else t.view(torch.int16).fill_(-1)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                sc.stack_forward(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"], out=out,
                                 workspace=ws, keep_rule=wl.keep_rule)
            g.replay()
        torch.cuda.synchronize()
    else:
        out = sc.stack_forward(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"],
                               workspace=ws, no_tail=True, keep_rule=wl.keep_rule)
    assert sc.workspace_status(ws) == 0
    return _host({k: v.cpu() for k, v in out.items()})


def _check(wl, res, got):
    check_stack(wl, res, got)
    for l in range(wl.n_layers):
        for b in range(wl.B):
            n = int(res["len"][l, b])
            if n:
                assert abs(float(got["scores"][l, b, :n].astype(np.float64).sum()) - 1.0) < 1e-4


def _host_route(sc, wl, inp):
    qkv = [torch.from_numpy(np.ascontiguousarray(inp[k]).view(np.int16)).view(torch.bfloat16)
           .pin_memory() for k in ("Q", "K", "V")]
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).pin_memory()
    out = sc.new_host_outputs(wl.n_layers, wl.B, wl.L, wl.H)
    ws = sc.new_stack_host_workspace(wl.n_layers, wl.B, wl.L, wl.H)
    sc.stack_forward_host(*qkv, mask, inp["global_pos"], wl.w, inp["alpha"], out=out,
                          workspace=ws, keep_rule=wl.keep_rule)
    assert sc.workspace_status(ws) == 0
    return _host(out)


@pytest.mark.parametrize("wl", FULL, ids=[w.name for w in FULL])
def test_full_size_stack(sc, wl):
    """The stored redraws are those the resampler finds (so the benchmark times
    resampled inputs), and all three routes match the oracle's whole stack."""
    inp, res, redraws = resample_stack(wl, redraws=stored_redraws(wl), o_dtype=np.float32)
    assert redraws == stored_redraws(wl), "tests/golden/redraws.json is out of date"
    _check(wl, res, _device_outputs(sc, wl, inp, graph=True))
    _check(wl, res, _device_outputs(sc, wl, inp, graph=False))
    _check(wl, res, _host_route(sc, wl, inp))
