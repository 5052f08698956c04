"""The failure path of the bounded device waits, on the GPU, without a fault.

Every wait inside the kernels gives up after a bounded time; the CTA then
abandons its work, drains its own copies and matrix products, frees its tensor
memory and records SC_ERR_TIMEOUT in the status word.  The test hook
sc_debug_stall_waits makes the first MMA-issuing thread of every per-layer
attention CTA wait on a barrier that nothing completes, for a short limit, so
that this path really runs; the status queries must then report the timeout,
and the next call (hook off) on the same workspace must match the oracle.
A status word written by hand checks the host-side decoding and reset.
"""
import numpy as np
import pytest
import torch

import workloads as wk
from parity_utils import bits_to_torch, check_o, check_scores, check_stack, layer_case, \
    resample_stack, torch_bf16_to_f64

pytestmark = pytest.mark.gpu

STALL_NS = 200_000   # 0.2 ms per CTA


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    yield sc
    sc.debug_stall_waits(0)


def _layer_tensors(case):
    t = {k: bits_to_torch(case[k], "cuda") for k in ("Q", "K", "V")}
    t["len"] = torch.from_numpy(case["len"]).cuda()
    t["pos"] = torch.from_numpy(case["pos"]).cuda()
    return t


def _check_layer(case, O, s, po, lo):
    O, s, po, lo = torch_bf16_to_f64(O), s.cpu().numpy(), po.cpu().numpy(), lo.cpu().numpy()
    for b, (Oe, se, kept) in enumerate(case["expected"]):
        n = int(case["len"][b])
        assert int(lo[b]) == len(kept)
        assert list(po[b, :len(kept)]) == kept
        if n:
            check_o(O[b, :n], Oe, f"sequence {b}")
            check_scores(s[b, :n], se, f"sequence {b}")


CASE = dict(B=2, L=700, H=12, lens=[700, 517], w=64, gpos=[0, 5, 300], alpha=0.8, seed=51)


def test_expired_wait_reports_timeout_then_recovers(sc):
    case = layer_case(**CASE)
    t = _layer_tensors(case)
    ws = sc.new_workspace(CASE["B"], CASE["L"], CASE["H"])
    sc.debug_stall_waits(STALL_NS)
    try:
        sc.layer_forward(t["Q"], t["K"], t["V"], t["len"], t["pos"], CASE["w"],
                         case["global_pos"], CASE["alpha"], workspace=ws)
    finally:
        sc.debug_stall_waits(0)
    assert sc.workspace_status(ws) == sc.SC_ERR_TIMEOUT
    assert sc.workspace_status(ws) == sc.SC_OK          # the query cleared the word
    out = sc.layer_forward(t["Q"], t["K"], t["V"], t["len"], t["pos"], CASE["w"],
                           case["global_pos"], CASE["alpha"], workspace=ws)
    assert sc.workspace_status(ws) == sc.SC_OK
    _check_layer(case, *out)


def test_expired_wait_in_a_stack_then_recovers(sc):
    """The per-layer part of a stack (every layer on the per-layer kernels):
    the timeout is reported, and the next call on the workspace is exact."""
    wl = wk.Workload("fail_stack", n_layers=3, B=2, L=900, w=64, n_extra_global=2, seed=52)
    inp, res, _ = resample_stack(wl)
    t = {k: bits_to_torch(inp[k], "cuda") for k in ("Q", "K", "V")}
    ws = sc.new_workspace(wl.B, wl.L, wl.H)
    sc.debug_stall_waits(STALL_NS)
    try:
        sc.stack_forward(t["Q"], t["K"], t["V"], None, inp["global_pos"], wl.w, inp["alpha"],
                         workspace=ws, no_tail=True)
    finally:
        sc.debug_stall_waits(0)
    assert sc.workspace_status(ws) == sc.SC_ERR_TIMEOUT
    out = sc.stack_forward(t["Q"], t["K"], t["V"], None, inp["global_pos"], wl.w, inp["alpha"],
                           workspace=ws, no_tail=True)
    assert sc.workspace_status(ws) == sc.SC_OK
    check_stack(wl, res, {"O": torch_bf16_to_f64(out["O"]), "scores": out["scores"].cpu().numpy(),
                          "pos": out["pos"].cpu().numpy(), "len": out["len"].cpu().numpy()})


def test_noalloc_timeout_is_reported(sc):
    """sc_layer_forward_noalloc keeps an expired wait in its array's status
    word until sc_layer_noalloc_status reads it."""
    case = layer_case(**CASE)
    t = _layer_tensors(case)
    B, L, H = CASE["B"], CASE["L"], CASE["H"]
    out = [torch.empty((B, L, H, 64), dtype=torch.bfloat16, device="cuda"),
           torch.empty((B, L), dtype=torch.float32, device="cuda"),
           torch.empty((B, L), dtype=torch.int32, device="cuda"),
           torch.empty((B,), dtype=torch.int32, device="cuda")]
    assert sc.layer_noalloc_status() in (sc.SC_OK, sc.SC_ERR_TIMEOUT)   # start clean
    assert sc.layer_noalloc_status() == sc.SC_OK

    def call():
        sc.layer_forward_noalloc(t["Q"], t["K"], t["V"], t["len"], t["pos"], CASE["w"],
                                 case["global_pos"], CASE["alpha"], O=out[0], scores=out[1],
                                 pos_out=out[2], len_out=out[3])

    sc.debug_stall_waits(STALL_NS)
    try:
        call()
    finally:
        sc.debug_stall_waits(0)
    call()   # a later call does not clear the earlier call's timeout
    assert sc.layer_noalloc_status() == sc.SC_ERR_TIMEOUT
    assert sc.layer_noalloc_status() == sc.SC_OK
    call()
    assert sc.layer_noalloc_status() == sc.SC_OK
    _check_layer(case, *out)


@pytest.mark.parametrize("word,expect", [(1, "SC_ERR_TIMEOUT"), (3, "SC_ERR_TIMEOUT"),
                                         (2, "SC_ERR_CUDA"), (0, "SC_OK")])
def test_status_word_decoding(sc, word, expect):
    """A status word written by hand: decoded, then cleared by the query."""
    ws = sc.new_workspace(1, 128, 1)
    ws[:4].view(torch.int32).fill_(word)
    assert sc.workspace_status(ws) == getattr(sc, expect)
    assert int(ws[:4].view(torch.int32).item()) == 0
    assert sc.workspace_status(ws) == sc.SC_OK
