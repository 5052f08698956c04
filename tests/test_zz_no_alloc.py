"""The no-allocation single-layer entry point (sc_layer_forward_noalloc).

For callers that cannot allocate device memory where they run a layer (hosts
whose device heap belongs to another allocator, fixed-budget deployments that
forbid allocation after start-up, services that cannot afford cudaMalloc's
implicit synchronisation), the library offers a variant of the layer that takes
its scratch from a fixed array compiled into the library.  This test checks it
against the workspace-based entry point on the same inputs, on two calls in a
row (the array keeps the previous call's contents), through the C ABI.

Kept last in collection order so that a failure here never hides the others.
"""
import numpy as np
import pytest
import torch

from parity_utils import O_ATOL, SCORE_ATOL, bits_to_torch
import workloads as wk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2310_07109_gb300 import binding
    binding.load(build_if_missing=True)
    return binding


def _inputs(B, L, H, lens, seed, dev):
    Q, K, V = (np.empty((B, L, H, 64), np.uint16) for _ in range(3))
    for b in range(B):
        Q[b], K[b], V[b] = wk.random_layer(L, H, 64, seed * 10 + b, scale_k=2.0)
    t = {k: bits_to_torch(x, dev) for k, x in (("Q", Q), ("K", K), ("V", V))}
    t["len"] = torch.tensor(lens, dtype=torch.int32, device=dev)
    t["pos"] = torch.arange(L, dtype=torch.int32, device=dev).repeat(B, 1).contiguous()
    return t


def _outputs(B, L, H, dev):
    return {"O": torch.zeros((B, L, H, 64), dtype=torch.bfloat16, device=dev),
            "scores": torch.zeros((B, L), dtype=torch.float32, device=dev),
            "pos_out": torch.full((B, L), -1, dtype=torch.int32, device=dev),
            "len_out": torch.full((B,), -1, dtype=torch.int32, device=dev)}


def test_noalloc_matches_workspace_entry_point_twice(sc):
    dev = "cuda"
    B, L, H, w, gl, alpha = 2, 700, 12, 64, [0, 5, 300], 0.8
    lens = [700, 517]
    x = _inputs(B, L, H, lens, seed=31, dev=dev)
    ws = sc.new_workspace(B, L, H, dev)
    ref = _outputs(B, L, H, dev)
    sc.layer_forward(x["Q"], x["K"], x["V"], x["len"], x["pos"], w, gl, alpha, O=ref["O"],
                     scores=ref["scores"], pos_out=ref["pos_out"], len_out=ref["len_out"],
                     workspace=ws)
    assert sc.workspace_status(ws) == 0
    for call in range(2):
        got = _outputs(B, L, H, dev)
        sc.layer_forward_noalloc(x["Q"], x["K"], x["V"], x["len"], x["pos"], w, gl, alpha,
                                 O=got["O"], scores=got["scores"], pos_out=got["pos_out"],
                                 len_out=got["len_out"])
        torch.cuda.synchronize()
        assert torch.equal(got["len_out"], ref["len_out"]), call
        for b in range(B):
            k = int(ref["len_out"][b])
            assert torch.equal(got["pos_out"][b, :k], ref["pos_out"][b, :k]), (call, b)
            n = lens[b]
            np.testing.assert_allclose(got["scores"][b, :n].cpu().numpy(),
                                       ref["scores"][b, :n].cpu().numpy(), rtol=0,
                                       atol=SCORE_ATOL)
            np.testing.assert_allclose(got["O"][b, :n].float().cpu().numpy(),
                                       ref["O"][b, :n].float().cpu().numpy(), rtol=0,
                                       atol=O_ATOL)


def test_noalloc_rejects_sizes_beyond_its_array(sc):
    dev = "cuda"
    B, L, H = 16, 4096, 12   # about 786k rows of scratch: more than the array holds
    x = {k: torch.zeros((B, L, H, 64), dtype=torch.bfloat16, device=dev) for k in "QKV"}
    o = _outputs(B, L, H, dev)
    length = torch.full((B,), L, dtype=torch.int32, device=dev)
    pos = torch.arange(L, dtype=torch.int32, device=dev).repeat(B, 1).contiguous()
    with pytest.raises(sc.SparseCoderError) as err:
        sc.layer_forward_noalloc(x["Q"], x["K"], x["V"], length, pos, 64, [0], 0.5, O=o["O"],
                                 scores=o["scores"], pos_out=o["pos_out"], len_out=o["len_out"])
    assert err.value.code == sc.SC_ERR_UNSUPPORTED
    assert int(o["len_out"][0]) == -1   # nothing was launched
