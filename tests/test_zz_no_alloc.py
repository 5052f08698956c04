"""The no-allocation single-layer entry point (sc_layer_forward_noalloc).

For callers that cannot allocate device memory where they run a layer (hosts
whose device heap belongs to another allocator, fixed-budget deployments that
forbid allocation after start-up, services that cannot afford cudaMalloc's
implicit synchronisation), the library offers a variant of the layer that takes
its scratch from a fixed array compiled into the library.  This test checks it
against the workspace-based entry point on the same inputs, on two calls in a
row (the array keeps the previous call's contents), through the C ABI, and on
the largest benchmark shape against the fp64 oracle as well.

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


def _compare(sc, x, B, L, H, w, gl, alpha, lens, expected=None):
    """Two no-allocation calls in a row against the workspace entry point (the
    same kernels: bit for bit) and, given the oracle's results, against those."""
    dev = "cuda"
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
        assert sc.layer_noalloc_status() == sc.SC_OK, call
        assert torch.equal(got["len_out"], ref["len_out"]), call
        for b in range(B):
            k = int(ref["len_out"][b])
            assert torch.equal(got["pos_out"][b, :k], ref["pos_out"][b, :k]), (call, b)
            n = lens[b]
            assert torch.equal(got["scores"][b, :n], ref["scores"][b, :n]), (call, b)
            assert torch.equal(got["O"][b, :n].view(torch.int16),
                               ref["O"][b, :n].view(torch.int16)), (call, b)
            if expected is not None:
                Oe, se, kept = expected[b]
                assert got["pos_out"][b, :k].cpu().tolist() == kept, (call, b)
                o = got["O"][b, :n].float().cpu().numpy().astype(np.float64)
                assert np.abs(o - Oe).max() <= O_ATOL, (call, b)
                s = got["scores"][b, :n].cpu().numpy().astype(np.float64)
                assert np.abs(s - se).max() <= SCORE_ATOL, (call, b)


def test_noalloc_matches_workspace_entry_point_twice(sc):
    B, L, H, w, gl, alpha = 2, 700, 12, 64, [0, 5, 300], 0.8
    lens = [700, 517]
    x = _inputs(B, L, H, lens, seed=31, dev="cuda")
    _compare(sc, x, B, L, H, w, gl, alpha, lens)


def test_noalloc_largest_workload_shape_matches_the_oracle(sc):
    """B=2, L=4096, H=12, window 256, nine global tokens: the largest benchmark
    shape, whose scratch fills about 97% of the array (just under its size)."""
    from parity_utils import layer_case
    B, L, H, w, alpha = 2, 4096, 12, 256, 0.4
    gl = [0, 331, 802, 1500, 2047, 2048, 2900, 3555, 4095]
    case = layer_case(B, L, H, [L, L - 123], w, gl, alpha, seed=37, scale_k=2.0)
    x = {k: bits_to_torch(case[k], "cuda") for k in ("Q", "K", "V")}
    x["len"] = torch.from_numpy(case["len"]).cuda()
    x["pos"] = torch.from_numpy(case["pos"]).cuda()
    _compare(sc, x, B, L, H, w, case["global_pos"].tolist(), alpha, list(case["len"]),
             case["expected"])


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
    # just beyond the array: one head more than the largest benchmark shape
    B, L, H = 2, 4096, 13
    x = {k: torch.zeros((B, L, H, 64), dtype=torch.bfloat16, device=dev) for k in "QKV"}
    o = _outputs(B, L, H, dev)
    length = torch.full((B,), L, dtype=torch.int32, device=dev)
    pos = torch.arange(L, dtype=torch.int32, device=dev).repeat(B, 1).contiguous()
    with pytest.raises(sc.SparseCoderError) as err:
        sc.layer_forward_noalloc(x["Q"], x["K"], x["V"], length, pos, 64, [0], 0.5, O=o["O"],
                                 scores=o["scores"], pos_out=o["pos_out"], len_out=o["len_out"])
    assert err.value.code == sc.SC_ERR_UNSUPPORTED
    assert int(o["len_out"][0]) == -1
