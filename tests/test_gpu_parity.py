"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle.

Every expected value comes from the oracle on the same bf16 inputs.  Kept lists,
lengths and positions must match bit for bit (the inputs are resampled so that
no oracle score lies within 1e-4 / n of its threshold); O within max-abs 2e-2;
scores within 1e-5 absolute.
"""
import numpy as np
import pytest
import torch

import workloads as wk
from parity_utils import (bits_to_torch, check_o, check_scores, check_stack, layer_case,
                          resample_stack, torch_bf16_to_f64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    return sc


def _run_layer(sc, case, w):
    dev = "cuda"
    Q, K, V = (bits_to_torch(case[k], dev) for k in ("Q", "K", "V"))
    B, L, H, _ = Q.shape
    length = torch.from_numpy(case["len"]).to(dev)
    pos = torch.from_numpy(case["pos"]).to(dev)
    ws = sc.new_workspace(B, L, H, dev)
    O, s, po, lo = sc.layer_forward(Q, K, V, length, pos, w, case["global_pos"], case["alpha"],
                                    workspace=ws)
    assert sc.workspace_status(ws) == 0
    return torch_bf16_to_f64(O), s.cpu().numpy(), po.cpu().numpy(), lo.cpu().numpy()


def _check_layer(case, got):
    O, s, po, lo = got
    for b, (Oe, se, kept) in enumerate(case["expected"]):
        n = int(case["len"][b])
        assert int(lo[b]) == len(kept), f"sequence {b}: kept count"
        assert list(po[b, :len(kept)]) == kept, f"sequence {b}: kept positions"
        if n == 0:
            continue
        check_o(O[b, :n], Oe, f"sequence {b}")
        check_scores(s[b, :n], se, f"sequence {b}")
        assert abs(float(s[b, :n].astype(np.float64).sum()) - 1.0) < 1e-4


LAYER_CASES = [
    # B, L, lens, w, globals, alpha, gaps
    (2, 320, [300, 217], 64, [0, 5, 100], 0.8, False),
    (1, 128, [128], 256, [0], 0.9, False),                   # window covers the sequence
    (3, 700, [700, 1, 129], 64, [0, 127, 128, 255, 699], 0.7, False),  # n=1, tile-edge globals
    (2, 640, [640, 517], 300, [0, 3], 0.6, False),           # wide window, short sequence
    (2, 900, [0, 900], 256, [0, 450], 0.9, False),           # an empty sequence
    (2, 400, [400, 333], 32, [0], 1.0, True),                # gaps in original positions
    (1, 1024, [1024], 0, [0, 1, 2, 1023], 0.5, False),       # w = 0: diagonal + globals
    # wide windows on long sequences: one query tile per rows CTA, up to nine
    # key tiles per band
    (2, 1024, [1024, 700], 512, [0, 300], 0.6, False),
    (1, 2048, [2048], 300, [0, 1000, 2047], 0.7, False),
]


@pytest.mark.parametrize("B,L,lens,w,gl,alpha,gaps", LAYER_CASES)
def test_layer_matches_oracle(sc, B, L, lens, w, gl, alpha, gaps):
    case = layer_case(B, L, 12, lens, w, gl, alpha, seed=L + w, gaps=gaps)
    if gaps:  # globals are original positions: pick some that exist
        case["global_pos"] = np.unique(np.concatenate([[0], case["pos"][1, [5, 77]]])).astype(np.int32)
        case = layer_case(B, L, 12, lens, w, case["global_pos"], alpha, seed=L + w, gaps=gaps)
    _check_layer(case, _run_layer(sc, case, w))


def _run_stack(sc, wl, inp, no_tail=False):
    dev = "cuda"
    Q, K, V = (bits_to_torch(inp[k], dev) for k in ("Q", "K", "V"))
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).to(dev)
    ws = sc.new_workspace(wl.B, wl.L, wl.H, dev)
    out = sc.stack_forward(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"], workspace=ws,
                           no_tail=no_tail, keep_rule=wl.keep_rule)
    assert sc.workspace_status(ws) == 0
    return {"O": torch_bf16_to_f64(out["O"]), "scores": out["scores"].cpu().numpy(),
            "pos": out["pos"].cpu().numpy(), "len": out["len"].cpu().numpy()}


STACKS = [
    wk.Workload("small_12x700", n_layers=12, B=2, L=700, w=64, n_extra_global=3, seed=3),
    wk.Workload("ragged_6x600", n_layers=6, B=3, L=600, w=128, ragged=(200, 600), seed=4),
    wk.Workload("salient4_4x1000", n_layers=4, B=1, L=1000, w=256, n_extra_global=8,
                salient_frac=0.05, salient_scale=4.0, alpha_first=0.4, alpha_last=1.0, seed=5),
    wk.CFG1,
    wk.Workload("wide_w512_4x1024", n_layers=4, B=2, L=1024, w=512, n_extra_global=2,
                alpha_first=0.2, alpha_last=0.6, seed=6),
]


@pytest.mark.parametrize("no_tail", [False, True], ids=["with_tail", "per_layer_only"])
@pytest.mark.parametrize("wl", STACKS, ids=[w.name for w in STACKS])
def test_stack_matches_oracle(sc, wl, no_tail):
    inp, res, _ = resample_stack(wl)
    check_stack(wl, res, _run_stack(sc, wl, inp, no_tail))


def test_stack_theta_zero_keeps_everything(sc):
    wl = wk.Workload("theta0", n_layers=3, B=2, L=500, w=64, alpha_first=0.0, alpha_last=0.0)
    inp = wk.make_inputs(wl)
    got = _run_stack(sc, wl, inp)
    assert (got["len"] == 500).all()
    assert (got["pos"][:, :, :500] == np.arange(500)).all()


def test_stack_huge_theta_keeps_only_first(sc):
    wl = wk.Workload("thetaInf", n_layers=2, B=2, L=300, w=64, alpha_first=1e9, alpha_last=1e9,
                     ragged=(100, 300))
    inp = wk.make_inputs(wl)
    got = _run_stack(sc, wl, inp)
    assert (got["len"][1:] == 1).all()
    assert (got["pos"][1:, :, 0] == 0).all()


def test_stack_scattered_padding_uses_compacted_rows(sc):
    """Padding in the middle of sequences: every layer reads compacted rows."""
    import oracle
    wl = wk.Workload("holes", n_layers=3, B=2, L=400, w=64, n_extra_global=2,
                     alpha_first=0.0, alpha_last=0.0, seed=8)
    inp = wk.make_inputs(wl)
    rng = np.random.default_rng(8)
    mask = (rng.random((wl.B, wl.L)) < 0.8).astype(np.uint8)
    mask[:, 0] = 1
    mask[:, inp["global_pos"]] = 1
    inp["pad_mask"] = mask
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], mask, inp["global_pos"], wl.w, inp["alpha"])
    check_stack(wl, res, _run_stack(sc, wl, inp))
