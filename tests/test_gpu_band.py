"""GPU parity of the single-pass rows design (SC_ROWS_SINGLE_PASS) against the
fp64 oracle.

The design keeps every band tile's probabilities on chip in bf16 until the
row's normaliser is known and takes the column sums of Sec. "Pruning" from
them with tensor-core products, so each score carries a relative error of at
most 2^-9 (the bf16 rounding of the probabilities).  The cases here are those
whose sequences keep at least a few hundred tokens in the per-layer kernels;
shorter sequences finish in the cluster kernel, which is the same for both
designs.  The bars are those of every other parity test: kept lists exact, O
within max-abs 2e-2, scores within 1e-5 absolute.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wk
from parity_utils import (bits_to_torch, check_o, check_scores, check_stack, layer_case,
                          resample_stack, torch_bf16_to_f64)
from test_gpu_parity import LAYER_CASES, _check_layer, _run_layer, _run_stack

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    sc.select_rows_kernel(sc.SC_ROWS_SINGLE_PASS)
    yield sc
    sc.select_rows_kernel(sc.SC_ROWS_TWO_PASS)


def test_select_rows_kernel_rejects_unknown_values(sc):
    with pytest.raises(sc.SparseCoderError):
        sc.select_rows_kernel(7)
    sc.select_rows_kernel(sc.SC_ROWS_SINGLE_PASS)


@pytest.mark.parametrize("B,L,lens,w,gl,alpha,gaps", LAYER_CASES)
def test_single_pass_layer_matches_oracle(sc, B, L, lens, w, gl, alpha, gaps):
    case = layer_case(B, L, 12, lens, w, gl, alpha, seed=L + w, gaps=gaps)
    if gaps:
        case["global_pos"] = np.unique(np.concatenate([[0], case["pos"][1, [5, 77]]])).astype(np.int32)
        case = layer_case(B, L, 12, lens, w, case["global_pos"], alpha, seed=L + w, gaps=gaps)
    _check_layer(case, _run_layer(sc, case, w))


def test_single_pass_full_size_layer_matches_oracle(sc):
    """Layer 0 of the L = 4096 workload (B = 2, 9 global tokens, salient keys
    x4): every O row, score and kept position against the oracle's layer."""
    wl = wk.CFG4
    inp = wk.make_inputs(wl, wk.stored_redraws(wl))
    dev = "cuda"
    Q, K, V = (bits_to_torch(inp[k][0], dev) for k in ("Q", "K", "V"))
    length = torch.full((wl.B,), wl.L, dtype=torch.int32, device=dev)
    pos = torch.arange(wl.L, dtype=torch.int32, device=dev).repeat(wl.B, 1).contiguous()
    gpos = [int(g) for g in inp["global_pos"]]
    alpha = float(inp["alpha"][0])
    ws = sc.new_workspace(wl.B, wl.L, wl.H, dev)
    O, s, po, lo = sc.layer_forward(Q, K, V, length, pos, wl.w, gpos, alpha, workspace=ws)
    assert sc.workspace_status(ws) == 0
    O = torch_bf16_to_f64(O)
    s, po, lo = s.cpu().numpy(), po.cpu().numpy(), lo.cpu().numpy()
    isg = np.zeros(wl.L, bool)
    isg[gpos] = True
    for b in range(wl.B):
        q, k, v = (wk.bf16_bits_to_f64(inp[t][0, b]) for t in ("Q", "K", "V"))
        Oe, se, keep = oracle.layer(q, k, v, isg, wl.w, alpha / wl.L)
        kept = list(np.nonzero(keep)[0])
        assert int(lo[b]) == len(kept)
        assert list(po[b, :len(kept)]) == kept
        check_o(O[b], Oe, f"sequence {b}")
        check_scores(s[b], se, f"sequence {b}")


WITH_TAIL = [wk.Workload("small_12x700", n_layers=12, B=2, L=700, w=64, n_extra_global=3, seed=3),
             wk.Workload("ragged_6x600", n_layers=6, B=3, L=600, w=128, ragged=(200, 600), seed=4),
             wk.Workload("salient4_4x1000", n_layers=4, B=1, L=1000, w=256, n_extra_global=8,
                         salient_frac=0.05, salient_scale=4.0, alpha_first=0.4, alpha_last=1.0,
                         seed=5)]


@pytest.mark.parametrize("wl", WITH_TAIL, ids=[w.name for w in WITH_TAIL])
def test_single_pass_stack_matches_oracle(sc, wl):
    inp, res, _ = resample_stack(wl)
    check_stack(wl, res, _run_stack(sc, wl, inp))
