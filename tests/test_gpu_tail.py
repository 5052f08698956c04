"""GPU parity of the cluster kernel that runs the remaining layers of a
sequence once at most TAIL_MAX_LEN (384) tokens are left (one cluster of H CTAs
per sequence, all such layers in one launch), against the fp64 oracle.

Covered: every layer in the cluster kernel with a window narrower than the
sequence and global tokens (masked path), a window that covers every pair,
sequences of one, two and three 128-row tiles (above 256 tokens the keys and
queries are processed in two halves), cluster sizes H = 4, 12 and 16, more
clusters than the GPU holds at once, the hand-over from the per-layer kernels
in the middle of a stack, empty and one-token sequences, and the launch plan the
library reports.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wk
from parity_utils import check_stack, resample_stack
from test_gpu_parity import _run_stack

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    return sc


TAIL_STACKS = [
    wk.Workload("all_tail_w64_ragged", n_layers=6, B=3, L=256, w=64, n_extra_global=4,
                ragged=(40, 256), seed=11),
    wk.Workload("all_tail_full_window", n_layers=4, B=2, L=200, w=256, n_extra_global=2, seed=12),
    wk.Workload("all_tail_h4", n_layers=3, B=2, L=180, H=4, w=32, n_extra_global=1, seed=13),
    wk.Workload("all_tail_h16", n_layers=3, B=2, L=160, H=16, w=48, n_extra_global=3, seed=14),
    wk.Workload("many_clusters_b20", n_layers=3, B=20, L=130, w=40, seed=15),
    wk.Workload("handover_1200", n_layers=5, B=2, L=1200, w=128, n_extra_global=6,
                salient_frac=0.08, salient_scale=4.0, alpha_first=0.5, alpha_last=1.0, seed=16),
    # above 256 tokens: two key / query halves per tile
    wk.Workload("halves_384_w64", n_layers=4, B=2, L=384, w=64, n_extra_global=5, seed=19),
    wk.Workload("halves_320_full", n_layers=3, B=3, L=320, w=256, n_extra_global=2,
                ragged=(260, 320), seed=20),
    wk.Workload("halves_theta_small", n_layers=6, B=2, L=380, w=100, n_extra_global=3,
                alpha_first=0.05, alpha_last=0.2, seed=21),
]


@pytest.mark.parametrize("wl", TAIL_STACKS, ids=[w.name for w in TAIL_STACKS])
def test_tail_stack_matches_oracle(sc, wl):
    inp, res, _ = resample_stack(wl)
    check_stack(wl, res, _run_stack(sc, wl, inp))


def test_handover_happens_mid_stack(sc):
    """The hand-over workload really uses both paths: layer 0 has more than
    TAIL_MAX_LEN tokens and a later layer at most that many."""
    wl = next(w for w in TAIL_STACKS if w.name == "handover_1200")
    inp, res, _ = resample_stack(wl)
    assert (res["len"][0] > sc.TAIL_MAX_LEN).all()
    assert (res["len"][wl.n_layers - 1] <= sc.TAIL_MAX_LEN).all()


def test_halves_cases_have_more_than_two_tiles(sc):
    """The 'halves' workloads keep more than 256 tokens in some layer, so the
    two-half path of the cluster kernel runs."""
    for w in TAIL_STACKS:
        if w.name.startswith("halves"):
            _, res, _ = resample_stack(w)
            assert (res["len"][: w.n_layers] > 256).any(), w.name


def test_tail_empty_and_single_token_sequences(sc):
    wl = wk.Workload("degenerate", n_layers=4, B=3, L=96, w=16, n_extra_global=2, seed=17)
    inp = wk.make_inputs(wl)
    mask = np.ones((wl.B, wl.L), np.uint8)
    mask[0, :] = 0          # empty sequence
    mask[1, 1:] = 0         # only its first token
    inp["pad_mask"] = mask
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], mask, inp["global_pos"], wl.w, inp["alpha"])
    got = _run_stack(sc, wl, inp)
    assert (got["len"][:, 0] == 0).all()
    assert (got["len"][:, 1] == 1).all()
    check_stack(wl, res, got)


def test_tail_theta_zero_keeps_everything(sc):
    wl = wk.Workload("theta0_short", n_layers=3, B=2, L=256, w=100, n_extra_global=3,
                     alpha_first=0.0, alpha_last=0.0, seed=18)
    inp = wk.make_inputs(wl)
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], None, inp["global_pos"], wl.w, inp["alpha"])
    got = _run_stack(sc, wl, inp)
    assert (got["len"] == 256).all()
    check_stack(wl, res, got)


def test_launch_plan(sc):
    g = [0, 5]
    # every sequence starts in the cluster kernel: global lookup + one launch
    assert sc.stack_launch_count(12, 2, 256, 12, 64, g, False) == 2
    assert sc.stack_launch_count(12, 2, sc.TAIL_MAX_LEN, 12, 64, g, False) == 2
    # per-layer kernels (rows, cols, and a gather between layers) + the cluster kernel
    assert sc.stack_launch_count(12, 2, 700, 12, 64, g, False) == 1 + 12 * 2 + 11 + 1
    assert sc.stack_launch_count(12, 2, 700, 12, 64, g, True) == 2 + 12 * 2 + 11 + 1
    assert sc.stack_launch_count(12, 2, 700, 12, 64, g, False, no_tail=True) == 1 + 12 * 2 + 11
    # clusters of more than 16 CTAs cannot be formed: per-layer kernels only
    assert sc.stack_launch_count(3, 1, 200, 20, 64, g, False) == 1 + 3 * 2 + 2
