"""GPU parity of the keep rules besides theta = alpha / n, against the fp64
oracle: an absolute threshold per layer (the schedule of RQ4) and the top-ratio
rule (the "top-k of the sequence length" family of the Pruning section: a layer
keeps ceil(rho n) tokens, the first and the best others, ties to the lower
index), through the per-layer kernels, the cluster kernel and the hand-over
between them, and through the single-layer call.

Top-ratio inputs are resampled until no oracle score lies within 1e-4 / n of
the cut between kept and dropped scores, so the kept lists must match bit for
bit; exact ties (uniform attention) are checked against their closed form.
"""
import numpy as np
import pytest
import torch

import oracle
import workloads as wk
from parity_utils import (MARGIN, bits_to_torch, check_o, check_scores, check_stack,
                          resample_stack, torch_bf16_to_f64)
from test_gpu_parity import _run_stack

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    return sc


RULE_STACKS = [
    # per-layer kernels for the first layers, the cluster kernel after the hand-over
    wk.Workload("top_ratio_6x900", n_layers=6, B=2, L=900, w=64, n_extra_global=3,
                alpha_first=0.9, alpha_last=0.5, keep_rule=2, seed=31),
    wk.Workload("top_ratio_ragged_4x1300", n_layers=4, B=3, L=1300, w=128, ragged=(300, 1300),
                alpha_first=0.8, alpha_last=0.6, keep_rule=2, seed=32),
    wk.Workload("top_ratio_short_5x350", n_layers=5, B=2, L=350, w=48, n_extra_global=2,
                alpha_first=0.95, alpha_last=0.3, keep_rule=2, seed=33),
    wk.Workload("top_ratio_4096", n_layers=1, B=1, L=4096, w=256, n_extra_global=8,
                salient_frac=0.05, salient_scale=4.0, alpha_first=0.3, alpha_last=0.3,
                keep_rule=2, seed=34),
    wk.Workload("abs_theta_6x900", n_layers=6, B=2, L=900, w=64, n_extra_global=2,
                alpha_first=0.01 / 12, alpha_last=0.01 / 2, keep_rule=1, seed=35),
    wk.Workload("abs_theta_short_4x300", n_layers=4, B=2, L=300, w=64,
                alpha_first=0.002, alpha_last=0.006, keep_rule=1, seed=36),
]


_CACHE = {}


def _resampled(wl):
    if wl.name not in _CACHE:
        _CACHE[wl.name] = resample_stack(wl)
    return _CACHE[wl.name]


@pytest.mark.parametrize("no_tail", [False, True], ids=["with_tail", "per_layer_only"])
@pytest.mark.parametrize("wl", RULE_STACKS, ids=[w.name for w in RULE_STACKS])
def test_rule_stack_matches_oracle(sc, wl, no_tail):
    if no_tail and wl.L > 2 * sc.TAIL_MAX_LEN and wl.n_layers == 1:
        pytest.skip("a single long layer runs in the per-layer kernels either way")
    inp, res, _ = _resampled(wl)
    check_stack(wl, res, _run_stack(sc, wl, inp, no_tail))


def test_top_ratio_lengths_follow_the_ratio(sc):
    wl = RULE_STACKS[0]
    inp, res, _ = _resampled(wl)
    got = _run_stack(sc, wl, inp)
    for l in range(wl.n_layers):
        for b in range(wl.B):
            assert got["len"][l + 1, b] == oracle.top_count(inp["alpha"][l], got["len"][l, b])


@pytest.mark.parametrize("L", [300, 600], ids=["cluster_kernel", "per_layer"])
def test_top_ratio_exact_ties_keep_the_first(sc, L):
    """Zero queries and a window over the whole sequence: every score is the
    same, so the ties at the cut go to the lowest indices (tokens 0..k-1)."""
    wl = wk.Workload("ties", n_layers=2, B=2, L=L, w=L, alpha_first=0.5, alpha_last=0.3,
                     keep_rule=2, seed=37)
    inp = wk.make_inputs(wl)
    inp["Q"][:] = 0
    got = _run_stack(sc, wl, inp)
    n = L
    for l in range(wl.n_layers):
        k = oracle.top_count(inp["alpha"][l], n)
        assert (got["len"][l + 1] == k).all()
        assert (got["pos"][l + 1, :, :k] == np.arange(k)).all()
        assert (got["scores"][l, :, 1:n] == got["scores"][l, :, 1:2]).all()
        n = k


def test_top_ratio_extremes(sc):
    wl = wk.Workload("extremes", n_layers=2, B=2, L=700, w=64, alpha_first=1.0, alpha_last=0.0,
                     keep_rule=2, seed=38)
    inp = wk.make_inputs(wl)
    got = _run_stack(sc, wl, inp)
    assert (got["len"][1] == 700).all()          # ratio 1 keeps every token
    assert (got["len"][2] == 1).all()            # ratio 0 keeps the first token only
    assert (got["pos"][2, :, 0] == 0).all()


def test_layer_call_top_ratio(sc):
    """sc_layer_forward with the top-ratio rule: one layer, two sequences of
    different lengths, kept lists against the oracle's ranking."""
    dev = "cuda"
    B, L, H, w, rho = 2, 1024, 12, 128, 0.6
    lens = [1024, 777]
    rng_seed = 39
    Q, K, V = (np.empty((B, L, H, 64), np.uint16) for _ in range(3))
    exp = []
    for b in range(B):
        n = lens[b]
        for rnd in range(50):
            q, k, v = wk.random_layer(L, H, 64, rng_seed * 100 + b * 10 + rnd, 2.0)
            Q[b], K[b], V[b] = q, k, v
            O, s, _ = oracle.layer(wk.bf16_bits_to_f64(q[:n]), wk.bf16_bits_to_f64(k[:n]),
                                   wk.bf16_bits_to_f64(v[:n]), np.arange(n) == 0, w, 0.0)
            kk = oracle.top_count(rho, n)
            srt = np.sort(s[1:])[::-1]
            if srt[kk - 2] - srt[kk - 1] >= 2 * MARGIN / n:
                exp.append((O, s, np.nonzero(oracle.keep_top(s, kk))[0]))
                break
        else:
            raise RuntimeError("no draw with a clear cut")
    pos = np.tile(np.arange(L, dtype=np.int32), (B, 1))
    Qt, Kt, Vt = (bits_to_torch(x, dev) for x in (Q, K, V))
    ws = sc.new_workspace(B, L, H, dev)
    O, s, po, lo = sc.layer_forward(Qt, Kt, Vt, torch.tensor(lens, dtype=torch.int32, device=dev),
                                    torch.from_numpy(pos).to(dev), w, [0], rho, workspace=ws,
                                    keep_rule=sc.SC_KEEP_TOP_RATIO)
    assert sc.workspace_status(ws) == 0
    O, s, po, lo = torch_bf16_to_f64(O), s.cpu().numpy(), po.cpu().numpy(), lo.cpu().numpy()
    for b in range(B):
        n = lens[b]
        Oe, se, kept = exp[b]
        assert lo[b] == len(kept)
        assert list(po[b, :len(kept)]) == list(kept)
        check_o(O[b, :n], Oe, f"sequence {b}")
        check_scores(s[b, :n], se, f"sequence {b}")
