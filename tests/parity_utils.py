"""Shared helpers of the parity tests: oracle runs with near-threshold
resampling, host<->device conversion of the bf16 bit patterns, comparisons.

The GPU side is reached only through the C ABI (paper_2310_07109_gb300.binding);
the expected values come only from the oracle.
"""
from __future__ import annotations

import numpy as np

import oracle
import workloads as wk

# tolerances of the parity bar
# bf16 attention outputs: 2e-2 absolute on the computed value, plus the bf16
# rounding the output format itself applies at that magnitude (half an ulp,
# 2^-9 |O|) and that of a dominant bf16 probability in P V (2^-9 |O|):
# |O_gpu - O| <= 2e-2 + 2^-8 |O|.
O_ATOL = 2e-2
O_RTOL = 2.0 ** -8
SCORE_ATOL = 1e-5      # scores (fp32 accumulation), absolute
MARGIN = 1e-4          # a token whose oracle score lies within MARGIN / n of theta is resampled


def near_threshold(scores, n, theta):
    """Current indices j >= 1 with |s_j - theta| < MARGIN / n (token 0 is kept regardless)."""
    s = np.asarray(scores[:n])
    bad = np.nonzero(np.abs(s - theta) < MARGIN / n)[0]
    return [int(j) for j in bad if j != 0]


def near_cut(scores, n, k):
    """Top-ratio rule: current indices j >= 1 whose oracle score lies within
    MARGIN / n of the midpoint between the lowest kept and the highest dropped
    score (token 0 is kept regardless and takes no part in the ranking)."""
    s = np.asarray(scores[1:n])
    if k - 1 <= 0 or k - 1 >= len(s):
        return []
    srt = np.sort(s)[::-1]
    cut = 0.5 * (srt[k - 2] + srt[k - 1])
    return [int(j) + 1 for j in np.nonzero(np.abs(s - cut) < MARGIN / n)[0]]


def near_boundary(wl, scores, n, value):
    """Tokens of one (layer, sequence) too close to the keep decision of ``wl``'s rule."""
    if wl.keep_rule == oracle.KEEP_TOP_RATIO:
        return near_cut(scores, n, oracle.top_count(value, n))
    theta = value if wl.keep_rule == oracle.KEEP_ABSOLUTE else value / n
    return near_threshold(scores, n, theta)


def resample_stack(wl: wk.Workload, max_rounds: int = 50, nthreads=None, overrides=None):
    """Draw ``wl`` and redraw (layer, token) Q/K rows until no oracle score of any
    layer lies within MARGIN / n of its keep decision (the threshold, or the cut
    between kept and dropped scores of the top-ratio rule).  Layers interact
    only through the kept set, so fixing the first offending layer and
    re-running converges.  ``overrides`` replaces entries of the drawn inputs
    (e.g. global_pos, pad_mask)."""
    redraws = {}
    for _ in range(max_rounds):
        inp = wk.make_inputs(wl, redraws)
        inp.update(overrides or {})
        res = oracle.stack(inp["Q"], inp["K"], inp["V"], inp["pad_mask"], inp["global_pos"],
                           wl.w, inp["alpha"], nthreads=nthreads, keep_rule=wl.keep_rule)
        bad = []
        for l in range(wl.n_layers):
            for b in range(wl.B):
                n = int(res["len"][l, b])
                if n == 0:
                    continue
                for j in near_boundary(wl, res["scores"][l, b], n, inp["alpha"][l]):
                    bad.append((l, b, int(res["pos"][l, b, j])))
            if bad:
                break
        if not bad:
            return inp, res, redraws
        for key in bad:
            redraws[key] = redraws.get(key, 0) + 1
    raise RuntimeError("near-threshold resampling did not converge for %s" % wl.describe())


def bits_to_torch(bits, device):
    import torch
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.to(device).view(torch.bfloat16)


def torch_bf16_to_f64(t):
    import torch
    bits = t.detach().to("cpu").view(torch.int16).numpy().view(np.uint16).astype(np.uint32)
    with np.errstate(invalid="ignore"):   # unused output slots may hold NaN patterns
        return (bits << 16).view(np.float32).astype(np.float64)


def layer_case(B, L, H, lens, w, gpos, alpha, seed, scale_k=2.0, gaps=False, max_rounds=50):
    """Current-order single-layer inputs with resampled near-threshold tokens.

    Returns dict(Q, K, V bits [B,L,H,64], pos [B,L] int32, len [B], global_pos,
    alpha, expected: list per sequence of (O, scores, kept positions)).
    """
    rng = np.random.default_rng(seed)
    Q, K, V = (np.empty((B, L, H, 64), np.uint16) for _ in range(3))
    pos = np.zeros((B, L), np.int32)
    for b in range(B):
        q, k, v = wk.random_layer(L, H, 64, seed * 100 + b, scale_k)
        Q[b], K[b], V[b] = q, k, v
        if gaps:
            rest = np.sort(rng.choice(np.arange(1, 4 * L), L - 1, replace=False))
            pos[b] = np.concatenate([[0], rest]).astype(np.int32)
        else:
            pos[b] = np.arange(L, dtype=np.int32)
    gset = set(int(g) for g in gpos)
    expected = []
    for b in range(B):
        n = int(lens[b])
        for rnd in range(max_rounds):
            if n == 0:
                expected.append((np.zeros((0, H, 64)), np.zeros(0), []))
                break
            q = wk.bf16_bits_to_f64(Q[b, :n])
            k = wk.bf16_bits_to_f64(K[b, :n])
            v = wk.bf16_bits_to_f64(V[b, :n])
            isg = np.array([int(p) in gset for p in pos[b, :n]])
            theta = alpha / n
            O, s, keep = oracle.layer(q, k, v, isg, w, theta)
            bad = near_threshold(s, n, theta)
            if not bad:
                expected.append((O, s, [int(p) for p, kp in zip(pos[b, :n], keep) if kp]))
                break
            for j in bad:
                qn, kn, _ = wk.random_layer(1, H, 64, seed * 7919 + b * 131 + j * 7 + rnd, scale_k)
                Q[b, j], K[b, j] = qn[0], kn[0]
        else:
            raise RuntimeError("layer resampling did not converge")
    return {"Q": Q, "K": K, "V": V, "pos": pos, "len": np.asarray(lens, np.int32),
            "global_pos": np.asarray(sorted(gset), np.int32), "alpha": alpha,
            "expected": expected}


def check_stack(wl, res, got):
    """A stack's results (numpy dict O as float64, scores, pos, len) against the
    oracle's: lengths and positions exactly, O and scores within tolerance."""
    np.testing.assert_array_equal(got["len"], res["len"])
    for l in range(wl.n_layers + 1):
        for b in range(wl.B):
            n = int(res["len"][l, b])
            np.testing.assert_array_equal(got["pos"][l, b, :n], res["pos"][l, b, :n],
                                          err_msg=f"layer {l} seq {b}")
    for l in range(wl.n_layers):
        for b in range(wl.B):
            n = int(res["len"][l, b])
            if n == 0:
                continue
            np.testing.assert_allclose(got["O"][l, b, :n], res["O"][l, b, :n], rtol=O_RTOL,
                                       atol=O_ATOL, err_msg=f"O layer {l} seq {b}")
            np.testing.assert_allclose(got["scores"][l, b, :n], res["scores"][l, b, :n], rtol=0,
                                       atol=SCORE_ATOL, err_msg=f"scores layer {l} seq {b}")
