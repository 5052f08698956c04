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
O_ATOL = 2e-2          # bf16 attention outputs: max-abs against the fp64 oracle
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


def resample_stack(wl: wk.Workload, max_rounds: int = 50, nthreads=None, overrides=None,
                   o_dtype=None, redraws=None):
    """Draw ``wl`` and redraw (layer, token) Q/K rows until no oracle score of any
    layer lies within MARGIN / n of its keep decision (the threshold, or the cut
    between kept and dropped scores of the top-ratio rule).

    Sequences are independent and layers interact only through the kept set,
    so each sequence is run layer by layer with the oracle's single-layer call:
    a layer with offending tokens has their rows redrawn and is run again (only
    that layer of that sequence) before the next layer starts.  The stack
    semantics are those of ``oracle.stack``: padding removed before layer 0,
    layer l reads the rows of its current tokens at their original positions,
    the kept tokens move on in order.  ``overrides`` replaces entries of the
    drawn inputs (e.g. global_pos, pad_mask); ``redraws`` are redraws to start
    from (e.g. the stored ones of ``stored_redraws``).

    Returns (inputs, results, redraws); results is a dict like ``oracle.stack``'s
    (O [nl,B,L,H,d] in ``o_dtype``, float64 by default; NaN / -1 past each
    length).
    """
    redraws = dict(redraws or {})
    inp = wk.make_inputs(wl, redraws)
    inp.update(overrides or {})
    nl, B, L, H, d = wl.n_layers, wl.B, wl.L, wl.H, wl.d
    alpha = np.asarray(inp["alpha"], np.float64)
    gset = set(int(g) for g in inp["global_pos"])
    mask = inp["pad_mask"]
    O = np.full((nl, B, L, H, d), np.nan, dtype=o_dtype or np.float64)
    scores = np.full((nl, B, L), np.nan)
    pos = np.full((nl + 1, B, L), -1, np.int32)
    lens = np.zeros((nl + 1, B), np.int32)
    for b in range(B):
        cur = np.arange(L) if mask is None else np.nonzero(mask[b])[0]
        lens[0, b] = len(cur)
        pos[0, b, :len(cur)] = cur
        for l in range(nl):
            n = len(cur)
            if n > 0:
                isg = np.array([int(c) in gset for c in cur])
                for _ in range(max_rounds):
                    q, k, v = (wk.bf16_bits_to_f64(inp[t][l, b, cur]) for t in ("Q", "K", "V"))
                    if wl.keep_rule == oracle.KEEP_RELATIVE:
                        theta = alpha[l] / n
                    else:
                        theta = alpha[l] if wl.keep_rule == oracle.KEEP_ABSOLUTE else 0.0
                    Ol, sl, keep = oracle.layer(q, k, v, isg, wl.w, theta, nthreads=nthreads)
                    if wl.keep_rule == oracle.KEEP_TOP_RATIO:
                        keep = oracle.keep_top(sl, oracle.top_count(alpha[l], n))
                    bad = near_boundary(wl, sl, n, alpha[l])
                    if not bad:
                        break
                    for j in bad:
                        key = (l, b, int(cur[j]))
                        redraws[key] = redraws.get(key, 0) + 1
                        wk.redraw_row(wl, inp, l, b, int(cur[j]), redraws[key])
                else:
                    raise RuntimeError("near-threshold resampling did not converge for %s"
                                       % wl.describe())
                O[l, b, :n] = Ol
                scores[l, b, :n] = sl
                cur = cur[keep]
            lens[l + 1, b] = len(cur)
            pos[l + 1, b, :len(cur)] = cur
    return inp, {"O": O, "scores": scores, "pos": pos, "len": lens}, redraws


def stored_redraws(wl: wk.Workload):
    """The redraws of ``wl`` stored in tests/golden/redraws.json (written by
    tests/golden/make_redraws.py from the oracle alone); {} for workloads it
    does not list."""
    return wk.stored_redraws(wl)


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


# largest errors seen by the comparisons of this session, per test (printed in
# the terminal summary by conftest.py)
ERRORS = {}


def record(o_err=None, s_err=None):
    """Keep the largest O / score error of the running test."""
    import os
    name = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]
    cur = ERRORS.setdefault(name, [0.0, 0.0])
    if o_err is not None:
        cur[0] = max(cur[0], float(o_err))
    if s_err is not None:
        cur[1] = max(cur[1], float(s_err))


def check_o(got, ref, what=""):
    """Attention outputs: max |got - ref| <= O_ATOL (``got`` float, or bf16 bits
    as uint16); returns the max error."""
    got = np.asarray(got)
    if got.dtype == np.uint16:
        got = wk.bf16_bits_to_f32(got)
    err = float(np.max(np.abs(got.astype(np.float64) - np.asarray(ref, np.float64)),
                       initial=0.0))
    record(o_err=err)
    assert err <= O_ATOL, f"O max-abs error {err:.4g} > {O_ATOL} {what}"
    return err


def check_scores(got, ref, what=""):
    err = float(np.max(np.abs(np.asarray(got, np.float64) - np.asarray(ref, np.float64)),
                       initial=0.0))
    record(s_err=err)
    assert err <= SCORE_ATOL, f"score max-abs error {err:.4g} > {SCORE_ATOL} {what}"
    return err


def check_stack(wl, res, got):
    """A stack's results (dict: O as float or bf16 bits, scores, pos, len) against
    the oracle's: lengths and positions exactly, every O row and every score of
    every layer within the bar.  Returns (max O error, max score error)."""
    np.testing.assert_array_equal(got["len"], res["len"])
    for l in range(wl.n_layers + 1):
        for b in range(wl.B):
            n = int(res["len"][l, b])
            np.testing.assert_array_equal(got["pos"][l, b, :n], res["pos"][l, b, :n],
                                          err_msg=f"layer {l} seq {b}")
    eo = es = 0.0
    for l in range(wl.n_layers):
        for b in range(wl.B):
            n = int(res["len"][l, b])
            if n == 0:
                continue
            eo = max(eo, check_o(got["O"][l, b, :n], res["O"][l, b, :n], f"layer {l} seq {b}"))
            es = max(es, check_scores(got["scores"][l, b, :n], res["scores"][l, b, :n],
                                      f"layer {l} seq {b}"))
    return eo, es
