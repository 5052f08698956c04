"""Pins of the fp64 oracle against facts fixed outside itself (CPU only).

Each test pins the oracle to something other than its own code: hand-worked
fixtures under tests/golden/, a library routine (torch's fp64 scaled
dot-product attention) on the dense masked problem, closed forms (uniform
softmax, V = 1), invariants of a row-stochastic matrix, and brute force on tiny
inputs.  A plausible slip in the oracle -- a window off by one, a dropped
global row or column, a transposed Q/K, a wrong scale, row sums instead of
column sums, the wrong head normalisation, a strict instead of non-strict
threshold, a broken compaction -- fails at least one of them.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import workloads as wk

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    out = {"allowed": {}}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            if key == "allowed":
                out["allowed"][int(vals[0])] = [int(v) for v in vals[1:]]
            elif key in ("colsum", "alpha"):
                out[key] = [float(v) for v in vals]
            else:
                out[key] = [int(v) for v in vals]
    return out


def _globals_mask(n, gl):
    m = np.zeros(n, dtype=bool)
    m[list(gl)] = True
    return m


# --------------------------------------------------------------------------
# hand-worked fixtures
# --------------------------------------------------------------------------
def test_ten_token_example_uniform():
    g = _read_golden("ten_token_uniform.txt")
    n, w = g["n"][0], g["w"][0]
    isg = _globals_mask(n, g["global"])
    rng = np.random.default_rng(5)
    d = 4
    Q = np.zeros((n, 1, d))
    K = rng.standard_normal((n, 1, d))
    V = rng.standard_normal((n, 1, d))
    theta = g["alpha"][0] / n
    O, s, keep = oracle.layer(Q, K, V, isg, w, theta)
    # uniform attention: each output row is the mean of V over the hand-listed set
    for i, A in g["allowed"].items():
        np.testing.assert_allclose(O[i, 0], V[A, 0].mean(axis=0), rtol=0, atol=1e-13)
    np.testing.assert_allclose(s, np.array(g["colsum"]) / n, rtol=0, atol=1e-14)
    assert list(np.nonzero(keep)[0]) == g["kept"]


def test_four_token_two_heads_uniform():
    g = _read_golden("four_token_uniform.txt")
    n, w, H = g["n"][0], g["w"][0], g["H"][0]
    isg = _globals_mask(n, g["global"])
    rng = np.random.default_rng(6)
    Q = np.zeros((n, H, 3))
    K = rng.standard_normal((n, H, 3))
    V = rng.standard_normal((n, H, 3))
    _, s, _ = oracle.layer(Q, K, V, isg, w, 0.0)
    np.testing.assert_allclose(s, np.array(g["colsum"]) / n, rtol=0, atol=1e-14)


def test_hand_logits_global_row_and_column():
    """n = 4, d = 1, H = 1, w = 0, token 2 global, chosen logits.

    Keys carry log-weights (q = 1 for every row, k_j = ln a_j, scale 1/sqrt(1)),
    so P[i, j] = a_j / sum_{j' in A(i)} a_j'.  With w = 0 a non-global row sees
    itself and token 2; the global row 2 sees all four.  Worked by hand with
    a = (1, 2, 3, 4):
      row 0: {0, 2}       -> P = 1/4, 3/4
      row 1: {1, 2}       -> P = 2/5, 3/5
      row 2: {0, 1, 2, 3} -> P = 1/10, 2/10, 3/10, 4/10
      row 3: {2, 3}       -> P = 3/7, 4/7
    column sums: c0 = 1/4 + 1/10, c1 = 2/5 + 2/10, c2 = 3/4 + 3/5 + 3/10 + 3/7,
    c3 = 4/10 + 4/7.
    """
    a = np.array([1.0, 2.0, 3.0, 4.0])
    Q = np.ones((4, 1, 1))
    K = np.log(a).reshape(4, 1, 1)
    V = np.arange(4, dtype=np.float64).reshape(4, 1, 1) * 10.0  # v_j = 10 j
    isg = _globals_mask(4, [2])
    O, s, _ = oracle.layer(Q, K, V, isg, 0, 0.0)
    c = np.array([1 / 4 + 1 / 10, 2 / 5 + 2 / 10, 3 / 4 + 3 / 5 + 3 / 10 + 3 / 7,
                  4 / 10 + 4 / 7])
    np.testing.assert_allclose(s, c / 4, rtol=0, atol=1e-15)
    o = np.array([10 * 3 / 4 * 2, 10 * (2 / 5 * 1 + 3 / 5 * 2),
                  10 * (2 / 10 + 6 / 10 + 12 / 10), 10 * (3 / 7 * 2 + 4 / 7 * 3)])
    np.testing.assert_allclose(O[:, 0, 0], o, rtol=0, atol=1e-13)


# --------------------------------------------------------------------------
# library routine on the dense masked problem (brute force, tiny inputs)
# --------------------------------------------------------------------------
def _dense_mask(n, w, isg):
    i = np.arange(n)[:, None]
    j = np.arange(n)[None, :]
    return (np.abs(i - j) <= w) | isg[None, :] | isg[:, None]


CASES = [(1, 1, 4, 0, []), (2, 1, 4, 1, []), (5, 3, 4, 1, [0]), (17, 2, 64, 3, [0, 9]),
         (33, 3, 64, 0, [0, 32]), (33, 2, 8, 33, [0]), (40, 2, 16, 4, [0, 1, 2, 39]),
         (64, 1, 64, 7, [5])]


@pytest.mark.parametrize("n,H,d,w,gl", CASES)
def test_against_torch_sdpa_masked(n, H, d, w, gl):
    rng = np.random.default_rng(n * 100 + w)
    Q = rng.standard_normal((n, H, d))
    K = rng.standard_normal((n, H, d)) * 1.7
    V = rng.standard_normal((n, H, d))
    isg = _globals_mask(n, gl)
    O, s, _ = oracle.layer(Q, K, V, isg, w, 0.0)
    mask = torch.from_numpy(_dense_mask(n, w, isg))
    q = torch.from_numpy(Q).permute(1, 0, 2)  # [H, n, d]
    k = torch.from_numpy(K).permute(1, 0, 2)
    v = torch.from_numpy(V).permute(1, 0, 2)
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=mask)
    np.testing.assert_allclose(O, ref.permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)
    # probabilities themselves: attention applied to the identity gives P
    eye = torch.eye(n, dtype=torch.float64).expand(H, n, n)
    P = torch.nn.functional.scaled_dot_product_attention(q, k, eye, attn_mask=mask)
    np.testing.assert_allclose(s, P.sum(dim=(0, 1)).numpy() / (H * n), rtol=0, atol=1e-13)


@pytest.mark.parametrize("n,w", [(30, 29), (30, 45), (7, 6)])
def test_window_covering_sequence_is_full_attention(n, w):
    rng = np.random.default_rng(n + w)
    H, d = 2, 16
    Q, K, V = (rng.standard_normal((n, H, d)) for _ in range(3))
    O, s, _ = oracle.layer(Q, K, V, _globals_mask(n, [0]), w, 0.0)
    q, k, v = (torch.from_numpy(x).permute(1, 0, 2) for x in (Q, K, V))
    ref = torch.nn.functional.scaled_dot_product_attention(q, k, v)
    np.testing.assert_allclose(O, ref.permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)
    P = torch.softmax(q @ k.transpose(1, 2) / np.sqrt(d), dim=-1)
    np.testing.assert_allclose(s, P.sum(dim=(0, 1)).numpy() / (H * n), atol=1e-13)


# --------------------------------------------------------------------------
# invariants and closed forms
# --------------------------------------------------------------------------
def _medium(seed=3, n=200, H=4, d=64):
    rng = np.random.default_rng(seed)
    Q = rng.standard_normal((n, H, d))
    K = rng.standard_normal((n, H, d)) * 2.0
    V = rng.standard_normal((n, H, d))
    return Q, K, V


def test_scores_are_a_distribution():
    Q, K, V = _medium()
    n = Q.shape[0]
    isg = _globals_mask(n, [0, 50, 199])
    _, s, keep = oracle.layer(Q, K, V, isg, 16, 1.0 / n)
    assert abs(s.sum() - 1.0) < 1e-12
    assert abs(s.mean() - 1.0 / n) < 1e-15
    assert (s >= 0).all()
    assert keep[0]


def test_rows_sum_to_one_via_unit_values():
    Q, K, _ = _medium(seed=4)
    n, H, d = Q.shape
    isg = _globals_mask(n, [0, 13])
    O, _, _ = oracle.layer(Q, K, np.ones((n, H, d)), isg, 9, 0.0)
    np.testing.assert_allclose(O, 1.0, rtol=0, atol=1e-12)


def test_threshold_extremes_and_token0():
    Q, K, V = _medium(seed=5, n=64)
    n = Q.shape[0]
    isg = _globals_mask(n, [0])
    _, s, keep = oracle.layer(Q, K, V, isg, 8, 0.0)
    assert keep.all()
    _, _, keep = oracle.layer(Q, K, V, isg, 8, np.inf)
    assert list(np.nonzero(keep)[0]) == [0]
    # keep test is >=: a threshold equal to a score keeps that token
    _, s, _ = oracle.layer(Q, K, V, isg, 8, 0.0)
    j = int(np.argsort(s)[n // 2])
    _, _, keep = oracle.layer(Q, K, V, isg, 8, float(s[j]))
    assert keep[j]
    assert (keep[1:] == (s[1:] >= s[j])).all()


def test_sampled_matches_full():
    Q, K, V = _medium(seed=6, n=150, H=3)
    n = Q.shape[0]
    isg = _globals_mask(n, [0, 70])
    O, s, _ = oracle.layer(Q, K, V, isg, 11, 0.0)
    rows = [0, 1, 70, 71, 149]
    cols = [0, 5, 70, 100, 149]
    Os, ss = oracle.layer_sampled(Q, K, V, isg, 11, rows, cols)
    np.testing.assert_allclose(Os, O[rows], rtol=0, atol=1e-13)
    np.testing.assert_allclose(ss, s[cols], rtol=0, atol=1e-15)


# --------------------------------------------------------------------------
# the stack: gather by original position, compaction, padding
# --------------------------------------------------------------------------
def _small_stack(ragged=None, extra=0, L=96, nl=4, w=5):
    wl = wk.Workload("t", n_layers=nl, B=3, L=L, H=2, w=w, n_extra_global=extra,
                     ragged=ragged, alpha_first=0.5, alpha_last=1.1, seed=9)
    return wl, wk.make_inputs(wl)


def test_stack_equals_composed_layers():
    wl, inp = _small_stack(ragged=(40, 96), extra=3)
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], inp["pad_mask"], inp["global_pos"],
                       wl.w, inp["alpha"])
    gset = set(inp["global_pos"].tolist())
    for b in range(wl.B):
        pos = [p for p in range(wl.L) if inp["pad_mask"][b, p]]
        assert res["len"][0, b] == len(pos)
        for l in range(wl.n_layers):
            n = len(pos)
            assert list(res["pos"][l, b, :n]) == pos
            q = wk.bf16_bits_to_f64(inp["Q"][l, b, pos])
            k = wk.bf16_bits_to_f64(inp["K"][l, b, pos])
            v = wk.bf16_bits_to_f64(inp["V"][l, b, pos])
            isg = np.array([p in gset for p in pos])
            O, s, keep = oracle.layer(q, k, v, isg, wl.w, inp["alpha"][l] / n)
            np.testing.assert_array_equal(res["scores"][l, b, :n], s)
            np.testing.assert_array_equal(res["O"][l, b, :n], O)
            pos = [p for p, kp in zip(pos, keep) if kp]
            assert res["len"][l + 1, b] == len(pos)
            assert pos[0] == res["pos"][0, b, 0]  # the first token always survives


def test_padding_is_inert():
    wl, inp = _small_stack(ragged=(30, 80))
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], inp["pad_mask"], inp["global_pos"],
                       wl.w, inp["alpha"])
    rng = np.random.default_rng(1)
    Q2, K2, V2 = (x.copy() for x in (inp["Q"], inp["K"], inp["V"]))
    pad = inp["pad_mask"] == 0
    for X in (Q2, K2, V2):
        X[:, pad] = rng.integers(0, 0x3F80, size=X[:, pad].shape, dtype=np.uint16)
    res2 = oracle.stack(Q2, K2, V2, inp["pad_mask"], inp["global_pos"], wl.w, inp["alpha"])
    for key in ("pos", "len"):
        np.testing.assert_array_equal(res[key], res2[key])
    np.testing.assert_array_equal(np.nan_to_num(res["scores"]), np.nan_to_num(res2["scores"]))
    np.testing.assert_array_equal(np.nan_to_num(res["O"]), np.nan_to_num(res2["O"]))


def test_pruning_shrinks_and_preserves_order():
    wl, inp = _small_stack(L=128, nl=6)
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], None, inp["global_pos"], wl.w,
                       inp["alpha"])
    for b in range(wl.B):
        for l in range(wl.n_layers):
            n0, n1 = res["len"][l, b], res["len"][l + 1, b]
            assert 1 <= n1 <= n0
            cur, nxt = res["pos"][l, b, :n0], res["pos"][l + 1, b, :n1]
            assert (np.diff(nxt) > 0).all()
            assert set(nxt.tolist()) <= set(cur.tolist())
            s = res["scores"][l, b, :n0]
            theta = inp["alpha"][l] / n0
            expect = [p for c, p in enumerate(cur) if c == 0 or s[c] >= theta]
            assert list(nxt) == expect


# --------------------------------------------------------------------------
# the generator's bf16 rounding against torch's conversion
# --------------------------------------------------------------------------
def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).standard_normal(100_000).astype(np.float32) * 7
    x[:4] = [1.00390625, 1.01171875, -2.0078125, 0.0]  # exact ties
    ours = wk.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)
    np.testing.assert_array_equal(wk.bf16_bits_to_f32(ours),
                                  torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_generator_is_deterministic_and_redraw_is_local():
    wl = wk.Workload("t", n_layers=2, B=2, L=64, H=2, seed=4)
    a = wk.make_inputs(wl)
    b = wk.make_inputs(wl)
    for k in ("Q", "K", "V"):
        np.testing.assert_array_equal(a[k], b[k])
    c = wk.make_inputs(wl, {(1, 0, 7): 1})
    diff = np.argwhere((a["Q"] != c["Q"]).any(axis=(3, 4)))
    assert diff.tolist() == [[1, 0, 7]]
    assert (a["V"] == c["V"]).all()


# --------------------------------------------------------------------------
# the other keep rules: an absolute threshold per layer (RQ4's schedule) and
# a kept ratio per layer (the "top-k of the sequence length" family of the
# Pruning section)
# --------------------------------------------------------------------------
def test_top_count_closed_forms():
    assert oracle.top_count(1.0, 37) == 37
    assert oracle.top_count(0.0, 37) == 1
    assert oracle.top_count(0.5, 7) == 4
    assert oracle.top_count(0.5, 8) == 4
    assert oracle.top_count(2.0, 5) == 5
    assert oracle.top_count(0.25, 0) == 0
    # the ratio is the float32 a library caller passes: float32(0.3) is a
    # little above 0.3, so 10 tokens keep 4
    assert float(np.float32(0.3)) > 0.3
    assert oracle.top_count(0.3, 10) == 4


@pytest.mark.parametrize("n,k,seed", [(1, 1, 0), (2, 1, 1), (2, 2, 2), (50, 1, 3),
                                      (50, 17, 4), (50, 50, 5), (300, 123, 6)])
def test_keep_top_matches_stable_sort(n, k, seed):
    rng = np.random.default_rng(seed)
    s = rng.random(n)
    if n > 10:
        s[5:9] = s[20 % n]          # ties, resolved by the lower index
    keep = oracle.keep_top(s, k)
    order = 1 + np.argsort(-s[1:], kind="stable")   # numpy's stable sort
    expect = np.zeros(n, bool)
    expect[0] = True
    expect[order[:k - 1]] = True
    np.testing.assert_array_equal(keep, expect)
    assert keep.sum() == k


def test_keep_top_ignores_token0_score():
    s = np.array([0.0, 0.3, 0.1, 0.3, 0.2])
    assert list(np.nonzero(oracle.keep_top(s, 3))[0]) == [0, 1, 3]
    s[0] = 9.0   # a large first score takes no other token's place
    assert list(np.nonzero(oracle.keep_top(s, 3))[0]) == [0, 1, 3]


def test_uniform_attention_keeps_the_first_k():
    # zero queries with a window covering the sequence: every probability is
    # 1/n, every score the same, so the ties keep the lowest indices
    n, H, d = 40, 3, 8
    rng = np.random.default_rng(2)
    Q = np.zeros((n, H, d))
    K = rng.standard_normal((n, H, d))
    V = rng.standard_normal((n, H, d))
    _, s, _ = oracle.layer(Q, K, V, _globals_mask(n, [0]), n, 0.0)
    assert (s == s[0]).all()
    k = oracle.top_count(0.3, n)
    assert list(np.nonzero(oracle.keep_top(s, k))[0]) == list(range(k))


def test_stack_top_ratio_lengths_and_sets():
    wl, inp = _small_stack(ragged=(40, 96), extra=2, nl=5)
    rho = np.array([0.9, 0.75, 0.6, 0.5, 0.35])
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], inp["pad_mask"], inp["global_pos"],
                       wl.w, rho, keep_rule=oracle.KEEP_TOP_RATIO)
    for b in range(wl.B):
        for l in range(wl.n_layers):
            n = int(res["len"][l, b])
            k = int(np.ceil(float(np.float32(rho[l])) * n))   # closed form of the chain
            assert res["len"][l + 1, b] == min(max(k, 1), n)
            s = res["scores"][l, b, :n]
            keep = oracle.keep_top(s, k)
            cur = res["pos"][l, b, :n]
            assert list(res["pos"][l + 1, b, :res["len"][l + 1, b]]) == list(cur[keep])


def test_stack_absolute_threshold():
    wl, inp = _small_stack(L=128, nl=4)
    theta = np.array([0.002, 0.004, 0.006, 0.008])
    res = oracle.stack(inp["Q"], inp["K"], inp["V"], None, inp["global_pos"], wl.w, theta,
                       keep_rule=oracle.KEEP_ABSOLUTE)
    for b in range(wl.B):
        for l in range(wl.n_layers):
            n0, n1 = res["len"][l, b], res["len"][l + 1, b]
            s = res["scores"][l, b, :n0]
            cur = res["pos"][l, b, :n0]
            assert list(res["pos"][l + 1, b, :n1]) == [
                p for c, p in enumerate(cur) if c == 0 or s[c] >= theta[l]]
    # one layer without padding: theta = alpha / L is the relative rule
    one = {k: inp[k][:1] for k in ("Q", "K", "V")}
    a = oracle.stack(one["Q"], one["K"], one["V"], None, inp["global_pos"], wl.w, [0.8])
    t = oracle.stack(one["Q"], one["K"], one["V"], None, inp["global_pos"], wl.w, [0.8 / wl.L],
                     keep_rule=oracle.KEEP_ABSOLUTE)
    for key in ("pos", "len"):
        np.testing.assert_array_equal(a[key], t[key])


@pytest.mark.parametrize("rule,values", [(oracle.KEEP_TOP_RATIO, (0.9, 0.6)),
                                         (oracle.KEEP_ABSOLUTE, (0.004, 0.012))])
def test_resampling_clears_the_keep_decision(rule, values):
    from parity_utils import MARGIN, resample_stack
    wl = wk.Workload("t", n_layers=3, B=2, L=160, H=2, w=12, alpha_first=values[0],
                     alpha_last=values[1], keep_rule=rule, seed=21)
    inp, res, _ = resample_stack(wl)
    for l in range(wl.n_layers):
        for b in range(wl.B):
            n = int(res["len"][l, b])
            s = res["scores"][l, b, 1:n]
            kept = res["len"][l + 1, b] - 1
            if rule == oracle.KEEP_TOP_RATIO:
                srt = np.sort(s)[::-1]
                if 0 < kept < len(s):
                    assert srt[kept - 1] - srt[kept] >= 2 * MARGIN / n
            else:
                assert (np.abs(s - inp["alpha"][l]) >= MARGIN / n).all()


@pytest.mark.parametrize("wl", [
    wk.Workload("rs_rel", n_layers=4, B=3, L=200, H=2, w=20, n_extra_global=3, seed=31),
    wk.Workload("rs_ragged", n_layers=3, B=3, L=180, H=3, w=16, ragged=(60, 180), seed=32),
    wk.Workload("rs_abs", n_layers=3, B=2, L=150, H=2, w=12, alpha_first=0.004,
                alpha_last=0.012, keep_rule=oracle.KEEP_ABSOLUTE, seed=33),
    wk.Workload("rs_top", n_layers=3, B=2, L=150, H=2, w=12, alpha_first=0.9,
                alpha_last=0.6, keep_rule=oracle.KEEP_TOP_RATIO, seed=34),
], ids=lambda w: w.name)
def test_resampled_results_equal_the_oracle_stack(wl):
    """The resampler's layer-by-layer results are those of the oracle's own
    stack driver on the final (redrawn) inputs, and the redraws are exactly
    what make_inputs reproduces from the returned redraw counts."""
    from parity_utils import resample_stack
    inp, res, redraws = resample_stack(wl)
    again = wk.make_inputs(wl, redraws)
    for t in ("Q", "K", "V"):
        np.testing.assert_array_equal(again[t], inp[t])
    ref = oracle.stack(inp["Q"], inp["K"], inp["V"], inp["pad_mask"], inp["global_pos"], wl.w,
                       inp["alpha"], keep_rule=wl.keep_rule)
    np.testing.assert_array_equal(res["len"], ref["len"])
    np.testing.assert_array_equal(res["pos"], ref["pos"])
    np.testing.assert_array_equal(res["scores"], ref["scores"])
    np.testing.assert_array_equal(res["O"], ref["O"])


def test_stored_redraws_clear_the_benchmark_workload():
    """The benchmark times config 4 with the redraws stored in
    tests/golden/redraws.json: starting from them the resampler finds no token
    of any layer within the margin of its threshold, so they are complete."""
    from parity_utils import resample_stack
    stored = wk.stored_redraws(wk.CFG4)
    assert stored, "no stored redraws for the benchmark workload"
    _, _, redraws = resample_stack(wk.CFG4, redraws=stored, o_dtype=np.float32)
    assert redraws == stored
