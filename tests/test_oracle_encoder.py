"""Pins of the encoder-layer oracle (oracle/encoder.py) against definitions it
does not share code with: brute-force sums over integers, the normal CDF,
torch's layer norm, and closed forms of degenerate weights."""
import math

import numpy as np
import pytest
import torch

from oracle import encoder as enc


def test_linear_against_brute_force_integers():
    rng = np.random.default_rng(1)
    x = rng.integers(-4, 5, size=(5, 7)).astype(np.float64)
    W = rng.integers(-3, 4, size=(3, 7)).astype(np.float64)
    b = np.array([1.0, -2.0, 0.5])
    y = enc.linear(x, W, b)
    for i in range(5):
        for j in range(3):
            s = b[j]
            for k in range(7):
                s += x[i, k] * W[j, k]
            assert y[i, j] == s


def test_gelu_is_x_times_normal_cdf():
    from scipy.stats import norm
    x = np.linspace(-6, 6, 97)
    np.testing.assert_allclose(enc.gelu(x), x * norm.cdf(x), rtol=0, atol=1e-14)
    assert enc.gelu(np.array([0.0]))[0] == 0.0
    # erf is odd: gelu(x) - gelu(-x) = x
    np.testing.assert_allclose(enc.gelu(x) - enc.gelu(-x), x, rtol=0, atol=1e-14)


def test_layer_norm_moments_and_torch():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((6, 768)) * 3 + 1.5
    y = enc.layer_norm(x, np.ones(768), np.zeros(768))
    var = x.var(axis=1)
    np.testing.assert_allclose(y.mean(axis=1), 0, atol=1e-12)
    np.testing.assert_allclose((y ** 2).mean(axis=1), var / (var + enc.LN_EPS), rtol=1e-12)
    g, b = rng.standard_normal(768), rng.standard_normal(768)
    ref = torch.nn.functional.layer_norm(torch.from_numpy(x), (768,), torch.from_numpy(g),
                                         torch.from_numpy(b), eps=enc.LN_EPS).numpy()
    np.testing.assert_allclose(enc.layer_norm(x, g, b), ref, rtol=0, atol=1e-12)


def test_qkv_splits_the_rows_of_the_weight():
    rng = np.random.default_rng(3)
    D = 8
    X = rng.standard_normal((4, D))
    W = rng.standard_normal((3 * D, D))
    bq = rng.standard_normal(3 * D)
    q, k, v = enc.qkv(X, W, bq)
    np.testing.assert_allclose(q, X @ W[:D].T + bq[:D], atol=1e-13)
    np.testing.assert_allclose(k, X @ W[D:2 * D].T + bq[D:2 * D], atol=1e-13)
    np.testing.assert_allclose(v, X @ W[2 * D:].T + bq[2 * D:], atol=1e-13)


def _weights(D, rng, zero_o=False, zero_2=False):
    W_o = np.zeros((D, D)) if zero_o else rng.standard_normal((D, D)) / math.sqrt(D)
    b_o = np.zeros(D) if zero_o else rng.standard_normal(D) * 0.1
    W_1 = rng.standard_normal((4 * D, D)) / math.sqrt(D)
    W_2 = np.zeros((D, 4 * D)) if zero_2 else rng.standard_normal((D, 4 * D)) / math.sqrt(4 * D)
    b_2 = np.zeros(D) if zero_2 else rng.standard_normal(D) * 0.1
    return dict(W_o=W_o, b_o=b_o, g1=1 + 0.1 * rng.standard_normal(D), be1=0.1 * rng.standard_normal(D),
                W_1=W_1, b_1=0.1 * rng.standard_normal(4 * D), W_2=W_2, b_2=b_2,
                g2=1 + 0.1 * rng.standard_normal(D), be2=0.1 * rng.standard_normal(D))


def test_zero_output_projection_and_ffn_reduce_to_layer_norms():
    rng = np.random.default_rng(4)
    D = 16
    X, O = rng.standard_normal((5, D)), rng.standard_normal((5, D))
    w = _weights(D, rng, zero_o=True, zero_2=True)
    r = enc.output_and_ffn(X, O, **w)
    np.testing.assert_allclose(r["S1"], X, atol=0)
    h1 = enc.layer_norm(X, w["g1"], w["be1"])
    np.testing.assert_allclose(r["Y"], enc.layer_norm(h1, w["g2"], w["be2"]), atol=1e-13)


def test_output_and_ffn_against_torch_modules():
    rng = np.random.default_rng(5)
    D = 32
    X, O = rng.standard_normal((7, D)), rng.standard_normal((7, D))
    w = _weights(D, rng)
    r = enc.output_and_ffn(X, O, **w)
    t = {k: torch.from_numpy(np.asarray(v)) for k, v in w.items()}
    x, o = torch.from_numpy(X), torch.from_numpy(O)
    F = torch.nn.functional
    h1 = F.layer_norm(x + F.linear(o, t["W_o"], t["b_o"]), (D,), t["g1"], t["be1"], eps=enc.LN_EPS)
    ff = F.linear(F.gelu(F.linear(h1, t["W_1"], t["b_1"])), t["W_2"], t["b_2"])
    y = F.layer_norm(h1 + ff, (D,), t["g2"], t["be2"], eps=enc.LN_EPS)
    np.testing.assert_allclose(r["Y"], y.numpy(), rtol=0, atol=1e-12)
