"""Plain fp64 CPU oracle of the encoder layer around the hot path.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``): the tests and the
benchmark's CPU legs may use it; the CUDA library never does.

SparseCoder modifies the self-attention of a RoBERTa-style encoder (Sec.
"Transformer-based models", Fig. "sparsecoder": sparse attention and token
pruning inside each of the 12 encoder layers, the rest of the layer as in the
Transformer).  One layer on the n current tokens of a sequence, hidden size
D = 64 H, feed-forward width 4 D, post-layer normalisation:

    Q, K, V = X W_q^T + b_q, X W_k^T + b_k, X W_v^T + b_v      (per head: 64 columns)
    O, s, keep = sparse attention with token pruning          (oracle.layer)
    for the kept tokens only (pruning happens after the attention):
    H1 = LN(X + O W_o^T + b_o)
    Y  = LN(H1 + GELU(H1 W_1^T + b_1) W_2^T + b_2)

LN(x) = (x - mean) / sqrt(var + eps) * gamma + beta over the D features
(population variance, eps = 1e-5); GELU(x) = x/2 (1 + erf(x / sqrt 2)).

Each step is a plain definition on float64 arrays (numpy's matmul serves as the
matrix product); the caller decides which stored values are rounded to bf16,
as the GPU stores them, so that every stage can be checked on the GPU's own
inputs to that stage.
"""
from __future__ import annotations

import math

import numpy as np

LN_EPS = 1e-5


def linear(x, W, b=None):
    """x [m, k] @ W[n, k]^T + b[n], in float64."""
    y = np.asarray(x, np.float64) @ np.asarray(W, np.float64).T
    if b is not None:
        y = y + np.asarray(b, np.float64)[None, :]
    return y


def gelu(x):
    """x/2 (1 + erf(x / sqrt(2))), elementwise."""
    x = np.asarray(x, np.float64)
    erf = np.vectorize(math.erf, otypes=[np.float64])
    return 0.5 * x * (1.0 + erf(x / math.sqrt(2.0)))


def layer_norm(x, gamma, beta, eps=LN_EPS):
    """Normalise each row over its features: population mean and variance."""
    x = np.asarray(x, np.float64)
    mean = x.mean(axis=1, keepdims=True)
    var = ((x - mean) ** 2).mean(axis=1, keepdims=True)
    return (x - mean) / np.sqrt(var + eps) * np.asarray(gamma, np.float64)[None, :] \
        + np.asarray(beta, np.float64)[None, :]


def qkv(X, W_qkv, b_qkv):
    """The three projections: X [n, D], W_qkv [3D, D] (rows: Q's D outputs, then
    K's, then V's), b_qkv [3D].  Returns three [n, D] arrays."""
    D = np.asarray(X).shape[1]
    y = linear(X, W_qkv, b_qkv)
    return y[:, :D], y[:, D:2 * D], y[:, 2 * D:]


def output_and_ffn(X_kept, O_kept, W_o, b_o, g1, be1, W_1, b_1, W_2, b_2, g2, be2,
                   round_h1=None, round_f=None):
    """The rest of the layer on the kept tokens: X_kept, O_kept [n', D].
    ``round_h1`` / ``round_f`` (callables or None) apply the storage rounding of
    the layer-norm output H1 and of the GELU output before they are used.
    Returns dict(S1, H1, F, S2, Y) (S1, S2 the sums before the layer norms)."""
    S1 = np.asarray(X_kept, np.float64) + linear(O_kept, W_o, b_o)
    H1 = layer_norm(S1, g1, be1)
    if round_h1 is not None:
        H1 = round_h1(H1)
    F = gelu(linear(H1, W_1, b_1))
    if round_f is not None:
        F = round_f(F)
    S2 = H1 + linear(F, W_2, b_2)
    Y = layer_norm(S2, g2, be2)
    return {"S1": S1, "H1": H1, "F": F, "S2": S2, "Y": Y}
