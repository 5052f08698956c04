"""Seeded synthetic inputs shaped like SparseCoder's workloads.

This module only draws random numbers: it holds none of the method's
arithmetic, imports neither the CUDA package nor the oracle, and serves both.

Shapes follow the paper's setting: a RoBERTa-base encoder (12 layers, 12 heads
of width 64; Sec. "Experimental Design" and the RQ1 setup, which fixes 12
layers) over function-level C/C++ code whose token lengths are long-tailed,
with 95% of functions within 1024 tokens (Sec. "Dataset").  The dataset itself
is not available, so per-layer Q/K/V rows are drawn N(0,1) per head and
position, a seeded subset of positions gets its key rows scaled up (salient
tokens that attract attention), and the inputs are rounded to bf16 with
round-to-nearest-even.  The bf16 bit patterns are what both the CUDA path and
the oracle read.

Random streams are counter-based through ``numpy.random.SeedSequence`` with a
tuple key per (purpose, layer, sequence[, position, redraw]), so any part of a
workload can be regenerated alone and redraws do not disturb other rows.
"""
from __future__ import annotations

from dataclasses import dataclass, replace
from typing import Dict, Optional, Tuple

import json
import os

import numpy as np

HEAD_DIM = 64

_TAG_QKV = 11
_TAG_SALIENT = 12
_TAG_GLOBAL = 13
_TAG_LENGTH = 14
_TAG_REDRAW = 15
_TAG_WEIGHTS = 16
_TAG_HIDDEN = 17


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round finite float32 values to bf16 (round to nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    return bf16_bits_to_f32(b).astype(np.float64)


def _rng(*key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(list(key))))


@dataclass(frozen=True)
class Workload:
    """One synthetic workload.

    alpha schedule: linear from ``alpha_first`` (layer 1) to ``alpha_last``
    (layer n_layers), endpoints included; the paper scales its per-layer
    thresholds linearly with depth (RQ4 discussion).  ``keep_rule`` says what
    the per-layer value is: 0 = alpha_l with theta_l = alpha_l / n_l, 1 = an
    absolute threshold theta_l, 2 = the ratio of tokens a layer keeps.
    """
    name: str
    n_layers: int
    B: int
    L: int
    H: int = 12
    d: int = HEAD_DIM
    w: int = 256
    n_extra_global: int = 0
    salient_frac: float = 0.10
    salient_scale: float = 3.0
    alpha_first: float = 0.3
    alpha_last: float = 0.9
    ragged: Optional[Tuple[int, int]] = None
    seed: int = 1
    keep_rule: int = 0

    def alphas(self) -> np.ndarray:
        if self.n_layers == 1:
            return np.array([self.alpha_first], dtype=np.float64)
        t = np.arange(self.n_layers, dtype=np.float64) / (self.n_layers - 1)
        return self.alpha_first + (self.alpha_last - self.alpha_first) * t

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)

    def describe(self) -> str:
        s = (f"{self.name}: {self.n_layers} layers, B={self.B}, L={self.L}, H={self.H}, "
             f"d={self.d}, window +-{self.w}, globals 1+{self.n_extra_global}, "
             f"salient {self.salient_frac:.0%} x{self.salient_scale:g}, "
             + ("alpha", "theta", "kept ratio")[self.keep_rule]
             + f" {self.alpha_first:g}->{self.alpha_last:g}")
        if self.ragged:
            s += f", true lengths U[{self.ragged[0]},{self.ragged[1]}]"
        return s + f", seed {self.seed}"


# The five workloads, as stated for this hot path.
CFG1 = Workload("cfg1_L512_1layer", n_layers=1, B=1, L=512, w=64,
                alpha_first=0.7, alpha_last=0.7)
CFG2 = Workload("cfg2_L1024_B8", n_layers=12, B=8, L=1024)
CFG3 = Workload("cfg3_L2048_B4_ragged", n_layers=12, B=4, L=2048, ragged=(1024, 2048))
CFG4 = Workload("cfg4_L4096_B2_9global", n_layers=12, B=2, L=4096, n_extra_global=8,
                salient_frac=0.05, salient_scale=4.0, alpha_first=0.4, alpha_last=1.0)


def cfg5(L: int, control: bool = False) -> Workload:
    """Throughput sweep point: B = 16384 / L; ``control`` sets theta = 0 (no pruning)."""
    assert L in (512, 1024, 2048, 4096)
    wl = Workload(f"cfg5_L{L}_B{16384 // L}" + ("_theta0" if control else ""),
                  n_layers=12, B=16384 // L, L=L)
    if control:
        wl = wl.with_(alpha_first=0.0, alpha_last=0.0)
    return wl


CONFIGS = {"cfg1": CFG1, "cfg2": CFG2, "cfg3": CFG3, "cfg4": CFG4}


def window_sweep(w: int) -> Workload:
    """The window-size ablation (Table "window_size", RQ3): sparse attention
    alone (nothing pruned) over inputs of maximum length 1024, one-sided window
    ``w`` in {16, 32, 64, 128, 256, 512}; 12 layers, B = 8."""
    assert w in (16, 32, 64, 128, 256, 512)
    return Workload(f"window_w{w}_L1024_B8", n_layers=12, B=8, L=1024, w=w,
                    alpha_first=0.0, alpha_last=0.0)


# The paper's own threshold schedule (RQ4): absolute thresholds scaled
# linearly with depth up to 0.01 at the 12th layer (0.01 l / 12), over the
# config-2 shape.
ABS_THETA = Workload("abs_theta_L1024_B8", n_layers=12, B=8, L=1024,
                     alpha_first=0.01 / 12, alpha_last=0.01, keep_rule=1)

# The top-k family of Sec. "Pruning": each layer keeps a fixed ratio of its
# current tokens (0.95 at layer 1 down to 0.8 at layer 12), config-2 shape.
TOP_RATIO = Workload("top_ratio_L1024_B8", n_layers=12, B=8, L=1024,
                     alpha_first=0.95, alpha_last=0.8, keep_rule=2)


def global_positions(wl: Workload) -> np.ndarray:
    """Token 0 plus ``n_extra_global`` seeded distinct positions, sorted."""
    extra = np.zeros(0, dtype=np.int64)
    if wl.n_extra_global > 0:
        extra = _rng(wl.seed, _TAG_GLOBAL).choice(np.arange(1, wl.L), wl.n_extra_global,
                                                  replace=False)
    return np.sort(np.concatenate([[0], extra])).astype(np.int32)


def pad_mask(wl: Workload) -> Optional[np.ndarray]:
    """[B, L] uint8 (1 = real token) for ragged workloads, else None."""
    if wl.ragged is None:
        return None
    lo, hi = wl.ragged
    lens = _rng(wl.seed, _TAG_LENGTH).integers(lo, hi + 1, size=wl.B)
    return (np.arange(wl.L)[None, :] < lens[:, None]).astype(np.uint8)


def salient_mask(wl: Workload) -> np.ndarray:
    """[B, L] bool: the seeded salient positions of each sequence (fixed across layers)."""
    m = np.zeros((wl.B, wl.L), dtype=bool)
    cnt = int(round(wl.salient_frac * wl.L))
    for b in range(wl.B):
        if cnt > 0:
            m[b, _rng(wl.seed, _TAG_SALIENT, b).choice(wl.L, cnt, replace=False)] = True
    return m


def make_inputs(wl: Workload, redraws: Optional[Dict[Tuple[int, int, int], int]] = None):
    """Draw the workload.

    Returns a dict with ``Q``, ``K``, ``V`` (uint16 bf16 bits, [n_layers, B, L, H, d],
    original-position order), ``pad_mask`` ([B, L] uint8 or None), ``global_pos``
    (int32), ``alpha`` (float64 [n_layers]) and ``salient`` ([B, L] bool).

    ``redraws`` maps (layer, sequence, original position) to a redraw count; the
    Q and K rows of that token at that layer are replaced by a fresh draw keyed
    by the count (the near-threshold resampling of the parity fixtures).
    """
    nl, B, L, H, d = wl.n_layers, wl.B, wl.L, wl.H, wl.d
    sal = salient_mask(wl)
    Q = np.empty((nl, B, L, H, d), np.uint16)
    K = np.empty_like(Q)
    V = np.empty_like(Q)
    for l in range(nl):
        for b in range(B):
            g = _rng(wl.seed, _TAG_QKV, l, b)
            q = g.standard_normal((L, H, d), dtype=np.float32)
            k = g.standard_normal((L, H, d), dtype=np.float32)
            v = g.standard_normal((L, H, d), dtype=np.float32)
            k[sal[b]] *= np.float32(wl.salient_scale)
            Q[l, b] = f32_to_bf16_bits(q)
            K[l, b] = f32_to_bf16_bits(k)
            V[l, b] = f32_to_bf16_bits(v)
    inp = {"Q": Q, "K": K, "V": V, "pad_mask": pad_mask(wl),
           "global_pos": global_positions(wl), "alpha": wl.alphas(), "salient": sal}
    for (l, b, p), cnt in (redraws or {}).items():
        redraw_row(wl, inp, l, b, p, cnt)
    return inp


def redraw_row(wl: Workload, inp, l: int, b: int, p: int, cnt: int) -> None:
    """Replace, in place, the Q and K rows of token ``p`` of sequence ``b`` at
    layer ``l`` in ``inp`` (from ``make_inputs``) by draw number ``cnt`` of its
    redraw stream (V is kept; a salient token's key row keeps its scale)."""
    g = _rng(wl.seed, _TAG_REDRAW, l, b, p, cnt)
    q = g.standard_normal((wl.H, wl.d), dtype=np.float32)
    k = g.standard_normal((wl.H, wl.d), dtype=np.float32)
    if inp["salient"][b, p]:
        k *= np.float32(wl.salient_scale)
    inp["Q"][l, b, p] = f32_to_bf16_bits(q)
    inp["K"][l, b, p] = f32_to_bf16_bits(k)


def random_layer(n: int, H: int, d: int, seed: int, scale_k: float = 1.0):
    """Q, K, V bf16 bits [n, H, d] for single-layer tests (current order)."""
    g = _rng(seed, _TAG_QKV, 10_000, n)
    q = g.standard_normal((n, H, d), dtype=np.float32)
    k = g.standard_normal((n, H, d), dtype=np.float32) * np.float32(scale_k)
    v = g.standard_normal((n, H, d), dtype=np.float32)
    return f32_to_bf16_bits(q), f32_to_bf16_bits(k), f32_to_bf16_bits(v)


# ---------------------------------------------------------------------------
# the encoder layer around the path: random-init weights and input hidden states
# ---------------------------------------------------------------------------
ENCODER_CFG2 = Workload("encoder_cfg2_L1024_B8", n_layers=12, B=8, L=1024)


def encoder_weights(D: int, layer: int, seed: int = 1):
    """Random-init weights of one RoBERTa-size layer (no checkpoint is available):
    matrices N(0, 1/fan_in) as bf16 bits [out][in], biases N(0, 0.02^2), layer-norm
    gains 1 + N(0, 0.1^2) and shifts N(0, 0.1^2) as float32."""
    g = _rng(seed, _TAG_WEIGHTS, layer)
    def mat(o, i):
        return f32_to_bf16_bits(g.standard_normal((o, i), dtype=np.float32) / np.float32(np.sqrt(i)))
    def vec(n, scale, shift=0.0):
        return (np.float32(shift) + np.float32(scale) * g.standard_normal(n, dtype=np.float32))
    return {"W_qkv": mat(3 * D, D), "b_qkv": vec(3 * D, 0.02), "W_o": mat(D, D), "b_o": vec(D, 0.02),
            "ln1_gamma": vec(D, 0.1, 1.0), "ln1_beta": vec(D, 0.1), "W_1": mat(4 * D, D),
            "b_1": vec(4 * D, 0.02), "W_2": mat(D, 4 * D), "b_2": vec(D, 0.02),
            "ln2_gamma": vec(D, 0.1, 1.0), "ln2_beta": vec(D, 0.1)}


def encoder_input(wl: Workload):
    """Layer-0 hidden states: bf16 bits [B, L, D], N(0, 1)."""
    g = _rng(wl.seed, _TAG_HIDDEN)
    return f32_to_bf16_bits(g.standard_normal((wl.B, wl.L, wl.H * wl.d), dtype=np.float32))


# ---------------------------------------------------------------------------
# stored redraws: the near-threshold resampling of each named workload, found
# by the oracle (tests/golden/make_redraws.py writes the file; nothing here
# computes them)
# ---------------------------------------------------------------------------
_REDRAWS_FILE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                             "tests", "golden", "redraws.json")


def stored_redraws(wl: Workload) -> Dict[Tuple[int, int, int], int]:
    """{(layer, sequence, original position): redraw count} stored for ``wl``
    (matched by name and seed), or {} when the file has no entry for it."""
    try:
        with open(_REDRAWS_FILE) as f:
            table = json.load(f)
    except FileNotFoundError:
        return {}
    entry = table.get(wl.name)
    if entry is None or entry.get("seed") != wl.seed:
        return {}
    return {tuple(int(x) for x in k.split(",")): int(c) for k, c in entry["redraws"].items()}
