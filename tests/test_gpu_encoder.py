"""GPU parity of the encoder layer around the path (sc_linear_forward,
sc_layer_norm_forward, sc_encoder_layer_forward) against the float64 oracle.

The GEMM and the layer norm are checked on random inputs.  The layer is
checked stage by stage on the GPU's own inputs to each stage: the attention
outputs against the oracle's attention on the oracle's projections (bf16 as
stored), the kept list against the kernels' own scores (exactly) and against
the oracle outside a margin, and the output projection + feed-forward block on
the GPU's own O and kept list.  A second layer takes the first one's outputs.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads as wk
from oracle import encoder as enc
from parity_utils import (O_ATOL, SCORE_ATOL, bits_to_torch, check_o, check_scores,
                          torch_bf16_to_f64)

# The stages around the attention (GEMM outputs, the layer output Y) are not
# attention outputs: their values reach several units, where the bf16 storage
# rounding alone is half an ulp = 2^-9 |y|; their bar adds that rounding and one
# more of the same size for a bf16 operand rounded inside the stage.
STAGE_RTOL = 2.0 ** -8

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2310_07109_gb300 as sc
    sc.load()
    return sc


def _bf16(x):
    """float64 values rounded to bf16 (through float32), as float64."""
    return wk.bf16_bits_to_f64(wk.f32_to_bf16_bits(np.asarray(x, np.float32)))


def _t_bf16(x64):
    return bits_to_torch(wk.f32_to_bf16_bits(np.asarray(x64, np.float32)), "cuda")


LINEAR_CASES = [
    # B, L, rows, N, K, gather, gelu, res, res_gathered, out_f32
    (1, 128, None, 128, 64, False, False, False, False, True),
    (2, 300, [300, 77], 256, 768, True, False, True, True, True),
    (2, 256, [200, 256], 384, 192, False, True, False, False, False),
    (3, 130, [130, 1, 129], 768, 3072, False, False, True, False, True),
    (1, 512, [431], 3072, 768, True, True, False, False, False),
    # 192-column tiles (the width that fills whole rounds of tiles best here)
    (8, 1024, [1024, 1000, 517, 3, 1024, 900, 128, 129], 768, 768, False, False, True, False,
     False),
    (4, 1664, [1664, 1600, 1, 830], 384, 128, False, True, False, False, True),
]


@pytest.mark.parametrize("B,L,rows,N,K,gather,gelu,res,res_g,out_f32", LINEAR_CASES)
def test_linear_matches_oracle(sc, B, L, rows, N, K, gather, gelu, res, res_g, out_f32):
    rng = np.random.default_rng(B * 1000 + L + N + K)
    A = _bf16(rng.standard_normal((B * L, K)))
    W = _bf16(rng.standard_normal((N, K)) / math.sqrt(K))
    bias = rng.standard_normal(N).astype(np.float32) * 0.1
    R = _bf16(rng.standard_normal((B * L, N))) if res else None
    nrows = np.array(rows if rows is not None else [L] * B, np.int32)
    gidx = np.stack([rng.permutation(L) for _ in range(B)]).astype(np.int32) if gather else None
    out = torch.full((B * L, N), float("nan"), dtype=torch.float32 if out_f32 else torch.bfloat16,
                     device="cuda")
    sc.linear_forward(_t_bf16(A), _t_bf16(W), B=B, L=L,
                      rows=torch.from_numpy(nrows).cuda() if rows is not None else None,
                      gidx=torch.from_numpy(gidx).cuda() if gather else None,
                      bias=torch.from_numpy(bias).cuda(), gelu=gelu,
                      res=_t_bf16(R) if res else None, res_gathered=res_g, out=out,
                      out_f32=out_f32)
    torch.cuda.synchronize()
    got = out.float().cpu().numpy().astype(np.float64) if out_f32 else torch_bf16_to_f64(out)
    for b in range(B):
        n = int(nrows[b])
        src = b * L + (gidx[b, :n] if gather else np.arange(n))
        y = enc.linear(A[src], W, bias)
        if gelu:
            y = enc.gelu(y)
        if res:
            y = y + R[src if res_g else b * L + np.arange(n)]
        g = got[b * L:b * L + n]
        tol = (1e-4 * np.abs(y).max(), 0) if out_f32 else (O_ATOL / 4, STAGE_RTOL)
        np.testing.assert_allclose(g, y, atol=tol[0], rtol=tol[1], err_msg=f"sequence {b}")
        assert np.isnan(got[b * L + n:(b + 1) * L]).all(), "rows past the sequence were written"


def test_gelu_epilogue_accuracy(sc):
    """The GEMM's GELU (erf by Abramowitz & Stegun 7.1.26, |error| <= 1.5e-7)
    against the fp64 definition: a 0/1 selector weight makes each fp32 output
    GELU of one bf16 input exactly, so only the GELU's own error remains."""
    K, N, M = 64, 128, 512
    x = _bf16(np.linspace(-9.0, 9.0, M * K).reshape(M, K))
    x[0, :8] = [0.0, -0.0, 1e-3, -1e-3, 2.0 ** -20, -(2.0 ** -20), 40.0, -40.0]
    W = np.zeros((N, K))
    W[np.arange(N), np.arange(N) % K] = 1.0
    out = torch.empty((M, N), dtype=torch.float32, device="cuda")
    sc.linear_forward(_t_bf16(x), _t_bf16(W), B=1, L=M, bias=None, gelu=True, out=out,
                      out_f32=True)
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    want = enc.gelu(x[:, np.arange(N) % K])
    err = np.abs(got - want)
    assert (err <= 2e-6 * np.maximum(1.0, np.abs(want))).all(), err.max()


@pytest.mark.parametrize("D", [768, 128, 96, 1024], ids=lambda d: f"D{d}")
def test_layer_norm_matches_oracle(sc, D):
    """D a multiple of 128 takes the four-features-per-access path, D = 96 the
    one-feature path."""
    rng = np.random.default_rng(7 + D)
    B, L = 2, 200
    x = (rng.standard_normal((B * L, D)) * 2.5 + 0.7).astype(np.float32)
    g = (1 + 0.1 * rng.standard_normal(D)).astype(np.float32)
    be = (0.1 * rng.standard_normal(D)).astype(np.float32)
    rows = np.array([200, 63], np.int32)
    out = torch.full((B * L, D), float("nan"), dtype=torch.bfloat16, device="cuda")
    sc.layer_norm_forward(torch.from_numpy(x).cuda(), torch.from_numpy(g).cuda(),
                          torch.from_numpy(be).cuda(), B=B, L=L,
                          rows=torch.from_numpy(rows).cuda(), out=out)
    torch.cuda.synchronize()
    got = torch_bf16_to_f64(out)
    for b in range(B):
        n = int(rows[b])
        y = enc.layer_norm(x[b * L:b * L + n], g, be)
        np.testing.assert_allclose(got[b * L:b * L + n], y, atol=1e-2, rtol=2.0 ** -8)
        assert np.isnan(got[b * L + n:(b + 1) * L]).all()


def _weights(D, seed):
    rng = np.random.default_rng(seed)
    w = {"W_qkv": _bf16(rng.standard_normal((3 * D, D)) / math.sqrt(D)),
         "b_qkv": (0.02 * rng.standard_normal(3 * D)).astype(np.float32),
         "W_o": _bf16(rng.standard_normal((D, D)) / math.sqrt(D)),
         "b_o": (0.02 * rng.standard_normal(D)).astype(np.float32),
         "ln1_gamma": (1 + 0.1 * rng.standard_normal(D)).astype(np.float32),
         "ln1_beta": (0.1 * rng.standard_normal(D)).astype(np.float32),
         "W_1": _bf16(rng.standard_normal((4 * D, D)) / math.sqrt(D)),
         "b_1": (0.02 * rng.standard_normal(4 * D)).astype(np.float32),
         "W_2": _bf16(rng.standard_normal((D, 4 * D)) / math.sqrt(4 * D)),
         "b_2": (0.02 * rng.standard_normal(D)).astype(np.float32),
         "ln2_gamma": (1 + 0.1 * rng.standard_normal(D)).astype(np.float32),
         "ln2_beta": (0.1 * rng.standard_normal(D)).astype(np.float32)}
    dev = {k: (_t_bf16(v) if k.startswith("W") else torch.from_numpy(v).cuda()) for k, v in w.items()}
    return w, dev


def _check_layer(sc, X, lens, pos, w64, wdev, L, H, wwin, gpos, alpha):
    """Run one encoder layer and check it stage by stage; returns the GPU outputs."""
    B = X.shape[0]
    D = H * 64
    ws = sc.new_encoder_workspace(B, L, H)
    out = sc.encoder_layer_forward(_t_bf16(X.reshape(B, L, D)),
                                   torch.from_numpy(lens).cuda(), torch.from_numpy(pos).cuda(),
                                   wwin, gpos, wdev, alpha, workspace=ws)
    assert sc.workspace_status(ws) == 0
    torch.cuda.synchronize()
    O = torch_bf16_to_f64(out["O"]).reshape(B, L, D)
    Y = torch_bf16_to_f64(out["Y"]).reshape(B, L, D)
    s = out["scores"].cpu().numpy()
    po = out["pos_out"].cpu().numpy()
    lo = out["len_out"].cpu().numpy()
    gset = set(int(g) for g in gpos)
    for b in range(B):
        n = int(lens[b])
        theta = alpha / n
        # attention on the oracle's projections (rounded to bf16 as stored)
        q, k, v = (_bf16(t) for t in enc.qkv(X[b, :n], w64["W_qkv"], w64["b_qkv"]))
        isg = np.array([int(p) in gset for p in pos[b, :n]])
        Oe, se, keep_e = oracle.layer(q.reshape(n, H, 64), k.reshape(n, H, 64),
                                      v.reshape(n, H, 64), isg, wwin, theta)
        check_o(O[b, :n], Oe.reshape(n, D), f"sequence {b}")
        check_scores(s[b, :n], se, f"sequence {b}")
        # the kept list: the kernels' own decision on their own scores, and the
        # oracle's wherever its score is clear of the threshold
        keep_g = (np.arange(n) == 0) | (s[b, :n] >= np.float32(alpha) / np.float32(n))
        kept_pos = pos[b, :n][keep_g]
        assert int(lo[b]) == len(kept_pos)
        assert list(po[b, :len(kept_pos)]) == list(kept_pos)
        clear = np.abs(se - theta) > 1e-5
        assert (keep_g[clear] == keep_e[clear]).all()
        # output projection + feed-forward on the GPU's own O and kept tokens
        kc = np.nonzero(keep_g)[0]
        r = enc.output_and_ffn(X[b, kc], O[b, kc], w64["W_o"], w64["b_o"], w64["ln1_gamma"],
                               w64["ln1_beta"], w64["W_1"], w64["b_1"], w64["W_2"], w64["b_2"],
                               w64["ln2_gamma"], w64["ln2_beta"], round_h1=_bf16, round_f=_bf16)
        np.testing.assert_allclose(Y[b, :len(kc)], r["Y"], rtol=STAGE_RTOL, atol=O_ATOL,
                                   err_msg=f"sequence {b}")
    return Y, po, lo


@pytest.mark.parametrize("L,lens,wwin,gpos,alpha", [
    (300, [300, 211], 64, [0, 5], 0.6),
    (700, [700, 450], 128, [0], 0.8),
])
def test_encoder_layer_matches_oracle(sc, L, lens, wwin, gpos, alpha):
    H = 12
    D = H * 64
    B = len(lens)
    rng = np.random.default_rng(L + wwin)
    X = _bf16(rng.standard_normal((B, L, D)))
    lens = np.array(lens, np.int32)
    pos = np.tile(np.arange(L, dtype=np.int32), (B, 1))
    w64, wdev = _weights(D, seed=L)
    _check_layer(sc, X, lens, pos, w64, wdev, L, H, wwin, gpos, alpha)


def test_encoder_two_layers_chain(sc):
    """Layer 2 reads layer 1's compacted outputs (Y, len_out, pos_out)."""
    H, L, B = 12, 500, 2
    D = H * 64
    rng = np.random.default_rng(9)
    X = _bf16(rng.standard_normal((B, L, D)))
    lens = np.array([500, 333], np.int32)
    pos = np.tile(np.arange(L, dtype=np.int32), (B, 1))
    w1, d1 = _weights(D, seed=1)
    w2, d2 = _weights(D, seed=2)
    Y, po, lo = _check_layer(sc, X, lens, pos, w1, d1, L, H, 64, [0, 7], 0.7)
    Y2 = np.zeros_like(Y)
    for b in range(B):
        Y2[b, :lo[b]] = Y[b, :lo[b]]
    _check_layer(sc, Y2, lo.astype(np.int32), po.astype(np.int32), w2, d2, L, H, 64, [0, 7], 0.9)
