"""Pins of the target-layer oracle (RMSNorm, linear, SwiGLU, one decoder
layer around the tree attention) against closed forms, brute force and
special cases that reduce the layer to a known expression."""

import math

import numpy as np

from oracle.layer import decoder_layer, linear, rmsnorm, silu, swiglu
from oracle.tree import tree_build


def test_rmsnorm_closed_forms():
    w = np.array([0.5, -1.0, 2.0, 3.0])
    # a constant row c: mean square c^2, so the output is sign(c) * w (eps = 0)
    for c in (2.0, -0.25):
        out = rmsnorm(np.full((1, 4), c), w, eps=0.0)
        np.testing.assert_allclose(out[0], math.copysign(1.0, c) * w, rtol=1e-14)
    rng = np.random.default_rng(1)
    x = rng.normal(size=(5, 64))
    ones = np.ones(64)
    y = rmsnorm(x, ones, eps=0.0)
    np.testing.assert_allclose((y * y).mean(axis=1), np.ones(5), rtol=1e-12)   # unit mean square
    np.testing.assert_allclose(rmsnorm(3.5 * x, ones, eps=0.0), y, rtol=1e-12)  # scale invariant
    # eps shrinks a tiny row toward zero: x = 1e-4, eps = 1e-5 -> 1e-4 / sqrt(1e-8 + 1e-5)
    out = rmsnorm(np.full((1, 8), 1e-4), np.ones(8), eps=1e-5)
    np.testing.assert_allclose(out, np.full((1, 8), 1e-4 / math.sqrt(1e-8 + 1e-5)), rtol=1e-12)


def test_linear_and_silu():
    rng = np.random.default_rng(2)
    x = rng.normal(size=(3, 5))
    W = rng.normal(size=(4, 5))
    ref = np.array([[sum(x[r, k] * W[n, k] for k in range(5)) for n in range(4)] for r in range(3)])
    np.testing.assert_allclose(linear(x, W), ref, rtol=1e-12)
    z = np.linspace(-8, 8, 33)
    assert silu(np.array([0.0]))[0] == 0.0
    np.testing.assert_allclose(silu(z) - silu(-z), z, rtol=1e-12, atol=1e-15)   # z(s(z) + s(-z)) = z
    assert abs(silu(np.array([40.0]))[0] - 40.0) < 1e-12
    np.testing.assert_allclose(swiglu(x, W, np.zeros_like(W)), np.zeros((3, 4)))


def _layer_weights(rng, H, Hq, Hkv, d, F, scale=0.1):
    return {"attn_norm": rng.normal(size=H), "Wq": rng.normal(size=(Hq * d, H)) * scale,
            "Wk": rng.normal(size=(Hkv * d, H)) * scale, "Wv": rng.normal(size=(Hkv * d, H)) * scale,
            "Wo": rng.normal(size=(H, Hq * d)) * scale, "mlp_norm": rng.normal(size=H),
            "Wg": rng.normal(size=(F, H)) * scale, "Wu": rng.normal(size=(F, H)) * scale,
            "Wd": rng.normal(size=(H, F)) * scale}


def test_layer_without_outputs_is_identity():
    rng = np.random.default_rng(3)
    B, N, Hq, Hkv, d, F, S = 1, 4, 2, 1, 8, 24, 16
    H = Hq * d
    w = _layer_weights(rng, H, Hq, Hkv, d, F)
    w["Wo"][:] = 0.0
    w["Wd"][:] = 0.0
    parents = np.array([[-1, 0, 0, 1]])
    P = np.array([5])
    depth, pos, anc, st = tree_build(parents, P)
    h = rng.normal(size=(B * N, H))
    cK = rng.normal(size=(B, Hkv, S, d))
    cV = rng.normal(size=(B, Hkv, S, d))
    h2, _, _ = decoder_layer(h, w, cK, cV, P, pos, anc, 1e4, B, N, Hq, Hkv, d)
    np.testing.assert_array_equal(h2, h)


def test_single_token_layer_closed_form():
    # One node, no prefix (MHA): the attention of every head is its own v,
    # so the layer is h + x Wv^T Wo^T + SwiGLU(x2) Wd^T with x = RMSNorm(h).
    rng = np.random.default_rng(4)
    B, N, Hq, Hkv, d, F, S = 1, 1, 2, 2, 8, 16, 4
    H = Hq * d
    w = _layer_weights(rng, H, Hq, Hkv, d, F)
    parents = np.array([[-1]])
    P = np.array([0])
    depth, pos, anc, st = tree_build(parents, P)
    h = rng.normal(size=(1, H))
    cK = np.zeros((B, Hkv, S, d))
    cV = np.zeros((B, Hkv, S, d))
    got, _, _ = decoder_layer(h, w, cK, cV, P, pos, anc, 1e4, B, N, Hq, Hkv, d)

    def norm(v, g):
        return v / np.sqrt((v * v).mean() + 1e-5) * g

    x = norm(h[0], w["attn_norm"])
    h1 = h[0] + w["Wo"] @ (w["Wv"] @ x)
    x2 = norm(h1, w["mlp_norm"])
    gate = w["Wg"] @ x2
    ref = h1 + w["Wd"] @ (gate / (1.0 + np.exp(-gate)) * (w["Wu"] @ x2))
    np.testing.assert_allclose(got[0], ref, rtol=1e-10)
