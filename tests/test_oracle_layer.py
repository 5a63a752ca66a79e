"""Pins of the target-layer oracle (RMSNorm, linear, SwiGLU, one decoder
layer around the tree attention) against closed forms, brute force,
special cases that reduce the layer to a known expression, and an ordinary
causal LLaMA layer written with torch's library attention."""

import math

import numpy as np
import torch
import torch.nn.functional as F

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


def _rope_complex_torch(x, base):
    """RoPE of x [S][heads][d] at positions 0 .. S-1 as the complex product
    (x[j] + i x[j + d/2]) exp(i pos base^(-2j/d))."""
    S, _, d = x.shape
    half = d // 2
    theta = torch.tensor([base ** (-2.0 * j / d) for j in range(half)], dtype=torch.float64)
    ang = torch.arange(S, dtype=torch.float64)[:, None] * theta[None, :]
    z = torch.complex(x[..., :half], x[..., half:]) * torch.polar(torch.ones_like(ang), ang)[:, None, :]
    return torch.cat([z.real, z.imag], dim=-1)


def _torch_llama_layer(hs, w, base, Hq, Hkv, d, eps=1e-5):
    """A LLaMA decoder layer over a whole sequence in torch float64, causal
    attention by scaled_dot_product_attention; returns the outputs and every
    position's rotated key and value."""
    t = {k: torch.from_numpy(np.asarray(v, dtype=np.float64)) for k, v in w.items()}
    h = torch.from_numpy(hs)
    S = h.shape[0]

    def norm(v, g):
        return v * torch.rsqrt(v.pow(2).mean(dim=-1, keepdim=True) + eps) * g

    x = norm(h, t["attn_norm"])
    q = _rope_complex_torch((x @ t["Wq"].T).view(S, Hq, d), base)
    k = _rope_complex_torch((x @ t["Wk"].T).view(S, Hkv, d), base)
    v = (x @ t["Wv"].T).view(S, Hkv, d)
    G = Hq // Hkv
    o = F.scaled_dot_product_attention(q.transpose(0, 1)[None], k.repeat_interleave(G, dim=1).transpose(0, 1)[None],
                                       v.repeat_interleave(G, dim=1).transpose(0, 1)[None], is_causal=True)
    h1 = h + o[0].transpose(0, 1).reshape(S, Hq * d) @ t["Wo"].T
    x2 = norm(h1, t["mlp_norm"])
    h2 = h1 + (F.silu(x2 @ t["Wg"].T) * (x2 @ t["Wu"].T)) @ t["Wd"].T
    return h2.numpy(), k.numpy(), v.numpy()


def test_chain_layer_equals_a_causal_llama_layer():
    # A two-node chain after a three-token prefix is the last two positions of
    # a five-token causal sequence: the tree layer, fed the prefix's rotated
    # keys and values as its cache, must give what an ordinary LLaMA layer
    # (torch, causal SDPA, RoPE as a complex product, GQA by repeated KV heads)
    # gives there.  Unlike the one-token case, the keys decide the weights.
    rng = np.random.default_rng(11)
    Hq, Hkv, d, Fw, base = 4, 2, 8, 48, 1e4
    H = Hq * d
    w = _layer_weights(rng, H, Hq, Hkv, d, Fw, scale=0.3)
    hs = rng.normal(size=(5, H))
    ref, rk, rv = _torch_llama_layer(hs, w, base, Hq, Hkv, d)
    P = np.array([3])
    parents = np.array([[-1, 0]])
    depth, pos, anc, st = tree_build(parents, P)
    S = 8
    cK = np.zeros((1, Hkv, S, d))
    cV = np.zeros((1, Hkv, S, d))
    cK[0, :, :3] = rk[:3].transpose(1, 0, 2)
    cV[0, :, :3] = rv[:3].transpose(1, 0, 2)
    got, tK, tV = decoder_layer(hs[3:], w, cK, cV, P, pos, anc, base, 1, 2, Hq, Hkv, d)
    np.testing.assert_allclose(got, ref[3:], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(tK[0], rk[3:].transpose(1, 0, 2), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(tV[0], rv[3:].transpose(1, 0, 2), rtol=1e-10, atol=1e-12)
