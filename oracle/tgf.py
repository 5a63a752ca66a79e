"""Oracle: the Token-Guided Fusion module of GRIFFIN's draft model.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Section 4.2 (Token-Alignable Draft Model), Eqs. 6-8: before the draft model's
autoregressive layer, TGF fuses each position's input feature F (the target's
or the drafter's own feature) with the embedding x of its token:

1. embedding fusion (Eq. 6):         h = C(F, x) W_m + b_m
2. normalisation and expansion (7):  z = C(N(h), N(x)) W_u + b_u
3. refinement (Eq. 8):               o = silu(z) W_d + b_d + h

with C the concatenation, N layer normalisation, W_m [2d -> d], W_u
[2d -> e] (the expansion e is 4d in the text; the appendix sets it to the
target's FFN width, 11008 for a LLaMA-2-7B drafter) and W_d [e -> d].

Readings: weights are stored ``W[out][in]`` (so the paper's ``v W`` is
``v @ W.T`` here); each of the two layer norms has its own gain and bias
(``N(v) = (v - mean(v)) / sqrt(var(v) + eps) * g + b``, population variance,
eps = 1e-5); silu(z) = z / (1 + exp(-z)).  Float64, numpy primitives.
"""

import numpy as np

from .layer import linear, silu


def layernorm(x, g, b, eps=1e-5):
    """``(x - mean) / sqrt(var + eps) * g + b`` per row (population variance)."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * np.asarray(g, dtype=np.float64) + np.asarray(b, dtype=np.float64)


def tgf_forward(F, x, w, eps=1e-5):
    """Eqs. 6-8 over rows of features F [R][d] and token embeddings x [R][d].
    ``w`` holds Wm [d][2d], bm [d], g_h, b_h, g_x, b_x [d], Wu [e][2d], bu [e],
    Wd [d][e], bd [d].  Returns (o, h)."""
    F = np.asarray(F, dtype=np.float64)
    x = np.asarray(x, dtype=np.float64)
    h = linear(np.concatenate([F, x], axis=1), w["Wm"]) + w["bm"]
    zin = np.concatenate([layernorm(h, w["g_h"], w["b_h"], eps), layernorm(x, w["g_x"], w["b_x"], eps)], axis=1)
    z = linear(zin, w["Wu"]) + w["bu"]
    o = linear(silu(z), w["Wd"]) + w["bd"] + h
    return o, h
