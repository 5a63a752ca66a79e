"""Pins of the Token-Guided Fusion oracle (GRIFFIN Eqs. 6-8): layer-norm
closed forms, and weight choices that reduce the module to a known map."""

import math

import numpy as np

from oracle.tgf import layernorm, tgf_forward


def test_layernorm_closed_forms():
    rng = np.random.default_rng(1)
    x = rng.normal(size=(6, 40)) * 3 + 5
    y = layernorm(x, np.ones(40), np.zeros(40), eps=0.0)
    np.testing.assert_allclose(y.mean(axis=1), np.zeros(6), atol=1e-12)
    np.testing.assert_allclose((y * y).mean(axis=1), np.ones(6), rtol=1e-12)
    # shift and scale invariance
    np.testing.assert_allclose(layernorm(2.5 * x - 7, np.ones(40), np.zeros(40), eps=0.0), y, rtol=1e-10, atol=1e-12)
    # a two-valued row [a, b]: (+-1) after normalisation (eps = 0), then gain and bias
    out = layernorm(np.array([[1.0, 3.0]]), np.array([2.0, 3.0]), np.array([0.5, -1.0]), eps=0.0)
    np.testing.assert_allclose(out, [[-2.0 + 0.5, 3.0 - 1.0]], rtol=1e-12)
    # a constant row normalises to the bias
    np.testing.assert_allclose(layernorm(np.full((1, 5), 4.0), np.ones(5), np.arange(5.0)), [np.arange(5.0)])


def _w(rng, d, e, scale=0.2):
    return {"Wm": rng.normal(size=(d, 2 * d)) * scale, "bm": rng.normal(size=d),
            "g_h": rng.normal(size=d), "b_h": rng.normal(size=d), "g_x": rng.normal(size=d),
            "b_x": rng.normal(size=d), "Wu": rng.normal(size=(e, 2 * d)) * scale, "bu": rng.normal(size=e),
            "Wd": rng.normal(size=(d, e)) * scale, "bd": rng.normal(size=d)}


def test_refinement_off_returns_the_fusion():
    # Wd = 0 and bd = 0: o = h = C(F, x) Wm^T + bm; with Wm = [I 0] and bm = 0, h = F.
    rng = np.random.default_rng(2)
    d, e = 8, 32
    w = _w(rng, d, e)
    w["Wd"][:] = 0
    w["bd"][:] = 0
    w["Wm"] = np.concatenate([np.eye(d), np.zeros((d, d))], axis=1)
    w["bm"][:] = 0
    F = rng.normal(size=(5, d))
    x = rng.normal(size=(5, d))
    o, h = tgf_forward(F, x, w)
    np.testing.assert_allclose(h, F, rtol=1e-14)
    np.testing.assert_allclose(o, F, rtol=1e-14)


def test_single_row_written_out():
    rng = np.random.default_rng(3)
    d, e = 4, 12
    w = _w(rng, d, e)
    F = rng.normal(size=(1, d))
    x = rng.normal(size=(1, d))
    o, h = tgf_forward(F, x, w)
    # the same computation written element by element
    cat = list(F[0]) + list(x[0])
    hh = [sum(cat[k] * w["Wm"][i, k] for k in range(2 * d)) + w["bm"][i] for i in range(d)]

    def ln(v, g, b):
        mu = sum(v) / len(v)
        var = sum((t - mu) ** 2 for t in v) / len(v)
        return [(t - mu) / math.sqrt(var + 1e-5) * g[i] + b[i] for i, t in enumerate(v)]

    zin = ln(hh, w["g_h"], w["b_h"]) + ln(list(x[0]), w["g_x"], w["b_x"])
    z = [sum(zin[k] * w["Wu"][j, k] for k in range(2 * d)) + w["bu"][j] for j in range(e)]
    s = [t / (1 + math.exp(-t)) for t in z]
    oo = [sum(s[j] * w["Wd"][i, j] for j in range(e)) + w["bd"][i] + hh[i] for i in range(d)]
    np.testing.assert_allclose(h[0], hh, rtol=1e-12)
    np.testing.assert_allclose(o[0], oo, rtol=1e-12)
