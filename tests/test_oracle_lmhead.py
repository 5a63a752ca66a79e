"""Pins for the LM-head / selection oracle.

* projection against explicit per-element dot products on tiny shapes;
* planted hidden states (the generator's closed form) make the planted token
  the argmax, for every workload's vocabulary and hidden sizes;
* argmax / top-k tie rules against exhaustive Python sorting;
* log-sum-exp against ``scipy.special.logsumexp`` and the closed form of a
  constant row.
"""

import math

import numpy as np
import pytest
import torch
from scipy.special import logsumexp

from oracle.lmhead import lmhead_logits, select_argmax, select_topk, row_logsumexp
from paper_2502_11018_gb300 import inputs


def test_projection_brute_force():
    rng = np.random.default_rng(0)
    h = rng.normal(size=(5, 7))
    W = rng.normal(size=(11, 7))
    logits = lmhead_logits(h, W)
    for r in range(5):
        for v in range(11):
            acc = 0.0
            for k in range(7):
                acc += h[r, k] * W[v, k]
            assert abs(logits[r, v] - acc) < 1e-12


@pytest.mark.parametrize("V,H,dtype", [(4096, 512, torch.float32), (32000, 1024, torch.bfloat16),
                                       (9000, 4096, torch.bfloat16)])
def test_planted_argmax_closed_form(V, H, dtype):
    gen = torch.Generator().manual_seed(5)
    W = (torch.randn(V, H, generator=gen) * 0.02).to(dtype)
    targets = torch.randint(0, V, (24,), generator=gen)
    h = inputs.planted_hidden(gen, W, targets)
    logits = lmhead_logits(h.double().numpy(), W.double().numpy())
    ids, vals = select_argmax(logits)
    np.testing.assert_array_equal(ids, targets.numpy())
    top2 = np.sort(logits, axis=1)[:, -2:]
    assert ((top2[:, 1] - top2[:, 0]) > 1e-2 * np.abs(logits).max()).all()


def test_argmax_ties_lowest_id():
    logits = np.array([[0.0, 3.0, 1.0, 3.0], [2.0, 2.0, 2.0, 2.0], [-1.0, -5.0, -1.0, -7.0]])
    ids, vals = select_argmax(logits)
    assert ids.tolist() == [1, 0, 0]
    assert vals.tolist() == [3.0, 2.0, -1.0]


@pytest.mark.parametrize("k", [1, 3, 10])
def test_topk_against_exhaustive_sort(k):
    rng = np.random.default_rng(k)
    logits = np.round(rng.normal(size=(6, 40)), 1)   # rounding forces many ties
    ids, vals = select_topk(logits, k)
    for r in range(6):
        ref = sorted(range(40), key=lambda v: (-logits[r, v], v))[:k]
        assert ids[r].tolist() == ref
        assert vals[r].tolist() == [logits[r, v] for v in ref]


def test_logsumexp():
    rng = np.random.default_rng(9)
    logits = rng.normal(scale=30.0, size=(4, 1000))
    m, lse = row_logsumexp(logits)
    np.testing.assert_allclose(lse, logsumexp(logits, axis=1), rtol=0, atol=1e-12)
    np.testing.assert_array_equal(m, logits.max(axis=1))
    const = np.full((1, 64), 2.5)
    _, lse_c = row_logsumexp(const)
    assert abs(lse_c[0] - (2.5 + math.log(64))) < 1e-13
