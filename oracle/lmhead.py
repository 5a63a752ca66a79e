"""Oracle: LM head projection and per-row selection.

GRIFFIN Section 3 / Eq. 1: the LM head maps a final hidden feature to a
token, ``x = H(F)``.  In the verify pass every draft node's final hidden state
``h[r]`` (a row of ``h[rows][H]``) is projected by ``W[V][H]``:
``logits[r][v] = sum_k h[r][k] * W[v][k]``.  Section 4.1 uses the top-k of
these scores; Section 5 uses greedy choice (T = 0) and sampling (T = 1).

Selections (readings where the paper is silent):

* argmax: the largest logit, ties broken toward the lowest token id;
* top-k: ``k`` ids by decreasing logit, ties broken toward the lower id;
* log-sum-exp of a row: ``m + log(sum exp(logit - m))`` with ``m`` the row max.
"""

import numpy as np


def lmhead_logits(h, W):
    """``logits[r][v] = h[r] . W[v]`` in float64 (one matmul)."""
    return np.asarray(h, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T


def select_argmax(logits):
    """Per row: ``(id, value)`` of the maximum, lowest id on ties."""
    logits = np.asarray(logits, dtype=np.float64)
    rows = logits.shape[0]
    ids = np.zeros(rows, dtype=np.int32)
    vals = np.zeros(rows, dtype=np.float64)
    for r in range(rows):
        # np.argmax returns the first maximal index, i.e. the lowest id.
        best = int(np.argmax(logits[r]))
        ids[r] = best
        vals[r] = logits[r, best]
    return ids, vals


def select_topk(logits, k):
    """Per row: ``k`` ids by decreasing logit (lower id first on ties)."""
    logits = np.asarray(logits, dtype=np.float64)
    # A stable sort of the negated values keeps equal logits in id order.
    order = np.argsort(-logits, axis=1, kind="stable")[:, :k]
    vals = np.take_along_axis(logits, order, axis=1)
    return order.astype(np.int32), vals


def row_logsumexp(logits):
    """Per row ``(max, lse)`` with ``lse = max + log(sum(exp(logit - max)))``."""
    logits = np.asarray(logits, dtype=np.float64)
    m = logits.max(axis=1)
    lse = m + np.log(np.exp(logits - m[:, None]).sum(axis=1))
    return m, lse
