"""Oracle: the token-alignable training objective of the draft model.

TEST INFRASTRUCTURE ONLY (see the package docstring): only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU legs may use it.

GRIFFIN Section 4.1 trains the draft model in passes n = 1, 2, ...; in pass n
the draft model predicts, at every position t of a training sequence, a
feature Fd_t and draft logits Xd_t[V], conditioned on its own outputs of the
earlier passes.  With the ground-truth tokens x_t and the target model's
features Ft_t:

* predictable mask (Section 4.1): mbar_t = 1 iff x_t is among the top-k
  tokens of Xd_t;
* alignment mask (Eq. 3): m_t = product of the predictable masks of the draft
  tokens that the pass-n prediction at t was conditioned on;
* per-step loss (Implementation Details appendix):
  ell_t = lam_tok * (-log softmax(Xd_t)[x_t]) + lam_feat * ||Fd_t - Ft_t||_1,
  with lam_tok = 1 and lam_feat = 0.1 by default;
* pass loss (Eq. 5): L = sum_t m_t ell_t / sum_t m_t; the first pass (Eq. 2)
  uses m_t = 1 everywhere.

Readings where the paper is silent or ambiguous:

* ties in the top-k: the top-k are the k largest logits with ties broken
  toward the lower token id (the rule of every selection in this project), so
  x_t is predictable iff fewer than k tokens v have Xd_t[v] > Xd_t[x_t], or
  Xd_t[v] == Xd_t[x_t] and v < x_t; the comparisons use the logits as given
  (float64 widening of fp32 / bf16 values is exact);
* Eq. 3 writes the product over positions t-n+1 .. t-1 without a pass index.
  It is read along the draft chain that produced the pass-n prediction at t:
  the chain started at position t-n+1 in pass 1, and its j-th token (position
  t-n+j) was predicted in pass j, so m_t = prod_{j=1}^{n-1} mbar^(j)_{t-n+j};
  a position whose chain would start before the sequence (t < n-1) gets
  m_t = 0;
* Eq. 5 is a per-sequence loss; a sequence with sum_t m_t = 0 has loss 0.

Every function works in float64 with plain loops over rows and single numpy
primitives inside a row, in the order the definitions above state.
"""

import numpy as np


def predictable_mask(logits, tokens, k):
    """``mbar[r] = 1`` iff ``tokens[r]`` is among the top-k of ``logits[r]``
    (ties toward the lower id).  logits [R][V], tokens [R] -> uint8 [R]."""
    logits = np.asarray(logits, dtype=np.float64)
    tokens = np.asarray(tokens)
    R, V = logits.shape
    ids = np.arange(V)
    out = np.zeros(R, dtype=np.uint8)
    for r in range(R):
        x = int(tokens[r])
        lx = logits[r, x]
        ahead = np.count_nonzero((logits[r] > lx) | ((logits[r] == lx) & (ids < x)))
        out[r] = 1 if ahead < k else 0
    return out


def token_loss(logits, tokens):
    """Cross-entropy of the one-hot target: ``logsumexp(logits[r]) -
    logits[r][tokens[r]]`` (the max is subtracted before the exponentials)."""
    logits = np.asarray(logits, dtype=np.float64)
    R = logits.shape[0]
    out = np.zeros(R, dtype=np.float64)
    for r in range(R):
        m = logits[r].max()
        lse = m + np.log(np.exp(logits[r] - m).sum())
        out[r] = lse - logits[r, int(tokens[r])]
    return out


def feature_loss(feat_draft, feat_target):
    """``||Fd_r - Ft_r||_1`` per row.  [R][H] -> [R]."""
    fd = np.asarray(feat_draft, dtype=np.float64)
    ft = np.asarray(feat_target, dtype=np.float64)
    return np.abs(fd - ft).sum(axis=1)


def alignment_mask(mbar_prev, n, B, T):
    """Eq. 3 along the draft chain: ``m[b][t] = prod_{j=1}^{n-1}
    mbar_prev[j-1][b][t-n+j]``, 0 where the chain would start before the
    sequence, 1 everywhere for n = 1.  mbar_prev [n-1][B][T] -> uint8 [B][T]."""
    m = np.zeros((B, T), dtype=np.uint8)
    for b in range(B):
        for t in range(T):
            if t - n + 1 < 0:
                continue
            v = 1
            for j in range(1, n):
                v *= int(mbar_prev[j - 1][b][t - n + j])
            m[b, t] = v
    return m


def tat_pass(logits, tokens, feat_draft, feat_target, k, n, mbar_prev=None,
             lam_tok=1.0, lam_feat=0.1):
    """One training pass n (Eqs. 2-5).  logits [B][T][V], tokens [B][T],
    features [B][T][H], mbar_prev [n-1][B][T] (None for n = 1).

    Returns a dict: ``mbar`` [B][T] (this pass's predictable mask), ``mask``
    [B][T] (m_t), ``ell`` [B][T] (per-step loss), ``seq_loss`` [B]."""
    logits = np.asarray(logits, dtype=np.float64)
    B, T, V = logits.shape
    H = np.asarray(feat_draft).shape[-1]
    rows_logits = logits.reshape(B * T, V)
    rows_tok = np.asarray(tokens).reshape(B * T)
    mbar = predictable_mask(rows_logits, rows_tok, k).reshape(B, T)
    ell = (lam_tok * token_loss(rows_logits, rows_tok)
           + lam_feat * feature_loss(np.asarray(feat_draft).reshape(B * T, H),
                                     np.asarray(feat_target).reshape(B * T, H))).reshape(B, T)
    if n == 1:
        mask = np.ones((B, T), dtype=np.uint8)
    else:
        mask = alignment_mask(mbar_prev, n, B, T)
    seq_loss = np.zeros(B, dtype=np.float64)
    for b in range(B):
        den = float(mask[b].sum())
        num = float((mask[b] * ell[b]).sum())
        seq_loss[b] = num / den if den > 0 else 0.0
    return {"mbar": mbar, "mask": mask, "ell": ell, "seq_loss": seq_loss}
