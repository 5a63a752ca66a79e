"""Oracle: construction of the dynamic draft tree (the draft side of one
GRIFFIN cycle).

TEST INFRASTRUCTURE ONLY (see the package docstring).

GRIFFIN's draft trees are dynamic, 60 draft tokens deep 6 (Implementation
Details appendix), built the EAGLE-2 way from top-k expansions (Section 4.1:
each draft forward pass yields a top-k list per position).  The steps, for
one sequence:

* the pool starts with the root (the last verified token), score 0;
* expansion step j = 0 .. D-1: each node being expanded (the root at step
  0; afterwards the k nodes selected from the previous step's candidates)
  proposes the k tokens of highest draft probability; a candidate's score is
  its parent's score plus the log-probability of its token (log softmax of
  that node's draft logits).  All candidates join the pool; the k best of
  this step's candidates are the nodes expanded at the next step;
* rerank: the N - 1 pool nodes of highest score, with the root, form the tree
  given to the verify pass, listed in pool order (parents before children).

Readings (the paper names the construction but not its rules): scores are
summed log-probabilities (the log of EAGLE-2's product of confidences); every
ordering is by score, larger first, then by the earlier pool position;
top-k within a row is by logit, larger first, then by the lower token id; the
logits of step j >= 1 are given per expanded slot, slot s being the s-th best
node selected after step j - 1; N counts the root (60 nodes = the root and
59 drafted tokens; depth D = 6 drafted levels).  Log-probabilities are taken
in float64 of the given logits.

Because every log-probability is <= 0, a node never scores above its parent
and precedes it in no ordering here, so the kept set is closed under
ancestors.
"""

import numpy as np


def log_softmax(row):
    """Float64 log-probabilities of one logit row."""
    x = np.asarray(row, dtype=np.float64)
    m = x.max()
    return x - (m + np.log(np.exp(x - m).sum()))


def topk_ids(row, k):
    """The k ids of largest value, larger first, lower id first on ties."""
    x = np.asarray(row, dtype=np.float64)
    order = np.lexsort((np.arange(x.size), -x))
    return order[:k]


def expand_step(pool, expanded, logits, k):
    """One expansion step.  ``pool`` is a dict of lists (token, parent, score,
    depth), ``expanded`` the pool ids being expanded (slot order), ``logits``
    [len(expanded)][V].  Appends the candidates to the pool and returns their
    pool ids in slot-major, rank-minor order."""
    cands = []
    for s, pid in enumerate(expanded):
        row = np.asarray(logits[s], dtype=np.float64)
        lp = log_softmax(row)
        ids = topk_ids(row, k)
        for t in ids:
            pool["token"].append(int(t))
            pool["parent"].append(int(pid))
            pool["score"].append(pool["score"][pid] + lp[t])
            pool["depth"].append(pool["depth"][pid] + 1)
            cands.append(len(pool["token"]) - 1)
    return cands


def best(pool, ids, n):
    """The n ids of highest score, ties to the earlier pool id; and the score
    gap between the n-th and the (n+1)-th (a decision margin: the scores are
    sums of log-probabilities, so a computation in another precision can
    order a near-tie differently; an exact tie of equal computations cannot)."""
    ids = list(ids)
    sc = np.array([pool["score"][i] for i in ids])
    order = np.lexsort((np.array(ids), -sc))
    chosen = [ids[o] for o in order[:n]]
    gap = sc[order[n - 1]] - sc[order[n]] if len(ids) > n else np.inf
    return chosen, gap


def draft_tree(root_token, step_logits, k, D, N):
    """Build one sequence's tree.  ``step_logits[0]`` is [1][V] (the root's
    logits), ``step_logits[j]`` for 1 <= j < D is [k][V] (slot order).
    Returns a dict: ``parents`` int [N] (-1 for the root, else an index < i),
    ``tokens`` int [N], ``pool`` (token, parent, score, depth lists),
    ``expanded`` (the pool ids expanded at each step), ``margin`` (the
    smallest score gap at a selection boundary; the top-k of a row compares
    the given logits themselves and needs none)."""
    pool = {"token": [int(root_token)], "parent": [-1], "score": [0.0], "depth": [0]}
    expanded = [0]
    steps = [list(expanded)]
    margin = np.inf
    for j in range(D):
        cands = expand_step(pool, expanded, step_logits[j], k)
        if j + 1 < D:
            expanded, gap = best(pool, cands, k)
            margin = min(margin, gap)
            steps.append(list(expanded))
    kept, gap = best(pool, range(1, len(pool["token"])), N - 1)
    margin = min(margin, gap)
    keep = sorted([0] + kept)
    where = {pid: i for i, pid in enumerate(keep)}
    parents = np.array([-1 if pid == 0 else where[pool["parent"][pid]] for pid in keep], dtype=np.int64)
    tokens = np.array([pool["token"][pid] for pid in keep], dtype=np.int64)
    return {"parents": parents, "tokens": tokens, "pool": pool, "expanded": steps, "keep": keep,
            "margin": float(margin)}


def pool_size(k, D):
    """Pool nodes of a full construction: the root, k at depth 1, k*k at each
    deeper level."""
    return 1 + k + (D - 1) * k * k
