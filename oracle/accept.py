"""Oracle: acceptance of a verified draft tree.

Greedy acceptance (temperature 0).  Section 3 of GRIFFIN: the target model
verifies the draft tokens and accepts a subset; Section 4.1: rejecting a draft
token discards every later token of its draft sequence; Section 5: the method
is lossless, which for T = 0 means the output equals greedy decoding.  A
non-root node ``j`` *matches* when its token equals the target's choice at its
parent, ``tokens[j] == choice[parents[j]]``.  A node is *accepted* when every
non-root node of its root chain matches.  The accepted path is the chain of
the deepest accepted node (ties toward the smallest node index; the root is
always accepted).  Outputs per sequence:

* ``path``: the chain's node indices root first, ``accept_len = depth + 1``
  entries, padded with -1 to ``D + 1``;
* ``out_tokens``: the accepted draft tokens (``path[1:]``) followed by the
  bonus token ``choice[last node]``, padded with -1 to ``D + 1``.

Temperature-1 acceptance.  Section 5 claims losslessness at T = 1 "like prior
speculative decoding methods"; Section 3 cites speculative sampling and
Section 2 SpecInfer for tree verification.  The reading taken is multi-draft
recursive rejection sampling with the children of a node drawn from the draft
distribution at that node:

1. ``u = root``.
2. ``p = softmax(target_logits[u] / T)``, ``q = softmax(draft_logits[u] / T)``.
3. For each child ``c`` of ``u`` in increasing index order, with ``x = tokens[c]``:
   accept ``c`` when ``u_acc[c] <= p(x) / q(x)`` (always when ``q(x) == 0``);
   on acceptance set ``u = c`` and go to 2; on rejection replace ``p`` by
   ``max(p - q, 0) / sum(max(p - q, 0))`` (kept unchanged if that sum is 0).
4. When no child of ``u`` is accepted (or ``u`` is a leaf) the bonus token is
   the inverse-CDF draw of the current ``p`` at ``u_res[u]``: the smallest
   ``v`` with ``sum_{w <= v} p(w) > u_res[u] * sum_w p(w)``.

Variant without a draft distribution (``draft_logits`` None): the children are
deterministic proposals (EAGLE-style top-k drafts), so ``q(x)`` is taken as 1
for every drafted token.  Step 3 then accepts ``c`` when ``u_acc[c] <= p(x)``,
and a rejection sets ``p(x) = 0`` and renormalises ``p`` (kept unchanged if
nothing is left).  With distinct children this draws the emitted token from
``p`` exactly (sampling without replacement), so it is lossless too.
"""

import numpy as np

from .tree import GV_OK, GV_ERR_INVALID_TREE, tree_is_valid, chain


def _pad(seq, width):
    out = np.full(width, -1, dtype=np.int32)
    out[: len(seq)] = seq
    return out


def accept_greedy(parents, tokens, choice, D, seq_status=None):
    """Greedy acceptance; returns ``(path, accept_len, out_tokens, status)``.

    ``choice`` is the target's argmax per node, ``choice[b * N + i]``.
    A sequence whose input status is non-zero is skipped (``accept_len = 0``,
    rows of -1, status kept).  A tree with a node deeper than ``D`` gets
    ``GV_ERR_INVALID_TREE`` and is skipped the same way.
    """
    parents = np.asarray(parents)
    tokens = np.asarray(tokens)
    B, N = parents.shape
    choice = np.asarray(choice).reshape(B, N)
    path = np.full((B, D + 1), -1, dtype=np.int32)
    out_tokens = np.full((B, D + 1), -1, dtype=np.int32)
    accept_len = np.zeros(B, dtype=np.int32)
    status = np.zeros(B, dtype=np.int32) if seq_status is None else np.array(seq_status, dtype=np.int32)
    for b in range(B):
        if status[b] != GV_OK:
            continue
        if not tree_is_valid(parents[b]):
            status[b] = GV_ERR_INVALID_TREE
            continue
        chains = [chain(parents[b], i) for i in range(N)]
        if max(len(c) for c in chains) - 1 > D:
            status[b] = GV_ERR_INVALID_TREE
            continue
        best = 0
        for i in range(N):
            ok = all(int(tokens[b, j]) == int(choice[b, parents[b, j]]) for j in chains[i][1:])
            if ok and len(chains[i]) > len(chains[best]):
                best = i
        p = chains[best]
        path[b] = _pad(p, D + 1)
        accept_len[b] = len(p)
        out_tokens[b] = _pad([int(tokens[b, j]) for j in p[1:]] + [int(choice[b, best])], D + 1)
    return path, accept_len, out_tokens, status


def _softmax(x, T):
    z = np.asarray(x, dtype=np.float64) / T
    z = z - z.max()
    e = np.exp(z)
    return e / e.sum()


def _children(parents_row, u):
    return [c for c in range(len(parents_row)) if int(parents_row[c]) == u]


def _inverse_cdf(p, u):
    """Smallest ``v`` with ``cumsum(p)[v] > u * sum(p)``, and its margin.

    The margin is the distance of ``u * sum(p)`` from the nearer of the two
    CDF boundaries that bracket it, divided by ``sum(p)``.
    """
    c = np.cumsum(p)
    tot = c[-1]
    target = u * tot
    v = int(np.searchsorted(c, target, side="right"))
    v = min(v, len(p) - 1)
    lo = c[v - 1] if v > 0 else 0.0
    margin = min(target - lo, c[v] - target) / tot
    return v, margin


def _residual(p, q, x):
    """The unnormalised distribution after a rejected draft token ``x``:
    ``max(p - q, 0)``, or ``p`` with ``p(x) = 0`` when there is no draft
    distribution (``q`` None)."""
    if q is None:
        r = p.copy()
        r[x] = 0.0
        return r
    return np.maximum(p - q, 0.0)


def accept_sampling(parents, tokens, target_logits, draft_logits, u_acc, u_res, D,
                    temperature=1.0, seq_status=None):
    """Temperature sampling acceptance; returns ``(path, accept_len, out_tokens,
    status, min_margin)``.

    ``min_margin[b]`` is the smallest distance, over every decision the oracle
    took for sequence ``b``, between the uniform and the threshold it was
    compared with (``|u_acc - p/q|``, or the CDF margin of the final draw).
    """
    parents = np.asarray(parents)
    tokens = np.asarray(tokens)
    B, N = parents.shape
    path = np.full((B, D + 1), -1, dtype=np.int32)
    out_tokens = np.full((B, D + 1), -1, dtype=np.int32)
    accept_len = np.zeros(B, dtype=np.int32)
    min_margin = np.full(B, np.inf)
    status = np.zeros(B, dtype=np.int32) if seq_status is None else np.array(seq_status, dtype=np.int32)
    for b in range(B):
        if status[b] != GV_OK:
            continue
        if not tree_is_valid(parents[b]) or max(len(chain(parents[b], i)) for i in range(N)) - 1 > D:
            status[b] = GV_ERR_INVALID_TREE
            continue
        u = 0
        trail = [0]
        emitted = []
        while True:
            p = _softmax(target_logits[b, u], temperature)
            q = None if draft_logits is None else _softmax(draft_logits[b, u], temperature)
            nxt = None
            for c in _children(parents[b], u):
                x = int(tokens[b, c])
                qx = 1.0 if q is None else q[x]
                if qx == 0.0:
                    nxt = c
                    break
                ratio = p[x] / qx
                min_margin[b] = min(min_margin[b], abs(float(u_acc[b, c]) - ratio))
                if float(u_acc[b, c]) <= ratio:
                    nxt = c
                    break
                r = _residual(p, q, x)
                s = r.sum()
                if s > 0.0:
                    p = r / s
            if nxt is None:
                v, m = _inverse_cdf(p, float(u_res[b, u]))
                min_margin[b] = min(min_margin[b], m)
                emitted.append(v)
                break
            trail.append(nxt)
            emitted.append(int(tokens[b, nxt]))
            u = nxt
        path[b] = _pad(trail, D + 1)
        accept_len[b] = len(trail)
        out_tokens[b] = _pad(emitted, D + 1)
    return path, accept_len, out_tokens, status, min_margin


def check_sampling_trail(parents_row, tokens_row, target_logits_row, draft_logits_row,
                         u_acc_row, u_res_row, trail, bonus, temperature=1.0, tol=1e-5):
    """Check that a given acceptance trail is one the rule above could take.

    Replays steps 2-4 along ``trail`` (root first) with float64 ``p`` and
    ``q``.  Every child rejected before the trail's next node must satisfy
    ``u_acc > p/q - tol``, the trail's next node ``u_acc <= p/q + tol``, and the
    bonus must lie within ``tol`` (in CDF units) of the inverse-CDF draw.
    Returns ``(valid, ambiguous)``: ``ambiguous`` counts decisions that fell
    within ``tol`` of their threshold (either outcome is then accepted).
    """
    ambiguous = 0
    for step, u in enumerate(trail):
        p = _softmax(target_logits_row[u], temperature)
        q = None if draft_logits_row is None else _softmax(draft_logits_row[u], temperature)
        nxt = trail[step + 1] if step + 1 < len(trail) else None
        for c in _children(parents_row, u):
            x = int(tokens_row[c])
            qx = 1.0 if q is None else q[x]
            ratio = np.inf if qx == 0.0 else p[x] / qx
            ua = float(u_acc_row[c])
            if abs(ua - ratio) <= tol:
                ambiguous += 1
            if c == nxt:
                if not ua <= ratio + tol:
                    return False, ambiguous
                break
            if not ua > ratio - tol:
                return False, ambiguous
            r = _residual(p, q, x)
            s = r.sum()
            if s > 0.0:
                p = r / s
        else:
            if nxt is not None:
                return False, ambiguous   # trail names a node that is not a child
        if nxt is None:
            cdf = np.cumsum(p)
            tot = cdf[-1]
            target = float(u_res_row[u]) * tot
            lo = cdf[bonus - 1] if bonus > 0 else 0.0
            hi = cdf[bonus]
            if not (lo - tol * tot <= target < hi + tol * tot):
                return False, ambiguous
            if min(abs(target - lo), abs(hi - target)) <= tol * tot:
                ambiguous += 1
    return True, ambiguous
