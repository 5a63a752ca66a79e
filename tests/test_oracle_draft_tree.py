"""Pins of the draft-tree oracle (dynamic tree from top-k expansions, the
EAGLE-2 construction GRIFFIN uses): a hand-worked example, the greedy-chain
special case, and invariants checked by brute force on random trees."""

import math

import numpy as np
import pytest

from oracle.draft_tree import draft_tree, pool_size


def test_hand_example():
    # V = 4, k = 2, D = 2.  Root logits [2, 0, 1, -1]: top-2 = tokens 0, 2 with
    # log-probs 2 - lse0 and 1 - lse0, lse0 = log(e^2 + 1 + e + e^-1).
    # Step 1, slot 0 (token 0, the better node) logits [0, 3, 0, 0]: top-2 =
    # tokens 1, then 0 (the lowest id of the tied zeros); slot 1 (token 2)
    # logits [5, 0, 0, 0]: tokens 0, then 1.
    steps = [np.array([[2.0, 0.0, 1.0, -1.0]]), np.array([[0.0, 3.0, 0.0, 0.0], [5.0, 0.0, 0.0, 0.0]])]
    lse0 = math.log(math.exp(2) + 1 + math.exp(1) + math.exp(-1))
    la = math.log(3 + math.exp(3))
    lb = math.log(math.exp(5) + 3)
    s1, s2 = 2 - lse0, 1 - lse0                      # pool 1 (token 0), pool 2 (token 2)
    s3, s4 = s1 + 3 - la, s1 + 0 - la                # pool 3 (token 1), pool 4 (token 0), parent 1
    s5, s6 = s2 + 5 - lb, s2 + 0 - lb                # pool 5 (token 0), pool 6 (token 1), parent 2
    # scores: s1 -0.440 > s3 -0.579 > s2 -1.440 > s5 -1.460 > s4 -3.579 > s6 -6.460
    out = draft_tree(7, steps, k=2, D=2, N=4)
    np.testing.assert_allclose(out["pool"]["score"], [0, s1, s2, s3, s4, s5, s6], rtol=1e-12, atol=1e-12)
    assert out["pool"]["token"] == [7, 0, 2, 1, 0, 0, 1]
    assert out["pool"]["parent"] == [-1, 0, 0, 1, 1, 2, 2]
    assert out["keep"] == [0, 1, 2, 3]
    assert out["parents"].tolist() == [-1, 0, 0, 1] and out["tokens"].tolist() == [7, 0, 2, 1]
    out5 = draft_tree(7, steps, k=2, D=2, N=5)
    assert out5["keep"] == [0, 1, 2, 3, 5]
    assert out5["parents"].tolist() == [-1, 0, 0, 1, 2] and out5["tokens"].tolist() == [7, 0, 2, 1, 0]
    assert out5["margin"] == pytest.approx(s5 - s4, rel=1e-9)      # the rerank boundary


def test_greedy_chain():
    # k = 1: every step expands its single best candidate, so the tree is the
    # chain of each step's argmax token.
    rng = np.random.default_rng(4)
    D, V = 6, 50
    steps = [rng.normal(size=(1, V)) for _ in range(D)]
    out = draft_tree(3, steps, k=1, D=D, N=D + 1)
    assert pool_size(1, D) == D + 1
    assert out["parents"].tolist() == [-1] + list(range(D))
    assert out["tokens"].tolist() == [3] + [int(np.argmax(s[0])) for s in steps]


def _prob(row, t):
    e = np.exp(np.asarray(row, dtype=np.float64))
    return e[t] / e.sum()


@pytest.mark.parametrize("k,D,N,V,seed", [(10, 6, 60, 200, 1), (4, 5, 20, 30, 2), (3, 3, 8, 3, 3), (16, 2, 64, 500, 4)])
def test_invariants_by_brute_force(k, D, N, V, seed):
    rng = np.random.default_rng(seed)
    steps = [rng.normal(size=(1, V)) * 2] + [rng.normal(size=(k, V)) * 2 for _ in range(D - 1)]
    out = draft_tree(11, steps, k, D, N)
    pool = out["pool"]
    P = len(pool["token"])
    assert P == pool_size(k, D)
    # which expansion slot each pool node was expanded from
    slot = {}
    for j, ids in enumerate(out["expanded"]):
        for s, pid in enumerate(ids):
            slot[pid] = (j, s)
        # expanded nodes are listed best first (the slot order)
        sc = [pool["score"][i] for i in ids]
        assert all(a >= b for a, b in zip(sc, sc[1:]))
    # every pool score is the log of the product of its path's draft probabilities
    for i in range(1, P):
        prod, n = 1.0, i
        while n != 0:
            par = pool["parent"][n]
            j, s = slot[par]
            prod *= _prob(steps[j][s], pool["token"][n])
            n = par
        assert pool["score"][i] == pytest.approx(math.log(prod), rel=1e-9, abs=1e-9)
        assert pool["score"][i] < pool["score"][pool["parent"][i]]          # log-probs < 0
        assert pool["depth"][i] == pool["depth"][pool["parent"][i]] + 1
    # each step expands the k best of that step's candidates (by probability)
    for j in range(1, D):
        cands = [i for i in range(1, P) if pool["depth"][i] == j]
        best = sorted(cands, key=lambda i: (-pool["score"][i], i))[:k]
        assert out["expanded"][j] == best
    # the children of an expanded node are its k most probable tokens
    for pid, (j, s) in slot.items():
        kids = [pool["token"][i] for i in range(P) if pool["parent"][i] == pid]
        assert kids == sorted(range(V), key=lambda t: (-steps[j][s][t], t))[:k]
    # the kept set: N nodes, the root first, closed under parents, and no
    # dropped node scores above a kept one
    keep = out["keep"]
    assert len(keep) == N and keep[0] == 0 and keep == sorted(keep)
    ks = set(keep)
    assert all(pool["parent"][i] in ks for i in keep[1:])
    dropped = [i for i in range(1, P) if i not in ks]
    if dropped:
        assert min(pool["score"][i] for i in keep[1:]) >= max(pool["score"][i] for i in dropped)
    par = out["parents"]
    assert par[0] == -1 and all(0 <= par[i] < i for i in range(1, N))
    for i in range(1, N):
        assert keep[par[i]] == pool["parent"][keep[i]]
        assert out["tokens"][i] == pool["token"][keep[i]]
    assert max(pool["depth"][i] for i in keep) <= D


def test_flat_tail_keeps_the_first_level():
    # the root spreads its mass over k tokens (log-probs -1.42 .. -1.82) and
    # every deeper step is uniform over 40 tokens (-3.69 a level): the best
    # N - 1 = k nodes are exactly the root's children, best first
    V, k, D = 40, 5, 4
    root = np.full((1, V), -20.0)
    root[0, [3, 9, 1, 30, 22]] = [5.0, 4.9, 4.8, 4.7, 4.6]
    steps = [root] + [np.zeros((k, V)) for _ in range(D - 1)]
    out = draft_tree(0, steps, k, D, N=k + 1)
    assert out["parents"].tolist() == [-1] * 1 + [0] * k
    assert out["tokens"].tolist() == [0, 3, 9, 1, 30, 22]


def test_uniform_logits_tie_rules_by_hand():
    # Every logit equal (V = 4, k = 2, D = 3, N = 6): every candidate of a
    # step scores the same, so the tie rules alone decide the tree.
    # Step 0 expands the root: tokens 0, 1 (lower ids first) -> pool 1, 2,
    # both -log 4.  Selection of the two nodes expanded next, ties toward the
    # earlier pool node: slot 0 = pool 1, slot 1 = pool 2.  Step 1: slot 0's
    # children are pool 3, 4 (tokens 0, 1), slot 1's pool 5, 6, all -2 log 4;
    # the next expansion takes pool 3, 4 (both children of pool 1).  Step 2
    # adds pool 7 .. 10 (children of 3 and 4), -3 log 4 each.  Rerank of the
    # N - 1 = 5 best: pool 1, 2 and the three earliest of 3 .. 6, i.e. 3, 4, 5.
    V, k, D, N = 4, 2, 3, 6
    steps = [np.zeros((1, V)), np.zeros((k, V)), np.zeros((k, V))]
    out = draft_tree(9, steps, k=k, D=D, N=N)
    l4 = math.log(4)
    assert out["expanded"] == [[0], [1, 2], [3, 4]]
    assert out["pool"]["parent"] == [-1, 0, 0, 1, 1, 2, 2, 3, 3, 4, 4]
    assert out["pool"]["token"] == [9, 0, 1, 0, 1, 0, 1, 0, 1, 0, 1]
    np.testing.assert_allclose(out["pool"]["score"], [0] + [-l4] * 2 + [-2 * l4] * 4 + [-3 * l4] * 4,
                               rtol=1e-13)
    assert out["keep"] == [0, 1, 2, 3, 4, 5]
    assert out["parents"].tolist() == [-1, 0, 0, 1, 1, 2]
    assert out["tokens"].tolist() == [9, 0, 1, 0, 1, 0]
