"""Pins for the tree-build oracle (ancestor sets, depths, positions).

The oracle walks parent chains.  These tests check it against closed forms
(chain and star trees), against a different method (a top-down traversal
from the root that propagates ancestor sets to children), and against the
validity rules of the parent-array encoding.
"""

import os

import numpy as np
import pytest

import oracle
from oracle.tree import tree_build, GV_OK, GV_ERR_INVALID_TREE
from paper_2502_11018_gb300 import inputs


def test_chain_tree_closed_form():
    N, P = 64, 37
    parents = np.arange(-1, N - 1, dtype=np.int32)[None, :]
    depth, pos, anc, st = tree_build(parents, [P])
    assert st[0] == 0
    for i in range(N):
        assert depth[0, i] == i
        assert pos[0, i] == P + i
        assert int(anc[0, i]) == (1 << (i + 1)) - 1


def test_star_tree_closed_form():
    N = 17
    parents = np.zeros((1, N), dtype=np.int32)
    parents[0, 0] = -1
    depth, pos, anc, st = tree_build(parents, [5])
    assert int(anc[0, 0]) == 1 and depth[0, 0] == 0 and pos[0, 0] == 5
    for i in range(1, N):
        assert depth[0, i] == 1
        assert pos[0, i] == 6
        assert int(anc[0, i]) == (1 | (1 << i))


def _top_down(parents):
    """Ancestor sets by a breadth-first pass from the root over child lists."""
    N = len(parents)
    kids = [[] for _ in range(N)]
    for i in range(1, N):
        kids[parents[i]].append(i)
    sets = {0: {0}}
    depth = {0: 0}
    frontier = [0]
    while frontier:
        nxt = []
        for u in frontier:
            for c in kids[u]:
                sets[c] = sets[u] | {c}
                depth[c] = depth[u] + 1
                nxt.append(c)
        frontier = nxt
    return sets, depth


@pytest.mark.parametrize("seed", range(12))
def test_random_trees_against_top_down(seed):
    rng = np.random.default_rng(seed)
    B = 3
    N = int(rng.integers(1, 65))
    parents = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        if N == 1:
            parents[b] = [-1]
            continue
        # depth 1 holds at most 8 nodes below the root; deeper trees hold more
        D = int(rng.integers(1 if N <= 9 else 2, min(N - 1, 10) + 1))
        parents[b], _ = inputs.make_tree(rng, N, D, 8, 1000)
    P = rng.integers(0, 5000, size=B)
    depth, pos, anc, st = tree_build(parents, P)
    assert (st == 0).all()
    for b in range(B):
        sets, dep = _top_down(parents[b])
        for i in range(N):
            bits = int(anc[b, i])
            assert {j for j in range(N) if (bits >> j) & 1} == sets[i]
            assert bin(bits).count("1") == depth[b, i] + 1
            assert depth[b, i] == dep[i]
            assert pos[b, i] == P[b] + dep[i]


@pytest.mark.parametrize("bad", [
    [0, 0, 1],            # root not -1
    [-1, 1, 1],           # self reference
    [-1, 0, 3, 1],        # forward reference
    [-1, 0, -1],          # second root
    [-1, 0, 5],           # out of range
])
def test_invalid_trees(bad):
    parents = np.array([bad], dtype=np.int32)
    depth, pos, anc, st = tree_build(parents, [9])
    assert st[0] == GV_ERR_INVALID_TREE
    N = len(bad)
    assert (depth == 0).all() and (pos == 9).all()
    assert [int(a) for a in anc[0]] == [1 << i for i in range(N)]


def test_too_many_nodes_invalid():
    parents = np.arange(-1, 64, dtype=np.int32)[None, :]   # 65 nodes
    _, _, _, st = tree_build(parents, [0])
    assert st[0] == GV_ERR_INVALID_TREE


def test_generator_tree_shape():
    """The EAGLE-2 style generator yields topological, sibling-unique trees
    of exactly the requested size and depth (Appendix C: 60 tokens)."""
    rng = np.random.default_rng(7)
    for N, D in [(60, 6), (60, 8), (16, 4), (64, 8), (7, 6)]:
        parents, tokens = inputs.make_tree(rng, N, D, 10 if N > 16 else 4, 32000)
        depth, _, _, st = tree_build(parents[None], [0])
        assert st[0] == 0
        assert depth.max() == D
        for u in range(N):
            kids = [int(tokens[c]) for c in range(1, N) if parents[c] == u]
            assert len(kids) == len(set(kids))
    assert oracle.GV_OK == 0


def _golden(name):
    path = os.path.join(os.path.dirname(__file__), "golden", name)
    vals = {}
    with open(path) as f:
        for line in f:
            line = line.split("#", 1)[0].split()
            if len(line) == 2:
                vals[line[0]] = int(line[1])
    return vals


def test_paper_tree_configuration():
    """The tree size and depth the paper prints (Appendix, draft tree
    structure) yield, through the generator and the oracle, a valid tree of
    exactly that many nodes whose deepest node sits at that depth, with
    positions P + depth and one ancestor bit per level."""
    g = _golden("draft_tree_config.txt")
    N, D = g["draft_tokens"], g["depth"]
    rng = np.random.default_rng(11)
    parents, _ = inputs.make_tree(rng, N, D, 10, 32000)
    P = 37
    depth, pos, anc, st = tree_build(parents[None], [P])
    assert st[0] == GV_OK and parents.shape == (N,)
    assert depth.max() == D
    np.testing.assert_array_equal(pos[0], P + depth[0])
    assert all(bin(int(a)).count("1") == int(dd) + 1 for a, dd in zip(anc[0], depth[0]))
