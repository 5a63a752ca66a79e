"""Pins for the acceptance oracles.

Greedy (T = 0): against a top-down search that descends from the root only
into matching children (a different formulation of "longest accepted root
chain"), the bounds ``1 <= accept_len <= D + 1``, a fully planted chain
(``D + 1``), no planting (``1``), and the tie rule for duplicate siblings.

Temperature 1: losslessness (Section 5).  With children drawn from the draft
distribution at their parent, the first emitted token must follow the
target distribution at the root, and the token emitted after an accepted
child must follow the target distribution at that child; both are checked by
chi-square tests on seeded trials.  A planted mistake in a copy of the oracle
(no residual update after a rejection) must fail the same test.
"""

import numpy as np
import pytest
from scipy.stats import chisquare

import oracle.accept as acc
from oracle.accept import accept_greedy, accept_sampling, check_sampling_trail
from oracle.tree import GV_ERR_INVALID_TREE, chain
from paper_2502_11018_gb300 import inputs


def _search(parents, tokens, choice):
    """Deepest node reachable from the root through matching children,
    smallest index among equally deep ones."""
    N = len(parents)
    kids = [[] for _ in range(N)]
    for i in range(1, N):
        kids[parents[i]].append(i)
    best, best_depth = 0, 0
    stack = [(0, 0)]
    while stack:
        u, dep = stack.pop()
        if dep > best_depth or (dep == best_depth and u < best):
            best, best_depth = u, dep
        for c in kids[u]:
            if tokens[c] == choice[u]:
                stack.append((c, dep + 1))
    return best


@pytest.mark.parametrize("seed", range(20))
def test_greedy_against_search(seed):
    rng = np.random.default_rng(seed)
    B, N, D, V = 3, int(rng.integers(2, 61)), 6, 50
    D = min(D, N - 1)
    parents = np.zeros((B, N), dtype=np.int32)
    tokens = np.zeros((B, N), dtype=np.int32)
    choice = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        parents[b], tokens[b] = inputs.make_tree(rng, N, D, 10, V)
        choice[b] = inputs.plant_choices(rng, parents[b], tokens[b], V, p_match=0.7)
    path, alen, out, st = accept_greedy(parents, tokens, choice.reshape(-1), D)
    assert (st == 0).all()
    for b in range(B):
        best = _search(parents[b], tokens[b], choice[b])
        ch = chain(parents[b], best)
        assert 1 <= alen[b] <= D + 1
        assert alen[b] == len(ch)
        assert path[b, :alen[b]].tolist() == ch
        assert (path[b, alen[b]:] == -1).all()
        assert out[b, :alen[b]].tolist() == [int(tokens[b, j]) for j in ch[1:]] + [int(choice[b, best])]
        assert (out[b, alen[b]:] == -1).all()


def test_full_chain_and_no_match():
    rng = np.random.default_rng(1)
    N, D, V = 60, 8, 1000
    parents, tokens = inputs.make_tree(rng, N, D, 10, V)
    # Choices that match the first child at every node: the top-1 chain of
    # depth D is accepted in full.
    kids = inputs.children_of(parents)
    choice = np.array([tokens[kids[u][0]] if kids[u] else 0 for u in range(N)], dtype=np.int32)
    _, alen, out, _ = accept_greedy(parents[None], tokens[None], choice, D)
    assert alen[0] == D + 1
    # Choices no child carries: only the root, and the bonus is the root's choice.
    choice = np.full(N, V + 5, dtype=np.int32)
    path, alen, out, _ = accept_greedy(parents[None], tokens[None], choice, D)
    assert alen[0] == 1 and path[0, 0] == 0 and out[0, 0] == V + 5


def test_duplicate_siblings_tie_rule():
    # root -> {1, 2} both carry token 7; 1 -> 3 (token 9), 2 -> 4 (token 9)
    parents = np.array([[-1, 0, 0, 1, 2]])
    tokens = np.array([[0, 7, 7, 9, 9]])
    choice = np.array([7, 9, 9, 1, 2])
    path, alen, out, _ = accept_greedy(parents, tokens, choice, 3)
    assert path[0].tolist() == [0, 1, 3, -1]
    assert out[0].tolist() == [7, 9, 1, -1]


def test_greedy_status_and_depth_errors():
    parents = np.array([[-1, 0, 1, 2], [-1, 0, 1, 2]])
    tokens = np.zeros((2, 4), dtype=np.int32)
    choice = np.zeros(8, dtype=np.int32)
    path, alen, out, st = accept_greedy(parents, tokens, choice, 2, seq_status=[0, -2])
    assert st.tolist() == [GV_ERR_INVALID_TREE, -2]     # depth 3 > D = 2; input status kept
    assert alen.tolist() == [0, 0] and (path == -1).all() and (out == -1).all()


# ---------------------------------------------------------------- T = 1 ---

V1 = 6
SHAPE = np.array([-1, 0, 0, 0, 1, 1, 2, 3, 3])     # root: 3 children; depth 2


def _tables(seed):
    rng = np.random.default_rng(seed)
    tgt = {(): rng.normal(scale=1.2, size=V1)}
    drf = {(): tgt[()] + rng.normal(scale=1.0, size=V1)}
    for x in range(V1):
        tgt[(x,)] = rng.normal(scale=1.2, size=V1)
        drf[(x,)] = tgt[(x,)] + rng.normal(scale=1.0, size=V1)
    return tgt, drf


def _softmax(z):
    e = np.exp(z - z.max())
    return e / e.sum()


def _trials(seed, n, tgt, drf, T=1.0):
    """Seeded trials: children drawn from q at the parent (the drafter), at
    temperature T."""
    rng = np.random.default_rng(seed)
    N = len(SHAPE)
    parents = np.tile(SHAPE, (n, 1))
    tokens = np.zeros((n, N), dtype=np.int64)
    tl = np.zeros((n, N, V1))
    dl = np.zeros((n, N, V1))
    for b in range(n):
        paths = {0: ()}
        for i in range(N):
            if i > 0:
                par = SHAPE[i]
                qd = _softmax(drf[paths[par]] / T)
                tokens[b, i] = rng.choice(V1, p=qd)
                paths[i] = paths[par] + (int(tokens[b, i]),)
            key = paths[i] if len(paths[i]) < 2 else None
            if key is not None:
                tl[b, i] = tgt[key]
                dl[b, i] = drf[key]
    ua = rng.random((n, N))
    ur = rng.random((n, N))
    return parents, tokens, tl, dl, ua, ur


def _first_two(out, alen):
    first = out[:, 0]
    sec = {}
    for b in range(len(alen)):
        if alen[b] >= 2:
            sec.setdefault(int(first[b]), []).append(int(out[b, 1]))
    return first, sec


def _chi2_p(samples, p):
    counts = np.bincount(samples, minlength=len(p))
    return chisquare(counts, p * counts.sum()).pvalue


def test_sampling_lossless_first_and_second_token():
    tgt, drf = _tables(21)
    parents, tokens, tl, dl, ua, ur = _trials(22, 20000, tgt, drf)
    path, alen, out, st, margin = accept_sampling(parents, tokens, tl, dl, ua, ur, 2, 1.0)
    assert (st == 0).all() and (alen >= 1).all() and (alen <= 3).all()
    first, sec = _first_two(out, alen)
    assert _chi2_p(first, _softmax(tgt[()])) > 1e-3
    tested = 0
    for x, s in sec.items():
        if len(s) >= 500:
            assert _chi2_p(np.array(s), _softmax(tgt[(x,)])) > 1e-3, x
            tested += 1
    assert tested >= 3


def test_sampling_planted_mistake_is_caught(monkeypatch):
    """The oracle with ``|p - q|`` in place of ``max(p - q, 0)`` must fail."""
    tgt, drf = _tables(21)
    parents, tokens, tl, dl, ua, ur = _trials(23, 20000, tgt, drf)

    class _Mutated:
        def __getattr__(self, name):
            return getattr(np, name)

        @staticmethod
        def maximum(a, b):
            return np.abs(a)

    monkeypatch.setattr(acc, "np", _Mutated())
    _, alen, out, _, _ = accept_sampling(parents, tokens, tl, dl, ua, ur, 2, 1.0)
    monkeypatch.undo()
    first, _ = _first_two(out, alen)
    assert _chi2_p(first, _softmax(tgt[()])) < 1e-3


def test_sampling_special_cases():
    V = 5
    parents = np.array([[-1, 0, 0, 1]])
    tokens = np.array([[0, 2, 3, 4]])
    logits = np.random.default_rng(0).normal(size=(1, 4, V))
    # draft == target: p/q = 1 for every child, any u <= 1 accepts the first child
    ua = np.full((1, 4), 0.999)
    ur = np.zeros((1, 4))
    path, alen, out, _, _ = accept_sampling(parents, tokens, logits, logits, ua, ur, 2)
    assert path[0].tolist() == [0, 1, 3] and alen[0] == 3
    # leaf 3 resamples from its own p with u_res = 0: first token with p > 0
    assert out[0].tolist() == [2, 4, 0]
    # a draft that puts almost no mass on a token the target likes: ratio >> 1
    tl = np.zeros((1, 4, V))
    dl = np.zeros((1, 4, V))
    dl[0, 0, 2] = -30.0
    ua = np.full((1, 4), 0.99)
    path, alen, _, _, _ = accept_sampling(parents, tokens, tl, dl, ua, ur, 2)
    assert path[0, 1] == 1


def test_trail_checker_accepts_oracle_and_rejects_others():
    tgt, drf = _tables(30)
    parents, tokens, tl, dl, ua, ur = _trials(31, 300, tgt, drf)
    path, alen, out, _, margin = accept_sampling(parents, tokens, tl, dl, ua, ur, 2, 1.0)
    wrong = 0
    for b in range(300):
        trail = path[b, :alen[b]].tolist()
        bonus = int(out[b, alen[b] - 1])
        ok, _ = check_sampling_trail(parents[b], tokens[b], tl[b], dl[b], ua[b], ur[b], trail, bonus)
        assert ok
        if margin[b] > 1e-3:
            alt = (bonus + 1) % V1
            ok2, _ = check_sampling_trail(parents[b], tokens[b], tl[b], dl[b], ua[b], ur[b], trail, alt)
            wrong += not ok2
    assert wrong > 200


def test_sampling_lossless_at_temperature_07():
    # T != 1: children drawn from softmax(draft / T), emitted tokens follow
    # softmax(target / T).
    T = 0.7
    tgt, drf = _tables(41)
    parents, tokens, tl, dl, ua, ur = _trials(42, 20000, tgt, drf, T=T)
    path, alen, out, st, margin = accept_sampling(parents, tokens, tl, dl, ua, ur, 2, T)
    first, _ = _first_two(out, alen)
    assert _chi2_p(first, _softmax(tgt[()] / T)) > 1e-3
    # ... and not softmax(target) at T = 1
    assert _chi2_p(first, _softmax(tgt[()])) < 1e-3


def test_draftless_variant_hand_example():
    # No draft distribution: q(x) = 1 for drafted tokens, a rejection zeroes p(x).
    # Root p = [0.5, 0.3, 0.2]; children 1, 2 (leaves) carry tokens 0, 1.
    parents = np.array([[-1, 0, 0]])
    tokens = np.array([[0, 0, 1]])
    tl = np.zeros((1, 3, 3))
    tl[0, 0] = np.log([0.5, 0.3, 0.2])
    tl[0, 2] = np.log([0.1, 0.2, 0.7])
    tl[0, 1] = np.log([0.2, 0.2, 0.6])
    # child 1: u = 0.6 > p(0) = 0.5 -> rejected, p -> [0, 0.6, 0.4];
    # child 2: u = 0.55 <= 0.6 -> accepted; leaf 2 draws its bonus from its
    # own p at u_res = 0.25: CDF [0.1, 0.3, 1.0] -> token 1.
    ua = np.array([[0.0, 0.6, 0.55]])
    ur = np.array([[0.9, 0.0, 0.25]])
    path, alen, out, st, _ = accept_sampling(parents, tokens, tl, None, ua, ur, 1, 1.0)
    assert path[0].tolist() == [0, 2] and alen[0] == 2 and out[0].tolist() == [1, 1]
    # both rejected (0.7 > 0.6): p -> [0, 0, 1], the bonus is token 2 whatever u_res
    ua[0, 2] = 0.7
    path, alen, out, st, _ = accept_sampling(parents, tokens, tl, None, ua, ur, 1, 1.0)
    assert path[0].tolist() == [0, -1] and alen[0] == 1 and out[0].tolist() == [2, -1]


def test_draftless_variant_lossless():
    # Deterministic distinct drafts (the root's children carry tokens 0, 1, 2,
    # as a top-3 proposal would): the first emitted token follows p exactly.
    V = 6
    rng = np.random.default_rng(51)
    z = rng.normal(scale=1.3, size=V)
    n = 20000
    parents = np.tile(np.array([-1, 0, 0, 0]), (n, 1))
    tokens = np.tile(np.array([0, 2, 0, 5]), (n, 1))
    tl = np.zeros((n, 4, V))
    tl[:, :, :] = z
    ua = rng.random((n, 4))
    ur = rng.random((n, 4))
    path, alen, out, st, _ = accept_sampling(parents, tokens, tl, None, ua, ur, 1, 1.0)
    assert (st == 0).all()
    assert _chi2_p(out[:, 0], _softmax(z)) > 1e-3
    # the same trials under the draft-distribution rule with q = p would accept
    # the first child always: a different distribution
    path2, alen2, out2, _, _ = accept_sampling(parents, tokens, tl, tl, ua, ur, 1, 1.0)
    assert (out2[:, 0] == 2).all()
