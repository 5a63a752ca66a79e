"""Pins of the token-alignable training oracle (GRIFFIN Section 4.1, Eqs. 2-5,
and the per-step loss of the Implementation Details appendix) against closed
forms, brute force and hand-worked cases -- none of which re-types the
oracle's own formulas."""

import math

import numpy as np

from oracle.tat import alignment_mask, feature_loss, predictable_mask, tat_pass, token_loss


def test_uniform_logits_closed_forms():
    # Every logit equal: the cross-entropy is log V, and the tie rule puts
    # exactly the ids 0 .. k-1 in the top-k.
    V, k = 37, 3
    logits = np.full((V, V), 0.25)
    tokens = np.arange(V)
    np.testing.assert_allclose(token_loss(logits, tokens), np.full(V, math.log(V)), rtol=1e-13)
    np.testing.assert_array_equal(predictable_mask(logits, tokens, k), (tokens < k).astype(np.uint8))


def test_two_token_cross_entropy():
    for a, b in [(0.0, 0.0), (1.5, -2.0), (-3.0, 4.0), (30.0, -30.0)]:
        lg = np.array([[a, b], [a, b]])
        ce = token_loss(lg, np.array([0, 1]))
        assert abs(ce[0] - math.log1p(math.exp(b - a))) < 1e-12
        assert abs(ce[1] - math.log1p(math.exp(a - b))) < 1e-12


def test_cross_entropy_is_minus_log_probability():
    # exp(-CE) against the softmax probability formed another way:
    # p(x) = 1 / sum_v exp(l_v - l_x).
    rng = np.random.default_rng(3)
    lg = rng.normal(size=(20, 50)) * 3
    tok = rng.integers(0, 50, size=20)
    ce = token_loss(lg, tok)
    p = np.array([1.0 / sum(math.exp(lg[r, v] - lg[r, tok[r]]) for v in range(50)) for r in range(20)])
    np.testing.assert_allclose(np.exp(-ce), p, rtol=1e-12)
    # shifting a row by a constant changes nothing
    np.testing.assert_allclose(token_loss(lg + 7.25, tok), ce, rtol=1e-12)


def test_topk_membership_brute_force_with_ties():
    # Integer logits over a small vocabulary: many ties.  The top-k list is
    # built by sorting (value descending, id ascending).
    rng = np.random.default_rng(11)
    for k in (1, 2, 3, 5):
        lg = rng.integers(-3, 4, size=(200, 12)).astype(np.float64)
        tok = rng.integers(0, 12, size=200)
        got = predictable_mask(lg, tok, k)
        for r in range(200):
            order = sorted(range(12), key=lambda v: (-lg[r, v], v))
            assert got[r] == (1 if tok[r] in order[:k] else 0), (k, r)


def test_feature_loss_constant_vectors():
    H = 64
    fd = np.full((3, H), -0.75)
    ft = np.zeros((3, H))
    np.testing.assert_allclose(feature_loss(fd, ft), np.full(3, H * 0.75), rtol=1e-13)
    ft2 = np.full((3, H), 0.25)
    np.testing.assert_allclose(feature_loss(fd, ft2), np.full(3, H * 1.0), rtol=1e-13)


def test_alignment_mask_hand_example():
    # n = 3: m_t = mbar1[t-2] * mbar2[t-1] for t >= 2, worked by hand.
    mb1 = np.array([[1, 1, 0, 1, 1, 1]], dtype=np.uint8)
    mb2 = np.array([[1, 0, 1, 1, 1, 1]], dtype=np.uint8)
    m = alignment_mask([mb1, mb2], 3, 1, 6)
    np.testing.assert_array_equal(m[0], [0, 0, 0, 1, 0, 1])
    # n = 2: the pass-1 mask shifted by one position
    m2 = alignment_mask([mb1], 2, 1, 6)
    np.testing.assert_array_equal(m2[0], [0, 1, 1, 0, 1, 1])


def _random_pass(seed, B=2, T=9, V=40, H=16):
    rng = np.random.default_rng(seed)
    lg = rng.normal(size=(B, T, V))
    tok = rng.integers(0, V, size=(B, T))
    fd = rng.normal(size=(B, T, H))
    ft = rng.normal(size=(B, T, H))
    return rng, lg, tok, fd, ft


def test_first_pass_is_the_plain_mean():
    # Eq. 2: no masking in the first pass, so the pass loss is the mean of
    # the per-step losses, and ell = CE + 0.1 * L1 with the default weights.
    _, lg, tok, fd, ft = _random_pass(5)
    out = tat_pass(lg, tok, fd, ft, k=3, n=1)
    assert (out["mask"] == 1).all()
    ce = np.array([[-math.log(math.exp(lg[b, t, tok[b, t]]) / np.exp(lg[b, t]).sum())
                    for t in range(9)] for b in range(2)])
    l1 = np.abs(fd - ft).sum(axis=2)
    np.testing.assert_allclose(out["ell"], ce + 0.1 * l1, rtol=1e-12)
    np.testing.assert_allclose(out["seq_loss"], out["ell"].mean(axis=1), rtol=1e-12)


def test_masked_positions_do_not_count():
    rng, lg, tok, fd, ft = _random_pass(8)
    prev = [rng.integers(0, 2, size=(2, 9)).astype(np.uint8) for _ in range(2)]
    base = tat_pass(lg, tok, fd, ft, k=3, n=3, mbar_prev=prev)
    m = base["mask"]
    assert m.sum() > 0 and (m == 0).sum() > 0
    # A different loss at a masked position leaves the pass loss unchanged ...
    lg2 = lg.copy()
    b0, t0 = np.argwhere(m == 0)[0]
    lg2[b0, t0] += rng.normal(size=lg.shape[2]) * 5
    same = tat_pass(lg2, tok, fd, ft, k=3, n=3, mbar_prev=prev)
    np.testing.assert_allclose(same["seq_loss"], base["seq_loss"], rtol=1e-13)
    # ... and at an aligned position it changes it.
    lg3 = lg.copy()
    b1, t1 = np.argwhere(m == 1)[0]
    lg3[b1, t1, tok[b1, t1]] -= 3.0
    diff = tat_pass(lg3, tok, fd, ft, k=3, n=3, mbar_prev=prev)
    assert diff["seq_loss"][b1] > base["seq_loss"][b1]
    # the chain cannot start before the sequence
    assert (m[:, :2] == 0).all()


def test_sequence_without_aligned_tokens_has_zero_loss():
    _, lg, tok, fd, ft = _random_pass(9)
    prev = [np.zeros((2, 9), dtype=np.uint8)]
    out = tat_pass(lg, tok, fd, ft, k=3, n=2, mbar_prev=prev)
    assert (out["mask"] == 0).all()
    np.testing.assert_array_equal(out["seq_loss"], [0.0, 0.0])


def test_pass_loss_is_the_mean_over_aligned_steps_hand_example():
    # Eq. 5 by hand.  One sequence of T = 5 steps, V = 4 uniform logits (each
    # step's cross-entropy is exactly log 4) and features differing by a
    # constant c_t in each of H = 2 components (L1 distance 2 |c_t|), so with
    # lam_feat = 0.1 the per-step losses are log 4 + (1.0, 0.2, 0.4, 1.4, 0.6).
    # Pass n = 2 with the first pass's predictable mask (1, 1, 0, 1, 0): the
    # alignment mask is (0, 1, 1, 0, 1) (step t looks at step t - 1; step 0
    # has no chain), and the pass loss is the mean over those three steps,
    # log 4 + (0.2 + 0.4 + 0.6) / 3 = log 4 + 0.4.
    T, V, H = 5, 4, 2
    logits = np.zeros((1, T, V))
    tokens = np.array([[0, 1, 2, 3, 0]])
    c = np.array([5.0, 1.0, 2.0, 7.0, 3.0])
    ft = np.zeros((1, T, H))
    fd = np.repeat(c[None, :, None], H, axis=2)
    prev = [np.array([[1, 1, 0, 1, 0]], dtype=np.uint8)]
    out = tat_pass(logits, tokens, fd, ft, k=2, n=2, mbar_prev=prev)
    np.testing.assert_array_equal(out["mask"], [[0, 1, 1, 0, 1]])
    np.testing.assert_allclose(out["ell"][0], math.log(4) + np.array([1.0, 0.2, 0.4, 1.4, 0.6]), rtol=1e-13)
    assert abs(out["seq_loss"][0] - (math.log(4) + 0.4)) < 1e-13
