"""Pins for the KV-compaction oracle: only the accepted rows change, they hold
the tree rows named by the path, ``new_len = P + accept_len``, and capacity or
status errors leave the cache untouched."""

import numpy as np

from oracle.compact import kv_compact
from oracle.tree import GV_ERR_CAPACITY


def _case(rng, L=2, B=3, H=2, N=9, S=24, d=4):
    tK = rng.normal(size=(L, B, H, N, d))
    tV = rng.normal(size=(L, B, H, N, d))
    cK = rng.normal(size=(L, B, H, S, d))
    cV = rng.normal(size=(L, B, H, S, d))
    return tK, tV, cK, cV


def test_only_accepted_rows_change():
    rng = np.random.default_rng(0)
    tK, tV, cK, cV = _case(rng)
    path = np.array([[0, 2, 5, -1], [0, -1, -1, -1], [0, 1, 3, 8]])
    alen = np.array([3, 1, 4])
    P = np.array([4, 0, 20])
    nK, nV, new_len, st = kv_compact(tK, tV, cK, cV, path, alen, P)
    assert new_len.tolist() == [7, 1, 24] and (st == 0).all()
    for b in range(3):
        rows = set(range(P[b], P[b] + alen[b]))
        for s in range(cK.shape[3]):
            if s in rows:
                t = s - P[b]
                np.testing.assert_array_equal(nK[:, b, :, s], tK[:, b, :, path[b, t]])
                np.testing.assert_array_equal(nV[:, b, :, s], tV[:, b, :, path[b, t]])
            else:
                np.testing.assert_array_equal(nK[:, b, :, s], cK[:, b, :, s])
                np.testing.assert_array_equal(nV[:, b, :, s], cV[:, b, :, s])


def test_capacity_and_status():
    rng = np.random.default_rng(1)
    tK, tV, cK, cV = _case(rng, S=10)
    path = np.array([[0, 1, 2, -1]] * 3)
    alen = np.array([3, 3, 3])
    P = np.array([8, 7, 2])
    nK, nV, new_len, st = kv_compact(tK, tV, cK, cV, path, alen, P, seq_status=[0, 0, -2])
    assert st.tolist() == [GV_ERR_CAPACITY, 0, -2]
    assert new_len.tolist() == [8, 10, 2]
    np.testing.assert_array_equal(nK[:, 0], cK[:, 0])
    np.testing.assert_array_equal(nK[:, 2], cK[:, 2])
    np.testing.assert_array_equal(nV[:, 1, :, 7:10], tV[:, 1, :, 0:3])
