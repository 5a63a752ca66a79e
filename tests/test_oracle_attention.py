"""Pins for the tree-attention oracle.

Checks against things other than the oracle itself:

* RoPE against the complex-number form ``(a + ib) * exp(i * pos * theta)``
  and against the relative-position identity ``<R(m)q, R(n)k>`` depending
  only on ``m - n``;
* path-causal equivalence: node ``i``'s output equals textbook causal
  attention (``torch.nn.functional.scaled_dot_product_attention`` in float64)
  of the last query of ``[prefix ; root chain of i]``, for every node of random
  small trees;
* a chain tree reduces to ordinary causal attention over the whole sequence;
* one node (N = 1) is single-query decode attention; an empty prefix makes
  the root's output its own value row;
* grouped-query attention equals multi-head attention with each KV head
  repeated for its query heads.
"""

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle.attention import rope_rotate, tree_attention
from oracle.tree import tree_build, chain
from paper_2502_11018_gb300 import inputs


def rope_complex(x, positions, base):
    """RoPE as complex multiplication of (x[j] + i x[j + d/2])."""
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    theta = np.array([base ** (-2.0 * j / d) for j in range(half)])
    z = x[..., :half] + 1j * x[..., half:]
    rot = np.exp(1j * np.asarray(positions, dtype=np.float64)[:, None] * theta[None, :])
    z = z * rot[:, None, :]
    return np.concatenate([z.real, z.imag], axis=-1)


@pytest.mark.parametrize("base", [10000.0, 500000.0, 1e6])
def test_rope_matches_complex_form(base):
    rng = np.random.default_rng(3)
    x = rng.normal(size=(7, 3, 16))
    pos = np.array([0, 1, 5, 100, 4097, 16383, 20000])
    np.testing.assert_allclose(rope_rotate(x, pos, base), rope_complex(x, pos, base),
                               rtol=0, atol=1e-12)


def test_rope_relative_position():
    rng = np.random.default_rng(4)
    q = rng.normal(size=(1, 1, 32))
    k = rng.normal(size=(1, 1, 32))
    ref = None
    for m in [3, 50, 1000, 9000]:
        n = m - 3
        s = float((rope_rotate(q, [m], 1e4) * rope_rotate(k, [n], 1e4)).sum())
        if ref is None:
            ref = s
        assert abs(s - ref) < 1e-9


def sdpa_last_query(qvec, keys, vals):
    q = torch.from_numpy(qvec)[None, None, None, :]
    k = torch.from_numpy(keys)[None, None]
    v = torch.from_numpy(vals)[None, None]
    return F.scaled_dot_product_attention(q, k, v)[0, 0, 0].numpy()


def _random_case(rng, B, N, Hq, Hkv, d, Pmax, D):
    parents = np.zeros((B, N), dtype=np.int32)
    for b in range(B):
        if N == 1:
            parents[b] = [-1]
        else:
            parents[b], _ = inputs.make_tree(rng, N, min(D, N - 1), 4, 100)
    P = rng.integers(0, Pmax + 1, size=B)
    S = Pmax + 2
    q = rng.normal(size=(B, N, Hq, d))
    k = rng.normal(size=(B, N, Hkv, d))
    v = rng.normal(size=(B, N, Hkv, d))
    cK = rng.normal(size=(B, Hkv, S, d))
    cV = rng.normal(size=(B, Hkv, S, d))
    return parents, P, q, k, v, cK, cV


@pytest.mark.parametrize("seed,N,Hq,Hkv,d", [
    (0, 12, 1, 1, 16), (1, 9, 2, 2, 8), (2, 12, 4, 2, 16), (3, 7, 4, 1, 8),
    (4, 1, 2, 1, 8), (5, 12, 4, 4, 4),
])
def test_path_causal_equivalence(seed, N, Hq, Hkv, d):
    rng = np.random.default_rng(seed)
    B = 2
    parents, P, q, k, v, cK, cV = _random_case(rng, B, N, Hq, Hkv, d, 16, 4)
    depth, pos, anc, st = tree_build(parents, P)
    base = 10000.0
    out, treeK, treeV = tree_attention(q, k, v, cK, cV, P, pos, anc, base)
    G = Hq // Hkv
    for b in range(B):
        for i in range(N):
            path = chain(parents[b], i)
            positions = [P[b] + t for t in range(len(path))]
            for h in range(Hq):
                g = h // G
                kp = rope_complex(k[b, path, g][:, None, :], positions, base)[:, 0]
                keys = np.concatenate([cK[b, g, :P[b]], kp])
                vals = np.concatenate([cV[b, g, :P[b]], v[b, path, g]])
                qv = rope_complex(q[b, i, h][None, None], [P[b] + len(path) - 1], base)[0, 0]
                ref = sdpa_last_query(qv, keys, vals)
                np.testing.assert_allclose(out[b, i, h], ref, rtol=0, atol=1e-12)
        # tree scratch holds the rotated keys at each node's position and raw values
        for g in range(Hkv):
            np.testing.assert_allclose(treeK[b, g], rope_complex(k[b, :, g][:, None], pos[b], base)[:, 0],
                                       atol=1e-12)
            np.testing.assert_array_equal(treeV[b, g], v[b, :, g])


def test_chain_tree_is_causal_attention():
    rng = np.random.default_rng(11)
    N, H, d, P = 10, 2, 16, 13
    parents = np.arange(-1, N - 1, dtype=np.int32)[None]
    depth, pos, anc, _ = tree_build(parents, [P])
    # Prefix keys/values plus queries for every position of the full sequence.
    qs = rng.normal(size=(P + N, H, d))
    ks = rng.normal(size=(P + N, H, d))
    vs = rng.normal(size=(P + N, H, d))
    allpos = np.arange(P + N)
    qr = rope_complex(qs, allpos, 1e4)
    kr = rope_complex(ks, allpos, 1e4)
    cK = np.zeros((1, H, P + N, d))
    cV = np.zeros((1, H, P + N, d))
    cK[0, :, :P] = kr[:P].transpose(1, 0, 2)
    cV[0, :, :P] = vs[:P].transpose(1, 0, 2)
    out, _, _ = tree_attention(qs[None, P:], ks[None, P:], vs[None, P:], cK, cV, [P], pos, anc, 1e4)
    ref = F.scaled_dot_product_attention(
        torch.from_numpy(qr.transpose(1, 0, 2))[None], torch.from_numpy(kr.transpose(1, 0, 2))[None],
        torch.from_numpy(vs.transpose(1, 0, 2))[None], is_causal=True)[0].numpy()  # [H][P+N][d]
    np.testing.assert_allclose(out[0], ref[:, P:].transpose(1, 0, 2), atol=1e-12)


def test_single_node_is_decode_attention():
    rng = np.random.default_rng(12)
    P, H, d = 40, 3, 8
    q = rng.normal(size=(1, 1, H, d))
    k = rng.normal(size=(1, 1, H, d))
    v = rng.normal(size=(1, 1, H, d))
    cK = rng.normal(size=(1, H, P + 1, d))
    cV = rng.normal(size=(1, H, P + 1, d))
    depth, pos, anc, _ = tree_build(np.array([[-1]]), [P])
    out, _, _ = tree_attention(q, k, v, cK, cV, [P], pos, anc, 1e4)
    for h in range(H):
        keys = np.concatenate([cK[0, h, :P], rope_complex(k[0, :, h][:, None], [P], 1e4)[:, 0]])
        vals = np.concatenate([cV[0, h, :P], v[0, :, h]])
        qv = rope_complex(q[0, :, h][:, None], [P], 1e4)[0, 0]
        np.testing.assert_allclose(out[0, 0, h], sdpa_last_query(qv, keys, vals), atol=1e-12)


def test_empty_prefix_root_sees_only_itself():
    rng = np.random.default_rng(13)
    N, H, d = 6, 2, 8
    parents, _ = inputs.make_tree(rng, N, 3, 3, 50)
    depth, pos, anc, _ = tree_build(parents[None], [0])
    q = rng.normal(size=(1, N, H, d))
    k = rng.normal(size=(1, N, H, d))
    v = rng.normal(size=(1, N, H, d))
    out, _, _ = tree_attention(q, k, v, np.zeros((1, H, 4, d)), np.zeros((1, H, 4, d)),
                               [0], pos, anc, 1e4)
    np.testing.assert_allclose(out[0, 0], v[0, 0], atol=1e-15)


def test_gqa_equals_repeated_mha():
    rng = np.random.default_rng(14)
    B, N, Hq, Hkv, d = 2, 9, 8, 2, 8
    parents, P, q, k, v, cK, cV = _random_case(rng, B, N, Hq, Hkv, d, 20, 4)
    depth, pos, anc, _ = tree_build(parents, P)
    out, _, _ = tree_attention(q, k, v, cK, cV, P, pos, anc, 5e5)
    G = Hq // Hkv
    rep = lambda x, ax: np.repeat(x, G, axis=ax)  # noqa: E731  kv head g -> query heads gG..gG+G-1
    out_mha, _, _ = tree_attention(q, rep(k, 2), rep(v, 2), rep(cK, 1), rep(cV, 1), P, pos, anc, 5e5)
    np.testing.assert_allclose(out, out_mha, atol=1e-13)
