"""Pins of the whole-step composition (``oracle.verify_step``, Section 3: one
target forward over all draft tokens, then acceptance and the cache commit).

Each stage oracle is pinned on its own; these pins check how the step wires
the stages together (which layer's cache meets which queries, the positions
RoPE is given, the offsets of the commit), against facts that come from
outside the oracle: the generator's planted greedy choices (each row's argmax
by a wide margin by construction), a brute-force search for the accepted
chain, textbook causal attention (torch's scaled_dot_product_attention over
the prefix and the node's root chain, RoPE as a complex product) for sampled
nodes of every layer and sequence, and the committed cache rows against the
rotated tree keys and the values of the accepted chain.
"""

import numpy as np
import pytest

import oracle
from paper_2502_11018_gb300 import inputs
from test_oracle_accept import _search
from test_oracle_attention import rope_complex, sdpa_last_query


def _chain(parents_row, i):
    out = [int(i)]
    while parents_row[out[-1]] != -1:
        out.append(int(parents_row[out[-1]]))
    return out[::-1]


def _f64(t):
    return t.detach().cpu().double().numpy()


@pytest.mark.parametrize("name,over,seed", [
    # GQA, two sequences with ragged prefixes (one shorter than a block), three
    # layers; the seed accepts chains of 4 and 3 nodes
    ("llama3_8b", dict(B=2, L=3, H=64, Hq=4, Hkv=2, d=16, V=300, P=(37, 130), N=12, D=4, branch=3,
                       S_max=160), 27),
    # MHA, one sequence with an empty prefix, two layers; a chain of 3 nodes
    ("llama2_7b", dict(L=2, H=48, Hq=3, Hkv=3, d=8, V=200, P=(0,), N=9, D=3, branch=2, S_max=16), 12),
])
def test_step_composition(name, over, seed):
    cfg = inputs.config(name, **over)
    inp = inputs.make_step_inputs(cfg, seed)
    res = oracle.verify_step(inp)
    B, L, N, Hq, Hkv, d = cfg["B"], cfg["L"], cfg["N"], cfg["Hq"], cfg["Hkv"], cfg["d"]
    G = Hq // Hkv
    parents = inp.parents.numpy()
    tokens = inp.tokens.numpy()
    P = inp.prefix_len.numpy()
    planted = inp.planted.numpy()

    # Greedy choices are the planted tokens; the accepted chain is the deepest
    # matching one found by search (longer than the root alone); new lengths
    # count it.
    assert (res["accept_len"] >= 3).all()
    np.testing.assert_array_equal(res["choice"].reshape(B, N), planted)
    for b in range(B):
        best = _search(parents[b], tokens[b], planted[b])
        ch = _chain(parents[b], best)
        assert res["accept_len"][b] == len(ch)
        assert res["path"][b, :len(ch)].tolist() == ch
        assert res["out_tokens"][b, :len(ch)].tolist() == [int(tokens[b, j]) for j in ch[1:]] + [int(planted[b, best])]
        assert res["new_len"][b] == P[b] + len(ch)

    # Attention of sampled nodes of every layer and sequence: the last query
    # of [prefix ; root chain] under causal attention.
    for l in range(L):
        q, kn, vn = _f64(inp.q[l]), _f64(inp.k_new[l]), _f64(inp.v_new[l])
        cK, cV = _f64(inp.cacheK[l]), _f64(inp.cacheV[l])
        for b in range(B):
            for i in sorted({0, N // 2, N - 1}):
                ch = _chain(parents[b], i)
                pos = P[b] + np.arange(len(ch))          # a node's position: the prefix plus its depth
                for h in range(Hq):
                    g = h // G
                    keys = np.concatenate([cK[b, g, :P[b]], rope_complex(kn[b, ch, g][:, None, :], pos, cfg["rope_base"])[:, 0]])
                    vals = np.concatenate([cV[b, g, :P[b]], vn[b, ch, g]])
                    qv = rope_complex(q[b, i, h][None, None, :], pos[-1:], cfg["rope_base"])[0, 0]
                    ref = sdpa_last_query(qv, keys, vals)
                    np.testing.assert_allclose(res["attn_out"][l][b, i, h], ref, rtol=1e-9, atol=1e-12)

    # The commit: rows P .. P + accept_len - 1 of every layer's cache hold the
    # accepted chain's rotated keys and its values; every other row is unchanged.
    for l in range(L):
        kn, vn = _f64(inp.k_new[l]), _f64(inp.v_new[l])
        cK0, cV0 = _f64(inp.cacheK[l]), _f64(inp.cacheV[l])
        for b in range(B):
            n = int(res["accept_len"][b])
            ch = res["path"][b, :n].tolist()
            pos = P[b] + np.arange(n)
            for g in range(Hkv):
                rk = rope_complex(kn[b, ch, g][:, None, :], pos, cfg["rope_base"])[:, 0]
                np.testing.assert_allclose(res["cacheK"][l, b, g, P[b]:P[b] + n], rk, rtol=1e-9, atol=1e-12)
                np.testing.assert_array_equal(res["cacheV"][l, b, g, P[b]:P[b] + n], vn[b, ch, g])
                keep = np.ones(cK0.shape[2], dtype=bool)
                keep[P[b]:P[b] + n] = False
                np.testing.assert_array_equal(res["cacheK"][l, b, g, keep], cK0[b, g, keep])
                np.testing.assert_array_equal(res["cacheV"][l, b, g, keep], cV0[b, g, keep])
