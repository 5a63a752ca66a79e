"""Losslessness pin for the composed oracle (Section 5: greedy speculative
decoding reproduces greedy decoding token for token).

A tiny random-init target model (token embedding, one attention layer with
RoPE, LM head) decodes greedily in two ways:

* plain autoregressive decoding, one token per step, with textbook causal
  attention (``scaled_dot_product_attention`` in float64) and RoPE written as
  complex multiplication: this part uses nothing from ``oracle/``;
* draft-tree speculative decoding through the oracle: ``tree_build``,
  ``tree_attention``, ``lmhead_logits`` + ``select_argmax``,
  ``accept_greedy`` and ``kv_compact``, with draft trees whose tokens are
  partly planted from the reference continuation so that accepted lengths
  range from 1 to D + 1.

Both must emit the same tokens.  Seeds whose reference decode has a top-1 /
top-2 logit gap below 1e-9 are skipped (a tie would make "greedy" ambiguous).
"""

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle
from paper_2502_11018_gb300 import inputs

V, H, HQ, HKV, DH = 48, 32, 4, 2, 8
BASE = 10000.0


class TinyModel:
    def __init__(self, seed):
        rng = np.random.default_rng(seed)
        self.E = rng.normal(size=(V, H))
        self.Wq = rng.normal(size=(H, HQ * DH)) / np.sqrt(H)
        self.Wk = rng.normal(size=(H, HKV * DH)) / np.sqrt(H)
        self.Wv = rng.normal(size=(H, HKV * DH)) / np.sqrt(H)
        self.Wlm = rng.normal(size=(V, HQ * DH))

    def qkv(self, toks):
        x = self.E[np.asarray(toks)]
        return (x @ self.Wq).reshape(-1, HQ, DH), (x @ self.Wk).reshape(-1, HKV, DH), \
            (x @ self.Wv).reshape(-1, HKV, DH)


def rope_c(x, positions):
    half = DH // 2
    theta = BASE ** (-2.0 * np.arange(half) / DH)
    z = x[..., :half] + 1j * x[..., half:]
    z = z * np.exp(1j * np.asarray(positions, dtype=np.float64)[:, None, None] * theta[None, None, :])
    return np.concatenate([z.real, z.imag], axis=-1)


def ar_decode(model, prompt, steps):
    """Plain greedy decoding, recomputing causal attention over the sequence."""
    seq = list(prompt)
    margins = []
    for _ in range(steps):
        q, k, v = model.qkv(seq)
        pos = np.arange(len(seq))
        q, k = rope_c(q, pos), rope_c(k, pos)
        rep = HQ // HKV
        k = np.repeat(k, rep, axis=1)
        v = np.repeat(v, rep, axis=1)
        o = F.scaled_dot_product_attention(torch.from_numpy(q.transpose(1, 0, 2)),
                                           torch.from_numpy(k.transpose(1, 0, 2)),
                                           torch.from_numpy(v.transpose(1, 0, 2)),
                                           is_causal=True).numpy()[:, -1, :]   # [HQ][DH]
        logits = model.Wlm @ o.reshape(-1)
        srt = np.sort(logits)
        margins.append(srt[-1] - srt[-2])
        seq.append(int(np.argmax(logits)))
    return seq[len(prompt):], min(margins)


def spec_decode(model, prompt, steps, ref, rng, N=12, D=4):
    S_max = len(prompt) + steps + N + 8
    cK = np.zeros((1, 1, HKV, S_max, DH))
    cV = np.zeros((1, 1, HKV, S_max, DH))
    # Commit the prompt except its last token (the first root).
    P = len(prompt) - 1
    _, k, v = model.qkv(prompt[:-1])
    cK[0, 0, :, :P] = rope_c(k, np.arange(P)).transpose(1, 0, 2)
    cV[0, 0, :, :P] = v.transpose(1, 0, 2)
    root = prompt[-1]
    out = []
    lens = []
    while len(out) < steps:
        parents, tokens = inputs.make_tree(rng, N, D, 3, V)
        tokens[0] = root
        # Plant: along the reference continuation, the first child of an
        # on-path node carries the true next token with probability 0.6.
        done = len(out)
        kids = inputs.children_of(parents)
        onpath = {0: 0}
        for u in range(N):
            if u not in onpath or not kids[u]:
                continue
            t = done + onpath[u]
            if t < len(ref) and rng.random() < 0.6:
                want = ref[t]
                for c in kids[u][1:]:
                    if tokens[c] == want:
                        tokens[c] = (want + 1 + rng.integers(V - 1)) % V
                        while tokens[c] in [tokens[x] for x in kids[u] if x != c] or tokens[c] == want:
                            tokens[c] = (tokens[c] + 1) % V
                tokens[kids[u][0]] = want
                onpath[kids[u][0]] = onpath[u] + 1
        depth, pos, anc, st = oracle.tree_build(parents[None], [P])
        q, k, v = model.qkv(tokens)
        o, tK, tV = oracle.tree_attention(q[None], k[None], v[None], cK[0], cV[0], [P], pos, anc, BASE)
        logits = oracle.lmhead_logits(o[0].reshape(N, -1), model.Wlm)
        choice, _ = oracle.select_argmax(logits)
        path, alen, toks, st = oracle.accept_greedy(parents[None], tokens[None], choice, D)
        cK, cV, new_len, st = oracle.kv_compact(tK[None], tV[None], cK, cV, path, alen, [P])
        n = int(alen[0])
        out.extend(int(x) for x in toks[0, :n])
        lens.append(n)
        P = int(new_len[0])
        root = int(toks[0, n - 1])
    return out[:steps], lens


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_greedy_speculative_equals_autoregressive(seed):
    model = TinyModel(100 + seed)
    rng = np.random.default_rng(seed)
    prompt = [int(x) for x in rng.integers(0, V, size=9)]
    steps = 200
    ref, margin = ar_decode(model, prompt, steps)
    if margin < 1e-9:
        pytest.skip("tie in the reference decode")
    got, lens = spec_decode(model, prompt, steps, ref, rng)
    assert got == ref
    assert min(lens) >= 1 and max(lens) <= 5
    assert max(lens) >= 3          # planting produced multi-token acceptances
