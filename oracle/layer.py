"""Oracle: the target model's decoder layers around the tree attention.

TEST INFRASTRUCTURE ONLY (see the package docstring).

GRIFFIN Section 3: the target model verifies every draft token in one forward
pass.  The verify step's hot path (tree attention, LM head, acceptance,
compaction) sits inside that forward; this module is the rest of it, for
LLaMA-style targets (the paper's LLaMA-2/3, Vicuna, Qwen2 and the attention
of Mixtral): per layer, with the hidden states ``h[R][H]`` of the R = B * N
tree nodes,

    x  = RMSNorm(h) * w_attn
    q, k, v = x Wq^T, x Wk^T, x Wv^T
    h  = h + TreeAttention(q, k, v) Wo^T
    x  = RMSNorm(h) * w_mlp
    h  = h + (silu(x Wg^T) * (x Wu^T)) Wd^T

and after the last layer ``RMSNorm(h) * w_final`` feeds the LM head.
``RMSNorm(h) = h / sqrt(mean(h^2) + eps)``, ``silu(z) = z / (1 + exp(-z))``.

Readings (the paper does not restate the target architecture): the public
LLaMA layer order above; no biases; eps = 1e-5; the tree attention is
``oracle.attention.tree_attention`` (RoPE inside it, rotate-half); weights are
stored ``W[out][in]`` as the LM head's are.

Every function works in float64, with single numpy matmuls as steps.
"""

import numpy as np

from .attention import tree_attention


def rmsnorm(x, w, eps=1e-5):
    """``x / sqrt(mean(x^2) + eps) * w`` per row.  x [R][H], w [H]."""
    x = np.asarray(x, dtype=np.float64)
    ms = (x * x).mean(axis=1, keepdims=True)
    return x / np.sqrt(ms + eps) * np.asarray(w, dtype=np.float64)


def linear(x, W):
    """``x W^T``: x [R][K], W [N][K] -> [R][N]."""
    return np.asarray(x, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T


def silu(z):
    z = np.asarray(z, dtype=np.float64)
    return z / (1.0 + np.exp(-z))


def swiglu(x, Wg, Wu):
    """``silu(x Wg^T) * (x Wu^T)``."""
    return silu(linear(x, Wg)) * linear(x, Wu)


def decoder_layer(h, w, cacheK, cacheV, P, pos, anc, rope_base, B, N, Hq, Hkv, d, eps=1e-5):
    """One layer over the tree's hidden states.  h [B*N][H]; ``w`` holds
    attn_norm [H], Wq [Hq*d][H], Wk/Wv [Hkv*d][H], Wo [H][Hq*d], mlp_norm [H],
    Wg/Wu [F][H], Wd [H][F]; caches [B][Hkv][S][d].  Returns (h', treeK,
    treeV) with the layer's rotated tree keys and values."""
    h = np.asarray(h, dtype=np.float64)
    x = rmsnorm(h, w["attn_norm"], eps)
    q = linear(x, w["Wq"]).reshape(B, N, Hq, d)
    k = linear(x, w["Wk"]).reshape(B, N, Hkv, d)
    v = linear(x, w["Wv"]).reshape(B, N, Hkv, d)
    o, tK, tV = tree_attention(q, k, v, cacheK, cacheV, P, pos, anc, rope_base)
    h = h + linear(o.reshape(B * N, Hq * d), w["Wo"])
    x = rmsnorm(h, w["mlp_norm"], eps)
    h = h + linear(swiglu(x, w["Wg"], w["Wu"]), w["Wd"])
    return h, tK, tV
