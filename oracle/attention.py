"""Oracle: tree-masked attention of the draft tokens (one layer).

Section 3 of GRIFFIN: the target model verifies all draft tokens in a single
forward pass.  In one attention layer of that pass, draft node ``i`` of
sequence ``b`` attends to

* every cached prefix row ``0 .. P_b - 1`` (keys stored already rotated), and
* every tree node ``j`` on its own root chain (bit ``j`` of ``anc[b][i]``),
  whose key is rotated at that node's position ``pos[b][j]``,

so that its output equals ordinary causal attention of the last query of the
sequence ``[prefix ; root chain of i]``.  Section 4.1 (a rejected token takes
its whole subtree with it) is what makes the ancestor set the right mask.

Readings where the paper is silent (the models are LLaMA/Mixtral-shaped):
rotate-half RoPE with frequencies ``base ** (-2j/d)``, angles formed in
float64; softmax scale ``1/sqrt(d)``; grouped-query attention with query head
``h`` reading KV head ``h // (Hq/Hkv)``; no bias, ALiBi or soft-capping.

Layouts: ``q[B][N][Hq][d]``, ``k_new, v_new[B][N][Hkv][d]`` (unrotated),
``cacheK, cacheV[B][Hkv][S_max][d]``.  Returns ``out[B][N][Hq][d]`` and the
tree scratch ``treeK`` (rotated) / ``treeV`` as ``[B][Hkv][N][d]``.
"""

import numpy as np


def rope_rotate(x, positions, base):
    """Rotate-half RoPE of ``x[..., n, heads, d]`` at ``positions[n]``.

    For ``j < d/2``: ``x'[j] = x[j] cos(a) - x[j + d/2] sin(a)`` and
    ``x'[j + d/2] = x[j + d/2] cos(a) + x[j] sin(a)`` with
    ``a = pos * base ** (-2j/d)`` computed in float64.
    """
    x = np.asarray(x, dtype=np.float64)
    d = x.shape[-1]
    half = d // 2
    j = np.arange(half, dtype=np.float64)
    theta = np.power(float(base), -2.0 * j / d)                  # [half]
    ang = np.asarray(positions, dtype=np.float64)[:, None] * theta[None, :]  # [n, half]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    lo = x[..., :half]
    hi = x[..., half:]
    out = np.empty_like(x)
    out[..., :half] = lo * c - hi * s
    out[..., half:] = hi * c + lo * s
    return out


def ancestor_list(anc_bits, n):
    """Indices ``j < n`` whose bit is set in the 64-bit ancestor word."""
    a = int(anc_bits)
    return [j for j in range(n) if (a >> j) & 1]


def tree_attention(q, k_new, v_new, cacheK, cacheV, prefix_len, pos, anc, rope_base):
    """Float64 tree attention for one layer; see the module docstring.

    For each sequence ``b`` and KV head ``g`` the scores of all draft queries
    of that head group against the prefix keys and against the ``N`` tree keys
    are formed with two matmuls; tree keys that are not on the query node's
    root chain are excluded (set to minus infinity) before the softmax, so
    every row's softmax runs over exactly the key set of the definition.
    """
    q = np.asarray(q, dtype=np.float64)
    k_new = np.asarray(k_new, dtype=np.float64)
    v_new = np.asarray(v_new, dtype=np.float64)
    B, N, Hq, d = q.shape
    Hkv = k_new.shape[2]
    G = Hq // Hkv
    scale = 1.0 / np.sqrt(d)
    out = np.zeros((B, N, Hq, d), dtype=np.float64)
    treeK = np.zeros((B, Hkv, N, d), dtype=np.float64)
    treeV = np.zeros((B, Hkv, N, d), dtype=np.float64)
    for b in range(B):
        P = int(prefix_len[b])
        qr = rope_rotate(q[b], pos[b], rope_base)        # [N][Hq][d]
        kr = rope_rotate(k_new[b], pos[b], rope_base)    # [N][Hkv][d]
        allowed = np.zeros((N, N), dtype=bool)           # allowed[i][j]: j on i's chain
        for i in range(N):
            allowed[i, ancestor_list(anc[b, i], N)] = True
        for g in range(Hkv):
            treeK[b, g] = kr[:, g, :]
            treeV[b, g] = v_new[b, :, g, :]
            Kp = np.asarray(cacheK[b, g, :P, :], dtype=np.float64)
            Vp = np.asarray(cacheV[b, g, :P, :], dtype=np.float64)
            for hl in range(G):
                h = g * G + hl
                Q = qr[:, h, :]                                   # [N][d]
                s_pre = (Q @ Kp.T) * scale                        # [N][P]
                s_tree = (Q @ kr[:, g, :].T) * scale              # [N][N]
                s_tree = np.where(allowed, s_tree, -np.inf)
                s = np.concatenate([s_pre, s_tree], axis=1)
                s = s - s.max(axis=1, keepdims=True)
                p = np.exp(s)
                p = p / p.sum(axis=1, keepdims=True)
                out[b, :, h, :] = p[:, :P] @ Vp + p[:, P:] @ v_new[b, :, g, :]
    return out, treeK, treeV
