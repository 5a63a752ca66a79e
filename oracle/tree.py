"""Oracle: positions, depths and ancestor sets of a draft tree.

The draft tree is the dynamic tree of GRIFFIN Appendix C ("Draft Tree
Structure": 60 draft tokens, depth 6, following EAGLE-2).  The paper does not
write down an encoding; this oracle fixes the one the whole library uses:

* ``parents[b][i]`` is the parent of node ``i`` of sequence ``b``; node 0 is
  the root (the last committed token, whose K/V is not cached yet) and has
  ``parents[b][0] == -1``; every other node has ``0 <= parents[b][i] < i``
  (topological order), so ancestors always have smaller indices.
* ``depth[i]`` is the number of edges from the root, ``pos[i] = P_b + depth[i]``
  is the token position used for RoPE, and ``anc[i]`` is the 64-bit set of
  ancestor-or-self nodes: bit ``j`` is set iff ``j`` lies on the root-to-``i``
  chain.  Section 4.1 states that rejecting a token discards every later token
  of its draft sequence, so ``anc`` is exactly the set that decides both the
  attention mask and acceptance.

Computed by walking each node's parent chain (the definition), not by a
recurrence over parents.
"""

import numpy as np

GV_OK = 0
GV_ERR_INVALID_TREE = -2
GV_ERR_CAPACITY = -3

MAX_NODES = 64


def tree_is_valid(parents_row):
    """Topological-order rule: root first with parent -1, others point back."""
    n = len(parents_row)
    if n < 1 or n > MAX_NODES:
        return False
    if int(parents_row[0]) != -1:
        return False
    for i in range(1, n):
        p = int(parents_row[i])
        if p < 0 or p >= i:
            return False
    return True


def tree_build(parents, prefix_len):
    """Return ``(depth, pos, anc, status)`` for ``parents[B][N]``.

    ``anc`` is returned as ``uint64[B][N]``.  For a sequence whose parent array
    breaks the topological-order rule the status is ``GV_ERR_INVALID_TREE``
    and the outputs are the safe defaults ``depth = 0``, ``pos = P_b``,
    ``anc[i] = 1 << i`` (each node sees only itself).
    """
    parents = np.asarray(parents, dtype=np.int64)
    prefix_len = np.asarray(prefix_len, dtype=np.int64)
    B, N = parents.shape
    depth = np.zeros((B, N), dtype=np.int32)
    pos = np.zeros((B, N), dtype=np.int32)
    anc = np.zeros((B, N), dtype=np.uint64)
    status = np.zeros(B, dtype=np.int32)
    for b in range(B):
        if not tree_is_valid(parents[b]):
            status[b] = GV_ERR_INVALID_TREE
            for i in range(N):
                depth[b, i] = 0
                pos[b, i] = prefix_len[b]
                anc[b, i] = np.uint64(1) << np.uint64(i)
            continue
        for i in range(N):
            bits = 0
            edges = 0
            j = i
            while j != -1:
                bits |= 1 << j
                j = int(parents[b, j])
                if j != -1:
                    edges += 1
            depth[b, i] = edges
            pos[b, i] = prefix_len[b] + edges
            anc[b, i] = np.uint64(bits)
    return depth, pos, anc, status


def chain(parents_row, i):
    """Root-to-``i`` node list, by walking parents (used by accept and tests)."""
    out = []
    j = int(i)
    while j != -1:
        out.append(j)
        j = int(parents_row[j])
    return out[::-1]
