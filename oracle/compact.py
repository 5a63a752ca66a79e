"""Oracle: commit the accepted tokens' K/V into the contiguous cache.

Section 4.1 of GRIFFIN: a rejected draft token is discarded together with all
later tokens of its draft sequence, so only the accepted root chain survives
the verify pass.  Its keys and values (computed during verification and held
in a separate tree scratch) are appended to the cache; nothing else is
written.  For every layer ``l``, sequence ``b``, KV head ``h`` and
``t < accept_len[b]``::

    cache[l][b][h][P_b + t][:] = tree[l][b][h][path[b][t]][:]

and ``new_len[b] = P_b + accept_len[b]``.  Readings: the root (node 0) is the
last committed token whose K/V was not cached yet, so it is committed first;
a sequence whose status is already non-zero is left untouched
(``new_len = P_b``); a sequence whose ``P_b + accept_len`` exceeds ``S_max``
gets ``GV_ERR_CAPACITY`` and is left untouched.

Layouts: ``treeK, treeV[L][B][Hkv][N][d]``, ``cacheK, cacheV[L][B][Hkv][S_max][d]``.
Works on copies; returns ``(cacheK, cacheV, new_len, status)``.
"""

import numpy as np

from .tree import GV_OK, GV_ERR_CAPACITY


def kv_compact(treeK, treeV, cacheK, cacheV, path, accept_len, prefix_len, seq_status=None):
    cacheK = np.array(cacheK, copy=True)
    cacheV = np.array(cacheV, copy=True)
    L, B, Hkv, S_max, d = cacheK.shape
    status = np.zeros(B, dtype=np.int32) if seq_status is None else np.array(seq_status, dtype=np.int32)
    new_len = np.zeros(B, dtype=np.int32)
    for b in range(B):
        P = int(prefix_len[b])
        n = int(accept_len[b])
        new_len[b] = P
        if status[b] != GV_OK:
            continue
        if P + n > S_max:
            status[b] = GV_ERR_CAPACITY
            continue
        for layer in range(L):
            for h in range(Hkv):
                for t in range(n):
                    src = int(path[b][t])
                    cacheK[layer, b, h, P + t, :] = treeK[layer, b, h, src, :]
                    cacheV[layer, b, h, P + t, :] = treeV[layer, b, h, src, :]
        new_len[b] = P + n
    return cacheK, cacheV, new_len, status
