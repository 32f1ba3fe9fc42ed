"""Tree-verification attention oracle.  TEST INFRASTRUCTURE ONLY.

The packed tree is verified in one target forward (Sec. 4.2): every drafted
node is a query whose attention may see the verified prefix, itself and its
root-to-node ancestors (the tree mask of Appendix A, "Tensor
implementation").  This module restates one attention layer of that forward
in float64, for grouped-query heads:

    for request r, node i < n_nodes[r], query head h (KV head h // G):
        allowed keys  = prefix slots 0 .. T-1, and tree slots T + m for m on
                        the path from i to the root (the ancestor-or-self
                        mask row of i, here derived from the packed parent
                        indices the tree tensors carry)
        s_j  = scale * <Q[r, i, h], K[r, j, h // G]>
        out  = sum_j softmax(s)_j * V[r, j, h // G]
    rows i >= n_nodes[r] are 0.

Layouts (readings: the paper fixes none): Q and out are
``[batch][N][Hq][D]`` (token-major, as a forward produces them); the K and V
caches of the layer are ``[batch][slots][Hkv][D]`` with the tree's node i
written at slot T + i, T = prefix_len[r].  Rotary position embeddings are
applied by the caller before attention (node positions are depth + T,
Appendix A), so they are not part of this step.

Only ``tests/`` and ``bench.py``'s CPU legs may import this module.  It
shares no code with the CUDA library.
"""
from __future__ import annotations

import numpy as np


def ancestors_or_self(parent, i: int):
    """Packed indices on the path from node i up to the root."""
    path = []
    while i >= 0:
        path.append(i)
        i = int(parent[i])
    return path


def allowed_keys(T: int, parent, i: int) -> np.ndarray:
    """Slots node i may attend to: the whole prefix, then the tree slots of
    its ancestors and itself, in slot order."""
    tree = sorted(T + m for m in ancestors_or_self(parent, i))
    return np.concatenate([np.arange(T), np.asarray(tree, dtype=np.int64)])


def tree_attention(Q, K, V, prefix_len, n_nodes, parent, scale,
                   rows=None):
    """Q ``[batch][N][Hq][D]``, K/V ``[batch][slots][Hkv][D]`` (float arrays,
    any precision: computed in float64), parent ``[batch][N]`` (packed
    parent index, -1 at the root).  Returns float64 ``[batch][N][Hq][D]``;
    ``rows`` (pairs ``(r, i)``) limits the nodes computed, the others stay 0."""
    Q = np.asarray(Q, dtype=np.float64)
    K = np.asarray(K, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    batch, N, Hq, D = Q.shape
    Hkv = K.shape[2]
    G = Hq // Hkv
    out = np.zeros((batch, N, Hq, D))
    todo = rows if rows is not None else [
        (r, i) for r in range(batch) for i in range(int(n_nodes[r]))]
    for r, i in todo:
        T = int(prefix_len[r])
        if i >= int(n_nodes[r]):
            continue
        keys = allowed_keys(T, parent[r], i)
        for h in range(Hq):
            kv = h // G
            s = scale * (K[r, keys, kv] @ Q[r, i, h])
            p = np.exp(s - s.max())
            out[r, i, h] = (p / p.sum()) @ V[r, keys, kv]
    return out
