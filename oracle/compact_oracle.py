"""Accepted-row compaction oracle.  TEST INFRASTRUCTURE ONLY.

After the target has verified a packed tree and the longest accepted
root-to-leaf row has been chosen, the KV rows the verification forward wrote
for the tree and the target's hidden states are gathered along that row and
placed right after the verified prefix (Appendix A, "Tensor implementation").

Plain definition written out here, per request ``r`` with verified prefix
length ``T = prefix_len[r]``, accepted node indices ``a = accepted_idx[r]``
(root first, ``a[0] = 0``) and ``L = accepted_len[r]`` accepted draft
tokens:

* every cache plane (each layer's K and V, or any other per-token tensor
  laid out the same way): slot ``T + j`` afterwards holds what slot
  ``T + a[j]`` held before, for ``j = 0 .. L``; every other slot keeps its
  content;
* hidden states: ``hidden_out[r][j] = hidden_in[r][a[j]]`` for
  ``j = 0 .. L``; rows ``j > L`` of ``hidden_out`` are left as they were.

Readings (the paper gives no layout): caches are byte rows addressed by
``(layer, plane, request, slot)`` with caller-chosen strides; a request whose
``accepted_idx`` is not a valid accepted path (``a[0] != 0``, not strictly
increasing, an index >= N) or whose ``T + N`` exceeds the slots of a row is
left untouched and reported as invalid.

Only ``tests/`` and ``bench.py``'s CPU legs may import this module.  It
shares no code with the CUDA library.
"""
from __future__ import annotations

import numpy as np


def path_ok(acc, length, n_tree):
    """True iff ``acc[0..length]`` is a path the greedy tree rule can accept:
    it starts at the root and node indices strictly increase (parents are
    packed before their children), all below ``n_tree``."""
    if length < 0 or length + 1 > len(acc):
        return False
    a = [int(x) for x in acc[: length + 1]]
    if a[0] != 0:
        return False
    for j in range(1, len(a)):
        if not (a[j - 1] < a[j] < n_tree):
            return False
    return True


def compact(cache, hidden_in, hidden_out, accepted_idx, accepted_len,
            prefix_len, n_tree):
    """Returns ``(cache_after, hidden_out_after, valid)``.

    ``cache``:      uint8 ``[layers][planes][batch][slots][row_bytes]``
    ``hidden_in``:  uint8 ``[batch][n_tree][hidden_bytes]`` or None
    ``hidden_out``: uint8 ``[batch][B+1][hidden_bytes]`` or None
    ``accepted_idx``: int ``[batch][B+1]``; ``accepted_len``, ``prefix_len``:
    int ``[batch]``.  ``valid[r]`` says whether request r was compacted.
    Inputs are not modified.
    """
    before = np.asarray(cache)
    after = before.copy()
    h_after = None if hidden_out is None else np.asarray(hidden_out).copy()
    n_layers, n_planes, batch, slots, _ = before.shape
    valid = np.zeros(batch, dtype=bool)
    for r in range(batch):
        T = int(prefix_len[r])
        L = int(accepted_len[r])
        acc = accepted_idx[r]
        if T < 0 or T + n_tree > slots or not path_ok(acc, L, n_tree):
            continue
        valid[r] = True
        for j in range(L + 1):
            src = T + int(acc[j])
            for layer in range(n_layers):
                for plane in range(n_planes):
                    after[layer, plane, r, T + j] = before[layer, plane, r, src]
            if h_after is not None:
                h_after[r, j] = hidden_in[r, int(acc[j])]
    return after, h_after, valid
