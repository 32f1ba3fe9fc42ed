"""Pins of the accepted-row compaction oracle (Appendix A, "Tensor
implementation": KV tensors and target hidden states are gathered along the
accepted row and compacted after the verified prefix).

Each pin checks the oracle against something other than its own copy loop:
labelled rows decoded back to the slot they came from, identity and empty
paths, untouched requests on invalid input, an in-place forward sweep, and a
whole draft -> accept -> compact chain through the tree oracle, where the
compacted rows must spell out the tokens the target agreed with.
"""
import numpy as np
import pytest

from oracle import compact_oracle as co
from oracle import pctree_oracle as po
from workloads import (COMPACT_WORKLOADS, CompactWorkload, WORKLOADS,
                       draw_compaction, draw_round, target_for_tree)


def labelled_cache(cw):
    """Row (layer, plane, r, slot) holds its own coordinates, so a row's
    origin can be read back after any permutation."""
    shape = (cw.layers, cw.planes, cw.batch, cw.slots, cw.row_bytes // 4)
    lab = np.zeros(shape, dtype=np.int32)
    idx = np.indices(shape[:4])
    lab[...] = (((idx[0] * 8 + idx[1]) * 64 + idx[2]) * 4096 + idx[3])[..., None]
    return lab.view(np.uint8).reshape(shape[:4] + (cw.row_bytes,))


def decode(cache):
    return cache.view(np.int32)[..., 0] % 4096   # the slot a row came from


@pytest.mark.parametrize("name", ["small", "ragged"])
def test_rows_come_from_the_accepted_nodes(name):
    cw = COMPACT_WORKLOADS[name]
    ci = draw_compaction(cw)
    cache = labelled_cache(cw)
    # hidden row i of request r holds (r, i); output rows start at -1
    hid_in = np.zeros((cw.batch, cw.N, cw.hidden_bytes // 4), np.int32)
    hid_in[...] = (np.arange(cw.batch)[:, None] * 1000 +
                   np.arange(cw.N)[None, :])[..., None]
    hid_out = np.full((cw.batch, cw.B + 1, cw.hidden_bytes // 4), -1, np.int32)
    after, hid, valid = co.compact(cache, hid_in.view(np.uint8),
                                   hid_out.view(np.uint8), ci.accepted_idx,
                                   ci.accepted_len, ci.prefix_len, cw.N)
    assert valid.all()
    hid = hid.view(np.int32)[..., 0]
    for r in range(cw.batch):
        n = int(ci.accepted_len[r])
        np.testing.assert_array_equal(hid[r, :n + 1],
                                      r * 1000 + ci.accepted_idx[r, :n + 1])
        assert (hid[r, n + 1:] == -1).all()
    slot_of = decode(after)
    for r in range(cw.batch):
        T, n = int(ci.prefix_len[r]), int(ci.accepted_len[r])
        want = np.arange(cw.slots)
        want[T:T + n + 1] = T + ci.accepted_idx[r, :n + 1]
        for layer in range(cw.layers):
            for p in range(cw.planes):
                np.testing.assert_array_equal(slot_of[layer, p, r], want)
    # the other coordinates survive too: nothing crosses layers or requests
    full = after.view(np.int32)[..., 0]
    idx = np.indices(full.shape)
    np.testing.assert_array_equal(full // 4096,
                                  (idx[0] * 8 + idx[1]) * 64 + idx[2])


def test_identity_and_empty_paths_change_nothing():
    cw = COMPACT_WORKLOADS["small"]
    ci = draw_compaction(cw)
    acc = np.full_like(ci.accepted_idx, -1)
    lens = np.array([cw.B, 0, 2], dtype=np.int32)
    acc[0, :cw.B + 1] = np.arange(cw.B + 1)
    acc[1, 0] = 0
    acc[2, :3] = [0, 1, 2]
    after, hid, valid = co.compact(ci.cache, ci.hidden_in, ci.hidden_out, acc,
                                   lens, ci.prefix_len, cw.N)
    assert valid.all()
    np.testing.assert_array_equal(after, ci.cache)
    # hidden rows are gathered out of place: row j = hidden_in[a[j]]
    for r in range(cw.batch):
        n = lens[r]
        np.testing.assert_array_equal(hid[r, :n + 1], ci.hidden_in[r, :n + 1])
        np.testing.assert_array_equal(hid[r, n + 1:], ci.hidden_out[r, n + 1:])


@pytest.mark.parametrize("bad", [
    ("root not first", lambda a, n: a.__setitem__(0, 1), None),
    ("repeated node", lambda a, n: a.__setitem__(2, a[1]), None),
    ("decreasing", lambda a, n: a.__setitem__(slice(1, 3), [5, 3]), None),
    ("node beyond tree", lambda a, n: a.__setitem__(2, n), None),
    ("negative len", None, -1),
    ("len beyond B", None, 99),
])
def test_invalid_paths_leave_the_request_untouched(bad):
    cw = COMPACT_WORKLOADS["small"]
    ci = draw_compaction(cw)
    acc = ci.accepted_idx.copy()
    lens = ci.accepted_len.copy()
    acc[1, :4] = [0, 2, 4, 6]
    lens[1] = 3
    _, edit, new_len = bad
    if edit is not None:
        edit(acc[1], cw.N)
    if new_len is not None:
        lens[1] = new_len
    after, hid, valid = co.compact(ci.cache, ci.hidden_in, ci.hidden_out, acc,
                                   lens, ci.prefix_len, cw.N)
    assert not valid[1] and valid[0] and valid[2]
    np.testing.assert_array_equal(after[:, :, 1], ci.cache[:, :, 1])
    np.testing.assert_array_equal(hid[1], ci.hidden_out[1])


def test_prefix_overflow_is_invalid():
    cw = COMPACT_WORKLOADS["small"]
    ci = draw_compaction(cw)
    prefix = ci.prefix_len.copy()
    prefix[2] = cw.prefix_max + 1          # the tree would end past the row
    _, _, valid = co.compact(ci.cache, None, None, ci.accepted_idx,
                             ci.accepted_len, prefix, cw.N)
    assert list(valid) == [True, True, False]
    prefix[2] = -1
    _, _, valid = co.compact(ci.cache, None, None, ci.accepted_idx,
                             ci.accepted_len, prefix, cw.N)
    assert not valid[2]


def test_forward_in_place_sweep_matches():
    """Because a[j] >= j, copying slot T+a[j] to T+j for j = 0, 1, ... in
    place reads every source before it is overwritten; the result equals
    the gather from an untouched copy."""
    cw = COMPACT_WORKLOADS["ragged"]
    for seed in range(5):
        ci = draw_compaction(cw, seed=seed)
        want, _, _ = co.compact(ci.cache, None, None, ci.accepted_idx,
                                ci.accepted_len, ci.prefix_len, cw.N)
        got = ci.cache.copy()
        for r in range(cw.batch):
            T = int(ci.prefix_len[r])
            for j in range(int(ci.accepted_len[r]) + 1):
                got[:, :, r, T + j] = got[:, :, r, T + int(ci.accepted_idx[r, j])]
        np.testing.assert_array_equal(got, want)


def test_draft_accept_compact_chain():
    """Cache rows stamped with each tree node's token: after compaction the
    slots after the prefix hold the root and then exactly the drafted tokens
    the target accepted, each equal to the target's token at the previous
    accepted node, and the bonus token follows the last of them."""
    wl = WORKLOADS["tiny"]
    ri = draw_round(wl)
    rnd = po.draft(ri.L[0], ri.E_in, ri.W_out, int(ri.root[0]), wl.B, wl.k,
                   wl.N)
    tree = rnd.tree
    # a target that agrees with the tree along the path to its deepest node
    n = tree.n_nodes
    u = int(np.argmax(tree.depth[:n]))
    path = [u]
    while path[-1] != 0:
        path.append(int(tree.parent[path[-1]]))
    path.reverse()
    target = target_for_tree(ri.greedy, tree.depth[None])[0]
    for a, b in zip(path, path[1:]):
        target[a] = tree.tokens[b]
    acc, n_acc, bonus = po.accept(tree, target, wl.B)
    assert n_acc == tree.depth[u] >= 2
    assert list(acc[:n_acc + 1]) == path
    cw = CompactWorkload("chain", layers=2, planes=2, row_bytes=16,
                         hidden_bytes=16, B=wl.B, N=wl.N, batch=1,
                         prefix_max=5, seed=0)
    T = 3
    cache = np.zeros((2, 2, 1, cw.slots, 4), dtype=np.int32) - 7
    cache[:, :, 0, T:T + tree.n_nodes, :] = tree.tokens[:tree.n_nodes, None]
    after, _, valid = co.compact(cache.view(np.uint8), None, None, acc[None],
                                 np.array([n_acc]), np.array([T]), wl.N)
    assert valid[0]
    toks = after.view(np.int32)[0, 0, 0, :, 0]
    assert toks[T] == int(ri.root[0]) == tree.tokens[0]
    for j in range(1, n_acc + 1):
        assert toks[T + j] == target[acc[j - 1]]
    assert bonus == target[acc[n_acc]]
    assert (toks[:T] == -7).all()
