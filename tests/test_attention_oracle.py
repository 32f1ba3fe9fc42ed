"""Pins of the tree-verification attention oracle (Sec. 4.2; Appendix A,
"Tensor implementation": a node attends to the verified prefix, itself and
its root-to-node ancestors).

The pins check the oracle against other formulations of the same facts:
each node's output equals ordinary causal attention at the last position of
the linear sequence prefix + root-to-node path; closed forms for uniform
keys and a lone key; grouped-query head sharing; independence from the
order the tree is packed in.
"""
import numpy as np
import pytest

from oracle import attention_oracle as ao
from workloads import (ATTN_WORKLOADS, AttnWorkload, bf16_bits_to_f32,
                       draw_attention)


def values(a):
    return bf16_bits_to_f32(a).astype(np.float64)


def causal_last(q, Ks, Vs, scale):
    """Textbook causal attention of a linear sequence, last query row: the
    full score matrix with the upper triangle masked, row-wise softmax."""
    n = Ks.shape[0]
    Qs = np.zeros((n, q.shape[0]))
    Qs[-1] = q
    S = scale * Qs @ Ks.T
    S[np.triu_indices(n, 1)] = -np.inf
    P = np.exp(S - S.max(axis=1, keepdims=True))
    P /= P.sum(axis=1, keepdims=True)
    return (P @ Vs)[-1]


def path_of(parent, i):
    p = []
    while i >= 0:
        p.append(i)
        i = int(parent[i])
    return p[::-1]


@pytest.mark.parametrize("name", ["small", "ragged"])
def test_equals_causal_attention_along_each_path(name):
    ai = draw_attention(ATTN_WORKLOADS[name])
    aw = ai.aw
    Q, K, V = values(ai.q), values(ai.k), values(ai.v)
    scale = 1.0 / np.sqrt(aw.D)
    out = ao.tree_attention(Q, K, V, ai.prefix_len, ai.n_nodes, ai.parent, scale)
    G = aw.Hq // aw.Hkv
    for r in range(aw.batch):
        T, n = int(ai.prefix_len[r]), int(ai.n_nodes[r])
        for i in range(aw.N):
            if i >= n:
                assert not out[r, i].any()
                continue
            seq = list(range(T)) + [T + m for m in path_of(ai.parent[r], i)]
            for h in range(0, aw.Hq, 3):
                want = causal_last(Q[r, i, h], K[r, seq, h // G],
                                   V[r, seq, h // G], scale)
                np.testing.assert_allclose(out[r, i, h], want, rtol=0,
                                           atol=1e-12)


def test_uniform_keys_average_the_allowed_values():
    ai = draw_attention(ATTN_WORKLOADS["small"])
    K = np.ones(ai.k.shape)                 # every score equal
    V = values(ai.v)
    out = ao.tree_attention(values(ai.q) * 0 + 1, K, V, ai.prefix_len,
                            ai.n_nodes, ai.parent, 0.3)
    for r in range(ai.aw.batch):
        T = int(ai.prefix_len[r])
        for i in range(int(ai.n_nodes[r])):
            depth = len(path_of(ai.parent[r], i)) - 1
            rows = np.r_[np.arange(T), [T + m for m in path_of(ai.parent[r], i)]]
            assert len(rows) == T + depth + 1
            np.testing.assert_allclose(out[r, i, 0], V[r, rows, 0].mean(axis=0),
                                       rtol=0, atol=1e-12)


def test_root_without_prefix_sees_only_itself():
    ai = draw_attention(ATTN_WORKLOADS["small"])
    assert ai.prefix_len[1] == 0
    V = values(ai.v)
    out = ao.tree_attention(values(ai.q), values(ai.k), V, ai.prefix_len,
                            ai.n_nodes, ai.parent, 1 / np.sqrt(128))
    G = ai.aw.Hq // ai.aw.Hkv
    for h in range(ai.aw.Hq):
        np.testing.assert_array_equal(out[1, 0, h], V[1, 0, h // G])


def test_query_heads_share_their_group_kv_head():
    aw = ATTN_WORKLOADS["ragged"]            # 10 query heads, 2 KV heads
    ai = draw_attention(aw)
    V = np.zeros(ai.v.shape)
    for c in range(aw.Hkv):
        V[:, :, c, :] = c + 1.0
    out = ao.tree_attention(values(ai.q), values(ai.k), V, ai.prefix_len,
                            ai.n_nodes, ai.parent, 1 / np.sqrt(128))
    G = aw.Hq // aw.Hkv
    for h in range(aw.Hq):
        np.testing.assert_allclose(out[0, 0, h], h // G + 1.0, rtol=1e-12)


def test_independent_of_packing_order():
    """Relabel the tree's nodes (moving their KV rows and queries along):
    every node's output is unchanged."""
    aw = AttnWorkload("perm", batch=1, N=12, Hq=4, Hkv=2, D=128, B=4,
                      prefix_max=9, seed=3)
    ai = draw_attention(aw)
    Q, K, V = values(ai.q), values(ai.k), values(ai.v)
    T, n = int(ai.prefix_len[0]), int(ai.n_nodes[0])
    scale = 0.1
    base = ao.tree_attention(Q, K, V, ai.prefix_len, ai.n_nodes, ai.parent, scale)
    rng = np.random.default_rng(0)
    new_of = np.arange(aw.N)
    new_of[:n] = rng.permutation(n)          # old index -> new index
    par = np.full_like(ai.parent, -1)
    Q2, K2, V2 = Q.copy(), K.copy(), V.copy()
    for old in range(n):
        new = new_of[old]
        par[0, new] = -1 if ai.parent[0, old] < 0 else new_of[ai.parent[0, old]]
        Q2[0, new] = Q[0, old]
        K2[0, T + new] = K[0, T + old]
        V2[0, T + new] = V[0, T + old]
    out = ao.tree_attention(Q2, K2, V2, ai.prefix_len, ai.n_nodes, par, scale)
    for old in range(n):
        np.testing.assert_allclose(out[0, new_of[old]], base[0, old],
                                   rtol=0, atol=1e-12)
