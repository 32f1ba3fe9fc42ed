"""Planted mistakes in the tree-attention oracle (on the CPU) must each fail
one of the pins in ``tests/test_attention_oracle.py``."""
import numpy as np
import pytest

from oracle import attention_oracle as ao
from tests import test_attention_oracle as pins

_real_allowed = ao.allowed_keys
_real_attention = ao.tree_attention


def _keys_without_self(T, parent, i):
    return np.asarray([j for j in _real_allowed(T, parent, i) if j != T + i])


def _keys_without_prefix(T, parent, i):
    return np.asarray([j for j in _real_allowed(T, parent, i) if j >= T])


def _keys_all_tree(T, parent, i):
    n = len(parent)
    return np.r_[np.arange(T), T + np.arange(n)[: max(i + 1, 1)]]


def _keys_short_prefix(T, parent, i):
    return np.asarray([j for j in _real_allowed(T, parent, i) if j != T - 1])


def _wrong_head_map(Q, K, V, prefix_len, n_nodes, parent, scale, rows=None):
    """Query head h reads KV head h % Hkv instead of h // G: per-head caches
    fed through the real code (one KV head per query head)."""
    Hq, Hkv = Q.shape[2], K.shape[2]
    heads = np.asarray([h % Hkv for h in range(Hq)])
    K2 = np.asarray(K, dtype=np.float64)[:, :, heads, :]
    V2 = np.asarray(V, dtype=np.float64)[:, :, heads, :]
    return _real_attention(Q, K2, V2, prefix_len, n_nodes, parent, scale, rows)


def _no_scale(Q, K, V, prefix_len, n_nodes, parent, scale, rows=None):
    return _real_attention(Q, K, V, prefix_len, n_nodes, parent, 1.0, rows)


def _all_pins():
    yield lambda: pins.test_equals_causal_attention_along_each_path("small")
    yield lambda: pins.test_equals_causal_attention_along_each_path("ragged")
    yield pins.test_uniform_keys_average_the_allowed_values
    yield pins.test_root_without_prefix_sees_only_itself
    yield pins.test_query_heads_share_their_group_kv_head
    yield pins.test_independent_of_packing_order


def _caught():
    for pin in _all_pins():
        try:
            pin()
        except (AssertionError, IndexError, ValueError):
            return True
    return False


@pytest.mark.parametrize("fn", [_keys_without_self, _keys_without_prefix,
                                _keys_all_tree, _keys_short_prefix])
def test_planted_key_set_mistake_is_caught(fn, monkeypatch):
    monkeypatch.setattr(ao, "allowed_keys", fn)
    assert _caught(), fn.__name__


@pytest.mark.parametrize("fn", [_wrong_head_map, _no_scale])
def test_planted_arithmetic_mistake_is_caught(fn, monkeypatch):
    monkeypatch.setattr(ao, "tree_attention", fn)
    assert _caught(), fn.__name__


def test_unplanted_oracle_passes():
    for pin in _all_pins():
        pin()
