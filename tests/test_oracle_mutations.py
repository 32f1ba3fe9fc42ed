"""Planted mistakes in the oracle (on the CPU) must each fail a pin.

Each test replaces one oracle function by a plausible wrong version and checks
that at least one of the pins in ``tests/pins.py`` catches it.
"""
import numpy as np
import pytest

from oracle import pctree_oracle as O
from tests import pins


def _bruteforce_any():
    for seed in range(6):
        pins.check_bruteforce(seed, 5, 3, 5, 4)


def _fails(*checks):
    for chk in checks:
        try:
            chk()
        except (AssertionError, O.ParityViolation, IndexError, ValueError):
            return True
    return False


def test_transposed_markov_operand_is_caught(monkeypatch):
    def wrong(E_in, W_out, parents):            # E_in and W_out swapped
        return W_out[np.asarray(parents)] @ E_in.T
    monkeypatch.setattr(O, "markov_bias", wrong)
    assert _fails(lambda: pins.check_markov_integer(0), _bruteforce_any)


def test_dropped_markov_bias_is_caught(monkeypatch):
    monkeypatch.setattr(O, "markov_bias",
                        lambda E, W, p: np.zeros((len(p), W.shape[0])))
    assert _fails(_bruteforce_any, lambda: pins.check_chain(0))


def test_unnormalised_scores_are_caught(monkeypatch):
    monkeypatch.setattr(O, "log_softmax", lambda z: (z, 0.0))
    assert _fails(_bruteforce_any)


def test_sign_error_in_log_softmax_is_caught(monkeypatch):
    real = O.log_softmax

    def wrong(z):
        lp, lse = real(z)
        return z + lse, lse
    monkeypatch.setattr(O, "log_softmax", wrong)
    assert _fails(pins.check_log_softmax, _bruteforce_any)


def test_wrong_child_tie_break_is_caught(monkeypatch):
    def wrong(z, k):                              # highest token first on ties
        order = np.lexsort((-np.arange(z.shape[0]), -z))
        return [int(v) for v in order[:k]]
    monkeypatch.setattr(O, "local_topk", wrong)
    assert _fails(pins.check_tie_children)


def test_frontier_by_id_is_caught(monkeypatch):
    monkeypatch.setattr(O, "layer_frontier",
                        lambda ids, s, k: sorted(ids)[:k])
    assert _fails(pins.check_pruning_example)


def test_frontier_tie_break_is_caught(monkeypatch):
    monkeypatch.setattr(O, "layer_frontier",
                        lambda ids, s, k: sorted(ids, key=lambda i: (-s[i], -i))[:k])
    assert _fails(pins.check_tie_frontier)


def test_no_frontier_pruning_is_caught(monkeypatch):
    monkeypatch.setattr(O, "layer_frontier", lambda ids, s, k: list(ids))
    assert _fails(pins.check_pruning_example,
                  lambda: pins.check_structure(0))


def test_global_selection_by_depth_first_is_caught(monkeypatch):
    monkeypatch.setattr(O, "global_topn", lambda s, depth, N: sorted(
        range(len(s)), key=lambda i: (depth[i], -s[i], i))[:N])
    assert _fails(_bruteforce_any, pins.check_pruning_example)


def test_wrong_accept_row_is_caught(monkeypatch):
    real = O.accept

    def wrong(tree, target, B):                  # stops one step early
        acc, length, bonus = real(tree, target, B)
        if length > 0:
            acc = acc.copy()
            acc[length] = -1
            return acc, length - 1, int(target[acc[length - 1]])
        return acc, length, bonus
    monkeypatch.setattr(O, "accept", wrong)
    assert _fails(lambda: pins.check_accept(0))


def test_mask_without_self_is_caught(monkeypatch):
    real = O.pack

    def wrong(pool, chosen, N, B, pos_offset=0):
        order, t = real(pool, chosen, N, B, pos_offset)
        for a in range(t.n_nodes):
            t.mask[a, a] = 0
        return order, t
    monkeypatch.setattr(O, "pack", wrong)
    assert _fails(lambda: pins.check_structure(0))


def test_shared_mode_conditioned_per_parent_is_caught(monkeypatch):
    real = O.draft

    def wrong(*args, **kw):                 # shared mode silently ignored
        if kw.get("mode") == "shared":
            kw["mode"] = "parent"
        return real(*args, **kw)
    monkeypatch.setattr(O, "draft", wrong)
    assert _fails(lambda: [pins.check_shared_bruteforce(s, 5, 3, 5, 4)
                           for s in range(6)],
                  lambda: pins.check_shared_children_identical(0))
