"""The oracle against what the paper and mathematics fix (no GPU)."""
import math

import numpy as np
import pytest

from oracle import pctree_oracle as O
from tests import pins


@pytest.mark.parametrize("V,B,N,k", [(5, 3, 5, 4), (8, 3, 8, 7), (4, 4, 4, 3),
                                     (3, 5, 4, 3)])
def test_bruteforce_topN_when_pruning_does_not_bind(V, B, N, k):
    done = sum(pins.check_bruteforce(seed, V, B, N, k) for seed in range(12))
    assert done >= 8


def test_pruning_example_hand_derived():
    pins.check_pruning_example()


def test_tie_breaks():
    pins.check_tie_children()
    pins.check_tie_frontier()


@pytest.mark.parametrize("seed", range(4))
def test_k1_is_greedy_chain(seed):
    pins.check_chain(seed)


@pytest.mark.parametrize("seed", range(3))
def test_markov_projection_exact_on_integers(seed):
    pins.check_markov_integer(seed)


def test_markov_projection_one_hot():
    pins.check_markov_one_hot()


def test_log_softmax():
    pins.check_log_softmax()


def test_decode_bf16():
    pins.check_decode_bf16()


@pytest.mark.parametrize("seed", range(6))
def test_tree_structure_invariants(seed):
    pins.check_structure(seed)


@pytest.mark.parametrize("seed", range(3))
def test_accept(seed):
    pins.check_accept(seed)


def test_k_equals_V_keeps_every_child():
    rng = np.random.default_rng(1)
    V, H, B = 5, 3, 2
    L = rng.normal(size=(B, V))
    rnd = O.draft(L, rng.normal(size=(V, H)), rng.normal(size=(V, H)),
                  root=0, B=B, k=V, N=100)
    assert sorted(rnd.pool.token[1:1 + V]) == list(range(V))
    assert rnd.tree.n_nodes == 1 + V + V * V     # N above the pool size


def test_single_node_budget():
    rnd, (V, B, k, N, off) = pins.random_round(0, N=1)
    t = rnd.tree
    assert t.n_nodes == 1 and t.n_leaves == 1
    assert t.retrieve[0].tolist() == [0] + [-1] * B
    acc, length, bonus = O.accept(t, np.array([7], np.int32), B)
    assert length == 0 and bonus == 7 and acc.tolist() == [0] + [-1] * B


def test_nonfinite_inputs_rejected():
    rng = np.random.default_rng(0)
    L = rng.normal(size=(2, 6))
    E, W = rng.normal(size=(6, 2)), rng.normal(size=(6, 2))
    for bad in (np.nan, np.inf):
        L2 = L.copy()
        L2[1, 3] = bad
        with pytest.raises(O.NonFiniteInput):
            O.draft(L2, E, W, 0, 2, 2, 4)
    W2 = W.copy()
    W2[0, 0] = np.nan
    with pytest.raises(O.NonFiniteInput):
        O.draft(L, E, W2, 0, 2, 2, 4)
    L3 = L.copy()
    L3[0, :] = -np.inf
    with pytest.raises(O.NonFiniteInput):
        O.draft(L3, E, W, 0, 2, 2, 4)


def test_neg_inf_logits_are_probability_zero():
    L = np.array([[0.0, -np.inf, 1.0, -np.inf], [0.0, 0.0, 0.0, 0.0]])
    rnd = O.draft(L, np.ones((4, 1)), np.zeros((4, 1)), 0, 2, 3, 20)
    kids = rnd.pool.token[1:4]
    assert kids == [2, 0, 1]                   # -inf tie broken by token id
    assert rnd.pool.s[3] == -np.inf
    t = rnd.tree
    # the -inf child and its three children are still pool nodes and fill
    # the budget last
    assert t.n_nodes == 1 + 3 + 9
    assert int(np.isneginf(t.logp[:t.n_nodes]).sum()) == 4
    rnd = O.draft(L, np.ones((4, 1)), np.zeros((4, 1)), 0, 2, 3, 9)
    assert not np.isneginf(rnd.tree.logp[:9]).any()


def test_replay_adopts_only_near_ties():
    rng = np.random.default_rng(5)
    V, H, B, k, N = 30, 4, 3, 3, 8
    L = rng.normal(size=(B, V)) * 3
    E, W = rng.normal(size=(V, H)), np.zeros((V, H))
    root = 0
    own = O.draft(L, E, W, root, B, k, N)
    hint = O.choices_from_pool(own.pool.token, own.pool.parent,
                               len(own.pool.token),
                               {own.pool.path[i] for i in own.selected})
    again = O.draft(L, E, W, root, B, k, N, hint=hint)
    assert again.n_ambiguous == 0
    assert np.array_equal(again.tree.tokens, own.tree.tokens)
    # make the k-th and (k+1)-th children of the root a near tie
    order = np.argsort(-L[0], kind="stable")
    a, b = int(order[k - 1]), int(order[k])
    L2 = L.copy()
    L2[0, b] = L2[0, a] - 1e-6
    # a hint from a round where b edges out a by 1e-6 instead
    L3 = L2.copy()
    L3[0, b] = L2[0, a] + 1e-6
    alt = O.draft(L3, E, W, root, B, k, N)
    alt_hint = O.choices_from_pool(alt.pool.token, alt.pool.parent,
                                   len(alt.pool.token),
                                   {alt.pool.path[i] for i in alt.selected})
    rep = O.draft(L2, E, W, root, B, k, N, hint=alt_hint)
    assert rep.n_ambiguous >= 1
    assert b in rep.pool.token[1:1 + k] and a not in rep.pool.token[1:1 + k]
    # each adopted choice records our own margin there: the root's children
    # were decided across a 1e-6 gap
    assert len(rep.adopted) == rep.n_ambiguous
    kinds = dict(rep.adopted)
    assert kinds["children"] == pytest.approx(1e-6, rel=1e-3)
    assert all(m <= 1e-6 * 1.001 for _, m in rep.adopted)
    # the same swap with a clear gap is refused
    L4 = L.copy()
    L4[0, b] = L4[0, a] - 0.5
    with pytest.raises(O.ParityViolation):
        O.draft(L4, E, W, root, B, k, N, hint=alt_hint)


def test_golden_tiny_round_regression():
    import json
    import os
    from workloads import WORKLOADS, draw_round, target_for_tree
    path = os.path.join(os.path.dirname(__file__), "golden",
                        "tiny_seed0_oracle.json")
    gold = json.load(open(path))
    wl = WORKLOADS["tiny"]
    inp = draw_round(wl)
    E, W = O.as_f64(inp.E_in, "f32"), O.as_f64(inp.W_out, "f32")
    rnd = O.draft(inp.L[0], E, W, int(inp.root[0]), wl.B, wl.k, wl.N)
    t = rnd.tree
    assert t.tokens.tolist() == gold["tokens"]
    assert t.parent.tolist() == gold["parent"]
    assert t.retrieve.tolist() == gold["retrieve"]
    assert np.allclose(t.logp, gold["logp"], atol=1e-12, rtol=0)
    target = target_for_tree(inp.greedy, t.depth[None, :])[0]
    acc, length, bonus = O.accept(t, target, wl.B)
    assert [acc.tolist(), length, bonus] == gold["accept"]


# --- Shared-Markov control (Sec. 5.3) --------------------------------------

@pytest.mark.parametrize("V,B,N,k", [(5, 3, 5, 4), (8, 3, 8, 7), (4, 4, 4, 3)])
def test_shared_bruteforce_topN(V, B, N, k):
    done = sum(pins.check_shared_bruteforce(seed, V, B, N, k)
               for seed in range(12))
    assert done >= 8


@pytest.mark.parametrize("seed", range(3))
def test_shared_equals_parent_without_bias(seed):
    pins.check_shared_equals_parent_without_bias(seed)


@pytest.mark.parametrize("seed", range(3))
def test_shared_children_identical(seed):
    pins.check_shared_children_identical(seed)


@pytest.mark.parametrize("seed", range(2))
def test_shared_k1_is_greedy_chain(seed):
    pins.check_chain(seed, mode="shared")
