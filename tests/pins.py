"""Checks that pin the oracle to facts fixed by the paper and by mathematics.

Each ``check_*`` raises ``AssertionError`` when the oracle disagrees.  The
tests in ``test_oracle_pins.py`` run them on the oracle as written; the tests
in ``test_oracle_mutations.py`` plant a plausible mistake in the oracle and
show that at least one check fails.
"""
from __future__ import annotations

import math
from fractions import Fraction
from itertools import product
from typing import Dict, List, Tuple

import numpy as np

from oracle import pctree_oracle as O


# ----------------------------------------------------------------------------
# bigram heads with exactly known conditionals
# ----------------------------------------------------------------------------

def bigram_case(seed: int, V: int, B: int):
    """A Markov head that is an exact bigram model.

    With ``E_in = I`` (H = V) and ``W_out[v][h] = log Q[h][v]``, the head's
    bias for parent p is ``log Q[p][.]``; with ``L_d = log P_d`` Eq. 2 gives
    ``pi_d(v | p) = P_d[v] Q[p][v] / sum_u P_d[u] Q[p][u]``, which is computed
    here in exact rational arithmetic.
    """
    rng = np.random.default_rng(seed)
    P = [[Fraction(int(x)) for x in rng.integers(1, 60, size=V)] for _ in range(B)]
    P = [[x / sum(row) for x in row] for row in P]
    Q = [[Fraction(int(x)) for x in rng.integers(1, 60, size=V)] for _ in range(V)]
    Q = [[x / sum(row) for x in row] for row in Q]
    L = np.array([[math.log(x) for x in row] for row in P], dtype=np.float64)
    E_in = np.eye(V, dtype=np.float64)
    W_out = np.array([[math.log(Q[h][v]) for h in range(V)] for v in range(V)],
                     dtype=np.float64)
    root = int(rng.integers(0, V))
    cond = [[[P[d][v] * Q[p][v] for v in range(V)] for p in range(V)]
            for d in range(B)]
    for d in range(B):
        for p in range(V):
            z = sum(cond[d][p])
            cond[d][p] = [x / z for x in cond[d][p]]
    return L, E_in, W_out, root, cond


def all_paths(cond, root: int, V: int, B: int) -> Dict[Tuple[int, ...], Fraction]:
    """Exact joint probability of every node of the full V-ary depth-B tree."""
    out = {(): Fraction(1)}
    for depth in range(1, B + 1):
        for path in product(range(V), repeat=depth):
            prev = root if depth == 1 else path[-2]
            out[path] = out[path[:-1]] * cond[depth - 1][prev][path[-1]]
    return out


def check_bruteforce(seed: int, V: int, B: int, N: int, k: int) -> bool:
    """If pruning never binds (k >= N-1, k <= V), the kept set is the N most
    probable nodes of the full tree (Sec. 4.2 selection rule).  Returns False
    if the seed draws a near-tie at the cut (the caller then skips it)."""
    assert N - 1 <= k <= V
    L, E_in, W_out, root, cond = bigram_case(seed, V, B)
    probs = all_paths(cond, root, V, B)
    ranked = sorted(probs.items(), key=lambda kv: (-kv[1], len(kv[0])))
    top = ranked[:N + 1]
    vals = [p for _, p in top]
    if len(set(vals)) != len(vals):
        return False
    if N < len(ranked) and (vals[N - 1] - vals[N]) / vals[N - 1] < 1e-9:
        return False
    want = {path for path, _ in ranked[:N]}
    rnd = O.draft(L, E_in, W_out, root, B, k, N)
    got = {rnd.pool.path[i] for i in rnd.selected}
    assert got == want, f"kept {sorted(got)} != most probable {sorted(want)}"
    # Eq. 4: every pool node's score is the exact log joint probability
    for i, path in enumerate(rnd.pool.path):
        exact = math.log(probs[path])
        assert abs(rnd.pool.s[i] - exact) < 1e-12, (path, rnd.pool.s[i], exact)
    for a in range(rnd.tree.n_nodes):
        assert abs(rnd.tree.logp[a] - rnd.pool.s[rnd.selected[a]]) == 0.0
    return True


# ----------------------------------------------------------------------------
# hand-derived pruning example (parent-independent head, exact probabilities)
# ----------------------------------------------------------------------------

def pruning_case():
    """W_out = 0, so every parent gets the same child distribution P_d.

    P_0 = (.5, .3, .2), P_1 = (.62, .28, .10), P_2 = (.7, .2, .1); k = 2.
    Stage 0: children of the root are tokens 0 (.5) and 1 (.3); token 2 (.2)
    is cut by the per-parent top-2.  Stage 1: (0,0)=.31 (0,1)=.14 (1,0)=.186
    (1,1)=.084; the frontier keeps (0,0) and (1,0).  Stage 2: (0,0,0)=.217
    (0,0,1)=.062 (1,0,0)=.1302 (1,0,1)=.0372.  The nine best pool nodes are
    (), (0), (0,0), (1), (0,0,0), (1,0), (0,1), (1,0,0), (1,1).  The full tree
    would instead hold (2)=.2 and (0,1,0)=.098 among its nine best: both
    were removed by pruning (Sec. 6, limitation 2).
    """
    P = [(.5, .3, .2), (.62, .28, .10), (.7, .2, .1)]
    L = np.log(np.array(P, dtype=np.float64))
    E_in = np.ones((3, 2))
    W_out = np.zeros((3, 2))
    return L, E_in, W_out


def check_pruning_example() -> None:
    L, E_in, W_out = pruning_case()
    rnd = O.draft(L, E_in, W_out, root=2, B=3, k=2, N=9)
    t = rnd.tree
    assert t.n_nodes == 9
    assert t.tokens.tolist() == [2, 0, 1, 0, 1, 0, 1, 0, 0], t.tokens
    assert t.parent.tolist() == [-1, 0, 0, 1, 1, 2, 2, 3, 5], t.parent
    assert t.depth.tolist() == [0, 1, 1, 2, 2, 2, 2, 3, 3]
    want = [1, .5, .3, .31, .14, .186, .084, .217, .1302]
    assert np.allclose(t.logp, np.log(want), atol=1e-12, rtol=0), t.logp
    assert len(rnd.pool.token) == 1 + 2 + 2 * 4


# ----------------------------------------------------------------------------
# planted exact ties: (z desc, token asc), (s desc, id asc), depth asc
# ----------------------------------------------------------------------------

def tie_case(B: int):
    L = np.tile(np.array([1.0, 1.0, 0.0, 0.0]), (B, 1))
    return L, np.ones((4, 2)), np.zeros((4, 2))


def check_tie_children() -> None:
    """Tied children are ranked by token id; tied nodes by id; a tied parent
    precedes its child."""
    L, E_in, W_out = tie_case(2)
    rnd = O.draft(L, E_in, W_out, root=3, B=2, k=2, N=4)
    assert rnd.tree.tokens.tolist() == [3, 0, 1, 0], rnd.tree.tokens
    assert rnd.tree.parent.tolist() == [-1, 0, 0, 1], rnd.tree.parent
    rnd = O.draft(L, E_in, W_out, root=3, B=2, k=2, N=5)
    assert rnd.tree.tokens.tolist() == [3, 0, 1, 0, 1]
    assert rnd.tree.parent.tolist() == [-1, 0, 0, 1, 1]


def check_tie_frontier() -> None:
    """A frontier cut between four tied nodes keeps the two lowest ids."""
    L, E_in, W_out = tie_case(3)
    rnd = O.draft(L, E_in, W_out, root=3, B=3, k=2, N=8)
    # 1 root + 2 at depth 1 + 4 at depth 2 + first depth-3 node by id
    assert rnd.tree.depth.tolist() == [0, 1, 1, 2, 2, 2, 2, 3]
    assert rnd.tree.tokens.tolist() == [3, 0, 1, 0, 1, 0, 1, 0]
    assert rnd.tree.parent.tolist() == [-1, 0, 0, 1, 1, 2, 2, 3]


# ----------------------------------------------------------------------------
# k = 1 recovers DSpark's greedy chain (Sec. 4.2, Eq. 1)
# ----------------------------------------------------------------------------

def greedy_chain(L, E_in, W_out, root: int, B: int) -> List[int]:
    """Eq. 1 written as plain loops: y_d = argmax_v L_d[v] + Markov(y_{d-1})[v]
    (lowest token on exact ties)."""
    V, H = W_out.shape
    y, out = root, []
    for d in range(B):
        best, best_v = -math.inf, -1
        for v in range(V):
            z = float(L[d][v])
            for h in range(H):
                z += float(W_out[v][h]) * float(E_in[y][h])
            if z > best:
                best, best_v = z, v
        y = best_v
        out.append(y)
    return out


def check_chain(seed: int, V: int = 40, H: int = 5, B: int = 6,
                mode: str = "parent") -> None:
    rng = np.random.default_rng(seed)
    L = rng.normal(size=(B, V)) * 2.0
    E_in = rng.normal(size=(V, H))
    W_out = rng.normal(size=(V, H))
    root = int(rng.integers(V))
    chain = greedy_chain(L, E_in, W_out, root, B)
    for N in (B + 1, B, 3, 1):
        rnd = O.draft(L, E_in, W_out, root, B, k=1, N=N, mode=mode)
        n = min(N, B + 1)
        assert rnd.tree.n_nodes == n
        assert rnd.tree.tokens[:n].tolist() == [root] + chain[:n - 1]
        assert rnd.tree.parent[:n].tolist() == list(range(-1, n - 1))
        assert rnd.markov_calls == [1] * B


# ----------------------------------------------------------------------------
# Markov projection and log-softmax
# ----------------------------------------------------------------------------

def check_markov_integer(seed: int) -> None:
    """Integer-valued heads: every product and sum is exact in float64, so
    the bias must equal the triple-loop sum exactly."""
    rng = np.random.default_rng(seed)
    V, H = 7, 5
    E = rng.integers(-4, 5, size=(V, H))
    W = rng.integers(-4, 5, size=(V, H))
    parents = [int(p) for p in rng.integers(0, V, size=3)]
    got = O.markov_bias(E.astype(np.float64), W.astype(np.float64), parents)
    for r, p in enumerate(parents):
        for v in range(V):
            want = sum(int(W[v][h]) * int(E[p][h]) for h in range(H))
            assert got[r][v] == want, (r, v, got[r][v], want)


def check_markov_one_hot() -> None:
    """With one-hot input rows the bias of parent p is W_out's column p."""
    rng = np.random.default_rng(3)
    V = 6
    W = rng.normal(size=(V, V))
    got = O.markov_bias(np.eye(V), W, [4, 1])
    assert np.array_equal(got[0], W[:, 4]) and np.array_equal(got[1], W[:, 1])


def check_log_softmax() -> None:
    # constant row: every log pi is -log V, lse = c + log V
    z = np.full(1000, 3.25)
    lp, lse = O.log_softmax(z)
    assert abs(lse - (3.25 + math.log(1000))) < 1e-12
    assert np.allclose(lp, -math.log(1000), atol=1e-12, rtol=0)
    # z = log p with sum p = 1 gives back log p
    p = np.array([.5, .25, .125, .0625, .0625])
    lp, lse = O.log_softmax(np.log(p) + 7.0)
    assert abs(lse - 7.0) < 1e-12 and np.allclose(lp, np.log(p), atol=1e-12)
    # against scipy's logsumexp on wide rows
    from scipy.special import logsumexp
    rng = np.random.default_rng(0)
    for _ in range(5):
        z = rng.normal(size=5000) * 6
        lp, lse = O.log_softmax(z)
        assert abs(lse - logsumexp(z)) < 1e-10
        assert abs(math.log(np.exp(lp).sum())) < 1e-10
    # -inf entries carry probability 0
    lp, lse = O.log_softmax(np.array([0.0, -np.inf, 0.0]))
    assert lp[1] == -np.inf and abs(lse - math.log(2)) < 1e-15


def check_decode_bf16() -> None:
    bits = np.array([0x3F80, 0xC000, 0x0000, 0x8000, 0x7F80, 0x3F81, 0x0001,
                     0x4049], dtype=np.uint16)
    want = [1.0, -2.0, 0.0, -0.0, math.inf, 1.0 + 2.0 ** -7, 2.0 ** -133,
            3.140625]
    got = O.decode_bf16(bits)
    assert got.tolist() == want, got
    assert math.copysign(1.0, got[3]) == -1.0


# ----------------------------------------------------------------------------
# tree tensors and acceptance
# ----------------------------------------------------------------------------

def random_round(seed: int, V=60, H=6, B=5, k=3, N=12, pos_offset=17):
    rng = np.random.default_rng(seed)
    L = rng.normal(size=(B, V)) * 3.0
    E_in = rng.normal(size=(V, H))
    W_out = rng.normal(size=(V, H)) * 0.8
    root = int(rng.integers(V))
    return O.draft(L, E_in, W_out, root, B, k, N, pos_offset), (V, B, k, N,
                                                               pos_offset)


def check_structure(seed: int) -> None:
    rnd, (V, B, k, N, off) = random_round(seed)
    t = rnd.tree
    n = t.n_nodes
    assert len(rnd.pool.token) == 1 + k + (B - 1) * k * k     # Sec. 4.1 bound
    assert rnd.markov_calls == [1] + [k] * (B - 1)             # b_0=1, b_d<=k
    assert n == min(N, len(rnd.pool.token))
    assert t.parent[0] == -1 and t.depth[0] == 0 and t.logp[0] == 0.0
    for a in range(1, n):
        p = t.parent[a]
        assert 0 <= p < a
        assert t.depth[a] == t.depth[p] + 1
        assert t.logp[a] <= t.logp[p]
    for a in range(n):                                          # siblings
        kids = [t.tokens[c] for c in range(n) if t.parent[c] == a]
        assert len(kids) == len(set(kids))
        assert kids == sorted(kids)
    assert (t.position_ids[:n] == t.depth[:n] + off).all()
    assert (t.position_ids[n:] == -1).all() and (t.tokens[n:] == -1).all()
    for a in range(n):
        anc = set()
        b = a
        while b >= 0:
            anc.add(b)
            b = t.parent[b]
        assert set(np.nonzero(t.mask[a])[0].tolist()) == anc
        assert t.mask[a].sum() == t.depth[a] + 1
    assert not t.mask[n:].any() and not t.mask[:, n:].any()
    leaves = [a for a in range(n) if not (t.parent[:n] == a).any()]
    assert t.n_leaves == len(leaves)
    for j, leaf in enumerate(leaves):
        row = t.retrieve[j]
        m = int((row >= 0).sum())
        assert (row[m:] == -1).all() and row[0] == 0 and row[m - 1] == leaf
        for x, y in zip(row[:m - 1], row[1:m]):
            assert t.parent[y] == x
    assert (t.retrieve[t.n_leaves:] == -1).all()
    # depth order then parent's index then token
    keys = [(t.depth[a], t.parent[a], t.tokens[a]) for a in range(n)]
    assert keys == sorted(keys)


def walk_accept(t: O.Tree, target: np.ndarray) -> Tuple[List[int], int]:
    """Greedy tree walk: from the root, follow the child whose token is the
    target's token at the current node."""
    cur, path = 0, [0]
    while True:
        nxt = [c for c in range(t.n_nodes)
               if t.parent[c] == cur and t.tokens[c] == target[cur]]
        assert len(nxt) <= 1
        if not nxt:
            return path, int(target[cur])
        cur = nxt[0]
        path.append(cur)


def check_accept(seed: int) -> None:
    rnd, (V, B, k, N, off) = random_round(seed)
    t = rnd.tree
    n = t.n_nodes
    rng = np.random.default_rng(seed + 100)
    # a target that follows the path to node u, then leaves the tree
    for u in range(n):
        path = []
        b = u
        while b >= 0:
            path.append(b)
            b = t.parent[b]
        path.reverse()
        target = np.full(N, -1, np.int32)
        for a in range(n):
            used = {int(t.tokens[c]) for c in range(n) if t.parent[c] == a}
            choices = [v for v in range(V) if v not in used]
            target[a] = choices[int(rng.integers(len(choices)))]
        for x, y in zip(path[:-1], path[1:]):
            target[x] = t.tokens[y]
        acc, length, bonus = O.accept(t, target, B)
        assert length == len(path) - 1
        assert acc[:length + 1].tolist() == path
        assert (acc[length + 1:] == -1).all()
        assert bonus == target[u]
        walk, wb = walk_accept(t, target)
        assert walk == path and wb == bonus
    # per-depth targets (the synthetic target model)
    for _ in range(20):
        g = rng.integers(0, V, size=B + 1)
        g[: B] = np.where(rng.random(B) < 0.7, g[: B], 0)
        target = np.where(t.depth >= 0, g[np.maximum(t.depth, 0)], -1)
        acc, length, bonus = O.accept(t, target, B)
        walk, wb = walk_accept(t, target)
        assert acc[:length + 1].tolist() == walk and bonus == wb


# ----------------------------------------------------------------------------
# Shared-Markov control (Sec. 5.3): one distribution per depth for all parents
# ----------------------------------------------------------------------------

def check_shared_bruteforce(seed: int, V: int, B: int, N: int, k: int) -> bool:
    """Shared mode: every node at depth d+1 takes q_d, the distribution of
    the greedy chain's depth-d step (Eq. 1).  With pruning unable to bind,
    the kept set is the N most probable nodes of the full tree under those
    shared distributions, computed exactly."""
    assert N - 1 <= k <= V
    L, E_in, W_out, root, cond = bigram_case(seed, V, B)
    chain, prev = [], root
    for d in range(B):
        row = cond[d][prev]
        best = max(range(V), key=lambda v: (row[v], -v))
        if sorted(row, reverse=True)[0] == sorted(row, reverse=True)[1]:
            return False                    # exact tie in the chain argmax
        chain.append(row)
        prev = best
    probs = {(): Fraction(1)}
    for depth in range(1, B + 1):
        for path in product(range(V), repeat=depth):
            probs[path] = probs[path[:-1]] * chain[depth - 1][path[-1]]
    ranked = sorted(probs.items(), key=lambda kv: (-kv[1], len(kv[0])))
    vals = [p for _, p in ranked[:N + 1]]
    if len(set(vals)) != len(vals):
        return False
    if N < len(ranked) and (vals[N - 1] - vals[N]) / vals[N - 1] < 1e-9:
        return False
    want = {path for path, _ in ranked[:N]}
    rnd = O.draft(L, E_in, W_out, root, B, k, N, mode="shared")
    got = {rnd.pool.path[i] for i in rnd.selected}
    assert got == want, f"kept {sorted(got)} != most probable {sorted(want)}"
    for i, path in enumerate(rnd.pool.path):
        assert abs(rnd.pool.s[i] - math.log(probs[path])) < 1e-12
    assert rnd.markov_calls == [1] * B
    return True


def check_shared_equals_parent_without_bias(seed: int) -> None:
    """With W_out = 0 the head adds nothing, so parent-conditioned and shared
    scoring are the same distribution and must build the same tree."""
    rng = np.random.default_rng(seed)
    V, H, B, k, N = 40, 4, 5, 3, 12
    L = rng.normal(size=(B, V)) * 2
    E_in, W_out = rng.normal(size=(V, H)), np.zeros((V, H))
    root = int(rng.integers(V))
    a = O.draft(L, E_in, W_out, root, B, k, N, mode="parent")
    b = O.draft(L, E_in, W_out, root, B, k, N, mode="shared")
    assert a.pool.path == b.pool.path and a.pool.s == b.pool.s
    assert (a.tree.tokens == b.tree.tokens).all()


def check_shared_children_identical(seed: int) -> None:
    """Every parent of a layer gets the same ranked children with the same
    log-probabilities; the depth-1 layer equals parent mode's."""
    rnd, _ = random_round(seed)
    rng = np.random.default_rng(seed)
    V, H, B, k, N = 60, 6, 5, 3, 12
    L = rng.normal(size=(B, V)) * 3.0
    E_in = rng.normal(size=(V, H))
    W_out = rng.normal(size=(V, H)) * 0.8
    root = int(rng.integers(V))
    sh = O.draft(L, E_in, W_out, root, B, k, N, mode="shared")
    pa = O.draft(L, E_in, W_out, root, B, k, N, mode="parent")
    assert sh.pool.token[1:1 + k] == pa.pool.token[1:1 + k]
    by_parent = {}
    for i in range(1, len(sh.pool.token)):
        p = sh.pool.parent[i]
        by_parent.setdefault(p, []).append(
            (sh.pool.token[i], sh.pool.s[i] - sh.pool.s[p]))
    for depth in range(1, B):
        lists = [v for p, v in by_parent.items() if sh.pool.depth[p] == depth]
        assert all(lst == lists[0] for lst in lists), depth
