"""PCTree drafting-round oracle.  TEST INFRASTRUCTURE ONLY.

A plain, slow, float64 restatement of one PCTree drafting round, written from
the paper: the parent-conditioned Markov expansion (Sec. 4.1, Eqs. 2-4) and
the Shared-Markov control of the mechanism study (Sec. 5.3), the
layer-wise frontier pruning and global budgeted selection (Sec. 4.1-4.2,
Algorithm 1), the tree tensors (Sec. 4.2; Appendix A "Tensor implementation")
and the greedy tree acceptance (Sec. 4.2; Appendix A).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
and reference legs may import this module.  It shares no code with the CUDA
library: it neither imports it nor is imported by it.

Readings of the paper taken here (each also listed in the design notes):

* Markov head.  The paper calls it a low-rank head that adds a bias fixed by
  the preceding token (Sec. 3.2) and names its cost "the Markov projection"
  (Sec. 5.6).  Reading: ``Markov(p) = W_out @ E_in[p]`` with
  ``E_in, W_out`` both ``[V][H]``, a rank-``H`` factorisation of a V x V
  bigram bias; no nonlinearity, no scale.
* Per-parent top-k ties: ``(log pi desc, token id asc)``.
* Stable node ids: creation order.  Root 0; then layer by layer; inside a
  layer, the parent's frontier slot major and the child's rank minor.
* Frontier: the ``k`` best nodes of the layer just created (Algorithm 1),
  ranked by ``(score desc, id asc)``.
* Global selection: ``(score desc, depth asc, id asc)``, ``N`` nodes with the
  root, ``n_nodes = min(N, pool size)``.
* Packing order (unspecified in the paper): breadth first, i.e. by
  ``(depth asc, parent's packed index asc, token asc)``; root at 0.
* Acceptance: retrieve rows are compared child by child against the target's
  token at the preceding node; the longest accepted row wins (first such row
  on ties; the accepted node sequence is unique since siblings carry distinct
  tokens).  ``tau = accepted_len + 1`` counts the bonus token (Sec. 5.1).
* Unused output rows (fewer than N pool nodes): token / parent / depth /
  position id -1, logp -inf, mask 0, retrieve -1.
* Non-finite inputs: NaN or +inf base logits, a depth whose logits are all
  -inf, or head weights that make a stage logit NaN or infinite where the
  base logit is finite, raise ``NonFiniteInput``; -inf base logits are legal
  (probability 0).

Replay of near-tie decisions.  The CUDA path computes in float32 and so can
order two candidates differently from this float64 oracle when their values
differ by less than the float32 error.  ``draft`` therefore accepts an
optional ``hint`` (the other implementation's choices, see ``Choices``): at
every decision (each parent's top-k list, each frontier, the global top-N) the
hinted choice is adopted only if it is a valid choice under a relaxation of
``delta`` -- every kept candidate is at least every dropped candidate minus
``delta``, and consecutive kept candidates are ordered within ``delta`` --
and ``ParityViolation`` is raised otherwise.  Adopted choices that differ from
the oracle's own are counted in ``n_ambiguous``.  With no hint the oracle
takes only its own decisions.

Pins (tests/test_oracle_pins.py): every function below is pinned against
something other than itself -- exact rational arithmetic on bigram heads with
brute-force enumeration of all paths (Eqs. 2-4, selection), a closed-form
greedy chain for k=1 (Sec. 4.2), one-hot heads (Markov projection), constant
rows (log-softmax), hand-derived pruning and tie examples, structural
invariants of the mask / positions / retrieve rows, and acceptance on
constructed targets.  No function here is "parity unpinned".
"""
from __future__ import annotations

import concurrent.futures
import dataclasses
import math
import os
from typing import Dict, List, Optional, Sequence, Set, Tuple

import numpy as np

#: decision slack: twice the 1e-4 absolute tolerance on cumulative log-probs
DELTA = 2e-4

Path = Tuple[int, ...]


class NonFiniteInput(ValueError):
    """NaN / +inf input, or a depth with no finite logit."""


class ParityViolation(AssertionError):
    """A hinted choice is not a valid choice within the decision slack."""


# ----------------------------------------------------------------------------
# number formats
# ----------------------------------------------------------------------------

def decode_bf16(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64.  bf16 is the top half of an
    IEEE binary32, so shifting the pattern left by 16 bits is exact.  Large
    arrays are decoded in independent slices on several threads."""
    src = np.ascontiguousarray(bits, dtype=np.uint16)
    out = np.empty(src.shape, dtype=np.float64)
    fin, fout = src.reshape(-1), out.reshape(-1)
    step = 1 << 22

    def part(i: int) -> None:
        sl = slice(i, min(i + step, fin.size))
        wide = fin[sl].astype(np.uint32) << np.uint32(16)
        fout[sl] = wide.view(np.float32)

    starts = range(0, fin.size, step)
    if len(starts) <= 1:
        for i in starts:
            part(i)
    else:
        with concurrent.futures.ThreadPoolExecutor(os.cpu_count() or 1) as ex:
            list(ex.map(part, starts))
    return out


def as_f64(w: np.ndarray, dtype: str) -> np.ndarray:
    """Head weights in the caller's storage format -> float64."""
    if dtype == "bf16":
        return decode_bf16(w)
    if dtype == "f32":
        return np.asarray(w, dtype=np.float32).astype(np.float64)
    raise ValueError(dtype)


def _values(a: np.ndarray) -> np.ndarray:
    """float64 values of an array stored as bf16 bits (uint16) or floats."""
    if a.dtype == np.uint16:
        return decode_bf16(a)
    return np.asarray(a, dtype=np.float64)


# ----------------------------------------------------------------------------
# Eq. 3: one batched Markov call; Eq. 2: log-softmax
# ----------------------------------------------------------------------------

def markov_bias(E_in: np.ndarray, W_out: np.ndarray,
                parents: Sequence[int]) -> np.ndarray:
    """Markov(P) for the stacked parent tokens P (Eq. 3): one row per parent,
    ``Markov(p)[v] = sum_h W_out[v, h] * E_in[p, h]``.  Weights may be given
    as bf16 bits (uint16) or floats; the product is taken in float64."""
    X = _values(E_in[np.asarray(parents, dtype=np.int64)])   # [b][H]
    return X @ _values(W_out).T                               # [b][V]


def stage_logits(L_d: np.ndarray, E_in: np.ndarray, W_out: np.ndarray,
                 parents: Sequence[int]) -> np.ndarray:
    """Z_d = 1 L_d^T + Markov(P_{d-1})  (Eq. 3), float64 ``[b][V]``."""
    return L_d.astype(np.float64)[None, :] + markov_bias(E_in, W_out, parents)


def log_softmax(z: np.ndarray) -> Tuple[np.ndarray, float]:
    """log pi = z - lse, lse = m + log(sum exp(z - m)), m = max z (Eq. 2)."""
    m = float(np.max(z))
    if not math.isfinite(m):
        raise NonFiniteInput("no finite logit in a row")
    lse = m + math.log(float(np.sum(np.exp(z - m))))
    return z - lse, lse


# ----------------------------------------------------------------------------
# the three ranked decisions
# ----------------------------------------------------------------------------

def local_topk(z: np.ndarray, k: int) -> List[int]:
    """The k children of one parent: tokens by (z desc, token asc)."""
    order = np.lexsort((np.arange(z.shape[0]), -z))
    return [int(v) for v in order[:k]]


def layer_frontier(layer_ids: Sequence[int], s: Sequence[float],
                   k: int) -> List[int]:
    """Next frontier: the k best nodes of the current layer by
    (score desc, id asc) (Algorithm 1, frontier step)."""
    return sorted(layer_ids, key=lambda i: (-s[i], i))[:k]


def global_topn(s: Sequence[float], depth: Sequence[int], N: int) -> List[int]:
    """Budgeted selection: N pool nodes by (score desc, depth asc, id asc)
    (Sec. 4.2, Algorithm 1)."""
    return sorted(range(len(s)), key=lambda i: (-s[i], depth[i], i))[:N]


def _margin(sorted_vals: Sequence[float], m: int) -> float:
    """Gap between the last kept and the first dropped value."""
    if m >= len(sorted_vals) or m == 0:
        return math.inf
    a, b = sorted_vals[m - 1], sorted_vals[m]
    if a == b:
        return 0.0
    return a - b


def _order_margin(sorted_vals: Sequence[float], m: int) -> float:
    """Smallest of the cut gap and the gaps between consecutive kept values:
    how far this decision is from one whose kept set or order differs."""
    gaps = [_margin(sorted_vals, m)]
    top = list(sorted_vals[:m])
    gaps += [0.0 if a == b else a - b for a, b in zip(top, top[1:])]
    return min(gaps)


def _check_choice(name: str, chosen: Sequence, candidates: Sequence,
                  val: Dict, delta: float, ordered: bool) -> None:
    """Raise unless ``chosen`` is a valid top-|chosen| of ``candidates``
    under a slack of ``delta`` (and, if ``ordered``, in valid order)."""
    cset = set(chosen)
    if len(cset) != len(chosen):
        raise ParityViolation(f"{name}: repeated element in {chosen}")
    if not cset.issubset(set(candidates)):
        raise ParityViolation(f"{name}: {sorted(cset - set(candidates))} "
                              "are not candidates")
    dropped = [c for c in candidates if c not in cset]
    if dropped and chosen:
        lo = min(val[c] for c in chosen)
        hi = max(val[c] for c in dropped)
        if not lo >= hi - delta:
            raise ParityViolation(
                f"{name}: kept value {lo!r} is below dropped value {hi!r} "
                f"by more than {delta}")
    if ordered:
        for a, b in zip(chosen, chosen[1:]):
            if not val[a] >= val[b] - delta:
                raise ParityViolation(
                    f"{name}: order {a}->{b} has {val[a]!r} < {val[b]!r} "
                    f"- {delta}")


# ----------------------------------------------------------------------------
# choices of another implementation, for near-tie replay
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class Choices:
    """Decisions of another implementation of one round, keyed by token paths
    (a node's tokens from depth 1 down to itself; the root is ``()``)."""

    children: Dict[Path, List[int]]     # parent path -> child tokens, by rank
    frontier: Dict[int, List[Path]]     # layer depth -> frontier paths, by slot
    selected: Set[Path]                 # kept node paths


def choices_from_pool(pool_token: Sequence[int], pool_parent: Sequence[int],
                      n_pool: int, selected_paths: Set[Path]) -> Choices:
    """Rebuild the decisions from a candidate pool listed in id order
    (``pool_parent[i]`` the parent's id, -1 for the root).  A parent's
    children appear in rank order; a layer's frontier is the order in which
    its nodes first appear as parents of the next layer."""
    paths: List[Path] = []
    depth: List[int] = []
    children: Dict[Path, List[int]] = {}
    frontier: Dict[int, List[Path]] = {}
    for i in range(n_pool):
        p = int(pool_parent[i])
        if i == 0:
            if p != -1:
                raise ParityViolation("pool node 0 is not the root")
            paths.append(())
            depth.append(0)
            continue
        if not 0 <= p < i:
            raise ParityViolation(f"pool node {i} has parent {p}")
        path = paths[p] + (int(pool_token[i]),)
        paths.append(path)
        depth.append(depth[p] + 1)
        children.setdefault(paths[p], []).append(int(pool_token[i]))
        layer = frontier.setdefault(depth[p], [])
        if paths[p] not in layer:
            layer.append(paths[p])
    return Choices(children, frontier, set(selected_paths))


# ----------------------------------------------------------------------------
# one request's drafting round (Algorithm 1)
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class Pool:
    token: List[int]
    parent: List[int]
    depth: List[int]
    s: List[float]
    path: List[Path]


@dataclasses.dataclass
class Tree:
    """Packed tree of one request (fixed-size arrays with N rows)."""

    n_nodes: int
    tokens: np.ndarray        # [N] int32
    parent: np.ndarray        # [N] int32, packed index of the parent
    depth: np.ndarray         # [N] int32
    logp: np.ndarray          # [N] float64, cumulative joint log-prob
    position_ids: np.ndarray  # [N] int32
    mask: np.ndarray          # [N][N] uint8, 1 iff column is ancestor-or-self
    retrieve: np.ndarray      # [N][B+1] int32, root-to-leaf packed indices
    n_leaves: int


@dataclasses.dataclass
class Round:
    pool: Pool
    selected: List[int]       # pool ids, in packed order
    tree: Tree
    n_ambiguous: int          # adopted hinted choices that differ from ours
    margins: Dict[str, float]  # smallest own margin per decision kind
    markov_calls: List[int]   # batch size b_d of each Markov call
    # per adopted differing choice: (decision kind, our own margin there --
    # the smaller of the cut gap and the gaps between consecutive kept values
    # for ordered decisions, the cut gap for the unordered global selection)
    adopted: List[Tuple[str, float]] = dataclasses.field(default_factory=list)


def _check_logits(L: np.ndarray) -> None:
    if np.isnan(L).any() or np.isposinf(L).any():
        raise NonFiniteInput("base logits hold NaN or +inf")
    if not np.isfinite(L).any(axis=1).all():
        raise NonFiniteInput("a depth has no finite base logit")


def _check_stage(Z: np.ndarray, L_d: np.ndarray) -> None:
    """A non-finite head weight shows up as a NaN / infinite stage logit where
    the base logit is finite."""
    bad = np.isnan(Z) | (np.isinf(Z) & np.isfinite(L_d)[None, :]) | np.isposinf(Z)
    if bad.any():
        raise NonFiniteInput("non-finite Markov bias")


MODES = ("parent", "shared")


def draft(L: np.ndarray, E_in: np.ndarray, W_out: np.ndarray, root: int,
          B: int, k: int, N: int, pos_offset: int = 0,
          hint: Optional[Choices] = None, delta: float = DELTA,
          mode: str = "parent") -> Round:
    """One drafting round for one request.

    ``mode="parent"``: PCTree -- every frontier parent gets its own Markov
    bias (Eqs. 2-3).  ``mode="shared"``: the Shared-Markov tree of the
    mechanism study (Sec. 5.3): the greedy DSpark chain of Eq. 1 is built
    alongside, and its distribution q_d at depth d serves every parent at
    that depth; frontier, budget, selection and packing are unchanged.

    ``L`` is ``[B][V]`` (float32 or float64); ``E_in``/``W_out`` are ``[V][H]``
    as floats or bf16 bits (uint16; pass ``W_out`` pre-decoded with
    ``as_f64`` to decode it once for many rounds).  Returns the candidate
    pool, the selection and the packed tree.
    """
    V = L.shape[1]
    if not (1 <= k <= V and N >= 1 and B >= 1 and 0 <= root < V):
        raise ValueError("invalid round parameters")
    if mode not in MODES:
        raise ValueError(mode)
    _check_logits(np.asarray(L, dtype=np.float64))
    pool = Pool([root], [-1], [0], [0.0], [()])       # root: score 0, id 0
    frontier = [0]
    chain = root                                      # greedy chain (shared)
    margins = {"children": math.inf, "frontier": math.inf, "global": math.inf}
    n_amb = 0
    adopted: List[Tuple[str, float]] = []
    calls = []
    for d in range(B):                                # stage d builds level d+1
        if mode == "shared":
            parents = [chain]                         # one batch-1 call, Eq. 1
        else:
            parents = [pool.token[i] for i in frontier]
        calls.append(len(parents))
        Z = stage_logits(L[d], E_in, W_out, parents)  # one batched call, Eq. 3
        _check_stage(Z, L[d])
        layer: List[int] = []
        first_kids: List[int] = []
        for slot, pid in enumerate(frontier):
            z = Z[0 if mode == "shared" else slot]
            logpi, _ = log_softmax(z)                 # Eq. 2
            mine = local_topk(z, k)
            zs = np.sort(z)[::-1]
            margins["children"] = min(margins["children"], _margin(zs, k))
            kids = mine
            if hint is not None:
                theirs = hint.children.get(pool.path[pid])
                if theirs is None:
                    raise ParityViolation(
                        f"no children for parent {pool.path[pid]}")
                zval = {v: float(z[v]) for v in set(theirs) | set(mine)}
                if list(theirs) != mine:
                    # every token is a candidate; only near-cut ones matter
                    cut = float(zs[min(k, V - 1)])
                    cands = sorted(set(theirs) | set(mine) |
                                   {int(v) for v in np.nonzero(z >= cut - delta)[0]})
                    for v in cands:
                        zval[v] = float(z[v])
                    _check_choice(f"children of {pool.path[pid]}", theirs,
                                  cands, zval, delta, ordered=True)
                    n_amb += 1
                    adopted.append(("children", _order_margin(zs, k)))
                    kids = list(theirs)
            if slot == 0:
                first_kids = list(kids)
            for v in kids:                            # Eq. 4, pushed to pool
                pool.token.append(v)
                pool.parent.append(pid)
                pool.depth.append(d + 1)
                pool.s.append(pool.s[pid] + float(logpi[v]))
                pool.path.append(pool.path[pid] + (v,))
                layer.append(len(pool.token) - 1)
        if mode == "shared":
            chain = first_kids[0]                     # argmax of q_d (Eq. 1)
        if d < B - 1:
            mine = layer_frontier(layer, pool.s, k)
            ranked = sorted((pool.s[i] for i in layer), reverse=True)
            margins["frontier"] = min(margins["frontier"], _margin(ranked, k))
            frontier = mine
            if hint is not None:
                theirs_p = hint.frontier.get(d + 1)
                if theirs_p is None:
                    raise ParityViolation(f"no frontier for layer {d + 1}")
                by_path = {pool.path[i]: i for i in layer}
                if any(p not in by_path for p in theirs_p):
                    raise ParityViolation(f"frontier of layer {d + 1} names "
                                          "a node outside the layer")
                theirs = [by_path[p] for p in theirs_p]
                if theirs != mine:
                    _check_choice(f"frontier of layer {d + 1}", theirs, layer,
                                  {i: pool.s[i] for i in layer}, delta,
                                  ordered=True)
                    n_amb += 1
                    adopted.append(("frontier", _order_margin(ranked, k)))
                    frontier = theirs
    n_pool = len(pool.token)
    mine = global_topn(pool.s, pool.depth, N)
    ranked = sorted(pool.s, reverse=True)
    margins["global"] = _margin(ranked, min(N, n_pool))
    chosen = mine
    if hint is not None:
        by_path = {pool.path[i]: i for i in range(n_pool)}
        if any(p not in by_path for p in hint.selected):
            raise ParityViolation("selection names a node outside the pool")
        theirs = sorted(by_path[p] for p in hint.selected)
        if set(theirs) != set(mine):
            _check_choice("global selection", theirs, list(range(n_pool)),
                          {i: pool.s[i] for i in range(n_pool)}, delta,
                          ordered=False)
            n_amb += 1
            adopted.append(("global", margins["global"]))
            chosen = theirs
    packed, tree = pack(pool, chosen, N, B, pos_offset)
    return Round(pool, packed, tree, n_amb, margins, calls, adopted)


# ----------------------------------------------------------------------------
# tree tensors (Sec. 4.2; Appendix A "Tensor implementation")
# ----------------------------------------------------------------------------

def pack(pool: Pool, chosen: Sequence[int], N: int, B: int,
         pos_offset: int = 0) -> Tuple[List[int], Tree]:
    """Flat draft tokens, parent indices, depths, scores, position ids,
    ancestor-only mask and retrieve rows of the selected node set."""
    chosen_set = set(chosen)
    for i in chosen:
        if i != 0 and pool.parent[i] not in chosen_set:
            raise ParityViolation(f"selection is not prefix-closed at {i}")
    out_idx: Dict[int, int] = {}
    order: List[int] = []
    by_depth: Dict[int, List[int]] = {}
    for i in chosen:
        by_depth.setdefault(pool.depth[i], []).append(i)
    for t in sorted(by_depth):
        nodes = sorted(by_depth[t], key=lambda i: (
            out_idx.get(pool.parent[i], -1), pool.token[i]))
        for i in nodes:
            out_idx[i] = len(order)
            order.append(i)
    n = len(order)
    tokens = np.full(N, -1, np.int32)
    parent = np.full(N, -1, np.int32)
    depth = np.full(N, -1, np.int32)
    logp = np.full(N, -np.inf, np.float64)
    pos = np.full(N, -1, np.int32)
    mask = np.zeros((N, N), np.uint8)
    retrieve = np.full((N, B + 1), -1, np.int32)
    for a, i in enumerate(order):
        tokens[a] = pool.token[i]
        parent[a] = out_idx[pool.parent[i]] if pool.parent[i] >= 0 else -1
        depth[a] = pool.depth[i]
        logp[a] = pool.s[i]
        pos[a] = pool.depth[i] + pos_offset   # siblings share a position
    for a in range(n):                        # attend to self and ancestors
        b = a
        while b >= 0:
            mask[a, b] = 1
            b = parent[b]
    has_child = np.zeros(N, bool)
    for a in range(1, n):
        has_child[parent[a]] = True
    n_leaves = 0
    for a in range(n):
        if has_child[a]:
            continue
        chain = []
        b = a
        while b >= 0:
            chain.append(b)
            b = parent[b]
        chain.reverse()
        retrieve[n_leaves, :len(chain)] = chain
        n_leaves += 1
    return order, Tree(n, tokens, parent, depth, logp, pos, mask, retrieve,
                       n_leaves)


# ----------------------------------------------------------------------------
# greedy tree acceptance (Sec. 4.2; Appendix A)
# ----------------------------------------------------------------------------

def accept(tree: Tree, target: np.ndarray, B: int) -> Tuple[np.ndarray, int, int]:
    """Longest retrieve row whose every child matches the target's token at
    the preceding node.  Returns ``(accepted [B+1] packed indices incl. the
    root, -1 padded; accepted draft tokens; bonus token)``."""
    best_len, best_row = -1, 0
    for j in range(tree.n_leaves):
        row = tree.retrieve[j]
        a = 0
        while (a + 1 < row.shape[0] and row[a + 1] >= 0 and
               tree.tokens[row[a + 1]] == target[row[a]]):
            a += 1
        if a > best_len:
            best_len, best_row = a, j
    acc = np.full(B + 1, -1, np.int32)
    acc[:best_len + 1] = tree.retrieve[best_row, :best_len + 1]
    bonus = int(target[acc[best_len]])
    return acc, best_len, bonus


# ----------------------------------------------------------------------------
# convenience over a batch of requests
# ----------------------------------------------------------------------------

def draft_batch(L: np.ndarray, E_in: np.ndarray, W_out: np.ndarray,
                roots: Sequence[int], B: int, k: int, N: int,
                pos_offset: int = 0, hints: Optional[Sequence[Choices]] = None,
                delta: float = DELTA, mode: str = "parent") -> List[Round]:
    return [draft(L[r], E_in, W_out, int(roots[r]), B, k, N, pos_offset,
                  None if hints is None else hints[r], delta, mode)
            for r in range(L.shape[0])]
