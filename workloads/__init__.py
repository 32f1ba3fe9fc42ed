"""Seeded synthetic inputs for PCTree drafting rounds.

This module is shared by the tests, the benchmark and the smoke check. It holds
no part of the drafting method's arithmetic (no Markov head, no softmax, no
selection): it only draws the inputs a drafting round consumes, with the shapes
and value distributions of Qwen3-shaped DSpark drafters (Sec. 5.1, Table 6;
Appendix A).  Both the oracle and the CUDA path read the arrays made here.

Draw order, per workload and seed (numpy PCG64 via ``SeedSequence(seed)``):

* ``SeedSequence(seed).spawn(1 + batch)``: child 0 draws the Markov-head
  weights, child ``1 + r`` draws everything that belongs to request ``r``.
* head (child 0): ``child0.spawn(2)`` gives one sequence for ``E_in`` and one
  for ``W_out``; each ``[V][H]`` matrix is cut into row chunks of
  ``_CHUNK_ROWS`` rows and chunk ``i`` is drawn from ``seq.spawn(n_chunks)[i]``
  as float32 standard normals times the head scale (chunks are independent,
  so they are drawn in parallel threads); bf16 workloads round each value to
  bf16 (round to nearest even).
* request ``r``: base-logit noise ``[B][V]`` float32 normals; then the
  per-depth structure (planted tokens, or Zipf rank permutations); then the
  per-depth temperature coins (mixed-temperature workloads only); then the
  root token; then, per depth, the target coin and the target's fallback token.

The target's greedy token ``g[r][d]`` (the token the target model wants at
draft depth ``d+1``) is a stand-in for the target model's forward, which is
outside the drafting round: with probability ``target_p`` it is the
generator's own "likely" token for that depth (the planted token, or the
argmax of the base logits ``L_d``), otherwise a uniform token.  A node ``i``
of a drafted tree at depth ``t`` then receives ``target[i] = g[r][t]``.
"""
from __future__ import annotations

import concurrent.futures
import dataclasses
import os
from typing import Dict, Optional

import numpy as np

_CHUNK_ROWS = 8192


@dataclasses.dataclass(frozen=True)
class Workload:
    """One drafting-round workload: shapes, hyper-parameters and input recipe."""

    name: str
    V: int              # vocabulary size |V|
    H: int              # Markov-head rank (hidden size of E_in / W_out)
    B: int              # block size = number of sequential Markov stages
    k: int              # local branching factor (per-parent top-k, frontier width)
    N: int              # verification node budget, root included
    batch: int          # independent requests drafted together
    weight_dtype: str   # "bf16" or "f32"
    logits: str         # "planted", "zipf" or "zipf_mixed_temp"
    head_scale_e: float  # std of E_in entries
    head_scale_w: float  # std of W_out entries
    target_p: float     # probability that the target's token is the likely one
    seed: int
    pos_offset: int = 0  # verified-prefix length added to tree depths
    mode: str = "parent"  # "parent" (PCTree) or "shared" (Shared-Markov)

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    @property
    def pool_size(self) -> int:
        """Candidate pool size, root included: 1 + k + (B-1) k^2 (Sec. 4.1)."""
        return 1 + self.k + (self.B - 1) * self.k * self.k

    def describe(self) -> Dict[str, object]:
        return {
            "workload": self.name, "V": self.V, "H": self.H, "B": self.B,
            "k": self.k, "N": self.N, "batch": self.batch,
            "weights": self.weight_dtype, "logits": self.logits,
        }


def _tiny() -> Workload:
    H = 64
    return Workload("tiny_V1024_H64_B4_k4_N8", V=1024, H=H, B=4, k=4, N=8,
                    batch=1, weight_dtype="f32", logits="planted",
                    head_scale_e=1.0, head_scale_w=2.0 / np.sqrt(H),
                    target_p=0.8, seed=0)


WORKLOADS: Dict[str, Workload] = {
    # small case the oracle finishes in milliseconds
    "tiny": _tiny(),
    # Qwen3-4B-shaped drafting rounds (V of the Qwen3 tokenizer, H=2560)
    "4b_b7": Workload("qwen3_4b_V151936_H2560_B7_k8_N32_bs1", V=151936,
                      H=2560, B=7, k=8, N=32, batch=1, weight_dtype="bf16",
                      logits="zipf", head_scale_e=0.02, head_scale_w=0.02,
                      target_p=0.85, seed=1),
    "4b_b16": Workload("qwen3_4b_V151936_H2560_B16_k8_N64_bs1", V=151936,
                       H=2560, B=16, k=8, N=64, batch=1, weight_dtype="bf16",
                       logits="zipf", head_scale_e=0.02, head_scale_w=0.02,
                       target_p=0.85, seed=2),
    # DSpark-chain control on the same inputs as 4b_b16 (k=1)
    "4b_b16_chain": Workload("qwen3_4b_V151936_H2560_B16_k1_N16_bs1_chain",
                             V=151936, H=2560, B=16, k=1, N=16, batch=1,
                             weight_dtype="bf16", logits="zipf",
                             head_scale_e=0.02, head_scale_w=0.02,
                             target_p=0.85, seed=2),
    # Qwen3-8B-shaped batched serving round
    "8b_b7_bs16": Workload("qwen3_8b_V151936_H4096_B7_k8_N64_bs16", V=151936,
                           H=4096, B=7, k=8, N=64, batch=16,
                           weight_dtype="bf16", logits="zipf",
                           head_scale_e=0.02, head_scale_w=0.02,
                           target_p=0.85, seed=3),
    # Qwen3-14B-shaped stress round (flat and peaked rows mixed per depth)
    "14b_b16_bs32": Workload("qwen3_14b_V151936_H5120_B16_k16_N128_bs32",
                             V=151936, H=5120, B=16, k=16, N=128, batch=32,
                             weight_dtype="bf16", logits="zipf_mixed_temp",
                             head_scale_e=0.02, head_scale_w=0.02,
                             target_p=0.85, seed=4),
}


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); return the bits."""
    u = np.array(x, dtype=np.float32, copy=True).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    u += np.uint32(0x7FFF)
    u += lsb
    u >>= np.uint32(16)
    return u.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to float32 (exact)."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def _draw_matrix(seq: np.random.SeedSequence, V: int, H: int, scale: float,
                 dtype: str) -> np.ndarray:
    out = np.empty((V, H), dtype=np.uint16 if dtype == "bf16" else np.float32)
    n_chunks = (V + _CHUNK_ROWS - 1) // _CHUNK_ROWS
    seeds = seq.spawn(n_chunks)

    def fill(i: int) -> None:
        r0, r1 = i * _CHUNK_ROWS, min(V, (i + 1) * _CHUNK_ROWS)
        blk = np.random.default_rng(seeds[i]).standard_normal(
            (r1 - r0, H), dtype=np.float32)
        blk *= np.float32(scale)
        out[r0:r1] = f32_to_bf16_bits(blk) if dtype == "bf16" else blk

    workers = max(1, min(n_chunks, os.cpu_count() or 1))
    with concurrent.futures.ThreadPoolExecutor(workers) as ex:
        list(ex.map(fill, range(n_chunks)))
    return out


@dataclasses.dataclass
class RoundInputs:
    """Host arrays for one drafting round (all requests)."""

    wl: Workload
    L: np.ndarray          # [batch][B][V] float32 base logits
    E_in: np.ndarray       # [V][H] uint16 (bf16 bits) or float32
    W_out: np.ndarray      # [V][H] uint16 (bf16 bits) or float32
    root: np.ndarray       # [batch] int32
    greedy: np.ndarray     # [batch][B+1] int32: target's token after depth t
    likely: np.ndarray     # [batch][B] int32: generator's likely token per depth


def draw_head(wl: Workload, seed: Optional[int] = None):
    """Markov-head weights ``(E_in, W_out)`` for a workload."""
    ss = np.random.SeedSequence(wl.seed if seed is None else seed)
    seq_e, seq_w = ss.spawn(1 + wl.batch)[0].spawn(2)
    E_in = _draw_matrix(seq_e, wl.V, wl.H, wl.head_scale_e, wl.weight_dtype)
    W_out = _draw_matrix(seq_w, wl.V, wl.H, wl.head_scale_w, wl.weight_dtype)
    return E_in, W_out


def draw_request(wl: Workload, r: int, seed: Optional[int] = None):
    """Base logits, root token and target tokens of request ``r``.

    Returns ``(L [B][V] f32, root, greedy [B+1], likely [B])``; ``greedy[t]``
    is the target's token after a node at depth ``t`` (``t = 0`` is the root).
    """
    ss = np.random.SeedSequence(wl.seed if seed is None else seed)
    rng = np.random.default_rng(ss.spawn(1 + wl.batch)[1 + r])
    B, V = wl.B, wl.V
    noise = rng.standard_normal((B, V), dtype=np.float32)
    if wl.logits == "planted":
        # 3 N(0,1) with a +6 spike at one uniformly drawn token per depth
        L = noise * np.float32(3.0)
        likely = rng.integers(0, V, size=B)
        L[np.arange(B), likely] += np.float32(6.0)
    elif wl.logits in ("zipf", "zipf_mixed_temp"):
        # 4 N(0,1) plus a Zipf(s=1.1) log-rank boost, ranks a random
        # permutation per depth: boost(v) = -1.1 ln rank_d(v)
        L = noise * np.float32(4.0)
        for d in range(B):
            rank = rng.permutation(V).astype(np.float32) + np.float32(1.0)
            L[d] -= np.float32(1.1) * np.log(rank)
        if wl.logits == "zipf_mixed_temp":
            # per depth: flat rows (temperature 2.0) or peaked (0.3), 50/50
            flat = rng.random(B) < 0.5
            temp = np.where(flat, np.float32(2.0), np.float32(0.3))
            L = L / temp[:, None].astype(np.float32)
        likely = np.argmax(L, axis=1)
    else:
        raise ValueError(f"unknown logits recipe {wl.logits!r}")
    root = int(rng.integers(0, V))
    coin = rng.random(B) < wl.target_p
    fallback = rng.integers(0, V, size=B + 1)
    # entry B is the token after a fully drafted block (bonus position)
    greedy = np.concatenate([np.where(coin, likely, fallback[:B]),
                             fallback[B:]])
    return (np.ascontiguousarray(L, dtype=np.float32), root,
            greedy.astype(np.int32), likely.astype(np.int32))


def draw_round(wl: Workload, seed: Optional[int] = None,
               requests: Optional[range] = None) -> RoundInputs:
    """All inputs of one drafting round.  ``requests`` limits the requests
    drawn (the head is always drawn in full)."""
    E_in, W_out = draw_head(wl, seed)
    reqs = range(wl.batch) if requests is None else requests
    Ls, roots, greedy, likely = [], [], [], []
    for r in reqs:
        L, root, g, lk = draw_request(wl, r, seed)
        Ls.append(L)
        roots.append(root)
        greedy.append(g)
        likely.append(lk)
    return RoundInputs(wl, np.stack(Ls), E_in, W_out,
                       np.asarray(roots, dtype=np.int32),
                       np.stack(greedy), np.stack(likely))


def target_for_tree(greedy: np.ndarray, depth: np.ndarray) -> np.ndarray:
    """Per-node target tokens of a drafted tree: ``target[i] = g[depth[i]]``.

    ``greedy`` is ``[batch][B+1]``, ``depth`` is ``[batch][N]`` (-1 for
    unused rows, which receive -1).
    """
    out = np.full(depth.shape, -1, dtype=np.int32)
    for r in range(depth.shape[0]):
        valid = (depth[r] >= 0) & (depth[r] < greedy.shape[1])
        out[r, valid] = greedy[r, depth[r, valid]]
    return out


# ----------------------------------------------------------------------------
# accepted-row compaction inputs (caches after a tree verification)
# ----------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class CompactWorkload:
    """Shapes of the per-token caches a verification forward leaves behind.

    A cache plane holds one row of ``row_bytes`` per (request, slot); each
    layer has ``planes`` of them (K and V).  ``hidden_bytes`` is one target
    hidden-state row.  Slots per request: ``prefix_max + N``.
    """

    name: str
    layers: int
    planes: int
    row_bytes: int
    hidden_bytes: int
    B: int
    N: int
    batch: int
    prefix_max: int
    seed: int

    @property
    def slots(self) -> int:
        return self.prefix_max + self.N

    def cache_bytes(self) -> int:
        return self.layers * self.planes * self.batch * self.slots * self.row_bytes


# Qwen3 KV shapes: 8 KV heads x head_dim 128 in bf16 = 2048 bytes per token
# and plane; 36 layers (4B, 8B) or 40 (14B); hidden 2560 / 4096 / 5120 bf16.
COMPACT_WORKLOADS: Dict[str, CompactWorkload] = {
    "small": CompactWorkload("small_L3_row64_B5_N16_bs3", layers=3, planes=2,
                             row_bytes=64, hidden_bytes=96, B=5, N=16,
                             batch=3, prefix_max=40, seed=20),
    "ragged": CompactWorkload("ragged_L2_row16_B9_N12_bs5", layers=2,
                              planes=3, row_bytes=16, hidden_bytes=32, B=9,
                              N=12, batch=5, prefix_max=7, seed=21),
    "4b_b16": CompactWorkload("qwen3_4b_L36_kv2048_B16_N64_bs1", layers=36,
                              planes=2, row_bytes=2048, hidden_bytes=5120,
                              B=16, N=64, batch=1, prefix_max=2048, seed=22),
    "8b_b7_bs16": CompactWorkload("qwen3_8b_L36_kv2048_B7_N64_bs16",
                                  layers=36, planes=2, row_bytes=2048,
                                  hidden_bytes=8192, B=7, N=64, batch=16,
                                  prefix_max=1024, seed=23),
    "14b_b16_bs32": CompactWorkload("qwen3_14b_L40_kv2048_B16_N128_bs32",
                                    layers=40, planes=2, row_bytes=2048,
                                    hidden_bytes=10240, B=16, N=128,
                                    batch=32, prefix_max=1024, seed=24),
}


@dataclasses.dataclass
class CompactInputs:
    cw: CompactWorkload
    accepted_idx: np.ndarray   # [batch][B+1] int32, -1 padded
    accepted_len: np.ndarray   # [batch] int32
    prefix_len: np.ndarray     # [batch] int32
    cache: Optional[np.ndarray]       # uint8 [layers][planes][batch][slots][row]
    hidden_in: Optional[np.ndarray]   # uint8 [batch][N][hidden_bytes]
    hidden_out: Optional[np.ndarray]  # uint8 [batch][B+1][hidden_bytes]


def draw_accepted_paths(cw: CompactWorkload, rng: np.random.Generator):
    """Accepted paths as the greedy tree rule returns them: the root (0)
    followed by ``len`` strictly increasing packed indices below N, -1
    padded.  Lengths mix 0, B (capped at N-1) and uniform values."""
    B, N = cw.B, cw.N
    top = min(B, N - 1)
    acc = np.full((cw.batch, B + 1), -1, dtype=np.int32)
    lens = np.zeros(cw.batch, dtype=np.int32)
    for r in range(cw.batch):
        u = rng.random()
        n = 0 if u < 0.1 else top if u < 0.2 else int(rng.integers(1, top + 1))
        nodes = np.sort(rng.choice(np.arange(1, N), size=n, replace=False))
        acc[r, 0] = 0
        acc[r, 1:n + 1] = nodes
        lens[r] = n
    return acc, lens


def draw_compaction(cw: CompactWorkload, seed: Optional[int] = None,
                    fill: bool = True) -> CompactInputs:
    """Seeded compaction inputs.  Request 0 has the longest prefix allowed
    (its tree ends at the last slot) and request 1, if any, an empty one.
    ``fill=False`` skips the random cache and hidden-state bytes."""
    ss = np.random.SeedSequence(cw.seed if seed is None else seed)
    s_path, s_cache, s_hid = ss.spawn(3)
    rng = np.random.default_rng(s_path)
    acc, lens = draw_accepted_paths(cw, rng)
    prefix = rng.integers(0, cw.prefix_max + 1, size=cw.batch).astype(np.int32)
    prefix[0] = cw.prefix_max
    if cw.batch > 1:
        prefix[1] = 0
    cache = hid_in = hid_out = None
    if fill:
        shape = (cw.layers, cw.planes, cw.batch, cw.slots, cw.row_bytes)
        cache = np.random.default_rng(s_cache).integers(
            0, 256, size=shape, dtype=np.uint8)
        g = np.random.default_rng(s_hid)
        hid_in = g.integers(0, 256, size=(cw.batch, cw.N, cw.hidden_bytes),
                            dtype=np.uint8)
        hid_out = g.integers(0, 256, size=(cw.batch, cw.B + 1, cw.hidden_bytes),
                             dtype=np.uint8)
    return CompactInputs(cw, acc, lens, prefix, cache, hid_in, hid_out)


# ----------------------------------------------------------------------------
# tree-verification attention inputs (one target layer)
# ----------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class AttnWorkload:
    """One attention layer of the target's tree-verification forward:
    ``Hq`` query heads sharing ``Hkv`` KV heads of size ``D``; ``N`` tree
    nodes of depth at most ``B`` after a prefix of up to ``prefix_max``."""

    name: str
    batch: int
    N: int
    Hq: int
    Hkv: int
    D: int
    B: int
    prefix_max: int
    seed: int
    q_scale: float = 1.5
    k_scale: float = 1.5

    @property
    def slots(self) -> int:
        return self.prefix_max + self.N


ATTN_WORKLOADS: Dict[str, AttnWorkload] = {
    "small": AttnWorkload("small_bs2_N16_Hq8_Hkv2", batch=2, N=16, Hq=8,
                          Hkv=2, D=128, B=5, prefix_max=200, seed=40),
    "ragged": AttnWorkload("ragged_bs3_N24_Hq10_Hkv2", batch=3, N=24, Hq=10,
                           Hkv=2, D=128, B=7, prefix_max=70, seed=41),
    # Qwen3 attention shapes: 32 query / 8 KV heads (4B, 8B), 40 / 8 (14B),
    # head_dim 128; the trees of the drafting workloads
    "4b_b16": AttnWorkload("qwen3_4b_Hq32_Hkv8_D128_N64_B16_bs1", batch=1,
                           N=64, Hq=32, Hkv=8, D=128, B=16, prefix_max=2048,
                           seed=42),
    "8b_b7_bs16": AttnWorkload("qwen3_8b_Hq32_Hkv8_D128_N64_B7_bs16",
                               batch=16, N=64, Hq=32, Hkv=8, D=128, B=7,
                               prefix_max=1024, seed=43),
    "14b_b16_bs32": AttnWorkload("qwen3_14b_Hq40_Hkv8_D128_N128_B16_bs32",
                                 batch=32, N=128, Hq=40, Hkv=8, D=128, B=16,
                                 prefix_max=1024, seed=44),
}


@dataclasses.dataclass
class AttnInputs:
    aw: AttnWorkload
    q: np.ndarray            # bf16 bits [batch][N][Hq][D]
    k: np.ndarray            # bf16 bits [batch][slots][Hkv][D]
    v: np.ndarray            # bf16 bits [batch][slots][Hkv][D]
    prefix_len: np.ndarray   # [batch] int32
    n_nodes: np.ndarray      # [batch] int32
    parent: np.ndarray       # [batch][N] int32, -1 at the root and padding


def draw_tree_parents(N: int, B: int, rng: np.random.Generator):
    """A random tree in breadth-first packed order: node 0 is the root,
    every other node's parent is an earlier node of depth < B, picked with
    weight favouring shallow nodes (bushy near the root, like budgeted
    drafting trees).  Returns ``(n_nodes, parent [N])``."""
    n = int(rng.integers(max(1, N // 2), N + 1))
    parent = np.full(N, -1, dtype=np.int32)
    depth = np.zeros(N, dtype=np.int64)
    for i in range(1, n):
        cand = np.flatnonzero(depth[:i] < B)
        w = 1.0 / (1.0 + depth[cand]) ** 2
        p = int(rng.choice(cand, p=w / w.sum()))
        parent[i] = p
        depth[i] = depth[p] + 1
    # breadth-first packing: parents before children, depth non-decreasing
    order = sorted(range(n), key=lambda i: (depth[i], i))
    pos = {old: new for new, old in enumerate(order)}
    out = np.full(N, -1, dtype=np.int32)
    for old in order[1:]:
        out[pos[old]] = pos[int(parent[old])]
    return n, out


def draw_attention(aw: AttnWorkload, seed: Optional[int] = None,
                   fill: bool = True) -> AttnInputs:
    """Seeded inputs of one tree-verification attention layer.  Request 0
    has the longest prefix allowed, request 1 (if any) an empty one; Q, K,
    V are normal with the workload's scales, rounded to bf16; cache slots
    past a request's tree hold random values too (they must be ignored)."""
    ss = np.random.SeedSequence(aw.seed if seed is None else seed)
    s_tree, s_q, s_k, s_v = ss.spawn(4)
    rng = np.random.default_rng(s_tree)
    prefix = rng.integers(0, aw.prefix_max + 1, size=aw.batch).astype(np.int32)
    prefix[0] = aw.prefix_max
    if aw.batch > 1:
        prefix[1] = 0
    n_nodes = np.zeros(aw.batch, dtype=np.int32)
    parent = np.full((aw.batch, aw.N), -1, dtype=np.int32)
    for r in range(aw.batch):           # request 0 fills the node budget
        draw = _full_tree if r == 0 else draw_tree_parents
        n_nodes[r], parent[r] = draw(aw.N, aw.B, rng)
    q = k = v = None
    if fill:
        def normal(seq, shape, scale):
            rows = int(np.prod(shape[:-1]))
            return _draw_matrix(seq, rows, shape[-1], scale, "bf16").reshape(shape)
        q = normal(s_q, (aw.batch, aw.N, aw.Hq, aw.D), aw.q_scale)
        k = normal(s_k, (aw.batch, aw.slots, aw.Hkv, aw.D), aw.k_scale)
        v = normal(s_v, (aw.batch, aw.slots, aw.Hkv, aw.D), 1.0)
    return AttnInputs(aw, q, k, v, prefix, n_nodes, parent)


def _full_tree(N: int, B: int, rng: np.random.Generator):
    while True:
        n, par = draw_tree_parents(N, B, rng)
        if n == N:
            return n, par
