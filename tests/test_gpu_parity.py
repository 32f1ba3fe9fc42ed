"""CUDA path (through the C ABI) against the oracle, element by element.

Small cases span several 128-row vocabulary tiles with a ragged tail, ragged
K, multi-pass parent batches and the method's degenerate cases; the
full-size cases are the Qwen3-shaped workloads in the launch configuration
the benchmark times (sampled requests where the oracle would be slow).
"""
import functools

import numpy as np
import pytest
import torch

from oracle import pctree_oracle as O
from tests import gpu_util as G
from workloads import WORKLOADS, draw_round

pytestmark = pytest.mark.gpu


def strong(wl, **kw):
    """Head scale of the tiny workload, so that parents change rankings."""
    H = kw.get("H", wl.H)
    return wl.with_(head_scale_e=1.0, head_scale_w=2.0 / np.sqrt(H), **kw)


BASE = WORKLOADS["4b_b16"]
SMALL = {
    "tiny_f32": WORKLOADS["tiny"],
    "ragged_V_bf16": strong(BASE, V=3000, H=256, B=5, k=4, N=16, batch=3, seed=11),
    "ragged_K_bf16": strong(BASE, V=1111, H=72, B=4, k=3, N=12, batch=2, seed=12),
    "multipass_bf16": strong(BASE, V=2000, H=64, B=3, k=8, N=40, batch=40, seed=13),
    "chain_k1_bf16": strong(BASE, V=5000, H=128, B=8, k=1, N=9, batch=2, seed=14),
    "budget1_bf16": strong(BASE, V=700, H=64, B=3, k=4, N=1, batch=2, seed=15),
    "budget_over_pool": strong(BASE, V=700, H=64, B=2, k=3, N=100, batch=2, seed=16),
    "k32_bf16": strong(BASE, V=4096, H=64, B=3, k=32, N=200, batch=1, seed=17),
    "B1_bf16": strong(BASE, V=999, H=64, B=1, k=5, N=4, batch=2, seed=18),
    "weak_head_bf16": BASE.with_(V=20000, H=512, B=6, k=8, N=32, batch=2, seed=19),
    # more W_out tiles than SMs and a ragged K chunk (64 + 64 + 8): the fused
    # round's equal shares cut tiles between neighbouring CTAs
    "cut_tiles_bf16": strong(BASE, V=40000, H=136, B=5, k=8, N=32, batch=1, seed=26),
    "mixed_temp_bf16": strong(WORKLOADS["14b_b16_bs32"], V=6000, H=128, B=6,
                              k=6, N=24, batch=4, seed=20),
    "f32_pos_offset": WORKLOADS["tiny"].with_(V=3001, H=37, B=5, k=3, N=20,
                                              batch=2, seed=21, pos_offset=123),
    # Shared-Markov control (Sec. 5.3)
    "shared_ragged_bf16": strong(BASE, V=3000, H=256, B=5, k=4, N=16, batch=3,
                                 seed=23, mode="shared"),
    "shared_batched_bf16": strong(BASE, V=2000, H=64, B=4, k=8, N=40,
                                  batch=12, seed=24, mode="shared"),
    "shared_f32": WORKLOADS["tiny"].with_(V=1500, H=40, B=4, k=3, N=10,
                                          batch=2, seed=25, mode="shared"),
}


PATHS = {"auto": 0, "stagewise": 1}


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("name", sorted(SMALL))
def test_small_parity(name, path):
    inp = draw_round(SMALL[name])
    host = G.run_gpu(inp, path=PATHS[path])
    rep = G.compare(inp, host)
    print(f"{name}/{path}: " + rep.summary())


def test_many_chunks_merge_scan():
    """An f32 head with more than 160 vocabulary chunks of 8192 logits: the
    per-stage merge takes each row's children by its candidate scan, not by
    the tournament over at most 5 lists per lane that every other case
    uses."""
    wl = WORKLOADS["tiny"].with_(V=1_320_000, H=16, B=3, k=4, N=12, batch=2, seed=27)
    assert -(-wl.V // 8192) > 160
    inp = draw_round(wl)
    host = G.run_gpu(inp)
    rep = G.compare(inp, host)
    print("many_chunks_f32: " + rep.summary())


def test_paths_agree_exactly_on_structure():
    inp = draw_round(SMALL["weak_head_bf16"])
    a = G.run_gpu(inp, path=0)
    b = G.run_gpu(inp, path=1)
    for name in ("tokens", "parent", "depth", "mask", "retrieve", "n_nodes"):
        np.testing.assert_array_equal(a[name], b[name])
    assert np.abs(a["logp"][:, :] - b["logp"][:, :])[np.isfinite(a["logp"])].max() <= 1e-4


def test_second_call_reuses_workspace_cleanly():
    """A second round in the same workspace matches the first and the oracle
    (structure exactly, logp to float32 rounding of the normaliser)."""
    inp = draw_round(SMALL["ragged_V_bf16"])
    a = G.run_gpu(inp)
    b = G.run_gpu(inp)
    for name in ("tokens", "parent", "mask", "retrieve", "depth", "n_nodes"):
        np.testing.assert_array_equal(a[name], b[name])
    fin = np.isfinite(a["logp"])
    np.testing.assert_array_equal(fin, np.isfinite(b["logp"]))
    assert np.abs(a["logp"][fin] - b["logp"][fin]).max() <= 1e-5
    G.compare(inp, a)
    G.compare(inp, b)


def _tie_inputs(dtype):
    V, H = 64, 16
    L = np.zeros((1, 2, V), np.float32)
    L[0, 0, :10] = [4, 4, 2, 2, 2, 0, 0, 0, 0, 0]
    L[0, 0, 10:] = -1
    from workloads import RoundInputs
    wl = BASE.with_(V=V, H=H, B=2, k=3, N=10, batch=1, weight_dtype=dtype)
    zeros = (np.zeros((V, H), np.uint16) if dtype == "bf16"
             else np.zeros((V, H), np.float32))
    ones = (np.full((V, H), 0x3F80, np.uint16) if dtype == "bf16"
            else np.ones((V, H), np.float32))
    return RoundInputs(wl, L, ones, zeros, np.array([7], np.int32),
                       np.zeros((1, 3), np.int32), np.zeros((1, 2), np.int32))


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_planted_ties_exact(dtype, path):
    """Exact ties everywhere: the tie-break rules alone decide, so the GPU
    must equal the oracle's own decisions with no replay."""
    inp = _tie_inputs(dtype)
    host = G.run_gpu(inp, path=PATHS[path])
    G.compare(inp, host, strict=True)
    # root children: tokens 0, 1 (tie at 4, token order), then 2
    assert host["pool_token"][0][1:4].tolist() == [0, 1, 2]


@pytest.mark.parametrize("path", sorted(PATHS))
def test_neg_inf_logits(path):
    wl = strong(BASE, V=300, H=64, B=3, k=4, N=30, batch=1, seed=22)
    inp = draw_round(wl)
    inp.L[0, 0, :] = -np.inf
    inp.L[0, 0, [5, 77]] = [1.0, 0.5]        # two finite children only
    inp.L[0, 1, 100:] = -np.inf
    host = G.run_gpu(inp, path=PATHS[path])
    G.compare(inp, host)
    assert np.isneginf(host["pool_logp"][0]).sum() > 0


@pytest.mark.parametrize("path", sorted(PATHS))
def test_nonfinite_and_bad_root_set_status(path):
    inp = draw_round(SMALL["ragged_V_bf16"])
    inp.L[1, 2, 17] = np.nan
    host = G.run_gpu(inp, accept=False, path=PATHS[path])
    assert int(host["status"][0]) == -5       # PCTREE_ERR_NONFINITE
    inp = draw_round(SMALL["ragged_V_bf16"])
    inp.root[0] = inp.wl.V + 3
    host = G.run_gpu(inp, accept=False, path=PATHS[path])
    assert int(host["status"][0]) == -1       # PCTREE_ERR_INVALID_ARG


def test_host_errors_need_no_work():
    from paper_2608_02123_gb300 import pctree as P
    wl = SMALL["ragged_V_bf16"]
    cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, wl.batch)
    dr = P.Drafter(cfg)
    L, E, W, root = G.device_inputs(draw_round(wl))
    with pytest.raises(P.PctreeError) as ei:
        P.pctree_draft(cfg, L, E, W, root, dr.tree, dr.workspace[:100])
    assert ei.value.code == -2
    with pytest.raises(P.PctreeError) as ei:
        P.pctree_draft(cfg, L, E.view(-1)[1:], W, root, dr.tree,
                       dr.workspace)                       # misaligned E_in
    assert ei.value.code == -1


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("name", ["ragged_V_bf16", "multipass_bf16", "tiny_f32"])
def test_base_logits_in_pinned_host_memory(name, path):
    """Base logits and root tokens in page-locked host memory are read by
    the kernels over the host link, with no copy: the round is the same, bit
    for bit, as from device memory (also through draft_from_host, which
    reads all outputs back with one copy)."""
    from paper_2608_02123_gb300 import pctree as P
    inp = draw_round(SMALL[name])
    wl = inp.wl
    cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, inp.L.shape[0],
                        wl.pos_offset, wl.weight_dtype, wl.mode)
    L, E, W, root = G.device_inputs(inp)
    L_pinned = L.cpu().pin_memory()
    root_pinned = root.cpu().pin_memory()
    assert L_pinned.is_pinned() and root_pinned.is_pinned()
    P.pctree_set_path(PATHS[path])
    try:
        a = P.Drafter(cfg)
        ha = a.draft(L, E, W, root).to_host()
        b = P.Drafter(cfg)
        hb = b.draft(L_pinned, E, W, root_pinned).to_host()
        torch.cuda.synchronize()
        c = P.Drafter(cfg)
        hc = c.draft_from_host(L_pinned, root_pinned, E, W)
    finally:
        P.pctree_set_path(P.PATH_AUTO)
    a.check_status()
    b.check_status()
    for key in ha:
        np.testing.assert_array_equal(ha[key], hb[key], err_msg=key)
        if key in hc:
            np.testing.assert_array_equal(ha[key], hc[key], err_msg=key)


def test_pageable_base_logits_refused():
    """A host pointer CUDA cannot read from the device is refused on the
    host, before any launch."""
    import ctypes
    from paper_2608_02123_gb300 import pctree as P
    wl = SMALL["ragged_V_bf16"]
    cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, wl.batch)
    dr = P.Drafter(cfg)
    _, E, W, root = G.device_inputs(draw_round(wl))
    pageable = np.zeros((wl.batch, wl.B, wl.V), np.float32)
    ts = dr.tree.c_struct()
    rc = P.LIB.pctree_draft(ctypes.byref(cfg), ctypes.c_void_p(pageable.ctypes.data),
                            E.data_ptr(), W.data_ptr(), root.data_ptr(),
                            ctypes.byref(ts), dr.workspace.data_ptr(),
                            dr.workspace.numel(),
                            torch.cuda.current_stream().cuda_stream)
    assert rc == -1
    with pytest.raises(ValueError):
        P.pctree_draft(cfg, torch.from_numpy(pageable), E, W, root, dr.tree,
                       dr.workspace)


# ---------------------------------------------------------------------------
# full-size Qwen3-shaped workloads
# ---------------------------------------------------------------------------

@functools.lru_cache(maxsize=1)
def _full(name, requests=None):
    if name == "4b_b16_shared":
        wl = WORKLOADS["4b_b16"].with_(mode="shared")
        return draw_round(wl)
    wl = WORKLOADS[name]
    reqs = None if requests is None else range(requests)
    return draw_round(wl.with_(batch=wl.batch if requests is None else requests),
                      requests=reqs)


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("name", ["4b_b16", "4b_b16_chain", "4b_b7",
                                  "4b_b16_shared"])
def test_full_size_batch1(name, path):
    inp = _full(name)
    host = G.run_gpu(inp, path=PATHS[path])
    rep = G.compare(inp, host)
    print(f"{name}/{path}: " + rep.summary())


def _flat_depths(L: np.ndarray) -> np.ndarray:
    """Per request, the depths drawn flat (temperature 2.0) rather than
    peaked (0.3) in the mixed-temperature workload: the two differ 6.7x in
    spread, so the row's standard deviation tells them apart."""
    sd = L.std(axis=2)
    return (sd < np.sqrt(sd.min() * sd.max())).sum(axis=1)


def _checked_requests(name: str, inp) -> list:
    """Requests compared element by element.  8B: all 16.  14B: both ends of
    each 256-row projection pass (0, 15 | 16, 31: with 16 Markov rows per
    request, requests 16..31 run in the second pass) and the requests with
    the most flat and the most peaked depths."""
    if name == "8b_b7_bs16":
        return list(range(inp.L.shape[0]))
    flat = _flat_depths(inp.L)
    picks = [0, 15, 16, 31, int(np.argmax(flat)), int(np.argmin(flat))]
    return sorted(set(picks))


@pytest.mark.parametrize("name", ["8b_b7_bs16", "14b_b16_bs32"])
def test_full_size_batched(name):
    """Whole batch on the GPU in the benchmark's launch configuration; the
    oracle checks the requests of ``_checked_requests`` element by element
    (requests are independent) and every request's tree is checked for its
    structural invariants."""
    wl = WORKLOADS[name]
    inp = draw_round(wl)
    host = G.run_gpu(inp)
    reqs = _checked_requests(name, inp)
    rep = G.compare(inp, host, requests=reqs)
    flat = _flat_depths(inp.L) if name == "14b_b16_bs32" else None
    print(f"{name}: checked {reqs} "
          + (f"(flat depths {[int(flat[r]) for r in reqs]} of {wl.B}) "
             if flat is not None else "")
          + rep.summary() + f" adopted={rep.adopted}")
    # every request: structural invariants of its tree
    for r in range(wl.batch):
        n = int(host["n_nodes"][r])
        assert n == min(wl.N, wl.pool_size)
        par = host["parent"][r][:n]
        assert par[0] == -1 and (par[1:] < np.arange(1, n)).all()
        lp = host["logp"][r][:n]
        assert (lp[1:] <= lp[par[1:]]).all()
        assert (host["mask"][r][:n, :n].sum(1) == host["depth"][r][:n] + 1).all()


# ---------------------------------------------------------------------------
# the accept walk on constructed targets (Sec. 4.2 greedy tree rule;
# Appendix A retrieve rows; Sec. 5.1: tau counts the bonus token)
# ---------------------------------------------------------------------------

def _path_to(parent, u):
    path = [u]
    while path[-1] != 0:
        path.append(int(parent[path[-1]]))
    return path[::-1]


def _leave_token(tokens, parent, n, u, V):
    """A vocabulary token that none of node u's children carries."""
    kids = {int(tokens[c]) for c in range(1, n) if parent[c] == u}
    t = (int(tokens[u]) + 1) % V
    while t in kids:
        t = (t + 1) % V
    return t


def _constructed_targets(tokens, parent, n, N, V, seed):
    """Row u < n: the target follows path(u) and then wants, at u, a token
    none of u's children carries (filler tokens elsewhere).  Row n: the
    target misses at the root."""
    rng = np.random.default_rng(seed)
    rows = []
    for u in range(n + 1):
        t = rng.integers(0, V, size=N).astype(np.int32)
        if u < n:
            path = _path_to(parent, u)
            for a, b in zip(path, path[1:]):
                t[a] = tokens[b]
            t[u] = _leave_token(tokens, parent, n, u, V)
        else:
            t[0] = _leave_token(tokens, parent, n, 0, V)
        rows.append(t)
    return np.stack(rows)


def _accept_replicated(cfg_one, host, targets, n_nodes_override=None):
    """pctree_accept over one drafted tree replicated once per target row."""
    from paper_2608_02123_gb300 import pctree as P
    R = targets.shape[0]
    cfg = P.make_config(cfg_one.V, cfg_one.H, cfg_one.B, cfg_one.k, cfg_one.N, R)
    tree = P.alloc_tree(cfg, "cuda")
    n = int(host["n_nodes"][0]) if n_nodes_override is None else n_nodes_override
    tree.n_nodes.fill_(n)
    tree.tokens.copy_(torch.from_numpy(host["tokens"][0]).expand(R, -1))
    tree.parent.copy_(torch.from_numpy(host["parent"][0]).expand(R, -1))
    i32 = dict(dtype=torch.int32, device="cuda")
    acc = torch.full((R, cfg.B + 1), -7, **i32)
    length = torch.full((R,), -7, **i32)
    bonus = torch.full((R,), -7, **i32)
    P.pctree_accept(cfg, tree, torch.from_numpy(targets).cuda(), acc, length,
                    bonus)
    torch.cuda.synchronize()
    return acc.cpu().numpy(), length.cpu().numpy(), bonus.cpu().numpy()


def _oracle_tree(host, r=0):
    return O.Tree(int(host["n_nodes"][r]), host["tokens"][r], host["parent"][r],
                  host["depth"][r], host["logp"][r].astype(np.float64),
                  host["position_ids"][r], host["mask"][r], host["retrieve"][r],
                  int(host["n_leaves"][r]))


def test_accept_constructed_targets_full_size():
    """Every node u of the full-size 4b_b16 tree: a target that follows
    path(u) and leaves the tree at u gives accepted path(u), length depth(u)
    and u's target token as the bonus; an all-miss target accepts nothing.
    One accept launch covers every row (the tree replicated over a batch)."""
    from paper_2608_02123_gb300 import pctree as P
    inp = _full("4b_b16")
    host = G.run_gpu(inp, accept=False)
    wl = inp.wl
    n = int(host["n_nodes"][0])
    targets = _constructed_targets(host["tokens"][0], host["parent"][0], n,
                                   wl.N, wl.V, seed=3)
    cfg1 = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, 1)
    acc, length, bonus = _accept_replicated(cfg1, host, targets)
    t = _oracle_tree(host)
    for u in range(n + 1):
        a_ref, len_ref, b_ref = O.accept(t, targets[u], wl.B)
        np.testing.assert_array_equal(acc[u], a_ref, err_msg=f"row {u}")
        assert int(length[u]) == len_ref and int(bonus[u]) == b_ref, u
        if u < n:
            path = _path_to(host["parent"][0], u)
            assert int(length[u]) == len(path) - 1 == host["depth"][0][u]
            assert acc[u][:len(path)].tolist() == path
            assert int(bonus[u]) == targets[u][u]
        else:
            assert int(length[u]) == 0 and acc[u][0] == 0
            assert (acc[u][1:] == -1).all()


def test_accept_full_depth_chain():
    """A chain drafted to full depth (k = 1, N = B + 1 on the 4b_b16 inputs):
    the target that follows it accepts all B tokens and returns the token
    after the leaf as the bonus (tau = B + 1)."""
    import dataclasses
    from paper_2608_02123_gb300 import pctree as P
    base = _full("4b_b16")
    wl = base.wl.with_(k=1, N=base.wl.B + 1)
    inp = dataclasses.replace(base, wl=wl)
    host = G.run_gpu(inp, accept=False)
    n = int(host["n_nodes"][0])
    assert n == wl.B + 1 and host["depth"][0][n - 1] == wl.B
    G.compare(inp, host)
    targets = _constructed_targets(host["tokens"][0], host["parent"][0], n,
                                   wl.N, wl.V, seed=4)
    cfg1 = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, 1)
    acc, length, bonus = _accept_replicated(cfg1, host, targets)
    leaf = n - 1
    assert int(length[leaf]) == wl.B
    assert acc[leaf].tolist() == list(range(wl.B + 1))
    assert int(bonus[leaf]) == targets[leaf][leaf]
    t = _oracle_tree(host)
    for u in range(n + 1):
        a_ref, len_ref, b_ref = O.accept(t, targets[u], wl.B)
        np.testing.assert_array_equal(acc[u], a_ref)
        assert int(length[u]) == len_ref and int(bonus[u]) == b_ref


def test_accept_clamps_node_count_to_budget():
    """A caller-built tree whose n_nodes exceeds N walks only the request's
    N rows: the result equals that of the true node count."""
    from paper_2608_02123_gb300 import pctree as P
    inp = draw_round(SMALL["ragged_V_bf16"].with_(batch=1))
    host = G.run_gpu(inp, accept=False)
    wl = inp.wl
    n = int(host["n_nodes"][0])
    targets = _constructed_targets(host["tokens"][0], host["parent"][0], n,
                                   wl.N, wl.V, seed=5)
    cfg1 = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, 1)
    ref = _accept_replicated(cfg1, host, targets)
    for bad in (wl.N + 1000, 1 << 30):
        got = _accept_replicated(cfg1, host, targets, n_nodes_override=bad)
        for a, b in zip(got, ref):
            np.testing.assert_array_equal(a, b)


@pytest.mark.skipif(not torch.cuda.is_available() or torch.cuda.device_count() < 2,
                    reason="needs two visible GPUs")
def test_second_device_after_first():
    """Kernel attributes are set per device: a round on device 1 after one on
    device 0 runs and matches."""
    inp = draw_round(SMALL["cut_tiles_bf16"])
    a = G.run_gpu(inp, accept=False)
    with torch.cuda.device(1):
        from paper_2608_02123_gb300 import pctree as P
        wl = inp.wl
        cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, wl.batch)
        L, E, W, root = G.device_inputs(inp, device="cuda:1")
        dr = P.Drafter(cfg, "cuda:1")
        tree = dr.draft(L, E, W, root)
        torch.cuda.synchronize()
        b = tree.to_host()
    for name in ("tokens", "parent", "mask", "n_nodes"):
        np.testing.assert_array_equal(a[name], b[name])
