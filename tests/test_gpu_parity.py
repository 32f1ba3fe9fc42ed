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
    print(f"{name}/{path}: ambiguous={rep.ambiguous} "
          f"max|dlogp|={rep.max_logp_err:.2e}")


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
    print(f"{name}/{path}: ambiguous={rep.ambiguous} "
          f"max|dlogp|={rep.max_logp_err:.2e} min margin={rep.min_margin:.2e}")


@pytest.mark.parametrize("name,n_check", [("8b_b7_bs16", 2), ("14b_b16_bs32", 1)])
def test_full_size_batched_sampled(name, n_check):
    """Whole batch on the GPU in the benchmark's launch configuration; the
    oracle checks the first requests (each request is independent)."""
    wl = WORKLOADS[name]
    inp = draw_round(wl)
    host = G.run_gpu(inp)
    rep = G.compare(inp, host, requests=range(n_check))
    print(f"{name}: ambiguous={rep.ambiguous} max|dlogp|={rep.max_logp_err:.2e}")
    # every request: structural invariants of its tree
    for r in range(wl.batch):
        n = int(host["n_nodes"][r])
        assert n == min(wl.N, wl.pool_size)
        par = host["parent"][r][:n]
        assert par[0] == -1 and (par[1:] < np.arange(1, n)).all()
        lp = host["logp"][r][:n]
        assert (lp[1:] <= lp[par[1:]]).all()
        assert (host["mask"][r][:n, :n].sum(1) == host["depth"][r][:n] + 1).all()
