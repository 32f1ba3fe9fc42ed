"""Helpers shared by the GPU parity tests: run the CUDA path through the C
ABI and compare it with the oracle on the same seeded inputs."""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

from oracle import pctree_oracle as O
from workloads import RoundInputs, target_for_tree

LOGP_TOL = 1e-4      # absolute, on cumulative log-probs


def device_inputs(inp: RoundInputs, device="cuda"):
    wl = inp.wl
    if wl.weight_dtype == "bf16":
        E = torch.from_numpy(inp.E_in.view(np.int16)).to(device).view(torch.bfloat16)
        W = torch.from_numpy(inp.W_out.view(np.int16)).to(device).view(torch.bfloat16)
    else:
        E = torch.from_numpy(inp.E_in).to(device)
        W = torch.from_numpy(inp.W_out).to(device)
    L = torch.from_numpy(np.ascontiguousarray(inp.L)).to(device)
    root = torch.from_numpy(inp.root.astype(np.int32)).to(device)
    return L, E, W, root


def run_gpu(inp: RoundInputs, with_pool=True, accept=True,
            path: int = 0) -> Dict[str, np.ndarray]:
    """One round through the C ABI; ``path`` 0 = automatic (fused round
    kernel where it applies), 1 = per-stage kernels."""
    from paper_2608_02123_gb300 import pctree as P
    wl = inp.wl
    cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, inp.L.shape[0],
                        wl.pos_offset, wl.weight_dtype, wl.mode)
    L, E, W, root = device_inputs(inp)
    dr = P.Drafter(cfg, with_pool=with_pool)
    P.pctree_set_path(path)
    try:
        tree = dr.draft(L, E, W, root)
        torch.cuda.synchronize()
    finally:
        P.pctree_set_path(P.PATH_AUTO)
    host = tree.to_host()
    if accept:
        target = target_for_tree(inp.greedy, host["depth"])
        acc, length, bonus = dr.accept(torch.from_numpy(target).cuda())
        torch.cuda.synchronize()
        host["target"] = target
        host["accepted_idx"] = acc.cpu().numpy()
        host["accepted_len"] = length.cpu().numpy()
        host["bonus"] = bonus.cpu().numpy()
    return host


def tree_paths(tokens, parent, n) -> List[tuple]:
    paths: List[tuple] = []
    for a in range(n):
        paths.append(() if a == 0 else paths[parent[a]] + (int(tokens[a]),))
    return paths


def gpu_choices(host: Dict[str, np.ndarray], r: int) -> O.Choices:
    n = int(host["n_nodes"][r])
    sel = set(tree_paths(host["tokens"][r], host["parent"][r], n))
    P = host["pool_token"].shape[1]
    return O.choices_from_pool(host["pool_token"][r], host["pool_parent"][r],
                               P, sel)


@dataclasses.dataclass
class Report:
    ambiguous: int = 0
    max_logp_err: float = 0.0
    requests: int = 0
    min_margin: float = np.inf


def _close(got: np.ndarray, want: np.ndarray, r: int) -> float:
    """|got - want| <= LOGP_TOL where finite; -inf exactly where -inf."""
    got = got.astype(np.float64)
    fin = np.isfinite(want)
    np.testing.assert_array_equal(np.isneginf(got), np.isneginf(want),
                                  err_msg=f"-inf pattern request {r}")
    assert np.isfinite(got[fin]).all()
    err = np.abs(got[fin] - want[fin])
    worst = float(err.max()) if err.size else 0.0
    assert worst <= LOGP_TOL, (r, worst)
    return worst


def weights_f64(inp: RoundInputs):
    return (O.as_f64(inp.E_in, inp.wl.weight_dtype),
            O.as_f64(inp.W_out, inp.wl.weight_dtype))


def compare(inp: RoundInputs, host: Dict[str, np.ndarray],
            requests: Optional[Sequence[int]] = None, weights=None,
            strict: bool = False) -> Report:
    """Element-by-element comparison with the oracle.  With ``strict`` the
    oracle takes only its own decisions (used where exact ties are planted)."""
    wl = inp.wl
    E64, W64 = weights if weights is not None else weights_f64(inp)
    rep = Report()
    reqs = range(inp.L.shape[0]) if requests is None else requests
    for r in reqs:
        assert int(host["status"][0]) == 0, host["status"]
        hint = None if strict else gpu_choices(host, r)
        rnd = O.draft(inp.L[r], E64, W64, int(inp.root[r]), wl.B, wl.k, wl.N,
                      wl.pos_offset, hint=hint, mode=wl.mode)
        t = rnd.tree
        rep.requests += 1
        rep.ambiguous += rnd.n_ambiguous
        rep.min_margin = min(rep.min_margin, *rnd.margins.values())
        assert int(host["n_nodes"][r]) == t.n_nodes
        for name in ("tokens", "parent", "depth", "position_ids"):
            np.testing.assert_array_equal(host[name][r], getattr(t, name),
                                          err_msg=f"{name} request {r}")
        np.testing.assert_array_equal(host["mask"][r], t.mask,
                                      err_msg=f"mask request {r}")
        np.testing.assert_array_equal(host["retrieve"][r], t.retrieve,
                                      err_msg=f"retrieve request {r}")
        assert int(host["n_leaves"][r]) == t.n_leaves
        n = t.n_nodes
        rep.max_logp_err = max(rep.max_logp_err,
                               _close(host["logp"][r][:n], t.logp[:n], r))
        assert np.isneginf(host["logp"][r][n:]).all()
        if "pool_logp" in host and host["pool_logp"] is not None:
            _close(host["pool_logp"][r], np.asarray(rnd.pool.s), r)
            np.testing.assert_array_equal(host["pool_token"][r],
                                          np.asarray(rnd.pool.token))
            np.testing.assert_array_equal(host["pool_parent"][r],
                                          np.asarray(rnd.pool.parent))
        if "accepted_len" in host:
            acc, length, bonus = O.accept(t, host["target"][r], wl.B)
            np.testing.assert_array_equal(host["accepted_idx"][r], acc)
            assert int(host["accepted_len"][r]) == length
            assert int(host["bonus"][r]) == bonus
    return rep
