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

# Largest own margin at which the CUDA path may legitimately decide otherwise
# than the float64 oracle.  Children are ranked on float32 stage logits
# z = L + bias (rounding of the sum and of the float32 dot product: a few
# 1e-6 for |z| up to ~100); frontier and budget on float32 scores whose error
# grows over up to 16 stages to at most ~5e-5 (twice that for a pair).  A
# near-tie adopted at a wider margin is a regression, not float32 noise.
FLOAT32_DECISION_BOUND = {"children": 5e-5, "frontier": 1e-4, "global": 1e-4}


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


# ---------------------------------------------------------------------------
# canary padding: every output tensor and the workspace sit inside a larger
# buffer whose margins hold a fixed bit pattern; a write past either end of
# any of them changes the pattern
# ---------------------------------------------------------------------------

CANARY_PAD = 512          # elements before and after each tensor
_CANARY = {torch.int32: 0x5A5A5A5A, torch.float32: 0x7FA5A5A5,
           torch.uint8: 0xA5}


class Canaries:
    def __init__(self, device="cuda"):
        self.device = device
        self.bufs = []           # (name, padded buffer, inner element count)

    def tensor(self, name, shape, dtype):
        n = int(np.prod(shape))
        bits = torch.int32 if dtype == torch.float32 else dtype
        buf = torch.full((n + 2 * CANARY_PAD,), _CANARY[dtype], dtype=bits,
                         device=self.device)
        if dtype == torch.float32:
            buf = buf.view(torch.float32)
        self.bufs.append((name, buf, n))
        return buf[CANARY_PAD:CANARY_PAD + n].view(*shape)

    def check(self):
        for name, buf, n in self.bufs:
            raw = buf.view(torch.int32) if buf.dtype == torch.float32 else buf
            want = _CANARY[buf.dtype]
            head = raw[:CANARY_PAD].cpu().numpy()
            tail = raw[CANARY_PAD + n:].cpu().numpy()
            if buf.dtype == torch.uint8:
                ok = (head == want).all() and (tail == want).all()
            else:
                ok = ((head.view(np.uint32) == np.uint32(want)).all() and
                      (tail.view(np.uint32) == np.uint32(want)).all())
            assert ok, f"canary around {name} overwritten"


def canary_drafter(P, cfg, with_pool: bool):
    """A Drafter whose tree, accept outputs and workspace are canary-padded."""
    dr = P.Drafter(cfg, with_pool=with_pool)
    cz = Canaries()
    R, N, B = cfg.batch, cfg.N, cfg.B
    Pn = P.pctree_pool_capacity(cfg)
    i32, f32, u8 = torch.int32, torch.float32, torch.uint8
    dr.tree = P.Tree(
        n_nodes=cz.tensor("n_nodes", (R,), i32),
        tokens=cz.tensor("tokens", (R, N), i32),
        parent=cz.tensor("parent", (R, N), i32),
        depth=cz.tensor("depth", (R, N), i32),
        logp=cz.tensor("logp", (R, N), f32),
        position_ids=cz.tensor("position_ids", (R, N), i32),
        mask=cz.tensor("mask", (R, N, N), u8),
        retrieve=cz.tensor("retrieve", (R, N, B + 1), i32),
        n_leaves=cz.tensor("n_leaves", (R,), i32),
        status=cz.tensor("status", (1,), i32),
        pool_token=cz.tensor("pool_token", (R, Pn), i32) if with_pool else None,
        pool_parent=cz.tensor("pool_parent", (R, Pn), i32) if with_pool else None,
        pool_logp=cz.tensor("pool_logp", (R, Pn), f32) if with_pool else None)
    # the workspace keeps its 256-byte alignment: the pad is 512 bytes
    nbytes = dr.workspace.numel()
    dr.workspace = cz.tensor("workspace", (nbytes,), u8)
    dr.accepted_idx = cz.tensor("accepted_idx", (R, B + 1), i32)
    dr.accepted_len = cz.tensor("accepted_len", (R,), i32)
    dr.bonus = cz.tensor("bonus", (R,), i32)
    return dr, cz


def run_gpu(inp: RoundInputs, with_pool=True, accept=True,
            path: int = 0, tiled: bool = False) -> Dict[str, np.ndarray]:
    """One round through the C ABI; ``path`` 0 = automatic (fused round
    kernel where it applies), 1 = per-stage kernels; ``tiled``: W_out
    repacked by pctree_pack_head and drafted in the tiled layout.  Every
    output tensor and the workspace are canary-padded and checked
    afterwards."""
    from paper_2608_02123_gb300 import pctree as P
    wl = inp.wl
    cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, inp.L.shape[0],
                        wl.pos_offset, wl.weight_dtype, wl.mode,
                        "tiled" if tiled else "rowmajor")
    L, E, W, root = device_inputs(inp)
    if tiled:
        W = P.pack_head(cfg, W)
    dr, canaries = canary_drafter(P, cfg, with_pool)
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
    canaries.check()
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
    # smallest own margin per decision kind over the compared requests
    margins: Dict[str, float] = dataclasses.field(default_factory=dict)
    # (request, kind, own margin) of every adopted near-tie decision
    adopted: List[tuple] = dataclasses.field(default_factory=list)

    def summary(self) -> str:
        m = " ".join(f"{k}={v:.1e}" for k, v in sorted(self.margins.items()))
        return (f"requests={self.requests} ambiguous={self.ambiguous} "
                f"max|dlogp|={self.max_logp_err:.2e} min margins: {m}")


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
        for kind, m in rnd.margins.items():
            rep.margins[kind] = min(rep.margins.get(kind, np.inf), m)
        for kind, m in rnd.adopted:
            rep.adopted.append((r, kind, m))
            assert m <= FLOAT32_DECISION_BOUND[kind], (
                f"request {r}: the CUDA path decided a {kind} choice "
                f"otherwise than the oracle across a margin of {m:.2e}, "
                f"wider than float32 noise ({FLOAT32_DECISION_BOUND[kind]:.0e})")
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
