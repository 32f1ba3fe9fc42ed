"""Writes the oracle's regression fixtures.  Calls only ``oracle/`` (and the
seeded input generators); run from the repository root:

    python tests/golden/make_golden.py
"""
import json
import os
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

from oracle import pctree_oracle as O  # noqa: E402
from workloads import WORKLOADS, draw_round, target_for_tree  # noqa: E402


def tiny():
    wl = WORKLOADS["tiny"]
    inp = draw_round(wl)
    E, W = O.as_f64(inp.E_in, "f32"), O.as_f64(inp.W_out, "f32")
    rnd = O.draft(inp.L[0], E, W, int(inp.root[0]), wl.B, wl.k, wl.N)
    t = rnd.tree
    target = target_for_tree(inp.greedy, t.depth[None, :])[0]
    acc, length, bonus = O.accept(t, target, wl.B)
    return {
        "about": "oracle output for the tiny workload (V=1024, H=64 f32, "
                 "B=4, k=4, N=8, seed 0): Algorithm 1 + Appendix A packing "
                 "and greedy acceptance; regression fixture, written by "
                 "tests/golden/make_golden.py",
        "tokens": t.tokens.tolist(), "parent": t.parent.tolist(),
        "depth": t.depth.tolist(), "logp": t.logp.tolist(),
        "retrieve": t.retrieve.tolist(), "n_leaves": t.n_leaves,
        "accept": [acc.tolist(), int(length), int(bonus)],
        "margins": rnd.margins,
    }


if __name__ == "__main__":
    with open(os.path.join(HERE, "tiny_seed0_oracle.json"), "w") as f:
        json.dump(tiny(), f, indent=1)
        f.write("\n")
