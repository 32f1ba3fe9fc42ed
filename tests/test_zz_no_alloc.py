"""pctree_draft_noalloc: the drafting round for callers that cannot allocate
device memory (a host framework that owns a fixed memory budget, a plug-in
that only receives its host's buffers, a latency-critical loop where
cudaMalloc would synchronise the device).  Its scratch is a fixed array
inside the library; these tests check, through the C ABI, that two calls in
a row give the same trees as pctree_draft with a caller workspace, and that
rounds too large for the array are refused.  Collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

from tests import gpu_util as G
from workloads import WORKLOADS, draw_round

pytestmark = pytest.mark.gpu

TREE_FIELDS = ("n_nodes", "tokens", "parent", "depth", "position_ids", "mask",
               "retrieve", "n_leaves")


def _workload(seed, **kw):
    base = WORKLOADS["4b_b16"].with_(V=20000, H=512, B=6, k=8, N=32, batch=1,
                                     head_scale_e=1.0, head_scale_w=0.09,
                                     seed=seed)
    return base.with_(**kw)


def _reference(inp):
    """The round through pctree_draft with a torch-allocated workspace."""
    return G.run_gpu(inp, with_pool=False, accept=False)


@pytest.mark.parametrize("weights", ["bf16", "f32"])
def test_noalloc_matches_workspace_round_on_two_calls(weights):
    from paper_2608_02123_gb300 import pctree as P
    for call, seed in enumerate((41, 42)):
        wl = _workload(seed, weight_dtype=weights)
        inp = draw_round(wl)
        ref = _reference(inp)
        L, E, W, root = G.device_inputs(inp)
        cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, wl.batch, 0,
                            wl.weight_dtype)
        tree = P.alloc_tree(cfg, "cuda")
        P.pctree_draft_noalloc(cfg, L, E, W, root, tree)
        torch.cuda.synchronize()
        got = tree.to_host()
        assert int(got["status"][0]) == 0, (call, got["status"])
        for name in TREE_FIELDS:
            np.testing.assert_array_equal(got[name], ref[name],
                                          err_msg=f"{name}, call {call}")
        fin = np.isfinite(ref["logp"])
        np.testing.assert_array_equal(np.isfinite(got["logp"]), fin)
        assert np.abs(got["logp"][fin] - ref["logp"][fin]).max() <= G.LOGP_TOL


def test_noalloc_refuses_rounds_beyond_its_array():
    from paper_2608_02123_gb300 import pctree as P
    wl = WORKLOADS["14b_b16_bs32"]
    cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, wl.batch)
    assert P.pctree_workspace_bytes(cfg) > 16 << 20
    fake = 4096
    tree = P._Tree(*([256] * 10 + [None] * 3))
    rc = P.LIB.pctree_draft_noalloc(ctypes.byref(cfg), fake, fake, fake, fake,
                                    ctypes.byref(tree), None)
    assert rc == -2   # PCTREE_ERR_WORKSPACE, before any GPU work
