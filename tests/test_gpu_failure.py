"""Failure detection on the GPU without a fault: a test hook withholds the
cross-CTA release of one stage of the fused round, so every CTA's bounded
wait for it runs out.  The round must come back promptly with
PCTREE_ERR_TIMEOUT in its status word, and the same context must then draft
a correct round."""
import time

import numpy as np
import pytest
import torch

from tests import gpu_util as G
from workloads import WORKLOADS, draw_round

pytestmark = pytest.mark.gpu

WL = WORKLOADS["4b_b16"].with_(V=20000, H=256, B=5, k=4, N=16, batch=2,
                               head_scale_e=1.0, head_scale_w=2.0 / 16.0,
                               seed=31)


@pytest.fixture(scope="module")
def P():
    from paper_2608_02123_gb300 import pctree
    return pctree


@pytest.mark.parametrize("stage", [1, 3])
def test_withheld_release_times_out_and_context_recovers(P, stage):
    inp = draw_round(WL)
    cfg = P.make_config(WL.V, WL.H, WL.B, WL.k, WL.N, WL.batch, 0, "bf16")
    assert P.uses_fused_round(cfg)
    L, E, W, root = G.device_inputs(inp)
    dr = P.Drafter(cfg)
    dr.draft(L, E, W, root)                  # warm the kernel up
    torch.cuda.synchronize()
    dr.check_status()
    P.pctree_debug_stall_stage(stage, 5_000_000)          # 5 ms bound
    try:
        t0 = time.perf_counter()
        dr.draft(L, E, W, root)
        torch.cuda.synchronize()
        elapsed = time.perf_counter() - t0
    finally:
        P.pctree_debug_stall_stage(-1, 1_000_000_000)
    with pytest.raises(P.PctreeError) as err:
        dr.check_status()
    assert err.value.code == -4                         # PCTREE_ERR_TIMEOUT
    assert elapsed < 2.0, elapsed
    # the context is intact: a normal round matches the oracle
    host = G.run_gpu(inp)
    G.compare(inp, host)
