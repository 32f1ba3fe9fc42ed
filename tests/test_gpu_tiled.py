"""W_out in the tiled layout (PCTREE_HEAD_TILED): the repacking kernel
against the layout's definition, and drafting rounds from tiled weights
against the oracle (the layout is storage only: every result must match the
row-major rounds' parity bar)."""
import numpy as np
import pytest
import torch

from tests import gpu_util as G
from tests.test_gpu_parity import PATHS, SMALL, _full
from workloads import WORKLOADS, draw_round

pytestmark = pytest.mark.gpu


def tiled_reference(bits: np.ndarray) -> np.ndarray:
    """The layout's definition: [ceil(V/128)][ceil(H/64)][128][64] blocks of
    the [V][H] matrix, zero where a row >= V or a column >= H."""
    V, H = bits.shape
    nt, nk = -(-V // 128), -(-H // 64)
    pad = np.zeros((nt * 128, nk * 64), bits.dtype)
    pad[:V, :H] = bits
    return pad.reshape(nt, 128, nk, 64).transpose(0, 2, 1, 3).copy()


@pytest.mark.parametrize("V,H", [(3000, 72), (1111, 64), (128, 8), (40000, 136)])
def test_pack_head_matches_layout(V, H):
    from paper_2608_02123_gb300 import pctree as P
    rng = np.random.default_rng(V + H)
    bits = rng.integers(0, 1 << 16, size=(V, H), dtype=np.uint16)
    W = torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)
    cfg = P.make_config(V, H, 2, 2, 4)
    assert P.pctree_packed_head_bytes(cfg) == tiled_reference(bits).nbytes
    # a dirty buffer: padding must be written, not assumed
    packed = torch.full((P.pctree_packed_head_bytes(cfg) // 2,), -1,
                        dtype=torch.int16, device="cuda").view(torch.bfloat16)
    P.pctree_pack_head(cfg, W, packed)
    torch.cuda.synchronize()
    got = packed.view(torch.int16).cpu().numpy().view(np.uint16)
    np.testing.assert_array_equal(got.reshape(-1), tiled_reference(bits).reshape(-1))


TILED_CASES = ["ragged_V_bf16", "ragged_K_bf16", "cut_tiles_bf16",
               "multipass_bf16", "shared_batched_bf16", "k32_bf16"]


@pytest.mark.parametrize("path", sorted(PATHS))
@pytest.mark.parametrize("name", TILED_CASES)
def test_tiled_small_parity(name, path):
    inp = draw_round(SMALL[name])
    host = G.run_gpu(inp, path=PATHS[path], tiled=True)
    rep = G.compare(inp, host)
    print(f"{name}/{path}/tiled: " + rep.summary())


def test_tiled_full_size_batch1():
    inp = _full("4b_b16")
    host = G.run_gpu(inp, tiled=True)
    rep = G.compare(inp, host)
    print("4b_b16/tiled: " + rep.summary())


def test_tiled_full_size_batched_sampled():
    wl = WORKLOADS["8b_b7_bs16"]
    inp = draw_round(wl)
    host = G.run_gpu(inp, tiled=True)
    rep = G.compare(inp, host, requests=[0, 7, 15])
    print("8b_b7_bs16/tiled: " + rep.summary())


def test_tiled_needs_bf16():
    from paper_2608_02123_gb300 import pctree as P
    cfg = P.make_config(100, 8, 2, 2, 4, 1, 0, "f32", "parent", "tiled")
    assert P.pctree_check_config(cfg) == -1
    assert P.pctree_packed_head_bytes(cfg) == 0
