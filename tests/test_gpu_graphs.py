"""Drafting rounds and attention layers captured in a CUDA graph and replayed
give what direct calls give.  The per-stage kernels and the attention
kernels are launched with programmatic stream serialization; a capture
turns that into programmatic graph edges, and every kernel still waits for
its predecessor before it touches global memory."""
import numpy as np
import pytest
import torch

from tests import gpu_util as G
from workloads import ATTN_WORKLOADS, WORKLOADS, draw_attention, draw_round

pytestmark = pytest.mark.gpu


def _captured(fn, stream):
    """A graph of fn(stream) captured on `stream`, after one direct call
    outside the capture (which sets kernel attributes once)."""
    stream.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(stream):
        fn(stream)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn(torch.cuda.current_stream())
    return g


# (batch, path): batch 2 x k 4 = 8 Markov rows takes the fused round on the
# automatic path; 24 rows, and any batch on path 1, take the per-stage kernels
@pytest.mark.parametrize("batch,path", [(2, 0), (2, 1), (6, 0)])
def test_round_replayed_from_a_cuda_graph(batch, path):
    from paper_2608_02123_gb300 import pctree as P
    wl = WORKLOADS["4b_b16"].with_(V=3000, H=256, B=5, k=4, N=16, batch=batch, seed=31,
                                   head_scale_e=1.0, head_scale_w=0.125)
    inp = draw_round(wl)
    cfg = P.make_config(wl.V, wl.H, wl.B, wl.k, wl.N, inp.L.shape[0])
    L, E, W, root = G.device_inputs(inp)
    P.pctree_set_path(path)
    try:
        want = P.Drafter(cfg).draft(L, E, W, root).to_host()
        dr = P.Drafter(cfg)
        g = _captured(lambda s: dr.draft(L, E, W, root, s), torch.cuda.Stream())
        for _ in range(3):
            dr.tree.tokens.fill_(-7)      # each replay writes the round again
            g.replay()
        torch.cuda.synchronize()
        got = dr.tree.to_host()
    finally:
        P.pctree_set_path(P.PATH_AUTO)
    dr.check_status()
    for key, value in want.items():
        if value is not None:
            np.testing.assert_array_equal(value, got[key], err_msg=key)


@pytest.mark.parametrize("name", ["small", "ragged"])
def test_attention_replayed_from_a_cuda_graph(name):
    from paper_2608_02123_gb300 import pctree as P
    ai = draw_attention(ATTN_WORKLOADS[name])
    aw = ai.aw
    cfg = P.attn_config(aw.batch, aw.N, aw.Hq, aw.Hkv, aw.slots)
    dev = lambda bits: torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)
    q, k, v = dev(ai.q), dev(ai.k), dev(ai.v)
    pre = torch.from_numpy(ai.prefix_len).cuda()
    nn = torch.from_numpy(ai.n_nodes).cuda()
    par = torch.from_numpy(ai.parent).cuda()
    nb = P.pctree_tree_attention_workspace_bytes(cfg)
    ws = torch.empty(max(nb, 1), dtype=torch.uint8, device="cuda") if nb else None
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    want = torch.empty_like(q)
    P.pctree_tree_attention(cfg, q, k, v, pre, nn, par, want, ws, st)
    out = torch.empty_like(q)
    g = _captured(lambda s: P.pctree_tree_attention(cfg, q, k, v, pre, nn, par, out, ws, st, s),
                  torch.cuda.Stream())
    for _ in range(3):
        out.fill_(float("nan"))
        g.replay()
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    assert torch.equal(out.view(torch.int16), want.view(torch.int16))
