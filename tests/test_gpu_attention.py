"""Tree-verification attention on the GPU against the float64 oracle (Sec.
4.2; Appendix A).

Tolerance: an output row is a convex combination of V rows (|V| < 6 for the
drawn N(0,1) values).  The kernel rounds the probabilities to bf16 before
the P.V product (relative error <= 2^-9 each, in numerator and denominator
alike) and rounds the output to bf16 (<= 2^-9 relative), with float32
accumulation elsewhere; so |gpu - oracle| <= 2 * 2^-9 * max|V| + 2^-9 |out|
<= 0.024 + 0.002 |out|.  The tests use atol 0.025, rtol 0.004, and check
that the mean error is far smaller (< 2e-3), which a systematic mistake
would not meet.
"""
import numpy as np
import pytest
import torch

from oracle import attention_oracle as ao
from workloads import (ATTN_WORKLOADS, AttnWorkload, bf16_bits_to_f32,
                       draw_attention)

pytestmark = pytest.mark.gpu

ATOL, RTOL, MEAN_TOL = 0.025, 0.004, 2e-3


@pytest.fixture(scope="module")
def P():
    from paper_2608_02123_gb300 import pctree
    return pctree


def to_dev(bits):
    return torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16)


def run(P, ai, prefix=None, n_nodes=None, k_bits=None, v_bits=None):
    aw = ai.aw
    cfg = P.attn_config(aw.batch, aw.N, aw.Hq, aw.Hkv, aw.slots)
    q = to_dev(ai.q)
    k = to_dev(ai.k if k_bits is None else k_bits)
    v = to_dev(ai.v if v_bits is None else v_bits)
    pre = torch.from_numpy(ai.prefix_len if prefix is None else prefix).cuda()
    nn = torch.from_numpy(ai.n_nodes if n_nodes is None else n_nodes).cuda()
    par = torch.from_numpy(ai.parent).cuda()
    out = torch.full_like(q, float("nan"))
    nb = P.pctree_tree_attention_workspace_bytes(cfg)
    ws = torch.empty(max(nb, 1), dtype=torch.uint8, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    P.pctree_tree_attention(cfg, q, k, v, pre, nn, par, out,
                            ws if nb else None, st)
    torch.cuda.synchronize()
    return out.float().cpu().numpy(), int(st.item())


def reference(ai, rows=None, prefix=None, n_nodes=None):
    f = lambda b: bf16_bits_to_f32(b)
    return ao.tree_attention(f(ai.q), f(ai.k), f(ai.v),
                             ai.prefix_len if prefix is None else prefix,
                             ai.n_nodes if n_nodes is None else n_nodes,
                             ai.parent, 1.0 / np.sqrt(ai.aw.D), rows)


def compare(got, want, rows=None):
    if rows is not None:
        idx = tuple(np.asarray(rows).T)
        got, want = got[idx], want[idx]
    assert np.isfinite(got).all()
    err = np.abs(got - want)
    assert (err <= ATOL + RTOL * np.abs(want)).all(), err.max()
    assert err.mean() < MEAN_TOL, err.mean()


@pytest.mark.parametrize("name", ["small", "ragged"])
@pytest.mark.parametrize("seed", [0, 1])
def test_matches_oracle(P, name, seed):
    ai = draw_attention(ATTN_WORKLOADS[name], seed=seed)
    got, st = run(P, ai)
    assert st == 0
    compare(got, reference(ai))


def test_split_keys_and_long_prefix(P):
    """Prefixes spanning many key blocks, split over CTAs and merged."""
    aw = AttnWorkload("long", batch=2, N=32, Hq=8, Hkv=2, D=128, B=6,
                      prefix_max=900, seed=50)
    ai = draw_attention(aw)
    got, st = run(P, ai)
    assert st == 0
    compare(got, reference(ai))


def test_non_finite_cache_past_the_tree_is_ignored(P):
    aw = ATTN_WORKLOADS["small"]
    ai = draw_attention(aw, seed=3)
    k, v = ai.k.copy(), ai.v.copy()
    for r in range(aw.batch):
        end = int(ai.prefix_len[r] + ai.n_nodes[r])
        k[r, end:] = 0x7fc0          # NaN
        v[r, end:] = 0x7f80          # +inf
    got, st = run(P, ai, k_bits=k, v_bits=v)
    assert st == 0
    compare(got, reference(ai))


def test_empty_tree_and_invalid_request(P):
    aw = ATTN_WORKLOADS["small"]
    ai = draw_attention(aw, seed=4)
    nn = ai.n_nodes.copy()
    nn[0] = 0                                  # no nodes: all rows 0
    got, st = run(P, ai, n_nodes=nn)
    assert st == 0
    assert not got[0].any()
    compare(got[1:], reference(ai, n_nodes=nn)[1:])
    pre = ai.prefix_len.copy()
    pre[1] = aw.slots                           # tree would end past the row
    got, st = run(P, ai, prefix=pre)
    assert st == -1
    assert not got[1].any()
    compare(got[:1], reference(ai)[:1])


def sampled_rows(ai, per_request=4, seed=0):
    rng = np.random.default_rng(seed)
    rows = []
    for r in range(ai.aw.batch):
        n = int(ai.n_nodes[r])
        pick = {0, n - 1} | set(rng.integers(0, n, size=per_request).tolist())
        rows += [(r, int(i)) for i in sorted(pick)]
    return rows


def test_full_size_qwen3_4b(P):
    ai = draw_attention(ATTN_WORKLOADS["4b_b16"])
    got, st = run(P, ai)
    assert st == 0
    compare(got, reference(ai))


@pytest.mark.parametrize("name", ["8b_b7_bs16", "14b_b16_bs32"])
def test_full_size_batched_sampled_rows(P, name):
    ai = draw_attention(ATTN_WORKLOADS[name])
    got, st = run(P, ai)
    assert st == 0
    rows = sampled_rows(ai)
    compare(got, reference(ai, rows=rows), rows)
    # rows past each request's tree are 0
    for r in range(ai.aw.batch):
        assert not got[r, int(ai.n_nodes[r]):].any()
