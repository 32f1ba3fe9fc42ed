"""Accepted-row compaction on the GPU against the oracle (Appendix A, "Tensor
implementation"): bit-exact bytes of every cache plane and hidden-state row."""
import numpy as np
import pytest
import torch

from oracle import compact_oracle as co
from workloads import COMPACT_WORKLOADS, CompactWorkload, draw_compaction

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    from paper_2608_02123_gb300 import pctree
    return pctree


def run(P, ci, layout=None, cache_dev=None, status=True):
    cw = ci.cw
    dev = torch.device("cuda")
    lay = layout or P.compact_layout(cw.batch, cw.B, cw.N, cw.layers,
                                     cw.planes, cw.slots, cw.row_bytes,
                                     hidden_bytes=cw.hidden_bytes)
    cache = cache_dev if cache_dev is not None else \
        torch.from_numpy(ci.cache).to(dev)
    hin = torch.from_numpy(ci.hidden_in).to(dev)
    hout = torch.from_numpy(ci.hidden_out).to(dev)
    acc = torch.from_numpy(ci.accepted_idx).to(dev)
    ln = torch.from_numpy(ci.accepted_len).to(dev)
    pre = torch.from_numpy(ci.prefix_len).to(dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev) if status else None
    P.pctree_compact(lay, acc, ln, pre, cache, hin, hout, st)
    torch.cuda.synchronize()
    return cache, hout, (int(st.item()) if status else None)


@pytest.mark.parametrize("name", ["small", "ragged"])
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_matches_oracle(P, name, seed):
    ci = draw_compaction(COMPACT_WORKLOADS[name], seed=seed)
    cache, hout, st = run(P, ci)
    want, want_h, valid = co.compact(ci.cache, ci.hidden_in, ci.hidden_out,
                                     ci.accepted_idx, ci.accepted_len,
                                     ci.prefix_len, ci.cw.N)
    assert valid.all() and st == 0
    np.testing.assert_array_equal(cache.cpu().numpy(), want)
    np.testing.assert_array_equal(hout.cpu().numpy(), want_h)


def test_strided_layout_with_padding(P):
    """[batch][layers][planes][slots] order with 32 padding bytes per slot:
    the padding and every row outside the compacted ones keep their bytes."""
    cw = COMPACT_WORKLOADS["small"]
    ci = draw_compaction(cw, seed=7)
    pad = 32
    ss = cw.row_bytes + pad
    rng = np.random.default_rng(99)
    big = rng.integers(0, 256, size=(cw.batch, cw.layers, cw.planes,
                                     cw.slots, ss), dtype=np.uint8)
    lay = P.compact_layout(cw.batch, cw.B, cw.N, cw.layers, cw.planes,
                           cw.slots, cw.row_bytes, hidden_bytes=cw.hidden_bytes,
                           slot_stride=ss, plane_stride=cw.slots * ss,
                           layer_stride=cw.planes * cw.slots * ss,
                           request_stride=cw.layers * cw.planes * cw.slots * ss)
    cache = torch.from_numpy(big).cuda()
    got, _, st = run(P, ci, layout=lay, cache_dev=cache)
    assert st == 0
    # the oracle's [layers][planes][batch][slots][row] view of the same rows
    view = np.ascontiguousarray(big.transpose(1, 2, 0, 3, 4)[..., :cw.row_bytes])
    want, _, _ = co.compact(view, None, None, ci.accepted_idx, ci.accepted_len,
                            ci.prefix_len, cw.N)
    got = got.cpu().numpy()
    np.testing.assert_array_equal(got.transpose(1, 2, 0, 3, 4)[..., :cw.row_bytes],
                                  want)
    np.testing.assert_array_equal(got[..., cw.row_bytes:], big[..., cw.row_bytes:])


def test_invalid_requests_are_untouched_and_reported(P):
    cw = COMPACT_WORKLOADS["small"]
    ci = draw_compaction(cw, seed=3)
    ci.accepted_idx[1, :4] = [0, 4, 4, 9]        # repeated node
    ci.accepted_len[1] = 3
    ci.prefix_len[2] = cw.prefix_max + 1         # tree would end past the row
    cache, hout, st = run(P, ci)
    want, want_h, valid = co.compact(ci.cache, ci.hidden_in, ci.hidden_out,
                                     ci.accepted_idx, ci.accepted_len,
                                     ci.prefix_len, cw.N)
    assert list(valid) == [True, False, False]
    assert st == -1                              # PCTREE_ERR_INVALID_ARG
    np.testing.assert_array_equal(cache.cpu().numpy(), want)
    np.testing.assert_array_equal(hout.cpu().numpy(), want_h)


def test_identity_empty_and_full_paths(P):
    cw = COMPACT_WORKLOADS["small"]
    ci = draw_compaction(cw, seed=4)
    ci.accepted_idx[:] = -1
    ci.accepted_idx[0, :cw.B + 1] = np.arange(cw.B + 1)      # in place
    ci.accepted_len[0] = cw.B
    ci.accepted_idx[1, 0] = 0                                # root only
    ci.accepted_len[1] = 0
    ci.accepted_idx[2, :cw.B + 1] = [0] + list(range(cw.N - cw.B, cw.N))
    ci.accepted_len[2] = cw.B                                # deepest nodes
    cache, hout, st = run(P, ci)
    want, want_h, valid = co.compact(ci.cache, ci.hidden_in, ci.hidden_out,
                                     ci.accepted_idx, ci.accepted_len,
                                     ci.prefix_len, cw.N)
    assert valid.all() and st == 0
    np.testing.assert_array_equal(cache.cpu().numpy(), want)
    np.testing.assert_array_equal(hout.cpu().numpy(), want_h)


def test_long_paths_cross_the_load_batches(P):
    """Paths longer than the kernel's batch of loads in flight (k = 1 trees
    with a deep draft): in-place order must hold across batches."""
    cw = CompactWorkload("deep", layers=2, planes=2, row_bytes=32,
                         hidden_bytes=16, B=40, N=48, batch=4, prefix_max=9,
                         seed=30)
    for seed in range(3):
        ci = draw_compaction(cw, seed=seed)
        ci.accepted_idx[0, :] = np.arange(41) + np.r_[0, np.full(40, 7)]
        ci.accepted_len[0] = 40
        cache, hout, st = run(P, ci)
        want, want_h, valid = co.compact(ci.cache, ci.hidden_in, ci.hidden_out,
                                         ci.accepted_idx, ci.accepted_len,
                                         ci.prefix_len, cw.N)
        assert valid.all() and st == 0
        np.testing.assert_array_equal(cache.cpu().numpy(), want)
        np.testing.assert_array_equal(hout.cpu().numpy(), want_h)


def test_full_size_qwen3_4b(P):
    ci = draw_compaction(COMPACT_WORKLOADS["4b_b16"])
    cache, hout, st = run(P, ci)
    want, want_h, _ = co.compact(ci.cache, ci.hidden_in, ci.hidden_out,
                                 ci.accepted_idx, ci.accepted_len,
                                 ci.prefix_len, ci.cw.N)
    assert st == 0
    np.testing.assert_array_equal(cache.cpu().numpy(), want)
    np.testing.assert_array_equal(hout.cpu().numpy(), want_h)


def test_full_size_qwen3_14b_batch32_labelled(P):
    """40 layers x K/V x 32 requests x 1152 slots x 2 KB (6 GB): each row is
    filled with its own row number, the oracle compacts the array of row
    numbers, and every row of the device cache must hold the expected number
    in all of its 512 words."""
    cw = COMPACT_WORKLOADS["14b_b16_bs32"]
    ci = draw_compaction(cw, fill=False)
    g = np.random.default_rng(5)
    ci.hidden_in = g.integers(0, 256, (cw.batch, cw.N, cw.hidden_bytes), np.uint8)
    ci.hidden_out = g.integers(0, 256, (cw.batch, cw.B + 1, cw.hidden_bytes),
                               np.uint8)
    n_rows = cw.layers * cw.planes * cw.batch * cw.slots
    words = cw.row_bytes // 4
    labels = np.arange(n_rows, dtype=np.int32)
    cache = torch.empty((n_rows, words), dtype=torch.int32, device="cuda")
    cache.copy_(torch.from_numpy(labels).cuda()[:, None].expand(-1, words))
    _, hout, st = run(P, ci, cache_dev=cache)
    assert st == 0
    shape = (cw.layers, cw.planes, cw.batch, cw.slots, 4)
    want, want_h, valid = co.compact(labels.view(np.uint8).reshape(shape),
                                     ci.hidden_in, ci.hidden_out,
                                     ci.accepted_idx, ci.accepted_len,
                                     ci.prefix_len, cw.N)
    assert valid.all()
    assert bool((cache == cache[:, :1]).all())
    np.testing.assert_array_equal(cache[:, 0].cpu().numpy(),
                                  want.view(np.int32).reshape(-1))
    np.testing.assert_array_equal(hout.cpu().numpy(), want_h)
    del cache
    torch.cuda.empty_cache()
