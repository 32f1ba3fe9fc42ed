"""The C ABI library loads and exports every declared symbol, and its host
side rejects bad arguments before touching a GPU (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pctree.h")


@pytest.fixture(scope="module")
def P():
    from paper_2608_02123_gb300 import build
    if not os.path.exists(build.LIB):
        build.build()
    from paper_2608_02123_gb300 import pctree
    return pctree


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"PCTREE_API\s+[\w\s\*]+?\b(pctree_\w+)\(", text)))


def test_header_declares_the_api():
    names = declared_symbols()
    for n in ("pctree_draft", "pctree_accept", "pctree_workspace_bytes",
              "pctree_pool_capacity", "pctree_check_config"):
        assert n in names


def test_every_declared_symbol_is_exported(P):
    lib = ctypes.CDLL(P.LIB_PATH)
    for name in declared_symbols():
        assert hasattr(lib, name), name


def test_config_checks(P):
    mk = P.make_config
    assert P.pctree_check_config(mk(151936, 2560, 16, 8, 64, 1)) == 0
    assert P.pctree_check_config(mk(1024, 64, 4, 4, 8, 1, 0, "f32")) == 0
    assert P.pctree_check_config(mk(10, 8, 2, 11, 4, 1)) == -1      # k > V
    assert P.pctree_check_config(mk(100, 12, 2, 2, 4, 1)) == -1     # H % 8
    assert P.pctree_check_config(mk(100, 12, 2, 2, 4, 1, 0, "f32")) == 0
    assert P.pctree_check_config(mk(100, 8, 2, 33, 4, 1)) == -6     # k limit
    assert P.pctree_check_config(mk(100, 8, 2, 2, 1025, 1)) == -6   # N limit
    assert P.pctree_check_config(mk(100, 8, 2, 8, 4, 513)) == -6    # rows
    assert P.pctree_check_config(mk(100, 8, 300, 8, 4, 1)) == -6    # pool
    assert P.pctree_check_config(mk(100, 8, 0, 2, 4, 1)) == -1
    assert P.pctree_check_config(mk(100, 8, 2, 2, 0, 1)) == -1


def test_sizes(P):
    c = P.make_config(151936, 2560, 16, 8, 64, 1)
    assert P.pctree_pool_capacity(c) == 1 + 8 + 15 * 64
    ws = P.pctree_workspace_bytes(c)
    # bf16 heads never hold a stage's logits (8 rows x V floats) in memory
    assert ws % 256 == 0 and ws < 8 * 151936 * 4
    c32 = P.make_config(151936, 2560, 16, 8, 64, 1, 0, "f32")
    assert P.pctree_workspace_bytes(c32) > 8 * 151936 * 4
    assert P.pctree_workspace_bytes(P.make_config(10, 8, 2, 11, 4, 1)) == 0


def test_draft_rejects_bad_arguments_on_the_host(P):
    c = P.make_config(1000, 64, 3, 4, 8, 1)
    tree = P._Tree(*([256] * 10 + [None] * 3))
    fake = 4096
    lib = P.LIB
    # missing output pointer
    t2 = P._Tree(*([256] * 9 + [None] * 4))
    assert lib.pctree_draft(ctypes.byref(c), fake, fake, fake, fake,
                            ctypes.byref(t2), fake, 1 << 30, None) == -1
    # misaligned weights
    assert lib.pctree_draft(ctypes.byref(c), fake, fake + 2, fake, fake,
                            ctypes.byref(tree), fake, 1 << 30, None) == -1
    # workspace too small or misaligned
    assert lib.pctree_draft(ctypes.byref(c), fake, fake, fake, fake,
                            ctypes.byref(tree), fake, 16, None) == -2
    assert lib.pctree_draft(ctypes.byref(c), fake, fake, fake, fake,
                            ctypes.byref(tree), fake + 8, 1 << 30, None) == -2
    # only some of the optional pool outputs
    t3 = P._Tree(*([256] * 11 + [None] * 2))
    assert lib.pctree_draft(ctypes.byref(c), fake, fake, fake, fake,
                            ctypes.byref(t3), fake, 1 << 30, None) == -1
    # bad config
    bad = P.make_config(10, 8, 2, 11, 4, 1)
    assert lib.pctree_draft(ctypes.byref(bad), fake, fake, fake, fake,
                            ctypes.byref(tree), fake, 1 << 30, None) == -1
    assert lib.pctree_accept(ctypes.byref(c), ctypes.byref(t2), None, fake,
                             fake, fake, None) == -1


def test_status_strings(P):
    assert P.pctree_status_string(0) == "ok"
    assert "timed out" in P.pctree_status_string(-4)
    assert P.pctree_version() >= 100


def test_compact_rejects_bad_layouts_on_the_host(P):
    lib, fake = P.LIB, 4096
    good = P.compact_layout(2, 5, 16, 3, 2, 40, 64, hidden_bytes=96)

    def call(lay, cache=fake, hin=fake, hout=fake * 64, acc=fake):
        return lib.pctree_compact(ctypes.byref(lay), acc, fake, fake, cache,
                                  hin, hout, None, None)

    def variant(**kw):
        f = {n: getattr(good, n) for n, _ in P.CompactLayout._fields_}
        f.update(kw)
        return P.CompactLayout(**f)

    assert call(good, acc=None) == -1
    assert call(good, cache=None) == -1
    assert call(good, cache=fake + 8) == -1                 # misaligned
    assert call(good, hin=None) == -1
    assert call(good, hout=fake + 64) == -1                 # overlaps hidden_in
    for kw in [dict(batch=0), dict(B=0), dict(N=0), dict(max_slots=15),
               dict(row_bytes=8), dict(row_bytes=72), dict(slot_stride=48),
               dict(request_stride=40), dict(plane_stride=-16),
               dict(layer_stride=8), dict(hidden_bytes=20),
               dict(layers=-1)]:
        assert call(variant(**kw)) == -1, kw
    # nothing to move: no planes and no hidden states
    assert call(variant(layers=0, hidden_bytes=0), cache=None, hin=None,
                hout=None) == 0


def test_stall_hook_argument_checks(P):
    lib = P.LIB
    assert lib.pctree_debug_stall_stage(-2, 10**9) == -1
    assert lib.pctree_debug_stall_stage(1, 10) == -1
    assert lib.pctree_debug_stall_stage(1, 2 * 10**10) == -1
    assert lib.pctree_debug_stall_stage(-1, 10**9) == 0      # the default


def test_batch1_qwen3_rounds_fit_the_noalloc_array(P):
    """pctree_draft_noalloc serves batch-1 Qwen3-shaped rounds from its fixed
    16 MiB array: a layout change that outgrows it fails here."""
    limit = 16 << 20
    for V, H, B, k, N in ((151936, 2560, 16, 8, 64), (151936, 2560, 7, 8, 32),
                          (151936, 4096, 7, 8, 64), (151936, 5120, 16, 16, 128)):
        ws = P.pctree_workspace_bytes(P.make_config(V, H, B, k, N, 1))
        assert 0 < ws <= limit, (V, H, B, k, N, ws)


def test_tiled_head_layout_config(P):
    mk = P.make_config
    assert P.pctree_check_config(mk(151936, 2560, 16, 8, 64, 1, 0, "bf16", "parent", "tiled")) == 0
    assert P.pctree_check_config(mk(1024, 64, 4, 4, 8, 1, 0, "f32", "parent", "tiled")) == -1
    bad = mk(1024, 64, 4, 4, 8)
    bad.head_layout = 7
    assert P.pctree_check_config(bad) == -1
    # ceil(V/128) * ceil(H/64) blocks of 128 x 64 bf16
    assert P.pctree_packed_head_bytes(mk(151936, 2560, 16, 8, 64)) == 1187 * 40 * 128 * 64 * 2
    assert P.pctree_packed_head_bytes(mk(3000, 72, 2, 2, 4)) == 24 * 2 * 128 * 64 * 2


def test_outputs_share_one_buffer(P):
    """The round's outputs and any extra tensors are views of one buffer,
    each on a 256-byte boundary and disjoint, so that one copy brings all of
    them back."""
    import torch
    cfg = P.make_config(1000, 64, 5, 4, 24, 3)
    extra = (("accepted_idx", (3, 6), torch.int32), ("bonus", (3,), torch.int32))
    tree = P.alloc_tree(cfg, "cpu", extra=extra)
    base = tree.blob.data_ptr()
    spans = []
    for name in ("n_nodes", "tokens", "parent", "depth", "logp", "position_ids",
                 "mask", "retrieve", "n_leaves", "status"):
        t = getattr(tree, name)
        spans.append((t.data_ptr() - base, t.numel() * t.element_size(), name))
    for name, shape, dt in extra:
        t = tree.extra[name]
        assert tuple(t.shape) == shape and t.dtype == dt
        spans.append((t.data_ptr() - base, t.numel() * t.element_size(), name))
    assert tuple(tree.mask.shape) == (3, 24, 24) and tree.mask.dtype == torch.uint8
    assert tuple(tree.retrieve.shape) == (3, 24, 6)
    spans.sort()
    for (o, n, name), (o2, _, name2) in zip(spans, spans[1:]):
        assert o % 256 == 0, name
        assert o + n <= o2, (name, name2)
    o, n, name = spans[-1]
    assert o % 256 == 0 and o + n <= tree.blob.numel()
