"""Seeded input generators: determinism, shapes and number formats."""
import numpy as np

from workloads import (WORKLOADS, bf16_bits_to_f32, draw_request,
                       draw_round, f32_to_bf16_bits, target_for_tree)


def test_bf16_rounding_ties_to_even():
    x = np.array([1.0, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -2.5, 3.0e-3],
                 dtype=np.float32)
    bits = f32_to_bf16_bits(x)
    assert bits[:4].tolist() == [0x3F80, 0x3F80, 0x3F82, 0xC020]
    back = bf16_bits_to_f32(bits)
    assert abs(back[4] - 3.0e-3) <= 3.0e-3 * 2.0 ** -8


def test_tiny_round_is_deterministic_and_shaped():
    wl = WORKLOADS["tiny"]
    a, b = draw_round(wl), draw_round(wl)
    assert np.array_equal(a.L, b.L) and np.array_equal(a.W_out, b.W_out)
    assert a.L.shape == (1, wl.B, wl.V) and a.E_in.shape == (wl.V, wl.H)
    assert a.greedy.shape == (1, wl.B + 1)
    # one planted token per depth, in range
    assert a.likely.shape == (1, wl.B)
    assert ((a.likely >= 0) & (a.likely < wl.V)).all()


def test_requests_are_independent_of_batch_slicing():
    wl = WORKLOADS["tiny"].with_(batch=3, V=300, H=8)
    full = draw_round(wl)
    L1, root1, g1, _ = draw_request(wl, 1)
    assert np.array_equal(full.L[1], L1) and full.root[1] == root1


def test_zipf_logits_shape_small():
    wl = WORKLOADS["14b_b16_bs32"].with_(V=2000, H=16, batch=2, B=4)
    L, root, g, likely = draw_request(wl, 0)
    assert L.shape == (4, 2000) and L.dtype == np.float32
    assert np.isfinite(L).all() and (np.argmax(L, 1) == likely).all()


def test_target_for_tree():
    g = np.array([[5, 6, 7]])
    depth = np.array([[0, 1, 1, 2, -1]])
    assert target_for_tree(g, depth).tolist() == [[5, 6, 6, 7, -1]]
