"""Planted mistakes in the compaction oracle (on the CPU) must each fail one
of the pins in ``tests/test_compact_oracle.py``."""
import numpy as np
import pytest

from oracle import compact_oracle as co
from tests import test_compact_oracle as pins


def _variant(kind):
    def wrong(cache, hidden_in, hidden_out, accepted_idx, accepted_len,
              prefix_len, n_tree):
        before = np.asarray(cache)
        after = before.copy()
        h_after = None if hidden_out is None else np.asarray(hidden_out).copy()
        batch, slots = before.shape[2], before.shape[3]
        valid = np.zeros(batch, dtype=bool)
        for r in range(batch):
            T, L, acc = int(prefix_len[r]), int(accepted_len[r]), accepted_idx[r]
            if kind != "no_checks" and (T < 0 or T + n_tree > slots or
                                        not co.path_ok(acc, L, n_tree)):
                continue
            valid[r] = True
            n_rows = L if kind == "drop_last" else L + 1
            for j in range(max(n_rows, 0)):
                a = int(acc[j])
                if kind == "scatter":
                    after[:, :, r, T + a] = before[:, :, r, T + j]
                elif kind == "no_prefix_on_source":
                    after[:, :, r, T + j] = before[:, :, r, a]
                elif kind == "other_request":
                    after[:, :, r, T + j] = before[:, :, (r + 1) % batch, T + a]
                else:
                    after[:, :, r, T + j] = before[:, :, r, T + a]
                if h_after is not None:
                    h_after[r, j] = hidden_in[r, j if kind == "hidden_in_place" else a]
        return after, h_after, valid
    return wrong


def _all_pins():
    yield lambda: pins.test_rows_come_from_the_accepted_nodes("small")
    yield lambda: pins.test_rows_come_from_the_accepted_nodes("ragged")
    yield pins.test_identity_and_empty_paths_change_nothing
    yield pins.test_prefix_overflow_is_invalid
    yield pins.test_draft_accept_compact_chain
    for bad in [("decreasing", lambda a, n: a.__setitem__(slice(1, 3), [5, 3]), None),
                ("len beyond B", None, 99)]:
        yield lambda bad=bad: pins.test_invalid_paths_leave_the_request_untouched(bad)


@pytest.mark.parametrize("kind", ["scatter", "no_prefix_on_source",
                                  "other_request", "drop_last", "no_checks",
                                  "hidden_in_place"])
def test_planted_mistake_is_caught(kind, monkeypatch):
    monkeypatch.setattr(co, "compact", _variant(kind))
    caught = False
    for pin in _all_pins():
        try:
            pin()
        except (AssertionError, IndexError, ValueError):
            caught = True
            break
    assert caught, kind


def test_unplanted_variant_passes(monkeypatch):
    monkeypatch.setattr(co, "compact", _variant("none"))
    for pin in _all_pins():
        pin()
