"""bench.py's accounting, on the CPU: the algorithmic bytes behind every roofline fraction it
reports, the census of rows an eviction moved (checked against the oracle's own eviction of the
same units, Eq. 7-9, ordered and hole-filling), the per-launch durations it reads from an
instrumented graph's events, and the rule that a committed profile's DRAM ratio is used only while
the kernel's sources are the ones it was captured on."""
import hashlib

import numpy as np
import pytest
import torch

import bench
import oracle
from paper_2608_08569_gb300 import workloads as W


def _bytes(shape, dtype):
    return int(np.prod(shape)) * np.dtype(dtype).itemsize


@pytest.mark.parametrize("name", ["tiny", "short", "stress"])
def test_decode_bytes_is_a_census_of_what_one_step_touches(name):
    w = W.CONFIGS[name]
    e = np.float32 if w.dtype == torch.float32 else np.uint16  # bf16 stored as 2-byte words
    D, G = w.head_dim, w.group
    rng = np.random.default_rng(0)
    n_after = rng.integers(1, 5000, size=w.batch)
    total = 0
    for n in n_after:
        unit = (_bytes((n, D), e) * 2            # every cached K and V row, read once
                + _bytes((n,), np.float32) * 2   # each score read and written
                + _bytes((G, D), e) * 2          # the group's queries in, its outputs out
                + _bytes((D,), e) * 2            # k_new and v_new in
                + _bytes((D,), e) * 2            # the appended K and V rows written
                + _bytes((1,), np.int32))        # the appended position
        total += unit * w.layers * w.kv_heads
    assert bench.decode_bytes(w, n_after) == total


def test_evict_bytes_counts_the_selection_and_every_moved_row_both_ways():
    w = W.CONFIGS["stress"]
    n_before = np.array([2333, 2333, 2400])
    moved = np.array([10, 0, 2000])
    row = _bytes((w.head_dim,), np.uint16) * 2 + 4 + 4  # K and V, score, position
    assert bench.evict_bytes(w, n_before, moved) == 8 * n_before.sum() + 2 * row * moved.sum()


def _units(rng, n_units, C, budgets, extra):
    """Seeded unit states: n = budget + extra slots in time order, distinct scores."""
    caches = []
    for u in range(n_units):
        n = budgets[u] + extra[u]
        K = rng.standard_normal((n, 4))
        c = oracle.UnitCache.from_rows(C, K, K, np.arange(n, dtype=np.int32) * 3 + 7,
                                       score=rng.random(n) + np.arange(n) * 1e-9)
        caches.append(c)
    return caches


@pytest.mark.parametrize("fill", [False, True])
def test_moved_rows_matches_the_oracles_eviction(fill):
    rng = np.random.default_rng(3)
    C, n_units = 600, 6
    budgets = [150, 150, 200, 300, 120, 400]
    extra = [32, 0, 1, 250, 32, 16]  # one unit at its budget (no eviction)
    caches = _units(rng, n_units, C, budgets, extra)
    pos_before = torch.tensor(np.stack([c.pos for c in caches]))
    n_before = torch.tensor([c.n for c in caches], dtype=torch.int32)
    expected_moved, expected_n = [], []
    for c, bud in zip(caches, budgets):
        n0 = c.n
        if n0 <= bud:  # no eviction: no row moves, and its length is not listed
            expected_moved.append(0)
            continue
        _, kept = oracle.evict(c, bud, fill=fill)
        slots = np.flatnonzero(kept)
        if fill:  # kept rows at or beyond the budget fill the evicted slots below it
            expected_moved.append(int((slots >= bud).sum()))
        else:     # ordered compaction: a kept row moves iff an evicted slot precedes it
            expected_moved.append(int((slots != np.arange(len(slots))).sum()))
        expected_n.append(n0)
    pos_after = torch.tensor(np.stack([c.pos for c in caches]))
    n_after = torch.tensor([c.n for c in caches], dtype=torch.int32)
    nb, moved = bench.moved_rows(pos_before, n_before, pos_after, n_after)
    assert list(nb) == expected_n           # lengths of the units that evicted
    assert list(moved) == expected_moved    # rows moved, one count per unit
    if not fill:
        assert sum(expected_moved) > 0


class _Ev:
    def __init__(self, t):
        self.t = t

    def elapsed_time(self, other):
        return other.t - self.t


def test_launch_durations_spread_a_run_of_decodes_over_its_launches():
    events = [("decode", _Ev(0.0), _Ev(3.2), 32), ("evict", _Ev(3.2), _Ev(3.5), 1),
              ("decode", _Ev(3.5), _Ev(5.1), 16)]
    dec, ev = bench.launch_durations(events)
    assert len(dec) == 48 and len(ev) == 1
    assert dec[:32] == [pytest.approx(0.1)] * 32 and dec[32:] == [pytest.approx(0.1)] * 16
    assert ev == [pytest.approx(0.3)]


def test_profile_ratio_is_used_only_for_the_sources_it_was_captured_on(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2608_08569_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "k.cu").write_text("kernel A\n")
    (csrc / "c.cuh").write_text("common\n")
    h = hashlib.sha256(b"kernel A\n" + b"common\n").hexdigest()[:16]
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "k.md").write_text(f"- `traffic_ratio: 1.031`\n- `source_sha256: {h}` (k.cu, c.cuh)\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.profiled_traffic_ratio("k.md", ["k.cu", "c.cuh"]) == pytest.approx(1.031)
    assert bench.profiled_traffic_ratio("k.md", ["c.cuh", "k.cu"]) is None  # order is part of the hash
    (csrc / "k.cu").write_text("kernel B\n")
    assert bench.profiled_traffic_ratio("k.md", ["k.cu", "c.cuh"]) is None
    assert bench.profiled_traffic_ratio("missing.md", ["k.cu"]) is None

