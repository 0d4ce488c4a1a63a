"""The host-side Eq. 3 helper of the C library (voxzip_segments_to_spans: confidence filter,
time-to-index map) against the oracle's, bit-exact, on the hand-worked fixture, synthetic ASR
output and edge cases. It is host code, so these run without a GPU."""
import json
import os

import numpy as np
import pytest

import oracle
from paper_2608_08569_gb300 import VoxZipError, voxzip_segments_to_spans
from paper_2608_08569_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _same(a, b):
    for k in ("start", "end", "groups", "seg_index"):
        np.testing.assert_array_equal(a[k], b[k], err_msg=k)


def test_golden_fixture():
    g = json.load(open(os.path.join(GOLDEN, "eq3_segments.json")))
    r = voxzip_segments_to_spans(g["t_start"], g["t_end"], g["confidence"], g["text_len"], g["tau_total"], g["La"],
                                 g["audio_begin"], g["threshold"])
    np.testing.assert_array_equal(r["start"], g["expected_start"])
    np.testing.assert_array_equal(r["end"], g["expected_end"])
    np.testing.assert_array_equal(r["groups"], g["expected_groups"])
    np.testing.assert_array_equal(r["seg_index"], g["expected_seg_index"])
    e = g["boundary"]  # a segment on exact token boundaries (the order of Eq. 3's operations shows)
    r = voxzip_segments_to_spans(e["t_start"], e["t_end"], e["confidence"], e["text_len"], e["tau_total"], e["La"],
                                 e["audio_begin"], e["threshold"])
    np.testing.assert_array_equal(r["start"], e["expected_start"])
    np.testing.assert_array_equal(r["end"], e["expected_end"])
    e = g["nested"]  # a segment inside the previous one: an empty span that keeps its text rows
    r = voxzip_segments_to_spans(e["t_start"], e["t_end"], e["confidence"], e["text_len"], e["tau_total"], e["La"],
                                 e["audio_begin"], e["threshold"])
    for k in ("start", "end", "groups", "seg_index"):
        np.testing.assert_array_equal(r[k], e["expected_" + k], err_msg=k)


@pytest.mark.parametrize("name", sorted(W.EMBED_CONFIGS))
def test_synthetic_asr_matches_oracle(name):
    w = W.EMBED_CONFIGS[name]
    for b, s in enumerate(W.make_segments(w)):
        args = (s.t_start, s.t_end, s.confidence, s.text_len, s.tau_total, w.audio_len[b], w.audio_begin)
        for thr in (0.3, 0.0, 0.95, -1.0):
            _same(voxzip_segments_to_spans(*args, threshold=thr), oracle.segments_to_spans(*args, threshold=thr))


def test_random_edges_match_oracle():
    rng = np.random.default_rng(7)
    for trial in range(300):
        n = int(rng.integers(0, 15))
        tau = float(rng.choice([1.0, 48.0, 3600.0, float(rng.uniform(0.1, 100.0))]))
        La = int(rng.choice([0, 1, 7, 600, 45000]))
        # times may leave [0, tau], sit on token boundaries, be equal, or be infinite
        ts = np.sort(np.concatenate([rng.uniform(-0.2 * tau, 1.2 * tau, n // 2),
                                     np.round(rng.uniform(0, tau, n - n // 2) * La / tau) * tau / max(La, 1)]))
        te = ts + rng.choice([0.0, 0.0, 1.0], n) * rng.uniform(0, 0.3 * tau, n)
        if n and rng.random() < 0.1:
            te[-1] = np.inf
        if n and rng.random() < 0.1:
            ts[0] = -np.inf
        conf = rng.choice([0.3, 0.29999999, 0.30000001, 0.9, 0.1], n)
        tl = rng.integers(1, 9, n)
        ab = int(rng.integers(0, 100))
        args = (ts, te, conf, tl, tau, La, ab)
        _same(voxzip_segments_to_spans(*args), oracle.segments_to_spans(*args))


@pytest.mark.parametrize("args", [
    ([1.0, 0.5], [2.0, 2.0], [1.0, 1.0], [1, 1], 2.0, 20),   # unsorted
    ([0.0], [1.0], [1.0], [0], 2.0, 20),                       # no text tokens
    ([0.0], [1.0], [1.0], [1], 0.0, 20),                       # zero duration
    ([0.0], [1.0], [1.0], [1], float("inf"), 20),              # infinite duration
    ([1.0], [0.5], [1.0], [1], 2.0, 20),                       # ends before it starts
    ([float("nan")], [1.0], [1.0], [1], 2.0, 20),              # NaN time
    ([0.0], [1.0], [1.0], [1], 2.0, -1),                       # negative audio length
])
def test_rejected_like_the_oracle(args):
    with pytest.raises(VoxZipError):
        voxzip_segments_to_spans(*args)
    with pytest.raises(oracle.OracleError):
        oracle.segments_to_spans(*args)


def test_embed_generator_shape():
    """The synthetic ASR output is sorted, inside the audio, and its kept segments compress the
    covered audio to about a quarter (the paper's ~0.25x)."""
    w = W.EMBED_CONFIGS["embed_stress"]
    for b, s in enumerate(W.make_segments(w)):
        assert np.all(np.diff(s.t_start) >= 0) and np.all(s.t_end >= s.t_start)
        assert s.t_end.max() <= s.tau_total + 1.0 and s.t_start.min() >= 0.0
        r = voxzip_segments_to_spans(s.t_start, s.t_end, s.confidence, s.text_len, s.tau_total, w.audio_len[b],
                                     w.audio_begin)
        covered = int((r["end"] - r["start"]).sum())
        assert 0.8 * w.audio_len[b] < covered < w.audio_len[b]
        assert 0.22 < r["groups"].sum() / covered < 0.3
