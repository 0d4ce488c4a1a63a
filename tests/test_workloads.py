"""The synthetic input generator: shapes, seeding and the span recipe (CPU only)."""
import numpy as np
import pytest
import torch

from paper_2608_08569_gb300 import workloads as W


@pytest.mark.parametrize("name", sorted(W.CONFIGS))
def test_spans_tile_the_audio_region(name):
    w = W.CONFIGS[name]
    sp = W.make_spans(w)
    assert sp.off[0] == 0 and len(sp.off) == w.batch + 1 and np.all(np.diff(sp.off) >= 1)
    for b in range(w.batch):
        st, en, gr = sp.of(b)
        ab, al = w.audio_begin, w.audio_len[b]
        assert st[0] >= ab and en[-1] <= ab + al
        assert np.all(en > st) and np.all(st[1:] >= en[:-1]) and np.all(gr == 1)
        covered = int((en - st).sum())
        if w.silence_prob == 0:
            assert covered == al and np.all(st[1:] == en[:-1])   # spans cover the audio contiguously
        else:
            assert 0.5 * al < covered < al                       # silence gaps stay uncovered


def test_span_statistics_follow_the_recipe():
    sp = W.make_spans(W.CONFIGS["tiny"])
    assert len(sp.start) == 40 and int((sp.end - sp.start).sum()) == 600
    for name, mean in (("short", 4), ("long", 5), ("stress", 6)):
        w = W.CONFIGS[name]
        sp = W.make_spans(w)
        lens = (sp.end - sp.start).astype(float)
        assert abs(lens.mean() - mean) < 0.15 * mean, (name, lens.mean())
    # one group per word span of mean length 4 gives the paper's ~0.25x stage-1 length ratio
    w = W.CONFIGS["short"]
    sp = W.make_spans(w)
    assert 0.2 < len(sp.start) / w.audio_len[0] < 0.3


def test_budgets_and_shapes():
    c = W.CONFIGS
    assert c["tiny"].budget == (150,) and c["long"].budget == (400,) and c["long_4x"].budget == (2003,)
    assert c["short"].budget == (157,) and c["stress"].budget == (2301,) * 4 and c["stress_4x"].budget == (11506,) * 4
    b = c["batched"]
    assert b.batch == 32 and all(1500 <= a <= 6000 for a in b.audio_len)
    assert all(bud == (a + 256) // 4 for a, bud in zip(b.audio_len, b.budget))
    for w in c.values():
        assert w.q_heads % w.kv_heads == 0 and w.capacity >= w.stride


def test_tensors_are_seeded_and_in_the_cache_dtype():
    w = W.scaled(W.CONFIGS["short"], layers=2)
    k1, v1 = W.make_prefill(w)
    k2, v2 = W.make_prefill(w)
    assert k1.dtype == torch.bfloat16 and k1.shape == (1, 2, 4, w.stride, 128)
    assert torch.equal(k1, k2) and torch.equal(v1, v2)
    q, kn, vn, npos = W.make_steps(w, steps=3)
    assert q.shape == (3, 2, 1, 32, 128) and kn.shape == (3, 2, 1, 4, 128)
    assert npos.tolist() == [[w.in_len[0]], [w.in_len[0] + 1], [w.in_len[0] + 2]]
    # outlier channels of K are scaled
    ch = W.outlier_channels(w)[0, 0]
    kk = k1[0, 0, 0, :w.in_len[0]].float()
    assert kk[:, ch].std() > 4 * kk[:, [c for c in range(128) if c not in ch]].std()


# The five workloads as stated: (name, layers, q/kv heads, head dim, dtype, batch, audio tokens per
# sequence (range for the batched one), text tokens, gamma, decode steps, eviction interval,
# compression ratio of the budget, K outlier scale).
STATED = [
    ("tiny", 1, 2, 1, 64, torch.float32, 1, (600, 600), 32, 0.95, 64, 16, None, None),
    ("short", 48, 32, 4, 128, torch.bfloat16, 1, (375, 375), 256, 0.98, 128, 32, 4, 8.0),
    ("long", 48, 32, 4, 128, torch.bfloat16, 1, (7500, 7500), 512, 0.99, 256, 32, 20, 8.0),
    ("batched", 48, 32, 4, 128, torch.bfloat16, 32, (1500, 6000), 256, 0.98, 512, 32, 4, 8.0),
    ("stress", 48, 32, 4, 128, torch.bfloat16, 4, (45000, 45000), 1024, 0.995, 1024, 32, 20, 16.0),
]


@pytest.mark.parametrize("row", STATED, ids=[r[0] for r in STATED])
def test_configs_are_the_stated_workloads(row):
    name, L, hq, hkv, d, dt, b, (a_lo, a_hi), text, gamma, steps, interval, ratio, outlier = row
    w = W.CONFIGS[name]
    assert (w.layers, w.q_heads, w.kv_heads, w.head_dim, w.dtype, w.batch) == (L, hq, hkv, d, dt, b)
    assert all(a_lo <= a <= a_hi for a in w.audio_len) and w.text_len == text
    assert (w.gamma, w.steps, w.interval) == (gamma, steps, interval)
    if ratio is not None:  # the 10-min 20x budget is the stated 400; every other is (audio + text) / ratio
        assert w.budget == tuple((a + text) // ratio for a in w.audio_len)
        assert w.outliers == 4 and w.outlier_scale == outlier
    assert (w.sink, w.recent_frac) == (4, 0.2)
    # audio at 12.5 tokens per second: 30 s, 10 min, 2-8 min and 60 min
    seconds = {"short": (30, 30), "long": (600, 600), "batched": (120, 480), "stress": (3600, 3600)}.get(name)
    if seconds:
        assert all(seconds[0] * 12.5 <= a <= seconds[1] * 12.5 for a in w.audio_len)


def test_the_60_min_workload_has_its_silence_gaps():
    w = W.CONFIGS["stress"]
    sp = W.make_spans(w)
    n_gaps, n_spans = 0, 0
    for b in range(w.batch):
        st, en, _ = sp.of(b)
        gaps = st[1:] - en[:-1]
        assert np.all((gaps == 0) | (gaps >= 20))   # a silence lasts 20-60 tokens
        n_gaps += int((gaps > 0).sum())
        n_spans += len(st)
    assert 0.035 < n_gaps / n_spans < 0.065         # about 5% of draws are silences
