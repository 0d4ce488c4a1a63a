"""Seeded synthetic workloads shaped like the Qwen3-Omni thinker (48 layers, GQA 32/4, D = 128).

This module only draws inputs: ASR-like token spans, prefilled K/V, per-step q/k/v. It holds none
of the compression arithmetic; the CUDA path and the oracle both consume what it produces.

Recipe (shared by tests and the benchmark):
  * prompt layout: text_len // 8 text tokens, then the audio tokens, then the remaining text;
  * spans tile the audio region left to right; each segment is, with probability
    ``silence_prob``, an uncovered silence gap of U{20..60} tokens (kept 1:1 as background),
    otherwise a span whose length is geometric with the configured mean (the last one clipped);
    the tiny configuration instead draws 40 lengths U{1..30} and rescales them to cover the
    audio exactly (largest-remainder rounding, each >= 1). Every span gets n_groups = 1, one
    anchor per ASR word;
  * K ~ N(0, 1) with ``outliers`` fixed channels per (layer, kv-head) scaled by ``outlier_scale``;
    V ~ N(0, 1); q = 0.5 N(0, 1) + 0.5 sum_k c_k u_k with 8 anchor directions u_k ~ N(0, I) per
    (layer, kv-head) and c ~ N(0, 1) / sqrt(8) per query; the tiny configuration draws q, K, V
    from N(0, 1) plainly. New keys and values of each decode step follow the K and V laws;
  * all values are rounded once to the cache dtype. Random numbers come from torch generators
    on the device the tensors are made on, one stream per (workload seed, kind, sequence or step,
    layer), so any slice can be drawn alone; CPU and CUDA streams differ, so both sides of a
    comparison always receive the same drawn tensors.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field, replace

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    dtype: torch.dtype
    batch: int
    audio_len: tuple            # per sequence
    text_len: int
    budget: tuple               # per sequence
    gamma: float
    steps: int
    interval: int
    span_kind: str = "geometric"    # "geometric" | "uniform40" | "unit"
    span_mean: float = 4.0
    silence_prob: float = 0.0
    outliers: int = 4
    outlier_scale: float = 8.0
    anchor_dirs: int = 8
    plain_normal: bool = False
    seed: int = 0
    sink: int = 4
    recent_frac: float = 0.2
    description: str = field(default="", compare=False)

    @property
    def group(self) -> int:
        return self.q_heads // self.kv_heads

    @property
    def in_len(self) -> tuple:
        return tuple(a + self.text_len for a in self.audio_len)

    @property
    def audio_begin(self) -> int:
        return self.text_len // 8

    @property
    def stride(self) -> int:
        return max(self.in_len)

    @property
    def capacity(self) -> int:
        # an upper bound needing no knowledge of stage 1: every prompt token plus every step
        return self.stride + self.steps

    @property
    def units(self) -> int:
        return self.batch * self.layers * self.kv_heads


def _ratio_budget(audio, text, ratio):
    return tuple((a + text) // ratio for a in audio)


def _make_configs():
    qwen = dict(layers=48, q_heads=32, kv_heads=4, head_dim=128, dtype=torch.bfloat16)
    c = {}
    c["tiny"] = Workload("tiny", layers=1, q_heads=2, kv_heads=1, head_dim=64, dtype=torch.float32, batch=1,
                         audio_len=(600,), text_len=32, budget=(150,), gamma=0.95, steps=64, interval=16,
                         span_kind="uniform40", plain_normal=True, outliers=0, seed=0,
                         description="1 layer, 2/1 heads, D 64, fp32; 600 audio + 32 text tokens; 40 spans")
    c["tiny_identity"] = replace(c["tiny"], name="tiny_identity", span_kind="unit",
                                 description="tiny with length-1 spans: stage 1 is the identity")
    c["short"] = Workload("short", **qwen, batch=1, audio_len=(375,), text_len=256,
                          budget=_ratio_budget((375,), 256, 4), gamma=0.98, steps=128, interval=32,
                          span_mean=4.0, seed=1, description="30 s clip, 4x budget")
    c["long"] = Workload("long", **qwen, batch=1, audio_len=(7500,), text_len=512, budget=(400,), gamma=0.99,
                         steps=256, interval=32, span_mean=5.0, seed=2, description="10 min audio, 20x budget")
    c["long_4x"] = replace(c["long"], name="long_4x", budget=_ratio_budget((7500,), 512, 4),
                           description="10 min audio, 4x budget")
    rng = np.random.default_rng(4)
    audio4 = tuple(int(x) for x in rng.integers(1500, 6001, 32))
    c["batched"] = Workload("batched", **qwen, batch=32, audio_len=audio4, text_len=256,
                            budget=_ratio_budget(audio4, 256, 4), gamma=0.98, steps=512, interval=32,
                            span_mean=4.0, seed=3, description="32 sequences of 2-8 min audio, 4x budget")
    c["stress"] = Workload("stress", **qwen, batch=4, audio_len=(45000,) * 4, text_len=1024,
                           budget=_ratio_budget((45000,) * 4, 1024, 20), gamma=0.995, steps=1024, interval=32,
                           span_mean=6.0, silence_prob=0.05, outlier_scale=16.0, seed=5,
                           description="4 x 60 min audio, 20x budget")
    c["stress_4x"] = replace(c["stress"], name="stress_4x", budget=_ratio_budget((45000,) * 4, 1024, 4),
                             description="4 x 60 min audio, 4x budget")
    return c


CONFIGS = _make_configs()


def scaled(w: Workload, *, layers=None, batch=None, steps=None, audio_scale=None, name=None) -> Workload:
    """A smaller copy of a workload (fewer layers, sequences, steps or audio) for quick checks."""
    kw = {}
    if layers is not None:
        kw["layers"] = layers
    if batch is not None:
        kw["batch"] = batch
        kw["audio_len"] = w.audio_len[:batch]
        kw["budget"] = w.budget[:batch]
    if steps is not None:
        kw["steps"] = steps
    if audio_scale is not None:
        audio = tuple(max(1, int(a * audio_scale)) for a in kw.get("audio_len", w.audio_len))
        kw["audio_len"] = audio
        ratio = (w.audio_len[0] + w.text_len) / w.budget[0]
        kw["budget"] = tuple(max(w.sink + 2, int((a + w.text_len) / ratio)) for a in audio)
    return replace(w, name=name or (w.name + "_scaled"), **kw)


# ----------------------------------------------------------------------------- spans

def _spans_one(w: Workload, b: int, rng: np.random.Generator):
    ab, al = w.audio_begin, w.audio_len[b]
    starts, ends = [], []
    if w.span_kind == "unit":
        starts = list(range(ab, ab + al))
        ends = [s + 1 for s in starts]
    elif w.span_kind == "uniform40":
        raw = rng.integers(1, 31, 40).astype(np.float64)
        exact = raw * al / raw.sum()
        lens = np.maximum(1, np.floor(exact)).astype(np.int64)
        short = al - int(lens.sum())
        order = np.argsort(-(exact - np.floor(exact)), kind="stable")
        k = 0
        while short > 0:
            lens[order[k % 40]] += 1
            short -= 1
            k += 1
        while short < 0:  # only if the floors of 1 overshot; take from the longest
            i = int(np.argmax(lens))
            lens[i] -= 1
            short += 1
        t = ab
        for ln in lens:
            starts.append(t)
            ends.append(t + int(ln))
            t += int(ln)
    else:
        t = ab
        while t < ab + al:
            if w.silence_prob > 0 and rng.random() < w.silence_prob:
                t = min(ab + al, t + int(rng.integers(20, 61)))
                continue
            ln = int(rng.geometric(1.0 / w.span_mean))
            e = min(ab + al, t + ln)
            starts.append(t)
            ends.append(e)
            t = e
    groups = [1] * len(starts)
    return starts, ends, groups


@dataclass
class Spans:
    """CSR span arrays for all sequences (host numpy, int32)."""
    off: np.ndarray
    start: np.ndarray
    end: np.ndarray
    groups: np.ndarray

    def of(self, b: int):
        s, e = int(self.off[b]), int(self.off[b + 1])
        return self.start[s:e], self.end[s:e], self.groups[s:e]


def make_spans(w: Workload) -> Spans:
    rng = np.random.default_rng(1000 + w.seed)
    off, st, en, gr = [0], [], [], []
    for b in range(w.batch):
        s, e, g = _spans_one(w, b, rng)
        st += s
        en += e
        gr += g
        off.append(len(st))
    as32 = lambda x: np.asarray(x, dtype=np.int32)
    return Spans(as32(off), as32(st), as32(en), as32(gr))


# ----------------------------------------------------------------------------- tensors

def _gen(w: Workload, device, *key) -> torch.Generator:
    """A generator seeded by (workload seed, key...): each slice has its own stream."""
    h = w.seed
    for k in key:
        h = (h * 1_000_003 + int(k) + 1) % (2 ** 62)
    g = torch.Generator(device=device)
    g.manual_seed(h)
    return g


def outlier_channels(w: Workload) -> np.ndarray:
    """[L][Hkv][outliers] channel indices scaled in K (fixed per layer and kv-head)."""
    rng = np.random.default_rng(2000 + w.seed)
    if w.outliers == 0:
        return np.zeros((w.layers, w.kv_heads, 0), np.int64)
    return np.stack([np.stack([rng.choice(w.head_dim, w.outliers, replace=False) for _ in range(w.kv_heads)])
                     for _ in range(w.layers)])


def _k_scale(w: Workload, device) -> torch.Tensor:
    """[L][Hkv][D] per-channel multiplier of K (1, or outlier_scale on the outlier channels)."""
    s = torch.ones(w.layers, w.kv_heads, w.head_dim)
    ch = outlier_channels(w)
    for l in range(w.layers):
        for h in range(w.kv_heads):
            s[l, h, torch.from_numpy(ch[l, h])] = w.outlier_scale
    return s.to(device)


_K, _V, _Q, _C, _KN, _VN, _U = range(7)   # stream kinds


def prefill_slice(w: Workload, b: int, l: int, device="cpu", ks=None):
    """K and V rows [Hkv][in_len[b]][D] of sequence b, layer l (cache dtype)."""
    n, H, D = w.in_len[b], w.kv_heads, w.head_dim
    ks = _k_scale(w, device) if ks is None else ks
    x = torch.randn(H, n, D, generator=_gen(w, device, _K, b, l), device=device)
    k = (x * ks[l][:, None, :]).to(w.dtype)
    v = torch.randn(H, n, D, generator=_gen(w, device, _V, b, l), device=device).to(w.dtype)
    return k, v


def make_prefill(w: Workload, device="cpu"):
    """Prefilled K and V, [B][L][Hkv][stride][D] in the cache dtype; rows past in_len are zero."""
    B, L, H, D, S = w.batch, w.layers, w.kv_heads, w.head_dim, w.stride
    k = torch.zeros(B, L, H, S, D, dtype=w.dtype, device=device)
    v = torch.zeros(B, L, H, S, D, dtype=w.dtype, device=device)
    ks = _k_scale(w, device)
    for b in range(B):
        n = w.in_len[b]
        for l in range(L):
            k[b, l, :, :n], v[b, l, :, :n] = prefill_slice(w, b, l, device, ks)
    return k, v


def step_slice(w: Workload, t: int, l: int, device="cpu", ks=None, u=None):
    """Decode inputs of step t (0-based), layer l: q [B][Hq][D], k_new and v_new [B][Hkv][D]."""
    B, Hq, H, D, G = w.batch, w.q_heads, w.kv_heads, w.head_dim, w.group
    ks = _k_scale(w, device) if ks is None else ks
    if w.plain_normal:
        q = torch.randn(B, Hq, D, generator=_gen(w, device, _Q, t, l), device=device)
    else:
        if u is None:   # anchor directions of layer l: [Hkv][A][D]
            u = torch.randn(H, w.anchor_dirs, D, generator=_gen(w, device, _U, l), device=device)
        noise = torch.randn(B, Hq, D, generator=_gen(w, device, _Q, t, l), device=device)
        c = torch.randn(B, Hq, w.anchor_dirs, generator=_gen(w, device, _C, t, l), device=device)
        mix = torch.einsum("bha,had->bhd", c / math.sqrt(w.anchor_dirs), u.repeat_interleave(G, dim=0))
        q = 0.5 * noise + 0.5 * mix
    kn = torch.randn(B, H, D, generator=_gen(w, device, _KN, t, l), device=device) * ks[l][None]
    vn = torch.randn(B, H, D, generator=_gen(w, device, _VN, t, l), device=device)
    return q.to(w.dtype), kn.to(w.dtype), vn.to(w.dtype)


def make_steps(w: Workload, device="cpu", steps=None):
    """Decode inputs for every step: q [S][L][B][Hq][D], k_new and v_new [S][L][B][Hkv][D],
    new_pos [S][B] int32 (the prompt length plus the step index)."""
    S = w.steps if steps is None else steps
    B, L, Hq, H, D = w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim
    q = torch.empty(S, L, B, Hq, D, dtype=w.dtype, device=device)
    kn = torch.empty(S, L, B, H, D, dtype=w.dtype, device=device)
    vn = torch.empty(S, L, B, H, D, dtype=w.dtype, device=device)
    ks = _k_scale(w, device)
    us = [None if w.plain_normal else
          torch.randn(H, w.anchor_dirs, D, generator=_gen(w, device, _U, l), device=device) for l in range(L)]
    for t in range(S):
        for l in range(L):
            q[t, l], kn[t, l], vn[t, l] = step_slice(w, t, l, device, ks, us[l])
    new_pos = torch.tensor([[w.in_len[b] + t for b in range(B)] for t in range(S)], dtype=torch.int32,
                           device=device)
    return q, kn, vn, new_pos


def unit_inputs(w: Workload, spans: Spans, k_pre, v_pre, q, kn, vn, new_pos, b: int, l: int, h: int,
                steps=None):
    """One unit's inputs as float64 numpy arrays, in the oracle's argument layout."""
    S = q.shape[0] if steps is None else steps
    G = w.group
    n = w.in_len[b]
    st, en, gr = spans.of(b)
    f64 = lambda t: t.detach().to("cpu", torch.float64).numpy()
    return dict(xk=f64(k_pre[b, l, h, :n]), xv=f64(v_pre[b, l, h, :n]), in_len=n, audio_begin=w.audio_begin,
                audio_len=w.audio_len[b], span_start=st, span_end=en, span_groups=gr,
                q=f64(q[:S, l, b, h * G:(h + 1) * G]), k_new=f64(kn[:S, l, b, h]), v_new=f64(vn[:S, l, b, h]),
                new_pos=new_pos[:S, b].cpu().numpy())


def unit_inputs_cpu(w: Workload, spans: Spans, b: int, l: int, h: int, steps=None):
    """One unit's inputs drawn on the CPU alone (the same recipe; CPU generator streams), for
    timing the oracle on a sample without building the whole workload."""
    S = w.steps if steps is None else steps
    G = w.group
    ks = _k_scale(w, "cpu")
    k, v = prefill_slice(w, b, l, "cpu", ks)
    u = None if w.plain_normal else torch.randn(w.kv_heads, w.anchor_dirs, w.head_dim,
                                                  generator=_gen(w, "cpu", _U, l))
    qs, kns, vns = [], [], []
    for t in range(S):
        q, kn, vn = step_slice(w, t, l, "cpu", ks, u)
        qs.append(q[b, h * G:(h + 1) * G])
        kns.append(kn[b, h])
        vns.append(vn[b, h])
    st, en, gr = spans.of(b)
    f64 = lambda t: t.to(torch.float64).numpy()
    return dict(xk=f64(k[h]), xv=f64(v[h]), in_len=w.in_len[b], audio_begin=w.audio_begin,
                audio_len=w.audio_len[b], span_start=st, span_end=en, span_groups=gr,
                q=f64(torch.stack(qs)), k_new=f64(torch.stack(kns)), v_new=f64(torch.stack(vns)),
                new_pos=np.array([w.in_len[b] + t for t in range(S)], np.int32))


# ----------------------------------------------------------------------------- embedding level

@dataclass(frozen=True)
class EmbedWorkload:
    """Stage 1 where the paper runs it: prompt embeddings [B][in_len][d_model] with an audio region,
    and the ASR output of that audio as timed segments.

    Recipe: the prompt is text_len // 8 text tokens, the audio tokens (12.5 per second, as the
    Qwen3-Omni audio encoder emits), then the rest of the text. The audio is cut left to right
    into ASR segments of U[seg_sec] seconds separated, with probability gap_prob, by silences of
    U[gap_sec] seconds; segment times are the token boundaries jittered by up to +-jitter_tok
    tokens (so the floor of Eq. 3 matters) and kept sorted; a segment's transcription has
    L_t = max(1, round(text_per_sec x duration)) tokens (about 0.26 text tokens per audio token,
    the paper's ~0.25x); its confidence is U(0, 0.3) with probability low_conf_prob, else
    U(0.3, 1). Embeddings are N(0, 1) (audio) and 0.5 N(0, 1) (text) rounded to the dtype; text
    embeddings are drawn for every segment, kept or not, in segment order."""
    name: str
    batch: int
    audio_len: tuple
    text_len: int
    d_model: int
    dtype: torch.dtype = torch.bfloat16
    rate: float = 12.5
    seg_sec: tuple = (2.0, 10.0)
    gap_prob: float = 0.1
    gap_sec: tuple = (0.5, 3.0)
    jitter_tok: float = 0.4
    text_per_sec: float = 3.2
    low_conf_prob: float = 0.1
    seed: int = 0
    description: str = field(default="", compare=False)

    @property
    def in_len(self) -> tuple:
        return tuple(a + self.text_len for a in self.audio_len)

    @property
    def audio_begin(self) -> int:
        return self.text_len // 8

    @property
    def stride(self) -> int:
        return max(self.in_len)

    @property
    def capacity(self) -> int:
        return self.stride


def _make_embed_configs():
    c = {}
    c["embed_tiny"] = EmbedWorkload("embed_tiny", batch=2, audio_len=(600, 430), text_len=32, d_model=256,
                                    dtype=torch.float32, seed=10, description="2 clips, d 256, fp32")
    c["embed_short"] = EmbedWorkload("embed_short", batch=1, audio_len=(375,), text_len=256, d_model=2048,
                                     seed=11, description="30 s clip, d 2048, bf16")
    c["embed_stress"] = EmbedWorkload("embed_stress", batch=4, audio_len=(45000,) * 4, text_len=1024, d_model=2048,
                                      seed=12, description="4 x 60 min audio, d 2048, bf16")
    return c


EMBED_CONFIGS = _make_embed_configs()


@dataclass
class Segments:
    """ASR output of one sequence: per segment start / end time (s), confidence, text tokens."""
    t_start: np.ndarray
    t_end: np.ndarray
    confidence: np.ndarray
    text_len: np.ndarray
    tau_total: float


def make_segments(w: EmbedWorkload) -> list:
    rng = np.random.default_rng(3000 + w.seed)
    out = []
    for b in range(w.batch):
        La = w.audio_len[b]
        tau = La / w.rate
        ts, te, cf, tl = [], [], [], []
        t = 0.0
        while t < tau:
            if rng.random() < w.gap_prob:
                t += float(rng.uniform(*w.gap_sec))
                continue
            dur = float(rng.uniform(*w.seg_sec))
            e = min(tau, t + dur)
            j0, j1 = rng.uniform(-w.jitter_tok, w.jitter_tok, 2) / w.rate
            s_t = max(0.0, t + j0) if not ts else max(ts[-1], t + j0)
            ts.append(s_t)
            te.append(max(s_t, e + j1))
            cf.append(float(rng.uniform(0.0, 0.3)) if rng.random() < w.low_conf_prob else float(rng.uniform(0.3, 1.0)))
            tl.append(max(1, int(round(w.text_per_sec * (e - t)))))
            t = e
        out.append(Segments(np.asarray(ts), np.asarray(te), np.asarray(cf), np.asarray(tl, np.int32), tau))
    return out


_E, _ET = 7, 8   # stream kinds of the embedding level


def make_embeddings(w: EmbedWorkload, device="cpu"):
    """Prompt embeddings [B][stride][d_model] in the dtype; rows past in_len are zero."""
    e = torch.zeros(w.batch, w.stride, w.d_model, dtype=w.dtype, device=device)
    for b in range(w.batch):
        n = w.in_len[b]
        e[b, :n] = torch.randn(n, w.d_model, generator=_gen(w, device, _E, b), device=device).to(w.dtype)
    return e


def make_text_embeddings(w: EmbedWorkload, segments: list, device="cpu"):
    """Embedded transcriptions of every segment, [B][max rows][d_model]: sequence b's segments'
    text tokens concatenated in segment order (rows past them zero)."""
    rows = [int(s.text_len.sum()) for s in segments]
    t = torch.zeros(w.batch, max(1, max(rows)), w.d_model, dtype=w.dtype, device=device)
    for b in range(w.batch):
        if rows[b]:
            x = torch.randn(rows[b], w.d_model, generator=_gen(w, device, _ET, b), device=device)
            t[b, :rows[b]] = (0.5 * x).to(w.dtype)
    return t
