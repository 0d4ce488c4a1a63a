"""Python access to the fp64 CPU oracle in ``voxzip_oracle.c``.

TEST INFRASTRUCTURE. Only the test suite, ``__graft_entry__.smoke()`` and ``bench.py``'s
CPU-baseline leg may import this package. It never touches the CUDA library.

Each method takes and returns numpy arrays; floating-point inputs are float64 holding values
exactly representable in the cache dtype. The C file's header lists the paper passage each
function follows (Sec. 3.1 Eq. 1-2, Sec. 3.2.1 Eq. 4-5, Sec. 3.2.2 Eq. 6-9).

``Oracle(path)`` wraps one compiled copy of the C file; the module-level functions use the
default copy, ``oracle/libvoxzip_oracle.so``, compiled on first use.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "voxzip_oracle.c")
LIB_PATH = os.path.join(_HERE, "libvoxzip_oracle.so")

OK, EINVAL, ECAPACITY, ENOMEM = 0, 1, 2, 3

_I32P = ctypes.POINTER(ctypes.c_int32)
_F64P = ctypes.POINTER(ctypes.c_double)
_i32 = ctypes.c_int32
_f64 = ctypes.c_double
_f32 = ctypes.c_float


def build(force: bool = False, src: str = SOURCE, out: str = LIB_PATH) -> str:
    """Compile the oracle with gcc (no fast-math, no FMA contraction, so x86 and Arm hosts give
    the same bits). By default builds ``oracle/libvoxzip_oracle.so``."""
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math", "-ffp-contract=off",
             "-o", tmp, src, "-lm"])
        os.replace(tmp, out)
    return out


class OracleError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} returned {code}")
        self.code = code


def _f64a(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _i32a(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def _p(a, t):
    return None if a is None else a.ctypes.data_as(t)


class UnitCache:
    """One unit's cache state in fp64: K, V [capacity][D], score, pos, length n."""

    def __init__(self, capacity: int, D: int):
        self.K = np.zeros((capacity, D))
        self.V = np.zeros((capacity, D))
        self.score = np.zeros(capacity)
        self.pos = np.full(capacity, -1, np.int32)
        self.n = 0
        self.capacity = capacity
        self.D = D

    @classmethod
    def from_rows(cls, capacity, K, V, pos, score=None):
        c = cls(capacity, np.asarray(K).shape[1])
        n = np.asarray(K).shape[0]
        c.K[:n] = K
        c.V[:n] = V
        c.pos[:n] = pos
        if score is not None:
            c.score[:n] = score
        c.n = n
        return c


class Oracle:
    """One loaded copy of the compiled oracle."""

    def __init__(self, path: str):
        lib = ctypes.CDLL(path)
        lib.vzo_stage1.argtypes = [_i32, _i32, _i32, _i32, _I32P, _I32P, _I32P, _i32, _F64P, _F64P,
                                   _i32, _i32, _F64P, _F64P, _I32P, _I32P, _I32P]
        lib.vzo_stage1_ex.argtypes = [_i32, _i32, _i32, _i32, _I32P, _I32P, _I32P, _i32, _F64P, _F64P,
                                      _i32, _i32, _i32, _F64P, _F64P, _I32P, _I32P, _I32P]
        lib.vzo_segments_to_spans.argtypes = [_i32, _F64P, _F64P, _F64P, _I32P, _f64, _i32, _i32, _f64,
                                              _I32P, _I32P, _I32P, _I32P, _I32P]
        lib.vzo_decode_step.argtypes = [_i32, _i32, _i32, _I32P, _F64P, _F64P, _F64P, _I32P, _F64P,
                                        _F64P, _F64P, _i32, _f64, _f64, _F64P]
        lib.vzo_evict.argtypes = [_i32, _I32P, _i32, _i32, _f32, _F64P, _F64P, _F64P, _I32P,
                                  _F64P, _I32P]
        lib.vzo_evict_ex.argtypes = [_i32, _I32P, _i32, _i32, _f32, _i32, _i32, _F64P, _F64P, _F64P,
                                     _I32P, _F64P, _I32P]
        lib.vzo_run_unit.argtypes = [_i32, _i32, _i32, _i32, _I32P, _I32P, _I32P, _i32, _F64P,
                                     _F64P, _F64P, _F64P, _i32, _i32, _i32, _i32, _F64P, _F64P,
                                     _F64P, _I32P, _f64, _f64, _i32, _i32, _i32, _f32, _F64P,
                                     _F64P, _I32P, _I32P, _F64P, _F64P, _F64P, _F64P, _I32P,
                                     _I32P, _I32P, _I32P]
        lib.vzo_run_unit_ex.argtypes = [_i32, _i32, _i32, _i32, _I32P, _I32P, _I32P, _i32, _F64P,
                                     _F64P, _F64P, _F64P, _i32, _i32, _i32, _i32, _F64P, _F64P,
                                     _F64P, _I32P, _f64, _f64, _i32, _i32, _i32, _f32, _i32, _i32, _F64P,
                                     _F64P, _I32P, _I32P, _I32P, _F64P, _F64P, _F64P, _F64P, _I32P,
                                     _I32P, _I32P, _I32P]
        for f in (lib.vzo_stage1, lib.vzo_stage1_ex, lib.vzo_segments_to_spans, lib.vzo_decode_step,
                  lib.vzo_evict, lib.vzo_evict_ex, lib.vzo_run_unit, lib.vzo_run_unit_ex):
            f.restype = ctypes.c_int
        self.lib = lib
        self.path = path

    def stage1(self, x, in_len, audio_begin, audio_len, span_start, span_end, span_groups, *,
               anchor=None, cache_is_bf16=False, capacity=None, keep_background=True):
        """Stage-1 fusion of one unit's rows (or of one sequence's embeddings). With
        keep_background=False the audio no span covers is dropped (the "Partial" ablation) and
        its tokens map to slot -1. Returns dict(exact, stored, pos, slot_map, n)."""
        x = _f64a(x)
        D = x.shape[1]
        ss, se, sg = _i32a(span_start), _i32a(span_end), _i32a(span_groups)
        cap = int(in_len if capacity is None else capacity)
        exact = np.zeros((max(cap, 1), D))
        stored = np.zeros((max(cap, 1), D))
        pos = np.full(max(cap, 1), -1, np.int32)
        slot_map = np.full(max(int(in_len), 1), -1, np.int32)
        n = np.zeros(1, np.int32)
        anc = None if anchor is None else _f64a(anchor)
        if keep_background:
            rc = self.lib.vzo_stage1(int(in_len), int(audio_begin), int(audio_len), len(ss),
                                     _p(ss, _I32P), _p(se, _I32P), _p(sg, _I32P), D, _p(x, _F64P),
                                     _p(anc, _F64P), int(bool(cache_is_bf16)), cap, _p(exact, _F64P),
                                     _p(stored, _F64P), _p(pos, _I32P), _p(slot_map, _I32P),
                                     _p(n, _I32P))
        else:
            rc = self.lib.vzo_stage1_ex(int(in_len), int(audio_begin), int(audio_len), len(ss),
                                        _p(ss, _I32P), _p(se, _I32P), _p(sg, _I32P), D, _p(x, _F64P),
                                        _p(anc, _F64P), int(bool(cache_is_bf16)), 0, cap,
                                        _p(exact, _F64P), _p(stored, _F64P), _p(pos, _I32P),
                                        _p(slot_map, _I32P), _p(n, _I32P))
        if rc != OK:
            raise OracleError("vzo_stage1", rc)
        k = int(n[0])
        return dict(exact=exact[:k], stored=stored[:k], pos=pos[:k],
                    slot_map=slot_map[:int(in_len)], n=k)

    def segments_to_spans(self, t_start, t_end, confidence, text_len, tau_total: float, audio_len: int,
                          audio_begin: int = 0, threshold: float = 0.3):
        """ASR segments -> token-index spans (confidence filter, Eq. 3). Returns
        dict(start, end, groups, seg_index) as int32 arrays, one entry per kept segment."""
        ts, te, cf = _f64a(t_start), _f64a(t_end), _f64a(confidence)
        tl = _i32a(text_len)
        n = len(ts)
        assert len(te) == n and len(cf) == n and len(tl) == n
        out = [np.zeros(max(n, 1), np.int32) for _ in range(4)]
        k = np.zeros(1, np.int32)
        rc = self.lib.vzo_segments_to_spans(n, _p(ts, _F64P), _p(te, _F64P), _p(cf, _F64P), _p(tl, _I32P),
                                            float(tau_total), int(audio_len), int(audio_begin), float(threshold),
                                            *[_p(a, _I32P) for a in out], _p(k, _I32P))
        if rc != OK:
            raise OracleError("vzo_segments_to_spans", rc)
        m = int(k[0])
        return dict(start=out[0][:m], end=out[1][:m], groups=out[2][:m], seg_index=out[3][:m])

    def decode_step(self, cache: UnitCache, q, k_new, v_new, new_pos: int, gamma: float,
                    scale: float):
        """Eq. 1, Eq. 2 and Eq. 6 for one unit, in place on ``cache``. Returns out [G][D]."""
        q = _f64a(q)
        G, D = q.shape
        k_new, v_new = _f64a(k_new), _f64a(v_new)
        out = np.zeros((G, D))
        n = np.array([cache.n], np.int32)
        rc = self.lib.vzo_decode_step(D, G, cache.capacity, _p(n, _I32P), _p(cache.K, _F64P),
                                      _p(cache.V, _F64P), _p(cache.score, _F64P),
                                      _p(cache.pos, _I32P), _p(q, _F64P), _p(k_new, _F64P),
                                      _p(v_new, _F64P), int(new_pos), float(gamma), float(scale),
                                      _p(out, _F64P))
        if rc != OK:
            raise OracleError("vzo_decode_step", rc)
        cache.n = int(n[0])
        return out

    def evict(self, cache: UnitCache, budget: int, sink: int = 4, recent_frac: float = 0.2, *,
              history: bool = True, fill: bool = False):
        """Eq. 7-9 for one unit, in place. history=False keeps sinks and a recent window only
        (StreamingLLM); fill=True selects sinks / recents by position and fills the evicted slots
        with the kept rows beyond the budget. Returns (margin, kept flags of the pre-eviction slots)."""
        n = np.array([cache.n], np.int32)
        margin = np.zeros(1)
        kept = np.zeros(max(cache.n, 1), np.int32)
        rc = self.lib.vzo_evict_ex(cache.D, _p(n, _I32P), int(budget), int(sink), float(recent_frac),
                                   int(bool(history)), int(bool(fill)), _p(cache.K, _F64P), _p(cache.V, _F64P),
                                   _p(cache.score, _F64P), _p(cache.pos, _I32P), _p(margin, _F64P),
                                   _p(kept, _I32P))
        if rc != OK:
            raise OracleError("vzo_evict", rc)
        pre_n = cache.n
        cache.n = int(n[0])
        return float(margin[0]), kept[:pre_n].astype(bool)

    def run_unit(self, xk, xv, in_len, audio_begin, audio_len, span_start, span_end, span_groups,
                 *, q, k_new, v_new, new_pos, gamma, scale, interval, budget, sink=4,
                 recent_frac=0.2, capacity, anchor_k=None, anchor_v=None, cache_is_bf16=False,
                 history=True, fill=False):
        """Stage 1, then len(q) decode steps with an eviction every ``interval`` steps.

        q [steps][G][D]; k_new, v_new [steps][D]; new_pos [steps]. Returns a dict with ``out``,
        the per-eviction records (score_before, len_before, kept_pos, margin), the final cache
        (K, V, score, pos, n) and the stage-1 slot map and length.
        """
        xk, xv = _f64a(xk), _f64a(xv)
        q, k_new, v_new = _f64a(q), _f64a(k_new), _f64a(v_new)
        new_pos = _i32a(new_pos)
        steps, G, D = q.shape
        ss, se, sg = _i32a(span_start), _i32a(span_end), _i32a(span_groups)
        n_ev = steps // interval
        out = np.zeros((max(steps, 1), G, D))
        score_before = np.zeros((max(n_ev, 1), capacity))
        pos_before = np.full((max(n_ev, 1), capacity), -1, np.int32)
        len_before = np.zeros(max(n_ev, 1), np.int32)
        kept_pos = np.full((max(n_ev, 1), max(budget, 1)), -1, np.int32)
        margin = np.zeros(max(n_ev, 1))
        K = np.zeros((capacity, D))
        V = np.zeros((capacity, D))
        score = np.zeros(capacity)
        pos = np.full(capacity, -1, np.int32)
        n_final = np.zeros(1, np.int32)
        slot_map = np.full(max(int(in_len), 1), -1, np.int32)
        stage1_len = np.zeros(1, np.int32)
        ak = None if anchor_k is None else _f64a(anchor_k)
        av = None if anchor_v is None else _f64a(anchor_v)
        rc = self.lib.vzo_run_unit_ex(
            int(in_len), int(audio_begin), int(audio_len), len(ss), _p(ss, _I32P), _p(se, _I32P),
            _p(sg, _I32P), D, _p(xk, _F64P), _p(xv, _F64P), _p(ak, _F64P), _p(av, _F64P),
            int(bool(cache_is_bf16)), G, int(capacity), steps, _p(q, _F64P), _p(k_new, _F64P),
            _p(v_new, _F64P), _p(new_pos, _I32P), float(gamma), float(scale), int(interval),
            int(budget), int(sink), float(recent_frac), int(bool(history)), int(bool(fill)),
            _p(out, _F64P), _p(score_before, _F64P), _p(pos_before, _I32P),
            _p(len_before, _I32P), _p(kept_pos, _I32P), _p(margin, _F64P), _p(K, _F64P),
            _p(V, _F64P), _p(score, _F64P), _p(pos, _I32P), _p(n_final, _I32P),
            _p(slot_map, _I32P), _p(stage1_len, _I32P))
        if rc != OK:
            raise OracleError("vzo_run_unit", rc)
        nf = int(n_final[0])
        return dict(out=out[:steps], score_before=score_before[:n_ev], pos_before=pos_before[:n_ev],
                    len_before=len_before[:n_ev], kept_pos=kept_pos[:n_ev], margin=margin[:n_ev],
                    K=K[:nf], V=V[:nf], score=score[:nf], pos=pos[:nf], n=nf,
                    slot_map=slot_map[:int(in_len)], stage1_len=int(stage1_len[0]))


_lock = threading.Lock()
_default: Oracle | None = None


def default() -> Oracle:
    """The oracle compiled from ``voxzip_oracle.c`` (built on first use)."""
    global _default
    with _lock:
        if _default is None:
            _default = Oracle(build())
    return _default


def stage1(*a, **k):
    return default().stage1(*a, **k)


def segments_to_spans(*a, **k):
    return default().segments_to_spans(*a, **k)


def decode_step(*a, **k):
    return default().decode_step(*a, **k)


def evict(*a, **k):
    return default().evict(*a, **k)


def run_unit(*a, **k):
    return default().run_unit(*a, **k)
