"""Isolated launches of each kernel of the path, for a profiler (ncu) to capture one of them.

    python -m paper_2608_08569_gb300.profile_cases decode [reps]   # decode step, 60-min 20x steady state
    python -m paper_2608_08569_gb300.profile_cases evict [reps]    # one eviction of that state
    python -m paper_2608_08569_gb300.profile_cases evict_small [reps]  # eviction, 10-min 4x steady state
    python -m paper_2608_08569_gb300.profile_cases evict_fill [reps]   # hole-filling eviction, 60-min 20x
    python -m paper_2608_08569_gb300.profile_cases fuse [reps]     # stage 1 of the 60-min request, 4 layers

Each case holds at most a few GB on the device (decode / evict: 0.94 GB of K/V, 4 sequences x 48
layers x 4 kv-heads at about 2 330 tokens; evict_small: 0.2 GB, one sequence at 2 035), restores the same seeded state before every launch and
synchronises after it, so `-s <reps-1> -c 1` captures one steady launch. Inputs are seeded synthetic
tensors; nothing here checks results (the tests do).
"""
import sys

import numpy as np
import torch

from . import (CacheDesc, allocate_cache, voxzip_anchor_fuse, voxzip_decode_step, voxzip_evict,
               voxzip_evict_ex, voxzip_get_status)
from . import workloads as W


def run(mode: str, reps: int = 6) -> None:
    g = torch.Generator(device="cuda")
    g.manual_seed(1)
    if mode in ("decode", "evict", "evict_small", "evict_fill"):
        B, L, Hq, H, D = (1 if mode == "evict_small" else 4), 48, 32, 4, 128
        # 60-min 20x: budget 2 301, up to 32 steps past it; 10-min 4x: budget 2 003
        budget = 2003 if mode == "evict_small" else 2301
        n = budget + 32 if mode != "decode" else 2330
        cap = n + 64
        desc = CacheDesc(B, L, Hq, H, D, cap, torch.bfloat16)
        c = allocate_cache(desc)
        for b in range(B):
            c["k"][b].normal_(generator=g)
            c["v"][b].normal_(generator=g)
        c["score"].uniform_(generator=g)
        c["pos"].copy_(torch.arange(cap, dtype=torch.int32, device="cuda").expand_as(c["pos"]))
        ref = {k: v.clone() for k, v in c.items()}
        q = torch.randn(L, B, Hq, D, device="cuda", generator=g).to(torch.bfloat16)
        kn = torch.randn(L, B, H, D, device="cuda", generator=g).to(torch.bfloat16)
        vn = torch.randn(L, B, H, D, device="cuda", generator=g).to(torch.bfloat16)
        out = torch.empty_like(q)
        npos = torch.full((B,), 99999, dtype=torch.int32, device="cuda")
        bud = torch.full((B,), budget, dtype=torch.int32, device="cuda")
        for _ in range(reps):
            for k in c:
                c[k].copy_(ref[k])
            c["len"].fill_(n)
            torch.cuda.synchronize()
            if mode == "decode":
                voxzip_decode_step(desc, 0, L, q, kn, vn, npos, c["k"], c["v"], c["score"], c["pos"], c["len"], 0.995,
                                   out, max_len=n + 1)
            elif mode == "evict_fill":
                voxzip_evict_ex(desc, 0, L, c["k"], c["v"], c["score"], c["pos"], c["len"], bud, compaction="fill")
            else:
                voxzip_evict(desc, 0, L, c["k"], c["v"], c["score"], c["pos"], c["len"], bud)
            torch.cuda.synchronize()
        # Algorithmic bytes of one launch, for the summary's traffic ratio. Decode: every K and V row
        # once, the score read and written, q and out, k_new and v_new and their append, the position.
        # Eviction: 8 B per slot for the selection, and K, V, score and position read and written for
        # every kept row that changed slot (counted from the positions before and after).
        e = 2
        if mode == "decode":
            alg = L * B * H * ((n + 1) * (2 * D * e + 8) + (2 * (Hq // H) * D + 4 * D) * e + 4)
        else:
            na = c["len"].reshape(-1).long()
            idx = torch.arange(cap, device="cuda")
            moved = ((ref["pos"].reshape(-1, cap) != c["pos"].reshape(-1, cap)) & (idx[None] < na[:, None])).sum()
            alg = 8 * n * L * B * H + 2 * (2 * D * e + 8) * int(moved)
        print("algorithmic_bytes_per_launch", int(alg))
    elif mode == "fuse":
        w = W.scaled(W.CONFIGS["stress"], layers=4, name="stress_l4")
        sp = W.make_spans(w)
        k, v = W.make_prefill(w, "cuda")

        def i32(a):
            return torch.as_tensor(np.asarray(a), dtype=torch.int32, device="cuda")

        desc = CacheDesc(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, w.capacity, w.dtype)
        c = allocate_cache(desc)
        for _ in range(reps):
            voxzip_anchor_fuse(desc, k, v, i32(w.in_len), i32([w.audio_begin] * w.batch), i32(w.audio_len),
                               i32(sp.off), i32(sp.start), i32(sp.end), i32(sp.groups), c["k"], c["v"], c["score"],
                               c["pos"], c["len"])
            torch.cuda.synchronize()
        # Algorithmic bytes of the fusion kernel: the prefill K and V read once, the stage-1 rows
        # written with their score and position.
        n1 = c["len"][:, 0, 0].long().cpu().tolist()
        e = 2 if w.dtype == torch.bfloat16 else 4
        alg = w.layers * w.kv_heads * sum(2 * il * w.head_dim * e + nn * (2 * w.head_dim * e + 8)
                                          for il, nn in zip(w.in_len, n1))
        print("algorithmic_bytes_per_launch", int(alg))
    else:
        raise SystemExit(f"unknown case {mode!r}: decode, evict, evict_small, evict_fill or fuse")
    if voxzip_get_status() != 0:
        raise SystemExit("device status word set")
    print("ok", mode)


if __name__ == "__main__":
    run(sys.argv[1], int(sys.argv[2]) if len(sys.argv) > 2 else 6)
