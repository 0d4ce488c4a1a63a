"""Planted mistakes: each mutation below is a plausible error in the oracle (a dropped term, a
wrong sign or index, a transposed operand, another rounding). It is applied to a temporary copy
of ``oracle/voxzip_oracle.c``, compiled, and the pins must reject that copy. CPU only; the
committed oracle is never modified."""
import os

import pytest

import oracle
import oracle_pins

MUTATIONS = [
    ("decay dropped", "score[j] *= gamma;", "score[j] *= 1.0;"),
    ("decay applied twice", "score[j] *= gamma;", "score[j] *= gamma * gamma;"),
    ("logit scale squared", "logit[j] = dot * scale;", "logit[j] = dot * scale * scale;"),
    ("softmax denominator off", "const double p = exp(logit[j] - m) / z;",
     "const double p = exp(logit[j] - m) / (z + 1.0);"),
    ("new token score not zero-padded", "score[n] = 0.0;", "score[n] = 1.0;"),
    ("append position off by one", "pos[n] = new_pos;", "pos[n] = new_pos + 1;"),
    ("PV reads K instead of V", "oh[d] += p * V[(int64_t)j * D + d];",
     "oh[d] += p * K[(int64_t)j * D + d];"),
    ("query reversed against key", "dot += qh[d] * K[(int64_t)j * D + d];",
     "dot += qh[D - 1 - d] * K[(int64_t)j * D + d];"),
    ("ceil group boundaries (short groups last)",
     "const int64_t lo = s + (j * l) / g;\n                const int64_t hi = s + ((j + 1) * l) / g;",
     "const int64_t lo = s + (j * l + g - 1) / g;\n                const int64_t hi = s + ((j + 1) * l + g - 1) / g;"),
    ("group count not clamped to span length", "span_groups[i] < l ? span_groups[i] : l",
     "span_groups[i]"),
    ("anchor row ignores the group index", "anchor[(anchor_row + j) * D + d]",
     "anchor[(anchor_row) * D + d]"),
    ("empty spans' anchor rows not counted",
     "while (i < n_spans && span_start[i] == span_end[i]) {\n            anchor_row += span_groups[i];",
     "while (i < n_spans && span_start[i] == span_end[i]) {"),
    ("group mean divides by |G|+1", "double exact = sum / (double)(hi - lo);",
     "double exact = sum / (double)(hi - lo + 1);"),
    ("stored mean divides by |G|+1", "float stored = acc / (float)(hi - lo);",
     "float stored = acc / (float)(hi - lo + 1);"),
    ("bf16 rounds half up", "u += 0x7fffu + lsb;", "u += 0x8000u;"),
    ("bf16 truncates", "u += 0x7fffu + lsb;", "u += 0u;"),
    ("background position off by one", "pos[slot] = t;\n            slot_map[t] = slot;",
     "pos[slot] = t + 1;\n            slot_map[t] = slot;"),
    ("group position is its last token", "pos[slot] = (int32_t)lo;", "pos[slot] = (int32_t)(hi - 1);"),
    ("ties go to the higher position", "return (x->pos > y->pos) - (x->pos < y->pos);",
     "return (x->pos < y->pos) - (x->pos > y->pos);"),
    ("lowest scores kept", "if (x->score > y->score)\n        return -1;\n    if (x->score < y->score)\n        return 1;",
     "if (x->score > y->score)\n        return 1;\n    if (x->score < y->score)\n        return -1;"),
    ("recent window rounded up", "floor((double)recent_frac * (double)budget)",
     "ceil((double)recent_frac * (double)budget)"),
    ("recent window one short", "for (int32_t r = n - M; r < n; ++r)\n        keep[all[r].slot] = 1;",
     "for (int32_t r = n - M + 1; r < n; ++r)\n        keep[all[r].slot] = 1;"),
    ("sinks one short", "for (int32_t r = 0; r < T; ++r)\n        keep[all[r].slot] = 1;",
     "for (int32_t r = 0; r < T - 1; ++r)\n        keep[all[r].slot] = 1;"),
    ("score not moved with its row", "score[w] = score[j];", "(void)0;"),
    ("position not moved with its row", "pos[w] = pos[j];", "(void)0;"),
    ("confidence filter keeps the threshold itself", "if (!(confidence[i] > threshold))",
     "if (!(confidence[i] >= threshold))"),
    ("Eq. 3 rounds instead of flooring", "double fs = floor((double)La * (t_start[i] / tau_total));",
     "double fs = round((double)La * (t_start[i] / tau_total));"),
    ("Eq. 3 end index rounded up", "double fe = floor((double)La * (t_end[i] / tau_total));",
     "double fe = ceil((double)La * (t_end[i] / tau_total));"),
    ("overlapping segments not clipped", "        if (s < prev_end)\n            s = prev_end;\n", ""),
    ("segment text length not carried", "span_groups[kept] = text_len[i];", "span_groups[kept] = 1;"),
    ("Partial keeps the background", "} else if (!keep_background && t >= audio_begin && t < audio_begin + audio_len) {",
     "} else if (0) {"),
    ("Partial drops the text too", "} else if (!keep_background && t >= audio_begin && t < audio_begin + audio_len) {",
     "} else if (!keep_background) {"),
    ("hole filling picks sinks and recents by slot", "    if (fill)\n        qsort(all, (size_t)n, sizeof(vzo_candidate), position_order);\n", ""),
    ("hole filling writes over kept rows", "while (h < budget && keep[h])", "while (h < budget && !keep[h])"),
    ("hole filling leaves the score behind", "            score[h] = score[j];\n            pos[h] = pos[j];",
     "            pos[h] = pos[j];"),
    ("hole filling leaves the position behind", "            score[h] = score[j];\n            pos[h] = pos[j];",
     "            score[h] = score[j];"),
    ("StreamingLLM window one short", ": budget - T;", ": budget - T - 1;"),
    ("history switch ignored", "history ? (int32_t)floor((double)recent_frac * (double)budget) : budget - T",
     "(int32_t)floor((double)recent_frac * (double)budget)"),
    ("margin against the wrong runner-up", "*margin = c[N - 1].score - c[N].score;",
     "*margin = c[N - 1].score - c[N + 1 < nc ? N + 1 : N].score;"),
    ("ordered compaction leaves K behind",
     "                memmove(K + (int64_t)w * D, K + (int64_t)j * D, sizeof(double) * (size_t)D);\n", ""),
    ("ordered compaction leaves V behind",
     "                memmove(V + (int64_t)w * D, V + (int64_t)j * D, sizeof(double) * (size_t)D);\n", ""),
    ("hole filling leaves V behind",
     "            memcpy(V + (int64_t)h * D, V + (int64_t)j * D, sizeof(double) * (size_t)D);\n", ""),
    ("V fused with the K anchors",
     "span_groups, D, xv, anchor_v, cache_is_bf16,", "span_groups, D, xv, anchor_k, cache_is_bf16,"),
    ("score sums one head of the group", "            score[j] += p;", "            score[j] += h == 0 ? p : 0.0;"),
    ("append writes k_new into V", "        V[(int64_t)n * D + d] = v_new[d];", "        V[(int64_t)n * D + d] = k_new[d];"),
    ("history candidates overlap the recent window", "    const int32_t nc = n - M - T;",
     "    const int32_t nc = n - T;"),
    ("ties broken by slot instead of position",
     "        return 1;\n    return (x->pos > y->pos) - (x->pos < y->pos);\n}\n\nstatic int position_order",
     "        return 1;\n    return (x->slot > y->slot) - (x->slot < y->slot);\n}\n\nstatic int position_order"),
    ("Eq. 3 multiplies before dividing", "double fs = floor((double)La * (t_start[i] / tau_total));",
     "double fs = floor((double)La * t_start[i] / tau_total);"),
    ("eviction one step late", "        if (t % interval == 0) {", "        if (t > 1 && (t - 1) % interval == 0) {"),
    ("segments emptied by clipping are dropped", "        span_start[kept] = (int32_t)(audio_begin + s);",
     "        if (e == s)\n            continue;\n        span_start[kept] = (int32_t)(audio_begin + s);"),
    ("clipped end not raised to the start", "        if (e < s)\n            e = s;\n", ""),
    ("clamp at L_a - 1", "int64_t e = fe < 0.0 ? 0 : (fe > (double)La ? La : (int64_t)fe);",
     "int64_t e = fe < 0.0 ? 0 : (fe > (double)La - 1 ? La - 1 : (int64_t)fe);"),
    ("no eviction one row over the budget", "    if (n <= budget)\n        return VZO_OK;",
     "    if (n <= budget + 1)\n        return VZO_OK;"),
    ("stage-1 scores not reset", "    for (int32_t j = 0; j < n; ++j)\n        score[j] = 0.0;\n\n    int32_t ev = 0;",
     "    for (int32_t j = 0; j < n; ++j)\n        score[j] = 1.0;\n\n    int32_t ev = 0;"),
    ("stored mean taken from the fp64 sum", "float stored = acc / (float)(hi - lo);",
     "float stored = (float)(sum / (double)(hi - lo));"),
    ("anchor added after the cache rounding",
     "out_stored[(int64_t)slot * D + d] = cache_is_bf16 ? bf16_round(stored) : (double)stored;",
     "out_stored[(int64_t)slot * D + d] = cache_is_bf16 ? bf16_round(acc / (float)(hi - lo)) + (anchor ? (float)anchor[(anchor_row + j) * D + d] : 0.0f) : (double)stored;"),
    ("custom softmax scale ignored", "logit[j] = dot * scale;", "logit[j] = dot / sqrt((double)D);"),
    ("top-N candidates include the sinks", "    const int32_t nc = n - M - T;\n    vzo_candidate *c = all + T;",
     "    const int32_t nc = n - M;\n    vzo_candidate *c = all;"),
    ("append overwrites the last row", "        K[(int64_t)n * D + d] = k_new[d];\n        V[(int64_t)n * D + d] = v_new[d];",
     "        K[(int64_t)(n > 0 ? n - 1 : 0) * D + d] = k_new[d];\n        V[(int64_t)(n > 0 ? n - 1 : 0) * D + d] = v_new[d];"),
    ("kept flags all set", "            kept[j] = keep[j];", "            kept[j] = 1;"),
    ("no-op eviction reports a zero margin", "    *margin = INFINITY;", "    *margin = 0.0;"),
    ("length before eviction recorded after it", "            len_before[ev] = n;\n            rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, fill, K, V, score, pos,\n                              &margin[ev], NULL);",
     "            rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, fill, K, V, score, pos,\n                              &margin[ev], NULL);\n            len_before[ev] = n;"),
    ("a whole run ignores the fill policy", "rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, fill, K, V, score, pos,",
     "rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, 0, K, V, score, pos,"),
    ("a whole run ignores the no-history policy", "rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, fill, K, V, score, pos,",
     "rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, 1, fill, K, V, score, pos,"),
    ("a whole run ignores the sink count", "rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, fill, K, V, score, pos,",
     "rc = vzo_evict_ex(D, &n, budget, 4, recent_frac, history, fill, K, V, score, pos,"),
    ("a whole run ignores the recent fraction", "rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, fill, K, V, score, pos,",
     "rc = vzo_evict_ex(D, &n, budget, sink, 0.2f, history, fill, K, V, score, pos,"),
    ("a whole run ignores the cache dtype", "D, xk, anchor_k, cache_is_bf16, capacity, scratch, K, pos, slot_map, &n);",
     "D, xk, anchor_k, 0, capacity, scratch, K, pos, slot_map, &n);"),
    ("a whole run decays with a fixed gamma", "v_new + (int64_t)(t - 1) * D, new_pos[t - 1], gamma, scale,",
     "v_new + (int64_t)(t - 1) * D, new_pos[t - 1], 0.9, scale,"),
    ("a whole run scales with a fixed factor", "v_new + (int64_t)(t - 1) * D, new_pos[t - 1], gamma, scale,",
     "v_new + (int64_t)(t - 1) * D, new_pos[t - 1], gamma, 0.3,"),
    ("hole filling orders by slot on a scrambled cache", "position_order);\n    for (int32_t r = 0; r < T; ++r)",
     "candidate_order);\n    for (int32_t r = 0; r < T; ++r)"),
]


def _caught(orc):
    for pin in oracle_pins.ALL_PINS:
        try:
            pin(orc)
        except (AssertionError, oracle.OracleError, ValueError, FloatingPointError):
            return pin.__name__
    return None


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(tmp_path, name, old, new):
    with open(oracle.SOURCE) as f:
        src = f.read()
    assert old in src, f"mutation anchor for '{name}' not found in the oracle source"
    mutated = tmp_path / "mutant.c"
    mutated.write_text(src.replace(old, new))
    lib = oracle.build(force=True, src=str(mutated), out=str(tmp_path / "libmutant.so"))
    by = _caught(oracle.Oracle(lib))
    assert by is not None, f"no pin catches the planted mistake: {name}"
    print(f"{name}: caught by {by}")
