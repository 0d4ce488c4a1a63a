/*
 * voxzip_oracle.c -- plain, slow fp64 CPU oracle for the VoxZip KV-cache compression path
 * (arxiv 2608.08569, "VoxZip: Semantic-Anchored Temporal KV Cache Compression for
 * Long-Context Audio Inference").
 *
 * TEST INFRASTRUCTURE. Only the test suite, the smoke check and the benchmark's CPU-baseline
 * leg may load this library. It shares no code, header, table or helper with the CUDA
 * library; neither includes the other. It processes one (sequence, layer, kv-head) unit at
 * a time, in the order the paper states its steps, with no blocking or fusion.
 *
 * Functions and the passages they follow:
 *   vzo_segments_to_spans  Sec. 3.2.1: the confidence filter on ASR segments (keep those above
 *                    the threshold, 0.3 in the paper) and the time-to-token-index map of Eq. 3.
 *   vzo_stage1       Sec. 3.2.1: semantic intervals given as token-index spans (Eq. 3 already
 *                    applied), uniform grouping + average pooling (Eq. 4), anchor addition,
 *                    background preservation and chronological concatenation (Eq. 5).
 *   vzo_stage1_ex    the same with the background optional: the "T+A (Partial)" configuration
 *                    of the stage-1 ablation (Sec. 4, Table of fusion strategies) drops the
 *                    audio no semantic interval covers.
 *   vzo_decode_step  Sec. 3.1: cache append (Eq. 1) and scaled dot-product attention (Eq. 2);
 *                    Sec. 3.2.2: temporally decayed accumulated score (Eq. 6).
 *   vzo_evict        Sec. 3.2.2: T attention sinks, a recent window of 20 % of the budget,
 *                    top-N history by decayed score, concatenation (Eq. 7-9).
 *   vzo_evict_ex     the same selection as a policy: without history (the StreamingLLM baseline
 *                    of Sec. 4), and with sinks / recents chosen by position and the kept rows
 *                    beyond the budget filling the evicted slots (a compaction that moves at most
 *                    n - budget rows; the kept set is the same as the ordered one on a cache in
 *                    time order).
 *   vzo_run_unit     the three above in the paper's order for one unit: stage 1 at prefill,
 *                    then decode steps with an eviction every `interval` steps.
 * Every function is pinned by the CPU tests (closed forms, invariants, brute force and
 * hand-worked fixtures); none is "parity unpinned".
 *
 * Readings where the paper is silent (each is listed in the design notes):
 *   - "a confidence score above a threshold" is strict (confidence > threshold);
 *   - Eq. 3 is evaluated as floor(L_a * (tau / tau_total)) in double, in that order; indices
 *     are clamped to [0, L_a]; a segment that would start before the previous kept one ends
 *     starts where that one ends (an empty interval if nothing is left); segments must come
 *     sorted by start time;
 *   - stage 1 acts on each layer's prefilled K and V rows (or on embeddings, the paper's own
 *     setting); the anchor term is an optional caller-supplied row per (span, group), zero
 *     when absent;
 *   - group j of a span of length l with g = min(n_groups, l) groups covers
 *     [s + floor(j*l/g), s + floor((j+1)*l/g)); empty spans yield nothing;
 *   - the slot of a fused group records the index of the group's first token as its position;
 *   - the decayed score of a (layer, kv-head) unit sums the softmax mass over the query heads
 *     of its GQA group; scores start at zero after stage 1;
 *   - M = floor(budget * recent_frac) evaluated in double, N = budget - T - M; ties in the
 *     top-N are broken by the lower position; kept rows stay in ascending slot order.
 *
 * Precision: fp64 throughout, except one quantisation the cache format forces: a fused
 * stage-1 row is stored in the cache dtype. That rounding decision is taken in the
 * kernel's precision (fp32 sum over the group in token order, IEEE division by the group
 * size, fp32 anchor add, then round-to-nearest-even to bf16 when the cache is bf16), so that
 * both sides store the same bits. The exact fp64 value is returned beside it.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define VZO_OK 0
#define VZO_EINVAL 1
#define VZO_ECAPACITY 2
#define VZO_ENOMEM 3

/* Round an fp32 value to the nearest bf16 (ties to even) and widen it back exactly. */
static double bf16_round(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu) != 0u) {
        u |= 0x00400000u; /* quiet NaN */
        u &= 0xffff0000u;
    } else {
        uint32_t lsb = (u >> 16) & 1u;
        u += 0x7fffu + lsb;
        u &= 0xffff0000u;
    }
    float r;
    memcpy(&r, &u, sizeof r);
    return (double)r;
}

/*
 * Stage 1 for one unit's rows (one of K or V of one layer and kv-head of one sequence).
 *
 *   x          [in_len][D]   prefill rows, already in the storage dtype, widened to double
 *   spans      token-index spans [span_start[i], span_end[i]) inside the audio region
 *              [audio_begin, audio_begin + audio_len), sorted, non-overlapping
 *   span_groups n_groups of each span (the text length L_t of the transcription)
 *   anchor     [sum(span_groups)][D] anchor rows, row (prefix of span_groups before i) + j is
 *              added to group j of span i; NULL means the anchor term is zero
 *   out_exact  [capacity][D] exact fp64 fused rows (Eq. 4 mean + anchor, or the copied row)
 *   out_stored [capacity][D] the same rows as the cache stores them (see the header)
 *   pos        [capacity]    original index of the first token of each output slot
 *   slot_map   [in_len]      output slot of every input token
 * Returns VZO_OK, VZO_EINVAL for malformed spans, VZO_ECAPACITY if the output exceeds capacity.
 */
int vzo_stage1_ex(int32_t in_len, int32_t audio_begin, int32_t audio_len, int32_t n_spans,
                  const int32_t *span_start, const int32_t *span_end, const int32_t *span_groups,
                  int32_t D, const double *x, const double *anchor, int32_t cache_is_bf16,
                  int32_t keep_background, int32_t capacity, double *out_exact,
                  double *out_stored, int32_t *pos, int32_t *slot_map, int32_t *out_len)
{
    if (in_len < 0 || audio_begin < 0 || audio_len < 0 || D <= 0 || capacity < 0 ||
        (int64_t)audio_begin + audio_len > in_len || n_spans < 0)
        return VZO_EINVAL;
    /* The semantic set: sorted, non-overlapping intervals inside the audio region. */
    int32_t prev_end = audio_begin;
    for (int32_t i = 0; i < n_spans; ++i) {
        if (span_start[i] < prev_end || span_end[i] < span_start[i] ||
            span_end[i] > audio_begin + audio_len || span_groups[i] < 1)
            return VZO_EINVAL;
        prev_end = span_end[i];
    }

    int32_t slot = 0;
    int32_t t = 0;
    int32_t i = 0;
    int64_t anchor_row = 0; /* first anchor row of span i */
    while (t < in_len) {
        /* Empty spans cover no token: skip them, keeping their anchor rows counted. */
        while (i < n_spans && span_start[i] == span_end[i]) {
            anchor_row += span_groups[i];
            ++i;
        }
        if (i < n_spans && t == span_start[i]) {
            /* A semantic interval: L_a = l tokens pooled into g consecutive groups (Eq. 4). */
            const int64_t s = span_start[i];
            const int64_t l = (int64_t)span_end[i] - span_start[i];
            const int64_t g = span_groups[i] < l ? span_groups[i] : l;
            for (int64_t j = 0; j < g; ++j) {
                const int64_t lo = s + (j * l) / g;
                const int64_t hi = s + ((j + 1) * l) / g;
                if (slot >= capacity)
                    return VZO_ECAPACITY;
                for (int32_t d = 0; d < D; ++d) {
                    double sum = 0.0;
                    float acc = 0.0f;
                    for (int64_t k = lo; k < hi; ++k) {
                        sum += x[k * D + d];
                        acc += (float)x[k * D + d];
                    }
                    double exact = sum / (double)(hi - lo);
                    float stored = acc / (float)(hi - lo);
                    if (anchor) {
                        /* Semantic anchor: element-wise addition of the aligned text row. */
                        exact += anchor[(anchor_row + j) * D + d];
                        stored = stored + (float)anchor[(anchor_row + j) * D + d];
                    }
                    out_exact[(int64_t)slot * D + d] = exact;
                    out_stored[(int64_t)slot * D + d] = cache_is_bf16 ? bf16_round(stored) : (double)stored;
                }
                pos[slot] = (int32_t)lo;
                for (int64_t k = lo; k < hi; ++k)
                    slot_map[k] = slot;
                ++slot;
            }
            t = span_end[i];
            anchor_row += span_groups[i];
            ++i;
        } else if (!keep_background && t >= audio_begin && t < audio_begin + audio_len) {
            /* "Partial": a background acoustic token is discarded; it maps to no slot. */
            slot_map[t] = -1;
            ++t;
        } else {
            /* Background audio or text token: preserved unchanged, in chronological order (Eq. 5). */
            if (slot >= capacity)
                return VZO_ECAPACITY;
            for (int32_t d = 0; d < D; ++d) {
                out_exact[(int64_t)slot * D + d] = x[(int64_t)t * D + d];
                out_stored[(int64_t)slot * D + d] = x[(int64_t)t * D + d];
            }
            pos[slot] = t;
            slot_map[t] = slot;
            ++slot;
            ++t;
        }
    }
    *out_len = slot;
    return VZO_OK;
}

/* Stage 1 as the paper's main method runs it: background acoustic intervals preserved. */
int vzo_stage1(int32_t in_len, int32_t audio_begin, int32_t audio_len, int32_t n_spans,
               const int32_t *span_start, const int32_t *span_end, const int32_t *span_groups,
               int32_t D, const double *x, const double *anchor, int32_t cache_is_bf16,
               int32_t capacity, double *out_exact, double *out_stored, int32_t *pos,
               int32_t *slot_map, int32_t *out_len)
{
    return vzo_stage1_ex(in_len, audio_begin, audio_len, n_spans, span_start, span_end,
                         span_groups, D, x, anchor, cache_is_bf16, 1, capacity, out_exact,
                         out_stored, pos, slot_map, out_len);
}

/*
 * The semantic set of one sequence (Sec. 3.2.1): ASR segments (start time, end time, text of
 * L_t tokens, confidence) become token-index spans of the audio region.
 *
 *   t_start, t_end, confidence, text_len   [n_seg] per segment, sorted by t_start
 *   tau_total   duration of the audio, seconds (> 0)
 *   La          number of audio tokens; audio_begin = index of the first one in the prompt
 *   threshold   a segment is kept when its confidence is above it
 * Outputs, one entry per kept segment, in order:
 *   span_start, span_end   [audio_begin + idx_start, audio_begin + idx_end) (Eq. 3)
 *   span_groups            L_t of the segment
 *   seg_index              which input segment it came from
 *   n_spans                how many were kept
 * Returns VZO_EINVAL for unsorted segments, t_end < t_start, L_t < 1, or a duration that is not
 * finite and positive (Eq. 3 divides by it).
 */
int vzo_segments_to_spans(int32_t n_seg, const double *t_start, const double *t_end,
                          const double *confidence, const int32_t *text_len, double tau_total,
                          int32_t La, int32_t audio_begin, double threshold, int32_t *span_start,
                          int32_t *span_end, int32_t *span_groups, int32_t *seg_index,
                          int32_t *n_spans)
{
    if (n_seg < 0 || !(tau_total > 0.0) || isinf(tau_total) || La < 0 || audio_begin < 0)
        return VZO_EINVAL;
    for (int32_t i = 0; i < n_seg; ++i) {
        if (!(t_end[i] >= t_start[i]) || text_len[i] < 1 || (i > 0 && t_start[i] < t_start[i - 1]))
            return VZO_EINVAL;
    }
    int32_t kept = 0;
    int64_t prev_end = 0;
    for (int32_t i = 0; i < n_seg; ++i) {
        /* Keep only segments whose confidence is above the threshold. */
        if (!(confidence[i] > threshold))
            continue;
        /* Eq. 3: idx = floor(L_a * (tau / tau_total)). */
        double fs = floor((double)La * (t_start[i] / tau_total));
        double fe = floor((double)La * (t_end[i] / tau_total));
        int64_t s = fs < 0.0 ? 0 : (fs > (double)La ? La : (int64_t)fs);
        int64_t e = fe < 0.0 ? 0 : (fe > (double)La ? La : (int64_t)fe);
        if (s < prev_end)
            s = prev_end;
        if (e < s)
            e = s;
        span_start[kept] = (int32_t)(audio_begin + s);
        span_end[kept] = (int32_t)(audio_begin + e);
        span_groups[kept] = text_len[i];
        seg_index[kept] = i;
        prev_end = e;
        ++kept;
    }
    *n_spans = kept;
    return VZO_OK;
}

/*
 * One decode step for one unit: Eq. 1 append, Eq. 2 attention for each of the G query heads of
 * the GQA group, Eq. 6 decayed score update summed over those heads.
 *
 *   n_io      in: cache length before the step; out: after the append
 *   K, V      [capacity][D] cache rows; score [capacity]; pos [capacity]
 *   q         [G][D] queries; k_new, v_new [D]; new_pos = the new token's original index
 *   scale     the logit scale, 1/sqrt(d) with d the head dimension in the paper
 *   out       [G][D] attention outputs
 */
int vzo_decode_step(int32_t D, int32_t G, int32_t capacity, int32_t *n_io, double *K, double *V,
                    double *score, int32_t *pos, const double *q, const double *k_new,
                    const double *v_new, int32_t new_pos, double gamma, double scale, double *out)
{
    int32_t n = *n_io;
    if (D <= 0 || G <= 0 || n < 0)
        return VZO_EINVAL;
    if (n >= capacity)
        return VZO_ECAPACITY;

    /* Eq. 1: K_t = [K_{t-1}, k_t], V_t = [V_{t-1}, v_t]. */
    for (int32_t d = 0; d < D; ++d) {
        K[(int64_t)n * D + d] = k_new[d];
        V[(int64_t)n * D + d] = v_new[d];
    }
    pos[n] = new_pos;
    /* Eq. 6 zero-pads the previous score vector for the new token. */
    score[n] = 0.0;
    n += 1;

    /* Eq. 6: A^(t) = gamma * [A^(t-1), 0] + softmax(q K^T / sqrt(d)), summed over the group. */
    for (int32_t j = 0; j < n; ++j)
        score[j] *= gamma;

    double *logit = (double *)malloc(sizeof(double) * (size_t)n);
    if (!logit)
        return VZO_ENOMEM;
    for (int32_t h = 0; h < G; ++h) {
        const double *qh = q + (int64_t)h * D;
        double m = -INFINITY;
        for (int32_t j = 0; j < n; ++j) {
            double dot = 0.0;
            for (int32_t d = 0; d < D; ++d)
                dot += qh[d] * K[(int64_t)j * D + d];
            logit[j] = dot * scale;
            if (logit[j] > m)
                m = logit[j];
        }
        double z = 0.0;
        for (int32_t j = 0; j < n; ++j)
            z += exp(logit[j] - m);
        double *oh = out + (int64_t)h * D;
        for (int32_t d = 0; d < D; ++d)
            oh[d] = 0.0;
        for (int32_t j = 0; j < n; ++j) {
            const double p = exp(logit[j] - m) / z;
            score[j] += p;
            for (int32_t d = 0; d < D; ++d)
                oh[d] += p * V[(int64_t)j * D + d];
        }
    }
    free(logit);
    *n_io = n;
    return VZO_OK;
}

typedef struct {
    double score;
    int32_t pos;
    int32_t slot;
} vzo_candidate;

/* Higher score first; on equal scores the lower original position comes first. */
static int candidate_order(const void *a, const void *b)
{
    const vzo_candidate *x = (const vzo_candidate *)a;
    const vzo_candidate *y = (const vzo_candidate *)b;
    if (x->score > y->score)
        return -1;
    if (x->score < y->score)
        return 1;
    return (x->pos > y->pos) - (x->pos < y->pos);
}

static int position_order(const void *a, const void *b)
{
    const vzo_candidate *x = (const vzo_candidate *)a;
    const vzo_candidate *y = (const vzo_candidate *)b;
    return (x->pos > y->pos) - (x->pos < y->pos);
}

/*
 * Budgeted eviction for one unit (Sec. 3.2.2, Eq. 7-9), with the policy variants of the same
 * selection. If the cache holds more than `budget` rows it keeps T = sink attention sinks, a
 * recent window of M rows and the N = budget - T - M history rows with the highest decayed score.
 *
 *   history = 1   M = floor(budget * recent_frac): VoxZip's top-N history (Eq. 9)
 *   history = 0   M = budget - T, N = 0: sinks and a recent window only (the StreamingLLM policy
 *                 the paper compares against)
 *   fill = 0      sinks are the first T slots, the recent window the last M slots, candidates
 *                 the slots between; the kept rows move to [0, budget) in ascending slot order
 *                 (Eq. 7-8 as concatenation in order)
 *   fill = 1      the same sets chosen by position instead of slot (sinks: the T lowest
 *                 positions, recent: the M highest), so the cache need not be in time order;
 *                 kept rows already below `budget` stay where they are and the kept rows at
 *                 slots >= budget fill the evicted slots below it, both taken in ascending slot
 *                 order. On a cache in time order both modes keep the same rows.
 * Ties in the top-N go to the lower position. K, V, score and pos move together.
 *   margin  score of the N-th kept history row minus that of the best evicted one (+inf when
 *           there is no such pair or nothing is evicted); parity tests gate on it
 *   kept    if non-NULL, [n] flags: 1 for every slot kept (before the move)
 */
int vzo_evict_ex(int32_t D, int32_t *n_io, int32_t budget, int32_t sink, float recent_frac,
                 int32_t history, int32_t fill, double *K, double *V, double *score, int32_t *pos,
                 double *margin, int32_t *kept)
{
    const int32_t n = *n_io;
    *margin = INFINITY;
    if (budget < 0 || sink < 0 || D <= 0 || !(recent_frac >= 0.0f && recent_frac <= 1.0f) ||
        (history != 0 && history != 1) || (fill != 0 && fill != 1))
        return VZO_EINVAL;
    const int32_t T = sink;
    const int32_t M = history ? (int32_t)floor((double)recent_frac * (double)budget) : budget - T;
    const int32_t N = budget - T - M;
    if (N < 0 || M < 0)
        return VZO_EINVAL;
    if (kept)
        for (int32_t j = 0; j < n; ++j)
            kept[j] = 1;
    if (n <= budget)
        return VZO_OK;

    vzo_candidate *all = (vzo_candidate *)malloc(sizeof(vzo_candidate) * (size_t)n);
    int32_t *keep = (int32_t *)calloc((size_t)n, sizeof(int32_t));
    if (!all || !keep) {
        free(all);
        free(keep);
        return VZO_ENOMEM;
    }
    /* The slots in the order that defines "first" and "last": slot order, or time (position). */
    for (int32_t j = 0; j < n; ++j) {
        all[j].score = score[j];
        all[j].pos = pos[j];
        all[j].slot = j;
    }
    if (fill)
        qsort(all, (size_t)n, sizeof(vzo_candidate), position_order);
    for (int32_t r = 0; r < T; ++r)
        keep[all[r].slot] = 1;
    for (int32_t r = n - M; r < n; ++r)
        keep[all[r].slot] = 1;
    /* Eq. 9: I_hist = Top_N over the rows between the sinks and the recent window. */
    const int32_t nc = n - M - T;
    vzo_candidate *c = all + T;
    qsort(c, (size_t)nc, sizeof(vzo_candidate), candidate_order);
    if (N >= 1 && N < nc)
        *margin = c[N - 1].score - c[N].score;
    for (int32_t r = 0; r < N; ++r)
        keep[c[r].slot] = 1;
    if (kept)
        for (int32_t j = 0; j < n; ++j)
            kept[j] = keep[j];

    if (!fill) {
        /* Eq. 7-8: concatenate sinks, selected history and recent rows, preserving their order. */
        int32_t w = 0;
        for (int32_t j = 0; j < n; ++j) {
            if (!keep[j])
                continue;
            if (w != j) {
                memmove(K + (int64_t)w * D, K + (int64_t)j * D, sizeof(double) * (size_t)D);
                memmove(V + (int64_t)w * D, V + (int64_t)j * D, sizeof(double) * (size_t)D);
                score[w] = score[j];
                pos[w] = pos[j];
            }
            ++w;
        }
    } else {
        /* Hole filling: kept rows at slots >= budget go, in slot order, to the evicted slots
           below budget, in slot order. There are as many of each. */
        int32_t h = 0;
        for (int32_t j = budget; j < n; ++j) {
            if (!keep[j])
                continue;
            while (h < budget && keep[h])
                ++h;
            if (h >= budget)
                break; /* cannot happen: the kept rows number exactly `budget` */
            memcpy(K + (int64_t)h * D, K + (int64_t)j * D, sizeof(double) * (size_t)D);
            memcpy(V + (int64_t)h * D, V + (int64_t)j * D, sizeof(double) * (size_t)D);
            score[h] = score[j];
            pos[h] = pos[j];
            ++h;
        }
    }
    free(all);
    free(keep);
    *n_io = budget;
    return VZO_OK;
}

/* VoxZip's eviction (history = 1) with ordered compaction. */
int vzo_evict(int32_t D, int32_t *n_io, int32_t budget, int32_t sink, float recent_frac,
              double *K, double *V, double *score, int32_t *pos, double *margin, int32_t *kept)
{
    return vzo_evict_ex(D, n_io, budget, sink, recent_frac, 1, 0, K, V, score, pos, margin, kept);
}

/*
 * The whole path for one unit: stage 1 over the prefill rows, then `steps` decode steps; after
 * step t (1-based) with t % interval == 0 the unit is evicted down to its budget.
 *
 * Inputs: the stage-1 arguments of vzo_stage1 for K and V rows (xk, xv, anchor_k, anchor_v),
 * q [steps][G][D], k_new and v_new [steps][D], new_pos [steps].
 * Outputs:
 *   out          [steps][G][D]
 *   score_before [steps/interval][capacity]  scores just before each eviction (0-padded)
 *   pos_before   [steps/interval][capacity]  (run_unit_ex, may be NULL) positions just before
 *                                            each eviction (-1 padded)
 *   len_before   [steps/interval]            cache length just before each eviction
 *   kept_pos     [steps/interval][budget]    positions of the rows after each eviction
 *                                            (-1 padded when the cache was within budget)
 *   margin       [steps/interval]            see vzo_evict
 *   K, V, score, pos, n_final                the final cache
 *   slot_map     [in_len]                    stage-1 slot of every prefill token
 *   stage1_len                               cache length after stage 1
 */
int vzo_run_unit_ex(int32_t in_len, int32_t audio_begin, int32_t audio_len, int32_t n_spans,
                    const int32_t *span_start, const int32_t *span_end, const int32_t *span_groups,
                    int32_t D, const double *xk, const double *xv, const double *anchor_k,
                    const double *anchor_v, int32_t cache_is_bf16, int32_t G, int32_t capacity,
                    int32_t steps, const double *q, const double *k_new, const double *v_new,
                    const int32_t *new_pos, double gamma, double scale, int32_t interval,
                    int32_t budget, int32_t sink, float recent_frac, int32_t history, int32_t fill,
                    double *out, double *score_before, int32_t *pos_before, int32_t *len_before,
                    int32_t *kept_pos, double *margin, double *K, double *V, double *score,
                    int32_t *pos, int32_t *n_final, int32_t *slot_map, int32_t *stage1_len)
{
    if (interval <= 0 || steps < 0)
        return VZO_EINVAL;
    double *scratch = (double *)malloc(sizeof(double) * (size_t)capacity * (size_t)D);
    int32_t *pos_v = (int32_t *)malloc(sizeof(int32_t) * (size_t)(capacity > 0 ? capacity : 1));
    if (!scratch || !pos_v) {
        free(scratch);
        free(pos_v);
        return VZO_ENOMEM;
    }
    int32_t n = 0, n_v = 0;
    int rc = vzo_stage1(in_len, audio_begin, audio_len, n_spans, span_start, span_end, span_groups,
                        D, xk, anchor_k, cache_is_bf16, capacity, scratch, K, pos, slot_map, &n);
    if (rc == VZO_OK)
        rc = vzo_stage1(in_len, audio_begin, audio_len, n_spans, span_start, span_end,
                        span_groups, D, xv, anchor_v, cache_is_bf16, capacity, scratch, V, pos_v,
                        slot_map, &n_v);
    free(scratch);
    free(pos_v);
    if (rc != VZO_OK)
        return rc;
    *stage1_len = n;
    for (int32_t j = 0; j < n; ++j)
        score[j] = 0.0;

    int32_t ev = 0;
    for (int32_t t = 1; t <= steps; ++t) {
        rc = vzo_decode_step(D, G, capacity, &n, K, V, score, pos,
                             q + (int64_t)(t - 1) * G * D, k_new + (int64_t)(t - 1) * D,
                             v_new + (int64_t)(t - 1) * D, new_pos[t - 1], gamma, scale,
                             out + (int64_t)(t - 1) * G * D);
        if (rc != VZO_OK)
            return rc;
        if (t % interval == 0) {
            for (int32_t j = 0; j < capacity; ++j) {
                score_before[(int64_t)ev * capacity + j] = j < n ? score[j] : 0.0;
                if (pos_before)
                    pos_before[(int64_t)ev * capacity + j] = j < n ? pos[j] : -1;
            }
            len_before[ev] = n;
            rc = vzo_evict_ex(D, &n, budget, sink, recent_frac, history, fill, K, V, score, pos,
                              &margin[ev], NULL);
            if (rc != VZO_OK)
                return rc;
            for (int32_t j = 0; j < budget; ++j)
                kept_pos[(int64_t)ev * budget + j] = j < n ? pos[j] : -1;
            ++ev;
        }
    }
    *n_final = n;
    return VZO_OK;
}

/* The whole path with VoxZip's eviction and ordered compaction. */
int vzo_run_unit(int32_t in_len, int32_t audio_begin, int32_t audio_len, int32_t n_spans,
                 const int32_t *span_start, const int32_t *span_end, const int32_t *span_groups,
                 int32_t D, const double *xk, const double *xv, const double *anchor_k,
                 const double *anchor_v, int32_t cache_is_bf16, int32_t G, int32_t capacity,
                 int32_t steps, const double *q, const double *k_new, const double *v_new,
                 const int32_t *new_pos, double gamma, double scale, int32_t interval,
                 int32_t budget, int32_t sink, float recent_frac, double *out,
                 double *score_before, int32_t *len_before, int32_t *kept_pos, double *margin,
                 double *K, double *V, double *score, int32_t *pos, int32_t *n_final,
                 int32_t *slot_map, int32_t *stage1_len)
{
    return vzo_run_unit_ex(in_len, audio_begin, audio_len, n_spans, span_start, span_end,
                           span_groups, D, xk, xv, anchor_k, anchor_v, cache_is_bf16, G, capacity,
                           steps, q, k_new, v_new, new_pos, gamma, scale, interval, budget, sink,
                           recent_frac, 1, 0, out, score_before, NULL, len_before, kept_pos,
                           margin, K, V, score, pos, n_final, slot_map, stage1_len);
}
