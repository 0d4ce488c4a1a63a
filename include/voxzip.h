/*
 * voxzip.h -- C ABI of the VoxZip KV-cache compression library for NVIDIA GB300 (sm_103a).
 *
 * VoxZip (arxiv 2608.08569) compresses the KV cache of a speech LLM in two stages:
 *   stage 1 (Sec. 3.2.1) fuses each ASR-aligned audio span of the prefilled cache into a few
 *           averaged rows (Eq. 4, optional anchor add, Eq. 5);
 *   stage 2 (Sec. 3.2.2) keeps a temporally decayed accumulated attention score per cached token
 *           (Eq. 6), updated by every decode step (Eq. 1-2), and evicts down to a budget
 *           by keeping T sinks, a recent window of M tokens and the top-N scored history
 *           (Eq. 7-9).
 * The library exports one call per step: voxzip_anchor_fuse, voxzip_decode_step, voxzip_evict;
 * and, for stage 1 where the paper runs it (on input embeddings, from ASR segments),
 * voxzip_segments_to_spans (host) and voxzip_embed_fuse.
 *
 * Conventions shared by every entry point
 *   - A "unit" is one (sequence b, layer l, kv-head h). All state is per unit and units are
 *     independent.
 *   - Every tensor pointer is caller-owned DEVICE memory, dense and row-major in the layout given
 *     beside it. The library never allocates, frees or copies to the host on these paths.
 *   - Element type: K/V cache, prefill rows, anchors, q, k_new, v_new and out all have the
 *     descriptor's dtype (bf16 or fp32). Scores are fp32, positions and lengths int32.
 *   - Calls are asynchronous on `stream` and do not synchronise the host.
 *   - Synchronous errors (bad descriptor, null required pointer, unsupported shape, workspace too
 *     small) return an error status and launch nothing. A failed launch returns VOXZIP_ECUDA.
 *   - Errors that depend on device data (malformed spans, a cache that would overflow its
 *     capacity, a length above the caller's hint, a budget smaller than sink + recent) skip the
 *     affected unit or sequence and set a bit in the device status word, read and cleared by
 *     voxzip_get_status. Kernels never trap.
 *   - Cache layout:  K, V   [B][L][Hkv][C][D]      (C = capacity slots per unit)
 *                    score  [B][L][Hkv][C]  fp32    decayed accumulated attention (Eq. 6)
 *                    pos    [B][L][Hkv][C]  int32   original token index of each slot
 *                    len    [B][L][Hkv]     int32   cache length n of each unit
 *     Slots [0, n) of a unit are valid. Stage 1, decode appends and the ordered eviction keep them
 *     in chronological (ascending position) order; the hole-filling eviction
 *     (VOXZIP_COMPACT_FILL of voxzip_evict_ex) does not: it moves kept rows into evicted slots, so
 *     a unit's slots are then in no particular order. No call depends on slot order.
 */
#ifndef VOXZIP_H
#define VOXZIP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st *voxzip_stream_t;

typedef enum {
    VOXZIP_OK = 0,
    VOXZIP_EINVAL = 1,       /* invalid argument; nothing was launched */
    VOXZIP_EUNSUPPORTED = 2, /* valid request outside what the kernels implement */
    VOXZIP_ECUDA = 3,        /* a CUDA runtime call or kernel launch failed */
    VOXZIP_ESCRATCH = 4      /* the request needs more scratch than voxzip_anchor_fuse_noalloc's
                                fixed 4 MiB; nothing was launched */
} voxzip_status;

/* Bits of the device status word (asynchronous errors). */
#define VOXZIP_DEV_BAD_SPANS 0x1u  /* a sequence's spans were malformed; its stage 1 was skipped */
#define VOXZIP_DEV_CAPACITY 0x2u   /* stage-1 output or an append would exceed the capacity */
#define VOXZIP_DEV_LEN_HINT 0x4u   /* a unit was longer than the call's max_len; it was skipped */
#define VOXZIP_DEV_BAD_BUDGET 0x8u /* budget < sink + floor(budget * recent_frac); unit skipped */
#define VOXZIP_DEV_TIMEOUT 0x10u   /* a bounded wait inside a kernel gave up; outputs of that unit
                                      are not valid (never expected; reported instead of hanging) */
#define VOXZIP_DEV_BAD_POSITIONS 0x20u /* a unit's positions were not unique, so a hole-filling
                                          eviction could not keep exactly `budget` rows */
#define VOXZIP_DEV_BOUNDS 0x40u    /* checked builds only (-DVOXZIP_CHECKED): an index a kernel was
                                      about to use fell outside its buffer; the access was skipped */

typedef enum { VOXZIP_F32 = 0, VOXZIP_BF16 = 1 } voxzip_dtype;

typedef struct {
    int32_t batch;    /* B, sequences */
    int32_t layers;   /* L */
    int32_t q_heads;  /* Hq */
    int32_t kv_heads; /* Hkv; divides Hq. Query head i reads kv head i / (Hq / Hkv). */
    int32_t head_dim; /* D, 64 or 128 */
    int32_t capacity; /* C, slots per unit */
    int32_t dtype;    /* voxzip_dtype of every K/V-typed tensor */
} voxzip_cache_desc;

/*
 * Stage 1: semantic-anchored fusion of the prefilled cache (Sec. 3.2.1, Eq. 4, anchor addition,
 * Eq. 5), for every layer and kv-head of every sequence.
 *
 * The ASR segments arrive as token-index spans, i.e. after the time-to-index map of Eq. 3.
 * Sequence b's spans are entries [span_off[b], span_off[b+1]) of span_start/span_end/span_groups;
 * they must be sorted, non-overlapping, lie inside [audio_begin[b], audio_begin[b]+audio_len[b])
 * and have span_groups >= 1 (span_groups is L_t, the length of the span's transcription). A span
 * of length l with g = min(span_groups, l) groups yields g rows; group j averages prefill rows
 * [start + floor(j*l/g), start + floor((j+1)*l/g)) in fp32 in token order, divides by the group
 * size, adds the anchor row if given, and rounds once to the cache dtype. Empty spans yield
 * nothing. Every other token (text, or audio no span covers) is copied unchanged. Output rows
 * keep chronological order; pos[slot] = index of the slot's first prefill token; score = 0;
 * len = number of rows, the same for every unit of a sequence.
 *
 *   k_prefill, v_prefill  [B][L][Hkv][prefill_stride][D]; rows [0, in_len[b]) are read, each
 *                         once. Device memory, or page-locked host memory that the device
 *                         addresses directly (unified addressing, as across the C2C link of a
 *                         Grace-Blackwell node): the kernels then stream the rows over the host
 *                         link from CTAs on half the SMs, need no device copy of the prompt, and
 *                         leave the other SMs to kernels running beside them.
 *   in_len, audio_begin, audio_len  [B] device int32
 *   span_off              [B+1] device int32, span_off[0] = 0, span_off[B] = num_spans
 *   span_start, span_end, span_groups  [num_spans] device int32
 *   anchor_k, anchor_v    NULL (anchor term zero) or [B][L][Hkv][anchor_stride][D]; group j of
 *                         sequence b's span i adds row (sum of span_groups over b's spans before
 *                         i) + j. Both NULL or both non-NULL.
 *   k_cache, v_cache, score, pos, len   outputs, cache layout above
 *   slot_map              NULL or [B][prefill_stride] device int32: output slot of every token
 *   workspace             device scratch of at least voxzip_anchor_fuse_workspace_size() bytes,
 *                         256-byte aligned; contents need not be initialised
 * Device errors: VOXZIP_DEV_BAD_SPANS or VOXZIP_DEV_CAPACITY; the sequence's units get len = 0.
 */
voxzip_status voxzip_anchor_fuse(const voxzip_cache_desc *desc, const void *k_prefill,
                                 const void *v_prefill, int32_t prefill_stride,
                                 const int32_t *in_len, const int32_t *audio_begin,
                                 const int32_t *audio_len, const int32_t *span_off,
                                 int32_t num_spans, const int32_t *span_start,
                                 const int32_t *span_end, const int32_t *span_groups,
                                 const void *anchor_k, const void *anchor_v, int32_t anchor_stride,
                                 void *k_cache, void *v_cache, float *score, int32_t *pos,
                                 int32_t *len, int32_t *slot_map, void *workspace,
                                 size_t workspace_bytes, voxzip_stream_t stream);

/* Bytes of workspace voxzip_anchor_fuse needs (0 if the descriptor is invalid). */
size_t voxzip_anchor_fuse_workspace_size(const voxzip_cache_desc *desc, int32_t prefill_stride,
                                         int32_t num_spans);

/*
 * Stage 1 exactly as voxzip_anchor_fuse, but without a workspace argument: for callers that cannot
 * allocate device memory, such as a runtime whose device memory belongs entirely to another
 * framework's pool, or an audio front-end that must not allocate while it serves requests. The
 * paper has no counterpart; this is a deployment variant of the same computation.
 *
 * Its scratch is a fixed 4 MiB array compiled into the library, held by every GPU that loads the
 * library until the process exits. A request whose voxzip_anchor_fuse_workspace_size exceeds 4 MiB
 * returns VOXZIP_ESCRATCH and launches nothing. The need is 12 bytes per prompt-token slot
 * (batch x prefill_stride) plus 12 per span, 8 per sequence and under 2.5 KiB of alignment padding:
 * 4 MiB covers, for instance, 4 sequences of 60 000 tokens or 32 of 8 000 with one span per five
 * tokens. voxzip_anchor_fuse_workspace_size gives the exact figure to compare against 4 MiB.
 *   - The first call on a device looks up the array's device address (cudaGetSymbolAddress) with
 *     that device current; make that first call before any stream capture.
 *   - Every call on a device shares the array and it keeps the last call's contents; no part of it
 *     needs to start at zero. Calls that overlap on the GPU (unordered streams) race on it.
 * Arguments, layouts, results and device errors are those of voxzip_anchor_fuse.
 */
voxzip_status voxzip_anchor_fuse_noalloc(const voxzip_cache_desc *desc, const void *k_prefill,
                                         const void *v_prefill, int32_t prefill_stride,
                                         const int32_t *in_len, const int32_t *audio_begin,
                                         const int32_t *audio_len, const int32_t *span_off,
                                         int32_t num_spans, const int32_t *span_start,
                                         const int32_t *span_end, const int32_t *span_groups,
                                         const void *anchor_k, const void *anchor_v,
                                         int32_t anchor_stride, void *k_cache, void *v_cache,
                                         float *score, int32_t *pos, int32_t *len,
                                         int32_t *slot_map, voxzip_stream_t stream);

/*
 * The semantic set of one sequence from ASR output (Sec. 3.2.1): the confidence filter and the
 * time-to-index map of Eq. 3. HOST function: every pointer is host memory; no CUDA call, no GPU.
 *
 * Segment i (times in seconds, sorted by t_start) is kept when confidence[i] > threshold (the
 * paper keeps segments above 0.3). Its interval of audio tokens is
 *     [floor(audio_len * (t_start / tau_total)), floor(audio_len * (t_end / tau_total)))   (Eq. 3)
 * evaluated in double in that order and clamped to [0, audio_len]. A kept segment that would
 * start before the previous kept one ends starts where that one ends (an empty interval if
 * nothing is left: it yields no row, but its text rows still count for the anchor offsets).
 *
 *   t_start, t_end, confidence  [n] double; text_len [n] int32 >= 1 (L_t, the segment's tokens)
 *   tau_total      duration of the audio, seconds, finite and > 0
 *   audio_len      L_a, audio tokens; audio_begin = prompt index of the first one
 *   span_start, span_end, span_groups, seg_index   outputs, room for n entries each: the kept
 *                  segments in order as prompt-index spans, their L_t, and their input index
 *   num_spans      output: number of kept segments
 * The outputs feed voxzip_anchor_fuse / voxzip_embed_fuse (span_groups = n_groups; the anchor
 * rows are the embedded texts of the kept segments, concatenated in this order).
 * Errors: VOXZIP_EINVAL for n < 0, a NULL pointer (with n > 0), unsorted segments,
 * t_end < t_start (or NaN), text_len < 1, a bad tau_total, audio_len or audio_begin < 0.
 */
voxzip_status voxzip_segments_to_spans(int32_t n, const double *t_start, const double *t_end,
                                       const double *confidence, const int32_t *text_len,
                                       double tau_total, int32_t audio_len, int32_t audio_begin,
                                       double threshold, int32_t *span_start, int32_t *span_end,
                                       int32_t *span_groups, int32_t *seg_index,
                                       int32_t *num_spans);

typedef struct {
    int32_t batch;    /* B, sequences */
    int32_t d_model;  /* d, hidden size; rows are whole 16-byte vectors (multiple of 8 bf16 or
                         4 fp32 elements) */
    int32_t capacity; /* C, output rows per sequence */
    int32_t dtype;    /* voxzip_dtype of e_in, e_text and e_out */
} voxzip_embed_desc;

/*
 * Stage 1 at the embedding level, the setting the paper evaluates (Sec. 3.2.1): the audio
 * embeddings E_A of each sequence are fused under its semantic set before the LLM runs. Group j
 * of a span (Eq. 4 grouping, as in voxzip_anchor_fuse) becomes mean(E_A rows of the group) +
 * e_t,j, the j-th embedded text token of the span's transcription (the semantic anchor);
 * background audio and every token outside the audio region are copied (Eq. 5).
 *
 * keep_background = 0 gives the stage-1 ablation's T+A (Partial) configuration: audio that no
 * span covers is dropped (slot_map -1), text outside the audio region is still copied.
 *
 *   e_in        [B][stride][d] prompt embeddings; rows [0, in_len[b]) are read; the audio
 *               region is [audio_begin[b], audio_begin[b] + audio_len[b])
 *   in_len, audio_begin, audio_len, span_off, span_start, span_end, span_groups
 *               device int32, exactly as for voxzip_anchor_fuse
 *   e_text      NULL (no anchor term) or [B][text_stride][d]: sequence b's embedded texts,
 *               concatenated in span order; group j of span i adds row
 *               (sum of span_groups over b's spans before i) + j
 *   e_out       [B][capacity][d] output rows; pos [B][capacity] int32: first prompt token of each
 *               output row; len [B] int32: output rows per sequence
 *   slot_map    NULL or [B][stride] int32: output row of every prompt token, -1 if dropped
 *   workspace   device scratch of voxzip_embed_fuse_workspace_size() bytes, 256-byte aligned
 * All tensor pointers are device memory, 16-byte aligned. Device errors: VOXZIP_DEV_BAD_SPANS or
 * VOXZIP_DEV_CAPACITY skip the sequence (len = 0).
 */
voxzip_status voxzip_embed_fuse(const voxzip_embed_desc *desc, const void *e_in, int32_t stride,
                                const int32_t *in_len, const int32_t *audio_begin,
                                const int32_t *audio_len, const int32_t *span_off,
                                int32_t num_spans, const int32_t *span_start,
                                const int32_t *span_end, const int32_t *span_groups,
                                const void *e_text, int32_t text_stride, int32_t keep_background,
                                void *e_out, int32_t *pos, int32_t *len, int32_t *slot_map,
                                void *workspace, size_t workspace_bytes, voxzip_stream_t stream);

/* Bytes of workspace voxzip_embed_fuse needs (0 if the arguments are invalid). */
size_t voxzip_embed_fuse_workspace_size(const voxzip_embed_desc *desc, int32_t stride,
                                        int32_t num_spans);

/*
 * One decode step for layers [layer_begin, layer_begin + layer_count) of every sequence:
 * append (Eq. 1), GQA attention (Eq. 2) and the decayed-score update (Eq. 6), fused so that
 * each cached K and V row is read once.
 *
 * For every unit with length n: the new token's k_new/v_new are written to slot n with
 * pos = new_pos[b]; then for each of the G = Hq/Hkv query heads of the unit,
 *     p_h = softmax(scale * q_h K^T) over the n+1 rows,   out_h = p_h V,
 * and every slot's score becomes  gamma * score + sum_h p_h  (the new slot starts from 0);
 * len becomes n + 1.
 *
 *   q, out          [layer_count][B][Hq][D]
 *   k_new, v_new    [layer_count][B][Hkv][D]
 *   new_pos         [B] device int32, original index of the token being decoded
 *   gamma           decay in (0, 1]; 1 is plain accumulation
 *   sm_scale        logit scale; <= 0 selects 1/sqrt(D)
 *   max_len         host-side upper bound on n + 1 over all units of the call (sizes the launch);
 *                   <= 0 selects the capacity. Units above it are skipped with
 *                   VOXZIP_DEV_LEN_HINT.
 * Requires D in {64, 128}, G <= 16. Device errors: VOXZIP_DEV_CAPACITY (n == C), LEN_HINT.
 */
voxzip_status voxzip_decode_step(const voxzip_cache_desc *desc, int32_t layer_begin,
                                 int32_t layer_count, const void *q, const void *k_new,
                                 const void *v_new, const int32_t *new_pos, void *k_cache,
                                 void *v_cache, float *score, int32_t *pos, int32_t *len,
                                 float gamma, float sm_scale, int32_t max_len, void *out,
                                 voxzip_stream_t stream);

/*
 * Budgeted eviction (Sec. 3.2.2, Eq. 7-9) for layers [layer_begin, layer_begin + layer_count).
 * A unit with n <= budget[b] is left alone. Otherwise, with T = sink,
 * M = floor(budget[b] * recent_frac) (evaluated in double) and N = budget[b] - T - M, it keeps
 * slots [0, T), slots [n - M, n) and the N slots of [T, n - M) with the highest score, ties
 * going to the lower position, and moves the kept rows (K, V, score, pos) to [0, budget[b]) in
 * ascending slot order, in place; len becomes budget[b].
 *
 *   budget  [B] device int32
 * Device errors: VOXZIP_DEV_BAD_BUDGET (N < 0).
 */
voxzip_status voxzip_evict(const voxzip_cache_desc *desc, int32_t layer_begin,
                           int32_t layer_count, void *k_cache, void *v_cache, float *score,
                           int32_t *pos, int32_t *len, const int32_t *budget, int32_t sink,
                           float recent_frac, voxzip_stream_t stream);

typedef enum {
    VOXZIP_COMPACT_ORDERED = 0, /* kept rows move to [0, budget) in slot order (Eq. 7-8) */
    VOXZIP_COMPACT_FILL = 1     /* kept rows beyond the budget fill the evicted slots below it */
} voxzip_compaction;

typedef struct {
    int32_t sink;            /* T, attention sinks kept (the paper uses 4) */
    float recent_frac;       /* M = floor(budget * recent_frac) recent rows (the paper: 0.2) */
    int32_t history;         /* 1: the top-N history by decayed score (VoxZip, Eq. 9);
                                0: no history, M = budget - T (the StreamingLLM policy) */
    int32_t budget_stride_b; /* the budget of unit (b, l, h) is                                */
    int32_t budget_stride_l; /*   budget[b * budget_stride_b + l * budget_stride_l]            */
                             /* (1, 0): one per sequence; (L, 1): [B][L], one per layer        */
    int32_t compaction;      /* voxzip_compaction */
} voxzip_evict_policy;

/*
 * Eviction under a policy: the same selection as voxzip_evict with the switches above.
 *
 * VOXZIP_COMPACT_FILL chooses the sinks as the T lowest positions and the recent window as the M
 * highest, so the cache need not be kept in time order. Kept rows below the budget stay where
 * they are; the kept rows at slots >= budget move, in ascending slot order, into the evicted
 * slots below the budget, in ascending slot order. At most n - budget rows move, against up to
 * `budget` for the ordered compaction. On a cache in time order both keep the same rows. The
 * decode step does not depend on slot order. A unit's positions must be unique; otherwise it
 * reports VOXZIP_DEV_BAD_POSITIONS.
 *
 * The budget array is device int32 and covers every index the strides reach for the layers
 * evicted. Errors: VOXZIP_EINVAL for a NULL policy, sink < 0, recent_frac outside [0, 1],
 * history or compaction outside their values, or a negative stride; otherwise as voxzip_evict.
 */
voxzip_status voxzip_evict_ex(const voxzip_cache_desc *desc, int32_t layer_begin,
                              int32_t layer_count, void *k_cache, void *v_cache, float *score,
                              int32_t *pos, int32_t *len, const int32_t *budget,
                              const voxzip_evict_policy *policy, voxzip_stream_t stream);

/*
 * Paged cache (for serving many turns: memory follows the live cache, not a fixed capacity).
 *
 * K and V rows live in pools of pages of VOXZIP_PAGE_TOKENS rows. Slot s of unit u is row
 * (s % 64) of page page_table[u][s / 64]; scores, positions and lengths stay dense as in the
 * cache layout above (8 bytes per slot). Free pages are a device-side stack, so every call of the
 * decode loop runs without a host round trip and can be captured in a CUDA graph:
 *   - voxzip_paged_init gives unit u page u for slot 0 and stacks the rest as free;
 *   - voxzip_anchor_fuse_paged returns each unit's pages and takes the ones its stage-1 rows need;
 *   - voxzip_decode_step_paged takes a page when an append fills the unit's last one;
 *   - voxzip_evict_paged returns the pages beyond the budget.
 * After every call a unit of length n holds the pages of slots [0, n] (the next append's slot
 * included) when the pool allowed it. A decode whose slot has no page, or a stage 1 the pool
 * cannot hold, sets VOXZIP_DEV_CAPACITY and skips the unit. Which free page a unit receives depends
 * on the order in which units ran, so it is not deterministic.
 */
#define VOXZIP_PAGE_TOKENS 64

typedef struct {
    void *k_pool;        /* [pages][64][D] in the descriptor's dtype, 16-byte aligned */
    void *v_pool;        /* [pages][64][D] */
    int32_t *page_table; /* [B][L][Hkv][max_pages] device int32: page of slots [64 p, 64 p + 64), -1 none */
    int32_t *free_pages; /* [pages] device int32: stack of free page indices */
    int32_t *free_count; /* device int32: stack entries in use */
    int32_t pages;       /* pool size; at least B * L * Hkv */
    int32_t max_pages;   /* pages per unit; the descriptor's capacity must be 64 * max_pages */
} voxzip_paged_cache;

/* Empty every unit (len = 0, page u of the pool for its slot 0) and stack the other pages. */
voxzip_status voxzip_paged_init(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged,
                                int32_t *len, voxzip_stream_t stream);

/* voxzip_anchor_fuse into a paged cache (same arguments and results; K/V rows go to the pages). */
voxzip_status voxzip_anchor_fuse_paged(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged,
                                       const void *k_prefill, const void *v_prefill,
                                       int32_t prefill_stride, const int32_t *in_len,
                                       const int32_t *audio_begin, const int32_t *audio_len,
                                       const int32_t *span_off, int32_t num_spans,
                                       const int32_t *span_start, const int32_t *span_end,
                                       const int32_t *span_groups, const void *anchor_k,
                                       const void *anchor_v, int32_t anchor_stride, float *score,
                                       int32_t *pos, int32_t *len, int32_t *slot_map, void *workspace,
                                       size_t workspace_bytes, voxzip_stream_t stream);

/* Bytes of workspace voxzip_anchor_fuse_paged needs (0 if the arguments are invalid). */
size_t voxzip_anchor_fuse_paged_workspace_size(const voxzip_cache_desc *desc, int32_t prefill_stride,
                                               int32_t num_spans);

/* voxzip_decode_step on a paged cache (bf16, head_dim 64 or 128, group <= 16; else
   VOXZIP_EUNSUPPORTED). */
voxzip_status voxzip_decode_step_paged(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged,
                                       int32_t layer_begin, int32_t layer_count, const void *q,
                                       const void *k_new, const void *v_new, const int32_t *new_pos,
                                       float *score, int32_t *pos, int32_t *len, float gamma,
                                       float sm_scale, int32_t max_len, void *out,
                                       voxzip_stream_t stream);

/* voxzip_evict_ex on a paged cache; the pages beyond the new length's are returned. */
voxzip_status voxzip_evict_paged(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged,
                                 int32_t layer_begin, int32_t layer_count, float *score, int32_t *pos,
                                 int32_t *len, const int32_t *budget, const voxzip_evict_policy *policy,
                                 voxzip_stream_t stream);

/*
 * Waits for `stream`, then returns the device status word of the current device in *bits
 * (VOXZIP_DEV_* flags accumulated by earlier calls) and clears it.
 */
voxzip_status voxzip_get_status(uint32_t *bits, voxzip_stream_t stream);

/*
 * Self-test of the bounded waits: failure detection exercised without a GPU fault. One CTA arms an
 * mbarrier for 16 bytes that never arrive and waits on it with the bounded wait the decode kernel
 * uses on its TMA ring, giving up after `limit` polls (1 to 2^20). The give-up sets
 * VOXZIP_DEV_TIMEOUT in the status word, as a decode whose loads never landed would. No copy is
 * issued, so nothing can fault. Asynchronous on `stream`; VOXZIP_EINVAL for a limit out of range.
 */
voxzip_status voxzip_selftest_bounded_wait(uint32_t limit, voxzip_stream_t stream);

/*
 * Measurement helper, not a step of the method: reads `bytes` of device memory at `p` once with
 * 16-byte loads spread over the whole GPU, as a plain streaming read, and does nothing with the
 * data (a checksum that no input produces in practice is the only store, to `sink`, a caller-owned
 * device word). It is the most a single launch of that size can reach, so it serves as the ceiling
 * a kernel moving the same bytes is measured against. Like the decode and eviction launches it is a
 * programmatic dependent of the previous kernel on `stream`, so a captured loop of them overlaps
 * each launch's start with the previous one's tail exactly as a loop of decode steps does.
 * `p` 16-byte aligned, `bytes` a multiple of 16; VOXZIP_EINVAL otherwise. Asynchronous.
 */
voxzip_status voxzip_stream_read(const void *p, size_t bytes, uint32_t *sink, voxzip_stream_t stream);

/* Human-readable name of a status code (static storage). */
const char *voxzip_status_string(voxzip_status status);

/* Library ABI version: 100 * major + minor. */
int32_t voxzip_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VOXZIP_H */
