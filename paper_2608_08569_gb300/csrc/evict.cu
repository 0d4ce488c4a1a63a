// Budgeted eviction of VoxZip (Sec. 3.2.2, Eq. 7-9): keep T sinks, the M most recent rows and
// the top-N history rows by decayed score, then compact K, V, score and pos in place.
// Policy switches: the budget of a unit is read at budget[b * stride_b + layer * stride_l] (one
// per sequence, or per layer); without history the recent window is budget - T rows (the
// StreamingLLM baseline).
//
// evict_kernel (ordered compaction):
// One CTA of 256 threads per unit:
//   select   MSB-first radix select (4 passes of 8 bits) over an order-preserving 32-bit image of
//            the history scores gives the N-th best score. Only when that score is tied and not all
//            tied rows fit does a second select over their positions (ascending) run, so that
//            equal scores keep the lower position. Positions within a unit are unique.
//   compact  slots are scanned 256 at a time; a block scan gives each kept slot its rank, and the
//            kept slots of up to kSegment ranks are listed in shared memory. Rows then move in
//            rank order, kRows rows per sub-chunk, through a kPipe-deep ring of shared-memory
//            stages filled by cp.async: the loads of the next kPipe-1 sub-chunks are in flight
//            while one is stored. A kept row never moves up (dest = rank <= src). Sources of a
//            later sub-chunk sit at slots >= its ranks, beyond every destination of an earlier one,
//            so in-flight loads never see a store; and a barrier after all of a sub-chunk's loads
//            have landed precedes its stores, so no row is overwritten before it is read. Neither
//            argument depends on how the rows travel:
//            - many units per launch: every thread copies 16-byte vectors by cp.async through a
//              narrow ring (8 KB stages, 3 deep, six CTAs per SM, so a 48-layer launch of four
//              sequences is resident at once);
//            - at most two units per SM: that few CTAs would each be bound by their own instruction
//              issue and latency, not by HBM. They take a wide ring instead (up to 96 KB of stages,
//              two CTAs per SM), in which one warp moves each run of consecutive source rows in,
//              and each sub-chunk's moving rows out, by 1-D bulk copies.
//
// evict_fill_kernel (hole filling): sinks are the T lowest positions and the recent window the M
// highest (both cuts in one radix sweep per digit), so the cache need not be in time order; the
// history select is the same. Kept rows below the budget stay; the kept rows at slots >= budget
// move, in ascending slot order, into the evicted slots below the budget, in ascending slot
// order: at most n - budget rows move. Sources lie at or above the budget and destinations below
// it, so no copy can read a row another one wrote. Its time is the latency of its passes, so the
// block size follows the unit count: 256 threads when the launch fits one wave of 4 CTAs per SM,
// else 192 threads (6 per SM).
#include "common.cuh"
#include "evict_policy.cuh"
#include "paged.cuh"
#include "ptx.cuh"

namespace voxzip {
namespace {

constexpr int kThreads = 256;
// Hole filling runs 256-thread CTAs (4 per SM) when a launch's units fit one wave of those, else
// 192-thread CTAs (6 per SM: the 768 units of 4 sequences x 48 layers x 4 kv-heads in one wave).
// Its time is the latency of its radix passes, so fewer waves beat more threads per pass.
template <int NT>
struct FillShape {
    static constexpr int kCtasPerSm = NT <= 192 ? 6 : 4;
};
constexpr int kSegment = 1024;   // ranks listed per compaction segment
constexpr uint32_t kEvictWaitLimit = 1u << 22;  // polls before an mbarrier wait gives up

// The narrow compaction ring: every thread copies kVecs 16-byte vectors per sub-chunk by cp.async,
// kDepth sub-chunks in flight (8 KB stages, six CTAs per SM).
struct NarrowRing {
    static constexpr int kVecs = 2, kDepth = 3, kCtasPerSm = 6;
};
// The wide ring: one warp moves 32 rows per sub-chunk, each K and V row by one bulk copy in and
// one out; up to 96 KB of stages (two CTAs per SM).
template <typename T, int D>
struct BulkRing {
    static constexpr int kRows = 32;
    static constexpr int kRowBytes = D * (int)sizeof(T);
    static constexpr int kStageBytes = 2 * kRows * kRowBytes;  // K rows, then V rows
    static constexpr int kDepth = 98304 / kStageBytes < 8 ? 98304 / kStageBytes : 8;
    static constexpr size_t kBytes = (size_t)kDepth * kStageBytes;
    static constexpr int kCtasPerSm = 2;
    static_assert(kDepth >= 3, "a sub-chunk in flight and two stores draining");
};

// 1-D bulk copies (the async proxy): global -> shared counted on an mbarrier, shared -> global in
// bulk groups. Addresses 16-byte aligned, sizes multiples of 16.
__device__ __forceinline__ void bulk_load(void *smem_dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     ptx::smem_u32(smem_dst)),
                 "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(ptx::smem_u32(bar))
                 : "memory");
}
__device__ __forceinline__ void bulk_store(void *dst, const void *smem_src, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(reinterpret_cast<uint64_t>(dst)),
                 "r"(ptx::smem_u32(smem_src)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void bulk_wait_read() {  // at most N groups still reading shared memory
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

struct EvictParams {
    void *k_cache, *v_cache;
    float *score;
    int32_t *pos, *len;
    const int32_t *budget;
    int32_t *status;
    int32_t B, L, Hkv, C, layer_begin, sink;
    int32_t budget_stride_b, budget_stride_l, history;
    float recent_frac;
    PageView pv;  // paged instantiations only: K/V rows through the page table, pools as k/v_cache
    int64_t rows; // K / V rows of the cache, or of the pools
};

// The unit's budget and its split into T sinks, M recent rows and N history rows.
struct Split {
    int32_t bud, T, M, N;
};
__device__ __forceinline__ Split split_of(const EvictParams &p, const UnitIdx &ui) {
    Split s;
    s.bud = p.budget[(int64_t)ui.b * p.budget_stride_b + (int64_t)(p.layer_begin + ui.l_local) * p.budget_stride_l];
    s.T = p.sink;
    s.M = p.history ? (int32_t)floor((double)p.recent_frac * (double)s.bud) : s.bud - s.T;
    s.N = s.bud - s.T - s.M;
    return s;
}

__device__ __forceinline__ uint32_t score_key(float s) {  // monotone map of fp32 order to uint32 order
    const uint32_t b = __float_as_uint(s);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Block-wide exclusive scan of one int per thread (NT threads).
template <int NT = kThreads>
__device__ int scan_excl(int v, int *total, int *warp_sums) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    constexpr int kWarps = NT / 32;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int s = lane < kWarps ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        if (lane < kWarps) warp_sums[lane] = s;
    }
    __syncthreads();
    const int r = (warp > 0 ? warp_sums[warp - 1] : 0) + x - v;
    *total = warp_sums[kWarps - 1];
    __syncthreads();
    return r;
}

// One radix pass: histogram of digit (key >> shift) & 255 over the keys that match `prefix` above
// the digit, then the digit holding the `rem`-th key counted from the top (descending = true) or
// from the bottom. Updates prefix and rem; returns the count of keys equal to the final prefix
// in the last pass (the bin size).
struct RadixState {
    uint32_t prefix;
    int rem;
    int bin;
};

// One warp finds the bin of the rem-th key of a 256-bin histogram, counted from the top bin
// (descending) or the bottom, and publishes the new prefix, remainder and bin size.
template <bool kDescending>
__device__ __forceinline__ void radix_find(int shift, uint32_t mask_hi, const RadixState &st, const unsigned *hist,
                                           RadixState *shared_st) {
    const int lane = threadIdx.x & 31;
    {
        // Lane l holds 8 consecutive bins in scan order (from the top bin when descending).
        unsigned c[8], s = 0;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int bin = kDescending ? 255 - (lane * 8 + k) : lane * 8 + k;
            c[k] = hist[bin];
            s += c[k];
        }
        unsigned incl = s;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned y = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += y;
        }
        const unsigned excl = incl - s;
        const bool hit = excl < (unsigned)st.rem && (unsigned)st.rem <= incl;
        const unsigned ballot = __ballot_sync(0xffffffffu, hit);
        if (lane == __ffs(ballot) - 1) {
            unsigned cum = excl;
            for (int k = 0; k < 8; ++k) {
                if (cum + c[k] >= (unsigned)st.rem) {
                    const int bin = kDescending ? 255 - (lane * 8 + k) : lane * 8 + k;
                    shared_st->prefix = (st.prefix & mask_hi) | ((uint32_t)bin << shift);
                    shared_st->rem = st.rem - (int)cum;
                    shared_st->bin = (int)c[k];
                    break;
                }
                cum += c[k];
            }
        }
    }
}

template <bool kDescending, int NT = kThreads, typename KeyFn>
__device__ void radix_pass(int shift, int lo, int hi, KeyFn key_of, RadixState &st, unsigned *hist,
                           RadixState *shared_st) {
    const int tid = threadIdx.x, warp = tid >> 5;
    for (int i = tid; i < 256; i += NT) hist[i] = 0u;
    __syncthreads();
    const uint32_t mask_hi = shift == 24 ? 0u : (0xffffffffu << (shift + 8));
    for (int j = lo + tid; j < hi; j += NT) {
        bool valid;
        const uint32_t k = key_of(j, valid);
        if (valid && (k & mask_hi) == (st.prefix & mask_hi)) atomicAdd(&hist[(k >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (warp == 0) radix_find<kDescending>(shift, mask_hi, st, hist, shared_st);
    __syncthreads();
    st = *shared_st;
}

// Two selects over the same keys in one sweep per digit: `lo_st` counts from the bottom (the
// rem-th smallest key), `hi_st` from the top, each with its own histogram; warp 0 and warp 1 find
// their bins at the same time.
template <int NT, typename KeyFn>
__device__ void radix_pass_both(int shift, int n, KeyFn key_of, RadixState &lo_st, RadixState &hi_st,
                                unsigned *hist_lo, unsigned *hist_hi, RadixState *shared_lo, RadixState *shared_hi) {
    const int tid = threadIdx.x, warp = tid >> 5;
    for (int i = tid; i < 256; i += NT) hist_lo[i] = hist_hi[i] = 0u;
    __syncthreads();
    const uint32_t mask_hi = shift == 24 ? 0u : (0xffffffffu << (shift + 8));
    for (int j = tid; j < n; j += NT) {
        bool valid;
        const uint32_t k = key_of(j, valid);
        if (!valid) continue;
        const unsigned bin = (k >> shift) & 255u;
        if ((k & mask_hi) == (lo_st.prefix & mask_hi)) atomicAdd(&hist_lo[bin], 1u);
        if ((k & mask_hi) == (hi_st.prefix & mask_hi)) atomicAdd(&hist_hi[bin], 1u);
    }
    __syncthreads();
    if (warp == 0) radix_find<false>(shift, mask_hi, lo_st, hist_lo, shared_lo);
    if (warp == 1) radix_find<true>(shift, mask_hi, hi_st, hist_hi, shared_hi);
    __syncthreads();
    lo_st = *shared_lo;
    hi_st = *shared_hi;
}

template <typename T, int D, bool kPaged, bool kWide>
__global__ void __launch_bounds__(kThreads, kWide ? BulkRing<T, D>::kCtasPerSm : NarrowRing::kCtasPerSm)
evict_kernel(const EvictParams p) {
    constexpr int kVecPerRow = D * (int)sizeof(T) / 16;  // 16-byte vectors in one K (or V) row
    using BR = BulkRing<T, D>;
    constexpr int kStageVecs = NarrowRing::kVecs;
    constexpr int kPipe = kWide ? BR::kDepth : NarrowRing::kDepth;
    constexpr int kRows = kWide ? BR::kRows : kThreads * kStageVecs / (2 * kVecPerRow);
    __shared__ int32_t src_list[kSegment];
    __shared__ uint4 ring_static[kWide ? 1 : kPipe][kWide ? 1 : kThreads * kStageVecs];  // narrow ring
    extern __shared__ uint4 ring_dyn[];                                                  // wide ring
    __shared__ uint64_t full[kWide ? kPipe : 1];  // wide: the stage's bulk loads have landed
    __shared__ float stage_sc[kPipe][kRows];
    __shared__ int32_t stage_ps[kPipe][kRows];
    __shared__ unsigned hist[256];
    __shared__ int warp_sums[32];
    __shared__ RadixState shared_st;

    const int tid = threadIdx.x;
    const UnitIdx ui = unit_of(blockIdx.x, p.B, p.L, p.Hkv, p.layer_begin);
    ptx::grid_dependency_wait();  // a programmatic dependent of the previous kernel: wait for its writes
    const int32_t n = p.len[ui.cache_unit];
    const Split sp = split_of(p, ui);
    const int32_t bud = sp.bud, M = sp.M, T_ = sp.T, N = sp.N;
    if (bud < 0 || N < 0 || M < 0) {
        if (tid == 0) raise_status(p.status, VOXZIP_DEV_BAD_BUDGET);
        return;
    }
    if (n <= bud) return;
    if (n > p.C) {
        if (tid == 0) raise_status(p.status, VOXZIP_DEV_CAPACITY);
        return;
    }
    float *sc = p.score + ui.cache_unit * p.C;
    int32_t *ps = p.pos + ui.cache_unit * p.C;
    if constexpr (kWide) {
        if (tid == 0) {
            for (int s = 0; s < kPipe; ++s) ptx::mbar_init(&full[s], 1);
            ptx::fence_mbar_init();
        }
        // (the next block-wide barrier, in the selection or else in the compaction's first scan,
        // orders the initialisation before any use)
    }
    // K/V rows: the unit's slots (dense), or pool rows through the page table (paged).
    uint4 *kc = reinterpret_cast<uint4 *>(static_cast<T *>(p.k_cache) + (kPaged ? 0 : ui.cache_unit * p.C * D));
    uint4 *vc = reinterpret_cast<uint4 *>(static_cast<T *>(p.v_cache) + (kPaged ? 0 : ui.cache_unit * p.C * D));
    auto slot_row = [&](int32_t slot) -> int64_t { return kPaged ? paged_row(p.pv, ui.cache_unit, slot) : slot; };
    auto row_ok = [&](int64_t r) { return !kPaged || (r >= 0 && r < p.rows); };  // checked builds only
    (void)row_ok;
    const int32_t c_end = n - M;  // history candidates are slots [T, c_end)

    // Eq. 9: the N-th best history score, then (only if needed) the position cut among its ties.
    uint32_t thr = 0u, pos_thr = 0xffffffffu;
    bool all_ties = true;
    if (N > 0) {
        RadixState st{0u, N, 0};
        auto skey = [&](int j, bool &valid) {
            valid = true;
            return score_key(sc[j]);
        };
        for (int shift = 24; shift >= 0; shift -= 8) radix_pass<true>(shift, T_, c_end, skey, st, hist, &shared_st);
        thr = st.prefix;
        all_ties = st.rem == st.bin;  // every candidate scoring exactly thr is kept
        if (!all_ties) {
            RadixState sp{0u, st.rem, 0};
            auto pkey = [&](int j, bool &valid) {
                valid = score_key(sc[j]) == thr;
                return (uint32_t)ps[j];
            };
            for (int shift = 24; shift >= 0; shift -= 8)
                radix_pass<false>(shift, T_, c_end, pkey, sp, hist, &shared_st);
            pos_thr = sp.prefix;
        }
    }

    // Eq. 7-8: ordered, in-place compaction of the kept rows.
    int cursor = 0, rank0 = 0;
    bool ok = true;          // wide: every mbarrier wait succeeded
    uint32_t g_sub = 0;      // wide: sub-chunks of earlier segments (stage and phase of the next one)
    uint32_t g_loaded = 0;   // wide: sub-chunks whose loads were issued
    uint32_t g_stored = 0;   // wide: sub-chunks whose loads were seen to land
    while (cursor < n) {
        int seg = 0;
        while (cursor < n && seg + kThreads <= kSegment) {
            const int j = cursor + tid;
            bool keep = false;
            if (j < n) {
                if (j < T_ || j >= c_end) {
                    keep = true;
                } else if (N > 0) {
                    const uint32_t k = score_key(sc[j]);
                    keep = k > thr || (k == thr && (all_ties || (uint32_t)ps[j] <= pos_thr));
                }
            }
            int total;
            const int r = scan_excl(keep ? 1 : 0, &total, warp_sums);
            if (keep) src_list[seg + r] = j;
            seg += total;
            cursor += kThreads;
        }
        __syncthreads();

        // Move ranks [rank0, rank0 + seg) in sub-chunks of kRows through the ring.
        const int nsub = (seg + kRows - 1) / kRows;
        if constexpr (kWide) {
            // One warp: lane l owns row l of every 32-row sub-chunk. Kept rows with consecutive
            // source slots form runs (split at page boundaries when paged); each run of K (and of V)
            // comes in by one bulk copy counted on the stage's mbarrier. The rows that move form a
            // suffix (once an evicted slot precedes a row, one precedes every later row) with
            // consecutive destinations, so a sub-chunk's moving rows go out by one bulk copy of K
            // and one of V (two each when they cross a page boundary). Loads run kAhead sub-chunks
            // ahead of stores, and a stage is reloaded only after the store that read it has read
            // it. Score and position travel by 4-byte cp.async and plain stores.
            constexpr int kAhead = kPipe - 2;
            constexpr uint32_t RB = BR::kRowBytes;
            if (tid < 32 && ok) {
                const int lane = tid;
                for (int it = 0; it < nsub + kAhead; ++it) {
                    const int sub = it - kAhead;
                    if (sub >= 0) {
                        const uint32_t gs = g_sub + (uint32_t)sub;
                        const int st = (int)(gs % kPipe);
                        if (!__all_sync(0xffffffffu, ptx::mbar_wait_bounded(&full[st], (gs / kPipe) & 1, kEvictWaitLimit))) {
                            ok = false;
                            break;
                        }
                        g_stored = gs + 1;
                        asm volatile("cp.async.wait_group %0;" ::"n"(kAhead - 1) : "memory");
                        const int row = sub * kRows + lane;
                        const int dst = rank0 + row;
                        const bool mv = row < seg && src_list[row] != dst &&
                                        VOXZIP_IN_RANGE(p.status, dst < n && row_ok(slot_row(dst)));
                        // The moving rows are a suffix of the sub-chunk with consecutive destinations;
                        // paged, a page boundary splits them in two.
                        const bool prev_mv = __shfl_up_sync(0xffffffffu, mv ? 1 : 0, 1) != 0;  // every lane
                        const bool piece = mv && (lane == 0 || !prev_mv || (kPaged && (dst & (kPageTokens - 1)) == 0));
                        const unsigned movers = __ballot_sync(0xffffffffu, mv);
                        const unsigned pieces = __ballot_sync(0xffffffffu, piece);
                        if (mv) {
                            sc[dst] = stage_sc[st][lane];
                            ps[dst] = stage_ps[st][lane];
                        }
                        if (piece) {
                            const unsigned after = lane == 31 ? 0u : (0xffffffffu << (lane + 1));
                            const unsigned stop = (pieces | ~movers) & after;
                            const uint32_t bytes = (uint32_t)((stop ? __ffs(stop) - 1 : 32) - lane) * RB;
                            uint8_t *stage = reinterpret_cast<uint8_t *>(ring_dyn) + st * BR::kStageBytes;
                            bulk_store(kc + slot_row(dst) * kVecPerRow, stage + lane * RB, bytes);
                            bulk_store(vc + slot_row(dst) * kVecPerRow, stage + (kRows + lane) * RB, bytes);
                        }
                        bulk_commit();
                    }
                    if (it < nsub) {
                        const uint32_t gl = g_sub + (uint32_t)it;
                        const int st = (int)(gl % kPipe);
                        bulk_wait_read<kPipe - kAhead>();  // the store that last read this stage is done reading
                        const int row = it * kRows + lane;
                        const int src = row < seg ? src_list[row] : -2;
                        const bool mv = row < seg && src != rank0 + row &&
                                        VOXZIP_IN_RANGE(p.status, src >= 0 && src < n && row_ok(slot_row(src)));
                        const int prev_src = __shfl_up_sync(0xffffffffu, src, 1);
                        const bool prev_mv = __shfl_up_sync(0xffffffffu, mv ? 1 : 0, 1) != 0;
                        const bool start = mv && (lane == 0 || !prev_mv || src != prev_src + 1 ||
                                                  (kPaged && (src & (kPageTokens - 1)) == 0));
                        const unsigned movers = __ballot_sync(0xffffffffu, mv);
                        const unsigned starts = __ballot_sync(0xffffffffu, start);
                        if (lane == 0) ptx::mbar_arrive_expect_tx(&full[st], (uint32_t)__popc(movers) * 2u * RB);
                        __syncwarp();
                        if (start) {  // this lane's run: up to the next run start or the next row that stays
                            const unsigned after = lane == 31 ? 0u : (0xffffffffu << (lane + 1));
                            const unsigned stop = (starts | ~movers) & after;
                            const int len = (stop ? __ffs(stop) - 1 : 32) - lane;
                            uint8_t *stage = reinterpret_cast<uint8_t *>(ring_dyn) + st * BR::kStageBytes;
                            bulk_load(stage + lane * RB, kc + slot_row(src) * kVecPerRow, (uint32_t)len * RB, &full[st]);
                            bulk_load(stage + (kRows + lane) * RB, vc + slot_row(src) * kVecPerRow, (uint32_t)len * RB,
                                      &full[st]);
                        }
                        if (mv) {
                            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_u32(&stage_sc[st][lane])),
                                         "l"(sc + src)
                                         : "memory");
                            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_u32(&stage_ps[st][lane])),
                                         "l"(ps + src)
                                         : "memory");
                        }
                        g_loaded = gl + 1;
                    }
                    // One 4-byte copy group per iteration (empty in the drain), so that the group of
                    // the sub-chunk stored next is always the kAhead-th most recent.
                    asm volatile("cp.async.commit_group;" ::: "memory");
                }
                bulk_wait_read<0>();  // the next segment may refill every stage
                asm volatile("cp.async.wait_all;" ::: "memory");
            }
            g_sub += (uint32_t)nsub;
            __syncthreads();  // src_list is free for the next segment
        } else {
        auto load_sub = [&](int sub) {
            const int st = sub % kPipe;
#pragma unroll
            for (int k = 0; k < kStageVecs; ++k) {
                const int v = tid + k * kThreads;
                const int row = sub * kRows + v / (2 * kVecPerRow), w = v % (2 * kVecPerRow);
                if (row < seg) {
                    const int src = src_list[row];
                    if (src != rank0 + row && VOXZIP_IN_RANGE(p.status, src >= 0 && src < n && row_ok(slot_row(src)))) {
                        const uint4 *from = (w < kVecPerRow ? kc : vc) + slot_row(src) * kVecPerRow + (w % kVecPerRow);
                        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                                         (uint32_t)__cvta_generic_to_shared(&ring_static[st][v])),
                                     "l"(from)
                                     : "memory");
                    }
                }
            }
            const int row = sub * kRows + tid;
            if (tid < kRows && row < seg) {
                const int src = src_list[row];
                if (src != rank0 + row) {
                    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                                     (uint32_t)__cvta_generic_to_shared(&stage_sc[st][tid])),
                                 "l"(sc + src)
                                 : "memory");
                    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                                     (uint32_t)__cvta_generic_to_shared(&stage_ps[st][tid])),
                                 "l"(ps + src)
                                 : "memory");
                }
            }
        };
        auto store_sub = [&](int sub) {
            const int st = sub % kPipe;
#pragma unroll
            for (int k = 0; k < kStageVecs; ++k) {
                const int v = tid + k * kThreads;
                const int row = sub * kRows + v / (2 * kVecPerRow), w = v % (2 * kVecPerRow);
                if (row < seg) {
                    const int dst = rank0 + row;
                    if (src_list[row] != dst && VOXZIP_IN_RANGE(p.status, dst < n && row_ok(slot_row(dst)))) {
                        uint4 *to = w < kVecPerRow ? kc : vc;
                        to[slot_row(dst) * kVecPerRow + (w % kVecPerRow)] = ring_static[st][v];
                    }
                }
            }
            const int row = sub * kRows + tid;
            if (tid < kRows && row < seg) {
                const int dst = rank0 + row;
                if (src_list[row] != dst) {
                    sc[dst] = stage_sc[st][tid];
                    ps[dst] = stage_ps[st][tid];
                }
            }
        };
        for (int it = 0; it < nsub + kPipe - 1; ++it) {
            if (it < nsub) load_sub(it);
            asm volatile("cp.async.commit_group;" ::: "memory");
            const int sub = it - (kPipe - 1);
            if (sub >= 0) {
                asm volatile("cp.async.wait_group %0;" ::"n"(kPipe - 1) : "memory");
                __syncthreads();  // every thread's loads of `sub` have landed
                store_sub(sub);
                __syncthreads();  // its stage is drained before the next refill
            }
        }
        }
        rank0 += seg;
    }
    if constexpr (kWide) {
        if (tid < 32) {
            if (!ok) {  // a wait gave up: let the loads still in flight land (bounded) before leaving
                raise_status(p.status, VOXZIP_DEV_TIMEOUT);
                for (uint32_t g = g_stored; g < g_loaded; ++g)
                    (void)ptx::mbar_wait_bounded(&full[g % kPipe], (g / kPipe) & 1, kEvictWaitLimit);
                asm volatile("cp.async.wait_all;" ::: "memory");
            }
            bulk_wait_all();  // this lane's bulk stores are complete
        }
    }
    if (tid == 0) p.len[ui.cache_unit] = rank0;  // == budget
    if constexpr (kPaged) {  // pages past the one holding slot bud go back to the pool
        __syncthreads();
        if (tid < 32) return_pages_warp(p.pv, ui.cache_unit, bud / kPageTokens + 1, n / kPageTokens + 1);
    }
}

template <typename T, int D, bool kPaged, int NT>
__global__ void __launch_bounds__(NT, FillShape<NT>::kCtasPerSm) evict_fill_kernel(const EvictParams p) {
    constexpr int kVecPerRow = D * (int)sizeof(T) / 16;
    __shared__ int32_t holes[kSegment];
    __shared__ int32_t movers[kSegment];
    __shared__ unsigned hist[256], hist2[256];
    __shared__ int warp_sums[32];
    __shared__ RadixState shared_st, shared_st2;
    __shared__ int resume_at;
    const int tid = threadIdx.x;
    const UnitIdx ui = unit_of(blockIdx.x, p.B, p.L, p.Hkv, p.layer_begin);
    ptx::grid_dependency_wait();  // a programmatic dependent of the previous kernel: wait for its writes
    const int32_t n = p.len[ui.cache_unit];
    const Split sp = split_of(p, ui);
    const int32_t bud = sp.bud, M = sp.M, T_ = sp.T, N = sp.N;
    if (bud < 0 || N < 0 || M < 0) {
        if (tid == 0) raise_status(p.status, VOXZIP_DEV_BAD_BUDGET);
        return;
    }
    if (n <= bud) return;
    if (n > p.C) {
        if (tid == 0) raise_status(p.status, VOXZIP_DEV_CAPACITY);
        return;
    }
    float *sc = p.score + ui.cache_unit * p.C;
    int32_t *ps = p.pos + ui.cache_unit * p.C;
    uint4 *kc = reinterpret_cast<uint4 *>(static_cast<T *>(p.k_cache) + (kPaged ? 0 : ui.cache_unit * p.C * D));
    uint4 *vc = reinterpret_cast<uint4 *>(static_cast<T *>(p.v_cache) + (kPaged ? 0 : ui.cache_unit * p.C * D));
    auto slot_row = [&](int32_t slot) -> int64_t { return kPaged ? paged_row(p.pv, ui.cache_unit, slot) : slot; };
    auto row_ok = [&](int64_t r) { return !kPaged || (r >= 0 && r < p.rows); };  // checked builds only
    (void)row_ok;

    // Sinks: the T lowest positions (<= p_lo); recent window: the M highest (>= p_hi). Positions
    // of a unit are unique, so each select cuts exactly.
    auto pkey = [&](int j, bool &valid) {
        valid = true;
        return (uint32_t)ps[j];
    };
    // The bits any position sets: radix passes over high digits that are zero in every position
    // (positions below 2^16, say) decide nothing and are skipped.
    uint32_t any = 0u;
    for (int j = tid; j < n; j += NT) any |= (uint32_t)ps[j];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) any |= __shfl_xor_sync(0xffffffffu, any, o);
    if ((tid & 31) == 0) warp_sums[tid >> 5] = (int)any;
    __syncthreads();
    any = 0u;
#pragma unroll
    for (int w = 0; w < NT / 32; ++w) any |= (uint32_t)warp_sums[w];
    __syncthreads();
    const int top_shift = any >> 24 ? 24 : any >> 16 ? 16 : any >> 8 ? 8 : 0;
    uint32_t p_lo = 0u, p_hi = 0xffffffffu;
    if (T_ > 0 && M > 0) {  // both cuts in one sweep per digit
        RadixState lo{0u, T_, 0}, hi{0u, M, 0};
        for (int shift = top_shift; shift >= 0; shift -= 8)
            radix_pass_both<NT>(shift, n, pkey, lo, hi, hist, hist2, &shared_st, &shared_st2);
        p_lo = lo.prefix;
        p_hi = hi.prefix;
    } else if (T_ > 0) {
        RadixState st{0u, T_, 0};
        for (int shift = top_shift; shift >= 0; shift -= 8)
            radix_pass<false, NT>(shift, 0, n, pkey, st, hist, &shared_st);
        p_lo = st.prefix;
    } else if (M > 0) {
        RadixState st{0u, M, 0};
        for (int shift = top_shift; shift >= 0; shift -= 8)
            radix_pass<true, NT>(shift, 0, n, pkey, st, hist, &shared_st);
        p_hi = st.prefix;
    }
    auto middle = [&](uint32_t q) { return !(T_ > 0 && q <= p_lo) && !(M > 0 && q >= p_hi); };

    // Eq. 9 over the rest, exactly as in the ordered eviction.
    uint32_t thr = 0u, pos_thr = 0xffffffffu;
    bool all_ties = true;
    if (N > 0) {
        RadixState st{0u, N, 0};
        auto skey = [&](int j, bool &valid) {
            valid = middle((uint32_t)ps[j]);
            return score_key(sc[j]);
        };
        for (int shift = 24; shift >= 0; shift -= 8) radix_pass<true, NT>(shift, 0, n, skey, st, hist, &shared_st);
        thr = st.prefix;
        all_ties = st.rem == st.bin;
        if (!all_ties) {
            RadixState sq{0u, st.rem, 0};
            auto tkey = [&](int j, bool &valid) {
                const uint32_t q = (uint32_t)ps[j];
                valid = middle(q) && score_key(sc[j]) == thr;
                return q;
            };
            for (int shift = top_shift; shift >= 0; shift -= 8)
                radix_pass<false, NT>(shift, 0, n, tkey, sq, hist, &shared_st);
            pos_thr = sq.prefix;
        }
    }
    auto kept = [&](int j) {
        const uint32_t q = (uint32_t)ps[j];
        if (!middle(q)) return true;
        if (N == 0) return false;
        const uint32_t k = score_key(sc[j]);
        return k > thr || (k == thr && (all_ties || q <= pos_thr));
    };

    // Pair the evicted slots below the budget with the kept slots at or above it, both in ascending
    // slot order. Sources lie at or above the budget and destinations below it, so a thread loads all
    // of its vectors of a round (kBatch of them) before it stores any.
    auto move_pairs = [&](int pairs) {
        constexpr int kBatch = 4;
        const int total = pairs * 2 * kVecPerRow;
        for (int v0 = tid; v0 < total; v0 += kBatch * NT) {
            uint4 x[kBatch];
            bool go[kBatch];
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int v = v0 + u * NT;
                const int r = v / (2 * kVecPerRow), w = v % (2 * kVecPerRow);
                go[u] = v < total && VOXZIP_IN_RANGE(p.status, holes[r] >= 0 && holes[r] < bud && movers[r] >= bud &&
                                                                   movers[r] < n && row_ok(slot_row(holes[r])) &&
                                                                   row_ok(slot_row(movers[r])));
                if (go[u]) x[u] = (w < kVecPerRow ? kc : vc)[slot_row(movers[r]) * kVecPerRow + w % kVecPerRow];
            }
#pragma unroll
            for (int u = 0; u < kBatch; ++u) {
                const int v = v0 + u * NT;
                const int r = v / (2 * kVecPerRow), w = v % (2 * kVecPerRow);
                if (go[u]) (w < kVecPerRow ? kc : vc)[slot_row(holes[r]) * kVecPerRow + w % kVecPerRow] = x[u];
            }
        }
        for (int r = tid; r < pairs; r += NT) {
            sc[holes[r]] = sc[movers[r]];
            ps[holes[r]] = ps[movers[r]];
        }
    };
    // One pass when it fits: each thread classifies a contiguous run of at most 64 slots into a bit
    // mask, and one block scan per region gives every hole and every mover its rank.
    {
        const int ch = (bud + NT - 1) / NT, cm = (n - bud + NT - 1) / NT;
        int fast = ch <= 64 && cm <= 64;
        int nh = 0, nm = 0;
        if (fast) {
            uint64_t hmask = 0, mmask = 0;
            const int h0 = tid * ch, m0 = bud + tid * cm;
            for (int i = 0; i < ch && h0 + i < bud; ++i)
                if (!kept(h0 + i)) hmask |= 1ull << i;
            for (int i = 0; i < cm && m0 + i < n; ++i)
                if (kept(m0 + i)) mmask |= 1ull << i;
            const int hr = scan_excl<NT>(__popcll(hmask), &nh, warp_sums);
            const int mr = scan_excl<NT>(__popcll(mmask), &nm, warp_sums);
            fast = nh <= kSegment && nm <= kSegment;  // the same decision in every thread
            if (fast) {
                for (int k = hr; hmask; hmask &= hmask - 1) holes[k++] = h0 + __ffsll((long long)hmask) - 1;
                for (int k = mr; mmask; mmask &= mmask - 1) movers[k++] = m0 + __ffsll((long long)mmask) - 1;
            }
            __syncthreads();
        }
        if (fast) {
            // equal when positions are unique (then exactly `bud` rows are kept)
            if (nh != nm && tid == 0) raise_status(p.status, VOXZIP_DEV_BAD_POSITIONS);
            move_pairs(min(nh, nm));
            __syncthreads();
            if (tid == 0) p.len[ui.cache_unit] = bud;
            if constexpr (kPaged) {  // pages past the one holding slot bud go back to the pool
                if (tid < 32) return_pages_warp(p.pv, ui.cache_unit, bud / kPageTokens + 1, n / kPageTokens + 1);
            }
            return;
        }
    }
    // Otherwise a segment of up to kSegment pairs at a time.
    int hcur = 0, mcur = bud;
    while (true) {
        int nh = 0;
        while (hcur < bud && nh + NT <= kSegment) {
            const int j = hcur + tid;
            const bool hole = j < bud && !kept(j);
            int total;
            const int r = scan_excl<NT>(hole ? 1 : 0, &total, warp_sums);
            if (hole) holes[nh + r] = j;
            nh += total;
            hcur += NT;
        }
        if (nh == 0) break;
        int nm = 0;
        while (nm < nh && mcur < n) {
            const int j = mcur + tid;
            const bool mv = j < n && kept(j);
            int total;
            const int r = scan_excl<NT>(mv ? 1 : 0, &total, warp_sums);
            if (mv && nm + r < nh) movers[nm + r] = j;
            if (nm + total <= nh) {
                nm += total;
                mcur += NT;
            } else {  // this step holds more movers than holes are left: resume after the last one taken
                if (mv && nm + r == nh - 1) resume_at = j + 1;
                __syncthreads();
                mcur = resume_at;
                nm = nh;
                __syncthreads();
            }
        }
        __syncthreads();
        const int pairs = min(nh, nm);  // equal when positions are unique (then exactly `bud` rows are kept)
        if (pairs < nh && tid == 0) raise_status(p.status, VOXZIP_DEV_BAD_POSITIONS);
        move_pairs(pairs);
        __syncthreads();
        if (pairs < nh) break;
    }
    // Every kept row at or above the budget has found a hole; one left over means more than
    // `bud` rows were kept (repeated positions).
    int extra = 0;
    for (int j = mcur + tid; j < n; j += NT) extra |= kept(j) ? 1 : 0;
    if (__syncthreads_or(extra) && tid == 0) raise_status(p.status, VOXZIP_DEV_BAD_POSITIONS);
    if (tid == 0) p.len[ui.cache_unit] = bud;
    if constexpr (kPaged) {  // pages past the one holding slot bud go back to the pool
        __syncthreads();
        if (tid < 32) return_pages_warp(p.pv, ui.cache_unit, bud / kPageTokens + 1, n / kPageTokens + 1);
    }
}

template <typename T, int D, bool kPaged = false>
cudaError_t launch_t(const EvictParams &prm, int units, bool fill, cudaStream_t stream) {
    // A programmatic dependent of the previous kernel (the decode step): the kernels wait for it
    // before their first read, and a launch without that attribute is the fallback.
    const bool wide = !fill && units <= BulkRing<T, D>::kCtasPerSm * sm_count();
    const bool fill_wide = fill && units <= FillShape<kThreads>::kCtasPerSm * sm_count();
    void (*kern)(EvictParams) = fill ? (fill_wide ? evict_fill_kernel<T, D, kPaged, kThreads>
                                                  : evict_fill_kernel<T, D, kPaged, 192>)
                                     : (wide ? evict_kernel<T, D, kPaged, true> : evict_kernel<T, D, kPaged, false>);
    if (wide) {  // above the default 48 KB of dynamic shared memory: opt in once
        static bool configured = false;
        if (!configured) {
            const cudaError_t e = cudaFuncSetAttribute(evict_kernel<T, D, kPaged, true>,
                                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                       (int)BulkRing<T, D>::kBytes);
            if (e != cudaSuccess) return e;
            configured = true;
        }
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)units, 1, 1);
    cfg.blockDim = dim3(fill && !fill_wide ? 192 : kThreads, 1, 1);
    cfg.dynamicSmemBytes = wide ? BulkRing<T, D>::kBytes : 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t err = cudaLaunchKernelEx(&cfg, kern, prm);
    if (err == cudaErrorNotSupported || err == cudaErrorInvalidValue) {
        cudaGetLastError();
        cfg.numAttrs = 0;
        err = cudaLaunchKernelEx(&cfg, kern, prm);
    }
    return err;
}

}  // namespace

cudaError_t launch_evict(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count,
                         void *k_cache, void *v_cache, float *score, int32_t *pos, int32_t *len,
                         const int32_t *budget, int32_t sink, float recent_frac, int32_t *status,
                         cudaStream_t stream) {
    voxzip_evict_policy pol{};
    pol.sink = sink;
    pol.recent_frac = recent_frac;
    pol.history = 1;
    pol.budget_stride_b = 1;
    pol.budget_stride_l = 0;
    pol.compaction = VOXZIP_COMPACT_ORDERED;
    return launch_evict_policy(d, layer_begin, layer_count, k_cache, v_cache, score, pos, len, budget, pol, status,
                               stream);
}

cudaError_t launch_evict_policy(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count,
                                void *k_cache, void *v_cache, float *score, int32_t *pos, int32_t *len,
                                const int32_t *budget, const voxzip_evict_policy &pol, int32_t *status,
                                cudaStream_t stream) {
    EvictParams prm;
    prm.k_cache = k_cache; prm.v_cache = v_cache; prm.score = score; prm.pos = pos; prm.len = len;
    prm.budget = budget; prm.status = status;
    prm.B = d.batch; prm.L = d.layers; prm.Hkv = d.kv_heads; prm.C = d.capacity;
    prm.layer_begin = layer_begin; prm.sink = pol.sink; prm.recent_frac = pol.recent_frac;
    prm.budget_stride_b = pol.budget_stride_b; prm.budget_stride_l = pol.budget_stride_l;
    prm.history = pol.history;
    prm.pv = PageView{nullptr, nullptr, nullptr, 0};
    prm.rows = (int64_t)d.batch * d.layers * d.kv_heads * d.capacity;
    const int units = layer_count * d.batch * d.kv_heads;
    const bool bf16 = d.dtype == VOXZIP_BF16, fill = pol.compaction == VOXZIP_COMPACT_FILL;
    if (d.head_dim == 128)
        return bf16 ? launch_t<__nv_bfloat16, 128>(prm, units, fill, stream)
                    : launch_t<float, 128>(prm, units, fill, stream);
    return bf16 ? launch_t<__nv_bfloat16, 64>(prm, units, fill, stream) : launch_t<float, 64>(prm, units, fill, stream);
}

cudaError_t launch_evict_paged(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, int32_t layer_begin,
                               int32_t layer_count, float *score, int32_t *pos, int32_t *len, const int32_t *budget,
                               const voxzip_evict_policy &pol, int32_t *status, cudaStream_t stream) {
    EvictParams prm;
    prm.k_cache = pc.k_pool; prm.v_cache = pc.v_pool; prm.score = score; prm.pos = pos; prm.len = len;
    prm.budget = budget; prm.status = status;
    prm.B = d.batch; prm.L = d.layers; prm.Hkv = d.kv_heads; prm.C = d.capacity;
    prm.layer_begin = layer_begin; prm.sink = pol.sink; prm.recent_frac = pol.recent_frac;
    prm.budget_stride_b = pol.budget_stride_b; prm.budget_stride_l = pol.budget_stride_l;
    prm.history = pol.history;
    prm.pv = PageView{pc.page_table, pc.free_pages, pc.free_count, pc.max_pages};
    prm.rows = (int64_t)pc.pages * kPageTokens;
    const int units = layer_count * d.batch * d.kv_heads;
    const bool bf16 = d.dtype == VOXZIP_BF16, fill = pol.compaction == VOXZIP_COMPACT_FILL;
    if (d.head_dim == 128)
        return bf16 ? launch_t<__nv_bfloat16, 128, true>(prm, units, fill, stream)
                    : launch_t<float, 128, true>(prm, units, fill, stream);
    return bf16 ? launch_t<__nv_bfloat16, 64, true>(prm, units, fill, stream)
                : launch_t<float, 64, true>(prm, units, fill, stream);
}

}  // namespace voxzip
