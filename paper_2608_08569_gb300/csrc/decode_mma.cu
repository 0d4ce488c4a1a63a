// Fast decode step for bf16 caches (head_dim 64 or 128, GQA group <= 16): append (Eq. 1), GQA
// attention (Eq. 2) and the decayed-score update (Eq. 6), reading each cached K and V row once.
//
// Grid: one thread-block cluster of S CTAs per (layer, sequence, kv-head) unit; CTA r owns the
// token range [r*ceil(n/S), (r+1)*ceil(n/S)). Per CTA, one producer warp streams the range's K
// tiles and then its V tiles (64 tokens each) with 2-D tensor-map TMA loads (128-byte swizzle)
// into a shared-memory ring guarded by mbarriers; four consumer warps take 16 tokens of every tile:
//   phase K  S = K_tile Q^T on the tensor cores (mma.sync m16n8k16, tokens as M, the group's
//            query heads as N); scaled logits kept in shared memory; a running per-head maximum
//            and normaliser (online softmax statistics; kept only when S = 1).
//   phase V  p = 2^(logit - max_cta); O^T += V_tile^T P^T on the tensor cores. A CTA that holds the
//            whole unit (S = 1) already has the final statistics: it rewrites the scores tile by
//            tile as gamma * s + sum_h p_h / Z_h. In a cluster p is kept in shared memory instead.
// As each tile issues, the tile one ring-depth ahead is requested into L2 (bulk prefetch), so an
// SM keeps more bytes in flight than its rings hold. Launches are programmatic dependents of the
// previous kernel on the stream: a CTA sets up (barriers, the L2 prefetch of its first tiles)
// while that kernel drains, then waits for it before its first dependent read.
// In a cluster, one exchange through distributed shared memory then gives the unit's per-head
// maximum and normaliser: every CTA rewrites its tokens' scores and combines one slice of the
// G x D outputs from all CTAs' partials. (Exchanging the statistics between the two phases instead
// makes every CTA wait twice for the slowest one of its cluster, which measured slower.)
// The appended row is patched into its tile in shared memory, so no load waits for its store; its
// cache stores go out at that patch, not in the prologue, where they would wait for their loads.
// Paged caches (kPaged): a CTA's range is whole 64-token pages, each tile is loaded from the pool
// row its page-table entry gives, and the CTA that completes a page takes the next one.
#include <cooperative_groups.h>

#include <type_traits>

#include "common.cuh"
#include "paged.cuh"
#include "ptx.cuh"
#include "tmap.cuh"

namespace cg = cooperative_groups;

namespace voxzip {
namespace {

#ifndef VOXZIP_DECODE_WARPS
#define VOXZIP_DECODE_WARPS 4      // consumer warps per CTA (16 tokens of every tile each)
#endif
#ifndef VOXZIP_DECODE_L2_AHEAD
#define VOXZIP_DECODE_L2_AHEAD 1           // tiles past the ring requested into L2 as each tile issues
#endif
#ifndef VOXZIP_DECODE_CTA_FIXED_US
#define VOXZIP_DECODE_CTA_FIXED_US 5.0     // a CTA's fixed latency: first tiles, exit
#endif
#ifndef VOXZIP_DECODE_CLUSTER_FIXED_US
#define VOXZIP_DECODE_CLUSTER_FIXED_US 0.0  // added by the cluster exchange (S > 1)
#endif
#ifndef VOXZIP_DECODE_STAGE_TOKENS_PER_US
#define VOXZIP_DECODE_STAGE_TOKENS_PER_US 20.0  // one CTA's streaming rate per ring stage in flight
#endif
#ifndef VOXZIP_DECODE_SM_TOKENS_PER_US
#define VOXZIP_DECODE_SM_TOKENS_PER_US 90.0     // one SM's share of HBM bandwidth (~46 GB/s of K+V)
#endif
#ifndef VOXZIP_DECODE_GPU_TOKENS_PER_US
#define VOXZIP_DECODE_GPU_TOKENS_PER_US 12000.0  // the whole GPU near HBM peak (~6.1 TB/s of K+V)
#endif

constexpr int kConsumerWarps = VOXZIP_DECODE_WARPS;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kTile = 16 * kConsumerWarps;      // tokens per pipeline stage
constexpr int kBoxCols = 64;                    // bf16 elements per TMA box row (128 bytes)
constexpr int kBoxBytes = kTile * kBoxCols * 2;
constexpr uint32_t kWaitLimit = 1u << 24;
constexpr size_t kMaxSmem = 227 * 1024;
constexpr int kMaxCluster = 16;
static_assert(kTile == kPageTokens, "a paged cache's page is one tile of the ring");

struct MmaParams {
    const __nv_bfloat16 *q, *k_new, *v_new;
    const int32_t *new_pos;
    __nv_bfloat16 *k_cache, *v_cache;
    float *score;
    int32_t *pos, *len;
    __nv_bfloat16 *out;
    int32_t *status;
    int32_t B, L, Hq, Hkv, G, C, layer_begin, chunk_cap, n_hint;
    int64_t rows;  // K / V rows the tensor maps cover (the cache, or the page pools)
    float gamma, scale_log2;
    PageView pv;  // paged instantiations: the pools are k_cache / v_cache
};

template <int D, int NT, int kStages>
struct Layout {
    static constexpr int kHalves = D / 64;
    static constexpr int kGP = 8 * NT;                         // heads padded to the MMA's N
    static constexpr int kStageBytes = kHalves * kBoxBytes;
    static constexpr int kStagesOff = 0;                       // the ring; reused for o_w afterwards
    static constexpr int kRingBytes = kStages * kStageBytes;
    static constexpr int kOStride = D + 4;                     // padded row of the output partials
    static constexpr int kOwBytes = kConsumerWarps * kGP * kOStride * 4;
    static constexpr int kRingAlloc = kRingBytes > kOwBytes ? kRingBytes : (kOwBytes + 1023) / 1024 * 1024;
    static constexpr int kBarOff = kRingAlloc;                 // full[kStages], empty[kStages]
    static constexpr int kPbufOff = kBarOff + 2 * kStages * 8;
    static constexpr int kPbufBytes = kConsumerWarps * 16 * kGP * 2;
    static constexpr int kStatOff = kPbufOff + kPbufBytes;     // m_w, z_w [warps][kGP]; m_cta, z_cta [kGP]; fac [S][kGP]
    static constexpr int kStatFloats = (2 * kConsumerWarps + 2 + kMaxCluster) * kGP;
    static constexpr int kLgOff = kStatOff + kStatFloats * 4;  // logits / p [chunk_cap][kGP] fp32, then old scores
    static size_t bytes(int chunk_cap) {  // + the pool row of each tile (paged)
        return 1024 + (size_t)kLgOff + (size_t)chunk_cap * kGP * 4 + (size_t)chunk_cap * 4 +
               (size_t)(chunk_cap / kTile + 1) * 4;
    }
};

__device__ __forceinline__ uint32_t swz(int row, int chunk) {  // byte offset in a 128B-swizzled box
    return (uint32_t)(row * 128 + ((chunk ^ (row & 7)) << 4));
}

// kCluster: launched in clusters of S > 1 CTAs (else one CTA holds the whole unit).
// kPaged: K/V rows live in page pools (see paged.cuh).
template <int D, int NT, int kStages, bool kCluster, bool kPaged>
__global__ void __launch_bounds__(kThreads)
decode_mma_kernel(const __grid_constant__ CUtensorMap tmk, const __grid_constant__ CUtensorMap tmv,
                  const MmaParams p) {
    using Lay = Layout<D, NT, kStages>;
    constexpr int GP = Lay::kGP;
    constexpr int kHalves = Lay::kHalves;
    constexpr int kKSteps = D / 16;

    cg::cluster_group cluster = cg::this_cluster();
    const int S = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    constexpr bool clustered = kCluster;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, qd = lane & 3;

    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *stages = smem + Lay::kStagesOff;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + Lay::kBarOff);
    uint64_t *empty = full + kStages;
    uint8_t *pbuf = smem + Lay::kPbufOff + warp * 16 * GP * 2;
    float *o_w = reinterpret_cast<float *>(stages);            // [warps][GP][D], valid after the ring drains
    float *o_cta = o_w;                                        // the sum over warps lands in warp 0's slot
    float *m_w = reinterpret_cast<float *>(smem + Lay::kStatOff);
    float *z_w = m_w + kConsumerWarps * GP;
    float *m_cta = z_w + kConsumerWarps * GP;                  // this CTA's per-head maximum (log2 units)
    float *z_cta = m_cta + GP;                                 // and normaliser relative to it
    float *fac = z_cta + GP;                                   // [S][GP]: 2^(m_r - m) / Z; 0 for padding heads
    float *lg = reinterpret_cast<float *>(smem + Lay::kLgOff);
    float *s_old = lg + (size_t)p.chunk_cap * GP;               // [chunk_cap] scores before the step
    int32_t *tile_rows = reinterpret_cast<int32_t *>(s_old + p.chunk_cap);  // [tiles] pool row (paged)

    const UnitIdx ui = unit_of(blockIdx.y, p.B, p.L, p.Hkv, p.layer_begin);
    const int64_t act_row = (int64_t)ui.l_local * p.B + ui.b;
    const int64_t row_base = ui.cache_unit * p.C;
    // While this unit's length is read, pull the first tiles of the range the launch's length hint
    // predicts into L2 (exact when the unit is as long as the hint; otherwise a few wasted KB).
    if (!kPaged && warp == kConsumerWarps && lane == 0) {
        const int est_j0 = rank * ((p.n_hint + S - 1) / S);
        const int rows = min(kStages * kTile, p.C - est_j0);
        if (rows > 0) ptx::prefetch_l2(p.k_cache + (row_base + est_j0) * D, (uint32_t)rows * D * 2);
    }
    // Launched as a programmatic dependent of the previous kernel on the stream, the CTA may start
    // before that kernel ends: everything from here on reads what it wrote (lengths, pages,
    // cache rows, scores, queries), so wait for its completion. (The prefetch above is a hint.)
    ptx::grid_dependency_wait();
    // Paged: before the length is known, the producer reads the page-table entries of the range the
    // launch's length hint predicts and pulls those tiles into L2 (kept when the prediction holds).
    int est_j0 = -1, est_tiles = 0;
    if constexpr (kPaged) {
        if (warp == kConsumerWarps) {
            const int est_chunk = ((p.n_hint + S - 1) / S + kTile - 1) / kTile * kTile;
            est_j0 = rank * est_chunk;
            est_tiles = max(0, min(est_chunk, p.n_hint - est_j0) + kTile - 1) / kTile;
            est_tiles = min(est_tiles, p.pv.max_pages - est_j0 / kTile);
            const int32_t *trow = p.pv.table + ui.cache_unit * p.pv.max_pages + est_j0 / kTile;
            for (int t = lane; t < est_tiles; t += 32) {
                const int32_t page = trow[t];
                tile_rows[t] = page * kTile;
                if (t < kStages && page >= 0)
                    ptx::prefetch_l2(p.k_cache + (int64_t)page * kTile * D, (uint32_t)kTile * D * 2);
            }
        }
    }
    // The queries do not depend on the length: load them first. Q^T is the B operand:
    // b0b1 = Q[head][16ks + 2qd .. +1], b2b3 = Q[head][16ks + 8 + 2qd .. +1].
    uint32_t qb[NT][kKSteps][2];
    if (warp < kConsumerWarps) {
        const __nv_bfloat16 *qg = p.q + (act_row * p.Hq + (int64_t)ui.h * p.G) * D;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            const int head = nt * 8 + g;
#pragma unroll
            for (int ks = 0; ks < kKSteps; ++ks) {
                if (head < p.G) {
                    qb[nt][ks][0] = *reinterpret_cast<const uint32_t *>(qg + head * D + ks * 16 + 2 * qd);
                    qb[nt][ks][1] = *reinterpret_cast<const uint32_t *>(qg + head * D + ks * 16 + 8 + 2 * qd);
                } else {
                    qb[nt][ks][0] = 0u;
                    qb[nt][ks][1] = 0u;
                }
            }
        }
    }
    const int32_t n_old = p.len[ui.cache_unit];
    const int32_t n = n_old + 1;
    if (n_old < 0 || n > p.C) {  // the same decision in every CTA of the cluster
        if (rank == 0 && tid == 0) raise_status(p.status, VOXZIP_DEV_CAPACITY);
        return;
    }
    int32_t page_new = 0;  // paged: page of the appended row (slot n - 1)
    if constexpr (kPaged) {
        page_new = p.pv.table[ui.cache_unit * p.pv.max_pages + (n_old >> 6)];
        if (page_new < 0) {  // the pool had no page for it: the same decision in every CTA
            if (rank == 0 && tid == 0) raise_status(p.status, VOXZIP_DEV_CAPACITY);
            return;
        }
    }
    const int chunk = kPaged ? ((n + S - 1) / S + kTile - 1) / kTile * kTile : (n + S - 1) / S;
    if (chunk > p.chunk_cap) {
        if (rank == 0 && tid == 0) raise_status(p.status, VOXZIP_DEV_LEN_HINT);
        return;
    }
    const int j0 = min(n, rank * chunk);
    const int cnt = min(n, j0 + chunk) - j0;
    const int ntiles = (cnt + kTile - 1) / kTile;

    // Eq. 1: the appended row is local row jn of the CTA whose range holds slot n-1. The consumer
    // warp that owns that row of its tile loads k_new / v_new into registers here, writes them over
    // the row the TMA brought in, so no load waits for the store, and stores them (with the position)
    // to the cache for later steps when it patches that tile: a store issued here would wait for its
    // load and hold back the barrier before the ring's first load.
    const int jn = n - 1 - j0;
    const bool own_new = jn >= 0 && jn < cnt;
    const int t_new = own_new ? jn / kTile : -1;
    const bool patcher = own_new && warp == (jn % kTile) / 16;
    const uint32_t patch_off = own_new ? (uint32_t)(lane >> 3) * kBoxBytes + swz(jn % kTile, lane & 7) : 0u;
    const int64_t drow = kPaged ? (int64_t)page_new * kPageTokens + (n_old & (kPageTokens - 1)) : row_base + n - 1;
    uint4 kn4 = make_uint4(0u, 0u, 0u, 0u), vn4 = make_uint4(0u, 0u, 0u, 0u);
    int32_t pos_new = 0;
    if (patcher && lane < D / 8) {
        const int64_t src = (act_row * p.Hkv + ui.h) * D + lane * 8;
        kn4 = *reinterpret_cast<const uint4 *>(p.k_new + src);
        vn4 = *reinterpret_cast<const uint4 *>(p.v_new + src);
        if (lane == 0) pos_new = p.new_pos[ui.b];
    }
    bool appended = false;  // the patcher warp has stored the appended row
    auto append = [&]() {
        if (lane < D / 8 && VOXZIP_IN_RANGE(p.status, drow >= 0 && drow < p.rows)) {
            *reinterpret_cast<uint4 *>(p.k_cache + drow * D + lane * 8) = kn4;
            *reinterpret_cast<uint4 *>(p.v_cache + drow * D + lane * 8) = vn4;
        }
        if (lane == 0) p.pos[row_base + n - 1] = pos_new;
        appended = true;
    };
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&full[s], 1);
            ptx::mbar_init(&empty[s], kConsumerWarps);
        }
        ptx::fence_mbar_init();
    }
    // The old scores of this CTA's tokens travel to shared memory while the tiles stream.
    if (warp < kConsumerWarps) {
        const float *src = p.score + row_base + j0;
        for (int i = tid; i < cnt; i += kConsumerWarps * 32)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(ptx::smem_u32(s_old + i)), "l"(src + i)
                         : "memory");
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    __syncthreads();

    bool ok = true;
    if (warp == kConsumerWarps) {
        // ------------------------------------------------------------- producer
        if constexpr (kPaged) {  // the pool row of every tile of the range (j0 is page-aligned)
            if (j0 != est_j0 || ntiles > est_tiles) {
                const int32_t *trow = p.pv.table + ui.cache_unit * p.pv.max_pages + j0 / kTile;
                for (int t = lane; t < ntiles; t += 32) tile_rows[t] = trow[t] * kTile;
            }
            __syncwarp();
        }
        if (lane == 0 && ntiles > 0) {
            ptx::prefetch_tmap(&tmk);
            ptx::prefetch_tmap(&tmv);
            for (int i = 0; i < 2 * ntiles; ++i) {
                const int s = i % kStages, use = i / kStages;
                if (use > 0 && !ptx::mbar_wait_bounded(&empty[s], (use - 1) & 1, kWaitLimit)) {
                    ok = false;
                    break;
                }
                ptx::mbar_arrive_expect_tx(&full[s], Lay::kStageBytes);
                const bool is_k = i < ntiles;
                const int tile = is_k ? i : i - ntiles;
                const int32_t y = kPaged ? tile_rows[tile] : (int32_t)(row_base + j0 + tile * kTile);
                // (a TMA load outside the map reads zeros, so a bad row is only recorded)
                (void)VOXZIP_IN_RANGE(p.status, y >= 0 && (int64_t)y < p.rows);
                uint8_t *dst = stages + s * Lay::kStageBytes;
#pragma unroll
                for (int h = 0; h < kHalves; ++h)
                    ptx::tma_load_2d(dst + h * kBoxBytes, is_k ? &tmk : &tmv, h * kBoxCols, y, &full[s]);
                // L2 look-ahead: the tile that will issue once the ring turns over starts toward L2
                // now. It costs no shared memory and keeps more of the SM's bytes in flight; its TMA
                // load then hits L2.
                if (VOXZIP_DECODE_L2_AHEAD > 0) {
                    const int ia = i + kStages + VOXZIP_DECODE_L2_AHEAD + (kStages == 2 ? 1 : 0) - 1;
                    if (ia < 2 * ntiles) {
                        const bool ak = ia < ntiles;
                        const int at = ak ? ia : ia - ntiles;
                        const int rows = min(kTile, cnt - at * kTile);
                        const int64_t row0 = kPaged ? (int64_t)tile_rows[at] : row_base + j0 + (int64_t)at * kTile;
                        if (rows > 0 && VOXZIP_IN_RANGE(p.status, row0 >= 0 && row0 + rows <= p.rows))
                            ptx::prefetch_l2((ak ? p.k_cache : p.v_cache) + row0 * D, (uint32_t)rows * D * 2);
                    }
                }
            }
        }
        __syncwarp();  // reconverge the producer warp
    } else {
        // ------------------------------------------------------------- consumers
        // Running maximum and normaliser of this thread's logits, per head slot (nt, j).
        float mx[NT][2], zx[NT][2];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mx[nt][0] = mx[nt][1] = -INFINITY, zx[nt][0] = zx[nt][1] = 0.f;
        const int r0 = warp * 16;

        // Phase K: logits of this warp's 16 tokens of every tile.
        for (int t = 0; t < ntiles && ok; ++t) {
            const int s = t % kStages;
            if (!__all_sync(0xffffffffu, ptx::mbar_wait_bounded(&full[s], (t / kStages) & 1, kWaitLimit))) {
                ok = false;
                break;
            }
            const int lt0 = t * kTile + r0;
            if (lt0 < cnt) {
                uint8_t *stage = stages + s * Lay::kStageBytes;
                const bool patch = patcher && t == t_new;
                if (patch) {
                    if (lane < D / 8) *reinterpret_cast<uint4 *>(stage + patch_off) = kn4;
                    append();
                    __syncwarp();
                }
                const uint32_t base = ptx::smem_u32(stage);
                // Two accumulators (even and odd k-steps), summed at the end: two independent mma
                // chains of half the length on the per-tile critical path.
                float acc2[2][NT][4];
#pragma unroll
                for (int c = 0; c < 2; ++c)
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt) acc2[c][nt][0] = acc2[c][nt][1] = acc2[c][nt][2] = acc2[c][nt][3] = 0.f;
                const int arow = r0 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
                for (int h = 0; h < kHalves; ++h) {
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        uint32_t a0, a1, a2, a3;
                        ptx::ldsm_x4(base + h * kBoxBytes + swz(arow, kk * 2 + (lane >> 4)), a0, a1, a2, a3);
#pragma unroll
                        for (int nt = 0; nt < NT; ++nt)
                            ptx::mma_bf16_16816(acc2[kk & 1][nt], a0, a1, a2, a3, qb[nt][h * 4 + kk][0],
                                                qb[nt][h * 4 + kk][1]);
                    }
                }
                float acc[NT][4];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[nt][e] = acc2[0][nt][e] + acc2[1][nt][e];
                // acc[nt][2 * half + j]: token lt0 + g + 8 * half, head nt * 8 + 2 * qd + j.
                const bool va = lt0 + g < cnt, vb = lt0 + g + 8 < cnt;
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    float la[2], lb[2];
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        la[j] = va ? acc[nt][j] * p.scale_log2 : -INFINITY;
                        lb[j] = vb ? acc[nt][2 + j] * p.scale_log2 : -INFINITY;
                        const float m_new = fmaxf(mx[nt][j], fmaxf(la[j], lb[j]));
                        // The normaliser is needed before phase V only without a cluster; keeping it
                        // off the per-tile path otherwise matters when one CTA fills an SM.
                        if (!clustered && m_new != -INFINITY)
                            zx[nt][j] = zx[nt][j] * exp2f(mx[nt][j] - m_new) + exp2f(la[j] - m_new) +
                                        exp2f(lb[j] - m_new);
                        mx[nt][j] = m_new;
                    }
                    if (va) *reinterpret_cast<float2 *>(lg + (lt0 + g) * GP + nt * 8 + 2 * qd) = make_float2(la[0], la[1]);
                    if (vb)
                        *reinterpret_cast<float2 *>(lg + (lt0 + g + 8) * GP + nt * 8 + 2 * qd) = make_float2(lb[0], lb[1]);
                }
                if (patch) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // before the slot's next TMA
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&empty[s]);
        }
        if (patcher && !appended) append();  // phase K ended early (a wait gave up)
        // Per-head statistics of the warp (merge over the 8 lanes that share qd), then of the CTA.
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                float m = mx[nt][j], z = zx[nt][j];
#pragma unroll
                for (int off = 4; off <= 16; off <<= 1) {
                    const float mo = __shfl_xor_sync(0xffffffffu, m, off);
                    const float zo = __shfl_xor_sync(0xffffffffu, z, off);
                    const float mm = fmaxf(m, mo);
                    z = (m == -INFINITY ? 0.f : z * exp2f(m - mm)) + (mo == -INFINITY ? 0.f : zo * exp2f(mo - mm));
                    m = mm;
                }
                if (g == 0) {
                    m_w[warp * GP + nt * 8 + 2 * qd + j] = m;
                    z_w[warp * GP + nt * 8 + 2 * qd + j] = z;
                }
            }
        asm volatile("cp.async.wait_all;" ::: "memory");  // this thread's old scores have landed
        asm volatile("bar.sync 1, %0;" ::"r"(kConsumerWarps * 32) : "memory");
        if (tid < GP) {
            float m = -INFINITY, z = 0.f;
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) m = fmaxf(m, m_w[w * GP + tid]);
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) {
                const float mw = m_w[w * GP + tid];
                if (mw != -INFINITY) z += z_w[w * GP + tid] * exp2f(mw - m);
            }
            m_cta[tid] = m;
            z_cta[tid] = z;
        }
        // A CTA that holds the whole unit has its final statistics now.
        if (!clustered && tid < GP) fac[tid] = tid < p.G ? 1.f / z_cta[tid] : 0.f;
        asm volatile("bar.sync 1, %0;" ::"r"(kConsumerWarps * 32) : "memory");

        // Phase V: probabilities with the CTA maximum, P V on the tensor cores; without a cluster
        // also the score update (Eq. 6), else p is kept for it.
        float oacc[kKSteps][NT][4];
#pragma unroll
        for (int i = 0; i < kKSteps; ++i)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) oacc[i][nt][0] = oacc[i][nt][1] = oacc[i][nt][2] = oacc[i][nt][3] = 0.f;
        float mc[NT][2], rc[NT][2], zv[NT][2];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                mc[nt][j] = m_cta[nt * 8 + 2 * qd + j];
                rc[nt][j] = clustered ? 0.f : fac[nt * 8 + 2 * qd + j];
                zv[nt][j] = 0.f;
            }
        float *sc = p.score + row_base + j0;
        for (int t = 0; t < ntiles && ok; ++t) {
            const int i = ntiles + t, s = i % kStages;
            if (!__all_sync(0xffffffffu, ptx::mbar_wait_bounded(&full[s], (i / kStages) & 1, kWaitLimit))) {
                ok = false;
                break;
            }
            const int lt0 = t * kTile + r0;
            if (lt0 < cnt) {
                uint8_t *stage = stages + s * Lay::kStageBytes;
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    const int lt = lt0 + g + half * 8;
                    const bool valid = lt < cnt;
                    float add = 0.f;
#pragma unroll
                    for (int nt = 0; nt < NT; ++nt) {
                        float p0 = 0.f, p1 = 0.f;
                        if (valid) {
                            const float2 l = *reinterpret_cast<const float2 *>(lg + lt * GP + nt * 8 + 2 * qd);
                            p0 = exp2f(l.x - mc[nt][0]);
                            p1 = exp2f(l.y - mc[nt][1]);
                            if (clustered) {
                                *reinterpret_cast<float2 *>(lg + lt * GP + nt * 8 + 2 * qd) = make_float2(p0, p1);
                                zv[nt][0] += p0;
                                zv[nt][1] += p1;
                            } else {
                                add += p0 * rc[nt][0] + p1 * rc[nt][1];
                            }
                        }
                        *reinterpret_cast<uint32_t *>(pbuf + (g + half * 8) * GP * 2 + (nt * 8 + 2 * qd) * 2) =
                            ptx::pack_bf16(p0, p1);
                    }
                    if (!clustered) {  // Eq. 6: A = gamma * [A, 0] + sum over the heads (a token's four lanes)
                        add += __shfl_xor_sync(0xffffffffu, add, 1);
                        add += __shfl_xor_sync(0xffffffffu, add, 2);
                        if (valid && qd == 0 && VOXZIP_IN_RANGE(p.status, j0 + lt < p.C))
                            sc[lt] = lt == jn ? add : p.gamma * s_old[lt] + add;
                    }
                }
                // Rows past the range may hold anything; zero them so 0 * garbage cannot be NaN.
                bool wrote = false;
                if (lt0 + 16 > cnt) {
                    for (int e = lane; e < 16 * kHalves * 8; e += 32) {
                        const int row = e / (kHalves * 8), rest = e % (kHalves * 8);
                        if (lt0 + row >= cnt)
                            *reinterpret_cast<uint4 *>(stage + (rest >> 3) * kBoxBytes + swz(r0 + row, rest & 7)) =
                                make_uint4(0u, 0u, 0u, 0u);
                    }
                    wrote = true;
                }
                if (patcher && t == t_new) {
                    if (lane < D / 8) *reinterpret_cast<uint4 *>(stage + patch_off) = vn4;
                    wrote = true;
                }
                if (wrote) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                uint32_t pb[NT][2];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
                    ptx::ldsm_x2_t(ptx::smem_u32(pbuf + (lane & 15) * GP * 2 + nt * 16), pb[nt][0], pb[nt][1]);
                const uint32_t base = ptx::smem_u32(stage);
                const int mi = lane >> 3;
                const int vrow = r0 + (lane & 7) + (mi >> 1) * 8;
#pragma unroll
                for (int h = 0; h < kHalves; ++h) {
#pragma unroll
                    for (int mt = 0; mt < 4; ++mt) {
                        uint32_t a0, a1, a2, a3;
                        ptx::ldsm_x4_t(base + h * kBoxBytes + swz(vrow, mt * 2 + (mi & 1)), a0, a1, a2, a3);
#pragma unroll
                        for (int nt = 0; nt < NT; ++nt)
                            ptx::mma_bf16_16816(oacc[h * 4 + mt][nt], a0, a1, a2, a3, pb[nt][0], pb[nt][1]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&empty[s]);
        }
        if (clustered) {  // per-head sums of the warp, then of the CTA (fixed order)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int j = 0; j < 2; ++j) {
                    float v = zv[nt][j];
                    v += __shfl_xor_sync(0xffffffffu, v, 4);
                    v += __shfl_xor_sync(0xffffffffu, v, 8);
                    v += __shfl_xor_sync(0xffffffffu, v, 16);
                    if (g == 0) z_w[warp * GP + nt * 8 + 2 * qd + j] = v;
                }
        }
        // Partial outputs of this warp, then of the CTA (fixed summation order).
        asm volatile("bar.sync 1, %0;" ::"r"(kConsumerWarps * 32) : "memory");  // the ring is drained
        constexpr int OS = Lay::kOStride;
        float *ow = o_w + warp * GP * OS;
#pragma unroll
        for (int i = 0; i < kKSteps; ++i)
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                const int d0 = i * 16 + g, h0 = nt * 8 + 2 * qd;
                ow[h0 * OS + d0] = oacc[i][nt][0];
                ow[(h0 + 1) * OS + d0] = oacc[i][nt][1];
                ow[h0 * OS + d0 + 8] = oacc[i][nt][2];
                ow[(h0 + 1) * OS + d0 + 8] = oacc[i][nt][3];
            }
        asm volatile("bar.sync 1, %0;" ::"r"(kConsumerWarps * 32) : "memory");
        for (int e = tid; e < GP * D; e += kConsumerWarps * 32) {
            const int at = (e / D) * OS + e % D;
            float v = o_w[at];
#pragma unroll
            for (int w = 1; w < kConsumerWarps; ++w) v += o_w[w * GP * OS + at];
            o_cta[at] = v;
        }
        if (clustered && tid < GP) {
            float v = 0.f;
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w) v += z_w[w * GP + tid];
            z_cta[tid] = v;
        }
    }
    if (!ok) raise_status(p.status, VOXZIP_DEV_TIMEOUT);
    ptx::launch_dependents();  // streaming is over: the next launch may begin its prologue
    __syncthreads();
    // CTA r writes slice r of the G x D outputs: the CTAs' partial outputs summed, normalised.
    constexpr int OS = Lay::kOStride;
    const int o_total = p.G * D;
    __nv_bfloat16 *og = p.out + (act_row * p.Hq + (int64_t)ui.h * p.G) * D;
    if (clustered) {
        cluster.sync();  // every CTA's m_cta, z_cta, o_cta are final
        // For a cluster of SS CTAs (a power of two), this thread's share of the slice is at most E
        // elements: all their partials from every CTA are requested before the statistics, so the
        // reads over the cluster take one round trip.
        auto combine = [&](auto ss_tag) {
            constexpr int SS = decltype(ss_tag)::value;
            constexpr int E = (GP * D / SS + kThreads - 1) / kThreads;
            const int per = (o_total + SS - 1) / SS;
            const int lo = rank * per, hi = min(o_total, lo + per);
            float part[E][SS];
#pragma unroll
            for (int e = 0; e < E; ++e) {
                const int i = lo + tid + e * kThreads;
                const int at = i < hi ? (i / D) * OS + i % D : 0;
#pragma unroll
                for (int r = 0; r < SS; ++r) part[e][r] = i < hi ? *cluster.map_shared_rank(&o_cta[at], r) : 0.f;
            }
            // The unit's per-head maximum m and normaliser Z; fac[r][h] = 2^(m_r - m) / Z.
            if (tid < GP) {
                float mr[SS], zr[SS];
#pragma unroll
                for (int r = 0; r < SS; ++r) {
                    mr[r] = *cluster.map_shared_rank(&m_cta[tid], r);
                    zr[r] = *cluster.map_shared_rank(&z_cta[tid], r);
                }
                float m = -INFINITY;
#pragma unroll
                for (int r = 0; r < SS; ++r) m = fmaxf(m, mr[r]);
                float z = 0.f;
#pragma unroll
                for (int r = 0; r < SS; ++r) {
                    mr[r] = mr[r] == -INFINITY ? 0.f : exp2f(mr[r] - m);
                    z += mr[r] * zr[r];
                }
                const float rzv = tid < p.G ? 1.f / z : 0.f;
#pragma unroll
                for (int r = 0; r < SS; ++r) fac[r * GP + tid] = mr[r] * rzv;
            }
            __syncthreads();
#pragma unroll
            for (int e = 0; e < E; ++e) {
                const int i = lo + tid + e * kThreads;
                if (i < hi) {
                    const int h = i / D;
                    float o = 0.f;
#pragma unroll
                    for (int r = 0; r < SS; ++r) o += fac[r * GP + h] * part[e][r];
                    og[i] = __float2bfloat16_rn(o);
                }
            }
        };
        switch (S) {
            case 2: combine(std::integral_constant<int, 2>{}); break;
            case 4: combine(std::integral_constant<int, 4>{}); break;
            case 8: combine(std::integral_constant<int, 8>{}); break;
            default: combine(std::integral_constant<int, 16>{}); break;
        }
        // This CTA is done reading its peers' shared memory (every value read has been used above);
        // they may leave once all have said so. The arrive orders nothing else, so it is relaxed and
        // does not wait for the output stores. The score update below touches only this CTA's own
        // shared memory and global memory.
        asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
        // Eq. 6 for this CTA's tokens: A = gamma * [A, 0] + sum over the group's heads.
        const float *fs = fac + rank * GP;
        float *sc = p.score + row_base + j0;
        for (int i = tid; i < cnt; i += kThreads) {
            float add = 0.f;
            const float4 *pr = reinterpret_cast<const float4 *>(lg + i * GP);
#pragma unroll
            for (int h4 = 0; h4 < GP / 4; ++h4) {
                const float4 v = pr[h4];
                add += v.x * fs[h4 * 4] + v.y * fs[h4 * 4 + 1] + v.z * fs[h4 * 4 + 2] + v.w * fs[h4 * 4 + 3];
            }
            if (VOXZIP_IN_RANGE(p.status, j0 + i < p.C)) sc[i] = i == jn ? add : p.gamma * s_old[i] + add;
        }
    } else {
        for (int i = tid; i < o_total; i += kThreads) {
            const int h = i / D;
            og[i] = __float2bfloat16_rn(o_cta[h * OS + i % D] * fac[h]);
        }
    }
    if (rank == 0 && tid == 0) {
        p.len[ui.cache_unit] = n;
        if constexpr (kPaged) {  // the next append starts a page: take one now
            if ((n & (kPageTokens - 1)) == 0 && (n >> 6) < p.pv.max_pages) {
                int32_t *entry = p.pv.table + ui.cache_unit * p.pv.max_pages + (n >> 6);
                if (*entry < 0) *entry = take_page(p.pv);
            }
        }
    }
    // No CTA leaves while a peer may still read its shared memory.
    if (clustered) asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// ---------------------------------------------------------------- host side
template <int D_, int NT_, int NS_>
struct Tag {
    static constexpr int D = D_, NT = NT_, NS = NS_;
};

// Calls f(Tag<D, NT, NS>{}) for the runtime shape; the kernel is instantiated for D in {64, 128},
// NT in {1, 2} (group <= 8 or <= 16) and a ring of NS in {3, 4, 6, 8} stages.
constexpr int kRingDepths[] = {2, 3, 4, 6, 8};

template <int D, int NT, typename F>
auto dispatch_ns(int NS, F &&f) {
    switch (NS) {
        case 2: return f(Tag<D, NT, 2>{});
        case 4: return f(Tag<D, NT, 4>{});
        case 6: return f(Tag<D, NT, 6>{});
        case 8: return f(Tag<D, NT, 8>{});
        default: return f(Tag<D, NT, 3>{});
    }
}
template <typename F>
auto dispatch(int D, int NT, int NS, F &&f) {
    if (D == 128) return NT == 1 ? dispatch_ns<128, 1>(NS, f) : dispatch_ns<128, 2>(NS, f);
    return NT == 1 ? dispatch_ns<64, 1>(NS, f) : dispatch_ns<64, 2>(NS, f);
}

using KernelFn = void (*)(CUtensorMap, CUtensorMap, MmaParams);

template <typename K>
KernelFn kernel_for(int S, bool paged = false) {
    if (paged)
        return S > 1 ? decode_mma_kernel<K::D, K::NT, K::NS, true, true> : decode_mma_kernel<K::D, K::NT, K::NS, false, true>;
    return S > 1 ? decode_mma_kernel<K::D, K::NT, K::NS, true, false> : decode_mma_kernel<K::D, K::NT, K::NS, false, false>;
}

template <typename K>
bool configure() {  // kernel attributes are per function; set once per process
    static bool done = false;
    if (!done) {
        for (KernelFn kern : {kernel_for<K>(1), kernel_for<K>(2), kernel_for<K>(1, true), kernel_for<K>(2, true)})
            if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMaxSmem) != cudaSuccess ||
                cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess)
                return false;
        done = true;
    }
    return true;
}

// How many clusters of S CTAs, each with `smem` bytes of shared memory, fit the GPU at once.
template <typename K>
int max_active_clusters(int S, size_t smem) {
    if (!configure<K>()) return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)S, 1024, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kernel_for<K>(S), &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n;
}

template <typename K>
cudaError_t launch_t(const CUtensorMap &tmk, const CUtensorMap &tmv, const MmaParams &prm, int S, int units,
                     cudaStream_t stream, bool paged) {
    const KernelFn kern = kernel_for<K>(S, paged);
    if (!configure<K>()) return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)S, (unsigned)units, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = Layout<K::D, K::NT, K::NS>::bytes(prm.chunk_cap);
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // overlap the previous kernel's tail
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    cudaError_t err = cudaLaunchKernelEx(&cfg, kern, tmk, tmv, prm);
    if (err == cudaErrorNotSupported || err == cudaErrorInvalidValue) {  // no programmatic launch here
        cudaGetLastError();
        cfg.numAttrs = 1;
        err = cudaLaunchKernelEx(&cfg, kern, tmk, tmv, prm);
    }
    return err;
}

struct Plan {
    int S, NS, chunk_cap;
};

struct PlanModel {
    double cta_fixed_us, cluster_fixed_us, stage_tokens_per_us, sm_tokens_per_us, gpu_tokens_per_us;
    int stage_cap;  // ring stages beyond this add no streaming rate
};
// A launch whose K and V stream from HBM.
constexpr PlanModel kPlanModel{VOXZIP_DECODE_CTA_FIXED_US, VOXZIP_DECODE_CLUSTER_FIXED_US,
                               VOXZIP_DECODE_STAGE_TOKENS_PER_US, VOXZIP_DECODE_SM_TOKENS_PER_US,
                               VOXZIP_DECODE_GPU_TOKENS_PER_US, 8};
// A launch whose K and V fit comfortably in L2 (at most VOXZIP_DECODE_L2_RESIDENT_MB): in a decode
// loop they stay there from step to step. Fitted to back-to-back graph loops on GB300 (10-min and
// 30-s requests, cluster sizes 1-4, ring depths 2-4): a CTA then consumes ~46 tokens/us whatever
// its ring depth past three stages, an SM ~120, and a cluster exchange adds ~2.6 us.
constexpr PlanModel kPlanModelL2{VOXZIP_DECODE_CTA_FIXED_US, 2.6, 46.0 / 3.0, 120.0, 30000.0, 3};
#ifndef VOXZIP_DECODE_L2_RESIDENT_MB
#define VOXZIP_DECODE_L2_RESIDENT_MB 64.0
#endif

// Chooses the cluster size S and ring depth NS with a time model. For each (S, NS) the CTAs hold
// ceil(nmax/S) tokens (shared memory sized for that, rounded up to 16 tokens); the occupancy API
// gives how many clusters are resident. Every resident cluster takes ceil(units / clusters) units
// in turn; a unit costs a CTA's fixed latency (more with a cluster exchange) plus its tokens at one
// CTA's streaming rate, which grows with the ring stages in flight until the CTAs resident on an SM
// share its bandwidth; and no launch beats the GPU's streaming rate. A launch small enough to stay
// in L2 across a decode loop is planned with the L2 constants instead.
Plan plan(int D, int NT, int units, int nmax, bool paged = false) {
    const bool l2 = (double)units * nmax * 4.0 * D <= VOXZIP_DECODE_L2_RESIDENT_MB * 1048576.0;
    const PlanModel &md = l2 ? kPlanModelL2 : kPlanModel;
    Plan best{0, 3, 0};
    double best_cost = 0.0;
    int sms = 148;
    {
        int dev = 0;
        if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    }
    const double total = (double)units * nmax;
    for (int S = 1; S <= kMaxCluster; S <<= 1) {
        int cap = (nmax + S - 1) / S;
        if (S > 1 && cap < kTile / 2) break;
        cap = paged ? (cap + kTile - 1) / kTile * kTile : (cap + 15) / 16 * 16;  // paged: whole pages per CTA
        for (int ns : kRingDepths) {
            const size_t sm = dispatch(D, NT, ns, [&](auto k) {
                using K = decltype(k);
                return Layout<K::D, K::NT, K::NS>::bytes(cap);
            });
            if (sm > kMaxSmem) continue;
            const int cl = dispatch(D, NT, ns, [&](auto k) { return max_active_clusters<decltype(k)>(S, sm); });
            if (cl <= 0) continue;
            const double per_sm = fmax(1.0, (double)min(units, cl) * S / sms);  // CTAs sharing an SM
            const double rate = fmin(md.stage_tokens_per_us * min(ns, md.stage_cap), md.sm_tokens_per_us / per_sm);
            const double rounds = (double)((units + cl - 1) / cl);
            const double per_cta = md.cta_fixed_us + (S > 1 ? md.cluster_fixed_us : 0.0) +
                                   (double)((nmax + S - 1) / S) / rate;
            const double cost = fmax(rounds * per_cta, total / md.gpu_tokens_per_us);
            if (best.S == 0 || cost < best_cost) {
                best = Plan{S, ns, cap};
                best_cost = cost;
            }
        }
    }
    return best;
}

}  // namespace

// Returns false when this path does not apply (fp32 cache, other head dims, group > 16).
bool decode_mma_supported(const voxzip_cache_desc &d) {
    const int G = d.q_heads / d.kv_heads;
    return d.dtype == VOXZIP_BF16 && (d.head_dim == 64 || d.head_dim == 128) && G >= 1 && G <= 16 &&
           tensor_map_encoder() != nullptr;
}

namespace {

// The dense and the paged launch: K/V rows are [rows][D] at k_base / v_base (the cache, or the
// page pools), pv.table is null for the dense layout.
cudaError_t launch_impl(const voxzip_cache_desc &d, void *k_base, void *v_base, int64_t rows, const PageView &pv,
                        int32_t layer_begin, int32_t layer_count, const void *q, const void *k_new, const void *v_new,
                        const int32_t *new_pos, float *score, int32_t *pos, int32_t *len, float gamma, float sm_scale,
                        int32_t max_len, void *out, int32_t *status, cudaStream_t stream, bool *unsupported) {
    *unsupported = false;
    const bool paged = pv.table != nullptr;
    const int G = d.q_heads / d.kv_heads;
    const int NT = G <= 8 ? 1 : 2;
    const int units = layer_count * d.batch * d.kv_heads;
    const int nmax = (max_len > 0 && max_len < d.capacity) ? max_len : d.capacity;
    // Plans are cached per (head dim, group tiles, units, length bucket of one tile, layout).
    struct Entry {
        int D, NT, units, bucket;
        bool paged;
        Plan p;
    };
    thread_local Entry cache[16];
    thread_local int cache_next = 0;
    const int bucket = (nmax + kTile - 1) / kTile;
    Plan pl{0, 0, 0};
    for (const Entry &e : cache)
        if (e.p.S != 0 && e.D == d.head_dim && e.NT == NT && e.units == units && e.bucket == bucket &&
            e.paged == paged)
            pl = e.p;
    if (pl.S == 0) {
        pl = plan(d.head_dim, NT, units, bucket * kTile, paged);
        if (pl.S == 0) {
            *unsupported = true;
            return cudaSuccess;
        }
        cache[cache_next] = Entry{d.head_dim, NT, units, bucket, paged, pl};
        cache_next = (cache_next + 1) % 16;
    }
    const int S = pl.S;
    const int chunk_cap = pl.chunk_cap;
    thread_local void *cached_k = nullptr, *cached_v = nullptr;
    thread_local int64_t cached_rows = 0;
    thread_local int cached_d = 0;
    thread_local CUtensorMap tmk, tmv;
    if (cached_k != k_base || cached_v != v_base || cached_rows != rows || cached_d != d.head_dim) {
        if (!make_cache_map(&tmk, k_base, rows, d.head_dim, kTile) ||
            !make_cache_map(&tmv, v_base, rows, d.head_dim, kTile)) {
            cached_k = cached_v = nullptr;
            *unsupported = true;
            return cudaSuccess;
        }
        cached_k = k_base;
        cached_v = v_base;
        cached_rows = rows;
        cached_d = d.head_dim;
    }
    MmaParams prm;
    prm.q = static_cast<const __nv_bfloat16 *>(q);
    prm.k_new = static_cast<const __nv_bfloat16 *>(k_new);
    prm.v_new = static_cast<const __nv_bfloat16 *>(v_new);
    prm.new_pos = new_pos;
    prm.k_cache = static_cast<__nv_bfloat16 *>(k_base);
    prm.v_cache = static_cast<__nv_bfloat16 *>(v_base);
    prm.score = score;
    prm.pos = pos;
    prm.len = len;
    prm.out = static_cast<__nv_bfloat16 *>(out);
    prm.status = status;
    prm.B = d.batch; prm.L = d.layers; prm.Hq = d.q_heads; prm.Hkv = d.kv_heads; prm.G = G;
    prm.C = d.capacity; prm.layer_begin = layer_begin; prm.chunk_cap = chunk_cap; prm.n_hint = nmax;
    prm.rows = rows;
    prm.gamma = gamma;
    prm.pv = pv;
    const float scale = sm_scale > 0.f ? sm_scale : 1.0f / sqrtf((float)d.head_dim);
    prm.scale_log2 = scale * 1.4426950408889634f;  // log2(e): exp(x) = 2^(x log2 e)
    return dispatch(d.head_dim, NT, pl.NS,
                    [&](auto k) { return launch_t<decltype(k)>(tmk, tmv, prm, S, units, stream, paged); });
}

}  // namespace

cudaError_t launch_decode_mma(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count, const void *q,
                              const void *k_new, const void *v_new, const int32_t *new_pos, void *k_cache,
                              void *v_cache, float *score, int32_t *pos, int32_t *len, float gamma, float sm_scale,
                              int32_t max_len, void *out, int32_t *status, cudaStream_t stream, bool *unsupported) {
    const int64_t rows = (int64_t)d.batch * d.layers * d.kv_heads * d.capacity;
    return launch_impl(d, k_cache, v_cache, rows, PageView{nullptr, nullptr, nullptr, 0}, layer_begin, layer_count, q,
                       k_new, v_new, new_pos, score, pos, len, gamma, sm_scale, max_len, out, status, stream,
                       unsupported);
}

bool decode_mma_paged_supported(const voxzip_cache_desc &d) { return decode_mma_supported(d); }

cudaError_t launch_decode_mma_paged(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, int32_t layer_begin,
                                    int32_t layer_count, const void *q, const void *k_new, const void *v_new,
                                    const int32_t *new_pos, float *score, int32_t *pos, int32_t *len, float gamma,
                                    float sm_scale, int32_t max_len, void *out, int32_t *status, cudaStream_t stream,
                                    bool *unsupported) {
    const int64_t rows = (int64_t)pc.pages * kPageTokens;
    return launch_impl(d, pc.k_pool, pc.v_pool, rows, PageView{pc.page_table, pc.free_pages, pc.free_count, pc.max_pages},
                       layer_begin, layer_count, q, k_new, v_new, new_pos, score, pos, len, gamma, sm_scale, max_len,
                       out, status, stream, unsupported);
}

}  // namespace voxzip
