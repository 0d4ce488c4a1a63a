// Budgeted eviction of VoxZip (Sec. 3.2.2, Eq. 7-9): keep T sinks, the M most recent rows and
// the top-N history rows by decayed score, then compact K, V, score and pos in place.
//
// One CTA per unit:
//   select   an 8-pass MSB-first radix select over 64-bit keys (order-preserving score bits,
//            then the complemented position, so equal scores rank the lower position higher)
//            finds the key of the N-th best history row. Keys are unique within a unit, so
//            "key >= threshold" keeps exactly N rows.
//   compact  slots are scanned in order, 1024 at a time; a block scan gives every kept slot its
//            destination (its rank among kept slots) and the rows move in sub-chunks of rank
//            order. A kept row never moves up (dest <= src), and the rows of a sub-chunk are all
//            read into shared memory before any is written, so no row is overwritten before it
//            is read: later sub-chunks read only slots at or beyond their own ranks, which lie
//            past every destination written earlier.
#include "common.cuh"

namespace voxzip {
namespace {

constexpr int kThreads = 1024;
constexpr int kStageBytes = 32 * 1024;

struct EvictParams {
    void *k_cache, *v_cache;
    float *score;
    int32_t *pos, *len;
    const int32_t *budget;
    int32_t *status;
    int32_t B, L, Hkv, C, layer_begin, sink;
    float recent_frac;
};

__device__ __forceinline__ uint64_t order_key(float s, int32_t p) {
    uint32_t b = __float_as_uint(s);
    b = (b & 0x80000000u) ? ~b : (b | 0x80000000u);  // monotone map of fp32 order to uint32 order
    return ((uint64_t)b << 32) | (uint64_t)(0xffffffffu - (uint32_t)p);
}

// Block-wide exclusive scan of one int per thread (blockDim.x == kThreads).
__device__ int scan_excl(int v, int *total, int *warp_sums) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int s = warp_sums[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        warp_sums[lane] = s;
    }
    __syncthreads();
    const int r = (warp > 0 ? warp_sums[warp - 1] : 0) + x - v;
    *total = warp_sums[31];
    __syncthreads();
    return r;
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) evict_kernel(const EvictParams p) {
    constexpr int kVecPerRow = D * (int)sizeof(T) / 16;      // 16-byte vectors per K (or V) row
    constexpr int kRowsPerStage = kStageBytes / (2 * D * (int)sizeof(T));
    __shared__ uint4 stage[kStageBytes / 16];
    __shared__ float stage_score[kRowsPerStage];
    __shared__ int32_t stage_pos[kRowsPerStage];
    __shared__ int32_t src_list[kThreads];
    __shared__ unsigned hist[256];
    __shared__ int warp_sums[32];
    __shared__ unsigned long long sel_prefix;
    __shared__ int sel_rem;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const UnitIdx ui = unit_of(blockIdx.x, p.B, p.L, p.Hkv, p.layer_begin);
    const int32_t n = p.len[ui.cache_unit];
    const int32_t bud = p.budget[ui.b];
    const int32_t M = (int32_t)floor((double)p.recent_frac * (double)bud);
    const int32_t T_ = p.sink;
    const int32_t N = bud - T_ - M;
    if (bud < 0 || N < 0) {
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
    uint4 *kc = reinterpret_cast<uint4 *>(static_cast<T *>(p.k_cache) + ui.cache_unit * p.C * D);
    uint4 *vc = reinterpret_cast<uint4 *>(static_cast<T *>(p.v_cache) + ui.cache_unit * p.C * D);
    const int32_t c_end = n - M;  // history candidates are slots [T, c_end)

    // Eq. 9: the key of the N-th largest candidate.
    uint64_t prefix = 0;
    int rem = N;
    if (N > 0) {
        for (int pass = 0; pass < 8; ++pass) {
            const int shift = 56 - 8 * pass;
            for (int i = tid; i < 256; i += kThreads) hist[i] = 0u;
            __syncthreads();
            for (int j = T_ + tid; j < c_end; j += kThreads) {
                const uint64_t key = order_key(sc[j], ps[j]);
                if (pass == 0 || (key >> (shift + 8)) == (prefix >> (shift + 8)))
                    atomicAdd(&hist[(unsigned)(key >> shift) & 255u], 1u);
            }
            __syncthreads();
            if (warp == 0) {
                // Lane l holds bins 255-8l down to 248-8l: counts accumulate from the top bin.
                const int top = 255 - lane * 8;
                unsigned c[8], s = 0;
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    c[k] = hist[top - k];
                    s += c[k];
                }
                unsigned incl = s;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const unsigned y = __shfl_up_sync(0xffffffffu, incl, o);
                    if (lane >= o) incl += y;
                }
                const unsigned excl = incl - s;
                const bool hit = excl < (unsigned)rem && (unsigned)rem <= incl;
                const unsigned ballot = __ballot_sync(0xffffffffu, hit);
                if (lane == __ffs(ballot) - 1) {
                    unsigned cum = excl;
                    for (int k = 0; k < 8; ++k) {
                        if (cum + c[k] >= (unsigned)rem) {
                            sel_prefix = prefix | ((unsigned long long)(top - k) << shift);
                            sel_rem = rem - (int)cum;
                            break;
                        }
                        cum += c[k];
                    }
                }
            }
            __syncthreads();
            prefix = sel_prefix;
            rem = sel_rem;
        }
    }
    const uint64_t thr = prefix;  // keys above thr are kept, plus the first `rem` equal to it

    // Eq. 7-8: ordered, in-place compaction of the kept rows.
    int base_rank = 0, eq_seen = 0;
    for (int c0 = 0; c0 < n; c0 += kThreads) {
        const int j = c0 + tid;
        const bool in = j < n;
        const bool cand = in && j >= T_ && j < c_end;
        const uint64_t key = cand ? order_key(sc[j], ps[j]) : 0ull;
        const bool eq = cand && N > 0 && key == thr;
        int eq_total;
        const int eq_rank = scan_excl(eq ? 1 : 0, &eq_total, warp_sums);
        const bool keep = in && (!cand || (N > 0 && (key > thr || (eq && eq_seen + eq_rank < rem))));
        int kept_total;
        const int k_rank = scan_excl(keep ? 1 : 0, &kept_total, warp_sums);
        if (keep) src_list[k_rank] = j;
        eq_seen += eq_total;
        __syncthreads();
        for (int r0 = 0; r0 < kept_total; r0 += kRowsPerStage) {
            const int rows = min(kRowsPerStage, kept_total - r0);
            for (int v = tid; v < rows * 2 * kVecPerRow; v += kThreads) {
                const int row = v / (2 * kVecPerRow), w = v % (2 * kVecPerRow);
                const int src = src_list[r0 + row], dst = base_rank + r0 + row;
                if (src != dst) {
                    const uint4 *from = w < kVecPerRow ? kc : vc;
                    stage[v] = from[(int64_t)src * kVecPerRow + (w % kVecPerRow)];
                }
            }
            for (int row = tid; row < rows; row += kThreads) {
                const int src = src_list[r0 + row];
                stage_score[row] = sc[src];
                stage_pos[row] = ps[src];
            }
            __syncthreads();
            for (int v = tid; v < rows * 2 * kVecPerRow; v += kThreads) {
                const int row = v / (2 * kVecPerRow), w = v % (2 * kVecPerRow);
                const int src = src_list[r0 + row], dst = base_rank + r0 + row;
                if (src != dst) {
                    uint4 *to = w < kVecPerRow ? kc : vc;
                    to[(int64_t)dst * kVecPerRow + (w % kVecPerRow)] = stage[v];
                }
            }
            for (int row = tid; row < rows; row += kThreads) {
                const int dst = base_rank + r0 + row;
                sc[dst] = stage_score[row];
                ps[dst] = stage_pos[row];
            }
            __syncthreads();
        }
        base_rank += kept_total;
    }
    if (tid == 0) p.len[ui.cache_unit] = base_rank;  // == budget
}

template <typename T, int D>
cudaError_t launch_t(const EvictParams &prm, int units, cudaStream_t stream) {
    evict_kernel<T, D><<<units, kThreads, 0, stream>>>(prm);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_evict(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count,
                         void *k_cache, void *v_cache, float *score, int32_t *pos, int32_t *len,
                         const int32_t *budget, int32_t sink, float recent_frac, int32_t *status,
                         cudaStream_t stream) {
    EvictParams prm;
    prm.k_cache = k_cache; prm.v_cache = v_cache; prm.score = score; prm.pos = pos; prm.len = len;
    prm.budget = budget; prm.status = status;
    prm.B = d.batch; prm.L = d.layers; prm.Hkv = d.kv_heads; prm.C = d.capacity;
    prm.layer_begin = layer_begin; prm.sink = sink; prm.recent_frac = recent_frac;
    const int units = layer_count * d.batch * d.kv_heads;
    const bool bf16 = d.dtype == VOXZIP_BF16;
    if (d.head_dim == 128)
        return bf16 ? launch_t<__nv_bfloat16, 128>(prm, units, stream) : launch_t<float, 128>(prm, units, stream);
    return bf16 ? launch_t<__nv_bfloat16, 64>(prm, units, stream) : launch_t<float, 64>(prm, units, stream);
}

}  // namespace voxzip
