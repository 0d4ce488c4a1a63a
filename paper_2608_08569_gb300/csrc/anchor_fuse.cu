// Stage 1 of VoxZip (Sec. 3.2.1): semantic-anchored fusion of the prefilled K/V cache, or of the
// input embeddings (the paper's own setting).
//
// Kernels, all launched on the caller's stream:
//   span_scan   one CTA per sequence: validates the semantic set (sorted, non-overlapping spans
//               inside the audio region) and scans, per span, the slot shift
//               delta = min(n_groups, l) - l, the anchor-row offset (prefix of n_groups) and the
//               background tokens before the span (dropped in the "Partial" configuration);
//   slot_map    one thread per prompt token: the output slot of the token (Eq. 4 grouping with
//               group j = [floor(j*l/g), floor((j+1)*l/g)), Eq. 5 chronological order); the first
//               token of each slot records the slot's source range and anchor row;
//   fuse_rows   K/V level, head_dim 64 or 128: one warp-slice per output slot of every (layer,
//               kv-head) unit (a lane owns one 16-byte vector of the row; four source rows in
//               flight): the fp32 mean of the slot's source rows (a copy when the range has one
//               row) plus the anchor row, rounded once to the cache dtype; K and V in the same
//               pass; pos and score = 0. A persistent grid walks (128-slot chunk, unit) items;
//               prefill rows in pinned host memory are streamed over the host link by CTAs on
//               half the SMs;
//   fuse_wide   embedding level, any width that is a whole number of 16-byte vectors: one warp per
//               output row of a sequence, the same arithmetic.
// Output slots cover the kept tokens of the prompt in order, each a contiguous source range.
#include <algorithm>

#include "common.cuh"
#include "embed.cuh"
#include "paged.cuh"

namespace voxzip {

// SMs of the current device (looked up once per device).
int sm_count() {
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (cached[dev] == 0) {
        int n = 0;
        cached[dev] = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0 ? n : 148;
    }
    return cached[dev];
}

namespace {

// acc[e] += element e of a 16-byte vector (4 fp32 or 8 bf16 values, low address first).
template <typename T>
__device__ __forceinline__ void accumulate16(float *acc, uint4 x);
template <>
__device__ __forceinline__ void accumulate16<float>(float *acc, uint4 x) {
    acc[0] += __uint_as_float(x.x);
    acc[1] += __uint_as_float(x.y);
    acc[2] += __uint_as_float(x.z);
    acc[3] += __uint_as_float(x.w);
}
template <>
__device__ __forceinline__ void accumulate16<__nv_bfloat16>(float *acc, uint4 x) {
    const uint32_t w[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        acc[2 * i] += __uint_as_float(w[i] << 16);
        acc[2 * i + 1] += __uint_as_float(w[i] & 0xffff0000u);
    }
}
// The 16-byte vector of acc rounded to T (round to nearest even).
template <typename T>
__device__ __forceinline__ uint4 pack16(const float *acc);
template <>
__device__ __forceinline__ uint4 pack16<float>(const float *acc) {
    return make_uint4(__float_as_uint(acc[0]), __float_as_uint(acc[1]), __float_as_uint(acc[2]),
                      __float_as_uint(acc[3]));
}
template <>
__device__ __forceinline__ uint4 pack16<__nv_bfloat16>(const float *acc) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * i]));
        const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(acc[2 * i + 1]));
        w[i] = lo | (hi << 16);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

#ifndef VOXZIP_FUSE_HOST_CTAS
#define VOXZIP_FUSE_HOST_CTAS 0  // stage-1 CTAs when the prefill rows are in host memory (0: half the SMs)
#endif

constexpr int kScanThreads = 512;
constexpr int kMapThreads = 256;
constexpr int kFuseWarps = 8;
constexpr int kSlotsPerWarp = 8;

struct FuseWorkspace {
    int32_t *seq_len;        // [B] stage-1 length, -1 when the sequence is skipped
    int32_t *bg_total;       // [B] background (uncovered audio) tokens of the sequence
    int32_t *delta_prefix;   // [num_spans] exclusive prefix of (g - l) within the sequence
    int32_t *anchor_prefix;  // [num_spans] exclusive prefix of n_groups within the sequence
    int32_t *bg_prefix;      // [num_spans] background tokens before the span's start
    int32_t *slot_src;       // [B][stride] first prompt token of each slot
    int32_t *slot_end;       // [B][stride] one past the last prompt token of each slot
    int32_t *slot_anchor;    // [B][stride] anchor row of each slot, -1 for copied rows
    int32_t *status;         // the call's device status word (not part of the workspace bytes)
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__host__ __device__ inline size_t carve(const voxzip_cache_desc &d, int32_t stride, int32_t num_spans,
                                        char *base, FuseWorkspace *ws) {
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base + off;
        off += align256(bytes);
        return reinterpret_cast<int32_t *>(p);
    };
    int32_t *a = take(sizeof(int32_t) * (size_t)d.batch);
    int32_t *a2 = take(sizeof(int32_t) * (size_t)d.batch);
    int32_t *b = take(sizeof(int32_t) * (size_t)num_spans);
    int32_t *c = take(sizeof(int32_t) * (size_t)num_spans);
    int32_t *c2 = take(sizeof(int32_t) * (size_t)num_spans);
    int32_t *e = take(sizeof(int32_t) * (size_t)d.batch * (size_t)stride);
    int32_t *e2 = take(sizeof(int32_t) * (size_t)d.batch * (size_t)stride);
    int32_t *f = take(sizeof(int32_t) * (size_t)d.batch * (size_t)stride);
    if (ws) {
        ws->seq_len = a;
        ws->bg_total = a2;
        ws->delta_prefix = b;
        ws->anchor_prefix = c;
        ws->bg_prefix = c2;
        ws->slot_src = e;
        ws->slot_end = e2;
        ws->slot_anchor = f;
    }
    return off;
}

// Block-wide exclusive scan of one int per thread; returns the block total in *total.
__device__ int block_excl_scan(int v, int *total) {
    __shared__ int warp_sums[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int s = lane < nw ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        warp_sums[lane] = s;  // inclusive over warps
    }
    __syncthreads();
    const int warp_off = warp > 0 ? warp_sums[warp - 1] : 0;
    *total = warp_sums[nw - 1];
    __syncthreads();
    return warp_off + x - v;
}

__global__ void __launch_bounds__(kScanThreads)
span_scan_kernel(int32_t B, int32_t stride, int32_t capacity, int32_t num_spans, int32_t anchor_stride,
                 bool has_anchor, bool keep_bg, const int32_t *__restrict__ in_len, const int32_t *__restrict__ audio_begin,
                 const int32_t *__restrict__ audio_len, const int32_t *__restrict__ span_off,
                 const int32_t *__restrict__ span_start, const int32_t *__restrict__ span_end,
                 const int32_t *__restrict__ span_groups, FuseWorkspace ws, int32_t *status) {
    const int b = blockIdx.x;
    __shared__ int bad;
    if (threadIdx.x == 0) bad = 0;
    __syncthreads();
    const int32_t n_in = in_len[b], ab = audio_begin[b], al = audio_len[b];
    const int32_t s0 = span_off[b], s1 = span_off[b + 1];
    const bool header_ok = n_in >= 0 && n_in <= stride && ab >= 0 && al >= 0 &&
                           (int64_t)ab + al <= n_in && s0 >= 0 && s0 <= s1 && s1 <= num_spans;
    if (!header_ok) {
        if (threadIdx.x == 0) {
            ws.seq_len[b] = -1;
            raise_status(status, VOXZIP_DEV_BAD_SPANS);
        }
        return;
    }
    int carry_delta = 0, carry_groups = 0, carry_gap = 0;
    for (int base = s0; base < s1; base += blockDim.x) {
        const int i = base + threadIdx.x;
        int delta = 0, groups = 0, gap = 0;
        if (i < s1) {
            const int32_t st = span_start[i], en = span_end[i], ng = span_groups[i];
            const int32_t prev_end = i > s0 ? span_end[i - 1] : ab;
            if (st < prev_end || en < st || en > ab + al || ng < 1) bad = 1;
            const int32_t l = en - st;
            delta = (ng < l ? ng : l) - l;
            groups = ng;
            gap = st - prev_end;  // background audio between the previous span (or the audio start) and this one
        }
        int tot_d, tot_g, tot_b;
        const int ex_d = block_excl_scan(delta, &tot_d);
        const int ex_g = block_excl_scan(groups, &tot_g);
        const int ex_b = block_excl_scan(gap, &tot_b);
        if (i < s1) {
            ws.delta_prefix[i] = carry_delta + ex_d;
            ws.anchor_prefix[i] = carry_groups + ex_g;
            ws.bg_prefix[i] = carry_gap + ex_b + gap;
        }
        carry_delta += tot_d;
        carry_groups += tot_g;
        carry_gap += tot_b;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const int32_t last_end = s1 > s0 ? span_end[s1 - 1] : ab;
        const int32_t bg = carry_gap + (ab + al - last_end);
        ws.bg_total[b] = bg;
        const int64_t out_len = (int64_t)n_in + carry_delta - (keep_bg ? 0 : bg);
        if (bad || (has_anchor && carry_groups > anchor_stride)) {
            ws.seq_len[b] = -1;
            raise_status(status, VOXZIP_DEV_BAD_SPANS);
        } else if (out_len > capacity) {
            ws.seq_len[b] = -1;
            raise_status(status, VOXZIP_DEV_CAPACITY);
        } else {
            ws.seq_len[b] = (int32_t)out_len;
        }
    }
}

__global__ void __launch_bounds__(kMapThreads)
slot_map_kernel(int32_t stride, bool keep_bg, const int32_t *__restrict__ in_len,
                const int32_t *__restrict__ audio_begin, const int32_t *__restrict__ audio_len,
                const int32_t *__restrict__ span_off, const int32_t *__restrict__ span_start,
                const int32_t *__restrict__ span_end, const int32_t *__restrict__ span_groups, FuseWorkspace ws,
                int32_t *__restrict__ slot_map) {
    const int b = blockIdx.y;
    const int32_t t = blockIdx.x * blockDim.x + threadIdx.x;
    const int32_t out_len = ws.seq_len[b];
    const int32_t n_in = in_len[b];
    if (out_len < 0 || t >= n_in) return;
    const int32_t s0 = span_off[b], s1 = span_off[b + 1];
    // Last span with start <= t.
    int lo = s0, hi = s1;  // answer in [s0 - 1, s1)
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (span_start[mid] <= t) lo = mid + 1;
        else hi = mid;
    }
    const int i = lo - 1;
    int32_t slot, end, anchor = -1;
    bool first;
    if (i >= s0 && t < span_end[i]) {
        const int64_t st = span_start[i], l = span_end[i] - st;
        const int64_t ng = span_groups[i];
        const int64_t g = ng < l ? ng : l;
        const int64_t r = t - st;
        const int64_t j = ((r + 1) * g - 1) / l;  // group j holds r iff floor(j*l/g) <= r < floor((j+1)*l/g)
        slot = (int32_t)(st + ws.delta_prefix[i] - (keep_bg ? 0 : ws.bg_prefix[i]) + j);
        first = r == (j * l) / g;
        end = (int32_t)(st + ((j + 1) * l) / g);
        anchor = (int32_t)(ws.anchor_prefix[i] + j);
    } else {
        const int32_t ab = audio_begin[b], ae = ab + audio_len[b];
        if (!keep_bg && t >= ab && t < ae) {  // background audio, dropped ("Partial")
            if (slot_map) slot_map[(int64_t)b * stride + t] = -1;
            return;
        }
        int32_t shift = i >= s0 ? ws.delta_prefix[i] + (min(span_groups[i], span_end[i] - span_start[i]) -
                                                       (span_end[i] - span_start[i]))
                                : 0;
        if (!keep_bg && t >= ae) shift -= ws.bg_total[b];  // a text token after the audio
        slot = t + shift;
        first = true;
        end = t + 1;
    }
    if (slot_map) slot_map[(int64_t)b * stride + t] = slot;
    if (first) {
        ws.slot_src[(int64_t)b * stride + slot] = t;
        ws.slot_end[(int64_t)b * stride + slot] = end;
        ws.slot_anchor[(int64_t)b * stride + slot] = anchor;
    }
}

// A persistent grid (as many CTAs as are resident at once) walks work items: chunk c of the output
// slots of unit u, item = c * units + u, so every CTA gets an equal share of the rows and no wave
// runs part-empty. A chunk is kSlotsPerPass consecutive slots: warp w owns kSlotsPerWarp groups of
// kRowsPerWarp slots. kPaged: k_cache / v_cache are page pools and output slot s goes to the row
// the page table gives.
template <typename T, int D, bool kPaged>
__global__ void __launch_bounds__(kFuseWarps * 32, 4)
fuse_rows_kernel(int32_t B, int32_t L, int32_t Hkv, int32_t C, int32_t stride, int32_t anchor_stride,
                 const T *__restrict__ k_prefill, const T *__restrict__ v_prefill,
                 const T *__restrict__ anchor_k, const T *__restrict__ anchor_v, FuseWorkspace ws,
                 T *__restrict__ k_cache, T *__restrict__ v_cache, float *__restrict__ score,
                 int32_t *__restrict__ pos, int32_t *__restrict__ len, PageView pv) {
    constexpr int kElems = 16 / (int)sizeof(T);  // each lane owns one 16-byte vector of a row
    constexpr int kLanesPerRow = D / kElems;
    constexpr int kRowsPerWarp = 32 / kLanesPerRow;
    constexpr int kRowVecs = D / kElems;          // 16-byte vectors per row
    constexpr int kSlotsPerPass = kFuseWarps * kSlotsPerWarp * kRowsPerWarp;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / kLanesPerRow, e = (lane % kLanesPerRow) * kElems;
    const int units = B * L * Hkv;
    // Chunks per unit: enough for the longest stage-1 output of the batch.
    int max_len = 0;
    for (int bb = 0; bb < B; ++bb) max_len = max(max_len, ws.seq_len[bb]);
    const int chunks = max(1, (max_len + kSlotsPerPass - 1) / kSlotsPerPass);
    for (int64_t item = blockIdx.x; item < (int64_t)units * chunks; item += gridDim.x) {
        const int u = (int)(item % units);   // cache unit (b, l, h)
        const int chunk = (int)(item / units);
        const int b = u / (L * Hkv);
        int32_t out_len = ws.seq_len[b];
        if (kPaged && pv.table[(int64_t)u * pv.max_pages] < 0) out_len = -1;  // the pool could not hold it
        if (chunk == 0 && threadIdx.x == 0) len[u] = out_len < 0 ? 0 : out_len;
        if (out_len <= chunk * kSlotsPerPass) continue;
        const int64_t in_base = (int64_t)u * stride * D;
        const int64_t out_base = kPaged ? 0 : (int64_t)u * C * D;
        const int64_t anc_base = (int64_t)u * anchor_stride * D;
        const uint4 *kin = reinterpret_cast<const uint4 *>(k_prefill + in_base + e);  // vector e of row 0
        const uint4 *vin = reinterpret_cast<const uint4 *>(v_prefill + in_base + e);
        const int32_t *src = ws.slot_src + (int64_t)b * stride;
        const int32_t *send = ws.slot_end + (int64_t)b * stride;
        const int32_t *anc = ws.slot_anchor + (int64_t)b * stride;
        const int slot0 = chunk * kSlotsPerPass + warp * kSlotsPerWarp * kRowsPerWarp;
        // The warp's slots' source ranges and anchor rows, one slot per lane, fetched together up
        // front, so no slot's row loads wait behind its own metadata load.
        static_assert(kSlotsPerWarp * kRowsPerWarp <= 32, "one slot per lane");
        int32_t m0 = 0, m1 = 0, ma = -1;
        if (lane < kSlotsPerWarp * kRowsPerWarp && slot0 + lane < out_len) {
            m0 = src[slot0 + lane];
            m1 = send[slot0 + lane];
            ma = anc[slot0 + lane];
        }
        for (int k = 0; k < kSlotsPerWarp; ++k) {
            const int li = k * kRowsPerWarp + sub;
            const int s = slot0 + li;
            const int32_t r0 = __shfl_sync(0xffffffffu, m0, li), r1 = __shfl_sync(0xffffffffu, m1, li);
            const int32_t a_row = __shfl_sync(0xffffffffu, ma, li);
            if (s >= out_len) continue;  // (every lane still takes the shuffles of every k)
            if (!VOXZIP_IN_RANGE(ws.status, r0 >= 0 && r0 < r1 && r1 <= stride && s < C)) continue;
            float sk[kElems], sv[kElems];
#pragma unroll
            for (int i = 0; i < kElems; ++i) sk[i] = sv[i] = 0.f;
            int32_t r = r0;
            for (; r + 4 <= r1; r += 4) {  // four rows' loads in flight, then their sums in token order
                uint4 xk[4], xv[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    xk[i] = __ldcs(kin + (int64_t)(r + i) * kRowVecs);
                    xv[i] = __ldcs(vin + (int64_t)(r + i) * kRowVecs);
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    accumulate16<T>(sk, xk[i]);
                    accumulate16<T>(sv, xv[i]);
                }
            }
            for (; r < r1; ++r) {
                accumulate16<T>(sk, __ldcs(kin + (int64_t)r * kRowVecs));
                accumulate16<T>(sv, __ldcs(vin + (int64_t)r * kRowVecs));
            }
            if (r1 - r0 > 1) {
                const float cnt = (float)(r1 - r0);
#pragma unroll
                for (int i = 0; i < kElems; ++i) {
                    sk[i] = __fdiv_rn(sk[i], cnt);
                    sv[i] = __fdiv_rn(sv[i], cnt);
                }
            }
            if (anchor_k != nullptr && a_row >= 0 && VOXZIP_IN_RANGE(ws.status, a_row < anchor_stride)) {
                float ak[kElems], av[kElems];
#pragma unroll
                for (int i = 0; i < kElems; ++i) ak[i] = av[i] = 0.f;
                accumulate16<T>(ak, *reinterpret_cast<const uint4 *>(anchor_k + anc_base + (int64_t)a_row * D + e));
                accumulate16<T>(av, *reinterpret_cast<const uint4 *>(anchor_v + anc_base + (int64_t)a_row * D + e));
#pragma unroll
                for (int i = 0; i < kElems; ++i) {
                    sk[i] = __fadd_rn(sk[i], ak[i]);
                    sv[i] = __fadd_rn(sv[i], av[i]);
                }
            }
            const int64_t orow = kPaged ? paged_row(pv, u, s) : s;
            *reinterpret_cast<uint4 *>(k_cache + out_base + orow * D + e) = pack16<T>(sk);
            *reinterpret_cast<uint4 *>(v_cache + out_base + orow * D + e) = pack16<T>(sv);
            if (e == 0) {
                pos[(int64_t)u * C + s] = r0;
                score[(int64_t)u * C + s] = 0.f;
            }
        }
    }
}

template <typename T, int D, bool kPaged = false>
cudaError_t launch_fuse_rows(const voxzip_cache_desc &d, int32_t stride, int32_t anchor_stride,
                             const void *kp, const void *vp, const void *ak, const void *av,
                             const FuseWorkspace &ws, void *kc, void *vc, float *score, int32_t *pos,
                             int32_t *len, cudaStream_t stream, PageView pv = PageView{nullptr, nullptr, nullptr, 0}) {
    constexpr int kRowsPerWarp = 32 / (D * (int)sizeof(T) / 16);  // as in the kernel
    const int slots_per_block = kFuseWarps * kSlotsPerWarp * kRowsPerWarp;
    const int64_t units = (int64_t)d.batch * d.layers * d.kv_heads;
    // As many CTAs as are resident at once (never more than the work items of the longest possible
    // output): each walks items grid-stride.
    static int per_sm = 0;
    if (per_sm == 0 && (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fuse_rows_kernel<T, D, kPaged>,
                                                                       kFuseWarps * 32, 0) != cudaSuccess ||
                        per_sm < 1)) {
        cudaGetLastError();
        per_sm = 4;
    }
    const int64_t items = units * ((stride + slots_per_block - 1) / slots_per_block);
    // Prefill rows in host memory the device addresses directly (page-locked memory under unified
    // addressing, across the Grace-Blackwell C2C link): the kernel streams them over the host link.
    // CTAs on half the SMs already keep the link busy (on GB300: 87 ms for the 18.1 GB of a 60-min
    // request, ~209 GB/s), and the rest of the GPU stays free for a kernel running beside it: a decode
    // loop of another request slows by ~2% (by 67% when every SM also runs a stage-1 CTA).
    cudaPointerAttributes pa{};
    const bool host_rows = cudaPointerGetAttributes(&pa, kp) == cudaSuccess && pa.type == cudaMemoryTypeHost;
    cudaGetLastError();
    const int64_t ctas = host_rows ? (VOXZIP_FUSE_HOST_CTAS > 0 ? VOXZIP_FUSE_HOST_CTAS : std::max(1, sm_count() / 2))
                                   : (int64_t)sm_count() * per_sm;
    const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(items, ctas));
    fuse_rows_kernel<T, D, kPaged><<<grid, kFuseWarps * 32, 0, stream>>>(
        d.batch, d.layers, d.kv_heads, d.capacity, stride, anchor_stride, (const T *)kp, (const T *)vp,
        (const T *)ak, (const T *)av, ws, (T *)kc, (T *)vc, score, pos, len, pv);
    return cudaGetLastError();
}

constexpr int kWideWarps = 8;

// Embedding-level fusion: one warp per output row of sequence b; each lane owns 16-byte vectors
// v and v + 32 of the row (two in flight per source row). The arithmetic is fuse_rows' (fp32 sum
// in token order, IEEE division by the group size, fp32 anchor add, one rounding).
template <typename T>
__global__ void __launch_bounds__(kWideWarps * 32)
fuse_wide_kernel(int32_t C, int32_t stride, int32_t D, int32_t text_stride, const T *__restrict__ e_in,
                 const T *__restrict__ e_text, FuseWorkspace ws, T *__restrict__ e_out, int32_t *__restrict__ pos,
                 int32_t *__restrict__ len) {
    constexpr int kElems = 16 / sizeof(T);
    const int b = blockIdx.y;
    const int32_t out_len = ws.seq_len[b];
    if (blockIdx.x == 0 && threadIdx.x == 0) len[b] = out_len < 0 ? 0 : out_len;
    if (out_len < 0) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int vecs = D / kElems;
    const T *in = e_in + (int64_t)b * stride * D;
    const T *txt = e_text ? e_text + (int64_t)b * text_stride * D : nullptr;
    T *out = e_out + (int64_t)b * C * D;
    const int32_t *src = ws.slot_src + (int64_t)b * stride;
    const int32_t *send = ws.slot_end + (int64_t)b * stride;
    const int32_t *anc = ws.slot_anchor + (int64_t)b * stride;
    for (int s = blockIdx.x * kWideWarps + warp; s < out_len; s += gridDim.x * kWideWarps) {
        const int32_t r0 = src[s], r1 = send[s], a_row = anc[s];
        if (!VOXZIP_IN_RANGE(ws.status, r0 >= 0 && r0 < r1 && r1 <= stride && s < C &&
                                         (txt == nullptr || a_row < text_stride)))
            continue;
        const float cnt = (float)(r1 - r0);
        for (int v0 = lane; v0 < vecs; v0 += 64) {
            const bool two = v0 + 32 < vecs;
            float acc[2][kElems];
#pragma unroll
            for (int h = 0; h < 2; ++h)
#pragma unroll
                for (int e = 0; e < kElems; ++e) acc[h][e] = 0.f;
            const uint4 *col = reinterpret_cast<const uint4 *>(in) + v0;   // vector v0 of row 0
            const int64_t rstride = vecs;                                    // vectors per row
            int32_t r = r0;
            // Four source rows' loads in flight, then their sums in token order.
            for (; r + 4 <= r1; r += 4) {
                uint4 x[4][2];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    x[i][0] = __ldcs(col + (int64_t)(r + i) * rstride);
                    x[i][1] = two ? __ldcs(col + (int64_t)(r + i) * rstride + 32) : x[i][0];
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    accumulate16<T>(acc[0], x[i][0]);
                    accumulate16<T>(acc[1], x[i][1]);
                }
            }
            for (; r < r1; ++r) {
                const uint4 x0 = __ldcs(col + (int64_t)r * rstride);
                const uint4 x1 = two ? __ldcs(col + (int64_t)r * rstride + 32) : x0;
                accumulate16<T>(acc[0], x0);
                accumulate16<T>(acc[1], x1);
            }
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                if (h == 1 && !two) break;
                const int v = v0 + 32 * h;
                if (r1 - r0 > 1)
#pragma unroll
                    for (int e = 0; e < kElems; ++e) acc[h][e] = __fdiv_rn(acc[h][e], cnt);
                if (txt != nullptr && a_row >= 0) {
                    float t[kElems];
#pragma unroll
                    for (int e = 0; e < kElems; ++e) t[e] = 0.f;
                    accumulate16<T>(t, *reinterpret_cast<const uint4 *>(txt + (int64_t)a_row * D + v * kElems));
#pragma unroll
                    for (int e = 0; e < kElems; ++e) acc[h][e] = __fadd_rn(acc[h][e], t[e]);
                }
                *reinterpret_cast<uint4 *>(out + (int64_t)s * D + v * kElems) = pack16<T>(acc[h]);
            }
        }
        if (lane == 0) pos[(int64_t)b * C + s] = r0;
    }
}

// Paged stage 1, step 1: every unit of the launch returns all its pages (one warp per unit).
__global__ void __launch_bounds__(256) page_release_kernel(int64_t units, PageView pv) {
    const int64_t u = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    if (u < units) return_pages_warp(pv, u, 0, pv.max_pages);
}

// Step 2: each unit takes the pages of slots [0, n] for its stage-1 length n (all or none; none
// leaves page 0 missing, which the fusion and later calls read as "skipped").
__global__ void __launch_bounds__(256) page_take_kernel(int64_t units, int32_t per_seq, FuseWorkspace ws, PageView pv,
                                                        int32_t *status) {
    const int64_t u = (int64_t)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (u >= units) return;
    const int32_t n = max(0, ws.seq_len[u / per_seq]);
    const int32_t need = min(n / kPageTokens + 1, pv.max_pages);  // a full unit needs no page for slot n
    int32_t top = 0;
    if (lane == 0) {
        top = atomicSub(pv.free_count, need);
        if (top < need) {  // not enough: give them back (whatever other units did meanwhile)
            atomicAdd(pv.free_count, need);
            raise_status(status, VOXZIP_DEV_CAPACITY);
            top = -1;
        }
    }
    top = __shfl_sync(0xffffffffu, top, 0);
    if (top < 0) return;
    for (int32_t p = lane; p < need; p += 32) pv.table[u * pv.max_pages + p] = pv.free_pages[top - need + p];
}

// span_scan then slot_map: the slot, source range and anchor row of every output row.
cudaError_t launch_slot_plan(int32_t B, int32_t capacity, int32_t stride, int32_t num_spans, int32_t anchor_stride,
                             bool has_anchor, bool keep_bg, const int32_t *in_len, const int32_t *audio_begin,
                             const int32_t *audio_len, const int32_t *span_off, const int32_t *span_start,
                             const int32_t *span_end, const int32_t *span_groups, const FuseWorkspace &ws,
                             int32_t *slot_map, int32_t *status, cudaStream_t stream) {
    span_scan_kernel<<<B, kScanThreads, 0, stream>>>(B, stride, capacity, num_spans, anchor_stride, has_anchor,
                                                    keep_bg, in_len, audio_begin, audio_len, span_off, span_start,
                                                    span_end, span_groups, ws, status);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    dim3 grid_map((unsigned)((stride + kMapThreads - 1) / kMapThreads), (unsigned)B);
    slot_map_kernel<<<grid_map, kMapThreads, 0, stream>>>(stride, keep_bg, in_len, audio_begin, audio_len, span_off,
                                                          span_start, span_end, span_groups, ws, slot_map);
    return cudaGetLastError();
}

}  // namespace

size_t anchor_fuse_workspace_bytes(const voxzip_cache_desc &d, int32_t prefill_stride, int32_t num_spans) {
    return carve(d, prefill_stride, num_spans, nullptr, nullptr);
}

cudaError_t launch_anchor_fuse(const voxzip_cache_desc &d, const void *k_prefill, const void *v_prefill,
                               int32_t prefill_stride, const int32_t *in_len, const int32_t *audio_begin,
                               const int32_t *audio_len, const int32_t *span_off, int32_t num_spans,
                               const int32_t *span_start, const int32_t *span_end,
                               const int32_t *span_groups, const void *anchor_k, const void *anchor_v,
                               int32_t anchor_stride, void *k_cache, void *v_cache, float *score,
                               int32_t *pos, int32_t *len, int32_t *slot_map, void *workspace,
                               int32_t *status, cudaStream_t stream) {
    FuseWorkspace ws;
    carve(d, prefill_stride, num_spans, static_cast<char *>(workspace), &ws);
    ws.status = status;
    cudaError_t err = launch_slot_plan(d.batch, d.capacity, prefill_stride, num_spans, anchor_stride,
                                       anchor_k != nullptr, true, in_len, audio_begin, audio_len, span_off,
                                       span_start, span_end, span_groups, ws, slot_map, status, stream);
    if (err != cudaSuccess) return err;
    const bool bf16 = d.dtype == VOXZIP_BF16;
    if (d.head_dim == 128)
        return bf16 ? launch_fuse_rows<__nv_bfloat16, 128>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                            anchor_k, anchor_v, ws, k_cache, v_cache, score, pos,
                                                            len, stream)
                    : launch_fuse_rows<float, 128>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                   anchor_k, anchor_v, ws, k_cache, v_cache, score, pos, len,
                                                   stream);
    return bf16 ? launch_fuse_rows<__nv_bfloat16, 64>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                       anchor_k, anchor_v, ws, k_cache, v_cache, score, pos, len,
                                                       stream)
                : launch_fuse_rows<float, 64>(d, prefill_stride, anchor_stride, k_prefill, v_prefill, anchor_k,
                                              anchor_v, ws, k_cache, v_cache, score, pos, len, stream);
}

size_t anchor_fuse_paged_workspace_bytes(const voxzip_cache_desc &d, int32_t prefill_stride, int32_t num_spans) {
    return carve(d, prefill_stride, num_spans, nullptr, nullptr);
}

cudaError_t launch_anchor_fuse_paged(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, const void *k_prefill,
                                     const void *v_prefill, int32_t prefill_stride, const int32_t *in_len,
                                     const int32_t *audio_begin, const int32_t *audio_len, const int32_t *span_off,
                                     int32_t num_spans, const int32_t *span_start, const int32_t *span_end,
                                     const int32_t *span_groups, const void *anchor_k, const void *anchor_v,
                                     int32_t anchor_stride, float *score, int32_t *pos, int32_t *len,
                                     int32_t *slot_map, void *workspace, int32_t *status, cudaStream_t stream) {
    FuseWorkspace ws;
    carve(d, prefill_stride, num_spans, static_cast<char *>(workspace), &ws);
    ws.status = status;
    const PageView pv{pc.page_table, pc.free_pages, pc.free_count, pc.max_pages};
    const int64_t units = (int64_t)d.batch * d.layers * d.kv_heads;
    const unsigned blocks = (unsigned)((units + 7) / 8);
    page_release_kernel<<<blocks, 256, 0, stream>>>(units, pv);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    err = launch_slot_plan(d.batch, d.capacity, prefill_stride, num_spans, anchor_stride, anchor_k != nullptr, true,
                           in_len, audio_begin, audio_len, span_off, span_start, span_end, span_groups, ws, slot_map,
                           status, stream);
    if (err != cudaSuccess) return err;
    page_take_kernel<<<blocks, 256, 0, stream>>>(units, d.layers * d.kv_heads, ws, pv, status);
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    const bool bf16 = d.dtype == VOXZIP_BF16;
    void *kc = pc.k_pool, *vc = pc.v_pool;
    if (d.head_dim == 128)
        return bf16 ? launch_fuse_rows<__nv_bfloat16, 128, true>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                                  anchor_k, anchor_v, ws, kc, vc, score, pos, len,
                                                                  stream, pv)
                    : launch_fuse_rows<float, 128, true>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                         anchor_k, anchor_v, ws, kc, vc, score, pos, len, stream, pv);
    return bf16 ? launch_fuse_rows<__nv_bfloat16, 64, true>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                             anchor_k, anchor_v, ws, kc, vc, score, pos, len, stream,
                                                             pv)
                : launch_fuse_rows<float, 64, true>(d, prefill_stride, anchor_stride, k_prefill, v_prefill, anchor_k,
                                                    anchor_v, ws, kc, vc, score, pos, len, stream, pv);
}

// Empty units: page u holds unit u's slot 0, the other pages are stacked free, lengths are 0.
__global__ void paged_init_kernel(int64_t units, int32_t max_pages, int32_t pages, int32_t *table,
                                  int32_t *free_pages, int32_t *free_count, int32_t *len) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const int64_t first = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    for (int64_t i = first; i < units * max_pages; i += stride)
        table[i] = i % max_pages == 0 ? (int32_t)(i / max_pages) : -1;
    for (int64_t j = first; j < pages - units; j += stride) free_pages[j] = (int32_t)(units + j);
    for (int64_t u = first; u < units; u += stride) len[u] = 0;
    if (first == 0) *free_count = (int32_t)(pages - units);
}

cudaError_t launch_paged_init(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, int32_t *len,
                              cudaStream_t stream) {
    const int64_t units = (int64_t)d.batch * d.layers * d.kv_heads;
    paged_init_kernel<<<sm_count() * 4, 256, 0, stream>>>(units, pc.max_pages, pc.pages, pc.page_table,
                                                          pc.free_pages, pc.free_count, len);
    return cudaGetLastError();
}

size_t embed_fuse_workspace_bytes(int32_t batch, int32_t stride, int32_t num_spans) {
    voxzip_cache_desc d{};
    d.batch = batch;
    return carve(d, stride, num_spans, nullptr, nullptr);
}

cudaError_t launch_embed_fuse(int32_t B, int32_t D, int32_t C, bool bf16, const void *e_in, int32_t stride,
                              const int32_t *in_len, const int32_t *audio_begin, const int32_t *audio_len,
                              const int32_t *span_off, int32_t num_spans, const int32_t *span_start,
                              const int32_t *span_end, const int32_t *span_groups, const void *e_text,
                              int32_t text_stride, bool keep_background, void *e_out, int32_t *pos, int32_t *len,
                              int32_t *slot_map, void *workspace, int32_t *status, cudaStream_t stream) {
    voxzip_cache_desc d{};
    d.batch = B;
    FuseWorkspace ws;
    carve(d, stride, num_spans, static_cast<char *>(workspace), &ws);
    ws.status = status;
    cudaError_t err = launch_slot_plan(B, C, stride, num_spans, text_stride, e_text != nullptr, keep_background,
                                       in_len, audio_begin, audio_len, span_off, span_start, span_end, span_groups,
                                       ws, slot_map, status, stream);
    if (err != cudaSuccess) return err;
    // A grid-stride loop over the output rows; about five CTAs of 8 warps per SM in all (the
    // output has far fewer rows than the prompt stride the slot plan is sized for).
    const int per_seq = (sm_count() * 5 + B - 1) / B;
    dim3 grid((unsigned)max(1, min((stride + kWideWarps - 1) / kWideWarps, per_seq)), (unsigned)B);
    if (bf16)
        fuse_wide_kernel<__nv_bfloat16><<<grid, kWideWarps * 32, 0, stream>>>(
            C, stride, D, text_stride, (const __nv_bfloat16 *)e_in, (const __nv_bfloat16 *)e_text, ws,
            (__nv_bfloat16 *)e_out, pos, len);
    else
        fuse_wide_kernel<float><<<grid, kWideWarps * 32, 0, stream>>>(C, stride, D, text_stride, (const float *)e_in,
                                                                      (const float *)e_text, ws, (float *)e_out, pos,
                                                                      len);
    return cudaGetLastError();
}

}  // namespace voxzip
