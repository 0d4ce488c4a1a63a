// Measurement helper: a plain streaming read of a device buffer, launched the way the decode and
// eviction kernels are (a programmatic dependent of the previous kernel on the stream). It is the
// ceiling a kernel that moves the same bytes is measured against; it computes nothing of the method.
#include "common.cuh"
#include "ptx.cuh"

namespace {

constexpr int kReadThreads = 256;
constexpr int kReadUnroll = 8;      // 16-byte loads in flight per thread (the asm below issues 8)
constexpr int kReadCtasPerSm = 8;  // 2 048 threads per SM

__global__ void __launch_bounds__(kReadThreads) stream_read_kernel(const uint4 *p, size_t n16, uint32_t *sink) {
    voxzip::ptx::grid_dependency_wait();
    uint32_t x = 0;
    const size_t stride = (size_t)gridDim.x * kReadThreads;
    size_t i = (size_t)blockIdx.x * kReadThreads + threadIdx.x;
    for (; i + (kReadUnroll - 1) * stride < n16; i += kReadUnroll * stride) {
        // all loads of the batch are issued (one asm statement) before any of them is used
        uint4 v[kReadUnroll];
        const uint4 *q = p + i;
        const size_t sb = stride * sizeof(uint4);
        asm volatile(
            "{\n\t.reg .u64 a;\n\t"
            "mov.u64 a, %32;\n\t"
            "ld.global.cs.v4.u32 {%0, %1, %2, %3}, [a];\n\tadd.u64 a, a, %33;\n\t"
            "ld.global.cs.v4.u32 {%4, %5, %6, %7}, [a];\n\tadd.u64 a, a, %33;\n\t"
            "ld.global.cs.v4.u32 {%8, %9, %10, %11}, [a];\n\tadd.u64 a, a, %33;\n\t"
            "ld.global.cs.v4.u32 {%12, %13, %14, %15}, [a];\n\tadd.u64 a, a, %33;\n\t"
            "ld.global.cs.v4.u32 {%16, %17, %18, %19}, [a];\n\tadd.u64 a, a, %33;\n\t"
            "ld.global.cs.v4.u32 {%20, %21, %22, %23}, [a];\n\tadd.u64 a, a, %33;\n\t"
            "ld.global.cs.v4.u32 {%24, %25, %26, %27}, [a];\n\tadd.u64 a, a, %33;\n\t"
            "ld.global.cs.v4.u32 {%28, %29, %30, %31}, [a];\n\t}"
            : "=r"(v[0].x), "=r"(v[0].y), "=r"(v[0].z), "=r"(v[0].w), "=r"(v[1].x), "=r"(v[1].y), "=r"(v[1].z),
              "=r"(v[1].w), "=r"(v[2].x), "=r"(v[2].y), "=r"(v[2].z), "=r"(v[2].w), "=r"(v[3].x), "=r"(v[3].y),
              "=r"(v[3].z), "=r"(v[3].w), "=r"(v[4].x), "=r"(v[4].y), "=r"(v[4].z), "=r"(v[4].w), "=r"(v[5].x),
              "=r"(v[5].y), "=r"(v[5].z), "=r"(v[5].w), "=r"(v[6].x), "=r"(v[6].y), "=r"(v[6].z), "=r"(v[6].w),
              "=r"(v[7].x), "=r"(v[7].y), "=r"(v[7].z), "=r"(v[7].w)
            : "l"(q), "l"(sb));
#pragma unroll
        for (int u = 0; u < kReadUnroll; ++u) x ^= v[u].x ^ v[u].y ^ v[u].z ^ v[u].w;
    }
    for (; i < n16; i += stride) {
        const uint4 v = __ldcs(p + i);
        x ^= v.x ^ v.y ^ v.z ^ v.w;
    }
    voxzip::ptx::launch_dependents();
    if (x == 0x9e3779b9u) atomicXor(sink, x);  // keeps the loads; practically never taken
}

}  // namespace

extern "C" voxzip_status voxzip_stream_read(const void *p, size_t bytes, uint32_t *sink, voxzip_stream_t stream) {
    if (p == nullptr || sink == nullptr || (reinterpret_cast<uintptr_t>(p) & 15u) != 0 || bytes % 16 != 0)
        return VOXZIP_EINVAL;
    if (bytes == 0) return VOXZIP_OK;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return VOXZIP_ECUDA;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(sms * kReadCtasPerSm), 1, 1);
    cfg.blockDim = dim3(kReadThreads, 1, 1);
    cfg.stream = reinterpret_cast<cudaStream_t>(stream);
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaError_t err = cudaLaunchKernelEx(&cfg, stream_read_kernel, reinterpret_cast<const uint4 *>(p), bytes / 16, sink);
    if (err == cudaErrorNotSupported || err == cudaErrorInvalidValue) {  // no programmatic launch here
        cudaGetLastError();
        cfg.numAttrs = 0;
        err = cudaLaunchKernelEx(&cfg, stream_read_kernel, reinterpret_cast<const uint4 *>(p), bytes / 16, sink);
    }
    return err == cudaSuccess ? VOXZIP_OK : VOXZIP_ECUDA;
}
