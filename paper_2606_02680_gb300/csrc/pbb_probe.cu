// pbb_stream_read: a read-only HBM streaming kernel, the roof a decode step is
// measured against next to the copy bandwidth.
//
// A decode step reads its K/V support and writes almost nothing (the fp32
// output and one ring row per (sequence, KV head)), so its ceiling is the
// DRAM read bandwidth, which is higher than the bandwidth of a copy (a copy
// turns the bus around between reads and writes). This kernel reads every
// 16-byte word of a buffer exactly once with streaming (evict-first) loads,
// four independent loads in flight per thread, and folds the words into one
// 64-bit xor so that no load can be dropped. No counterpart in the paper.
#include <cuda_runtime.h>

#include <cstdint>

#include "pbb.h"

namespace {

constexpr int kProbeThreads = 512;
constexpr int kProbeCtasPerSm = 4;

__global__ void __launch_bounds__(kProbeThreads) stream_read_kernel(const uint4* __restrict__ p, size_t n,
                                                                    unsigned long long* sink)
{
    const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
    size_t i = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    uint32_t acc = 0;
    for (; i + 3 * stride < n; i += 4 * stride) {
        const uint4 a = __ldcs(p + i);
        const uint4 b = __ldcs(p + i + stride);
        const uint4 c = __ldcs(p + i + 2 * stride);
        const uint4 d = __ldcs(p + i + 3 * stride);
        acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w ^ c.x ^ c.y ^ c.z ^ c.w ^ d.x ^ d.y ^ d.z ^ d.w;
    }
    for (; i < n; i += stride) {
        const uint4 a = __ldcs(p + i);
        acc ^= a.x ^ a.y ^ a.z ^ a.w;
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) acc ^= __shfl_xor_sync(0xffffffffu, acc, off);
    if ((threadIdx.x & 31) == 0 && acc != 0) atomicXor(sink, static_cast<unsigned long long>(acc));
}

}  // namespace

extern "C" int pbb_stream_read(const void* buf, size_t bytes, unsigned long long* sink, cudaStream_t stream)
{
    if (bytes == 0) return PBB_OK;
    if (!buf || !sink || (reinterpret_cast<uintptr_t>(buf) % 16) != 0 || (bytes % 16) != 0 ||
        (reinterpret_cast<uintptr_t>(sink) % 8) != 0)
        return PBB_ERR_INVALID_ARG;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        return PBB_ERR_CUDA;
    stream_read_kernel<<<sms * kProbeCtasPerSm, kProbeThreads, 0, stream>>>(static_cast<const uint4*>(buf),
                                                                           bytes / 16, sink);
    return cudaGetLastError() == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}
