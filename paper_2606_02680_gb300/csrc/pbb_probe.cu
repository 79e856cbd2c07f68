// pbb_stream_read: a read-only HBM streaming kernel, the roof a decode step is
// measured against next to the copy bandwidth.
//
// A decode step reads its K/V support and writes almost nothing (the fp32
// output and one ring row per (sequence, KV head)), so its ceiling is the DRAM
// read bandwidth, which is higher than the bandwidth of a copy (a copy turns
// the bus around between reads and writes). The probe reads the way the decode
// kernels do: one lane per CTA streams the buffer in 16 KiB bulk copies
// (cp.async.bulk) into an 8-stage shared-memory ring whose stages complete on
// mbarriers, one CTA per SM, each CTA taking every gridDim-th chunk. The data is
// never looked at; every wait is bounded, and a wait that runs out sets a bit
// in *sink instead of hanging. A tail shorter than a chunk is read by plain
// loads. No counterpart in the paper.
#include <cuda_runtime.h>

#include <cstdint>

#include "pbb.h"
#include "pbb_device.cuh"

namespace {

constexpr int kProbeChunk = 16384;                   // bytes per bulk copy
constexpr int kProbeStages = 8;                      // copies in flight per CTA
constexpr unsigned long long kProbeLimitNs = 1000000000ull;

__global__ void __launch_bounds__(32) stream_read_kernel(const unsigned char* __restrict__ p, size_t bytes,
                                                         unsigned long long* sink)
{
    extern __shared__ __align__(128) unsigned char ring[];
    __shared__ __align__(8) uint64_t full[kProbeStages];
    const size_t chunks = bytes / kProbeChunk;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kProbeStages; ++s) pbb::mbar_init(&full[s], 1);
        pbb::fence_mbar_init();
        uint32_t k = 0;
        bool ok = true;
        for (size_t c = blockIdx.x; c < chunks; c += gridDim.x, ++k) {
            const int s = k % kProbeStages;
            if (k >= kProbeStages &&
                !pbb::mbar_wait(&full[s], static_cast<uint32_t>(((k / kProbeStages) - 1) & 1u), kProbeLimitNs)) {
                ok = false;
                break;
            }
            pbb::mbar_expect_tx(&full[s], kProbeChunk);
            pbb::bulk_g2s(ring + s * kProbeChunk, p + c * kProbeChunk, kProbeChunk, &full[s]);
        }
        // every copy lands before the CTA (and its shared memory) goes away
        const uint32_t first = k > kProbeStages ? k - kProbeStages : 0;
        for (uint32_t j = first; j < k; ++j)
            if (!pbb::mbar_wait(&full[j % kProbeStages], static_cast<uint32_t>((j / kProbeStages) & 1u), kProbeLimitNs))
                ok = false;
        if (!ok) atomicOr(sink, 1ull << 63);
    }
    if (blockIdx.x == 0) {  // the tail after the last whole chunk, 16 bytes per lane
        uint32_t acc = 0;
        for (size_t i = chunks * kProbeChunk + 16 * threadIdx.x; i < bytes; i += 16 * blockDim.x) {
            const uint4 v = __ldcs(reinterpret_cast<const uint4*>(p + i));
            acc ^= v.x ^ v.y ^ v.z ^ v.w;
        }
        if (acc != 0) atomicXor(sink, static_cast<unsigned long long>(acc));
    }
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
    constexpr int smem = kProbeChunk * kProbeStages;
    if (cudaFuncSetAttribute(stream_read_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return PBB_ERR_CUDA;
    stream_read_kernel<<<sms, 32, smem, stream>>>(static_cast<const unsigned char*>(buf), bytes, sink);
    return cudaGetLastError() == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}
