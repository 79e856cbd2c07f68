// pbb_decode_step_noalloc: the bf16 decode step with its split scratch in a
// fixed device array compiled into the library, so that the call allocates no
// memory at all.
//
// Who needs it: callers that must not, or cannot, allocate device memory
// while they run decode steps. Examples are a serving runtime that hands all
// of HBM to its own pool up front and forbids any other allocation, and
// latency-critical loops where the device-wide synchronisation a cudaMalloc
// can bring is unacceptable. pbb_decode_step keeps its
// scratch in a workspace it grows with cudaMalloc on demand; this variant
// never calls cudaMalloc, cudaFree or any allocating library routine.
//
// The scratch is `g_noalloc_scratch` below: kNoallocScratchBytes per GPU
// that loads the library, held until the process exits. Host code cannot use
// the array's name as a device address (on the host it is only a stand-in
// symbol), so the first call on each device, with that device current, asks
// the runtime for the real address with cudaGetSymbolAddress and caches it.
// Make that first call before any stream capture.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <mutex>

#include "pbb.h"
#include "pbb_internal.h"

namespace {

constexpr size_t kNoallocScratchBytes = PBB_NOALLOC_SCRATCH_BYTES;
constexpr size_t kCounterBytes = 256 * 1024;  // queue words and counters: up to 65,534 (sequence, KV head) pairs
constexpr int kMaxDevices = 64;

// Scratch: [0, kCounterBytes) the work-queue words and the per-(sequence, KV
// head) counters, then the split partials.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

std::mutex g_setup_mutex;
unsigned char* g_scratch_addr[kMaxDevices] = {};

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Device address of the scratch array on the current device (set-up on first use).
int scratch_address(int dev, unsigned char** out)
{
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (g_scratch_addr[dev] == nullptr) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr)
            return PBB_ERR_CUDA;
        g_scratch_addr[dev] = static_cast<unsigned char*>(p);
    }
    *out = g_scratch_addr[dev];
    return PBB_OK;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

extern "C" int pbb_decode_step_noalloc(const void* q, const void* k_new, const void* v_new,
                                       void* k_ring, void* v_ring, const int32_t* pos, float* out,
                                       int batch, int Hq, int Hkv, int d, int B,
                                       cudaStream_t stream)
{
    // Same argument rules as pbb_decode_step (include/pbb.h).
    if (batch < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || B <= 0) return PBB_ERR_INVALID_ARG;
    if ((B % 2) != 0 || B > (1 << 20) || (d != 64 && d != 128) || batch > 65535 || Hkv > 65535)
        return PBB_ERR_UNSUPPORTED;
    if (Hq % Hkv != 0) return PBB_ERR_UNSUPPORTED;
    const int gq = Hq / Hkv;
    if (gq != 1 && gq != 2 && gq != 4 && gq != 6 && gq != 8) return PBB_ERR_UNSUPPORTED;
    if (batch == 0) return PBB_OK;
    if (!q || !k_new || !v_new || !k_ring || !v_ring || !pos || !out) return PBB_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(k_ring, 16) ||
        !aligned(v_ring, 16) || !aligned(out, 16) || !aligned(pos, 4))
        return PBB_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return PBB_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return PBB_ERR_UNSUPPORTED;

    pbb::DecodeArgs a{};
    a.q = q;
    a.k_new = k_new;
    a.v_new = v_new;
    a.k_ring = k_ring;
    a.v_ring = v_ring;
    a.pos = pos;
    a.out = out;
    a.batch = batch;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.d = d;
    a.B = B;
    a.gq = gq;
    a.pos_batch = batch;
    const pbb::SplitPlan sp = pbb::plan_split(batch, Hkv, d, B, 2, gq, 0);  // the same plan as pbb_decode_step
    if (sp.chunk <= 0) return PBB_ERR_CUDA;
    a.whole = sp.whole;
    a.chunk = sp.chunk;
    a.nchunk = sp.nchunk;
    if (a.nchunk > 65535) return PBB_ERR_UNSUPPORTED;
    a.timeout_ns = 1000000000ull;

    // the partials' head layout is the launched kernel's group: 8 on the tensor cores, and 8
    // for six heads on the CUDA cores
    const int group = (pbb::use_tensor_cores(a, 2) || gq == 6) ? 8 : gq;
    const size_t pairs = static_cast<size_t>(batch) * Hkv;
    const size_t parts = (pairs - static_cast<size_t>(sp.whole)) * a.nchunk * group;
    const size_t o_bytes = round_up(parts * d * sizeof(float), 256);
    const size_t need = kCounterBytes + o_bytes + parts * 2 * sizeof(float);
    if ((pairs + 2) * sizeof(int) > kCounterBytes || need > kNoallocScratchBytes)
        return PBB_ERR_SCRATCH_LIMIT;
    a.total_items = static_cast<int>(static_cast<size_t>(sp.whole) + (pairs - static_cast<size_t>(sp.whole)) * a.nchunk);
    unsigned char* base = nullptr;
    const int rc = scratch_address(dev, &base);
    if (rc != PBB_OK) return rc;
    a.ctl = reinterpret_cast<int*>(base);
    a.counters = reinterpret_cast<int*>(base) + 2;
    if (parts > 0) {
        a.part_o = reinterpret_cast<float*>(base + kCounterBytes);
        a.part_ml = reinterpret_cast<float*>(base + kCounterBytes + o_bytes);
    }
    // The array keeps whatever the previous call left: the queue words and the
    // counters must start at zero.
    if (cudaMemsetAsync(a.ctl, 0, (pairs + 2) * sizeof(int), stream) != cudaSuccess) return PBB_ERR_CUDA;
    return pbb::launch_decode(a, 2, stream) == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}
