// C ABI of libpbb (declared in include/pbb.h): argument checking, the split
// plan, the per-device workspace, and dispatch to the kernels in pbb_decode.cu.
#include <cuda_runtime.h>

#include <atomic>
#include <climits>
#include <cstdint>
#include <mutex>

#include "pbb.h"
#include "pbb_internal.h"

namespace {

constexpr int kMaxDevices = 64;
constexpr int kMaxBlock = 1 << 20;

// Library-owned scratch of one device: the work-queue control words and one
// counter per (sequence, KV head), all of which read zero between steps, and
// the split partials.
struct Workspace {
    int* counters = nullptr;  // [0, 2): queue control; then one per (sequence, KV head)
    size_t counter_cap = 0;   // ints allocated
    float* parts = nullptr;
    size_t parts_bytes = 0;
};

std::mutex g_mutex;
Workspace g_ws[kMaxDevices];
int g_sms[kMaxDevices] = {};
std::atomic<unsigned long long> g_timeout_ns{1000000000ull};
std::atomic<int> g_chunk_override{0};

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int elem_size(pbb_dtype dt) { return dt == PBB_BF16 ? 2 : (dt == PBB_F32 ? 4 : 0); }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Shape checks shared by every entry point (see include/pbb.h).
int check_shape(int batch, int Hkv, int d, int B, pbb_dtype dt)
{
    if (batch < 0 || Hkv <= 0 || d <= 0 || B <= 0) return PBB_ERR_INVALID_ARG;
    if (elem_size(dt) == 0) return PBB_ERR_INVALID_ARG;
    if ((B % 2) != 0 || B < 2 || B > kMaxBlock) return PBB_ERR_UNSUPPORTED;
    if (d != 64 && d != 128) return PBB_ERR_UNSUPPORTED;
    if (batch > 65535 || Hkv > 65535) return PBB_ERR_UNSUPPORTED;
    return PBB_OK;
}

int check_group(int Hq, int Hkv)
{
    if (Hq <= 0 || Hkv <= 0) return PBB_ERR_INVALID_ARG;
    if (Hq % Hkv != 0) return PBB_ERR_UNSUPPORTED;
    const int g = Hq / Hkv;
    if (g != 1 && g != 2 && g != 4 && g != 8) return PBB_ERR_UNSUPPORTED;
    return PBB_OK;
}

int current_device(int* dev)
{
    if (cudaGetDevice(dev) != cudaSuccess) return PBB_ERR_CUDA;
    if (*dev < 0 || *dev >= kMaxDevices) return PBB_ERR_UNSUPPORTED;
    return PBB_OK;
}

int sm_count(int dev)
{
    if (g_sms[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
        g_sms[dev] = n;
    }
    return g_sms[dev];
}

// Ring keys of the support per work item. The support of a (sequence, KV
// head) has at most B-1 ring keys besides the current token. Without an
// override the plan splits supports only when there are fewer of them than
// resident CTAs, into at most as many items as there are CTAs, and never into
// chunks of less than kMinChunkBytes of K+V, below which the combine would cost
// more than the parallel streaming saves. Measured on GB300 at 512 supports
// (batch 64 x 8 KV heads, or 256 x 2) on 456 resident CTAs, splitting into 2-4
// chunks was 5-25 % slower than running them whole (the per-item merge and the
// cross-CTA combine cost more than the shorter tail saves).
int plan_chunk(int batch, int Hkv, int d, int B, int elem, int group, int dev)
{
    const int tile = pbb::tile_keys(elem, d, group);
    const int max_keys = B - 1;
    int chunk;
    const int over = g_chunk_override.load();
    if (over > 0) {
        chunk = over;
    } else {
        constexpr int kWaves = 1;
        constexpr int kMinChunkBytes = 64 * 1024;
        const long long pairs = static_cast<long long>(batch) * Hkv;
        int per_sm = pbb::decode_ctas_per_sm(elem, d, group, B);
        if (per_sm <= 0) per_sm = 1;
        const long long want = static_cast<long long>(kWaves) * sm_count(dev) * per_sm;
        long long split = pairs > 0 ? (want + pairs - 1) / pairs : 1;
        int min_keys = kMinChunkBytes / (2 * d * elem);
        if (min_keys < tile) min_keys = tile;
        const long long max_split = (max_keys + min_keys - 1) / min_keys;
        if (split > max_split) split = max_split;
        if (split < 1) split = 1;
        chunk = static_cast<int>((max_keys + split - 1) / split);
    }
    chunk = static_cast<int>(round_up(static_cast<size_t>(chunk), static_cast<size_t>(tile)));
    if (chunk < tile) chunk = tile;
    return chunk;
}

// Bytes of split partials for a step: per (sequence, KV head, chunk, head)
// d floats of unnormalised output, then 2 floats (max, sum).
size_t parts_bytes(int batch, int Hkv, int d, int group, int nchunk)
{
    const size_t parts = static_cast<size_t>(batch) * Hkv * nchunk * group;
    return round_up(parts * d * sizeof(float), 256) + parts * 2 * sizeof(float);
}

// Make the workspace of device `dev` hold `pairs` counters and `pbytes` bytes
// of partials. Allocating is refused while `stream` is being captured.
// Caller holds g_mutex.
int grow_workspace(int dev, size_t pairs, size_t pbytes, cudaStream_t stream, bool check_capture)
{
    Workspace& ws = g_ws[dev];
    if (ws.counter_cap >= pairs && ws.parts_bytes >= pbytes) return PBB_OK;
    if (check_capture) {
        cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
        if (cudaStreamIsCapturing(stream, &cap) != cudaSuccess) return PBB_ERR_CUDA;
        if (cap != cudaStreamCaptureStatusNone) return PBB_ERR_WORKSPACE;
    }
    // Steps in flight may still use the old buffers.
    if (cudaDeviceSynchronize() != cudaSuccess) return PBB_ERR_CUDA;
    if (ws.counter_cap < pairs) {
        int* c = nullptr;
        if (cudaMalloc(&c, pairs * sizeof(int)) != cudaSuccess) return PBB_ERR_CUDA;
        if (cudaMemset(c, 0, pairs * sizeof(int)) != cudaSuccess) {
            cudaFree(c);
            return PBB_ERR_CUDA;
        }
        cudaFree(ws.counters);
        ws.counters = c;
        ws.counter_cap = pairs;
    }
    if (pbytes > 0 && ws.parts_bytes < pbytes) {
        void* p = nullptr;
        if (cudaMalloc(&p, pbytes) != cudaSuccess) return PBB_ERR_CUDA;
        cudaFree(ws.parts);
        ws.parts = static_cast<float*>(p);
        ws.parts_bytes = pbytes;
    }
    return cudaDeviceSynchronize() == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}

int decode_impl(const void* q, const void* k_new, const void* v_new, void* k_ring, void* v_ring,
                const int32_t* pos, float* out, int batch, int Hq, int Hkv, int d, int B,
                pbb_dtype dt, cudaStream_t stream)
{
    int rc = check_shape(batch, Hkv, d, B, dt);
    if (rc != PBB_OK) return rc;
    rc = check_group(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    if (batch == 0) return PBB_OK;
    if (!q || !k_new || !v_new || !k_ring || !v_ring || !pos || !out) return PBB_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k_new, 16) || !aligned(v_new, 16) || !aligned(k_ring, 16) ||
        !aligned(v_ring, 16) || !aligned(out, 16) || !aligned(pos, 4))
        return PBB_ERR_INVALID_ARG;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    const int elem = elem_size(dt);
    const int group = Hq / Hkv;

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
    a.chunk = plan_chunk(batch, Hkv, d, B, elem, group, dev);
    a.nchunk = (B - 1 + a.chunk - 1) / a.chunk;
    if (a.nchunk < 1) a.nchunk = 1;
    a.timeout_ns = g_timeout_ns.load();
    if (a.nchunk > 65535) return PBB_ERR_UNSUPPORTED;
    const size_t pairs = static_cast<size_t>(batch) * Hkv;
    a.total_items = static_cast<int>(pairs * a.nchunk);
    if (pairs * a.nchunk > static_cast<size_t>(INT_MAX)) return PBB_ERR_UNSUPPORTED;
    {
        const size_t pbytes = a.nchunk > 1 ? parts_bytes(batch, Hkv, d, group, a.nchunk) : 0;
        std::lock_guard<std::mutex> lock(g_mutex);
        rc = grow_workspace(dev, pairs + 2, pbytes, stream, true);
        if (rc != PBB_OK) return rc;
        const size_t parts = pairs * a.nchunk * group;
        a.ctl = g_ws[dev].counters;
        a.counters = g_ws[dev].counters + 2;
        if (a.nchunk > 1) {
            a.part_o = g_ws[dev].parts;
            a.part_ml = reinterpret_cast<float*>(reinterpret_cast<char*>(g_ws[dev].parts) +
                                                 round_up(parts * d * sizeof(float), 256));
        }
    }
    return pbb::launch_decode(a, elem, stream) == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}

}  // namespace

extern "C" {

size_t pbb_ring_bytes(int batch, int Hkv, int d, int B, pbb_dtype dtype)
{
    if (batch < 0 || Hkv <= 0 || d <= 0 || B <= 0 || elem_size(dtype) == 0) return 0;
    return static_cast<size_t>(batch) * Hkv * B * d * elem_size(dtype);
}

int pbb_ring_alloc(void** k_ring, void** v_ring, int batch, int Hkv, int d, int B,
                   pbb_dtype dtype, cudaStream_t stream)
{
    if (!k_ring || !v_ring) return PBB_ERR_INVALID_ARG;
    *k_ring = nullptr;
    *v_ring = nullptr;
    int rc = check_shape(batch, Hkv, d, B, dtype);
    if (rc != PBB_OK) return rc;
    const size_t bytes = pbb_ring_bytes(batch, Hkv, d, B, dtype);
    if (bytes == 0) return PBB_ERR_INVALID_ARG;
    void* k = nullptr;
    void* v = nullptr;
    if (cudaMallocAsync(&k, bytes, stream) != cudaSuccess) return PBB_ERR_CUDA;
    if (cudaMallocAsync(&v, bytes, stream) != cudaSuccess) {
        cudaFreeAsync(k, stream);
        return PBB_ERR_CUDA;
    }
    if (cudaMemsetAsync(k, 0, bytes, stream) != cudaSuccess ||
        cudaMemsetAsync(v, 0, bytes, stream) != cudaSuccess) {
        cudaFreeAsync(k, stream);
        cudaFreeAsync(v, stream);
        return PBB_ERR_CUDA;
    }
    *k_ring = k;
    *v_ring = v;
    return PBB_OK;
}

int pbb_ring_free(void* k_ring, void* v_ring, cudaStream_t stream)
{
    int rc = PBB_OK;
    if (k_ring && cudaFreeAsync(k_ring, stream) != cudaSuccess) rc = PBB_ERR_CUDA;
    if (v_ring && cudaFreeAsync(v_ring, stream) != cudaSuccess) rc = PBB_ERR_CUDA;
    return rc;
}

int pbb_ring_prefill(const void* k_hist, const void* v_hist, const int32_t* pos, void* k_ring,
                     void* v_ring, int batch, int Hkv, int d, int B, pbb_dtype dtype,
                     cudaStream_t stream)
{
    int rc = check_shape(batch, Hkv, d, B, dtype);
    if (rc != PBB_OK) return rc;
    if (batch == 0) return PBB_OK;
    if (!k_hist || !v_hist || !pos || !k_ring || !v_ring) return PBB_ERR_INVALID_ARG;
    if (!aligned(k_hist, 16) || !aligned(v_hist, 16) || !aligned(k_ring, 16) ||
        !aligned(v_ring, 16) || !aligned(pos, 4))
        return PBB_ERR_INVALID_ARG;
    const int row = d * elem_size(dtype);
    return pbb::launch_prefill(k_hist, v_hist, pos, k_ring, v_ring, batch, Hkv, B, row, stream) ==
                   cudaSuccess
               ? PBB_OK
               : PBB_ERR_CUDA;
}

int pbb_reserve_workspace(int max_batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype)
{
    int rc = check_shape(max_batch, Hkv, d, B, dtype);
    if (rc != PBB_OK) return rc;
    rc = check_group(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    const int elem = elem_size(dtype);
    const int group = Hq / Hkv;
    // Every batch up to max_batch: the plan's split shrinks as the batch grows.
    size_t need = 0;
    for (int bsz = 1; bsz <= max_batch; ++bsz) {
        const int chunk = plan_chunk(bsz, Hkv, d, B, elem, group, dev);
        const int nchunk = (B - 1 + chunk - 1) / chunk;
        if (nchunk <= 1) continue;
        const size_t w = parts_bytes(bsz, Hkv, d, group, nchunk);
        if (w > need) need = w;
    }
    std::lock_guard<std::mutex> lock(g_mutex);
    return grow_workspace(dev, static_cast<size_t>(max_batch) * Hkv + 2, need, nullptr, false);
}

int pbb_decode_step(const void* q, const void* k_new, const void* v_new, void* k_ring,
                    void* v_ring, const int32_t* pos, float* out, int batch, int Hq, int Hkv,
                    int d, int B, cudaStream_t stream)
{
    return decode_impl(q, k_new, v_new, k_ring, v_ring, pos, out, batch, Hq, Hkv, d, B, PBB_BF16,
                       stream);
}

int pbb_decode_step_f32(const float* q, const float* k_new, const float* v_new, float* k_ring,
                        float* v_ring, const int32_t* pos, float* out, int batch, int Hq,
                        int Hkv, int d, int B, cudaStream_t stream)
{
    return decode_impl(q, k_new, v_new, k_ring, v_ring, pos, out, batch, Hq, Hkv, d, B, PBB_F32,
                       stream);
}

int pbb_advance_positions(int32_t* pos, int batch, cudaStream_t stream)
{
    if (batch < 0) return PBB_ERR_INVALID_ARG;
    if (batch == 0) return PBB_OK;
    if (!pos || !aligned(pos, 4)) return PBB_ERR_INVALID_ARG;
    return pbb::launch_advance(pos, batch, stream) == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}

int pbb_get_device_status(cudaStream_t stream)
{
    int dev = 0;
    int rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    int status = 0;
    if (pbb::read_and_clear_status(&status, stream) != cudaSuccess) return PBB_ERR_CUDA;
    if (status == pbb::kDevOk) return PBB_OK;
    {
        // An aborted step can leave split counters behind: zero them.
        std::lock_guard<std::mutex> lock(g_mutex);
        Workspace& ws = g_ws[dev];
        if (ws.counters) {
            if (cudaMemset(ws.counters, 0, ws.counter_cap * sizeof(int)) != cudaSuccess) return PBB_ERR_CUDA;
            if (cudaDeviceSynchronize() != cudaSuccess) return PBB_ERR_CUDA;
        }
    }
    return status == pbb::kDevTimeout ? PBB_ERR_DEVICE_TIMEOUT : PBB_ERR_DEVICE_POSITION;
}

int pbb_set_wait_timeout_ns(unsigned long long ns)
{
    g_timeout_ns.store(ns);
    return PBB_OK;
}

int pbb_set_chunk_keys(int keys)
{
    if (keys < 0) return PBB_ERR_INVALID_ARG;
    return g_chunk_override.exchange(keys);
}

int pbb_plan_chunk_keys(int batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype)
{
    if (check_shape(batch, Hkv, d, B, dtype) != PBB_OK || check_group(Hq, Hkv) != PBB_OK) return 0;
    int dev = 0;
    if (current_device(&dev) != PBB_OK) return 0;
    return plan_chunk(batch, Hkv, d, B, elem_size(dtype), Hq / Hkv, dev);
}

int pbb_plan_kernel(int batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype)
{
    int rc = check_shape(batch, Hkv, d, B, dtype);
    if (rc != PBB_OK) return rc;
    rc = check_group(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    pbb::DecodeArgs a{};
    a.batch = batch;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.d = d;
    a.B = B;
    a.chunk = plan_chunk(batch, Hkv, d, B, elem_size(dtype), Hq / Hkv, dev);
    return pbb::use_tensor_cores(a, elem_size(dtype)) ? PBB_KERNEL_TENSOR_CORES : PBB_KERNEL_CUDA_CORES;
}

const char* pbb_error_string(int code)
{
    switch (code) {
        case PBB_OK: return "ok";
        case PBB_ERR_INVALID_ARG: return "invalid argument (null or misaligned pointer, negative size)";
        case PBB_ERR_UNSUPPORTED: return "unsupported shape (B odd or out of range, Hq % Hkv != 0, group or d not supported)";
        case PBB_ERR_CUDA: return "CUDA runtime error";
        case PBB_ERR_DEVICE_TIMEOUT: return "a kernel's bounded wait on a bulk copy ran out";
        case PBB_ERR_WORKSPACE: return "workspace too small while the stream is captured; call pbb_reserve_workspace first";
        case PBB_ERR_DEVICE_POSITION: return "a kernel saw a negative position; that sequence was skipped";
        case PBB_ERR_SCRATCH_LIMIT: return "the step needs more scratch than pbb_decode_step_noalloc's fixed array holds; use pbb_decode_step";
        default: return "unknown error code";
    }
}

}  // extern "C"
