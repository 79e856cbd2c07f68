// C ABI of libpbb (declared in include/pbb.h): argument checking, the split
// plan, the per-device workspace, and dispatch to the kernels in pbb_decode.cu.
#include <cuda_runtime.h>

#include <atomic>
#include <climits>
#include <cstdint>
#include <map>
#include <mutex>
#include <utility>

#include "pbb.h"
#include "pbb_forward_plan.h"
#include "pbb_internal.h"

namespace {

constexpr int kMaxDevices = 64;
constexpr int kMaxBlock = 1 << 20;

// Library-owned scratch of one (device, stream): the work-queue control words
// and one counter per (sequence, KV head), all of which read zero between
// steps, and the split partials. Steps issued on one stream run in order, so
// they never use a workspace at the same time; steps on different streams get
// different workspaces and may overlap on the GPU.
struct Workspace {
    int* counters = nullptr;  // [0, 2): queue control; then one per (sequence, KV head)
    size_t counter_cap = 0;   // ints allocated
    float* parts = nullptr;
    size_t parts_bytes = 0;
};

using WsKey = std::pair<int, uintptr_t>;  // (device, stream handle)

std::mutex g_mutex;
std::map<WsKey, Workspace> g_ws;  // guarded by g_mutex; entries are never erased
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

// Decode steps: groups 1, 2, 4, 6 and 8 (6, the paper's models with 12 query heads on 2 KV
// heads, runs on the group-8 kernel with two padded heads).
int check_group(int Hq, int Hkv)
{
    if (Hq <= 0 || Hkv <= 0) return PBB_ERR_INVALID_ARG;
    if (Hq % Hkv != 0) return PBB_ERR_UNSUPPORTED;
    const int g = Hq / Hkv;
    if (g != 1 && g != 2 && g != 4 && g != 6 && g != 8) return PBB_ERR_UNSUPPORTED;
    return PBB_OK;
}

// The whole-sequence kernels stack G heads x 128/G positions as 128 rows: G must divide 128.
int check_group_sequence(int Hq, int Hkv)
{
    const int rc = check_group(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    return (Hq / Hkv) == 6 ? PBB_ERR_UNSUPPORTED : PBB_OK;
}

// The group G a decode kernel runs, which lays out the split partials: the tensor-core kernel
// always runs 8 query columns, the CUDA-core kernel runs a group of 6 as 8. plan_split takes
// the real group.
int kernel_group(const pbb::DecodeArgs& a, int elem)
{
    if (pbb::use_tensor_cores(a, elem)) return 8;
    return a.gq == 6 ? 8 : a.gq;
}

// An upper bound of kernel_group for every step of this group.
int max_kernel_group(int group) { return (group == 6 || pbb::tc_group(group)) ? 8 : group; }

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

// The split plan of the CUDA-core kernel. Whole supports are the cheapest work
// items there (no cross-CTA combine), but a batch of P supports on G resident
// CTAs leaves P mod G supports for a last round; when that round would leave
// more than half the CTAs idle, those last supports are split into about
// G / (P mod G) chunks each, so the step ends on small items. A batch with
// fewer supports than CTAs splits every support so that there are about G
// items. Chunks never hold less than kMinChunkBytes of K+V (below that the
// combine costs more than the parallel streaming saves). Measured on GB300 at
// 512 supports on 456 CTAs, splitting every support into 2-4 chunks was 5-25 %
// slower than running them whole, while splitting only the last round's
// supports paid for long supports (see below).
//
// The tensor-core kernel ends items on a separate epilogue warp, so a split
// item costs its consumers little; its plan cuts every support into chunks of
// about (supports x mean support) / (PBB_TC_ROUNDS x G) keys, and at least
// PBB_TC_MIN_CHUNK_KB of K+V, so the persistent grid balances on small items and
// the step does not end on a few CTAs streaming long supports alone. A positive
// pbb_set_chunk_keys override splits every support into chunks of that many
// keys, for either kernel.
#ifndef PBB_MIN_CHUNK_KB
#define PBB_MIN_CHUNK_KB 64
#endif
#ifndef PBB_TC_ROUNDS
#define PBB_TC_ROUNDS 4
#endif
// Smallest chunk of the tensor-core plan, in KiB of K+V: smaller chunks cost more in item
// starts and split combines than they gain in balance (measured on GB300 at batch 64: 448 keys
// of d 128 beat 128-288 keys at B 512 and B 1024).
#ifndef PBB_TC_MIN_CHUNK_KB
#define PBB_TC_MIN_CHUNK_KB 224
#endif

int min_split_keys(int d, int elem, int tile)
{
    constexpr int kMinChunkBytes = PBB_MIN_CHUNK_KB * 1024;
    const int k = kMinChunkBytes / (2 * d * elem);
    return k < tile ? tile : k;
}

}  // namespace

namespace pbb {

SplitPlan plan_split(int batch, int Hkv, int d, int B, int elem, int group, int window)
{
    SplitPlan sp{0, 0, 1};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) dev = 0;
    const int tile = pbb::tile_keys(elem, d, group);
    const bool tc = pbb::tensor_core_shape(batch, Hkv, d, B, elem, group, window);
    // keys of the longest support in the kernel's key space: B-1 for PBB (phase B-1), w-1 for a
    // window of w; the tensor-core kernel counts a window's run from the tile-aligned slot below
    // its start, up to tile-1 keys more
    const int span = window > 0 ? window - 1 + (tc && window > 1 ? tile - 1 : 0) : B - 1;
    const int max_keys = span > 0 ? span : 1;
    const long long pairs = static_cast<long long>(batch) * Hkv;
    const int over = g_chunk_override.load();
    if (over > 0) {
        sp.whole = 0;
        int chunk = static_cast<int>(round_up(static_cast<size_t>(over), static_cast<size_t>(tile)));
        sp.chunk = chunk;
        sp.nchunk = (max_keys + chunk - 1) / chunk;
        return sp;
    }
    auto whole_plan = [&]() {
        sp.whole = static_cast<int>(pairs);
        sp.chunk = static_cast<int>(round_up(static_cast<size_t>(max_keys), static_cast<size_t>(tile)));
        sp.nchunk = 1;
        return sp;
    };
    auto chunks_of = [&](long long chunk) {
        const int min_keys = tc ? (PBB_TC_MIN_CHUNK_KB * 1024) / (2 * d * elem) : min_split_keys(d, elem, tile);
        if (chunk < min_keys) chunk = min_keys;
        chunk = static_cast<long long>(round_up(static_cast<size_t>(chunk), static_cast<size_t>(tile)));
        if (chunk >= max_keys) return whole_plan();
        sp.whole = 0;
        sp.chunk = static_cast<int>(chunk);
        sp.nchunk = (max_keys + sp.chunk - 1) / sp.chunk;
        return sp;
    };
    int per_sm = pbb::decode_ctas_per_sm(batch, Hkv, elem, d, group, B, window);
    if (per_sm <= 0) per_sm = 1;
    const long long G = static_cast<long long>(sm_count(dev)) * per_sm;
    if (tc) {
        // mean ring keys of a support: (3h+1)/2 - 1 for PBB at a uniform phase (App. F.1), w-1
        // for a window
        const long long mean = window > 0 ? window - 1 : (3LL * B) / 4;
        const long long want = static_cast<long long>(PBB_TC_ROUNDS) * G;
        return chunks_of((pairs * (mean > 0 ? mean : 1) + want - 1) / want);
    }
    auto finish = [&](long long split) {
        const long long max_split = (max_keys + min_split_keys(d, elem, tile) - 1) / min_split_keys(d, elem, tile);
        if (split > max_split) split = max_split;
        if (split < 1) split = 1;
        int chunk = static_cast<int>((max_keys + split - 1) / split);
        chunk = static_cast<int>(round_up(static_cast<size_t>(chunk), static_cast<size_t>(tile)));
        sp.chunk = chunk;
        sp.nchunk = (max_keys + chunk - 1) / chunk;
        if (sp.nchunk <= 1) {  // nothing to split
            sp.whole = static_cast<int>(pairs);
            sp.nchunk = 1;
        }
    };
    if (pairs >= G) {
        const long long R = pairs % G;
        // Splitting the last round pays only for long supports (measured: +29 % at B 4096 and
        // +6 % at B 2048, but -12 to -15 % at B <= 1024).
        const bool long_supports = max_keys >= 2047;
        if (R == 0 || 2 * R > G || !long_supports) return whole_plan();
        sp.whole = static_cast<int>(pairs - R);
        finish((G + R - 1) / R);
    } else {
        sp.whole = 0;
        finish(pairs > 0 ? (G + pairs - 1) / pairs : 1);
    }
    return sp;
}

}  // namespace pbb

namespace {

// Bytes of split partials for a step: per (split support, chunk, head) d floats
// of unnormalised output, then 2 floats (max, sum).
size_t parts_bytes(int batch, int Hkv, int d, int group, const pbb::SplitPlan& sp)
{
    const size_t split_pairs = static_cast<size_t>(batch) * Hkv - static_cast<size_t>(sp.whole);
    const size_t parts = split_pairs * sp.nchunk * group;
    return round_up(parts * d * sizeof(float), 256) + parts * 2 * sizeof(float);
}

// Make the workspace of (device `dev`, `stream`) hold `pairs` counters and
// `pbytes` bytes of partials, and return it. Allocating is refused while
// `stream` is being captured. Growth is rare (the first steps of a larger
// shape, or pbb_reserve_workspace) and waits for the whole device, so that no
// step still in flight, on any stream, can read a buffer it frees. Caller
// holds g_mutex.
int grow_workspace(int dev, cudaStream_t stream, size_t pairs, size_t pbytes, Workspace** out)
{
    Workspace& ws = g_ws[WsKey(dev, reinterpret_cast<uintptr_t>(stream))];
    *out = &ws;
    if (ws.counter_cap >= pairs && ws.parts_bytes >= pbytes) return PBB_OK;
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream, &cap) != cudaSuccess) return PBB_ERR_CUDA;
    if (cap != cudaStreamCaptureStatusNone) return PBB_ERR_WORKSPACE;
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

// Longest-first order of whole supports (DecodeArgs::order): on the tensor-core kernel, when every
// support is one work item and the step gives each resident CTA at least PBB_TC_ORDER_ROUNDS of
// them. A step of fewer rounds is latency-bound, and the ordering kernel would add a launch to it.
#ifndef PBB_TC_ORDER_ROUNDS
#define PBB_TC_ORDER_ROUNDS 4
#endif
bool support_order_pays(const pbb::DecodeArgs& a, int elem, size_t pairs, int dev)
{
    if (PBB_TC_ORDER_ROUNDS <= 0 || static_cast<size_t>(a.whole) != pairs || !pbb::use_tensor_cores(a, elem)) return false;
    const int per_sm = pbb::decode_ctas_per_sm(a.batch, a.Hkv, elem, a.d, a.gq, a.B, a.window);
    const size_t resident = static_cast<size_t>(sm_count(dev)) * (per_sm > 0 ? per_sm : 1);
    return pairs >= static_cast<size_t>(PBB_TC_ORDER_ROUNDS) * resident;
}

int decode_impl(const void* q, const void* k_new, const void* v_new, void* k_ring, void* v_ring,
                const int32_t* pos, float* out, int batch, int Hq, int Hkv, int d, int B,
                int window, pbb_dtype dt, cudaStream_t stream, int pos_batch = 0)
{
    int rc = check_shape(batch, Hkv, d, B, dt);
    if (rc != PBB_OK) return rc;
    if (window < 0 || window > B) return PBB_ERR_INVALID_ARG;
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
    a.gq = Hq / Hkv;
    a.window = window;
    a.pos_batch = pos_batch > 0 ? pos_batch : batch;
    const pbb::SplitPlan sp = pbb::plan_split(batch, Hkv, d, B, elem, Hq / Hkv, window);
    a.whole = sp.whole;
    a.chunk = sp.chunk;
    a.nchunk = sp.nchunk;
    a.timeout_ns = g_timeout_ns.load();
    if (a.nchunk > 65535) return PBB_ERR_UNSUPPORTED;
    const size_t pairs = static_cast<size_t>(batch) * Hkv;
    const size_t items = static_cast<size_t>(sp.whole) + (pairs - static_cast<size_t>(sp.whole)) * sp.nchunk;
    if (items > static_cast<size_t>(INT_MAX)) return PBB_ERR_UNSUPPORTED;
    a.total_items = static_cast<int>(items);
    const int group = kernel_group(a, elem);
    const bool order = support_order_pays(a, elem, pairs, dev);
    {
        const size_t pbytes = static_cast<size_t>(sp.whole) < pairs ? parts_bytes(batch, Hkv, d, group, sp) : 0;
        std::lock_guard<std::mutex> lock(g_mutex);
        Workspace* ws = nullptr;
        rc = grow_workspace(dev, stream, pairs + 2 + (order ? static_cast<size_t>(batch) : 0), pbytes, &ws);
        if (rc != PBB_OK) return rc;
        const size_t parts = (pairs - static_cast<size_t>(sp.whole)) * a.nchunk * group;
        a.ctl = ws->counters;
        a.counters = ws->counters + 2;
        if (pbytes > 0) {
            a.part_o = ws->parts;
            a.part_ml = reinterpret_cast<float*>(reinterpret_cast<char*>(ws->parts) +
                                                 round_up(parts * d * sizeof(float), 256));
        }
        if (order) {  // the sequences, longest support first, after the per-support counters
            int* ord = ws->counters + 2 + pairs;
            if (pbb::launch_support_order(a, ord, stream) != cudaSuccess) return PBB_ERR_CUDA;
            a.order = ord;
        }
        // launched with the lock held: a call on another host thread that grows a workspace
        // frees the old buffers only after its cudaDeviceSynchronize, which waits for this launch
        return pbb::launch_decode(a, elem, stream) == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
    }
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

int pbb_reserve_workspace(int max_batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype, cudaStream_t stream)
{
    int rc = check_shape(max_batch, Hkv, d, B, dtype);
    if (rc != PBB_OK) return rc;
    rc = check_group(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    const int elem = elem_size(dtype);
    const int group = max_kernel_group(Hq / Hkv);
    // Every batch up to max_batch (the plan's split depends on the batch), for
    // PBB steps and for window steps with window = B.
    size_t need = 0;
    for (int bsz = 1; bsz <= max_batch; ++bsz) {
        for (int window : {0, B}) {
            const pbb::SplitPlan sp = pbb::plan_split(bsz, Hkv, d, B, elem, Hq / Hkv, window);
            if (static_cast<size_t>(sp.whole) >= static_cast<size_t>(bsz) * Hkv) continue;
            const size_t w = parts_bytes(bsz, Hkv, d, group, sp);
            if (w > need) need = w;
        }
    }
    std::lock_guard<std::mutex> lock(g_mutex);
    Workspace* ws = nullptr;
    // per-support counters, the queue words and the longest-first order of the sequences
    return grow_workspace(dev, stream, static_cast<size_t>(max_batch) * Hkv + 2 + static_cast<size_t>(max_batch), need,
                          &ws);
}

int pbb_decode_step(const void* q, const void* k_new, const void* v_new, void* k_ring,
                    void* v_ring, const int32_t* pos, float* out, int batch, int Hq, int Hkv,
                    int d, int B, cudaStream_t stream)
{
    return decode_impl(q, k_new, v_new, k_ring, v_ring, pos, out, batch, Hq, Hkv, d, B, 0, PBB_BF16,
                       stream);
}

int pbb_decode_step_f32(const float* q, const float* k_new, const float* v_new, float* k_ring,
                        float* v_ring, const int32_t* pos, float* out, int batch, int Hq,
                        int Hkv, int d, int B, cudaStream_t stream)
{
    return decode_impl(q, k_new, v_new, k_ring, v_ring, pos, out, batch, Hq, Hkv, d, B, 0, PBB_F32,
                       stream);
}

int pbb_decode_step_layers(const void* q, const void* k_new, const void* v_new, void* k_ring, void* v_ring,
                           const int32_t* pos, float* out, int layers, int batch, int Hq, int Hkv, int d, int B,
                           pbb_dtype dtype, cudaStream_t stream)
{
    if (layers < 1 || batch < 0) return PBB_ERR_INVALID_ARG;
    if (static_cast<long long>(layers) * batch > 65535) return PBB_ERR_UNSUPPORTED;
    return decode_impl(q, k_new, v_new, k_ring, v_ring, pos, out, layers * batch, Hq, Hkv, d, B, 0, dtype,
                       stream, batch);
}

int pbb_swa_decode_step(const void* q, const void* k_new, const void* v_new, void* k_ring,
                        void* v_ring, const int32_t* pos, float* out, int batch, int Hq, int Hkv,
                        int d, int B, int window, pbb_dtype dtype, cudaStream_t stream)
{
    if (window < 1) return PBB_ERR_INVALID_ARG;
    return decode_impl(q, k_new, v_new, k_ring, v_ring, pos, out, batch, Hq, Hkv, d, B, window,
                       dtype, stream);
}

int pbb_forward(const void* q, const void* k, const void* v, void* out, float* lse, int batch, int Hq,
                int Hkv, int n, int d, int B, pbb_dtype out_dtype, cudaStream_t stream)
{
    int rc = check_shape(batch, Hkv, d, B, PBB_BF16);
    if (rc != PBB_OK) return rc;
    rc = check_group_sequence(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    if (n < 0 || elem_size(out_dtype) == 0) return PBB_ERR_INVALID_ARG;
    if (batch == 0 || n == 0) return PBB_OK;
    // TMA row coordinates are 32-bit: every (sequence, head, position) row must fit
    if (static_cast<long long>(batch) * Hq * n >= (1LL << 31)) return PBB_ERR_UNSUPPORTED;
    if (!q || !k || !v || !out) return PBB_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(out, 16) ||
        (lse != nullptr && !aligned(lse, 4)))
        return PBB_ERR_INVALID_ARG;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    pbb::ForwardArgs a{};
    a.q = q;
    a.k = k;
    a.v = v;
    a.out = out;
    a.lse = lse;
    a.batch = batch;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.n = n;
    a.d = d;
    a.B = B;
    a.out_f32 = out_dtype == PBB_F32 ? 1 : 0;
    a.timeout_ns = g_timeout_ns.load();
    return pbb::launch_forward(a, stream) == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}

int pbb_plan_forward(int batch, int Hq, int Hkv, int n, int d, int B, int* keys_per_tile, int* ctas_per_sm)
{
    if (!keys_per_tile || !ctas_per_sm) return PBB_ERR_INVALID_ARG;
    int rc = check_shape(batch, Hkv, d, B, PBB_BF16);
    if (rc != PBB_OK) return rc;
    rc = check_group_sequence(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    if (n < 0) return PBB_ERR_INVALID_ARG;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    pbb::ForwardArgs a{};
    a.batch = batch;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.n = n;
    a.d = d;
    a.B = B;
    pbb::ForwardPlan plan{};
    if (pbb::plan_forward(a, &plan) != cudaSuccess) return PBB_ERR_CUDA;
    *keys_per_tile = plan.keys_per_tile;
    *ctas_per_sm = plan.ctas_per_sm;
    return PBB_OK;
}

int pbb_plan_forward_query_tiles(int batch, int Hq, int Hkv, int n, int d, int B)
{
    int rc = check_shape(batch, Hkv, d, B, PBB_BF16);
    if (rc != PBB_OK) return rc;
    rc = check_group_sequence(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    if (n < 0) return PBB_ERR_INVALID_ARG;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    pbb::ForwardArgs a{};
    a.batch = batch;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.n = n;
    a.d = d;
    a.B = B;
    int tiles = 0;
    if (pbb::plan_forward_query_tiles(a, &tiles) != cudaSuccess) return PBB_ERR_CUDA;
    return tiles;
}

int pbb_backward(const void* q, const void* k, const void* v, const void* out, const void* dout, const float* lse,
                 float* delta, float* dq, float* dk, float* dv, int batch, int Hq, int Hkv, int n, int d, int B,
                 cudaStream_t stream)
{
    int rc = check_shape(batch, Hkv, d, B, PBB_BF16);
    if (rc != PBB_OK) return rc;
    rc = check_group_sequence(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    if (n < 0) return PBB_ERR_INVALID_ARG;
    if (batch == 0 || n == 0) return PBB_OK;
    if (static_cast<long long>(batch) * Hq * n >= (1LL << 31)) return PBB_ERR_UNSUPPORTED;
    if (!q || !k || !v || !out || !dout || !lse || !delta || !dq || !dk || !dv) return PBB_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(out, 16) || !aligned(dout, 16) ||
        !aligned(lse, 4) || !aligned(delta, 4) || !aligned(dq, 16) || !aligned(dk, 16) || !aligned(dv, 16))
        return PBB_ERR_INVALID_ARG;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    pbb::BackwardArgs a{};
    a.q = q;
    a.k = k;
    a.v = v;
    a.out = out;
    a.dout = dout;
    a.lse = lse;
    a.delta = delta;
    a.dq = dq;
    a.dk = dk;
    a.dv = dv;
    a.batch = batch;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.n = n;
    a.d = d;
    a.B = B;
    a.timeout_ns = g_timeout_ns.load();
    return pbb::launch_backward(a, stream) == cudaSuccess ? PBB_OK : PBB_ERR_CUDA;
}

int pbb_ring_from_sequence(const void* k, const void* v, int n, void* k_ring, void* v_ring, int batch,
                           int Hkv, int d, int B, pbb_dtype dtype, cudaStream_t stream)
{
    int rc = check_shape(batch, Hkv, d, B, dtype);
    if (rc != PBB_OK) return rc;
    if (n < 0) return PBB_ERR_INVALID_ARG;
    if (batch == 0) return PBB_OK;
    if (!k_ring || !v_ring || (n > 0 && (!k || !v))) return PBB_ERR_INVALID_ARG;
    if (!aligned(k_ring, 16) || !aligned(v_ring, 16) || (n > 0 && (!aligned(k, 16) || !aligned(v, 16))))
        return PBB_ERR_INVALID_ARG;
    return pbb::launch_seq_ring(k, v, k_ring, v_ring, batch, Hkv, n, B, d * elem_size(dtype), stream) ==
                   cudaSuccess
               ? PBB_OK
               : PBB_ERR_CUDA;
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
    int status = 0, fwd_status = 0, bwd_status = 0;
    if (pbb::read_and_clear_status(&status, stream) != cudaSuccess) return PBB_ERR_CUDA;
    if (pbb::read_and_clear_forward_status(&fwd_status) != cudaSuccess) return PBB_ERR_CUDA;
    if (pbb::read_and_clear_backward_status(&bwd_status) != cudaSuccess) return PBB_ERR_CUDA;
    if (status == pbb::kDevOk && (fwd_status != pbb::kDevOk || bwd_status != pbb::kDevOk))
        return PBB_ERR_DEVICE_TIMEOUT;  // forward and backward kernels only time out
    if (status == pbb::kDevOk) return PBB_OK;
    {
        // An aborted step can leave split counters behind: zero them in every workspace of
        // this device.
        std::lock_guard<std::mutex> lock(g_mutex);
        for (auto& kv : g_ws) {
            if (kv.first.first != dev || !kv.second.counters) continue;
            if (cudaMemset(kv.second.counters, 0, kv.second.counter_cap * sizeof(int)) != cudaSuccess)
                return PBB_ERR_CUDA;
        }
        if (cudaDeviceSynchronize() != cudaSuccess) return PBB_ERR_CUDA;
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

int pbb_set_kernel(int kernel)
{
    if (kernel != PBB_KERNEL_AUTO && kernel != PBB_KERNEL_CUDA_CORES && kernel != PBB_KERNEL_TENSOR_CORES)
        return PBB_ERR_INVALID_ARG;
    return pbb::set_kernel_choice(kernel);
}

int pbb_plan_chunk_keys(int batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype)
{
    if (check_shape(batch, Hkv, d, B, dtype) != PBB_OK || check_group(Hq, Hkv) != PBB_OK) return 0;
    int dev = 0;
    if (current_device(&dev) != PBB_OK) return 0;
    return pbb::plan_split(batch, Hkv, d, B, elem_size(dtype), Hq / Hkv, 0).chunk;
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
    a.gq = Hq / Hkv;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.d = d;
    a.B = B;
    const pbb::SplitPlan sp = pbb::plan_split(batch, Hkv, d, B, elem_size(dtype), Hq / Hkv, 0);
    a.chunk = sp.chunk;
    return pbb::use_tensor_cores(a, elem_size(dtype)) ? PBB_KERNEL_TENSOR_CORES : PBB_KERNEL_CUDA_CORES;
}

int pbb_plan_support_order(int batch, int Hq, int Hkv, int d, int B, int window, pbb_dtype dtype)
{
    int rc = check_shape(batch, Hkv, d, B, dtype);
    if (rc != PBB_OK) return rc;
    rc = check_group(Hq, Hkv);
    if (rc != PBB_OK) return rc;
    if (window < 0 || window > B) return PBB_ERR_INVALID_ARG;
    int dev = 0;
    rc = current_device(&dev);
    if (rc != PBB_OK) return rc;
    const int elem = elem_size(dtype);
    pbb::DecodeArgs a{};
    a.batch = batch;
    a.gq = Hq / Hkv;
    a.Hq = Hq;
    a.Hkv = Hkv;
    a.d = d;
    a.B = B;
    a.window = window;
    const pbb::SplitPlan sp = pbb::plan_split(batch, Hkv, d, B, elem, Hq / Hkv, window);
    a.whole = sp.whole;
    a.chunk = sp.chunk;
    a.nchunk = sp.nchunk;
    return support_order_pays(a, elem, static_cast<size_t>(batch) * Hkv, dev) ? 1 : 0;
}

const char* pbb_error_string(int code)
{
    switch (code) {
        case PBB_OK: return "ok";
        case PBB_ERR_INVALID_ARG: return "invalid argument (null or misaligned pointer, negative size, window outside [1, B])";
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
