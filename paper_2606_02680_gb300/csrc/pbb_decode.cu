// Kernels of the PBB decode step for sm_103a.
//
// The support. For a sequence whose current token is at t = p + r (block
// start p, phase r, B = 2h) the support is the interval [a(t), t]
// (Eq. pbb_relay). Apart from the current token, which comes from
// k_new/v_new, it occupies at most two contiguous runs of ring slots
// (Appendix F.1): a bridge phase (p > 0, r < h) reads slots h..B-1 (the
// previous block's tail, positions p-h..p-1) and then 0..r-1; the other
// phases read 0..r-1. In position order, ring key i of the support lives in
// slot (base + i) mod B, base = h for a bridge phase and 0 otherwise.
//
// Work items. An item covers one (sequence, KV head) support, or a chunk of C
// ring keys of one, for all G = Hq/Hkv query heads of the group, so each K/V
// byte is read from HBM once per step. The first `whole` supports are items of
// their own; each later support is split into chunks (the plan splits only
// the supports of a last, partly filled round, or all supports of a batch too
// small to fill the GPU). Chunk 0 of a support also carries the current token:
// it appends k_new/v_new to slot r (never a slot that is read) and folds the
// token into its softmax. Chunks past the end of a short support are skipped.
//
// Persistent CTAs, as many per SM as fit. A producer lane takes items from a device-wide
// queue (an atomic counter) and streams them without a break: every item
// becomes tiles of TK keys, and each tile lands in one stage of a 3-stage
// shared-memory ring through 1-D bulk copies (cp.async.bulk, completion
// counted in bytes on the stage's "full" mbarrier). The first tile of an item
// also brings the item's G query rows and, for chunk 0, the new K/V rows; a
// tile that straddles the end of the ring is fetched as two copies. The
// producer writes a small descriptor per stage (item, keys, first/last flags)
// before arming the barrier, so consumers learn item boundaries in order.
//
// Eight consumer warps share every tile (KW = TK/8 keys each) and keep
// independent fp32 online-softmax states in the base-2 domain (the scale
// log2(e)/sqrt(d) is folded into q), releasing the stage through its "empty"
// mbarrier:
//   scores: KL lanes per key (8, or 16 for G = 8 so the query registers fit);
//           a lane holds the queries of d/KL dims of all G heads and the
//           partial dot products are combined by a reduce-scatter over the
//           KL lanes, so each lane ends with the score of one (key, head);
//           products are packed fp32x2 FMAs;
//   P.V:    each lane owns d/32 output dims of all G heads and reads a key's
//           weights from shared memory as ready fp32x2 pairs.
// At an item's last tile the consumer warps merge their states in shared
// memory (Eq. lse). A single-item support writes `out`; otherwise the item
// stores its partial (max, sum, output) and the last item of the (sequence,
// KV head) to finish (an atomic counter, no spinning) fuses all partials in
// chunk order with Eq. (lse) and resets the counter, so results do not depend
// on scheduling. The last CTA to finish resets the queue.
//
// No wait can hang: waits on mbarriers and the consumers' software barrier are
// bounded by the global timer. A wait that runs out records kDevTimeout; the
// CTA then stops, waits (bounded) for the copies it issued and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <stdint.h>

#include <atomic>
#include <mutex>
#include <utility>

#include "pbb.h"
#include "pbb_device.cuh"
#include "pbb_internal.h"

namespace pbb {

__device__ int g_status;  // first device-side fault recorded, kDevOk if none

namespace {

// Launch shape. Chosen by measurement on GB300 (a sweep of consumer warps,
// tile bytes, stages and resident CTAs per SM); the macros let a build try
// other shapes without editing the kernel.
#ifndef PBB_CONSUMER_WARPS
#define PBB_CONSUMER_WARPS 4
#endif
#ifndef PBB_STAGES
#define PBB_STAGES 3
#endif
#ifndef PBB_TILE_BYTES
#define PBB_TILE_BYTES 8192
#endif
#ifndef PBB_TILE_BYTES_G8
#define PBB_TILE_BYTES_G8 8192
#endif
#ifndef PBB_MIN_CTAS
#define PBB_MIN_CTAS 3
#endif
#ifndef PBB_MIN_CTAS_G8
#define PBB_MIN_CTAS_G8 2
#endif
constexpr int kConsumers = PBB_CONSUMER_WARPS;   // warps that compute
constexpr int kThreads = (kConsumers + 1) * 32;  // plus one producer warp
constexpr int kStages = PBB_STAGES;
constexpr unsigned kFull = 0xffffffffu;
constexpr unsigned long long kGuardNs = 2000000000ull;  // waits only a broken GPU can exceed

enum : int { kFirst = 1, kLast = 2, kCurrent = 4, kEnd = 8 };

// Descriptor of the tile in one stage, written by the producer before it arms the stage.
struct __align__(16) TileMeta {
    int b, kvh, chunk, nk;  // item and ring keys in this tile
    int nch, r, flags, lo;  // chunks of the support, phase, kFirst/kLast/kCurrent/kEnd, and the
                            // first tile row in the support (tensor-core kernel; rows < lo masked)
};

// ---------------------------------------------------------- elements ----

template <int ELEM>
struct Elem;

template <>
struct Elem<2> {  // bf16: the high half of an fp32
    static __device__ __forceinline__ float to_float(const void* p)
    {
        return __bfloat162float(*static_cast<const __nv_bfloat16*>(p));
    }
    // Convert the 8 bf16 of a 16-byte vector.
    static __device__ __forceinline__ void vec16(const uint4& u, float* f)
    {
        const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            f[2 * i] = __uint_as_float(w[i] << 16);
            f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
        }
    }
};

template <>
struct Elem<4> {  // fp32
    static __device__ __forceinline__ float to_float(const void* p)
    {
        return *static_cast<const float*>(p);
    }
    static __device__ __forceinline__ void vec16(const uint4& u, float* f)
    {
        f[0] = __uint_as_float(u.x);
        f[1] = __uint_as_float(u.y);
        f[2] = __uint_as_float(u.z);
        f[3] = __uint_as_float(u.w);
    }
};

// Load N consecutive elements (N * ELEM in {4, 8, 16} bytes) as floats.
template <int ELEM, int N>
__device__ __forceinline__ void load_elems(const unsigned char* p, float* f)
{
    constexpr int BYTES = N * ELEM;
    if constexpr (BYTES == 16) {
        const uint4 u = *reinterpret_cast<const uint4*>(p);
        Elem<ELEM>::vec16(u, f);
    } else if constexpr (BYTES == 8) {
        const uint2 u = *reinterpret_cast<const uint2*>(p);
        if constexpr (ELEM == 2) {
            f[0] = __uint_as_float(u.x << 16);
            f[1] = __uint_as_float(u.x & 0xffff0000u);
            f[2] = __uint_as_float(u.y << 16);
            f[3] = __uint_as_float(u.y & 0xffff0000u);
        } else {
            f[0] = __uint_as_float(u.x);
            f[1] = __uint_as_float(u.y);
        }
    } else {
        static_assert(BYTES == 4, "row slice must be 4, 8 or 16 bytes");
        const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
        if constexpr (ELEM == 2) {
            f[0] = __uint_as_float(u << 16);
            f[1] = __uint_as_float(u & 0xffff0000u);
        } else {
            f[0] = __uint_as_float(u);
        }
    }
}

// --------------------------------------------------------- reductions ----

template <int N>
struct Log2 {
    static constexpr int value = (N <= 1) ? 0 : 1 + Log2<N / 2>::value;
};
template <>
struct Log2<1> {
    static constexpr int value = 0;
};

// Within each aligned group of KL lanes, every lane holds G partial sums, one
// per head, in a lane-specific order: position p holds head (myhead ^ p), where
// myhead = sub >> (log2 KL - log2 G). Each exchange step then keeps the first
// half of the positions and sends the second half, which are exactly the
// partner lane's first half, so no lane needs a select. Once a lane keeps one
// value the remaining steps are butterfly sums. Afterwards every lane holds the
// group's full sum for its own head.
template <int G, int KL>
__device__ __forceinline__ float reduce_scatter(float (&v)[G])
{
    int cnt = G;
#pragma unroll
    for (int lvl = KL / 2; lvl >= 1; lvl >>= 1) {
        if (cnt > 1) {
            const int half = cnt / 2;
#pragma unroll
            for (int i = 0; i < half; ++i) v[i] += __shfl_xor_sync(kFull, v[i + half], lvl);
            cnt = half;
        } else {
            v[0] += __shfl_xor_sync(kFull, v[0], lvl);
        }
    }
    return v[0];
}

// The ring keys of a support, i.e. all of it but the current token t (which
// comes from k_new/v_new). r = t mod B is the slot the step writes.
//   window == 0, PBB (Eq. pbb_relay, Appendix F.1): positions a(t) .. t-1,
//     n = h + r keys from slot h in a bridge phase (p > 0, r < h), else the r
//     keys of slots 0 .. r-1.
//   window == w in [1, B], the sliding window {t-w+1, ..., t} (Sec. 2.3):
//     n = min(t, w-1) keys from slot (t-n) mod B; the run may wrap past slot
//     B-1. Slot r holds position t-B <= t-w, outside the window.
// In both cases ring key i (position t-n+i) lives in slot (base + i) mod B.
__device__ __forceinline__ void support_keys(int t, int B, int window, int& r, int& n, int& base)
{
    const int blk = t / B;
    r = t - blk * B;
    if (window > 0) {
        n = min(t, window - 1);
        base = r - n;
        if (base < 0) base += B;
    } else {
        const int h = B >> 1;
        const bool bridge = (blk > 0) && (r < h);
        n = bridge ? h + r : r;
        base = bridge ? h : 0;
    }
}

// Barrier of the consumer warps through a shared-memory counter, bounded by
// `limit_ns` (a hardware named barrier could not be bounded). All lanes of all
// consumer warps call it; returns false if it gave up.
template <int NC>
__device__ __forceinline__ bool consumer_barrier(unsigned* count, volatile unsigned* gen, int lane,
                                                 unsigned long long limit_ns)
{
    bool ok = true;
    __syncwarp();
    if (lane == 0) {
        const unsigned g = *gen;
        __threadfence_block();
        if (atomicAdd(count, 1u) == NC - 1) {
            *count = 0;
            __threadfence_block();
            *gen = g + 1;
        } else {
            const unsigned long long t0 = global_ns();
            while (*gen == g) {
                if (global_ns() - t0 > limit_ns) {
                    ok = false;
                    break;
                }
            }
        }
        __threadfence_block();
    }
    return __shfl_sync(kFull, ok ? 1 : 0, 0) != 0;
}

// ------------------------------------------------------------ config ----

template <int ELEM, int D, int G>
struct Cfg {
    // resident CTAs per SM the registers and shared memory must allow
    static constexpr int MIN_CTAS = (G == 8) ? PBB_MIN_CTAS_G8 : PBB_MIN_CTAS;
    static constexpr int ROW = D * ELEM;                            // bytes of one K or V row
    static constexpr int KL = (G == 8 && ROW >= 256) ? 16 : 8;      // lanes per key, score phase
    static constexpr int KPS = 32 / KL;                             // keys per warp step
    static constexpr int MERGE = kConsumers * G * D * 4;            // per-warp outputs at a merge
    static constexpr int BUDGET = 218 * 1024 / MIN_CTAS;            // dynamic shared memory per CTA
    static constexpr int stage_bytes(int tile)
    {
        return (2 * tile + (G + 2) * ROW + 127) / 128 * 128;
    }
    // The requested K (and V) bytes per stage, halved until the stages and the
    // merge buffer fit the budget (fp32 rows are twice as wide).
    static constexpr int fit_tile(int tile)
    {
        while (kStages * stage_bytes(tile) + MERGE > BUDGET && tile > ROW * kConsumers * KPS) tile /= 2;
        return tile;
    }
    static constexpr int TILE_BYTES = fit_tile((G == 8) ? PBB_TILE_BYTES_G8 : PBB_TILE_BYTES);
    static constexpr int TK = TILE_BYTES / ROW;                     // keys per tile
    static constexpr int KW = TK / kConsumers;                      // keys per consumer warp per tile
    static constexpr int STEPS = KW / KPS;                          // score steps per tile
    static constexpr int VPL = ROW / (KL * 16);                     // 16-byte vectors per lane, score phase
    static constexpr int EPV = 16 / ELEM;                           // elements per 16-byte vector
    static constexpr int DPL = D / KL;                              // dims per lane, score phase
    static constexpr int PVD = D / 32;                              // dims per lane, P.V phase
    static constexpr int REP = Log2<KL>::value - Log2<G>::value;    // lanes per (key, head) = 2^REP
    static constexpr int KV = 2 * TK * ROW;                         // K tile then V tile
    static constexpr int Q_OFF = KV;                                // the item's G query rows
    static constexpr int KN_OFF = Q_OFF + G * ROW;                  // k_new row (chunk 0)
    static constexpr int VN_OFF = KN_OFF + ROW;                     // v_new row (chunk 0)
    static constexpr int STAGE = (VN_OFF + ROW + 127) / 128 * 128;
    static constexpr int SMEM = kStages * STAGE + MERGE;
    static_assert(KW % KPS == 0 && STEPS >= 1, "a warp needs whole score steps");
    static_assert(VPL >= 1 && VPL * EPV == DPL && (EPV % 2) == 0 && (PVD % 2) == 0, "lane slices");
    static_assert(REP >= 0, "group larger than the lanes of a key");
    static_assert(SMEM <= BUDGET, "shared memory budget (dynamic; the static part is a few KiB)");
};

// ----------------------------------------------------------- item end ----

// atomicAdd with acquire-release semantics at GPU scope (one round trip: it publishes the
// caller's earlier stores and sees the stores published before earlier updates).
__device__ __forceinline__ int atomic_add_acq_rel_gpu(int* p, int v)
{
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}


// End of a work item, run by all consumer threads: merge the consumer warps'
// (max, sum, output) states of the item (Eq. lse) from ml_s [NC][G] and
// merge_o [NC][G][D]; write `out` for an unsplit support, else the item's
// partial, and let the last item of the (sequence, KV head) to finish fuse all
// partials in chunk order. Returns false if a bounded barrier gave up.
template <int G, int D, int NC>
__device__ __forceinline__ bool finish_item(const DecodeArgs& a, const TileMeta& mt, size_t head, const float2* ml_s,
                                         float* merge_o, unsigned* sbar_count, volatile unsigned* sbar_gen,
                                         int* last_s, int tid, int lane, int warp)
{
    bool ok = consumer_barrier<NC>(sbar_count, sbar_gen, lane, kGuardNs);
    const int ctid = tid;  // 0 .. 32*NC-1 (consumer threads)
    const size_t part = (head - a.whole) * a.nchunk + mt.chunk;  // only split supports have partials
    if (ok) {
        for (int e = ctid; e < G * D; e += NC * 32) {
            const int j = e / D;
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < NC; ++w) M = fmaxf(M, ml_s[w * G + j].x);
            float L = 0.f, O = 0.f;
#pragma unroll
            for (int w = 0; w < NC; ++w) {
                const float sc = exp2f(ml_s[w * G + j].x - M);
                L = fmaf(ml_s[w * G + j].y, sc, L);
                O = fmaf(merge_o[(w * G) * D + e], sc, O);
            }
            if (mt.nch == 1) {
                if (j < a.gq) a.out[(static_cast<size_t>(mt.b) * a.Hq + static_cast<size_t>(mt.kvh) * a.gq) * D + e] = O / L;
            } else {
                a.part_o[part * G * D + e] = O;
                if ((e % D) == 0) reinterpret_cast<float2*>(a.part_ml)[part * G + j] = make_float2(M, L);
            }
        }
    }
    if (ok && mt.nch > 1) {
        // split combine (Eq. lse): the last item of this (sequence, KV head) fuses all partials.
        // The barrier orders every consumer thread's partial stores before thread 0's counter
        // update, which releases them to the GPU and, for the last item, acquires the other
        // items' partials (the semaphore pattern of a split-k reduction).
        ok = consumer_barrier<NC>(sbar_count, sbar_gen, lane, kGuardNs);
        if (ok && ctid == 0) *last_s = (atomic_add_acq_rel_gpu(a.counters + head, 1) == mt.nch - 1);
        ok = ok && consumer_barrier<NC>(sbar_count, sbar_gen, lane, kGuardNs);
        if (ok && *last_s) {
            const float* po = a.part_o + (head - a.whole) * a.nchunk * G * D;
            const float2* pml = reinterpret_cast<const float2*>(a.part_ml) + (head - a.whole) * a.nchunk * G;
            float* out_g = a.out + (static_cast<size_t>(mt.b) * a.Hq + static_cast<size_t>(mt.kvh) * a.gq) * D;
            if (mt.nch <= NC * D) {
                // weight of every (chunk, head) in shared memory: e^(m_c - M) / L, with M and
                // L reduced across the chunks by one warp per head
                float* wgt = merge_o;  // [nch][G], free after the barrier above
                for (int j = warp; j < G; j += NC) {
                    float M = -INFINITY;
                    for (int c = lane; c < mt.nch; c += 32) M = fmaxf(M, __ldcg(&pml[c * G + j]).x);
#pragma unroll
                    for (int off = 16; off >= 1; off >>= 1) M = fmaxf(M, __shfl_xor_sync(kFull, M, off));
                    float L = 0.f;
                    for (int c = lane; c < mt.nch; c += 32) {
                        const float2 ml = __ldcg(&pml[c * G + j]);
                        const float e = fast_exp2(ml.x - M);
                        wgt[c * G + j] = e;
                        L = fmaf(ml.y, e, L);
                    }
#pragma unroll
                    for (int off = 16; off >= 1; off >>= 1) L += __shfl_xor_sync(kFull, L, off);
                    const float inv = 1.f / L;
                    __syncwarp();
                    for (int c = lane; c < mt.nch; c += 32) wgt[c * G + j] *= inv;
                }
                ok = consumer_barrier<NC>(sbar_count, sbar_gen, lane, kGuardNs);
                if (ok) {
                    // four consecutive elements (one head: D is a multiple of 4) per thread, as
                    // 16-byte loads of every chunk's partial (partials and out are 16-byte aligned)
                    for (int e = 4 * ctid; e < a.gq * D; e += 4 * NC * 32) {  // the real query heads
                        const int j = e / D;
                        float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 8
                        for (int c = 0; c < mt.nch; ++c) {
                            const float4 p = __ldcg(reinterpret_cast<const float4*>(po + c * G * D + e));
                            const float w = wgt[c * G + j];
                            O.x = fmaf(p.x, w, O.x);
                            O.y = fmaf(p.y, w, O.y);
                            O.z = fmaf(p.z, w, O.z);
                            O.w = fmaf(p.w, w, O.w);
                        }
                        *reinterpret_cast<float4*>(out_g + e) = O;
                    }
                }
            } else {
                for (int e = ctid; e < a.gq * D; e += NC * 32) {  // the real query heads
                    const int j = e / D;
                    float M = -INFINITY;
                    for (int c = 0; c < mt.nch; ++c) M = fmaxf(M, __ldcg(&pml[c * G + j]).x);
                    float L = 0.f, O = 0.f;
                    for (int c = 0; c < mt.nch; ++c) {
                        const float2 ml = __ldcg(&pml[c * G + j]);
                        const float sc = fast_exp2(ml.x - M);
                        L = fmaf(ml.y, sc, L);
                        O = fmaf(__ldcg(po + c * G * D + e), sc, O);
                    }
                    out_g[e] = O / L;
                }
            }
            if (ctid == 0) a.counters[head] = 0;
        }
    }
    ok = ok && consumer_barrier<NC>(sbar_count, sbar_gen, lane, kGuardNs);  // merge buffers free again
    return ok;
}

// ------------------------------------------------------------ kernel ----

template <int ELEM, int D, int G>
__global__ void __launch_bounds__(kThreads, Cfg<ELEM, D, G>::MIN_CTAS) decode_kernel(const DecodeArgs a)
{
    using C = Cfg<ELEM, D, G>;
    extern __shared__ __align__(128) unsigned char dsmem[];
    __shared__ __align__(8) uint64_t full_bar[kStages];
    __shared__ __align__(8) uint64_t empty_bar[kStages];
    __shared__ TileMeta meta_s[kStages];
    __shared__ __align__(16) float p_s[kConsumers][C::KW][G];  // softmax weights of a tile
    __shared__ __align__(16) float alpha_s[kConsumers][G];     // rescale factors of a tile
    __shared__ float2 ml_s[kConsumers][G];
    __shared__ unsigned sbar_count;
    __shared__ volatile unsigned sbar_gen;
    __shared__ volatile int abort_s;
    __shared__ int last_s;
    __shared__ int issued_s;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
#pragma unroll
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], kConsumers);
        }
        fence_mbar_init();
        sbar_count = 0;
        sbar_gen = 0;
        abort_s = 0;
        issued_s = 0;
    }
    if (a.gq < G) {
        // a group of gq < G heads runs as G: the query rows gq .. G-1 of every stage are never
        // loaded and stay zero, so the padded heads compute finite values that are never written
        for (int s = 0; s < kStages; ++s)
            for (int x = threadIdx.x; x < (G - a.gq) * C::ROW / 16; x += blockDim.x)
                reinterpret_cast<uint4*>(dsmem + s * C::STAGE + C::Q_OFF + a.gq * C::ROW)[x] = make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();
    // the set-up above touches no global memory; everything below may read what the previous
    // grid of the stream wrote (rings, positions, the queue words)
    pdl_wait();
    pdl_launch_dependents();

    if (warp == kConsumers) {
        // ================= producer: one lane =================
        if (lane == 0) {
            int seq = 0;  // tiles issued so far (stage seq % kStages)
            bool ok = true;
            // the first item of a CTA is its index (no queue round trip before the first
            // tile); later ones come from the queue, which hands out items grid, grid+1, ...
            for (int item = blockIdx.x; ok && item < a.total_items;
                 item = static_cast<int>(gridDim.x) + atomicAdd(a.ctl, 1)) {
                // items [0, whole): whole supports; then nchunk chunks of each later support
                int pair, chunk;
                if (item < a.whole) {
                    pair = item;
                    chunk = 0;
                } else {
                    const int j = item - a.whole;
                    pair = a.whole + j / a.nchunk;
                    chunk = j % a.nchunk;
                }
                const int kvh = pair % a.Hkv, b = pair / a.Hkv;
                const int t = __ldg(a.pos + (b < a.pos_batch ? b : b % a.pos_batch));  // layers share positions
                if (t < 0) {
                    if (chunk == 0 && kvh == 0) atomicCAS(&g_status, kDevOk, kDevBadPosition);
                    continue;
                }
                const int B = a.B;
                int r, n, base;  // slot of t; ring keys of the support (positions t-n .. t-1); slot of key 0
                support_keys(t, B, a.window, r, n, base);
                const bool whole = pair < a.whole;
                const int csize = whole ? max(n, 1) : a.chunk;  // keys per chunk of this support
                const int nch = n > 0 ? (n + csize - 1) / csize : 1;
                if (chunk >= nch) continue;
                const int i0 = chunk * csize;
                const int i1 = min(i0 + csize, n);
                const int nkeys = max(i1 - i0, 0);
                const int ntiles = nkeys > 0 ? (nkeys + C::TK - 1) / C::TK : 1;
                const size_t head = static_cast<size_t>(b) * a.Hkv + kvh;
                const unsigned char* kring = static_cast<const unsigned char*>(a.k_ring) + head * B * C::ROW;
                const unsigned char* vring = static_cast<const unsigned char*>(a.v_ring) + head * B * C::ROW;
                for (int it = 0; it < ntiles; ++it, ++seq) {
                    const int s = seq % kStages;
                    if (seq >= kStages &&
                        !mbar_wait(&empty_bar[s], static_cast<uint32_t>((seq / kStages - 1) & 1), kGuardNs)) {
                        ok = false;
                        break;
                    }
                    if (abort_s) {
                        ok = false;
                        break;
                    }
                    const int k0 = i0 + it * C::TK;
                    const int nk = max(min(C::TK, i1 - k0), 0);
                    const bool first = it == 0;
                    const bool current = first && chunk == 0;
                    TileMeta mt;
                    mt.b = b;
                    mt.kvh = kvh;
                    mt.chunk = chunk;
                    mt.nk = nk;
                    mt.nch = nch;
                    mt.r = r;
                    mt.flags = (first ? kFirst : 0) | (it == ntiles - 1 ? kLast : 0) | (current ? kCurrent : 0);
                    mt.lo = 0;
                    meta_s[s] = mt;
                    unsigned char* st = dsmem + s * C::STAGE;
                    const uint32_t bytes = static_cast<uint32_t>(2 * nk * C::ROW + (first ? a.gq * C::ROW : 0) +
                                                                 (current ? 2 * C::ROW : 0));
                    fence_proxy_async();
                    mbar_expect_tx(&full_bar[s], bytes);  // arrives (release): the descriptor is visible
                    if (nk > 0) {
                        int slot = base + k0;
                        if (slot >= B) slot -= B;
                        const int len1 = min(nk, B - slot);
                        bulk_g2s(st, kring + static_cast<size_t>(slot) * C::ROW, len1 * C::ROW, &full_bar[s]);
                        bulk_g2s(st + C::TK * C::ROW, vring + static_cast<size_t>(slot) * C::ROW,
                                 len1 * C::ROW, &full_bar[s]);
                        if (len1 < nk) {  // wrapped past slot B-1: the rest starts at slot 0
                            bulk_g2s(st + len1 * C::ROW, kring, (nk - len1) * C::ROW, &full_bar[s]);
                            bulk_g2s(st + (C::TK + len1) * C::ROW, vring, (nk - len1) * C::ROW, &full_bar[s]);
                        }
                    }
                    if (first) {
                        const unsigned char* qg = static_cast<const unsigned char*>(a.q) +
                                                  (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(kvh) * a.gq) * C::ROW;
                        bulk_g2s(st + C::Q_OFF, qg, a.gq * C::ROW, &full_bar[s]);
                    }
                    if (current) {
                        bulk_g2s(st + C::KN_OFF, static_cast<const unsigned char*>(a.k_new) + head * C::ROW,
                                 C::ROW, &full_bar[s]);
                        bulk_g2s(st + C::VN_OFF, static_cast<const unsigned char*>(a.v_new) + head * C::ROW,
                                 C::ROW, &full_bar[s]);
                    }
                }
            }
            if (ok) {  // end-of-work descriptor: a plain arrival completes the stage's phase
                const int s = seq % kStages;
                if (seq >= kStages &&
                    !mbar_wait(&empty_bar[s], static_cast<uint32_t>((seq / kStages - 1) & 1), kGuardNs)) {
                    ok = false;
                } else {
                    TileMeta mt{};
                    mt.flags = kEnd;
                    meta_s[s] = mt;
                    mbar_arrive(&full_bar[s]);
                    ++seq;
                }
            }
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_status, kDevOk, kDevTimeout);
            }
            issued_s = seq;
        }
    } else {
        // ================= consumers =================
        const int sub = lane & (C::KL - 1), kq = lane / C::KL;
        const int myhead = sub >> C::REP;
        const bool primary = (sub & ((1 << C::REP) - 1)) == 0;
        const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
        float* merge_o = reinterpret_cast<float*>(dsmem + kStages * C::STAGE);  // [kConsumers][G][D]
        float2 qr[G][C::DPL / 2];  // this lane's query slice, scaled, as pairs
        float m_run = -INFINITY;   // running max of this lane's head (log2 domain)
        float l_run = 0.f;         // this lane's share of the running sum (primary lanes only)
        float2 o[G][C::PVD / 2];   // output dims lane*PVD .. +PVD of every head
#pragma unroll
        for (int j = 0; j < G; ++j)
#pragma unroll
            for (int x = 0; x < C::DPL / 2; ++x) qr[j][x] = make_float2(0.f, 0.f);

        for (int seq = 0;; ++seq) {
            const int s = seq % kStages;
            if (!mbar_wait(&full_bar[s], static_cast<uint32_t>((seq / kStages) & 1), a.timeout_ns)) {
                abort_s = 1;
                atomicCAS(&g_status, kDevOk, kDevTimeout);
                break;
            }
            const TileMeta mt = meta_s[s];
            if (mt.flags & kEnd) break;
            if (abort_s) break;
            const unsigned char* st = dsmem + s * C::STAGE;
            const size_t head = static_cast<size_t>(mt.b) * a.Hkv + mt.kvh;

            if (mt.flags & kFirst) {
                // the item's queries: position p of this lane holds head (myhead ^ p), the
                // order reduce_scatter expects; vector m covers dims (sub + KL*m)*EPV ...
#pragma unroll
                for (int p = 0; p < G; ++p)
#pragma unroll
                    for (int m = 0; m < C::VPL; ++m) {
                        float qf[C::EPV];
                        const uint4 u = *reinterpret_cast<const uint4*>(st + C::Q_OFF + (myhead ^ p) * C::ROW +
                                                                        (sub + C::KL * m) * 16);
                        Elem<ELEM>::vec16(u, qf);
#pragma unroll
                        for (int x = 0; x < C::EPV / 2; ++x)
                            qr[p][m * (C::EPV / 2) + x] = make_float2(qf[2 * x] * qscale, qf[2 * x + 1] * qscale);
                    }
                m_run = -INFINITY;
                l_run = 0.f;
#pragma unroll
                for (int j = 0; j < G; ++j)
#pragma unroll
                    for (int x = 0; x < C::PVD / 2; ++x) o[j][x] = make_float2(0.f, 0.f);
                if (mt.flags & kCurrent) {
                    if (warp == 0) {  // the current token seeds warp 0's softmax state
                        float kc[C::PVD], vc[C::PVD];
                        load_elems<ELEM, C::PVD>(st + C::KN_OFF + lane * C::PVD * ELEM, kc);
                        load_elems<ELEM, C::PVD>(st + C::VN_OFF + lane * C::PVD * ELEM, vc);
                        float zc[G];
#pragma unroll
                        for (int j = 0; j < G; ++j) {
                            float qf[C::PVD];
                            load_elems<ELEM, C::PVD>(st + C::Q_OFF + j * C::ROW + lane * C::PVD * ELEM, qf);
                            float acc = 0.f;
#pragma unroll
                            for (int x = 0; x < C::PVD; ++x) acc = fmaf(qf[x] * qscale, kc[x], acc);
#pragma unroll
                            for (int off = 16; off >= 1; off >>= 1) acc += __shfl_xor_sync(kFull, acc, off);
                            zc[j] = acc;
                        }
                        m_run = zc[0];
#pragma unroll
                        for (int j = 1; j < G; ++j)
                            if (myhead == j) m_run = zc[j];
                        l_run = (primary && kq == 0) ? 1.f : 0.f;
#pragma unroll
                        for (int j = 0; j < G; ++j)
#pragma unroll
                            for (int x = 0; x < C::PVD / 2; ++x) o[j][x] = make_float2(vc[2 * x], vc[2 * x + 1]);
                    }
                    if (warp == kConsumers - 1) {  // append: slot r of both rings <- the new rows
                        uint4* kd = reinterpret_cast<uint4*>(static_cast<unsigned char*>(a.k_ring) +
                                                             (head * a.B + mt.r) * C::ROW);
                        uint4* vd = reinterpret_cast<uint4*>(static_cast<unsigned char*>(a.v_ring) +
                                                             (head * a.B + mt.r) * C::ROW);
                        for (int x = lane; x < C::ROW / 16; x += 32) {
                            kd[x] = *reinterpret_cast<const uint4*>(st + C::KN_OFF + x * 16);
                            vd[x] = *reinterpret_cast<const uint4*>(st + C::VN_OFF + x * 16);
                        }
                    }
                }
            }

            const int nkw = min(max(mt.nk - warp * C::KW, 0), C::KW);
            if (nkw > 0) {
                const unsigned char* sK = st + warp * C::KW * C::ROW;
                const unsigned char* sV = st + (C::TK + warp * C::KW) * C::ROW;
                float zs[C::STEPS];
                float mx = -INFINITY;
#pragma unroll
                for (int stp = 0; stp < C::STEPS; ++stp) {
                    const int key = stp * C::KPS + kq;
                    float z = -INFINITY;
                    if (stp * C::KPS < nkw) {  // warp-uniform
                        float2 acc[G];
#pragma unroll
                        for (int j = 0; j < G; ++j) acc[j] = make_float2(0.f, 0.f);
#pragma unroll
                        for (int m = 0; m < C::VPL; ++m) {
                            float kf[C::EPV];
                            const uint4 u = *reinterpret_cast<const uint4*>(sK + key * C::ROW + (sub + C::KL * m) * 16);
                            Elem<ELEM>::vec16(u, kf);
#pragma unroll
                            for (int x = 0; x < C::EPV / 2; ++x) {
                                const float2 k2 = make_float2(kf[2 * x], kf[2 * x + 1]);
#pragma unroll
                                for (int j = 0; j < G; ++j)
                                    acc[j] = __ffma2_rn(qr[j][m * (C::EPV / 2) + x], k2, acc[j]);
                            }
                        }
                        float part[G];
#pragma unroll
                        for (int j = 0; j < G; ++j) part[j] = acc[j].x + acc[j].y;
                        const float zz = reduce_scatter<G, C::KL>(part);
                        z = key < nkw ? zz : -INFINITY;
                    }
                    zs[stp] = z;
                    mx = fmaxf(mx, z);
                }
#pragma unroll
                for (int off = C::KL; off < 32; off <<= 1) mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, off));
                const float m_new = fmaxf(m_run, mx);
                float lsum = 0.f;
#pragma unroll
                for (int stp = 0; stp < C::STEPS; ++stp) {
                    const float pz = fast_exp2(zs[stp] - m_new);
                    if (stp * C::KPS < nkw && primary) p_s[warp][stp * C::KPS + kq][myhead] = pz;
                    lsum += pz;
                }
                // rescale only when some head's running max moved (rare once it settles)
                const bool grew = m_new > m_run;
                if (__any_sync(kFull, grew)) {
                    const float alpha = fast_exp2(m_run - m_new);  // 2^-inf = 0 on the first keys
                    l_run *= alpha;
                    if (primary && kq == 0) alpha_s[warp][myhead] = alpha;
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < G; ++j) {
                        const float al = alpha_s[warp][j];
#pragma unroll
                        for (int x = 0; x < C::PVD / 2; ++x) o[j][x] = __fmul2_rn(o[j][x], make_float2(al, al));
                    }
                }
                l_run += primary ? lsum : 0.f;
                m_run = m_new;
                __syncwarp();
#pragma unroll 4
                for (int k = 0; k < nkw; ++k) {
                    float vf[C::PVD];
                    load_elems<ELEM, C::PVD>(sV + k * C::ROW + lane * C::PVD * ELEM, vf);
                    float pv[G];
#pragma unroll
                    for (int j = 0; j < G; ++j) pv[j] = p_s[warp][k][j];
#pragma unroll
                    for (int j = 0; j < G; ++j)
#pragma unroll
                        for (int x = 0; x < C::PVD / 2; ++x)
                            o[j][x] = __ffma2_rn(make_float2(pv[j], pv[j]), make_float2(vf[2 * x], vf[2 * x + 1]), o[j][x]);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty_bar[s]);
            if (!(mt.flags & kLast)) continue;

            // ---- end of the item: merge the consumer warps' states (Eq. lse)
            {
                float l = l_run;
#pragma unroll
                for (int off = C::KL; off < 32; off <<= 1) l += __shfl_xor_sync(kFull, l, off);
#pragma unroll
                for (int x = 1; x < (1 << C::REP); x <<= 1) l += __shfl_xor_sync(kFull, l, x);
                if (lane == (myhead << C::REP)) ml_s[warp][myhead] = make_float2(m_run, l);
            }
#pragma unroll
            for (int j = 0; j < G; ++j)
#pragma unroll
                for (int x = 0; x < C::PVD / 2; ++x)
                    *reinterpret_cast<float2*>(&merge_o[(warp * G + j) * D + lane * C::PVD + 2 * x]) = o[j][x];
            bool ok = finish_item<G, D, kConsumers>(a, mt, head, &ml_s[0][0], merge_o, &sbar_count, &sbar_gen,
                                                    &last_s, tid, lane, warp);
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_status, kDevOk, kDevTimeout);
                break;
            }
        }
    }
    __syncthreads();
    if (abort_s) {
        if (tid == 0) {
            // wait (bounded) for the last copy issued into each stage
            const int issued = issued_s;
            for (int s = 0; s < kStages && s < issued; ++s) {
                const int j = s + kStages * ((issued - 1 - s) / kStages);
                mbar_wait(&full_bar[s], static_cast<uint32_t>((j / kStages) & 1), kGuardNs);
            }
        }
        __syncthreads();
    }
    if (tid == 0) {  // the last CTA to finish resets the work queue for the next launch
        __threadfence();
        if (atomicAdd(a.ctl + 1, 1) == static_cast<int>(gridDim.x) - 1) {
            atomicExch(a.ctl, 0);
            atomicExch(a.ctl + 1, 0);
        }
    }
}

// ------------------------------------------------- tensor-core kernel ----
//
// GQA group 8 makes the score product a dense tile: for a block of 16 keys,
// S^T [16 keys x 8 heads] = K [16 x d] . Q^T [d x 8] is an mma.m16n8k16 chain
// over d, and the output O^T [d x 8 heads] += V^T [d x 16 keys] . P^T
// [16 keys x 8 heads] is one mma per 16 output dims. This kernel serves bf16
// steps with G = 8, or G = 4 and 6 with their query columns padded to 8 by
// zero rows (whose outputs are not written), and block sizes that are multiples
// of twice the tile. The step is bound by HBM (each K/V byte feeds 2G flops),
// so the warp-level mma is enough to keep up with the copies. Work items, the
// queue and the split are those of decode_kernel; per CTA:
//   - a producer warp (one lane) streams tiles of TK ring slots by 2-D TMA
//     copies with the 128-byte swizzle, one box per 64 columns. Tiles start at
//     multiples of TK in slot order and B is a multiple of 2 TK, so no box
//     crosses the end of a ring; a support whose run of slots starts or ends
//     inside a tile (a sliding window's run starts at any slot) masks the
//     tile's rows outside [lo, nk);
//   - two consumer warps take 16 rows of every tile each: A operands from
//     ldmatrix (K) and ldmatrix.trans (V^T), the Q^T operand from registers
//     loaded once per item; the scores (fp32) go through the online softmax;
//     the weights P are split into a bf16 high part and a bf16 low part
//     (p = hi + lo to about 2^-16) and both are multiplied, so P.V keeps
//     fp32-level accuracy; the C fragment of S^T becomes the B fragment of P^T
//     by an 8x8 movmatrix transpose;
//   - an epilogue warp ends the items. At an item's last tile the consumer
//     warps leave their (max, sum, output) states in one of two shared-memory
//     slots and go straight on to the next item's tiles; the epilogue warp
//     merges the states (Eq. lse), writes `out` or the item's split partial
//     and, for the last item of a split support to finish, fuses the partials
//     in chunk order. The item ends (shared-memory merges, global writes and
//     the L2 round trips of the split combine) thus overlap the streaming of
//     the next item instead of stalling it, which is what makes splitting
//     supports into chunks cheap enough to balance the persistent grid.
#ifndef PBB_TC_CONSUMER_WARPS
#define PBB_TC_CONSUMER_WARPS 2
#endif
#ifndef PBB_TC_STAGES
#define PBB_TC_STAGES 3
#endif
#ifndef PBB_TC_MIN_CTAS
#define PBB_TC_MIN_CTAS 3
#endif
constexpr int kTcConsumers = PBB_TC_CONSUMER_WARPS;
constexpr int kTcProducer = kTcConsumers;          // warp index of the producer
constexpr int kTcEpilogue = kTcConsumers + 1;      // warp index of the epilogue warp
constexpr int kTcThreads = (kTcConsumers + 2) * 32;
constexpr int kTcStages = PBB_TC_STAGES;
constexpr int kTcEpiSlots = 2;                     // item-end slots between consumers and epilogue

template <int D>
struct TcCfg {
    static constexpr int G = 8;
    static constexpr int ROW = D * 2;                      // bf16 row bytes
    static constexpr int BOXES = D / 64;                   // 64-column (128-byte) boxes per row
    static constexpr int TK = 16 * kTcConsumers;           // keys per tile: one m16 block per warp
    static constexpr int BOX_BYTES = TK * 128;             // one swizzled [TK rows x 128 B] box
    static constexpr int K_OFF = 0;
    static constexpr int V_OFF = BOXES * BOX_BYTES;
    static constexpr int Q_OFF = 2 * BOXES * BOX_BYTES;    // the item's 8 query rows (plain)
    static constexpr int KN_OFF = Q_OFF + G * ROW;         // k_new row (chunk 0)
    static constexpr int VN_OFF = KN_OFF + ROW;            // v_new row (chunk 0)
    static constexpr int STAGE = (VN_OFF + ROW + 1023) / 1024 * 1024;  // boxes stay 1024-aligned
    static constexpr int EPI_O = kTcConsumers * G * D * 4; // one slot: the consumer warps' outputs
    static constexpr int SMEM = kTcStages * STAGE + kTcEpiSlots * EPI_O + 1024;  // + alignment slack
    static constexpr int KSTEPS = D / 16;                  // k-steps of the score chain
    static constexpr int MTILES = D / 16;                  // 16-dim tiles of the output
    static constexpr int PVD = D / 32;                     // dims per lane for the current token
    static_assert(BOX_BYTES % 1024 == 0, "swizzle atoms");
    static_assert(D % 128 == 0 || D == 64, "head sizes");
};

// Work item -> (support, chunk) on the tensor-core kernel. Items [0, whole) are whole supports,
// then the chunks of each later support together. PBB_TC_CHUNK_MAJOR = 1 orders the chunks
// chunk-major instead (chunk 0 of every split support, then chunk 1, ...), so the queue ends on
// the short remainders of the longest supports; measured on GB300 it lost 5 % at B 2048 (the
// chunks past short supports, which the producer skips at two L2 round trips each, then pile up
// at the end of the queue) and tied elsewhere. A support is (sequence, KV head).
#ifndef PBB_TC_CHUNK_MAJOR
#define PBB_TC_CHUNK_MAJOR 0
#endif
__device__ __forceinline__ void tc_item(const DecodeArgs& a, int item, int& pair, int& chunk)
{
    if (item < a.whole) {
        // whole supports, longest first when the host ordered them (every support whole)
        pair = a.order ? __ldg(a.order + item / a.Hkv) * a.Hkv + item % a.Hkv : item;
        chunk = 0;
        return;
    }
    const int j = item - a.whole;
    if (PBB_TC_CHUNK_MAJOR) {
        const int split = a.batch * a.Hkv - a.whole;  // supports that are split
        pair = a.whole + j % split;
        chunk = j / split;
    } else {
        pair = a.whole + j / a.nchunk;
        chunk = j % a.nchunk;
    }
}

// Index into pos[] of work item `item` (the layers of a multi-layer step share the positions of
// their sequences).
__device__ __forceinline__ int tc_item_seq(const DecodeArgs& a, int item)
{
    int pair, chunk;
    tc_item(a, item, pair, chunk);
    const int b = pair / a.Hkv;
    return b < a.pos_batch ? b : b % a.pos_batch;
}

// Wait for phase `parity` of `bar`, giving up when another warp of the CTA has aborted or after
// kGuardNs. Returns false if it gave up.
__device__ __forceinline__ bool mbar_wait_or_abort(uint64_t* bar, uint32_t parity, volatile int* abort_flag)
{
    if (mbar_test(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try(bar, parity)) {
        if (*abort_flag) return false;
        if (global_ns() - t0 > kGuardNs) return false;
    }
    return true;
}

// End of one work item, run by the 32 lanes of the epilogue warp: merge the NC consumer
// warps' (max, sum, output) states of the item (Eq. lse), from ml [NC][G] and o [NC][G][D];
// write `out` for an unsplit support, else the item's partial, and let the last item of the
// (sequence, KV head) to finish fuse all partials in chunk order (so results do not depend on
// scheduling). `o` serves as scratch for the combine weights afterwards.
template <int G, int D, int NC>
__device__ __forceinline__ void epilogue_item(const DecodeArgs& a, const TileMeta& mt, const float2* ml, float* o,
                                              int lane)
{
    constexpr int V4 = D / 4;         // float4 per head row
    constexpr int HPI = 32 / V4;      // head rows per warp iteration (1 at d = 128, 2 at d = 64)
    const size_t head = static_cast<size_t>(mt.b) * a.Hkv + mt.kvh;
    const bool split = mt.nch > 1;
    const size_t part = split ? (head - a.whole) * a.nchunk + mt.chunk : 0;
    const int c4 = lane % V4;
    float* out_g = a.out + (static_cast<size_t>(mt.b) * a.Hq + static_cast<size_t>(mt.kvh) * a.gq) * D;
#pragma unroll
    for (int j0 = 0; j0 < G; j0 += HPI) {
        const int j = j0 + lane / V4;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < NC; ++w) M = fmaxf(M, ml[w * G + j].x);
        float L = 0.f;
        float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int w = 0; w < NC; ++w) {
            const float2 mw = ml[w * G + j];
            const float sc = exp2f(mw.x - M);
            const float4 ow = reinterpret_cast<const float4*>(o + (w * G + j) * D)[c4];
            L = fmaf(mw.y, sc, L);
            O.x = fmaf(ow.x, sc, O.x);
            O.y = fmaf(ow.y, sc, O.y);
            O.z = fmaf(ow.z, sc, O.z);
            O.w = fmaf(ow.w, sc, O.w);
        }
        if (!split) {
            if (j < a.gq) {
                const float inv = 1.f / L;
                reinterpret_cast<float4*>(out_g + j * D)[c4] = make_float4(O.x * inv, O.y * inv, O.z * inv, O.w * inv);
            }
        } else {
            reinterpret_cast<float4*>(a.part_o + (part * G + j) * D)[c4] = O;
            if (c4 == 0) reinterpret_cast<float2*>(a.part_ml)[part * G + j] = make_float2(M, L);
        }
    }
    if (!split) return;
    // split combine (Eq. lse): the last item of this (sequence, KV head) fuses all partials.
    // The partial stores of every lane are ordered before lane 0's counter update by the
    // warp barrier, and the update releases them to the GPU (and, for the last item,
    // acquires the other items' partials) in one atomic, the semaphore pattern of a
    // split-k reduction; under a saturated memory system each L2 round trip costs
    // microseconds, so the combine issues its loads in as few rounds as it can.
    __syncwarp();
    int last = 0;
    if (lane == 0) last = (atomic_add_acq_rel_gpu(a.counters + head, 1) == mt.nch - 1);
    last = __shfl_sync(kFull, last, 0);
    if (!last) return;
    const float* po = a.part_o + (head - a.whole) * a.nchunk * G * D;
    const float2* pml = reinterpret_cast<const float2*>(a.part_ml) + (head - a.whole) * a.nchunk * G;
    const int nch = mt.nch;
    constexpr int HPL = G / HPI;  // head rows per lane: each lane owns float4 c4 of them
    const int jl = lane / V4;     // head offset of this lane within a row group
    float4 acc[HPL];
#pragma unroll
    for (int x = 0; x < HPL; ++x) acc[x] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (nch <= 32) {
        // one round: every lane loads the (max, sum) pairs of chunk c = lane, and the
        // partials of chunks 0 and 1 are requested at the same time
        float2 m2[G];
#pragma unroll
        for (int j = 0; j < G; ++j)
            m2[j] = lane < nch ? __ldcg(&pml[lane * G + j]) : make_float2(-INFINITY, 0.f);
        float4 p0[HPL], p1[HPL];
#pragma unroll
        for (int x = 0; x < HPL; ++x) {
            const int j = x * HPI + jl;
            p0[x] = __ldcg(reinterpret_cast<const float4*>(po + j * D) + c4);
            p1[x] = nch > 1 ? __ldcg(reinterpret_cast<const float4*>(po + (G + j) * D) + c4)
                            : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        // weights e^(m_c - M) / L per (chunk, head), into the slot's scratch o [nch][G]
        float* wgt = o;
#pragma unroll
        for (int j = 0; j < G; ++j) {
            float M = m2[j].x;
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) M = fmaxf(M, __shfl_xor_sync(kFull, M, off));
            const float e = lane < nch ? fast_exp2(m2[j].x - M) : 0.f;
            float L = m2[j].y * e;
#pragma unroll
            for (int off = 16; off >= 1; off >>= 1) L += __shfl_xor_sync(kFull, L, off);
            if (lane < nch) wgt[lane * G + j] = e / L;
        }
        __syncwarp();
#pragma unroll
        for (int x = 0; x < HPL; ++x) {
            const int j = x * HPI + jl;
            const float w0 = wgt[j], w1 = nch > 1 ? wgt[G + j] : 0.f;
            acc[x].x = fmaf(p1[x].x, w1, p0[x].x * w0);
            acc[x].y = fmaf(p1[x].y, w1, p0[x].y * w0);
            acc[x].z = fmaf(p1[x].z, w1, p0[x].z * w0);
            acc[x].w = fmaf(p1[x].w, w1, p0[x].w * w0);
        }
#pragma unroll 2
        for (int c = 2; c < nch; ++c) {
#pragma unroll
            for (int x = 0; x < HPL; ++x) {
                const int j = x * HPI + jl;
                const float4 p = __ldcg(reinterpret_cast<const float4*>(po + (c * G + j) * D) + c4);
                const float w = wgt[c * G + j];
                acc[x].x = fmaf(p.x, w, acc[x].x);
                acc[x].y = fmaf(p.y, w, acc[x].y);
                acc[x].z = fmaf(p.z, w, acc[x].z);
                acc[x].w = fmaf(p.w, w, acc[x].w);
            }
        }
    } else {
        // many chunks: per head, the max, the sum and the weighted outputs in three passes
#pragma unroll
        for (int x = 0; x < HPL; ++x) {
            const int j = x * HPI + jl;
            float M = -INFINITY;
            for (int c = 0; c < nch; ++c) M = fmaxf(M, __ldcg(&pml[c * G + j]).x);
            float L = 0.f;
            for (int c = 0; c < nch; ++c) {
                const float2 m = __ldcg(&pml[c * G + j]);
                const float sc = fast_exp2(m.x - M);
                const float4 p = __ldcg(reinterpret_cast<const float4*>(po + (c * G + j) * D) + c4);
                L = fmaf(m.y, sc, L);
                acc[x].x = fmaf(p.x, sc, acc[x].x);
                acc[x].y = fmaf(p.y, sc, acc[x].y);
                acc[x].z = fmaf(p.z, sc, acc[x].z);
                acc[x].w = fmaf(p.w, sc, acc[x].w);
            }
            const float inv = 1.f / L;
            acc[x] = make_float4(acc[x].x * inv, acc[x].y * inv, acc[x].z * inv, acc[x].w * inv);
        }
    }
#pragma unroll
    for (int x = 0; x < HPL; ++x) {
        const int j = x * HPI + jl;
        if (j < a.gq) reinterpret_cast<float4*>(out_g + j * D)[c4] = acc[x];  // the real query heads
    }
    if (lane == 0) a.counters[head] = 0;
}

template <int D>
__global__ void __launch_bounds__(kTcThreads, PBB_TC_MIN_CTAS)
    decode_kernel_tc(const DecodeArgs a, const __grid_constant__ CUtensorMap kmap,
                     const __grid_constant__ CUtensorMap vmap)
{
    using C = TcCfg<D>;
    constexpr int G = C::G;
    constexpr int TK = C::TK;
    extern __shared__ unsigned char dsmem_raw[];
    __shared__ __align__(8) uint64_t full_bar[kTcStages];
    __shared__ __align__(8) uint64_t empty_bar[kTcStages];
    __shared__ __align__(8) uint64_t epi_full[kTcEpiSlots];   // consumers -> epilogue (count kTcConsumers)
    __shared__ __align__(8) uint64_t epi_empty[kTcEpiSlots];  // epilogue -> consumers (count 1)
    __shared__ TileMeta meta_s[kTcStages];
    __shared__ TileMeta epi_meta[kTcEpiSlots];
    __shared__ float2 epi_ml[kTcEpiSlots][kTcConsumers][G];
    __shared__ volatile int abort_s;
    __shared__ int issued_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    float* epi_o = reinterpret_cast<float*>(dsmem + kTcStages * C::STAGE);  // [kTcEpiSlots][kTcConsumers][G][D]

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (tid == 0) {
#pragma unroll
        for (int s = 0; s < kTcStages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], kTcConsumers);
        }
#pragma unroll
        for (int s = 0; s < kTcEpiSlots; ++s) {
            mbar_init(&epi_full[s], kTcConsumers);
            mbar_init(&epi_empty[s], 1);
        }
        fence_mbar_init();
        abort_s = 0;
        issued_s = 0;
    }
    if (a.gq < G) {
        // a group of gq < 8 heads fills the score tile's columns gq .. 7 with zero query rows,
        // never loaded: those heads compute finite values that are never written
        for (int s = 0; s < kTcStages; ++s)
            for (int x = threadIdx.x; x < (G - a.gq) * C::ROW / 16; x += blockDim.x)
                reinterpret_cast<uint4*>(dsmem + s * C::STAGE + C::Q_OFF + a.gq * C::ROW)[x] = make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();
    // the set-up above touches no global memory; everything below may read what the previous
    // grid of the stream wrote (rings, positions, the queue words)
    pdl_wait();
    pdl_launch_dependents();

    if (warp == kTcProducer) {
        // ================= producer: one lane =================
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&kmap)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&vmap)) : "memory");
            int seq = 0;
            bool ok = true;
            // The next item's index (an atomic on the queue) and its position are fetched while
            // the current item's last tiles are issued, so neither round trip to L2 sits between
            // two items.
            int item = blockIdx.x;
            int t_item = item < a.total_items ? __ldg(a.pos + tc_item_seq(a, item)) : 0;
            while (ok && item < a.total_items) {
                int next = -1, t_next = 0;
                int pair, chunk;
                tc_item(a, item, pair, chunk);
                const int kvh = pair % a.Hkv, b = pair / a.Hkv;
                const int t = t_item;
                const int B = a.B;
                int r = 0, n = 0, base = 0;
                if (t >= 0) support_keys(t, B, a.window, r, n, base);
                // the run of n slots from `base`, in tile-aligned key space: tiles start at slot
                // multiples of TK, the run occupies aligned keys [lo0, lo0 + n)
                const int lo0 = n > 0 ? base % TK : 0;
                const int tbase = base - lo0;         // slot of aligned key 0
                const int span = lo0 + n;             // aligned keys up to the end of the run
                const bool whole = pair < a.whole;
                const int csize = whole ? max(span, 1) : a.chunk;  // aligned keys per chunk (tiles)
                const int nch = span > 0 ? (span + csize - 1) / csize : 1;
                // a sequence with a negative position is skipped (and flagged once); so are the
                // chunks past the end of a short support
                const bool skip = t < 0 || chunk >= nch;
                if (t < 0 && chunk == 0 && kvh == 0) atomicCAS(&g_status, kDevOk, kDevBadPosition);
                const int i0 = chunk * csize;
                const int i1 = min(i0 + csize, span);
                const int nkeys = max(i1 - i0, 0);
                const int ntiles = skip ? 0 : (nkeys > 0 ? (nkeys + TK - 1) / TK : 1);
                const int head = b * a.Hkv + kvh;
                const int ahead = max(ntiles - 3, 0);  // tile at which the next index is fetched
                for (int it = 0; it < ntiles; ++it, ++seq) {
                    if (it == ahead) next = static_cast<int>(gridDim.x) + atomicAdd(a.ctl, 1);
                    if (it == ntiles - 1 && next < a.total_items) t_next = __ldg(a.pos + tc_item_seq(a, next));
                    const int s = seq % kTcStages;
                    if (seq >= kTcStages &&
                        !mbar_wait(&empty_bar[s], static_cast<uint32_t>((seq / kTcStages - 1) & 1), kGuardNs)) {
                        ok = false;
                        break;
                    }
                    if (abort_s) {
                        ok = false;
                        break;
                    }
                    const int k0 = i0 + it * TK;                  // aligned key of the tile's row 0
                    const int nk = max(min(TK, i1 - k0), 0);      // rows [lo, nk) are in the run
                    const int lo = min(max(lo0 - k0, 0), TK);
                    const bool first = it == 0;
                    const bool current = first && chunk == 0;
                    TileMeta mt;
                    mt.b = b;
                    mt.kvh = kvh;
                    mt.chunk = chunk;
                    mt.nk = nk;
                    mt.nch = nch;
                    mt.r = r;
                    mt.flags = (first ? kFirst : 0) | (it == ntiles - 1 ? kLast : 0) | (current ? kCurrent : 0);
                    mt.lo = lo;
                    meta_s[s] = mt;
                    unsigned char* st = dsmem + s * C::STAGE;
                    const bool rows = nk > lo;
                    const uint32_t bytes = static_cast<uint32_t>((rows ? 2 * C::BOXES * C::BOX_BYTES : 0) +
                                                                 (first ? a.gq * C::ROW : 0) + (current ? 2 * C::ROW : 0));
                    fence_proxy_async();
                    mbar_expect_tx(&full_bar[s], bytes);
                    if (rows) {
                        // whole boxes of TK rows at a slot multiple of TK: the box never crosses
                        // slot B-1 (B is a multiple of 2*TK); rows outside [lo, nk) are masked
                        int slot = tbase + k0;
                        if (slot >= B) slot -= B;
                        const int y = head * B + slot;
#pragma unroll
                        for (int bx = 0; bx < C::BOXES; ++bx) {
                            tma_load_2d(st + C::K_OFF + bx * C::BOX_BYTES, &kmap, bx * 64, y, &full_bar[s]);
                            tma_load_2d(st + C::V_OFF + bx * C::BOX_BYTES, &vmap, bx * 64, y, &full_bar[s]);
                        }
                    }
                    if (first) {
                        const unsigned char* qg = static_cast<const unsigned char*>(a.q) +
                                                  (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(kvh) * a.gq) * C::ROW;
                        bulk_g2s(st + C::Q_OFF, qg, a.gq * C::ROW, &full_bar[s]);
                    }
                    if (current) {
                        bulk_g2s(st + C::KN_OFF, static_cast<const unsigned char*>(a.k_new) + static_cast<size_t>(head) * C::ROW,
                                 C::ROW, &full_bar[s]);
                        bulk_g2s(st + C::VN_OFF, static_cast<const unsigned char*>(a.v_new) + static_cast<size_t>(head) * C::ROW,
                                 C::ROW, &full_bar[s]);
                    }
                }
                if (!ok) break;
                if (next < 0) next = static_cast<int>(gridDim.x) + atomicAdd(a.ctl, 1);  // a skipped item
                if (ntiles == 0 && next < a.total_items) t_next = __ldg(a.pos + tc_item_seq(a, next));
                item = next;
                t_item = t_next;
            }
            if (ok) {  // end-of-work descriptor
                const int s = seq % kTcStages;
                if (seq >= kTcStages &&
                    !mbar_wait(&empty_bar[s], static_cast<uint32_t>((seq / kTcStages - 1) & 1), kGuardNs)) {
                    ok = false;
                } else {
                    TileMeta mt{};
                    mt.flags = kEnd;
                    meta_s[s] = mt;
                    mbar_arrive(&full_bar[s]);
                    ++seq;
                }
            }
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_status, kDevOk, kDevTimeout);
            }
            issued_s = seq;
        }
    } else if (warp == kTcEpilogue) {
        // ================= epilogue: ends the items the consumers hand over =================
        for (int k = 0;; ++k) {
            const int es = k % kTcEpiSlots;
            if (!mbar_wait_or_abort(&epi_full[es], static_cast<uint32_t>((k / kTcEpiSlots) & 1), &abort_s)) {
                if (!abort_s) {
                    abort_s = 1;
                    atomicCAS(&g_status, kDevOk, kDevTimeout);
                }
                break;
            }
            const TileMeta mt = epi_meta[es];
            if (mt.flags & kEnd) break;
            epilogue_item<G, D, kTcConsumers>(a, mt, &epi_ml[es][0][0], epi_o + es * (kTcConsumers * G * D), lane);
            __syncwarp();
            if (lane == 0) mbar_arrive(&epi_empty[es]);
        }
    } else {
        // ================= consumers =================
        const int g = lane >> 2, tig = lane & 3;  // fragment row group and thread in group
        const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
        uint32_t qb[C::KSTEPS][2];  // Q^T B fragments: head g, dims 16kk + 2tig (+8)
        float o[C::MTILES][4];      // O^T C fragments: dims 16mt + g (+8), heads 2tig, 2tig+1
        float m0 = -INFINITY, m1 = -INFINITY;  // running max of heads 2tig, 2tig+1 (log2 domain)
        float l0 = 0.f, l1 = 0.f;               // this lane's share of their running sums
        int epi_seq = 0;                         // items handed to the epilogue warp
#pragma unroll
        for (int kk = 0; kk < C::KSTEPS; ++kk) qb[kk][0] = qb[kk][1] = 0u;
#pragma unroll
        for (int mt_ = 0; mt_ < C::MTILES; ++mt_)
#pragma unroll
            for (int x = 0; x < 4; ++x) o[mt_][x] = 0.f;
        // lane's ldmatrix row within a 16-row block and its chunk offset, for both operand orders
        const int lm = lane >> 3;                     // which 8x8 matrix this lane addresses
        const int rowA = 8 * (lm & 1) + (lane & 7);   // K (non-transposed): matrices (rows, +8) x (chunk, +1)
        const int chA = lm >> 1;
        const int rowV = 8 * (lm >> 1) + (lane & 7);  // V^T (transposed): matrices (chunk, +1) x (rows, +8)
        const int chV = lm & 1;

        for (int seq = 0;; ++seq) {
            const int s = seq % kTcStages;
            if (!mbar_wait(&full_bar[s], static_cast<uint32_t>((seq / kTcStages) & 1), a.timeout_ns)) {
                abort_s = 1;
                atomicCAS(&g_status, kDevOk, kDevTimeout);
                break;
            }
            const TileMeta mt = meta_s[s];
            if (abort_s) break;
            if (mt.flags & kEnd) {
                // hand the end marker to the epilogue warp through the next slot
                const int es = epi_seq % kTcEpiSlots;
                if (epi_seq >= kTcEpiSlots &&
                    !mbar_wait_or_abort(&epi_empty[es], static_cast<uint32_t>((epi_seq / kTcEpiSlots - 1) & 1),
                                        &abort_s)) {
                    if (!abort_s) {
                        abort_s = 1;
                        atomicCAS(&g_status, kDevOk, kDevTimeout);
                    }
                    break;
                }
                if (warp == 0 && lane == 0) epi_meta[es] = mt;
                __syncwarp();
                if (lane == 0) mbar_arrive(&epi_full[es]);
                break;
            }
            const unsigned char* st = dsmem + s * C::STAGE;
            const size_t head = static_cast<size_t>(mt.b) * a.Hkv + mt.kvh;

            if (mt.flags & kFirst) {
#pragma unroll
                for (int kk = 0; kk < C::KSTEPS; ++kk) {
                    qb[kk][0] = *reinterpret_cast<const uint32_t*>(st + C::Q_OFF + g * C::ROW + (16 * kk + 2 * tig) * 2);
                    qb[kk][1] = *reinterpret_cast<const uint32_t*>(st + C::Q_OFF + g * C::ROW + (16 * kk + 2 * tig + 8) * 2);
                }
                m0 = m1 = -INFINITY;
                l0 = l1 = 0.f;
#pragma unroll
                for (int mt_ = 0; mt_ < C::MTILES; ++mt_)
#pragma unroll
                    for (int x = 0; x < 4; ++x) o[mt_][x] = 0.f;
                if (mt.flags & kCurrent) {
                    if (warp == 0) {  // the current token seeds warp 0's state (weight 1 at its own max)
                        float kc[C::PVD];
                        load_elems<2, C::PVD>(st + C::KN_OFF + lane * C::PVD * 2, kc);
#pragma unroll
                        for (int j = 0; j < G; ++j) {
                            float qf[C::PVD];
                            load_elems<2, C::PVD>(st + C::Q_OFF + j * C::ROW + lane * C::PVD * 2, qf);
                            float acc = 0.f;
#pragma unroll
                            for (int x = 0; x < C::PVD; ++x) acc = fmaf(qf[x], kc[x], acc);
#pragma unroll
                            for (int off = 16; off >= 1; off >>= 1) acc += __shfl_xor_sync(kFull, acc, off);
                            const float zj = acc * qscale;
                            m0 = (j == 2 * tig) ? zj : m0;
                            m1 = (j == 2 * tig + 1) ? zj : m1;
                        }
                        l0 = l1 = (g == 0) ? 1.f : 0.f;
                        const __nv_bfloat16* vn = reinterpret_cast<const __nv_bfloat16*>(st + C::VN_OFF);
#pragma unroll
                        for (int mt_ = 0; mt_ < C::MTILES; ++mt_) {
                            const float va = __bfloat162float(vn[16 * mt_ + g]);
                            const float vb = __bfloat162float(vn[16 * mt_ + g + 8]);
                            o[mt_][0] = va;
                            o[mt_][1] = va;
                            o[mt_][2] = vb;
                            o[mt_][3] = vb;
                        }
                    }
                    if (warp == kTcConsumers - 1) {  // append: slot r of both rings <- the new rows
                        uint4* kd = reinterpret_cast<uint4*>(static_cast<unsigned char*>(a.k_ring) +
                                                             (head * a.B + mt.r) * C::ROW);
                        uint4* vd = reinterpret_cast<uint4*>(static_cast<unsigned char*>(a.v_ring) +
                                                             (head * a.B + mt.r) * C::ROW);
                        for (int x = lane; x < C::ROW / 16; x += 32) {
                            kd[x] = *reinterpret_cast<const uint4*>(st + C::KN_OFF + x * 16);
                            vd[x] = *reinterpret_cast<const uint4*>(st + C::VN_OFF + x * 16);
                        }
                    }
                }
            }

            // this warp's rows 16*warp .. 16*warp+15 of the tile; rows outside [lo, nk) are masked
            const int row0 = 16 * warp;
            const int lo = mt.lo;
            if (row0 + 16 > lo && row0 < mt.nk) {
                const uint32_t kbase = smem_addr(st + C::K_OFF);
                const uint32_t vbase = smem_addr(st + C::V_OFF);
                // ---- scores S^T [16 keys x 8 heads]: two independent mma chains (even and odd
                // k-steps) halve the dependent latency
                float c[4] = {0.f, 0.f, 0.f, 0.f};
                float c2[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int kk = 0; kk < C::KSTEPS; ++kk) {
                    const int chunk16 = 2 * kk + chA;  // 16-byte chunk of the 256-byte (or 128-byte) row
                    const int row = row0 + rowA;
                    uint32_t af[4];
                    ldmatrix_x4(af, kbase + (chunk16 >> 3) * C::BOX_BYTES + swz(row, chunk16 & 7));
                    if (kk & 1)
                        mma_bf16_16816(c2, af, qb[kk][0], qb[kk][1]);
                    else
                        mma_bf16_16816(c, af, qb[kk][0], qb[kk][1]);
                }
#pragma unroll
                for (int x = 0; x < 4; ++x) c[x] += c2[x];
                // keys g and g+8 of this warp's block; heads 2tig and 2tig+1
                const bool va = (row0 + g >= lo) && (row0 + g < mt.nk);
                const bool vb = (row0 + g + 8 >= lo) && (row0 + g + 8 < mt.nk);
                const float z0 = va ? c[0] * qscale : -INFINITY;
                const float z1 = va ? c[1] * qscale : -INFINITY;
                const float z2 = vb ? c[2] * qscale : -INFINITY;
                const float z3 = vb ? c[3] * qscale : -INFINITY;
                float mx0 = fmaxf(z0, z2), mx1 = fmaxf(z1, z3);
#pragma unroll
                for (int off = 4; off < 32; off <<= 1) {
                    mx0 = fmaxf(mx0, __shfl_xor_sync(kFull, mx0, off));
                    mx1 = fmaxf(mx1, __shfl_xor_sync(kFull, mx1, off));
                }
                const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
                if (__any_sync(kFull, (mn0 > m0) || (mn1 > m1))) {
                    const float al0 = fast_exp2(m0 - mn0), al1 = fast_exp2(m1 - mn1);
                    l0 *= al0;
                    l1 *= al1;
#pragma unroll
                    for (int mt_ = 0; mt_ < C::MTILES; ++mt_) {
                        o[mt_][0] *= al0;
                        o[mt_][1] *= al1;
                        o[mt_][2] *= al0;
                        o[mt_][3] *= al1;
                    }
                }
                m0 = mn0;
                m1 = mn1;
                const float p0 = fast_exp2(z0 - mn0), p1 = fast_exp2(z1 - mn1);
                const float p2 = fast_exp2(z2 - mn0), p3 = fast_exp2(z3 - mn1);
                l0 += p0 + p2;
                l1 += p1 + p3;
                // P^T B fragments: high and low bf16 parts, transposed from the S^T C layout
                const uint32_t h01 = pack_bf16x2(p0, p1), h23 = pack_bf16x2(p2, p3);
                const uint32_t r01 = pack_bf16x2(p0 - bf16_lo(h01), p1 - bf16_hi(h01));
                const uint32_t r23 = pack_bf16x2(p2 - bf16_lo(h23), p3 - bf16_hi(h23));
                const uint32_t bh0 = movmatrix_trans(h01), bh1 = movmatrix_trans(h23);
                const uint32_t bl0 = movmatrix_trans(r01), bl1 = movmatrix_trans(r23);
                // ---- O^T [d x 8 heads] += V^T [d x 16 keys] . P^T
#pragma unroll
                for (int mt_ = 0; mt_ < C::MTILES; ++mt_) {
                    const int chunk16 = 2 * mt_ + chV;
                    const int row = row0 + rowV;
                    uint32_t af[4];
                    ldmatrix_x4_trans(af, vbase + (chunk16 >> 3) * C::BOX_BYTES + swz(row, chunk16 & 7));
                    mma_bf16_16816(o[mt_], af, bh0, bh1);
                    mma_bf16_16816(o[mt_], af, bl0, bl1);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty_bar[s]);
            if (!(mt.flags & kLast)) continue;

            // ---- end of the item: this warp's (max, sum, output) into a free epilogue slot
            const int es = epi_seq % kTcEpiSlots;
            if (epi_seq >= kTcEpiSlots &&
                !mbar_wait_or_abort(&epi_empty[es], static_cast<uint32_t>((epi_seq / kTcEpiSlots - 1) & 1),
                                    &abort_s)) {
                if (!abort_s) {
                    abort_s = 1;
                    atomicCAS(&g_status, kDevOk, kDevTimeout);
                }
                break;
            }
            {
                float s0 = l0, s1 = l1;
#pragma unroll
                for (int off = 4; off < 32; off <<= 1) {
                    s0 += __shfl_xor_sync(kFull, s0, off);
                    s1 += __shfl_xor_sync(kFull, s1, off);
                }
                if (g == 0) {
                    epi_ml[es][warp][2 * tig] = make_float2(m0, s0);
                    epi_ml[es][warp][2 * tig + 1] = make_float2(m1, s1);
                }
            }
            float* ow = epi_o + es * (kTcConsumers * G * D) + (warp * G) * D;
#pragma unroll
            for (int mt_ = 0; mt_ < C::MTILES; ++mt_) {
                ow[(2 * tig) * D + 16 * mt_ + g] = o[mt_][0];
                ow[(2 * tig + 1) * D + 16 * mt_ + g] = o[mt_][1];
                ow[(2 * tig) * D + 16 * mt_ + g + 8] = o[mt_][2];
                ow[(2 * tig + 1) * D + 16 * mt_ + g + 8] = o[mt_][3];
            }
            if (warp == 0 && lane == 0) epi_meta[es] = mt;
            __syncwarp();
            if (lane == 0) mbar_arrive(&epi_full[es]);
            ++epi_seq;
        }
    }
    __syncthreads();
    if (abort_s) {
        if (tid == 0) {
            const int issued = issued_s;
            for (int s = 0; s < kTcStages && s < issued; ++s) {
                const int j = s + kTcStages * ((issued - 1 - s) / kTcStages);
                mbar_wait(&full_bar[s], static_cast<uint32_t>((j / kTcStages) & 1), kGuardNs);
            }
        }
        __syncthreads();
    }
    if (tid == 0) {  // the last CTA to finish resets the work queue for the next launch
        __threadfence();
        if (atomicAdd(a.ctl + 1, 1) == static_cast<int>(gridDim.x) - 1) {
            atomicExch(a.ctl, 0);
            atomicExch(a.ctl + 1, 0);
        }
    }
}

// --------------------------------------------------- prefill / advance ----

// Ring of a sequence resuming at t = pos[b]: row j of the history (position
// t - B + j) goes to slot (t - B + j) mod B; negative positions write zeros.
__global__ void prefill_kernel(const uint4* __restrict__ k_hist, const uint4* __restrict__ v_hist,
                               const int32_t* __restrict__ pos, uint4* __restrict__ k_ring,
                               uint4* __restrict__ v_ring, int Hkv, int B, int row16,
                               long long total)
{
    pdl_wait();
    pdl_launch_dependents();
    for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int x = static_cast<int>(i % row16);
        const long long rowi = i / row16;
        const int j = static_cast<int>(rowi % B);
        const long long head = rowi / B;
        const int b = static_cast<int>(head / Hkv);
        const int t = __ldg(pos + b);
        if (t < 0) {
            if (j == 0 && x == 0 && (head % Hkv) == 0) atomicCAS(&g_status, kDevOk, kDevBadPosition);
            continue;
        }
        const long long s = static_cast<long long>(t) - B + j;
        const long long slot = ((s % B) + B) % B;
        const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
        const size_t dst = (static_cast<size_t>(head) * B + static_cast<size_t>(slot)) * row16 + x;
        k_ring[dst] = s >= 0 ? __ldg(k_hist + i) : zero;
        v_ring[dst] = s >= 0 ? __ldg(v_hist + i) : zero;
    }
}

__global__ void advance_kernel(int32_t* pos, int batch)
{
    pdl_wait();
    pdl_launch_dependents();
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < batch; i += gridDim.x * blockDim.x) pos[i] += 1;
}

// The step's sequences by descending number of ring keys in their supports (support_keys' n):
// a counting sort on 256 length classes, largest first, by one block. When every support is a
// whole work item and the step runs several rounds of them per CTA, the tensor-core kernel takes
// them in this order, so the step ends on short supports and its CTAs finish together
// (longest processing time first). The order within a class is unspecified; the supports are
// independent work items, so no result depends on it.
__global__ void __launch_bounds__(1024) support_order_kernel(const int32_t* __restrict__ pos, int pos_batch,
                                                             int batch, int B, int window, int* __restrict__ order)
{
    __shared__ int cnt[256];
    pdl_wait();
    pdl_launch_dependents();
    for (int i = threadIdx.x; i < 256; i += blockDim.x) cnt[i] = 0;
    __syncthreads();
    auto cls = [&](int b) {  // class 0 holds the longest supports
        int r, n, base;
        support_keys(__ldg(pos + (b < pos_batch ? b : b % pos_batch)), B, window, r, n, base);
        const long long c = 255 - static_cast<long long>(n) * 256 / B;
        return static_cast<int>(c < 0 ? 0 : (c > 255 ? 255 : c));
    };
    for (int b = threadIdx.x; b < batch; b += blockDim.x) atomicAdd(&cnt[cls(b)], 1);
    __syncthreads();
    if (threadIdx.x < 32) {  // exclusive prefix sum over the classes, 8 a lane
        const int l = static_cast<int>(threadIdx.x);
        int v[8], sum = 0;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            v[i] = cnt[8 * l + i];
            sum += v[i];
        }
        int incl = sum;
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
            const int o = __shfl_up_sync(kFull, incl, off);
            if (l >= off) incl += o;
        }
        int run = incl - sum;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            cnt[8 * l + i] = run;
            run += v[i];
        }
    }
    __syncthreads();
    for (int b = threadIdx.x; b < batch; b += blockDim.x) order[atomicAdd(&cnt[cls(b)], 1)] = b;
}

// Launches of the decode-step kernels (decode, position advance, ring load) allow programmatic
// dependent launch: a kernel may be scheduled while the previous kernel of the stream finishes,
// so its launch and set-up overlap that kernel's tail; each of them calls pdl_wait before it
// touches global memory, so it sees everything the previous kernel wrote, as with plain stream
// order. PBB_PDL = 0 launches them plainly.
#ifndef PBB_PDL
#define PBB_PDL 1
#endif
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), int grid, int block, size_t smem, cudaStream_t stream, Args&&... args)
{
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(static_cast<unsigned>(block));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = PBB_PDL ? 1 : 0;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Opt the kernel in to its dynamic shared memory (above the 48 KiB default), once per device.
template <int ELEM, int D, int G>
cudaError_t ensure_smem_attr()
{
    static std::atomic<int> done[kMaxCachedDevices] = {};
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    const int ok = cached_per_device(done, dev, [&] {
        err = cudaFuncSetAttribute(decode_kernel<ELEM, D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   Cfg<ELEM, D, G>::SMEM);
        return err == cudaSuccess ? 1 : 0;
    });
    return ok > 0 ? cudaSuccess : err;
}

template <int ELEM, int D, int G>
int occupancy_t()
{
    static std::atomic<int> cache[kMaxCachedDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    return cached_per_device(cache, dev, [] {
        int n = 0;
        if (ensure_smem_attr<ELEM, D, G>() != cudaSuccess) return 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decode_kernel<ELEM, D, G>, kThreads,
                                                          Cfg<ELEM, D, G>::SMEM) != cudaSuccess)
            return 0;
        return n;
    });
}

template <int ELEM, int D, int G>
cudaError_t launch_t(const DecodeArgs& a, cudaStream_t stream)
{
    using C = Cfg<ELEM, D, G>;
    cudaError_t err = ensure_smem_attr<ELEM, D, G>();
    if (err != cudaSuccess) return err;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int per_sm = occupancy_t<ELEM, D, G>();
    if (per_sm < 1) per_sm = 1;
    const long long ctas = static_cast<long long>(sms) * per_sm;
    const int grid = static_cast<int>(a.total_items < ctas ? a.total_items : ctas);
    if (grid < 1) return cudaSuccess;
    return launch_pdl(decode_kernel<ELEM, D, G>, grid, kThreads, C::SMEM, stream, a);
}

// ---- tensor-core path: TMA tensor maps over the rings and the launch

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder()
{
    // looked up once: one thread initialises a function-local static while any others wait
    static const PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
        return static_cast<PFN_cuTensorMapEncodeTiled_v12000>(nullptr);
    }();
    return fn;
}

// Map a ring [rows][d] bf16 as a 2-D tensor read in boxes of 64 columns x box_rows
// rows with the 128-byte swizzle. Caches the last maps built (rings rarely move).
bool ring_tensor_map(CUtensorMap* map, const void* ring, unsigned long long rows, int d, int box_rows)
{
    struct Entry {
        const void* ring;
        unsigned long long rows;
        int d, box_rows;
        CUtensorMap map;
    };
    static std::mutex mu;
    static Entry cache[16];
    static int next = 0;
    std::lock_guard<std::mutex> lock(mu);
    for (auto& e : cache)
        if (e.ring == ring && e.rows == rows && e.d == d && e.box_rows == box_rows) {
            *map = e.map;
            return true;
        }
    PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(rows)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(d) * 2};
    const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1, 1};
    CUtensorMap m;
    if (enc(&m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ring), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) !=
        CUDA_SUCCESS)
        return false;
    cache[next] = Entry{ring, rows, d, box_rows, m};
    next = (next + 1) % 16;
    *map = m;
    return true;
}

template <int D>
int occupancy_tc()
{
    static std::atomic<int> cache[kMaxCachedDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    return cached_per_device(cache, dev, [] {
        if (cudaFuncSetAttribute(decode_kernel_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 TcCfg<D>::SMEM) != cudaSuccess)
            return 0;
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decode_kernel_tc<D>, kTcThreads, TcCfg<D>::SMEM) !=
            cudaSuccess)
            return 0;
        return n;
    });
}

int device_sms()
{
    static std::atomic<int> cache[kMaxCachedDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    return cached_per_device(cache, dev, [dev] {
        int n = 0;
        return cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess ? n : 0;
    });
}

// PBB_TC_PAD_MIN_FILL = 1 keeps padded groups (4 and 6 heads in the 8-column score tile) on the
// CUDA cores unless the supports fill the resident CTAs. That paid while the tensor-core kernel's
// two consumer warps ended the items themselves; with the epilogue warp the tensor cores win at
// small batches too (measured on GB300, Hq 32, Hkv 8: batch 8 / 32 at B 4096 25.4 / 74.5 against
// 33.5 / 105.7 us per step, batch 32 at B 1024 9.7 against 12.2 us), so it is off.
#ifndef PBB_TC_PAD_MIN_FILL
#define PBB_TC_PAD_MIN_FILL 0
#endif
// Sliding-window steps on the tensor-core kernel (0 keeps them on the CUDA cores).
#ifndef PBB_TC_WINDOWS
#define PBB_TC_WINDOWS 1
#endif

// Whether a step of this shape runs the tensor-core kernel, before the chunk check: a bf16 step
// (PBB or window; tiles start at slot multiples of the tile, and rows of a tile outside the
// support are masked), GQA group 8 (or 4 or 6, padded), d 64 or 128, block a multiple of two
// tiles (no tile straddles the ring end), row coordinates within int32.
std::atomic<int> g_kernel_choice{PBB_KERNEL_AUTO};

bool tc_shape(int batch, int Hkv, int d, int B, int elem_bytes, int group, int window)
{
    const int choice = g_kernel_choice.load();
    if (choice == PBB_KERNEL_CUDA_CORES) return false;
    if (elem_bytes != 2 || !tc_group(group) || (d != 64 && d != 128)) return false;
    if (window != 0 && !PBB_TC_WINDOWS) return false;
    if (B % (32 * kTcConsumers) != 0 || tensor_map_encoder() == nullptr) return false;
    const unsigned long long rows = static_cast<unsigned long long>(batch) * Hkv * B;
    if (rows >= (1ull << 31)) return false;
    if (PBB_TC_PAD_MIN_FILL && group != 8 && choice == PBB_KERNEL_AUTO) {
        const long long ctas = static_cast<long long>(device_sms()) * (d == 64 ? occupancy_tc<64>() : occupancy_tc<128>());
        if (static_cast<long long>(batch) * Hkv < ctas) return false;
    }
    return true;
}

// The tensor-core path also needs chunks of whole tiles.
bool tc_eligible(const DecodeArgs& a, int elem_bytes)
{
    constexpr int tk = 16 * kTcConsumers;
    return tc_shape(a.batch, a.Hkv, a.d, a.B, elem_bytes, a.gq, a.window) && a.chunk % tk == 0;
}

template <int D>
cudaError_t launch_tc(const DecodeArgs& a, cudaStream_t stream)
{
    using C = TcCfg<D>;
    const int per_sm = occupancy_tc<D>();
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const unsigned long long rows = static_cast<unsigned long long>(a.batch) * a.Hkv * a.B;
    CUtensorMap kmap, vmap;
    if (!ring_tensor_map(&kmap, a.k_ring, rows, D, C::TK) || !ring_tensor_map(&vmap, a.v_ring, rows, D, C::TK))
        return cudaErrorInvalidValue;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const long long ctas = static_cast<long long>(sms) * per_sm;
    const int grid = static_cast<int>(a.total_items < ctas ? a.total_items : ctas);
    if (grid < 1) return cudaSuccess;
    return launch_pdl(decode_kernel_tc<D>, grid, kTcThreads, C::SMEM, stream, a, kmap, vmap);
}

template <int ELEM, int D>
cudaError_t launch_g(const DecodeArgs& a, cudaStream_t stream)
{
    switch (a.Hq / a.Hkv) {
        case 1: return launch_t<ELEM, D, 1>(a, stream);
        case 2: return launch_t<ELEM, D, 2>(a, stream);
        case 4: return launch_t<ELEM, D, 4>(a, stream);
        case 6:  // six query heads per KV head run on the group-8 kernel with two padded heads
        case 8: return launch_t<ELEM, D, 8>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

template <int ELEM, int D>
int occupancy_g(int group)
{
    switch (group) {
        case 1: return occupancy_t<ELEM, D, 1>();
        case 2: return occupancy_t<ELEM, D, 2>();
        case 4: return occupancy_t<ELEM, D, 4>();
        case 6:
        case 8: return occupancy_t<ELEM, D, 8>();
        default: return 0;
    }
}

template <int ELEM, int D>
int tile_g(int group)
{
    switch (group) {
        case 1: return Cfg<ELEM, D, 1>::TK;
        case 2: return Cfg<ELEM, D, 2>::TK;
        case 4: return Cfg<ELEM, D, 4>::TK;
        case 6:
        case 8: return Cfg<ELEM, D, 8>::TK;
        default: return 0;
    }
}

}  // namespace

int tile_keys(int elem_bytes, int d, int group)
{
    if (elem_bytes == 2 && d == 64) return tile_g<2, 64>(group);
    if (elem_bytes == 2 && d == 128) return tile_g<2, 128>(group);
    if (elem_bytes == 4 && d == 64) return tile_g<4, 64>(group);
    if (elem_bytes == 4 && d == 128) return tile_g<4, 128>(group);
    return 0;
}

int set_kernel_choice(int kernel) { return g_kernel_choice.exchange(kernel); }

bool tensor_core_shape(int batch, int Hkv, int d, int B, int elem_bytes, int group, int window)
{
    return tc_shape(batch, Hkv, d, B, elem_bytes, group, window);
}

int decode_ctas_per_sm(int batch, int Hkv, int elem_bytes, int d, int group, int B, int window)
{
    if (tc_shape(batch, Hkv, d, B, elem_bytes, group, window)) return d == 64 ? occupancy_tc<64>() : occupancy_tc<128>();
    if (elem_bytes == 2 && d == 64) return occupancy_g<2, 64>(group);
    if (elem_bytes == 2 && d == 128) return occupancy_g<2, 128>(group);
    if (elem_bytes == 4 && d == 64) return occupancy_g<4, 64>(group);
    if (elem_bytes == 4 && d == 128) return occupancy_g<4, 128>(group);
    return 0;
}

bool use_tensor_cores(const DecodeArgs& a, int elem_bytes) { return tc_eligible(a, elem_bytes); }

cudaError_t launch_decode(const DecodeArgs& a, int elem_bytes, cudaStream_t stream)
{
    if (tc_eligible(a, elem_bytes)) return a.d == 64 ? launch_tc<64>(a, stream) : launch_tc<128>(a, stream);
    if (elem_bytes == 2 && a.d == 64) return launch_g<2, 64>(a, stream);
    if (elem_bytes == 2 && a.d == 128) return launch_g<2, 128>(a, stream);
    if (elem_bytes == 4 && a.d == 64) return launch_g<4, 64>(a, stream);
    if (elem_bytes == 4 && a.d == 128) return launch_g<4, 128>(a, stream);
    return cudaErrorInvalidValue;
}

cudaError_t launch_prefill(const void* k_hist, const void* v_hist, const int32_t* pos, void* k_ring,
                           void* v_ring, int batch, int Hkv, int B, int row_bytes,
                           cudaStream_t stream)
{
    const int row16 = row_bytes / 16;
    const long long total = static_cast<long long>(batch) * Hkv * B * row16;
    if (total == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const long long want = (total + 255) / 256;
    const int blocks = static_cast<int>(want < sms * 16LL ? want : sms * 16LL);
    return launch_pdl(prefill_kernel, blocks, 256, 0, stream, static_cast<const uint4*>(k_hist),
                      static_cast<const uint4*>(v_hist), pos, static_cast<uint4*>(k_ring),
                      static_cast<uint4*>(v_ring), Hkv, B, row16, total);
}

cudaError_t launch_support_order(const DecodeArgs& a, int* order, cudaStream_t stream)
{
    return launch_pdl(support_order_kernel, 1, 1024, 0, stream, a.pos, a.pos_batch, a.batch, a.B, a.window, order);
}

cudaError_t launch_advance(int32_t* pos, int batch, cudaStream_t stream)
{
    if (batch == 0) return cudaSuccess;
    const int blocks = (batch + 255) / 256 < 64 ? (batch + 255) / 256 : 64;
    return launch_pdl(advance_kernel, blocks, 256, 0, stream, pos, batch);
}

bool rows_tensor_map(CUtensorMap* map, const void* base, unsigned long long rows, int d, int box_rows)
{
    return ring_tensor_map(map, base, rows, d, box_rows);
}

cudaError_t read_and_clear_status(int* status, cudaStream_t stream)
{
    cudaError_t err = cudaStreamSynchronize(stream);
    if (err != cudaSuccess) return err;
    err = cudaMemcpyFromSymbol(status, g_status, sizeof(int));
    if (err != cudaSuccess) return err;
    if (*status != kDevOk) {
        const int zero = kDevOk;
        err = cudaMemcpyToSymbol(g_status, &zero, sizeof(int));
    }
    return err;
}

}  // namespace pbb
