// PBB attention over whole sequences (the forward pass / prefill) for sm_103a,
// on the fifth-generation tensor cores (tcgen05, accumulators in TMEM).
//
// Every position t of a sequence attends to the interval [a(t), t],
// a(t) = max(0, h(floor(t/h) - 1)) (Eq. pbb_relay, the interval form of
// Eq. pbb, Sec. 3): the whole previous half-block and the causal prefix of its
// own half-block, with the single softmax of Eq. (attention). Each output row
// also gets its natural-log partition lse = ln sum exp(z) (Eq. lse), which a
// backward pass reuses.
//
// Work items. An item is QT consecutive positions t0 .. t0+QT-1 of all G query
// heads of one KV head: M = G*QT = 128 query rows, stacked head-major, so every
// K/V tile serves all G heads (native GQA). Its keys are [a(t0), t_last] (a(t)
// only grows with t, so the range covers every row), streamed in tiles of 64
// keys; rows whose support starts later or ends earlier are masked in the tiles
// that cross their bounds. No dense mask exists anywhere. Persistent CTAs (one
// per SM with 128-key tiles for long supports; for short ones three per SM with
// 32-key tiles at d = 64, two with 64-key tiles at d = 128; see FwdCfg) take items
// round-robin; query tiles of a head are adjacent items, so CTAs running together
// share K/V tiles in L2.
//
// Roles (192 threads; 320 with two softmax warpgroups, whose warps come first):
//   warp 4, one lane   TMA producer: Q of an item (one 2-D tensor copy per head
//                      and 64-column box; one or two Q buffers), then K and V tiles
//                      into a 2- to 4-stage ring (128-byte swizzle), all on
//                      full/empty mbarriers;
//   warp 5, one lane   MMA issuer: S_j = Q K_j^T (M 128, N = tile keys, both operands
//                      K-major in shared memory) into one of two TMEM buffers, then
//                      O += P_j V_j with P read from tensor memory and V MN-major in
//                      shared memory, into the item's TMEM output buffer (two
//                      alternating between items, one for narrow tiles at d = 128);
//                      each group is completed through tcgen05.commit;
//   warps 0-3          softmax: thread r owns query row r (TMEM lane r; with two
//                      warpgroups each takes half of the row's columns and they
//                      exchange partial maxima and sums). It reads
//                      its row of S with tcgen05.ld, masks, keeps a running maximum
//                      (base-2 domain, 1/sqrt(d) folded into one FFMA) that moves
//                      only when it grows by more than 2^8 (then it rescales its O
//                      row in TMEM), writes exp2(z - m) as bf16 pairs over the first
//                      half of its S row (P aliases S, as the MMA reads it from TMEM),
//                      and at the item's end divides its O row by the row sum and
//                      writes O and lse.
// S_{j+1} is computed while the softmax of tile j runs. MMAs of the one issuing
// thread execute in order, so S_{j+2} overwrites a buffer only after P.V of tile
// j has read its P.
//
// Long supports with B a multiple of 256 run forward_pair_kernel instead (the
// "paired items" section below): two adjacent query items of a head share every K/V
// tile, each with its own softmax warpgroup, S buffer and O buffer in TMEM.
//
// Every wait is bounded by the global timer; a wait that runs out records a
// timeout in this file's status word and every role stops. Before the CTA exits,
// the MMA issuer waits (bounded) for its MMAs, the producer for its copies, and
// the TMEM columns are released.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pbb_device.cuh"
#include "pbb_forward_plan.h"
#include "pbb_internal.h"
#include "pbb_store.cuh"

namespace pbb {

__device__ int g_fwd_status;  // first fault recorded by a forward kernel, kDevOk if none

namespace {

constexpr unsigned long long kGuardNs = 2000000000ull;  // waits only a broken GPU can exceed

// Shapes of the same kernel (chosen by the block size, see launch_fwd_shape):
//   NK    keys per K/V tile (128, 64 or 32);
//   WGS   softmax warpgroups (1, or 2 sharing every tile: each takes half of the score
//         columns and half of the output columns);
//   CTAS  CTAs per SM: 1 owns all 512 TMEM columns, 2 to 4 share them (256 or 128 each) so
//         one CTA's latencies overlap the others' work.
// Long supports (many tiles per item) use one CTA per SM; short ones, where an item is one
// or two tiles, two CTAs per SM with 64-key tiles.
template <int D, int G, int NK_, int WGS_, int CTAS_>
struct FwdCfg {
    static constexpr int NK = NK_;
    static constexpr int WGS = WGS_;
    static constexpr int CTAS = CTAS_;
    static constexpr int TMEM_COLS = CTAS == 1 ? 512 : (CTAS == 2 ? 256 : 128);  // a power of 2
    static constexpr int M = 128;                       // query rows of an item (G heads x QT positions)
    static constexpr int QT = M / G;                    // positions of an item
    static constexpr int BOXES = D / 64;                // 64-column boxes of a row
    static constexpr int QBOX = M * 128;                // bytes of one Q box
    static constexpr int KBOX = NK * 128;               // bytes of one K (or V) box
    static constexpr int QBUF = (D == 64 && CTAS <= 2) ? 2 : 1;  // Q buffers (the next item's Q loads early)
    static constexpr int KV_STAGE = 2 * BOXES * KBOX;   // K boxes then V boxes
    static constexpr int Q_OFF = 0;
    static constexpr int Q_BYTES = BOXES * QBOX;
    static constexpr int KV_OFF = Q_OFF + QBUF * Q_BYTES;
    // the kernel's static shared memory (barriers; with two warpgroups the exchanges of the
    // partial row maxima and sums, 2 x 2 x 128 floats each)
    static constexpr int STATIC_SMEM = WGS == 2 ? 4608 : 512;
    // K/V tiles in flight: as many as the shared memory of this shape holds, at most 4
    static constexpr int STAGE_ROOM = (227 * 1024 / CTAS - STATIC_SMEM - 1024 - KV_OFF) / KV_STAGE;
    static constexpr int STAGES = STAGE_ROOM < 4 ? STAGE_ROOM : 4;
    static constexpr int SMEM = KV_OFF + STAGES * KV_STAGE + 1024;  // + alignment slack
    // TMEM columns: S buffers at 0 and NK, output buffers from 2 NK: two alternating between
    // items where they fit
    static constexpr int T_S = 0;
    static constexpr int T_O = 2 * NK;
    static constexpr int OBUF = T_O + 2 * D <= TMEM_COLS ? 2 : 1;
    static constexpr int THREADS = 128 * WGS + 64;      // softmax warps, producer warp, MMA warp
    static constexpr int PRODUCER_WARP = 4 * WGS;
    static constexpr int MMA_WARP = 4 * WGS + 1;
    static_assert(STAGES >= 2, "shared memory budget");
    static_assert(NK == 32 || NK % 64 == 0, "P is packed 32 or 64 scores at a time");
    static_assert(T_O + OBUF * D <= TMEM_COLS, "TMEM budget");
    static_assert(QT % 8 == 0, "a head's Q rows must start on a swizzle atom (8 rows)");
    static_assert(CTAS * (SMEM + STATIC_SMEM) <= 227 * 1024, "shared memory budget");
};

// Start of the PBB support of position t: a(t) = max(0, h (floor(t/h) - 1)).
__device__ __forceinline__ int support_start(int t, int h)
{
    const int m = t / h;
    return m > 0 ? h * (m - 1) : 0;
}

// A bounded wait whose outcome is the same in every lane of the warp (the
// softmax warps run warp-collective tcgen05 loads after it).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, unsigned long long limit)
{
    return __all_sync(0xffffffffu, mbar_wait(bar, parity, limit));
}

// 16-column TMEM load (the shapes with three or four CTAs per SM work in 16-column chunks to
// stay within their registers).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

// max(a, b, c) in one instruction (three-input max.f32, sm_100 and later).
__device__ __forceinline__ float fmax3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// Writes EC consecutive outputs o of one row, starting at element e0 of `out` (bf16, or fp32
// with f32). A thread's row is 256 or 128 bytes from its neighbours', so each store instruction
// of a warp touches 32 lines: 32-byte stores halve those instructions where the output base is
// 32-byte aligned (every chunk is then too); other bases take 16-byte stores.
template <int EC>
__device__ __forceinline__ void store_chunk(void* out, bool f32, size_t e0, const float (&o)[EC], bool wide)
{
    if (f32) {
        float* dst = static_cast<float*>(out) + e0;
        if (wide) {
#pragma unroll
            for (int y = 0; y < EC / 8; ++y) {
                uint32_t w[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) w[i] = __float_as_uint(o[8 * y + i]);
                st_global_v8(dst + 8 * y, w);
            }
        } else {
#pragma unroll
            for (int y = 0; y < EC / 4; ++y)
                reinterpret_cast<float4*>(dst)[y] = make_float4(o[4 * y], o[4 * y + 1], o[4 * y + 2], o[4 * y + 3]);
        }
    } else {
        uint32_t pk[EC / 2];
#pragma unroll
        for (int y = 0; y < EC / 2; ++y) pk[y] = pack_bf16x2(o[2 * y], o[2 * y + 1]);
        __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(out) + e0;
        if (wide) {
#pragma unroll
            for (int y = 0; y < EC / 16; ++y) st_global_v8(dst + 16 * y, pk + 8 * y);
        } else {
#pragma unroll
            for (int y = 0; y < EC / 8; ++y)
                reinterpret_cast<uint4*>(dst)[y] = make_uint4(pk[4 * y], pk[4 * y + 1], pk[4 * y + 2], pk[4 * y + 3]);
        }
    }
}

// One work item: (sequence, KV head) pair, first position, keys and tiles.
struct Item {
    int pair, t0, tl, lo, a_max, ntiles;
};

template <int QT, int NK>
__device__ __forceinline__ Item make_item(int idx, int n, int B)
{
    const int nq = (n + QT - 1) / QT;
    Item it;
    it.pair = idx / nq;
    it.t0 = (idx - it.pair * nq) * QT;
    it.tl = min(it.t0 + QT, n) - 1;  // last valid position
    const int h = B >> 1;
    it.lo = support_start(it.t0, h);  // first key any row needs
    it.a_max = support_start(it.tl, h);
    it.ntiles = (it.tl - it.lo + NK) / NK;
    return it;
}

template <int D, int G, int NK, int WGS_, int CTAS_>
__global__ void __launch_bounds__(FwdCfg<D, G, NK, WGS_, CTAS_>::THREADS, CTAS_)
forward_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
               const __grid_constant__ CUtensorMap vmap, const ForwardArgs a)
{
    using C = FwdCfg<D, G, NK, WGS_, CTAS_>;
    constexpr int STAGES = C::STAGES;
    constexpr int WGS = C::WGS;
    extern __shared__ unsigned char dsmem_raw[];
    constexpr int QBUF = C::QBUF;
    __shared__ __align__(8) uint64_t q_full[QBUF], q_empty[QBUF], done_bar, lsum_bar, xch_bar[2];
    __shared__ __align__(8) uint64_t kv_full[STAGES], kv_empty[STAGES];
    __shared__ __align__(8) uint64_t s_full[2], p_full[2], pv_done[2], o_free[2];
    // with two warpgroups, by tile (item) parity: each warpgroup's partial row maxima (sums)
    __shared__ float xch_s[WGS == 2 ? 2 : 1][WGS][WGS == 2 ? 128 : 1];
    __shared__ float lsum_s[WGS == 2 ? 2 : 1][WGS][WGS == 2 ? 128 : 1];
    __shared__ uint32_t tmem_base_s;
    __shared__ volatile int abort_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_items = a.batch * a.Hkv * ((a.n + C::QT - 1) / C::QT);

    if (tid == 0) {
#pragma unroll
        for (int q = 0; q < QBUF; ++q) {
            mbar_init(&q_full[q], 1);
            mbar_init(&q_empty[q], 1);
        }
        mbar_init(&done_bar, 1);
        mbar_init(&lsum_bar, 128 * WGS);
        mbar_init(&xch_bar[0], 128 * WGS);
        mbar_init(&xch_bar[1], 128 * WGS);
#pragma unroll
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&kv_full[s], 1);
            mbar_init(&kv_empty[s], 1);
        }
#pragma unroll
        for (int b = 0; b < 2; ++b) {
            mbar_init(&s_full[b], 1);
            mbar_init(&p_full[b], 128 * WGS);   // every softmax thread, after writing its P
            mbar_init(&pv_done[b], 1);
            mbar_init(&o_free[b], 128 * WGS);   // every softmax thread, after reading the output
        }
        fence_mbar_init();
        abort_s = 0;
    }
    if (warp == 0) tmem_alloc<C::TMEM_COLS>(&tmem_base_s);
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = tmem_base_s;
    const unsigned long long limit = a.timeout_ns;
    const bool wide_out = (reinterpret_cast<uintptr_t>(a.out) & 31u) == 0;  // 32-byte output stores

    if (warp == C::PRODUCER_WARP) {
        // ================= TMA producer =================
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&qmap)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&kmap)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&vmap)) : "memory");
            uint32_t gt = 0, ic = 0, q_issued = 0;  // tiles, items and Q loads issued
            bool ok = true;
            for (int rd = 0, idx = item_mirrored(0); ok && idx < n_items; ++rd, idx = item_mirrored(rd), ++ic) {
                const Item it = make_item<C::QT, C::NK>(idx, a.n, a.B);
                const int b = it.pair / a.Hkv, kvh = it.pair - b * a.Hkv;
                const uint32_t qb = ic % QBUF;
                if (ic >= QBUF && !mbar_wait(&q_empty[qb], ((ic / QBUF) - 1) & 1u, limit)) {
                    ok = false;
                    break;
                }
                mbar_expect_tx(&q_full[qb], static_cast<uint32_t>(C::Q_BYTES));
                const int qrow0 = (b * a.Hq + kvh * G) * a.n + it.t0;
                unsigned char* qdst = dsmem + C::Q_OFF + qb * C::Q_BYTES;
#pragma unroll
                for (int gi = 0; gi < G; ++gi)
#pragma unroll
                    for (int bx = 0; bx < C::BOXES; ++bx)
                        tma_load_2d(qdst + bx * C::QBOX + gi * C::QT * 128, &qmap, bx * 64, qrow0 + gi * a.n,
                                    &q_full[qb]);
                ++q_issued;
                const int krow0 = it.pair * a.n + it.lo;
                for (int j = 0; j < it.ntiles; ++j, ++gt) {
                    const int s = gt % STAGES;
                    if (gt >= STAGES && !mbar_wait(&kv_empty[s], ((gt / STAGES) - 1) & 1u, limit)) {
                        ok = false;
                        break;
                    }
                    if (abort_s) {
                        ok = false;
                        break;
                    }
                    unsigned char* st = dsmem + C::KV_OFF + s * C::KV_STAGE;
                    mbar_expect_tx(&kv_full[s], static_cast<uint32_t>(C::KV_STAGE));
#pragma unroll
                    for (int bx = 0; bx < C::BOXES; ++bx) {
                        tma_load_2d(st + bx * C::KBOX, &kmap, bx * 64, krow0 + j * C::NK, &kv_full[s]);
                        tma_load_2d(st + (C::BOXES + bx) * C::KBOX, &vmap, bx * 64, krow0 + j * C::NK, &kv_full[s]);
                    }
                }
            }
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
            }
            // drain: the last copies into each stage and into Q land before shared memory goes away
            for (uint32_t q = 0; q < QBUF && q < q_issued; ++q) {
                const uint32_t j = q + QBUF * ((q_issued - 1 - q) / QBUF);
                mbar_wait(&q_full[q], (j / QBUF) & 1u, kGuardNs);
            }
            for (uint32_t s = 0; s < STAGES && s < gt; ++s) {
                const uint32_t j = s + STAGES * ((gt - 1 - s) / STAGES);
                mbar_wait(&kv_full[s], (j / STAGES) & 1u, kGuardNs);
            }
        }
    } else if (warp == C::MMA_WARP) {
        // ================= MMA issuer =================
        if (lane == 0) {
            constexpr uint32_t idesc_s = umma_idesc_bf16(C::M, C::NK, 0);
            constexpr uint32_t idesc_o = umma_idesc_bf16(C::M, D, 1);
            const uint32_t kv_base = smem_addr(dsmem + C::KV_OFF);
            uint32_t gt = 0, ic = 0, q_base = 0;
            bool ok = true, issued_any = false;
            // S_g = Q K_g^T into S buffer g % 2
            auto issue_s = [&](uint32_t g) {
                const uint32_t kb = kv_base + (g % STAGES) * C::KV_STAGE;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (kk & 3) * 32;  // 16 columns = 32 bytes into the 128-byte row
                    const uint64_t ad = umma_desc_sw128(q_base + (kk >> 2) * C::QBOX + off, 16, 1024);
                    const uint64_t bd = umma_desc_sw128(kb + (kk >> 2) * C::KBOX + off, 16, 1024);
                    umma_bf16(tmem + C::T_S + (g & 1u) * C::NK, ad, bd, idesc_s, kk > 0 ? 1u : 0u);
                }
                umma_commit(&s_full[g & 1u]);
            };
            for (int rd = 0, idx = item_mirrored(0); ok && idx < n_items; ++rd, idx = item_mirrored(rd), ++ic) {
                const Item it = make_item<C::QT, C::NK>(idx, a.n, a.B);
                const uint32_t ob = ic % C::OBUF;
                const uint32_t qb = ic % QBUF;
                q_base = smem_addr(dsmem + C::Q_OFF + qb * C::Q_BYTES);
                if (!mbar_wait(&q_full[qb], (ic / QBUF) & 1u, limit) ||
                    !mbar_wait(&kv_full[gt % STAGES], (gt / STAGES) & 1u, limit)) {
                    ok = false;
                    break;
                }
                tmem_fence_after();
                issue_s(gt);
                issued_any = true;
                if (it.ntiles == 1) umma_commit(&q_empty[qb]);
                for (int j = 0; j < it.ntiles; ++j) {
                    const uint32_t g = gt + j;
                    if (j + 1 < it.ntiles) {
                        if (!mbar_wait(&kv_full[(g + 1) % STAGES], ((g + 1) / STAGES) & 1u, limit)) {
                            ok = false;
                            break;
                        }
                        tmem_fence_after();
                        issue_s(g + 1);
                        if (j + 2 == it.ntiles) umma_commit(&q_empty[qb]);  // the item's last read of Q
                    }
                    // before the item's first P.V: output buffer ob is free once every softmax thread
                    // has read the item before that used it
                    bool free_ok = true;
                    if (j == 0 && ic >= C::OBUF) free_ok = mbar_wait(&o_free[ob], ((ic / C::OBUF) - 1) & 1u, limit);
                    if (!free_ok || !mbar_wait(&p_full[g & 1u], (g >> 1) & 1u, limit)) {
                        ok = false;
                        break;
                    }
                    tmem_fence_after();
                    // O (+)= P_g V_g: P from TMEM (bf16 pairs over S buffer g % 2), V MN-major
                    const uint32_t pt = tmem + C::T_S + (g & 1u) * C::NK;
                    const uint32_t vb = kv_base + (g % STAGES) * C::KV_STAGE + C::BOXES * C::KBOX;
                    const uint32_t o_dst = tmem + C::T_O + ob * D;
                    const bool first = j == 0;
#pragma unroll
                    for (int kk = 0; kk < C::NK / 16; ++kk) {
                        const uint64_t bd = umma_desc_sw128(vb + kk * 2048, C::KBOX, 1024);
                        umma_bf16_tmem_a(o_dst, pt + 8 * kk, bd, idesc_o, (!first || kk > 0) ? 1u : 0u);
                    }
                    umma_commit(&pv_done[g & 1u]);
                    umma_commit(&kv_empty[g % STAGES]);
                }
                gt += it.ntiles;
            }
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
            }
            if (issued_any) {  // every MMA complete before TMEM is released
                umma_commit(&done_bar);
                mbar_wait(&done_bar, 0u, kGuardNs);
            }
        }
    } else {
        // ================= softmax =================
        // Thread r of a warpgroup owns query row r (TMEM lane r). With two warpgroups both take
        // every tile: warpgroup wg works on the score columns [wg NK/2, (wg+1) NK/2) and the
        // output columns [wg d/2, (wg+1) d/2) of its rows. They exchange their partial row maxima
        // through shared memory every tile, so both keep the same reference maximum, and their
        // partial row sums at the item's end.
        constexpr int HC = C::NK / WGS;  // score columns of this thread
        constexpr int OC = D / WGS;      // output columns of this thread
        const int wg = warp >> 2, r = tid & 127;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
        const int h = a.B >> 1;
        const int gi = r / C::QT, rp = r - gi * C::QT;
        uint32_t gt = 0, ic = 0;
        bool ok = true;
        for (int rd = 0, idx = item_mirrored(0); ok && idx < n_items; ++rd, idx = item_mirrored(rd), ++ic) {
            const Item it = make_item<C::QT, C::NK>(idx, a.n, a.B);
            const uint32_t ob = ic % C::OBUF;
            const uint32_t o_col = C::T_O + ob * D + wg * OC;  // this thread's output columns
            const int t = it.t0 + rp;               // this row's position
            const int as = support_start(t, h);     // and its support start
            float m_used = -INFINITY, l = 0.f;
            for (int j = 0; j < it.ntiles; ++j) {
                const uint32_t g = gt + j;
                if (!warp_wait(&s_full[g & 1u], (g >> 1) & 1u, limit) || __any_sync(0xffffffffu, abort_s != 0)) {
                    ok = false;
                    break;
                }
                tmem_fence_after();
                const uint32_t s_row = lane_base + C::T_S + (g & 1u) * C::NK;
                float z[HC];  // raw scores q.k of this thread's columns: every load issued, one wait
                if constexpr (HC >= 32) {
#pragma unroll
                    for (int c = 0; c < HC / 32; ++c) {
                        uint32_t v[32];
                        tmem_ld32(s_row + wg * HC + 32 * c, v);
#pragma unroll
                        for (int x = 0; x < 32; ++x) z[32 * c + x] = __uint_as_float(v[x]);
                    }
                } else {
                    uint32_t v[16];
                    tmem_ld16(s_row + wg * HC, v);
#pragma unroll
                    for (int x = 0; x < 16; ++x) z[x] = __uint_as_float(v[x]);
                }
                tmem_wait_ld();
                const int tile0 = it.lo + j * C::NK;   // first key of the tile
                const int key0 = tile0 + wg * HC;      // first key of this thread's columns
                if (tile0 + C::NK - 1 > it.t0) {       // the diagonal: keys past some row's own position
                    const int hi = t - key0;           // this row's last visible column
#pragma unroll
                    for (int c = 0; c < HC; ++c) z[c] = c <= hi ? z[c] : -INFINITY;
                }
                if (tile0 < it.a_max) {                // some row's support starts inside this tile
                    const int lo = as - key0;          // this row's first visible column
#pragma unroll
                    for (int c = 0; c < HC; ++c) z[c] = c >= lo ? z[c] : -INFINITY;
                }
                // row maximum: two independent chains of three-input maxima
                float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
                for (int c = 0; c < HC; c += 4) {
                    mx0 = fmax3(mx0, z[c], z[c + 1]);
                    mx1 = fmax3(mx1, z[c + 2], z[c + 3]);
                }
                float mx = fmaxf(mx0, mx1) * qscale;  // the scale is positive: the maximum of the scaled scores
                if constexpr (WGS == 2) {
                    // the other warpgroup's half of the row (both warps read both halves' maxima)
                    xch_s[g & 1u][wg][r] = mx;
                    mbar_arrive(&xch_bar[g & 1u]);
                    if (!warp_wait(&xch_bar[g & 1u], (g >> 1) & 1u, limit)) {
                        ok = false;
                        break;
                    }
                    mx = fmaxf(mx, xch_s[g & 1u][wg ^ 1][r]);
                }
                // the reference maximum moves only when the row maximum exceeds it by 2^8:
                // weights stay below 2^8, and O and l are rescaled together, so o = O / l is exact
                const bool grow = mx > m_used + 8.f;
                const float m_new = grow ? mx : m_used;
                if (__any_sync(0xffffffffu, grow)) {
                    const float f = grow ? (m_used == -INFINITY ? 0.f : fast_exp2(m_used - m_new)) : 1.f;
                    l *= f;
                    if (j > 0) {  // O holds the item's earlier tiles once P.V of the previous one is complete
                        const uint32_t gp = g - 1;
                        if (!warp_wait(&pv_done[gp & 1u], (gp >> 1) & 1u, limit)) {
                            ok = false;
                            break;
                        }
                        tmem_fence_after();
                        if constexpr (C::CTAS >= 3) {
#pragma unroll
                            for (int c = 0; c < OC / 16; ++c) {
                                uint32_t v[16];
                                const uint32_t ta = lane_base + o_col + 16 * c;
                                tmem_ld16(ta, v);
                                tmem_wait_ld();
#pragma unroll
                                for (int x = 0; x < 16; ++x) v[x] = __float_as_uint(__uint_as_float(v[x]) * f);
                                tmem_st16(ta, v);
                            }
                        } else {
#pragma unroll
                            for (int c = 0; c < OC / 32; ++c) {
                                uint32_t v[32];
                                const uint32_t ta = lane_base + o_col + 32 * c;
                                tmem_ld32(ta, v);
                                tmem_wait_ld();
#pragma unroll
                                for (int x = 0; x < 32; ++x) v[x] = __float_as_uint(__uint_as_float(v[x]) * f);
                                tmem_st32(ta, v);
                            }
                        }
                        tmem_wait_st();
                    }
                    m_used = m_new;
                }
                const float nbase = m_used == -INFINITY ? 0.f : -m_used;
                // P = exp2(z * scale - m) as bf16 pairs over the first NK/2 columns of the S row (this
                // thread's HC/2 of them, over columns read before the exchange); the arguments and the
                // row sum use packed two-lane FMA and add
                const float2 sc2 = make_float2(qscale, qscale), nb2 = make_float2(nbase, nbase);
                float2 lacc = make_float2(0.f, 0.f);
                if constexpr (HC == 32) {
                    uint32_t pk[16];
#pragma unroll
                    for (int x = 0; x < 16; ++x) {
                        const float2 arg = __ffma2_rn(make_float2(z[2 * x], z[2 * x + 1]), sc2, nb2);
                        const float2 e = make_float2(fast_exp2(arg.x), fast_exp2(arg.y));
                        lacc = __fadd2_rn(lacc, e);
                        pk[x] = pack_bf16x2(e.x, e.y);
                    }
                    tmem_st16(s_row + wg * 16, pk);
                } else {
#pragma unroll
                    for (int c = 0; c < HC / 64; ++c) {
                        uint32_t pk[32];
#pragma unroll
                        for (int x = 0; x < 32; ++x) {
                            const float2 arg = __ffma2_rn(make_float2(z[64 * c + 2 * x], z[64 * c + 2 * x + 1]), sc2, nb2);
                            const float2 e = make_float2(fast_exp2(arg.x), fast_exp2(arg.y));
                            lacc = __fadd2_rn(lacc, e);
                            pk[x] = pack_bf16x2(e.x, e.y);
                        }
                        tmem_st32(s_row + wg * (HC / 2) + 32 * c, pk);
                    }
                }
                l += lacc.x + lacc.y;
                tmem_wait_st();
                tmem_fence_before();   // P is in TMEM and this row of S has been read
                mbar_arrive(&p_full[g & 1u]);
            }
            if (!ok) break;
            // ---- epilogue: the item's last P.V, then o = O / l and lse
            {
                const uint32_t gl = gt + it.ntiles - 1;
                if (!warp_wait(&pv_done[gl & 1u], (gl >> 1) & 1u, limit)) {
                    ok = false;
                    break;
                }
            }
            float l_tot = l;
            if constexpr (WGS == 2) {  // the row sum is the two warpgroups' partial sums (same reference)
                lsum_s[ic & 1u][wg][r] = l;
                mbar_arrive(&lsum_bar);
                if (!warp_wait(&lsum_bar, ic & 1u, limit)) {
                    ok = false;
                    break;
                }
                l_tot = lsum_s[ic & 1u][0][r] + lsum_s[ic & 1u][1][r];
            }
            const bool valid = t < a.n;
            const int b = it.pair / a.Hkv, kvh = it.pair - b * a.Hkv;
            const size_t row = static_cast<size_t>(b * a.Hq + kvh * G + gi) * a.n + t;
            tmem_fence_after();
            const float inv = l_tot > 0.f ? 1.f / l_tot : 0.f;
            constexpr int EC = C::CTAS >= 3 ? 16 : 32;  // output columns per TMEM load
#pragma unroll
            for (int c = 0; c < OC / EC; ++c) {
                uint32_t v[EC];
                if constexpr (EC == 16) tmem_ld16(lane_base + o_col + EC * c, v);
                else tmem_ld32(lane_base + o_col + EC * c, v);
                tmem_wait_ld();
                float o[EC];
#pragma unroll
                for (int x = 0; x < EC; ++x) o[x] = __uint_as_float(v[x]) * inv;
                if (valid) store_chunk<EC>(a.out, a.out_f32, row * D + wg * OC + EC * c, o, wide_out);
            }
            tmem_fence_before();
            mbar_arrive(&o_free[ob]);  // the next item may overwrite the output buffer
            if (valid && a.lse != nullptr && wg == 0) {
                // ln sum exp(z) = (m + log2 l) ln 2, m the base-2 reference maximum
                a.lse[row] = (m_used + log2f(l_tot)) * 0.6931471805599453f;
            }
            gt += it.ntiles;
        }
        if (!ok) {
            abort_s = 1;
            atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
        }
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    if (warp == 0) tmem_dealloc<C::TMEM_COLS>(tmem);
}

// ------------------------------------------------------------ paired items ----
// Long supports (B a multiple of 256, so every support starts on a 128-key tile boundary):
// each CTA takes two consecutive query tiles (items A and B) of one (sequence, KV head), which
// need the same keys except where B's support starts a half-block later, and streams their
// union once. Warps 0-3 run the softmax of A, warps 4-7 that of B, each over its own S and
// output in TMEM, so one warpgroup's softmax runs while the tensor pipe works on the other's
// products, and the issuing thread queues four groups (S and P.V of both) per K/V tile. The
// softmax warpgroups take 216 registers a thread (setmaxnreg) from the warpgroup of the Q, K and
// V producers and the MMA issuer.
template <int D, int G>
struct PairCfg {
    static constexpr int NK = 128, M = 128, QT = M / G, BOXES = D / 64;
    static constexpr int QBOX = M * 128, KBOX = NK * 128;
    static constexpr int Q_BYTES = BOXES * QBOX;           // one item's Q
    static constexpr int TILE = BOXES * KBOX;              // one K or V tile
    static constexpr int Q_OFF = 0;                        // Q of A, then Q of B
    static constexpr int K_OFF = 2 * Q_BYTES;
    static constexpr int STATIC_SMEM = 1024;
    static constexpr int BUDGET = 228 * 1024 - 1024 - STATIC_SMEM - 1024;
    static constexpr int TILE_ROOM = (BUDGET - K_OFF) / TILE;
    static constexpr int KSTAGES = (TILE_ROOM + 1) / 2 < 4 ? (TILE_ROOM + 1) / 2 : 4;
    static constexpr int VSTAGES = TILE_ROOM - KSTAGES < 4 ? TILE_ROOM - KSTAGES : 4;
    static constexpr int V_OFF = K_OFF + KSTAGES * TILE;
    static constexpr int SMEM = V_OFF + VSTAGES * TILE + 1024;
    static constexpr int T_S = 0, T_O = 2 * NK;            // S of A and B, then the outputs
    // Iteration i of the issuing thread (K_j for S, V_{j-1} for P.V) waits on kv_full[i mod KVR],
    // which the K and the V producer each arrive on once per iteration, with their copy's bytes
    // or without a copy. Before copying tile t into a ring of S stages, a producer waits for tile
    // t - S to be freed, which happens after the issuing thread has passed that tile's
    // iteration. Those S tiles span at most 2 S iterations (one extra iteration per item, when
    // every item has one tile), and a copy may be followed by one arrival without a copy: a
    // producer arrives for iterations at most 2 S past the last one the issuing thread has
    // passed. A slot may take the arrivals of iteration i once the issuing thread has passed
    // i - KVR, so KVR >= 2 S + 1 suffices; it keeps one slot more: 8 at d = 128 (3 K and 2 V
    // stages), 10 at d = 64 (4 and 4).
    static constexpr int KVR = 2 * (KSTAGES > VSTAGES ? KSTAGES : VSTAGES) + 2;
    static_assert(KVR > 2 * KSTAGES && KVR > 2 * VSTAGES, "kv_full ring shorter than a producer's lead");
    // warps 0-7 softmax, 8 K producer, 9 V producer, 10 MMA issuer, 11 Q producer; at launch
    // 168 registers each (12 warps, three per SMSP). setmaxnreg is uniform per warpgroup and
    // the register file is split between the SMSPs, so each SMSP's three warps (two softmax,
    // one of warpgroup 2) must fit their launch share: 2 x 216 + 72 = 3 x 168, and over the
    // CTA 256 x 216 + 128 x 72 = 384 x 168
    static constexpr int THREADS = 384, W_K = 8, W_V = 9, W_MMA = 10, W_Q = 11;
    static constexpr int LAUNCH_REGS = 168;
    static constexpr int SOFTMAX_REGS = 216, OTHER_REGS = 72;
    static_assert(2 * SOFTMAX_REGS + OTHER_REGS <= 3 * LAUNCH_REGS, "register split per SMSP");
    static_assert(256 * SOFTMAX_REGS + 128 * OTHER_REGS <= THREADS * LAUNCH_REGS, "register split");
    static_assert(T_O + 2 * D <= 512, "TMEM budget");
    static_assert(KSTAGES >= 2 && VSTAGES >= 2, "shared memory budget");
    static_assert(SMEM + STATIC_SMEM + 1024 <= 228 * 1024, "shared memory budget");
    static_assert(QT % 8 == 0, "a head's Q rows must start on a swizzle atom (8 rows)");
};

// Two items of one (sequence, KV head): A = query tile 2s, B = 2s + 1 (absent past the end).
// Their keys are [loA, end], in tiles of NK from loA; A takes tiles [0, ntA), B [jB0, nt).
struct PItem {
    int pair, t0, tlA, tlB, loA, loB, amaxA, amaxB, nt, ntA, jB0;
    bool hasB;
};

template <int QT, int NK>
__device__ __forceinline__ PItem make_pitem(int sidx, int n, int B)
{
    const int nq = (n + QT - 1) / QT;
    const int nsp = (nq + 1) / 2;
    PItem it;
    it.pair = sidx / nsp;
    it.t0 = (sidx - it.pair * nsp) * 2 * QT;
    it.tlA = min(it.t0 + QT, n) - 1;
    it.hasB = it.t0 + QT < n;
    it.tlB = it.hasB ? min(it.t0 + 2 * QT, n) - 1 : it.tlA;
    const int h = B >> 1;
    it.loA = support_start(it.t0, h);
    it.amaxA = support_start(it.tlA, h);
    it.loB = it.hasB ? support_start(it.t0 + QT, h) : it.loA;
    it.amaxB = support_start(it.tlB, h);
    it.nt = (it.tlB - it.loA + NK) / NK;
    it.ntA = (it.tlA - it.loA + NK) / NK;
    it.jB0 = (it.loB - it.loA) / NK;  // exact: supports start on multiples of h, h a multiple of NK
    return it;
}

// setmaxnreg is a warpgroup instruction: the four warps of a warpgroup execute the same one.
__device__ __forceinline__ void regs_inc_softmax() { asm volatile("setmaxnreg.inc.sync.aligned.u32 216;\n" ::: "memory"); }
__device__ __forceinline__ void regs_dec_others() { asm volatile("setmaxnreg.dec.sync.aligned.u32 72;\n" ::: "memory"); }

template <int D, int G>
__global__ void __launch_bounds__(PairCfg<D, G>::THREADS, 1)
forward_pair_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                    const __grid_constant__ CUtensorMap vmap, const ForwardArgs a)
{
    using C = PairCfg<D, G>;
    constexpr int NK = C::NK, KS = C::KSTAGES, VS = C::VSTAGES;
    extern __shared__ unsigned char dsmem_raw[];
    __shared__ __align__(8) uint64_t q_full[2], q_empty[2], done_bar;
    __shared__ __align__(8) uint64_t kv_full[C::KVR], k_empty[KS], v_empty[VS];
    __shared__ __align__(8) uint64_t s_full[2], p_full[2], pv_last[2], o_free[2];  // per item (A, B)
    __shared__ uint32_t tmem_base_s;
    __shared__ volatile int abort_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nq = (a.n + C::QT - 1) / C::QT;
    const int n_sitems = a.batch * a.Hkv * ((nq + 1) / 2);

    if (tid == 0) {
#pragma unroll
        for (int x = 0; x < 2; ++x) {
            mbar_init(&q_full[x], 1);
            mbar_init(&q_empty[x], 1);
            mbar_init(&s_full[x], 1);
            mbar_init(&p_full[x], 128);
            mbar_init(&pv_last[x], 1);
            mbar_init(&o_free[x], 128);
        }
        mbar_init(&done_bar, 1);
#pragma unroll
        for (int s = 0; s < C::KVR; ++s) mbar_init(&kv_full[s], 2);  // the K and the V producer
#pragma unroll
        for (int s = 0; s < KS; ++s) mbar_init(&k_empty[s], 1);
#pragma unroll
        for (int s = 0; s < VS; ++s) mbar_init(&v_empty[s], 1);
        fence_mbar_init();
        abort_s = 0;
    }
    if (warp == 0) tmem_alloc<512>(&tmem_base_s);
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = tmem_base_s;
    const unsigned long long limit = a.timeout_ns;
    const bool wide_out = (reinterpret_cast<uintptr_t>(a.out) & 31u) == 0;  // 32-byte output stores
    // warpgroup 2 (producers, MMA issuer, spare) gives registers to warpgroups 0 and 1 (softmax):
    // each warpgroup's four warps run one setmaxnreg, at one place, ahead of its roles
    if (warp >= 8) {
        regs_dec_others();
        if (warp == C::W_K || warp == C::W_V || warp == C::W_Q) {
            // ================= TMA producers: Q of both items, K tiles, V tiles =================
            // (Q on a warp of its own, so that the K tiles of the next item need not wait for the
            // Q buffers, which free only after the current item's last S)
            const bool qk = warp == C::W_K;
            const bool q_role = warp == C::W_Q;
            const bool tiles = !q_role;
            if (lane == 0) {
                if (tiles) asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(qk ? &kmap : &vmap)) : "memory");
                if (q_role) asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&qmap)) : "memory");
                uint32_t gt = 0, gi = 0, armed = 0, ic[2] = {0, 0}, q_issued[2] = {0, 0};
                bool ok = true;
                for (int rd = 0, sidx = item_mirrored(0); ok && sidx < n_sitems; ++rd, sidx = item_mirrored(rd)) {
                    const PItem it = make_pitem<C::QT, NK>(sidx, a.n, a.B);
                    const int b = it.pair / a.Hkv, kvh = it.pair - b * a.Hkv;
                    if (q_role) {
                        for (int x = 0; x < (it.hasB ? 2 : 1); ++x) {
                            if (ic[x] >= 1 && !mbar_wait(&q_empty[x], (ic[x] - 1) & 1u, limit)) {
                                ok = false;
                                break;
                            }
                            mbar_expect_tx(&q_full[x], static_cast<uint32_t>(C::Q_BYTES));
                            const int qrow0 = (b * a.Hq + kvh * G) * a.n + it.t0 + x * C::QT;
                            unsigned char* qdst = dsmem + C::Q_OFF + x * C::Q_BYTES;
#pragma unroll
                            for (int gi = 0; gi < G; ++gi)
#pragma unroll
                                for (int bx = 0; bx < C::BOXES; ++bx)
                                    tma_load_2d(qdst + bx * C::QBOX + gi * C::QT * 128, &qmap, bx * 64,
                                                qrow0 + gi * a.n, &q_full[x]);
                            ++ic[x];
                            q_issued[x] = ic[x];
                        }
                        if (!ok) break;
                    }
                    const int row0 = it.pair * a.n + it.loA;
                    // iterations j = 0 .. nt: K_j for j < nt, V_{j-1} for j >= 1
                    for (int j = 0; tiles && j <= it.nt; ++j, ++gi) {
                        if (abort_s) {
                            ok = false;
                            break;
                        }
                        uint64_t* fullb = &kv_full[gi % C::KVR];
                        if (qk ? j == it.nt : j == 0) {
                            mbar_arrive(fullb);
                            continue;
                        }
                        const int ns = qk ? KS : VS;
                        const int s = gt % ns;
                        uint64_t* emptyb = qk ? &k_empty[s] : &v_empty[s];
                        if (gt >= static_cast<uint32_t>(ns) && !mbar_wait(emptyb, ((gt / ns) - 1) & 1u, limit)) {
                            ok = false;
                            break;
                        }
                        unsigned char* st = dsmem + (qk ? C::K_OFF : C::V_OFF) + s * C::TILE;
                        const int tile = qk ? j : j - 1;
                        mbar_expect_tx(fullb, static_cast<uint32_t>(C::TILE));
#pragma unroll
                        for (int bx = 0; bx < C::BOXES; ++bx)
                            tma_load_2d(st + bx * C::KBOX, qk ? &kmap : &vmap, bx * 64, row0 + tile * NK, fullb);
                        ++gt;
                        armed = gi + 1;
                    }
                }
                if (!ok) {
                    abort_s = 1;
                    atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
                }
                // drain the copies still in flight before shared memory goes away
                for (int x = 0; x < 2; ++x)
                    if (q_issued[x] > 0) mbar_wait(&q_full[x], (q_issued[x] - 1) & 1u, kGuardNs);
                for (uint32_t i = armed > C::KVR ? armed - C::KVR : 0; i < armed; ++i)
                    mbar_wait(&kv_full[i % C::KVR], (i / C::KVR) & 1u, kGuardNs);
            }
        } else if (warp == C::W_MMA) {
            // ================= MMA issuer =================
            if (lane == 0) {
                constexpr uint32_t idesc_s = umma_idesc_bf16(C::M, NK, 0);
                constexpr uint32_t idesc_o = umma_idesc_bf16(C::M, D, 1);
                const uint32_t q_base = smem_addr(dsmem + C::Q_OFF);
                const uint32_t k_base = smem_addr(dsmem + C::K_OFF), v_base = smem_addr(dsmem + C::V_OFF);
                uint32_t gk = 0, gv = 0, gi = 0;          // K and V tiles consumed, iterations
                uint32_t ic[2] = {0, 0}, gp[2] = {0, 0};  // items and P tiles consumed, per item slot
                bool ok = true, issued_any = false;
                for (int rd = 0, sidx = item_mirrored(0); ok && sidx < n_sitems; ++rd, sidx = item_mirrored(rd)) {
                    const PItem it = make_pitem<C::QT, NK>(sidx, a.n, a.B);
                    const int jb[2] = {0, it.hasB ? it.jB0 : it.nt};  // first and end tile of each item
                    const int je[2] = {it.ntA, it.nt};
                    for (int j = 0; ok && j <= it.nt; ++j, ++gi) {
                        const bool need_k = j < it.nt, need_v = j >= 1;  // K_j, V_{j-1}
                        if (!mbar_wait(&kv_full[gi % C::KVR], (gi / C::KVR) & 1u, limit)) {
                            ok = false;
                            break;
                        }
                        const uint32_t kb = k_base + (gk % KS) * C::TILE, vb = v_base + (gv % VS) * C::TILE;
#pragma unroll
                        for (int x = 0; x < 2; ++x) {
                            const bool pv = j >= jb[x] + 1 && j - 1 < je[x];  // P_x V of tile j - 1
                            const bool sk = j >= jb[x] && j < je[x];          // S_x of tile j
                            if (pv) {
                                const bool first = j - 1 == jb[x];
                                if ((first && ic[x] >= 1 && !mbar_wait(&o_free[x], (ic[x] - 1) & 1u, limit)) ||
                                    !mbar_wait(&p_full[x], gp[x] & 1u, limit)) {
                                    ok = false;
                                    break;
                                }
                                tmem_fence_after();
                                const uint32_t pt = tmem + C::T_S + x * NK, o_dst = tmem + C::T_O + x * D;
#pragma unroll
                                for (int kk = 0; kk < NK / 16; ++kk) {
                                    const uint64_t bd = umma_desc_sw128(vb + kk * 2048, C::KBOX, 1024);
                                    umma_bf16_tmem_a(o_dst, pt + 8 * kk, bd, idesc_o, (!first || kk > 0) ? 1u : 0u);
                                }
                                ++gp[x];
                            }
                            if (sk) {
                                if (j == jb[x]) {
                                    if (!mbar_wait(&q_full[x], ic[x] & 1u, limit)) {
                                        ok = false;
                                        break;
                                    }
                                    tmem_fence_after();
                                }
                                const uint32_t qb = q_base + x * C::Q_BYTES;
#pragma unroll
                                for (int kk = 0; kk < D / 16; ++kk) {
                                    const uint32_t off = (kk & 3) * 32;
                                    const uint64_t ad = umma_desc_sw128(qb + (kk >> 2) * C::QBOX + off, 16, 1024);
                                    const uint64_t bd = umma_desc_sw128(kb + (kk >> 2) * C::KBOX + off, 16, 1024);
                                    umma_bf16(tmem + C::T_S + x * NK, ad, bd, idesc_s, kk > 0 ? 1u : 0u);
                                }
                                umma_commit(&s_full[x]);      // S_x of tile j, and P_x V of tile j - 1
                                if (j == je[x] - 1) umma_commit(&q_empty[x]);
                            } else if (pv) {
                                umma_commit(&pv_last[x]);     // the item's last P.V
                                ++ic[x];
                            }
                            issued_any = true;
                        }
                        if (!ok) break;
                        gk += need_k;  // the softmax warpgroups release the K and V stages
                        gv += need_v;
                    }
                }
                if (!ok) {
                    abort_s = 1;
                    atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
                }
                if (issued_any) {  // every MMA complete before TMEM is released
                    umma_commit(&done_bar);
                    mbar_wait(&done_bar, 0u, kGuardNs);
                }
            }
        }
    } else {
        regs_inc_softmax();
        // ================= softmax of item x (warps 4x .. 4x + 3) =================
        const int x = warp >> 2, r = tid & 127;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        const uint32_t s_row = lane_base + C::T_S + x * NK, o_row = lane_base + C::T_O + x * D;
        const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
        const int h = a.B >> 1;
        const int gi = r / C::QT, rp = r - gi * C::QT;
        uint32_t g = 0, ic = 0;  // this item slot's tiles and items so far
        uint32_t gkv = 0;        // K (and V) tiles of the items before this one
        bool ok = true;
        for (int rd = 0, sidx = item_mirrored(0); ok && sidx < n_sitems; ++rd, sidx = item_mirrored(rd)) {
            const PItem it = make_pitem<C::QT, NK>(sidx, a.n, a.B);
            const uint32_t gk0 = gkv;
            gkv += it.nt;
            if (x == 1 && !it.hasB) continue;
            // K/V stages are freed here rather than by commits of the issuing thread, whose every
            // barrier operation delays its next products. Its last commit of iteration j (after S
            // of both items on K_j and P.V of both on V_{j-1}) is item B's s_full where B has tile
            // j, else item A's (A owns the iterations below jB0, all of them without B); iteration
            // nt, the last P.V, ends with pv_last of B, or of A without B. The owner's first thread
            // frees K_j and V_{j-1} once it has seen that commit: K_j sits in stage (gk0 + j) mod
            // KS, V_j in (gk0 + j) mod VS.
            const int jown = (tid & 127) != 0 ? -1 : x == 1 ? it.nt : (it.hasB ? it.jB0 : it.nt);
            const int t0 = it.t0 + x * C::QT, tl = x == 0 ? it.tlA : it.tlB;
            const int amax = x == 0 ? it.amaxA : it.amaxB;
            const int jb = x == 0 ? 0 : it.jB0, je = x == 0 ? it.ntA : it.nt;
            const int t = t0 + rp;                  // this row's position
            const int as = support_start(t, h);     // and its support start
            float m_used = -INFINITY, l = 0.f;
            for (int j = jb; j < je; ++j, ++g) {
                if (!warp_wait(&s_full[x], g & 1u, limit) || __any_sync(0xffffffffu, abort_s != 0)) {
                    ok = false;
                    break;
                }
                if (j < jown) {
                    mbar_arrive(&k_empty[(gk0 + j) % KS]);
                    if (j >= 1) mbar_arrive(&v_empty[(gk0 + j - 1) % VS]);
                }
                tmem_fence_after();
                float z[NK];  // raw scores q.k of this row: every load issued, one wait
#pragma unroll
                for (int c = 0; c < NK / 32; ++c) {
                    uint32_t v[32];
                    tmem_ld32(s_row + 32 * c, v);
#pragma unroll
                    for (int y = 0; y < 32; ++y) z[32 * c + y] = __uint_as_float(v[y]);
                }
                tmem_wait_ld();
                const int key0 = it.loA + j * NK;
                if (key0 + NK - 1 > t0) {  // the diagonal: keys past some row's own position
                    const int hi = t - key0;
#pragma unroll
                    for (int c = 0; c < NK; ++c) z[c] = c <= hi ? z[c] : -INFINITY;
                }
                if (key0 < amax) {         // some row's support starts inside this tile
                    const int lo = as - key0;
#pragma unroll
                    for (int c = 0; c < NK; ++c) z[c] = c >= lo ? z[c] : -INFINITY;
                }
                // P = exp2(z * scale - m) as bf16 pairs over the first half of this row's S
                // columns, one 64-key half at a time; the arguments and the row sum in packed
                // two-lane FMA and add
                const float2 sc2 = make_float2(qscale, qscale);
                auto write_p = [&](int c, float m) {
                    const float nb = m == -INFINITY ? 0.f : -m;
                    const float2 nb2 = make_float2(nb, nb);
                    float2 la = make_float2(0.f, 0.f), lb = la;
                    uint32_t pk[32];
#pragma unroll
                    for (int y = 0; y < 32; ++y) {
                        const float2 arg = __ffma2_rn(make_float2(z[64 * c + 2 * y], z[64 * c + 2 * y + 1]), sc2, nb2);
                        const float2 e = make_float2(fast_exp2(arg.x), fast_exp2(arg.y));
                        if (y & 1) lb = __fadd2_rn(lb, e);
                        else la = __fadd2_rn(la, e);
                        pk[y] = pack_bf16x2(e.x, e.y);
                    }
                    tmem_st32(s_row + 32 * c, pk);
                    return __fadd2_rn(la, lb);
                };
                // after the item's first tile the reference maximum seldom moves, so the first
                // half of P is formed against it while the row maximum is found, and formed again
                // only if it moved
                const bool first = j == jb;
                float2 l0 = make_float2(0.f, 0.f);
                if (!first) l0 = write_p(0, m_used);
                float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
#pragma unroll
                for (int c = 0; c < NK; c += 8) {
                    mx0 = fmax3(mx0, z[c], z[c + 1]);
                    mx1 = fmax3(mx1, z[c + 2], z[c + 3]);
                    mx2 = fmax3(mx2, z[c + 4], z[c + 5]);
                    mx3 = fmax3(mx3, z[c + 6], z[c + 7]);
                }
                const float mx = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * qscale;
                // the reference maximum moves only when the row maximum exceeds it by 2^8
                // (see forward_kernel); s_full of this tile also covers P.V of the previous one,
                // so O holds every earlier tile when it is rescaled
                const bool grow = mx > m_used + 8.f;
                const float m_new = grow ? mx : m_used;
                const bool moved = __any_sync(0xffffffffu, grow);
                if (moved) {
                    const float f = grow ? (m_used == -INFINITY ? 0.f : fast_exp2(m_used - m_new)) : 1.f;
                    l *= f;
                    if (j > jb) {
#pragma unroll
                        for (int c = 0; c < D / 32; ++c) {
                            uint32_t v[32];
                            tmem_ld32(o_row + 32 * c, v);
                            tmem_wait_ld();
#pragma unroll
                            for (int y = 0; y < 32; ++y) v[y] = __float_as_uint(__uint_as_float(v[y]) * f);
                            tmem_st32(o_row + 32 * c, v);
                        }
                        tmem_wait_st();
                    }
                    m_used = m_new;
                }
                if (first || moved) {
                    if (!first) tmem_wait_st();  // the first P's stores land before they are replaced
                    l0 = write_p(0, m_used);
                }
                const float2 l1 = write_p(1, m_used);
                l += (l0.x + l0.y) + (l1.x + l1.y);
                tmem_wait_st();
                tmem_fence_before();
                mbar_arrive(&p_full[x]);
            }
            if (!ok) break;
            // ---- epilogue: the item's last P.V, then o = O / l and lse
            if (!warp_wait(&pv_last[x], ic & 1u, limit)) {
                ok = false;
                break;
            }
            if ((tid & 127) == 0 && (x == 1 || !it.hasB)) mbar_arrive(&v_empty[(gk0 + it.nt - 1) % VS]);
            tmem_fence_after();
            const bool valid = t < a.n && t <= tl;
            const int b = it.pair / a.Hkv, kvh = it.pair - b * a.Hkv;
            const size_t row = static_cast<size_t>(b * a.Hq + kvh * G + gi) * a.n + t;
            const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t v[32];
                tmem_ld32(o_row + 32 * c, v);
                tmem_wait_ld();
                float o[32];
#pragma unroll
                for (int y = 0; y < 32; ++y) o[y] = __uint_as_float(v[y]) * inv;
                if (valid) store_chunk<32>(a.out, a.out_f32, row * D + 32 * c, o, wide_out);
            }
            tmem_fence_before();
            mbar_arrive(&o_free[x]);  // the next item of this slot may overwrite the output
            if (valid && a.lse != nullptr) a.lse[row] = (m_used + log2f(l)) * 0.6931471805599453f;
            ++ic;
        }
        if (!ok) {
            abort_s = 1;
            atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
        }
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    if (warp == 0) tmem_dealloc<512>(tmem);
}

// Sequence -> ring: slot j of each (sequence, KV head) ring gets the position
// s in [n-B, n-1] with s = j (mod B), zeros where s < 0 (Appendix F.1).
__global__ void seq_ring_kernel(const unsigned char* __restrict__ k, const unsigned char* __restrict__ v,
                                unsigned char* __restrict__ k_ring, unsigned char* __restrict__ v_ring,
                                long long pairs, int n, int B, int row_bytes)
{
    const int vecs = row_bytes / 16;
    const long long total = pairs * B * vecs;
    for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int x = static_cast<int>(i % vecs);
        const long long rs = i / vecs;
        const int slot = static_cast<int>(rs % B);
        const long long pr = rs / B;
        const long long first = static_cast<long long>(n) - B;  // oldest position the ring keeps
        long long off = (slot - first) % B;                      // s - first, s = slot (mod B)
        if (off < 0) off += B;
        const long long s = first + off;
        uint4 kv = make_uint4(0u, 0u, 0u, 0u), vv = kv;
        if (s >= 0) {
            const size_t src = (static_cast<size_t>(pr) * n + static_cast<size_t>(s)) * row_bytes + 16 * x;
            kv = *reinterpret_cast<const uint4*>(k + src);
            vv = *reinterpret_cast<const uint4*>(v + src);
        }
        const size_t dst = static_cast<size_t>(rs) * row_bytes + 16 * x;
        *reinterpret_cast<uint4*>(k_ring + dst) = kv;
        *reinterpret_cast<uint4*>(v_ring + dst) = vv;
    }
}

template <int D, int G, int NK, int WGS, int CTAS>
cudaError_t launch_fwd(const ForwardArgs& a, cudaStream_t stream, ForwardPlan* plan)
{
    using C = FwdCfg<D, G, NK, WGS, CTAS>;
    auto kernel = forward_kernel<D, G, NK, WGS, CTAS>;
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    // the shared-memory opt-in, then persistent CTAs: C::CTAS per SM where they fit, never more
    // than TMEM holds
    static std::atomic<int> per_sm_cache[kMaxCachedDevices] = {};
    const int per_sm = cached_per_device(per_sm_cache, dev, [&] {
        err = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        return err == cudaSuccess ? resident_ctas(kernel, C::THREADS, C::SMEM, C::CTAS, dev) : 0;
    });
    if (per_sm < 1) return err;
    const long long items = static_cast<long long>(a.batch) * a.Hkv * ((a.n + C::QT - 1) / C::QT);
    if (items < 1) {
        if (plan != nullptr) *plan = ForwardPlan{NK, 0, 0};
        return cudaSuccess;
    }
    if (items > 0x7fffffffLL) return cudaErrorInvalidValue;
    int sms = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    const long long slots = static_cast<long long>(sms) * per_sm;
    const int grid = static_cast<int>(items < slots ? items : slots);
    if (plan != nullptr) {
        *plan = ForwardPlan{NK, per_sm, grid};
        return cudaSuccess;
    }
    CUtensorMap qmap, kmap, vmap;
    const unsigned long long qrows = static_cast<unsigned long long>(a.batch) * a.Hq * a.n;
    const unsigned long long krows = static_cast<unsigned long long>(a.batch) * a.Hkv * a.n;
    if (!rows_tensor_map(&qmap, a.q, qrows, D, C::QT) || !rows_tensor_map(&kmap, a.k, krows, D, C::NK) ||
        !rows_tensor_map(&vmap, a.v, krows, D, C::NK))
        return cudaErrorInvalidValue;
    kernel<<<grid, C::THREADS, C::SMEM, stream>>>(qmap, kmap, vmap, a);
    return cudaGetLastError();
}

// The shape for long supports (B >= 512: an item spans several tiles) is a build-time choice:
// 0 = 128-key tiles, one softmax warpgroup; 1 = 128-key tiles, two softmax warpgroups sharing
// every tile.
#ifndef PBB_FWD_LONG_SHAPE
#define PBB_FWD_LONG_SHAPE 0
#endif

// Short supports (B < 512, an item is one to three tiles): 64-key tiles and two CTAs per SM, or
// at d = 64 (build option PBB_FWD_SHORT_SHAPE) 32-key tiles with three (1) or four (2) CTAs.
#ifndef PBB_FWD_SHORT_SHAPE
#define PBB_FWD_SHORT_SHAPE 1
#endif

// Long supports with B a multiple of 256 run the paired-item kernel (build option
// PBB_FWD_PAIR = 0 keeps them on forward_kernel's one-item shape).
#ifndef PBB_FWD_PAIR
#define PBB_FWD_PAIR 1
#endif

// 1: the paired kernel is usable on device dev; 2: its register split does not hold; 0: a
// runtime error (in *err). setmaxnreg moves registers within the block's launch allocation, so
// the split is only valid if the kernel launches with LAUNCH_REGS per thread (else an increase
// would wait forever); anything else falls back to the one-item kernel.
template <int D, int G>
int pair_kernel_usable(int dev, cudaError_t* err)
{
    using C = PairCfg<D, G>;
    auto kernel = forward_pair_kernel<D, G>;
    static std::atomic<int> state[kMaxCachedDevices] = {};
    return cached_per_device(state, dev, [&] {
        *err = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (*err != cudaSuccess) return 0;
        cudaFuncAttributes fa{};
        *err = cudaFuncGetAttributes(&fa, kernel);
        if (*err != cudaSuccess) return 0;
        return fa.numRegs == C::LAUNCH_REGS ? 1 : 2;
    });
}

template <int D, int G>
cudaError_t launch_fwd_pair(const ForwardArgs& a, cudaStream_t stream, ForwardPlan* plan)
{
    using C = PairCfg<D, G>;
    auto kernel = forward_pair_kernel<D, G>;
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    const int usable = pair_kernel_usable<D, G>(dev, &err);
    if (usable < 1) return err;
    if (usable != 1) return launch_fwd<D, G, 128, 1, 1>(a, stream, plan);
    const long long nq = (a.n + C::QT - 1) / C::QT;
    const long long sitems = static_cast<long long>(a.batch) * a.Hkv * ((nq + 1) / 2);
    if (sitems < 1) {
        if (plan != nullptr) *plan = ForwardPlan{C::NK, 0, 0};
        return cudaSuccess;
    }
    if (sitems > 0x7fffffffLL) return cudaErrorInvalidValue;
    int sms = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    const int grid = static_cast<int>(sitems < sms ? sitems : sms);
    if (plan != nullptr) {
        *plan = ForwardPlan{C::NK, 1, grid};
        return cudaSuccess;
    }
    CUtensorMap qmap, kmap, vmap;
    const unsigned long long qrows = static_cast<unsigned long long>(a.batch) * a.Hq * a.n;
    const unsigned long long krows = static_cast<unsigned long long>(a.batch) * a.Hkv * a.n;
    if (!rows_tensor_map(&qmap, a.q, qrows, D, C::QT) || !rows_tensor_map(&kmap, a.k, krows, D, C::NK) ||
        !rows_tensor_map(&vmap, a.v, krows, D, C::NK))
        return cudaErrorInvalidValue;
    kernel<<<grid, C::THREADS, C::SMEM, stream>>>(qmap, kmap, vmap, a);
    return cudaGetLastError();
}

// Blocks below this run the short-support shapes (measured at B = 4096, d = 128: the 64-key,
// two-CTA shape reaches 963 TFLOP/s against 1,186 for the 128-key, one-CTA shape).
#ifndef PBB_FWD_SHORT_MAX_B
#define PBB_FWD_SHORT_MAX_B 512
#endif

// Whether a call of these sizes takes the paired-item kernel's shape (which still falls back to
// the one-item kernel where its register split does not hold).
bool pair_shape(const ForwardArgs& a)
{
    return PBB_FWD_LONG_SHAPE != 1 && PBB_FWD_PAIR && a.B >= PBB_FWD_SHORT_MAX_B && (a.B / 2) % 128 == 0;
}

template <int D, int G>
cudaError_t launch_fwd_shape(const ForwardArgs& a, cudaStream_t stream, ForwardPlan* plan)
{
    if (a.B < PBB_FWD_SHORT_MAX_B) {
        if constexpr (D == 64 && PBB_FWD_SHORT_SHAPE == 1) return launch_fwd<D, G, 32, 1, 3>(a, stream, plan);
        if constexpr (D == 64 && PBB_FWD_SHORT_SHAPE == 2) return launch_fwd<D, G, 32, 1, 4>(a, stream, plan);
        return launch_fwd<D, G, 64, 1, 2>(a, stream, plan);
    }
#if PBB_FWD_LONG_SHAPE == 1
    return launch_fwd<D, G, 128, 2, 1>(a, stream, plan);
#else
    if (pair_shape(a)) return launch_fwd_pair<D, G>(a, stream, plan);
    return launch_fwd<D, G, 128, 1, 1>(a, stream, plan);
#endif
}

template <int D>
cudaError_t query_tiles_d(const ForwardArgs& a, int* query_tiles)
{
    *query_tiles = 1;
    if (!pair_shape(a)) return cudaSuccess;
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    int usable = 0;
    switch (a.Hq / a.Hkv) {
        case 1: usable = pair_kernel_usable<D, 1>(dev, &err); break;
        case 2: usable = pair_kernel_usable<D, 2>(dev, &err); break;
        case 4: usable = pair_kernel_usable<D, 4>(dev, &err); break;
        case 8: usable = pair_kernel_usable<D, 8>(dev, &err); break;
        default: return cudaErrorInvalidValue;
    }
    if (usable < 1) return err;
    if (usable == 1) *query_tiles = 2;
    return cudaSuccess;
}

template <int D>
cudaError_t launch_fwd_d(const ForwardArgs& a, cudaStream_t stream, ForwardPlan* plan)
{
    switch (a.Hq / a.Hkv) {
        case 1: return launch_fwd_shape<D, 1>(a, stream, plan);
        case 2: return launch_fwd_shape<D, 2>(a, stream, plan);
        case 4: return launch_fwd_shape<D, 4>(a, stream, plan);
        case 8: return launch_fwd_shape<D, 8>(a, stream, plan);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t forward_dispatch(const ForwardArgs& a, cudaStream_t stream, ForwardPlan* plan)
{
    if (a.d == 64) return launch_fwd_d<64>(a, stream, plan);
    if (a.d == 128) return launch_fwd_d<128>(a, stream, plan);
    return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_forward(const ForwardArgs& a, cudaStream_t stream) { return forward_dispatch(a, stream, nullptr); }

cudaError_t plan_forward(const ForwardArgs& a, ForwardPlan* plan) { return forward_dispatch(a, nullptr, plan); }

cudaError_t plan_forward_query_tiles(const ForwardArgs& a, int* query_tiles)
{
    if (a.d == 64) return query_tiles_d<64>(a, query_tiles);
    if (a.d == 128) return query_tiles_d<128>(a, query_tiles);
    return cudaErrorInvalidValue;
}

cudaError_t launch_seq_ring(const void* k, const void* v, void* k_ring, void* v_ring, int batch, int Hkv,
                            int n, int B, int row_bytes, cudaStream_t stream)
{
    const long long pairs = static_cast<long long>(batch) * Hkv;
    const long long total = pairs * B * (row_bytes / 16);
    if (total == 0) return cudaSuccess;
    const long long want = (total + 255) / 256;
    const int blocks = static_cast<int>(want < 4096 ? want : 4096);
    seq_ring_kernel<<<blocks, 256, 0, stream>>>(static_cast<const unsigned char*>(k),
                                                static_cast<const unsigned char*>(v),
                                                static_cast<unsigned char*>(k_ring),
                                                static_cast<unsigned char*>(v_ring), pairs, n, B, row_bytes);
    return cudaGetLastError();
}

cudaError_t read_and_clear_forward_status(int* status)
{
    cudaError_t err = cudaMemcpyFromSymbol(status, g_fwd_status, sizeof(int));
    if (err != cudaSuccess) return err;
    if (*status != kDevOk) {
        const int zero = kDevOk;
        err = cudaMemcpyToSymbol(g_fwd_status, &zero, sizeof(int));
    }
    return err;
}

}  // namespace pbb
