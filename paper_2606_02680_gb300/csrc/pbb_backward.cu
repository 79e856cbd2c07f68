// Gradients of the whole-sequence PBB attention (the backward pass) for sm_103a.
//
// With P_ts the softmax of z_ts = q_t.k_s / sqrt(d) over the support [a(t), t]
// (Eq. attention over Eq. pbb_relay), dO the upstream gradient and
// D_t = dO_t . o_t (= sum_s P_ts dP_ts):
//   dP_ts = dO_t . v_s,   dS_ts = P_ts (dP_ts - D_t),
//   dq_t = sum_s dS_ts k_s / sqrt(d),  dk_s = sum_t dS_ts q_t / sqrt(d),  dv_s = sum_t P_ts dO_t.
// P is recomputed from the forward's log-partition: P_ts = exp(z_ts - lse_t).
//
// Three kernels, none with floating-point atomics (results are deterministic):
//   delta_kernel       D for every row (dO . O);
//   bwd_kv_tc_kernel   items of 128 keys of one (sequence, KV head): it streams the
//                      query tiles (128 rows in the long shape, 32 in the short one: the
//                      G heads of the group stacked) whose supports hold any of its keys
//                      (positions s0 .. h(floor(s_last/h)+2)-1, the keys' own half-block
//                      and the next one, bridge rows included) and accumulates dK and dV
//                      in tensor memory;
//   bwd_q_tc_kernel    items of 128 query rows: it streams the key tiles of [a(t0), t_last]
//                      and accumulates dQ in tensor memory.
// Both are persistent on the fifth-generation tensor cores: a TMA producer warp
// (128-byte swizzle), one MMA-issuing lane (tcgen05.mma, completion through
// tcgen05.commit on mbarriers) and elementwise warpgroups; thread r of a warpgroup owns
// TMEM lane r. The long shape runs one CTA per SM with two elementwise warpgroups that
// share every tile, each on half of its columns (dQ pass: the scores of tile g sit in TMEM
// buffer g % 2, so tile g+1's products run while tile g's exponentials do; dK/dV pass: one
// buffer each for S^T and dP^T, the next dP^T issued once the warpgroups hold this one); the short shape
// (short supports, d = 64) runs two CTAs per SM with one warpgroup each, on half the TMEM. P, dS and their transposes are rounded
// to bf16 and written back over the scores in tensor memory as the A operands of the
// next products. Tiles with no masked entry take a packed path (two columns per
// ffma2/fadd2/fmul2, rounded like the scalar operations, so the results are the same
// bits). Every wait is bounded by the global timer; a wait that runs out records a
// timeout, every role stops, the MMAs and copies in flight are drained and TMEM is
// released.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pbb_device.cuh"
#include "pbb_internal.h"
#include "pbb_store.cuh"

namespace pbb {

__device__ int g_bwd_status;  // first fault recorded by a backward kernel, kDevOk if none

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr unsigned long long kGuardNs = 2000000000ull;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ int support_start(int t, int h)
{
    const int m = t / h;
    return m > 0 ? h * (m - 1) : 0;
}

// A bounded wait whose outcome is the same in every lane of the warp (warp-collective
// tcgen05 loads and stores follow it).
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, unsigned long long limit)
{
    return __all_sync(kFull, mbar_wait(bar, parity, limit));
}

// 32 fp32 gradients of one row, v scaled by f, to dst. A thread writes its own row, so each
// store instruction of a warp touches 32 lines: 32-byte stores halve those instructions where
// the gradient's base is 32-byte aligned (every 32-column chunk is then too); other bases take
// 16-byte stores.
__device__ __forceinline__ void store_row32(float* dst, const uint32_t (&v)[32], float f, bool wide)
{
    if (wide) {
#pragma unroll
        for (int x = 0; x < 4; ++x) {
            uint32_t w[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) w[i] = __float_as_uint(__uint_as_float(v[8 * x + i]) * f);
            st_global_v8(dst + 8 * x, w);
        }
    } else {
#pragma unroll
        for (int x = 0; x < 8; ++x)
            reinterpret_cast<float4*>(dst)[x] = make_float4(__uint_as_float(v[4 * x]) * f, __uint_as_float(v[4 * x + 1]) * f,
                                                            __uint_as_float(v[4 * x + 2]) * f, __uint_as_float(v[4 * x + 3]) * f);
    }
}

// 16 consecutive fp32 columns of this thread's TMEM lane, and 8 columns stored.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&r)[8])
{
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr), "r"(r[0]),
                 "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
                 : "memory");
}

// ---------------------------------------------------------------- delta ----

// D[row] = sum_c dO[row][c] O[row][c]; D/8 threads per row, 8 bf16 each.
template <int D>
__global__ void delta_kernel(const __nv_bfloat16* __restrict__ out, const __nv_bfloat16* __restrict__ dout,
                             float* __restrict__ delta, long long rows)
{
    constexpr int TPR = D / 8;
    const long long gid = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
    const long long row = gid / TPR;
    const int part = static_cast<int>(gid % TPR);
    float acc = 0.f;
    if (row < rows) {
        const uint4 o = *reinterpret_cast<const uint4*>(out + row * D + 8 * part);
        const uint4 g = *reinterpret_cast<const uint4*>(dout + row * D + 8 * part);
        const uint32_t ow[4] = {o.x, o.y, o.z, o.w}, gw[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            acc = fmaf(bf16_lo(ow[i]), bf16_lo(gw[i]), acc);
            acc = fmaf(bf16_hi(ow[i]), bf16_hi(gw[i]), acc);
        }
    }
#pragma unroll
    for (int off = TPR / 2; off >= 1; off >>= 1) acc += __shfl_xor_sync(kFull, acc, off);
    if (row < rows && part == 0) delta[row] = acc;
}

// ------------------------------------------------------------------ dQ ----
// Items of 128 query rows (G heads x QT positions), key tiles of NK. TMEM: S in two
// buffers (dS is written back over S as bf16 pairs, the A operand of dQ += dS K), dP in
// two buffers, or in one for 128-key tiles, and one or two dQ accumulators alternating
// between items. With one dP buffer the elementwise warpgroups release it as soon as
// they hold the tile's dP in registers (dp_free), and the MMA thread issues the next
// tile's dP then; the next tile's S is issued earlier still.
// Columns of S and dP the elementwise threads load before each wait (32 or 64).
#ifndef PBB_BWD_Q_QC
#define PBB_BWD_Q_QC 64
#endif

// With two elementwise warpgroups: both share every tile, warpgroup w taking columns
// [w N/2, (w+1) N/2) of its N score columns (1), or they take alternate tiles (0). Sharing keeps
// the tensor pipe busy: with alternate tiles, tile g+2's scores can only be issued after tile
// g's gradient products, which wait for tile g's exponentials, so both warpgroups went idle
// together while the pipe drained; with shared tiles, tile g+1's scores are ready when the
// warpgroups finish tile g.
#ifndef PBB_BWD_SPLIT_COLS
#define PBB_BWD_SPLIT_COLS 1
#endif

// TMEM column of the bf16-pair (P, dS or their transposes) operand for k-step kk (16 rows of
// the reduction) in a score buffer of N columns. Each warpgroup writes its pairs over the
// first columns it read itself: with split columns, warpgroup w's N/4 pair columns start at
// column w N/2; otherwise pairs of k-step kk sit at column 8 kk.
template <int N, bool SPLIT>
__host__ __device__ constexpr uint32_t pair_col(int kk)
{
    return SPLIT ? static_cast<uint32_t>((kk / (N / 32)) * (N / 2) + 8 * (kk % (N / 32)))
                 : static_cast<uint32_t>(8 * kk);
}

// Tiles with no masked entry take a packed path (1) or the masked one (0): PBB_BWD_Q_INNER for
// the dQ pass (every shape), PBB_BWD_KV_INNER for the dK/dV pass (one-CTA shapes; the two-CTA
// shape keeps the masked path, measured faster there).
#ifndef PBB_BWD_Q_INNER
#define PBB_BWD_Q_INNER 1
#endif
#ifndef PBB_BWD_KV_INNER
#define PBB_BWD_KV_INNER 1
#endif

// Shapes: NK keys per tile (64 or 32), WGS elementwise warpgroups (2 taking alternate
// tiles, or 1), CTAS CTAs per SM sharing its 512 TMEM columns (1, or 2 with 256 each).
template <int D, int G, int NK_, int WGS_, int CTAS_>
struct BqCfg {
    static constexpr int NK = NK_, WGS = WGS_, CTAS = CTAS_;
    static constexpr int M = 128, QT = M / G, BOXES = D / 64;
    static constexpr int THREADS = 128 * WGS + 64, PRODUCER = 4 * WGS, MMA = 4 * WGS + 1;
    static constexpr int TMEM_COLS = CTAS == 1 ? 512 : 256;
    static constexpr int QBOX = M * 128, KBOX = NK * 128;
    static constexpr int Q_OFF = 0, DO_OFF = BOXES * QBOX;
    // K and V in rings of their own: V is read by the dP product alone and its stage is free
    // again long before K's, which the dQ product reads too; K takes the odd stage (3 K + 2 V
    // at d = 128 in the long shape, where 2 + 2 left the MMA thread waiting for K)
    static constexpr int KV_OFF = 2 * BOXES * QBOX;
    static constexpr int K_STAGE = BOXES * KBOX;  // = V's
    static constexpr int ROOM = (227 * 1024 / CTAS - 2048 - KV_OFF) / K_STAGE;
    static constexpr int UNITS = ROOM < 8 ? ROOM : 8;
    static constexpr int KST = (UNITS + 1) / 2, VST = UNITS / 2;
    static constexpr int V_OFF = KV_OFF + KST * K_STAGE;
    static constexpr int SMEM = V_OFF + VST * K_STAGE + 1024;
    static constexpr int DPBUF = NK == 128 ? 1 : 2;            // dP buffers
    static constexpr int T_S = 0, T_DP = 2 * NK, T_DQ = T_DP + DPBUF * NK;
    static constexpr int OBUF = T_DQ + 2 * D <= TMEM_COLS ? 2 : 1;
    static constexpr bool INNER = PBB_BWD_Q_INNER;
    static constexpr bool SPLIT = WGS == 2 && PBB_BWD_SPLIT_COLS;
    static_assert(DPBUF == 2 || (PBB_BWD_Q_QC >= NK / (SPLIT ? 2 : 1)),
                  "one dP buffer: each warpgroup loads its columns of a tile before one wait");
    static_assert(VST >= 2, "shared memory budget");
    static_assert(T_DQ + OBUF * D <= TMEM_COLS, "TMEM budget");
    static_assert(CTAS * (SMEM + 1024) <= 227 * 1024, "shared memory budget");
    static_assert(QT % 8 == 0, "a head's rows must start on a swizzle atom");
    static_assert(NK % 32 == 0 && D % (32 * WGS) == 0, "32-column chunks");
};

struct QItem {
    int pair, t0, tl, lo, a_max, ntiles;
};

template <int QT, int NK>
__device__ __forceinline__ QItem make_qitem(int idx, int n, int B)
{
    const int nq = (n + QT - 1) / QT;
    QItem it;
    it.pair = idx / nq;
    it.t0 = (idx - it.pair * nq) * QT;
    it.tl = min(it.t0 + QT, n) - 1;
    const int h = B >> 1;
    it.lo = support_start(it.t0, h);
    it.a_max = support_start(it.tl, h);
    it.ntiles = (it.tl - it.lo + NK) / NK;
    return it;
}

template <int D, int G, int NK_, int WGS_, int CTAS_>
__global__ void __launch_bounds__(BqCfg<D, G, NK_, WGS_, CTAS_>::THREADS, CTAS_)
bwd_q_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                const __grid_constant__ CUtensorMap vmap, const __grid_constant__ CUtensorMap dmap,
                const BackwardArgs a)
{
    using C = BqCfg<D, G, NK_, WGS_, CTAS_>;
    constexpr int KST = C::KST, VST = C::VST, NK = C::NK, WGS = C::WGS, OBUF = C::OBUF;
    extern __shared__ unsigned char dsmem_raw[];
    __shared__ __align__(8) uint64_t q_full, q_empty, done_bar;
    __shared__ __align__(8) uint64_t k_full[KST], k_empty[KST], v_full[VST], v_empty[VST];
    __shared__ __align__(8) uint64_t s_full[2], ds_full[2], item_done[2], o_free[2], dp_free;
    __shared__ uint32_t tmem_base_s;
    __shared__ volatile int abort_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_items = a.batch * a.Hkv * ((a.n + C::QT - 1) / C::QT);
    if (tid == 0) {
        mbar_init(&q_full, 1);
        mbar_init(&q_empty, 1);
        mbar_init(&done_bar, 1);
#pragma unroll
        for (int s = 0; s < KST; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
        }
#pragma unroll
        for (int s = 0; s < VST; ++s) {
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], 1);
        }
#pragma unroll
        for (int b = 0; b < 2; ++b) {
            mbar_init(&s_full[b], 1);
            mbar_init(&ds_full[b], C::SPLIT ? 256 : 128);  // the warpgroups that handle buffer b
            mbar_init(&item_done[b], 1);
            mbar_init(&o_free[b], 128 * WGS);   // every warpgroup reads its share of the dQ row
        }
        mbar_init(&dp_free, C::SPLIT ? 256 : 128);  // one dP buffer: the warpgroups of a tile hold it
        fence_mbar_init();
        abort_s = 0;
    }
    if (warp == 0) tmem_alloc<C::TMEM_COLS>(&tmem_base_s);
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = tmem_base_s;
    const unsigned long long limit = a.timeout_ns;

    if (warp == C::PRODUCER) {
        if (lane == 0) {
            uint32_t gt = 0, ic = 0, q_issued = 0, k_issued = 0, v_issued = 0;
            bool ok = true;
            for (int rd = 0, idx = item_turned(0); ok && idx < n_items; ++rd, idx = item_turned(rd), ++ic) {
                const QItem it = make_qitem<C::QT, NK>(idx, a.n, a.B);
                const int b = it.pair / a.Hkv, kvh = it.pair - b * a.Hkv;
                if (ic > 0 && !mbar_wait(&q_empty, (ic - 1) & 1u, limit)) {
                    ok = false;
                    break;
                }
                mbar_expect_tx(&q_full, static_cast<uint32_t>(2 * C::BOXES * C::QBOX));
#pragma unroll
                for (int gi = 0; gi < G; ++gi) {
                    const int qrow = (b * a.Hq + kvh * G + gi) * a.n + it.t0;
#pragma unroll
                    for (int bx = 0; bx < C::BOXES; ++bx) {
                        tma_load_2d(dsmem + C::Q_OFF + bx * C::QBOX + gi * C::QT * 128, &qmap, bx * 64, qrow, &q_full);
                        tma_load_2d(dsmem + C::DO_OFF + bx * C::QBOX + gi * C::QT * 128, &dmap, bx * 64, qrow, &q_full);
                    }
                }
                ++q_issued;
                const int krow0 = it.pair * a.n + it.lo;
                for (int j = 0; j < it.ntiles; ++j, ++gt) {
                    const int sk = gt % KST, sv = gt % VST;
                    if (gt >= KST && !mbar_wait(&k_empty[sk], ((gt / KST) - 1) & 1u, limit)) {
                        ok = false;
                        break;
                    }
                    if (abort_s) {
                        ok = false;
                        break;
                    }
                    unsigned char* kst = dsmem + C::KV_OFF + sk * C::K_STAGE;
                    mbar_expect_tx(&k_full[sk], static_cast<uint32_t>(C::K_STAGE));
#pragma unroll
                    for (int bx = 0; bx < C::BOXES; ++bx)
                        tma_load_2d(kst + bx * C::KBOX, &kmap, bx * 64, krow0 + j * NK, &k_full[sk]);
                    ++k_issued;
                    if (gt >= VST && !mbar_wait(&v_empty[sv], ((gt / VST) - 1) & 1u, limit)) {
                        ok = false;
                        break;
                    }
                    unsigned char* vst = dsmem + C::V_OFF + sv * C::K_STAGE;
                    mbar_expect_tx(&v_full[sv], static_cast<uint32_t>(C::K_STAGE));
#pragma unroll
                    for (int bx = 0; bx < C::BOXES; ++bx)
                        tma_load_2d(vst + bx * C::KBOX, &vmap, bx * 64, krow0 + j * NK, &v_full[sv]);
                    ++v_issued;
                }
            }
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
            }
            // drain: the last copies into Q/dO and into each stage land before shared memory goes away
            if (q_issued > 0) mbar_wait(&q_full, (q_issued - 1) & 1u, kGuardNs);
            for (uint32_t s = 0; s < KST && s < k_issued; ++s) {
                const uint32_t j = s + KST * ((k_issued - 1 - s) / KST);
                mbar_wait(&k_full[s], (j / KST) & 1u, kGuardNs);
            }
            for (uint32_t s = 0; s < VST && s < v_issued; ++s) {
                const uint32_t j = s + VST * ((v_issued - 1 - s) / VST);
                mbar_wait(&v_full[s], (j / VST) & 1u, kGuardNs);
            }
        }
    } else if (warp == C::MMA) {
        if (lane == 0) {
            constexpr uint32_t idesc_s = umma_idesc_bf16(C::M, NK, 0);
            constexpr uint32_t idesc_q = umma_idesc_bf16(C::M, D, 1);
            const uint32_t q_base = smem_addr(dsmem + C::Q_OFF), do_base = smem_addr(dsmem + C::DO_OFF);
            const uint32_t k_base = smem_addr(dsmem + C::KV_OFF), v_base = smem_addr(dsmem + C::V_OFF);
            uint32_t gt = 0, ic = 0;
            bool ok = true, issued_any = false;
            // S = Q K^T into buffer g % 2, and dP = dO V^T into buffer g % DPBUF; the commit of
            // s_full covers both, and dP's own commit frees V's stage
            auto issue_s = [&](uint32_t g) {
                const uint32_t kb = k_base + (g % KST) * C::K_STAGE;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (kk >> 2) * C::QBOX + (kk & 3) * 32;
                    const uint32_t koff = (kk >> 2) * C::KBOX + (kk & 3) * 32;
                    umma_bf16(tmem + C::T_S + (g & 1u) * NK, umma_desc_sw128(q_base + off, 16, 1024),
                              umma_desc_sw128(kb + koff, 16, 1024), idesc_s, kk > 0 ? 1u : 0u);
                }
            };
            auto issue_dp = [&](uint32_t g) {
                const uint32_t vb = v_base + (g % VST) * C::K_STAGE;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t off = (kk >> 2) * C::QBOX + (kk & 3) * 32;
                    const uint32_t koff = (kk >> 2) * C::KBOX + (kk & 3) * 32;
                    umma_bf16(tmem + C::T_DP + (g % C::DPBUF) * NK, umma_desc_sw128(do_base + off, 16, 1024),
                              umma_desc_sw128(vb + koff, 16, 1024), idesc_s, kk > 0 ? 1u : 0u);
                }
                umma_commit(&v_empty[g % VST]);
                umma_commit(&s_full[g & 1u]);
            };
            auto k_ready = [&](uint32_t g) { return mbar_wait(&k_full[g % KST], (g / KST) & 1u, limit); };
            auto v_ready = [&](uint32_t g) {
                if (!mbar_wait(&v_full[g % VST], (g / VST) & 1u, limit)) return false;
                tmem_fence_after();
                return true;
            };
            // with one dP buffer, tile g's dP goes in once the warpgroups hold tile g-1's
            auto dp_ready = [&](uint32_t g) {
                if (C::DPBUF == 2 || g == 0) return true;
                if (!mbar_wait(&dp_free, (g - 1) & 1u, limit)) return false;
                tmem_fence_after();
                return true;
            };
            for (int rd = 0, idx = item_turned(0); ok && idx < n_items; ++rd, idx = item_turned(rd), ++ic) {
                const QItem it = make_qitem<C::QT, NK>(idx, a.n, a.B);
                const uint32_t ob = ic % OBUF;
                if (!mbar_wait(&q_full, ic & 1u, limit) || !k_ready(gt)) {
                    ok = false;
                    break;
                }
                tmem_fence_after();
                issue_s(gt);
                issued_any = true;
                if (!dp_ready(gt) || !v_ready(gt)) {
                    ok = false;
                    break;
                }
                issue_dp(gt);
                if (it.ntiles == 1) umma_commit(&q_empty);
                for (int j = 0; j < it.ntiles; ++j) {
                    const uint32_t g = gt + j;
                    if (j + 1 < it.ntiles) {
                        if (!k_ready(g + 1)) {
                            ok = false;
                            break;
                        }
                        tmem_fence_after();
                        issue_s(g + 1);
                        if (!dp_ready(g + 1) || !v_ready(g + 1)) {
                            ok = false;
                            break;
                        }
                        issue_dp(g + 1);
                        if (j + 2 == it.ntiles) umma_commit(&q_empty);  // the item's last read of Q and dO
                    }
                    if (!mbar_wait(&ds_full[g & 1u], (g >> 1) & 1u, limit) ||
                        (j == 0 && ic >= OBUF && !mbar_wait(&o_free[ob], ((ic / OBUF) - 1) & 1u, limit))) {
                        ok = false;
                        break;
                    }
                    tmem_fence_after();
                    // dQ (+)= dS K: dS from TMEM (over S buffer g % 2), K MN-major
                    const uint32_t kb = k_base + (g % KST) * C::K_STAGE;
#pragma unroll
                    for (int kk = 0; kk < NK / 16; ++kk)
                        umma_bf16_tmem_a(tmem + C::T_DQ + ob * D, tmem + C::T_S + (g & 1u) * NK + pair_col<NK, C::SPLIT>(kk),
                                         umma_desc_sw128(kb + kk * 2048, C::KBOX, 1024), idesc_q,
                                         (j > 0 || kk > 0) ? 1u : 0u);
                    umma_commit(&k_empty[g % KST]);
                }
                if (!ok) break;
                umma_commit(&item_done[ob]);
                gt += it.ntiles;
            }
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
            }
            if (issued_any) {  // every MMA complete before TMEM is released
                umma_commit(&done_bar);
                mbar_wait(&done_bar, 0u, kGuardNs);
            }
        }
    } else {
        // elementwise: with two warpgroups, warpgroup wg takes the tiles g with g % 2 == wg (S/dP
        // buffer wg); one warpgroup takes them all. Thread r owns query row r (TMEM lane r)
        const int wg = warp >> 2, r = tid & 127;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        const float sc2 = kLog2e * rsqrtf(static_cast<float>(D)), sc = rsqrtf(static_cast<float>(D));
        const int h = a.B >> 1;
        const int gi = r / C::QT, rp = r - gi * C::QT;
        uint32_t gt = 0, ic = 0;
        bool ok = true;
        for (int rd = 0, idx = item_turned(0); ok && idx < n_items; ++rd, idx = item_turned(rd), ++ic) {
            const QItem it = make_qitem<C::QT, NK>(idx, a.n, a.B);
            const uint32_t ob = ic % OBUF;
            const int b = it.pair / a.Hkv, kvh = it.pair - b * a.Hkv;
            const int t = it.t0 + rp, as = support_start(t, h);
            const bool valid = t < a.n;
            const size_t row = static_cast<size_t>(b * a.Hq + kvh * G + gi) * a.n + (valid ? t : 0);
            const float l2 = valid ? a.lse[row] * kLog2e : 0.f, dr = valid ? a.delta[row] : 0.f;
            for (int j = 0; j < it.ntiles; ++j) {
                const uint32_t g = gt + j;
                if (WGS == 2 && !C::SPLIT && static_cast<int>(g & 1u) != wg) continue;
                if (!warp_wait(&s_full[g & 1u], (g >> 1) & 1u, limit) || __any_sync(kFull, abort_s != 0)) {
                    ok = false;
                    break;
                }
                tmem_fence_after();
                const int key0 = it.lo + j * NK;
                const bool edge = (key0 + NK - 1 > it.t0) || (key0 < it.a_max);
                // every key of the tile in every valid row's support: the packed path
                const bool inner = C::INNER && !edge && __all_sync(kFull, valid);
                // QC columns at a time (all their loads before one wait): their dS (QC/2
                // bf16-pair columns) goes over columns already read; with split columns this
                // warpgroup takes columns [wg NK/2, (wg+1) NK/2)
                constexpr int NW = C::SPLIT ? NK / 2 : NK;  // this warpgroup's columns of the tile
                constexpr int QC = PBB_BWD_Q_QC < NW ? PBB_BWD_Q_QC : NW;
                const int col0 = C::SPLIT ? wg * NW : 0;
#pragma unroll
                for (int c = 0; c < NW / QC; ++c) {
                    uint32_t v1[QC], v2[QC];
#pragma unroll
                    for (int h32 = 0; h32 < QC / 32; ++h32) {
                        uint32_t* a1 = v1 + 32 * h32;
                        uint32_t* a2 = v2 + 32 * h32;
                        tmem_ld32(lane_base + C::T_S + (g & 1u) * NK + col0 + QC * c + 32 * h32,
                                  *reinterpret_cast<uint32_t(*)[32]>(a1));
                        tmem_ld32(lane_base + C::T_DP + (g % C::DPBUF) * NK + col0 + QC * c + 32 * h32,
                                  *reinterpret_cast<uint32_t(*)[32]>(a2));
                    }
                    tmem_wait_ld();
                    if constexpr (C::DPBUF == 1) {  // this warpgroup's dP of the tile is in registers
                        tmem_fence_before();
                        mbar_arrive(&dp_free);
                    }
                    uint32_t pk[QC / 2];
                    if (inner) {
#pragma unroll
                        for (int x = 0; x < QC / 2; ++x) {
                            const float2 arg = __ffma2_rn(
                                make_float2(__uint_as_float(v1[2 * x]), __uint_as_float(v1[2 * x + 1])),
                                make_float2(sc2, sc2), make_float2(-l2, -l2));
                            const float2 e = __fmul2_rn(
                                make_float2(fast_exp2(arg.x), fast_exp2(arg.y)),
                                __fadd2_rn(make_float2(__uint_as_float(v2[2 * x]), __uint_as_float(v2[2 * x + 1])),
                                           make_float2(-dr, -dr)));
                            pk[x] = pack_bf16x2(e.x, e.y);
                        }
                    } else {
                        // the row's visible columns of this chunk, [lo_c, hi_c]: worked out once, so
                        // each entry compares its constant column index (testing each entry's key
                        // against the support measured about 3,500 cycles per 32-column tile)
                        const int k0 = key0 + col0 + QC * c;
                        const int lo_c = edge ? as - k0 : 0, hi_c = valid ? (edge ? t - k0 : QC) : -1;
#pragma unroll
                        for (int x = 0; x < QC / 2; ++x) {
                            float e[2];
#pragma unroll
                            for (int y = 0; y < 2; ++y) {
                                const bool vis = 2 * x + y >= lo_c && 2 * x + y <= hi_c;
                                const float p = vis ? fast_exp2(fmaf(__uint_as_float(v1[2 * x + y]), sc2, -l2)) : 0.f;
                                e[y] = p * (__uint_as_float(v2[2 * x + y]) - dr);
                            }
                            pk[x] = pack_bf16x2(e[0], e[1]);
                        }
                    }
#pragma unroll
                    for (int h16 = 0; h16 < QC / 32; ++h16)
                        tmem_st16(lane_base + C::T_S + (g & 1u) * NK + col0 + (QC / 2) * c + 16 * h16,
                                  *reinterpret_cast<const uint32_t(*)[16]>(pk + 16 * h16));
                }
                tmem_wait_st();
                tmem_fence_before();
                mbar_arrive(&ds_full[g & 1u]);
            }
            if (!ok) break;
            if (!warp_wait(&item_done[ob], (ic / OBUF) & 1u, limit)) {
                ok = false;
                break;
            }
            tmem_fence_after();
#pragma unroll
            for (int c = 0; c < D / (32 * WGS); ++c) {  // this warpgroup's share of the row
                const int col = wg * (D / WGS) + 32 * c;
                uint32_t v[32];
                tmem_ld32(lane_base + C::T_DQ + ob * D + col, v);
                tmem_wait_ld();
                if (valid) store_row32(a.dq + row * D + col, v, sc, (reinterpret_cast<uintptr_t>(a.dq) & 31u) == 0);
            }
            tmem_fence_before();
            mbar_arrive(&o_free[ob]);
            gt += it.ntiles;
        }
        if (!ok) {
            abort_s = 1;
            atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
        }
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    if (warp == 0) tmem_dealloc<C::TMEM_COLS>(tmem);
}

// ------------------------------------------------------------- dK, dV ----
// Items of 128 keys, query tiles of NQ rows (G heads x QT positions). Per query tile the
// producer warp also stages, for each of its NQ columns, the base-2 log-partition, D, the
// position and its support start. TMEM:
//  - NQ = 64 or 32: S^T and dP^T, two buffers each (P^T and dS^T are written back over
//    them as bf16 pairs, the A operands of dV += P^T dO and dK += dS^T Q), then dV and dK;
//  - NQ = 128 (two elementwise warpgroups on split columns): S^T and dP^T one buffer each,
//    then dV and dK (4 x 128 columns at d = 128). Every score product is an N = 128 MMA:
//    with both operands in shared memory, an N = 64 product runs at 2/3 of the tensor rate.
//    The score products end with one more K step, a column of ones against the tile's
//    -lse2 / sc2 (S^T) or -D (dP^T) split into three bf16 terms, so the scores arrive with
//    the per-column terms applied and the elementwise threads read no per-column data on
//    unmasked tiles. P^T and dS^T both go back over the S^T buffer, and the next tile's S^T
//    follows the gradient products that read them; its dP^T follows (dp_full), and the
//    warpgroups compute a half's exponentials before they wait for it. They release the
//    dP^T buffer once they hold the tile's dP^T (dp_free).
// Shapes as for the dQ pass: NQ query rows per tile, WGS elementwise warpgroups, CTAS CTAs
// per SM.
// Columns of S^T and dP^T the elementwise threads load before each wait (16 or 32): fewer waits
// per tile against more registers.
#ifndef PBB_BWD_KV_KC
#define PBB_BWD_KV_KC 16
#endif
template <int D, int G, int NQ_, int WGS_, int CTAS_>
struct BkvCfg {
    static constexpr int NQ = NQ_, WGS = WGS_, CTAS = CTAS_;
    static constexpr int M = 128, QT = NQ / G, BOXES = D / 64;
    static constexpr int THREADS = 128 * WGS + 64, PRODUCER = 4 * WGS, MMA = 4 * WGS + 1;
    static constexpr int TMEM_COLS = CTAS == 1 ? 512 : 256;
    static constexpr int KBOX = M * 128, QBOX = NQ * 128;
    static constexpr int K_OFF = 0, V_OFF = BOXES * KBOX;
    // one-buffer shape: the score products take -lse2 / sc2 and -D as one more K step against
    // a column of ones (AUG): a 128 x 16 ones tile after K and V, and per stage the 16-wide
    // extra K step of S^T and of dP^T (32-byte swizzle, 32 bytes a row)
    static constexpr bool AUG = NQ == 128;
    static constexpr int ONES_OFF = 2 * BOXES * KBOX, XROW = 32;
    static constexpr int RING_OFF = ONES_OFF + (AUG ? M * XROW : 0);
    // per column (lse2, D, t, a(t)) as a float4 (one load per entry on the masked path); with
    // the packed path, (-lse2, -D) again as a float2 array (one load per column pair)
    static constexpr bool INNER = PBB_BWD_KV_INNER && CTAS == 1;
    static constexpr bool SPLIT = WGS == 2 && PBB_BWD_SPLIT_COLS;
    static constexpr int META = NQ * (INNER ? 24 : 16);
    static constexpr int META_OFF = 2 * BOXES * QBOX;
    static constexpr int XS_OFF = (META_OFF + META + 255) / 256 * 256, XD_OFF = XS_OFF + NQ * XROW;
    static constexpr int STAGE = ((AUG ? XD_OFF + NQ * XROW : META_OFF + META) + 1023) / 1024 * 1024;  // Q, dO, metadata (+ extra K steps)
    static constexpr int STAGE_ROOM = (227 * 1024 / CTAS - 2048 - RING_OFF) / STAGE;
    static constexpr int STAGE_MAX = CTAS == 1 ? 3 : 4;
    static constexpr int STAGES = STAGE_ROOM < STAGE_MAX ? STAGE_ROOM : STAGE_MAX;
    static constexpr int SMEM = RING_OFF + STAGES * STAGE + 1024;
    static constexpr int SBUF = NQ == 128 ? 1 : 2;  // S^T and dP^T buffers
    static constexpr int T_ST = 0, T_DPT = SBUF * NQ, T_DV = 2 * SBUF * NQ, T_DK = T_DV + D;
    static_assert(SBUF == 2 || (SPLIT && CTAS == 1 && NQ == 128 && AUG), "one score buffer: both warpgroups share every tile");
    static_assert(STAGES >= 2, "shared memory budget");
    static_assert(T_DK + D <= TMEM_COLS, "TMEM budget");
    static_assert(CTAS * (SMEM + 1024) <= 227 * 1024, "shared memory budget");
    static_assert(QT % 8 == 0, "a head's rows must start on a swizzle atom");
    static_assert(NQ % 32 == 0, "the producer warp stages NQ / 32 columns per lane");
};

// TMEM column of the P^T pairs for k-step kk (16 query rows) in the one-buffer dK/dV shape
// (128-row tiles, split columns): warpgroup kk / 4 holds query columns [64 (kk / 4), +64),
// and each 32-column half of them takes its 16 P^T pair columns, then its 16 dS^T pair
// columns, over its own S^T columns. dS^T's pairs for kk sit 16 columns further on.
__host__ __device__ constexpr uint32_t pds_col(int kk)
{
    return static_cast<uint32_t>(64 * (kk / 4) + 32 * ((kk % 4) / 2) + 8 * (kk % 2));
}

// The first 16-byte half of a 16-element bf16 K-step row holding x as three bf16 terms
// (hi, mid, lo: x to about 24 bits, summed exactly by the fp32 accumulation), then zeros.
__device__ __forceinline__ uint4 bf16_split3_row(float x)
{
    const float hi = __bfloat162float(__float2bfloat16_rn(x));
    const float mid = __bfloat162float(__float2bfloat16_rn(x - hi));
    const float lo = __bfloat162float(__float2bfloat16_rn(x - hi - mid));
    return make_uint4(pack_bf16x2(hi, mid), pack_bf16x2(lo, 0.f), 0u, 0u);
}

struct KItem {
    int pair, s0, tq0, nqt;
};

template <int QT>
__device__ __forceinline__ KItem make_kitem(int idx, int n, int B)
{
    const int nk = (n + 127) / 128;
    KItem it;
    it.pair = idx / nk;
    it.s0 = (idx - it.pair * nk) * 128;
    const int s_last = min(it.s0 + 128, n) - 1;
    const int h = B >> 1;
    const int t_end = min(n, h * (s_last / h + 2));  // queries past t_end - 1 never see these keys
    it.tq0 = (it.s0 / QT) * QT;
    it.nqt = (t_end - it.tq0 + QT - 1) / QT;
    return it;
}

template <int D, int G, int NQ_, int WGS_, int CTAS_>
__global__ void __launch_bounds__(BkvCfg<D, G, NQ_, WGS_, CTAS_>::THREADS, CTAS_)
bwd_kv_tc_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                 const __grid_constant__ CUtensorMap vmap, const __grid_constant__ CUtensorMap dmap,
                 const BackwardArgs a)
{
    using C = BkvCfg<D, G, NQ_, WGS_, CTAS_>;
    constexpr int STAGES = C::STAGES, NQ = C::NQ, WGS = C::WGS;
    constexpr int MV = NQ / 32;  // columns of metadata each producer lane stages per tile
    extern __shared__ unsigned char dsmem_raw[];
    __shared__ __align__(8) uint64_t kv_full, kv_empty, done_bar, item_done, o_free;
    __shared__ __align__(8) uint64_t qd_full[STAGES], qd_empty[STAGES];
    __shared__ __align__(8) uint64_t s_full[2], p_full[2], dp_free, dp_full;
    __shared__ uint32_t tmem_base_s;
    __shared__ volatile int abort_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int n_items = a.batch * a.Hkv * ((a.n + 127) / 128);
    if (tid == 0) {
        mbar_init(&kv_full, 1);
        mbar_init(&kv_empty, 1);
        mbar_init(&done_bar, 1);
        mbar_init(&item_done, 1);
        mbar_init(&o_free, 128 * WGS);  // with two warpgroups, 0 reads dV and 1 dK
#pragma unroll
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&qd_full[s], 1);
            mbar_init(&qd_empty[s], 1);
        }
#pragma unroll
        for (int b = 0; b < 2; ++b) {
            mbar_init(&s_full[b], 1);
            mbar_init(&p_full[b], C::SPLIT ? 256 : 128);  // the warpgroups that handle buffer b
        }
        mbar_init(&dp_free, C::SPLIT ? 256 : 128);  // one dP^T buffer: the warpgroups of a tile hold it
        mbar_init(&dp_full, 1);                     // one dP^T buffer: its product is complete
        fence_mbar_init();
        abort_s = 0;
    }
    if constexpr (C::AUG) {  // the ones operand of the extra K step (bf16 1.0 everywhere, so unswizzled)
        for (int i = tid; i < C::M * C::XROW / 16; i += C::THREADS)
            reinterpret_cast<uint4*>(dsmem + C::ONES_OFF)[i] = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
        fence_proxy_async();
    }
    if (warp == 0) tmem_alloc<C::TMEM_COLS>(&tmem_base_s);
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    const uint32_t tmem = tmem_base_s;
    const unsigned long long limit = a.timeout_ns;
    const int h = a.B >> 1;

    if (warp == C::PRODUCER) {
        // the whole warp: lane 0 issues the copies, every lane stages two columns' metadata
        uint32_t gt = 0, ic = 0, kv_issued = 0;
        bool ok = true;
        for (int rd = 0, idx = item_turned(0); ok && idx < n_items; ++rd, idx = item_turned(rd), ++ic) {
            const KItem it = make_kitem<C::QT>(idx, a.n, a.B);
            const int b = it.pair / a.Hkv, kvh = it.pair - b * a.Hkv;
            if (ic > 0 && !warp_wait(&kv_empty, (ic - 1) & 1u, limit)) {
                ok = false;
                break;
            }
            if (lane == 0) {
                mbar_expect_tx(&kv_full, static_cast<uint32_t>(2 * C::BOXES * C::KBOX));
#pragma unroll
                for (int bx = 0; bx < C::BOXES; ++bx) {
                    tma_load_2d(dsmem + C::K_OFF + bx * C::KBOX, &kmap, bx * 64, it.pair * a.n + it.s0, &kv_full);
                    tma_load_2d(dsmem + C::V_OFF + bx * C::KBOX, &vmap, bx * 64, it.pair * a.n + it.s0, &kv_full);
                }
            }
            ++kv_issued;
            for (int i = 0; i < it.nqt; ++i, ++gt) {
                const int s = gt % STAGES;
                const int t0 = it.tq0 + i * C::QT;
                // this tile's per-column data: the loads are issued before the wait for a free
                // stage, so their latency overlaps it
                float4 mv[MV];
#pragma unroll
                for (int e = 0; e < MV; ++e) {
                    const int c = lane + 32 * e;
                    const int gi = c / C::QT, t = t0 + (c - gi * C::QT);
                    const bool valid = t < a.n;
                    const size_t row = static_cast<size_t>(b * a.Hq + kvh * G + gi) * a.n + (valid ? t : 0);
                    mv[e] = make_float4(valid ? __ldg(a.lse + row) : 0.f, valid ? __ldg(a.delta + row) : 0.f,
                                        __int_as_float(valid ? t : -1), __int_as_float(support_start(t, h)));
                }
                if (gt >= STAGES && !warp_wait(&qd_empty[s], ((gt / STAGES) - 1) & 1u, limit)) {
                    ok = false;
                    break;
                }
                if (__any_sync(kFull, abort_s != 0)) {
                    ok = false;
                    break;
                }
                unsigned char* st = dsmem + C::RING_OFF + s * C::STAGE;
                float4* meta = reinterpret_cast<float4*>(st + C::META_OFF);
#pragma unroll
                for (int e = 0; e < MV; ++e) {
                    const int c = lane + 32 * e;
                    mv[e].x *= kLog2e;
                    meta[c] = mv[e];
                    if constexpr (C::INNER && !C::AUG)
                        reinterpret_cast<float2*>(meta + NQ)[c] = make_float2(-mv[e].x, -mv[e].y);
                    if constexpr (C::AUG) {
                        // row c of the extra K steps: -lse2 / sc2 for S^T (so that sc2 S^T is the
                        // exponent) and -D for dP^T, as bf16 hi/mid/lo; the second half zero
                        const float sc2 = kLog2e * rsqrtf(static_cast<float>(D));
                        *reinterpret_cast<uint4*>(st + C::XS_OFF + swz32(c, 0)) = bf16_split3_row(-mv[e].x / sc2);
                        *reinterpret_cast<uint4*>(st + C::XS_OFF + swz32(c, 1)) = make_uint4(0u, 0u, 0u, 0u);
                        *reinterpret_cast<uint4*>(st + C::XD_OFF + swz32(c, 0)) = bf16_split3_row(-mv[e].y);
                        *reinterpret_cast<uint4*>(st + C::XD_OFF + swz32(c, 1)) = make_uint4(0u, 0u, 0u, 0u);
                    }
                }
                if constexpr (C::AUG) fence_proxy_async();  // the MMAs read the extra K steps
                __threadfence_block();
                __syncwarp();
                if (lane == 0) {
                    mbar_expect_tx(&qd_full[s], static_cast<uint32_t>(2 * C::BOXES * C::QBOX));
#pragma unroll
                    for (int gi = 0; gi < G; ++gi) {
                        const int qrow = (b * a.Hq + kvh * G + gi) * a.n + t0;
#pragma unroll
                        for (int bx = 0; bx < C::BOXES; ++bx) {
                            tma_load_2d(st + bx * C::QBOX + gi * C::QT * 128, &qmap, bx * 64, qrow, &qd_full[s]);
                            tma_load_2d(st + (C::BOXES + bx) * C::QBOX + gi * C::QT * 128, &dmap, bx * 64, qrow,
                                        &qd_full[s]);
                        }
                    }
                }
            }
        }
        if (!ok && lane == 0) {
            abort_s = 1;
            atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
        }
        if (lane == 0) {  // drain the copies still in flight
            if (kv_issued > 0) mbar_wait(&kv_full, (kv_issued - 1) & 1u, kGuardNs);
            for (uint32_t s = 0; s < STAGES && s < gt; ++s) {
                const uint32_t j = s + STAGES * ((gt - 1 - s) / STAGES);
                mbar_wait(&qd_full[s], (j / STAGES) & 1u, kGuardNs);
            }
        }
    } else if (warp == C::MMA) {
        if (lane == 0) {
            constexpr uint32_t idesc_s = umma_idesc_bf16(C::M, NQ, 0);
            constexpr uint32_t idesc_o = umma_idesc_bf16(C::M, D, 1);
            const uint32_t k_base = smem_addr(dsmem + C::K_OFF), v_base = smem_addr(dsmem + C::V_OFF);
            const uint32_t ring = smem_addr(dsmem + C::RING_OFF);
            uint32_t gt = 0, ic = 0;
            bool ok = true, issued_any = false;
            auto issue_sdp = [&](uint32_t g) {  // S^T = K Q^T and dP^T = V dO^T into buffer g % 2
                if (!mbar_wait(&qd_full[g % STAGES], (g / STAGES) & 1u, limit)) return false;
                tmem_fence_after();
                const uint32_t qb = ring + (g % STAGES) * C::STAGE, db = qb + C::BOXES * C::QBOX;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint32_t koff = (kk >> 2) * C::KBOX + (kk & 3) * 32;
                    const uint32_t qoff = (kk >> 2) * C::QBOX + (kk & 3) * 32;
                    umma_bf16(tmem + C::T_ST + (g & 1u) * NQ, umma_desc_sw128(k_base + koff, 16, 1024),
                              umma_desc_sw128(qb + qoff, 16, 1024), idesc_s, kk > 0 ? 1u : 0u);
                    umma_bf16(tmem + C::T_DPT + (g & 1u) * NQ, umma_desc_sw128(v_base + koff, 16, 1024),
                              umma_desc_sw128(db + qoff, 16, 1024), idesc_s, kk > 0 ? 1u : 0u);
                }
                umma_commit(&s_full[g & 1u]);
                return true;
            };
            auto qd_ready = [&](uint32_t g) {
                if (!mbar_wait(&qd_full[g % STAGES], (g / STAGES) & 1u, limit)) return false;
                tmem_fence_after();
                return true;
            };
            if constexpr (C::SBUF == 1) {
                // one score buffer per kind: tile g's S^T goes in after tile g-1's gradient
                // products (they read P^T and dS^T from the S^T buffer), then its dP^T (once the
                // warpgroups hold tile g-1's). S^T = K Q^T - (lse2 / sc2) 1^T and
                // dP^T = V dO^T - D 1^T: the last K step is the ones tile against the stage's row
                // of -lse2 / sc2 (or -D) terms
                const uint32_t ones = smem_addr(dsmem + C::ONES_OFF);
                auto issue_one = [&](uint32_t g, bool dpt) {
                    const uint32_t sbase = ring + (g % STAGES) * C::STAGE;
                    const uint32_t qb = sbase + (dpt ? C::BOXES * C::QBOX : 0);
                    const uint32_t ab = dpt ? v_base : k_base;
                    const uint32_t dst = tmem + (dpt ? C::T_DPT : C::T_ST);
#pragma unroll
                    for (int kk = 0; kk < D / 16; ++kk)
                        umma_bf16(dst, umma_desc_sw128(ab + (kk >> 2) * C::KBOX + (kk & 3) * 32, 16, 1024),
                                  umma_desc_sw128(qb + (kk >> 2) * C::QBOX + (kk & 3) * 32, 16, 1024), idesc_s,
                                  kk > 0 ? 1u : 0u);
                    umma_bf16(dst, umma_desc_sw32(ones), umma_desc_sw32(sbase + (dpt ? C::XD_OFF : C::XS_OFF)), idesc_s, 1u);
                };
                auto dp_ready = [&](uint32_t g) {
                    if (g == 0) return true;
                    if (!mbar_wait(&dp_free, (g - 1) & 1u, limit)) return false;
                    tmem_fence_after();
                    return true;
                };
                for (int rd = 0, idx = item_turned(0); ok && idx < n_items; ++rd, idx = item_turned(rd), ++ic) {
                    const KItem it = make_kitem<C::QT>(idx, a.n, a.B);
                    if (!mbar_wait(&kv_full, ic & 1u, limit) || !qd_ready(gt)) {
                        ok = false;
                        break;
                    }
                    tmem_fence_after();
                    issue_one(gt, false);
                    umma_commit(&s_full[0]);
                    issued_any = true;
                    if (!dp_ready(gt)) {
                        ok = false;
                        break;
                    }
                    issue_one(gt, true);
                    umma_commit(&dp_full);
                    if (it.nqt == 1) umma_commit(&kv_empty);  // the item's last read of K and V
                    for (int i = 0; i < it.nqt; ++i) {
                        const uint32_t g = gt + i;
                        const bool more = i + 1 < it.nqt;
                        // the next tile's dP^T goes ahead of this tile's gradient products if its
                        // Q/dO stage has landed; else after its S^T, so that waiting for the copy
                        // does not hold back the products whose completion frees the other stage
                        // (the warpgroups compute the exponentials of S^T before they need dP^T)
                        bool dp_early = false;
                        if (more) {
                            if (!dp_ready(g + 1)) {
                                ok = false;
                                break;
                            }
                            dp_early = mbar_test(&qd_full[(g + 1) % STAGES], ((g + 1) / STAGES) & 1u);
                            if (dp_early) {
                                tmem_fence_after();
                                issue_one(g + 1, true);
                                umma_commit(&dp_full);
                            }
                        }
                        if (!mbar_wait(&p_full[0], g & 1u, limit) ||
                            (i == 0 && ic >= 1 && !mbar_wait(&o_free, (ic - 1) & 1u, limit))) {
                            ok = false;
                            break;
                        }
                        tmem_fence_after();
                        // dV (+)= P^T dO and dK (+)= dS^T Q: P^T and dS^T in the S^T buffer, B MN-major
                        const uint32_t qb = ring + (g % STAGES) * C::STAGE, db = qb + C::BOXES * C::QBOX;
#pragma unroll
                        for (int kk = 0; kk < NQ / 16; ++kk) {
                            const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
                            const uint32_t pc = C::T_ST + pds_col(kk);
                            umma_bf16_tmem_a(tmem + C::T_DV, tmem + pc, umma_desc_sw128(db + kk * 2048, C::QBOX, 1024),
                                             idesc_o, acc);
                            umma_bf16_tmem_a(tmem + C::T_DK, tmem + pc + 16,
                                             umma_desc_sw128(qb + kk * 2048, C::QBOX, 1024), idesc_o, acc);
                        }
                        umma_commit(&qd_empty[g % STAGES]);
                        if (more) {
                            if (!dp_early && !qd_ready(g + 1)) {
                                ok = false;
                                break;
                            }
                            issue_one(g + 1, false);
                            umma_commit(&s_full[0]);
                            if (!dp_early) {
                                issue_one(g + 1, true);
                                umma_commit(&dp_full);
                            }
                            if (i + 2 == it.nqt) umma_commit(&kv_empty);
                        }
                    }
                    if (!ok) break;
                    umma_commit(&item_done);
                    gt += it.nqt;
                }
            }
            for (int rd = 0, idx = item_turned(0); C::SBUF == 2 && ok && idx < n_items; ++rd, idx = item_turned(rd), ++ic) {
                const KItem it = make_kitem<C::QT>(idx, a.n, a.B);
                if (!mbar_wait(&kv_full, ic & 1u, limit)) {
                    ok = false;
                    break;
                }
                tmem_fence_after();
                if (!issue_sdp(gt)) {
                    ok = false;
                    break;
                }
                issued_any = true;
                for (int i = 0; i < it.nqt; ++i) {
                    const uint32_t g = gt + i;
                    if (i + 1 < it.nqt && !issue_sdp(g + 1)) {
                        ok = false;
                        break;
                    }
                    if (!mbar_wait(&p_full[g & 1u], (g >> 1) & 1u, limit) ||
                        (i == 0 && ic >= 1 && !mbar_wait(&o_free, (ic - 1) & 1u, limit))) {
                        ok = false;
                        break;
                    }
                    tmem_fence_after();
                    // dV (+)= P^T dO and dK (+)= dS^T Q: A from TMEM, B (dO, Q) MN-major
                    const uint32_t qb = ring + (g % STAGES) * C::STAGE, db = qb + C::BOXES * C::QBOX;
#pragma unroll
                    for (int kk = 0; kk < NQ / 16; ++kk) {
                        const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
                        umma_bf16_tmem_a(tmem + C::T_DV, tmem + C::T_ST + (g & 1u) * NQ + pair_col<NQ, C::SPLIT>(kk),
                                         umma_desc_sw128(db + kk * 2048, C::QBOX, 1024), idesc_o, acc);
                        umma_bf16_tmem_a(tmem + C::T_DK, tmem + C::T_DPT + (g & 1u) * NQ + pair_col<NQ, C::SPLIT>(kk),
                                         umma_desc_sw128(qb + kk * 2048, C::QBOX, 1024), idesc_o, acc);
                    }
                    umma_commit(&qd_empty[g % STAGES]);
                }
                if (!ok) break;
                umma_commit(&kv_empty);
                umma_commit(&item_done);
                gt += it.nqt;
            }
            if (!ok) {
                abort_s = 1;
                atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
            }
            if (issued_any) {  // every MMA complete before TMEM is released
                umma_commit(&done_bar);
                mbar_wait(&done_bar, 0u, kGuardNs);
            }
        }
    } else {
        // elementwise: with two warpgroups, warpgroup wg takes the query tiles g with g % 2 == wg
        // (S^T/dP^T buffer wg); one warpgroup takes them all. Thread r owns key row r (TMEM lane r)
        const int wg = warp >> 2, r = tid & 127;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * (warp & 3)) << 16);
        const float sc2 = kLog2e * rsqrtf(static_cast<float>(D)), sc = rsqrtf(static_cast<float>(D));
        uint32_t gt = 0, ic = 0;
        bool ok = true;
        for (int rd = 0, idx = item_turned(0); ok && idx < n_items; ++rd, idx = item_turned(rd), ++ic) {
            const KItem it = make_kitem<C::QT>(idx, a.n, a.B);
            const int key = it.s0 + r;
            const bool kvalid = key < a.n;
            for (int i = 0; i < it.nqt; ++i) {
                const uint32_t g = gt + i;
                if (WGS == 2 && !C::SPLIT && static_cast<int>(g & 1u) != wg) continue;
                const uint32_t sb = g % C::SBUF;
                const float4* meta =
                    reinterpret_cast<const float4*>(dsmem + C::RING_OFF + (g % STAGES) * C::STAGE + C::META_OFF);
                const float2* meta_ld = reinterpret_cast<const float2*>(meta + NQ);
                // a tile whose every query sees every key of the warp's rows needs no mask: the
                // packed path (bit-identical arithmetic, half the instructions)
                const int tq0 = it.tq0 + i * C::QT, tql = tq0 + C::QT - 1;
                const bool inner =
                    C::INNER && __all_sync(kFull, kvalid && tql < a.n && key <= tq0 && key >= support_start(tql, h));
                if (!warp_wait(&s_full[sb], (g / C::SBUF) & 1u, limit) || __any_sync(kFull, abort_s != 0)) {
                    ok = false;
                    break;
                }
                tmem_fence_after();
                // KC columns at a time: their P^T and dS^T (KC/2 bf16-pair columns each) go over
                // columns already read; with split columns this warpgroup takes columns
                // [wg NQ/2, (wg+1) NQ/2)
                constexpr int NW = C::SPLIT ? NQ / 2 : NQ;  // this warpgroup's columns of the tile
                constexpr int KC = PBB_BWD_KV_KC < NW ? PBB_BWD_KV_KC : NW;
                const int col0 = C::SPLIT ? wg * NW : 0;
                if constexpr (C::SBUF == 1) {
                    // 32 columns at a time: S^T and its exponentials first, then (once its product
                    // is complete) dP^T; after the last half's dP^T loads the dP^T buffer is free.
                    // Each half takes its own P^T and dS^T pairs (16 columns each, pds_col) over
                    // its S^T columns. The scores already hold -lse2 / sc2 and -D (the extra K
                    // step), so the packed path reads no per-column data: P = 2^(sc2 S^T),
                    // dS = P dP^T
#pragma unroll
                    for (int hh = 0; hh < NW / 32; ++hh) {
                        uint32_t v1[32], v2[32];
                        tmem_ld32(lane_base + C::T_ST + col0 + 32 * hh, v1);
                        tmem_wait_ld();
                        float pr[32];
                        if (inner) {
#pragma unroll
                            for (int x = 0; x < 16; ++x) {
                                const float2 arg = __fmul2_rn(
                                    make_float2(__uint_as_float(v1[2 * x]), __uint_as_float(v1[2 * x + 1])), make_float2(sc2, sc2));
                                pr[2 * x] = fast_exp2(arg.x);
                                pr[2 * x + 1] = fast_exp2(arg.y);
                            }
                        } else {
#pragma unroll
                            for (int j = 0; j < 32; ++j) {
                                const float4 m = meta[col0 + 32 * hh + j];  // (lse2, D, t, a(t)); t = -1 past n
                                const int t = __float_as_int(m.z), at = __float_as_int(m.w);
                                const bool vis = kvalid && key <= t && key >= at;
                                pr[j] = vis ? fast_exp2(__uint_as_float(v1[j]) * sc2) : 0.f;
                            }
                        }
                        if (hh == 0 && !warp_wait(&dp_full, g & 1u, limit)) {
                            ok = false;
                            break;
                        }
                        if (hh == 0) tmem_fence_after();
                        tmem_ld32(lane_base + C::T_DPT + col0 + 32 * hh, v2);
                        tmem_wait_ld();
                        if (hh + 1 == NW / 32) {
                            tmem_fence_before();
                            mbar_arrive(&dp_free);
                        }
#pragma unroll
                        for (int c2 = 0; c2 < 2; ++c2) {
                            uint32_t pk[8], dk[8];
#pragma unroll
                            for (int x = 0; x < 8; ++x) {
                                const int j = 16 * c2 + 2 * x;
                                const float2 p = make_float2(pr[j], pr[j + 1]);
                                const float2 ds = __fmul2_rn(p, make_float2(__uint_as_float(v2[j]), __uint_as_float(v2[j + 1])));
                                pk[x] = pack_bf16x2(p.x, p.y);
                                dk[x] = pack_bf16x2(ds.x, ds.y);
                            }
                            tmem_st8(lane_base + C::T_ST + col0 + 32 * hh + 8 * c2, pk);
                            tmem_st8(lane_base + C::T_ST + col0 + 32 * hh + 16 + 8 * c2, dk);
                        }
                    }
                    if (!ok) break;
                }
#pragma unroll
                for (int c = 0; C::SBUF == 2 && c < NW / KC; ++c) {
                    uint32_t v1[KC], v2[KC];
                    if constexpr (KC == 32) {
                        tmem_ld32(lane_base + C::T_ST + (g & 1u) * NQ + col0 + KC * c, v1);
                        tmem_ld32(lane_base + C::T_DPT + (g & 1u) * NQ + col0 + KC * c, v2);
                    } else {
                        tmem_ld16(lane_base + C::T_ST + (g & 1u) * NQ + col0 + KC * c, v1);
                        tmem_ld16(lane_base + C::T_DPT + (g & 1u) * NQ + col0 + KC * c, v2);
                    }
                    tmem_wait_ld();
                    uint32_t pk[KC / 2], dk[KC / 2];
                    if (inner) {
#pragma unroll
                        for (int x = 0; x < KC / 2; ++x) {
                            // (-lse2, -D) of columns cc and cc + 1
                            const float4 m = *reinterpret_cast<const float4*>(meta_ld + col0 + KC * c + 2 * x);
                            const float2 arg = __ffma2_rn(
                                make_float2(__uint_as_float(v1[2 * x]), __uint_as_float(v1[2 * x + 1])),
                                make_float2(sc2, sc2), make_float2(m.x, m.z));
                            const float2 p = make_float2(fast_exp2(arg.x), fast_exp2(arg.y));
                            const float2 ds = __fmul2_rn(
                                p, __fadd2_rn(make_float2(__uint_as_float(v2[2 * x]), __uint_as_float(v2[2 * x + 1])),
                                              make_float2(m.y, m.w)));
                            pk[x] = pack_bf16x2(p.x, p.y);
                            dk[x] = pack_bf16x2(ds.x, ds.y);
                        }
                    } else {
#pragma unroll
                        for (int x = 0; x < KC / 2; ++x) {
                            float pe[2], de[2];
#pragma unroll
                            for (int y = 0; y < 2; ++y) {
                                const int cc = col0 + KC * c + 2 * x + y;
                                const float4 m = meta[cc];  // (lse2, D, t, a(t)) of column cc; t = -1 past n
                                const int t = __float_as_int(m.z), at = __float_as_int(m.w);
                                const bool vis = kvalid && key <= t && key >= at;
                                const float p = vis ? fast_exp2(fmaf(__uint_as_float(v1[2 * x + y]), sc2, -m.x)) : 0.f;
                                pe[y] = p;
                                de[y] = p * (__uint_as_float(v2[2 * x + y]) - m.y);
                            }
                            pk[x] = pack_bf16x2(pe[0], pe[1]);
                            dk[x] = pack_bf16x2(de[0], de[1]);
                        }
                    }
                    if constexpr (KC == 32) {
                        tmem_st16(lane_base + C::T_ST + (g & 1u) * NQ + col0 + 16 * c, pk);
                        tmem_st16(lane_base + C::T_DPT + (g & 1u) * NQ + col0 + 16 * c, dk);
                    } else {
                        tmem_st8(lane_base + C::T_ST + (g & 1u) * NQ + col0 + 8 * c, pk);
                        tmem_st8(lane_base + C::T_DPT + (g & 1u) * NQ + col0 + 8 * c, dk);
                    }
                }
                tmem_wait_st();
                tmem_fence_before();
                mbar_arrive(&p_full[sb]);
            }
            if (!ok) break;
            if (!warp_wait(&item_done, ic & 1u, limit)) {
                ok = false;
                break;
            }
            tmem_fence_after();
            const size_t row = static_cast<size_t>(it.pair) * a.n + (kvalid ? key : 0);
            // dV, then dK scaled by 1/sqrt(d): with two warpgroups, 0 writes dV and 1 writes dK
#pragma unroll
            for (int o = 0; o < 2; ++o) {
                if (WGS == 2 && o != wg) continue;
                const float f = o == 0 ? 1.f : sc;
                float* dst_row = (o == 0 ? a.dv : a.dk) + row * D;
                const bool wide = (reinterpret_cast<uintptr_t>(o == 0 ? a.dv : a.dk) & 31u) == 0;
                const uint32_t src = lane_base + (o == 0 ? C::T_DV : C::T_DK);
#pragma unroll
                for (int c = 0; c < D / 32; ++c) {
                    uint32_t v[32];
                    tmem_ld32(src + 32 * c, v);
                    tmem_wait_ld();
                    if (kvalid) store_row32(dst_row + 32 * c, v, f, wide);
                }
            }
            tmem_fence_before();
            mbar_arrive(&o_free);
            gt += it.nqt;
        }
        if (!ok) {
            abort_s = 1;
            atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
        }
    }
    tmem_fence_before();
    __syncthreads();
    tmem_fence_after();
    if (warp == 0) tmem_dealloc<C::TMEM_COLS>(tmem);
}

// One backward call: delta, the dK/dV pass (shape CK) and the dQ pass (shape CQ), each pass a
// persistent grid of CTAS CTAs per SM where they fit.
template <int D, typename CQ, typename CK>
cudaError_t launch_bwd_shape(const BackwardArgs& a, cudaStream_t stream)
{
    constexpr int G = CQ::M / CQ::QT;
    auto kv_kernel = bwd_kv_tc_kernel<D, G, CK::NQ, CK::WGS, CK::CTAS>;
    auto q_kernel = bwd_q_tc_kernel<D, G, CQ::NK, CQ::WGS, CQ::CTAS>;
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    // each pass's shared-memory opt-in and its resident CTAs per SM, once per device
    static std::atomic<int> kv_cache[kMaxCachedDevices] = {}, q_cache[kMaxCachedDevices] = {};
    const int kv_per_sm = cached_per_device(kv_cache, dev, [&] {
        err = cudaFuncSetAttribute(kv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, CK::SMEM);
        return err == cudaSuccess ? resident_ctas(kv_kernel, CK::THREADS, CK::SMEM, CK::CTAS, dev) : 0;
    });
    if (kv_per_sm < 1) return err;
    const int q_per_sm = cached_per_device(q_cache, dev, [&] {
        err = cudaFuncSetAttribute(q_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, CQ::SMEM);
        return err == cudaSuccess ? resident_ctas(q_kernel, CQ::THREADS, CQ::SMEM, CQ::CTAS, dev) : 0;
    });
    if (q_per_sm < 1) return err;
    int sms = 0;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    const unsigned long long qrows = static_cast<unsigned long long>(a.batch) * a.Hq * a.n;
    const unsigned long long krows = static_cast<unsigned long long>(a.batch) * a.Hkv * a.n;
    // dQ pass: Q/dO in items of 128 rows, K/V in tiles of NK; dK/dV pass: K/V in items of
    // 128 keys, Q/dO in tiles of NQ rows
    CUtensorMap q1, d1, k1, v1, q2, d2, k2, v2;
    if (!rows_tensor_map(&q1, a.q, qrows, D, CQ::QT) || !rows_tensor_map(&d1, a.dout, qrows, D, CQ::QT) ||
        !rows_tensor_map(&k1, a.k, krows, D, CQ::NK) || !rows_tensor_map(&v1, a.v, krows, D, CQ::NK) ||
        !rows_tensor_map(&q2, a.q, qrows, D, CK::QT) || !rows_tensor_map(&d2, a.dout, qrows, D, CK::QT) ||
        !rows_tensor_map(&k2, a.k, krows, D, CK::M) || !rows_tensor_map(&v2, a.v, krows, D, CK::M))
        return cudaErrorInvalidValue;
    {
        constexpr int TPR = D / 8;
        const long long threads = static_cast<long long>(qrows) * TPR;
        const long long blocks = (threads + 255) / 256;
        if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
        delta_kernel<D><<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
            static_cast<const __nv_bfloat16*>(a.out), static_cast<const __nv_bfloat16*>(a.dout), a.delta,
            static_cast<long long>(qrows));
        err = cudaGetLastError();
        if (err != cudaSuccess) return err;
    }
    const long long kv_items = static_cast<long long>(a.batch) * a.Hkv * ((a.n + 127) / 128);
    const long long q_items = static_cast<long long>(a.batch) * a.Hkv * ((a.n + CQ::QT - 1) / CQ::QT);
    if (kv_items > 0x7fffffffLL || q_items > 0x7fffffffLL) return cudaErrorInvalidValue;
    const long long kv_slots = static_cast<long long>(sms) * kv_per_sm;
    const long long q_slots = static_cast<long long>(sms) * q_per_sm;
    const int kv_grid = static_cast<int>(kv_items < kv_slots ? kv_items : kv_slots);
    const int q_grid = static_cast<int>(q_items < q_slots ? q_items : q_slots);
    kv_kernel<<<kv_grid, CK::THREADS, CK::SMEM, stream>>>(q2, k2, v2, d2, a);
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    q_kernel<<<q_grid, CQ::THREADS, CQ::SMEM, stream>>>(q1, k1, v1, d1, a);
    return cudaGetLastError();
}

// Shapes: long supports (B >= 512), and d = 128 or GQA group 8, run both passes with 64-row
// tiles, two elementwise warpgroups and one CTA per SM (512 TMEM columns). Short supports at
// d = 64 and G <= 4 run 32-row tiles, one elementwise warpgroup and two CTAs per SM (256
// columns each), so one CTA's per-item latencies overlap the other's work. Build option
// PBB_BWD_SHORT_SHAPE = 0 keeps every call on the long shape.
#ifndef PBB_BWD_SHORT_SHAPE
#define PBB_BWD_SHORT_SHAPE 1
#endif
// Keys per tile of the dQ pass in the long shape: 128 (one dP buffer, released early) or 64 (two).
#ifndef PBB_BWD_Q_NK
#define PBB_BWD_Q_NK 128
#endif
// Query rows per tile of the dK/dV pass in the long shape: 128 (one S^T and one dP^T buffer) or 64
// (two each).
#ifndef PBB_BWD_KV_NQ
#define PBB_BWD_KV_NQ 128
#endif

template <int D, int G>
cudaError_t launch_bwd(const BackwardArgs& a, cudaStream_t stream)
{
    if constexpr (D == 64 && G <= 4 && PBB_BWD_SHORT_SHAPE == 1) {
        if (a.B < 512)
            return launch_bwd_shape<D, BqCfg<D, G, 32, 1, 2>, BkvCfg<D, G, 32, 1, 2>>(a, stream);
    }
    return launch_bwd_shape<D, BqCfg<D, G, PBB_BWD_Q_NK, 2, 1>, BkvCfg<D, G, PBB_BWD_KV_NQ, 2, 1>>(a, stream);
}

template <int D>
cudaError_t launch_bwd_d(const BackwardArgs& a, cudaStream_t stream)
{
    switch (a.Hq / a.Hkv) {
        case 1: return launch_bwd<D, 1>(a, stream);
        case 2: return launch_bwd<D, 2>(a, stream);
        case 4: return launch_bwd<D, 4>(a, stream);
        case 8: return launch_bwd<D, 8>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_backward(const BackwardArgs& a, cudaStream_t stream)
{
    if (a.d == 64) return launch_bwd_d<64>(a, stream);
    if (a.d == 128) return launch_bwd_d<128>(a, stream);
    return cudaErrorInvalidValue;
}

cudaError_t read_and_clear_backward_status(int* status)
{
    cudaError_t err = cudaMemcpyFromSymbol(status, g_bwd_status, sizeof(int));
    if (err != cudaSuccess) return err;
    if (*status != kDevOk) {
        const int zero = kDevOk;
        err = cudaMemcpyToSymbol(g_bwd_status, &zero, sizeof(int));
    }
    return err;
}

}  // namespace pbb
