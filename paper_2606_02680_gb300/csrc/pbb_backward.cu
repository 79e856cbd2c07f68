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
//   delta_kernel   D for every row (dO . O);
//   bwd_kv_kernel  one CTA per (sequence, KV head, tile of 64 keys): it streams
//                  the query tiles whose supports hold any of its keys (positions
//                  s0 .. h(floor(s_last/h) + 2) - 1: the key's own half-block and
//                  the next one, bridge rows included) with all G heads of the group
//                  stacked as 64 rows, and accumulates dK and dV for its keys in
//                  registers (each warp owns 16 keys);
//   bwd_q_kernel   one CTA per (sequence, KV head, 64 query rows): it streams the
//                  key tiles of [a(t0), t_last] and accumulates dQ (each warp owns
//                  16 query rows).
// Tiles arrive by TMA (128-byte swizzle) through a full/empty mbarrier ring fed by
// one producer lane; the products are mma.sync m16n8k16 (bf16 operands, fp32
// accumulation), with P and dS rounded to bf16 as operands. Every wait is bounded by
// the global timer; a wait that runs out records a timeout and the CTA drains its
// copies and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pbb_device.cuh"
#include "pbb_internal.h"

namespace pbb {

__device__ int g_bwd_status;  // first fault recorded by a backward kernel, kDevOk if none

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr unsigned long long kGuardNs = 2000000000ull;
constexpr int kBwdConsumers = 4;
constexpr int kBwdThreads = (kBwdConsumers + 1) * 32;
constexpr float kLog2e = 1.4426950408889634f;

template <int D, int G>
struct BwdCfg {
    static constexpr int M = 64;              // query rows of a query tile (G heads x QT positions)
    static constexpr int QT = M / G;
    static constexpr int KT = 64;             // keys of a key tile (16 per warp)
    static constexpr int BOXES = D / 64;
    static constexpr int BOX = 64 * 128;      // one 64-row x 64-column bf16 box
    static constexpr int TILE = BOXES * BOX;  // one 64-row tile of d columns
    static constexpr int STAGES = 2;
    static constexpr int STAGE = 2 * TILE;    // (Q, dO) or (K, V)
    static constexpr int FIX_OFF = 0;         // the CTA's fixed pair of tiles
    static constexpr int RING_OFF = 2 * TILE;
    static constexpr int SMEM = RING_OFF + STAGES * STAGE + 1024;
    static constexpr int KSTEPS = D / 16;
    static constexpr int RC = D == 128 ? 16 : 32;  // query rows per inner step of the dK/dV kernel
    static_assert(QT % 8 == 0, "a head's rows must start on a swizzle atom");
};

__device__ __forceinline__ int support_start(int t, int h)
{
    const int m = t / h;
    return m > 0 ? h * (m - 1) : 0;
}

// Byte offset of 16-byte chunk ch (0 .. D/8 - 1) of row r in a 64-row tile of BOXES boxes.
template <int BOX>
__device__ __forceinline__ uint32_t tile_off(int r, int ch)
{
    return static_cast<uint32_t>((ch >> 3) * BOX) + swz(r, ch & 7);
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

// ------------------------------------------------------------- dK, dV ----

template <int D, int G>
__global__ void __launch_bounds__(kBwdThreads, 1)
bwd_kv_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
              const __grid_constant__ CUtensorMap vmap, const __grid_constant__ CUtensorMap dmap,
              const BackwardArgs a)
{
    using C = BwdCfg<D, G>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ unsigned char dsmem_raw[];
    __shared__ __align__(8) uint64_t fix_bar, full_bar[STAGES], empty_bar[STAGES];
    __shared__ volatile int abort_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    const int nk = (a.n + C::KT - 1) / C::KT;
    const int ktile = static_cast<int>(blockIdx.x % static_cast<unsigned>(nk));
    const int pair = static_cast<int>(blockIdx.x / static_cast<unsigned>(nk));
    const int b = pair / a.Hkv, kvh = pair - b * a.Hkv;
    const int h = a.B >> 1;
    const int s0 = ktile * C::KT;
    const int s_last = min(s0 + C::KT, a.n) - 1;
    const int t_end = min(a.n, h * (s_last / h + 2));  // queries past t_end - 1 never see these keys
    const int tq0 = (s0 / C::QT) * C::QT;             // first query tile (key s is seen from t = s)
    const int nqt = (t_end - tq0 + C::QT - 1) / C::QT;

    if (tid == 0) {
        mbar_init(&fix_bar, 1);
#pragma unroll
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], kBwdConsumers);
        }
        fence_mbar_init();
        abort_s = 0;
    }
    __syncthreads();

    int issued = 0;
    if (warp == kBwdConsumers) {
        if (lane == 0) {
            mbar_expect_tx(&fix_bar, static_cast<uint32_t>(2 * C::TILE));
            const int krow = pair * a.n + s0;
#pragma unroll
            for (int bx = 0; bx < C::BOXES; ++bx) {
                tma_load_2d(dsmem + C::FIX_OFF + bx * C::BOX, &kmap, bx * 64, krow, &fix_bar);
                tma_load_2d(dsmem + C::FIX_OFF + C::TILE + bx * C::BOX, &vmap, bx * 64, krow, &fix_bar);
            }
            for (int it = 0; it < nqt; ++it) {
                const int s = it % STAGES;
                if (it >= STAGES &&
                    !mbar_wait(&empty_bar[s], static_cast<uint32_t>((it / STAGES - 1) & 1), a.timeout_ns)) {
                    abort_s = 1;
                    atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
                    break;
                }
                if (abort_s) break;
                unsigned char* st = dsmem + C::RING_OFF + s * C::STAGE;
                mbar_expect_tx(&full_bar[s], static_cast<uint32_t>(C::STAGE));
                const int t0 = tq0 + it * C::QT;
#pragma unroll
                for (int gi = 0; gi < G; ++gi) {
                    const int qrow = (b * a.Hq + kvh * G + gi) * a.n + t0;
#pragma unroll
                    for (int bx = 0; bx < C::BOXES; ++bx) {
                        tma_load_2d(st + bx * C::BOX + gi * C::QT * 128, &qmap, bx * 64, qrow, &full_bar[s]);
                        tma_load_2d(st + C::TILE + bx * C::BOX + gi * C::QT * 128, &dmap, bx * 64, qrow,
                                    &full_bar[s]);
                    }
                }
                ++issued;
            }
        }
    } else {
        const int g = lane >> 2, tig = lane & 3, lm = lane >> 3;
        const float sc2 = kLog2e * rsqrtf(static_cast<float>(D));  // base-2 logits
        const float sc = rsqrtf(static_cast<float>(D));
        const int key_a = s0 + 16 * warp + g, key_b = key_a + 8;   // this thread's keys (S^T rows)
        float dk[D / 8][4], dv[D / 8][4];
#pragma unroll
        for (int nt = 0; nt < D / 8; ++nt)
#pragma unroll
            for (int x = 0; x < 4; ++x) dk[nt][x] = dv[nt][x] = 0.f;
        bool ok = mbar_wait(&fix_bar, 0u, a.timeout_ns);
        const uint32_t kbase = smem_addr(dsmem + C::FIX_OFF), vbase = kbase + C::TILE;
        for (int it = 0; ok && it < nqt; ++it) {
            const int s = it % STAGES;
            if (!mbar_wait(&full_bar[s], static_cast<uint32_t>((it / STAGES) & 1), a.timeout_ns) || abort_s) {
                ok = false;
                break;
            }
            const uint32_t qbase = smem_addr(dsmem + C::RING_OFF + s * C::STAGE), dbase = qbase + C::TILE;
            const int t0 = tq0 + it * C::QT;
            constexpr int RC = C::RC, NT = RC / 8, KQ = RC / 16;
#pragma unroll 1
            for (int rc = 0; rc < C::M / RC; ++rc) {  // RC query rows at a time
                // per-row data of the columns (query rows) this thread's fragments touch
                float l2[NT][2], dl[NT][2];
                int tpos[NT][2], tstart[NT][2];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        const int R = RC * rc + 8 * nt + 2 * tig + e;
                        const int gi = R / C::QT;
                        const int t = t0 + (R - gi * C::QT);
                        tpos[nt][e] = t;
                        tstart[nt][e] = support_start(t, h);
                        const size_t row = static_cast<size_t>(b * a.Hq + kvh * G + gi) * a.n + (t < a.n ? t : 0);
                        l2[nt][e] = (t < a.n) ? a.lse[row] * kLog2e : 0.f;
                        dl[nt][e] = (t < a.n) ? a.delta[row] : 0.f;
                    }
                // S^T = K_w Q^T and dP^T = V_w dO^T (16 keys x RC rows)
                float st[NT][4], dpt[NT][4];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                    for (int x = 0; x < 4; ++x) st[nt][x] = dpt[nt][x] = 0.f;
#pragma unroll
                for (int kk = 0; kk < C::KSTEPS; ++kk) {
                    uint32_t ka[4], va[4];
                    const int arow = 16 * warp + 8 * (lm & 1) + (lane & 7);
                    const int ach = 2 * kk + (lm >> 1);
                    ldmatrix_x4(ka, kbase + tile_off<C::BOX>(arow, ach));
                    ldmatrix_x4(va, vbase + tile_off<C::BOX>(arow, ach));
#pragma unroll
                    for (int p = 0; p < KQ; ++p) {
                        const int brow = RC * rc + 16 * p + 8 * (lm >> 1) + (lane & 7);
                        const int bch = 2 * kk + (lm & 1);
                        uint32_t qb[4], db[4];
                        ldmatrix_x4(qb, qbase + tile_off<C::BOX>(brow, bch));
                        ldmatrix_x4(db, dbase + tile_off<C::BOX>(brow, bch));
                        mma_bf16_16816(st[2 * p], ka, qb[0], qb[1]);
                        mma_bf16_16816(st[2 * p + 1], ka, qb[2], qb[3]);
                        mma_bf16_16816(dpt[2 * p], va, db[0], db[1]);
                        mma_bf16_16816(dpt[2 * p + 1], va, db[2], db[3]);
                    }
                }
                // P^T and dS^T, masked to a(t) <= s <= t
                uint32_t pa[KQ][4], sa[KQ][4];
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    float p4[4], d4[4];
#pragma unroll
                    for (int x = 0; x < 4; ++x) {
                        const int key = (x < 2) ? key_a : key_b;
                        const int e = x & 1;
                        const int t = tpos[nt][e];
                        const bool vis = key < a.n && t < a.n && key <= t && key >= tstart[nt][e];
                        const float p = vis ? fast_exp2(fmaf(st[nt][x], sc2, -l2[nt][e])) : 0.f;
                        p4[x] = p;
                        d4[x] = p * (dpt[nt][x] - dl[nt][e]);
                    }
                    const int kq = nt >> 1, hf = nt & 1;
                    pa[kq][2 * hf] = pack_bf16x2(p4[0], p4[1]);
                    pa[kq][2 * hf + 1] = pack_bf16x2(p4[2], p4[3]);
                    sa[kq][2 * hf] = pack_bf16x2(d4[0], d4[1]);
                    sa[kq][2 * hf + 1] = pack_bf16x2(d4[2], d4[3]);
                }
                // dV_w += P^T dO and dK_w += dS^T Q over these RC rows
#pragma unroll
                for (int kq = 0; kq < KQ; ++kq) {
                    const int vrow = RC * rc + 16 * kq + 8 * (lm & 1) + (lane & 7);
#pragma unroll
                    for (int j = 0; j < D / 16; ++j) {
                        const int ch = 2 * j + (lm >> 1);
                        uint32_t db[4], qb[4];
                        ldmatrix_x4_trans(db, dbase + tile_off<C::BOX>(vrow, ch));
                        ldmatrix_x4_trans(qb, qbase + tile_off<C::BOX>(vrow, ch));
                        mma_bf16_16816(dv[2 * j], pa[kq], db[0], db[1]);
                        mma_bf16_16816(dv[2 * j + 1], pa[kq], db[2], db[3]);
                        mma_bf16_16816(dk[2 * j], sa[kq], qb[0], qb[1]);
                        mma_bf16_16816(dk[2 * j + 1], sa[kq], qb[2], qb[3]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty_bar[s]);
        }
        if (!ok) {
            abort_s = 1;
            atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
        } else {
            // rows key_a, key_b; columns 8 nt + 2 tig, +1
            const size_t base = static_cast<size_t>(pair) * a.n;
#pragma unroll
            for (int nt = 0; nt < D / 8; ++nt) {
                const int col = 8 * nt + 2 * tig;
                if (key_a < a.n) {
                    *reinterpret_cast<float2*>(a.dk + (base + key_a) * D + col) = make_float2(dk[nt][0] * sc, dk[nt][1] * sc);
                    *reinterpret_cast<float2*>(a.dv + (base + key_a) * D + col) = make_float2(dv[nt][0], dv[nt][1]);
                }
                if (key_b < a.n) {
                    *reinterpret_cast<float2*>(a.dk + (base + key_b) * D + col) = make_float2(dk[nt][2] * sc, dk[nt][3] * sc);
                    *reinterpret_cast<float2*>(a.dv + (base + key_b) * D + col) = make_float2(dv[nt][2], dv[nt][3]);
                }
            }
        }
    }
    __syncthreads();
    if (abort_s && warp == kBwdConsumers && lane == 0) {
        mbar_wait(&fix_bar, 0u, kGuardNs);
        for (int s = 0; s < STAGES && s < issued; ++s) {
            const int j = s + STAGES * ((issued - 1 - s) / STAGES);
            mbar_wait(&full_bar[s], static_cast<uint32_t>((j / STAGES) & 1), kGuardNs);
        }
    }
}

// ------------------------------------------------------------------ dQ ----

template <int D, int G>
__global__ void __launch_bounds__(kBwdThreads, 1)
bwd_q_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
             const __grid_constant__ CUtensorMap vmap, const __grid_constant__ CUtensorMap dmap,
             const BackwardArgs a)
{
    using C = BwdCfg<D, G>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ unsigned char dsmem_raw[];
    __shared__ __align__(8) uint64_t fix_bar, full_bar[STAGES], empty_bar[STAGES];
    __shared__ volatile int abort_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    const int nq = (a.n + C::QT - 1) / C::QT;
    const int qtile = static_cast<int>(blockIdx.x % static_cast<unsigned>(nq));
    const int pair = static_cast<int>(blockIdx.x / static_cast<unsigned>(nq));
    const int b = pair / a.Hkv, kvh = pair - b * a.Hkv;
    const int h = a.B >> 1;
    const int t0 = qtile * C::QT;
    const int tl = min(t0 + C::QT, a.n) - 1;
    const int lo = support_start(t0, h);
    const int ntiles = (tl - lo + C::KT) / C::KT;
    const int a_max = support_start(tl, h);

    if (tid == 0) {
        mbar_init(&fix_bar, 1);
#pragma unroll
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], kBwdConsumers);
        }
        fence_mbar_init();
        abort_s = 0;
    }
    __syncthreads();

    int issued = 0;
    if (warp == kBwdConsumers) {
        if (lane == 0) {
            mbar_expect_tx(&fix_bar, static_cast<uint32_t>(2 * C::TILE));
#pragma unroll
            for (int gi = 0; gi < G; ++gi) {
                const int qrow = (b * a.Hq + kvh * G + gi) * a.n + t0;
#pragma unroll
                for (int bx = 0; bx < C::BOXES; ++bx) {
                    tma_load_2d(dsmem + C::FIX_OFF + bx * C::BOX + gi * C::QT * 128, &qmap, bx * 64, qrow, &fix_bar);
                    tma_load_2d(dsmem + C::FIX_OFF + C::TILE + bx * C::BOX + gi * C::QT * 128, &dmap, bx * 64, qrow,
                                &fix_bar);
                }
            }
            const int krow0 = pair * a.n + lo;
            for (int it = 0; it < ntiles; ++it) {
                const int s = it % STAGES;
                if (it >= STAGES &&
                    !mbar_wait(&empty_bar[s], static_cast<uint32_t>((it / STAGES - 1) & 1), a.timeout_ns)) {
                    abort_s = 1;
                    atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
                    break;
                }
                if (abort_s) break;
                unsigned char* st = dsmem + C::RING_OFF + s * C::STAGE;
                mbar_expect_tx(&full_bar[s], static_cast<uint32_t>(C::STAGE));
#pragma unroll
                for (int bx = 0; bx < C::BOXES; ++bx) {
                    tma_load_2d(st + bx * C::BOX, &kmap, bx * 64, krow0 + it * C::KT, &full_bar[s]);
                    tma_load_2d(st + C::TILE + bx * C::BOX, &vmap, bx * 64, krow0 + it * C::KT, &full_bar[s]);
                }
                ++issued;
            }
        }
    } else {
        const int g = lane >> 2, tig = lane & 3, lm = lane >> 3;
        const float sc2 = kLog2e * rsqrtf(static_cast<float>(D));
        const float sc = rsqrtf(static_cast<float>(D));
        const int r0 = 16 * warp + g, r1 = r0 + 8;
        const int gi0 = r0 / C::QT, gi1 = r1 / C::QT;
        const int tp0 = t0 + r0 - gi0 * C::QT, tp1 = t0 + r1 - gi1 * C::QT;
        const int as0 = support_start(tp0, h), as1 = support_start(tp1, h);
        const size_t row0 = static_cast<size_t>(b * a.Hq + kvh * G + gi0) * a.n + tp0;
        const size_t row1 = static_cast<size_t>(b * a.Hq + kvh * G + gi1) * a.n + tp1;
        const bool w0 = tp0 < a.n, w1 = tp1 < a.n;
        const float l20 = w0 ? a.lse[row0] * kLog2e : 0.f, l21 = w1 ? a.lse[row1] * kLog2e : 0.f;
        const float dl0 = w0 ? a.delta[row0] : 0.f, dl1 = w1 ? a.delta[row1] : 0.f;
        float dq[D / 8][4];
#pragma unroll
        for (int nt = 0; nt < D / 8; ++nt)
#pragma unroll
            for (int x = 0; x < 4; ++x) dq[nt][x] = 0.f;
        bool ok = mbar_wait(&fix_bar, 0u, a.timeout_ns);
        uint32_t qa[C::KSTEPS][4], da[C::KSTEPS][4];
        if (ok) {
            const uint32_t qbase = smem_addr(dsmem + C::FIX_OFF), dbase = qbase + C::TILE;
            const int row = 16 * warp + 8 * (lm & 1) + (lane & 7);
#pragma unroll
            for (int kk = 0; kk < C::KSTEPS; ++kk) {
                const int ch = 2 * kk + (lm >> 1);
                ldmatrix_x4(qa[kk], qbase + tile_off<C::BOX>(row, ch));
                ldmatrix_x4(da[kk], dbase + tile_off<C::BOX>(row, ch));
            }
        }
        for (int it = 0; ok && it < ntiles; ++it) {
            const int s = it % STAGES;
            if (!mbar_wait(&full_bar[s], static_cast<uint32_t>((it / STAGES) & 1), a.timeout_ns) || abort_s) {
                ok = false;
                break;
            }
            const uint32_t kbase = smem_addr(dsmem + C::RING_OFF + s * C::STAGE), vbase = kbase + C::TILE;
            const int key0 = lo + it * C::KT;
            // S = Q_w K^T and dP = dO_w V^T (16 rows x 64 keys)
            float sf[8][4], dp[8][4];
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                for (int x = 0; x < 4; ++x) sf[nt][x] = dp[nt][x] = 0.f;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int krow = 16 * j + 8 * (lm >> 1) + (lane & 7);
#pragma unroll
                for (int kk = 0; kk < C::KSTEPS; ++kk) {
                    const int ch = 2 * kk + (lm & 1);
                    uint32_t kb[4], vb[4];
                    ldmatrix_x4(kb, kbase + tile_off<C::BOX>(krow, ch));
                    ldmatrix_x4(vb, vbase + tile_off<C::BOX>(krow, ch));
                    mma_bf16_16816(sf[2 * j], qa[kk], kb[0], kb[1]);
                    mma_bf16_16816(sf[2 * j + 1], qa[kk], kb[2], kb[3]);
                    mma_bf16_16816(dp[2 * j], da[kk], vb[0], vb[1]);
                    mma_bf16_16816(dp[2 * j + 1], da[kk], vb[2], vb[3]);
                }
            }
            const bool edge = (key0 + C::KT - 1 > t0) || (key0 < a_max);
            uint32_t sa[4][4];  // dS as bf16 A-fragments, one per 16-key k-step
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                float d4[4];
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    const int key = key0 + 8 * nt + 2 * tig + (x & 1);
                    const bool hi = x >= 2;
                    bool vis = hi ? w1 : w0;
                    if (edge) vis = vis && (hi ? (key >= as1 && key <= tp1) : (key >= as0 && key <= tp0));
                    const float p = vis ? fast_exp2(fmaf(sf[nt][x], sc2, -(hi ? l21 : l20))) : 0.f;
                    d4[x] = p * (dp[nt][x] - (hi ? dl1 : dl0));
                }
                const int kq = nt >> 1, hf = nt & 1;
                sa[kq][2 * hf] = pack_bf16x2(d4[0], d4[1]);
                sa[kq][2 * hf + 1] = pack_bf16x2(d4[2], d4[3]);
            }
            // dQ_w += dS K
#pragma unroll
            for (int kq = 0; kq < 4; ++kq) {
                const int krow = 16 * kq + 8 * (lm & 1) + (lane & 7);
#pragma unroll
                for (int j = 0; j < D / 16; ++j) {
                    const int ch = 2 * j + (lm >> 1);
                    uint32_t kb[4];
                    ldmatrix_x4_trans(kb, kbase + tile_off<C::BOX>(krow, ch));
                    mma_bf16_16816(dq[2 * j], sa[kq], kb[0], kb[1]);
                    mma_bf16_16816(dq[2 * j + 1], sa[kq], kb[2], kb[3]);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty_bar[s]);
        }
        if (!ok) {
            abort_s = 1;
            atomicCAS(&g_bwd_status, kDevOk, kDevTimeout);
        } else {
#pragma unroll
            for (int nt = 0; nt < D / 8; ++nt) {
                const int col = 8 * nt + 2 * tig;
                if (w0) *reinterpret_cast<float2*>(a.dq + row0 * D + col) = make_float2(dq[nt][0] * sc, dq[nt][1] * sc);
                if (w1) *reinterpret_cast<float2*>(a.dq + row1 * D + col) = make_float2(dq[nt][2] * sc, dq[nt][3] * sc);
            }
        }
    }
    __syncthreads();
    if (abort_s && warp == kBwdConsumers && lane == 0) {
        mbar_wait(&fix_bar, 0u, kGuardNs);
        for (int s = 0; s < STAGES && s < issued; ++s) {
            const int j = s + STAGES * ((issued - 1 - s) / STAGES);
            mbar_wait(&full_bar[s], static_cast<uint32_t>((j / STAGES) & 1), kGuardNs);
        }
    }
}

template <int D, int G>
cudaError_t launch_bwd(const BackwardArgs& a, cudaStream_t stream)
{
    using C = BwdCfg<D, G>;
    static bool attr_set[64] = {};
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 64 && !attr_set[dev]) {
        err = cudaFuncSetAttribute(bwd_kv_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (err != cudaSuccess) return err;
        err = cudaFuncSetAttribute(bwd_q_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (err != cudaSuccess) return err;
        attr_set[dev] = true;
    }
    const unsigned long long qrows = static_cast<unsigned long long>(a.batch) * a.Hq * a.n;
    const unsigned long long krows = static_cast<unsigned long long>(a.batch) * a.Hkv * a.n;
    CUtensorMap qmap, kmap, vmap, dmap;
    if (!rows_tensor_map(&qmap, a.q, qrows, D, C::QT) || !rows_tensor_map(&dmap, a.dout, qrows, D, C::QT) ||
        !rows_tensor_map(&kmap, a.k, krows, D, C::KT) || !rows_tensor_map(&vmap, a.v, krows, D, C::KT))
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
    const long long kv_ctas = static_cast<long long>(a.batch) * a.Hkv * ((a.n + C::KT - 1) / C::KT);
    const long long q_ctas = static_cast<long long>(a.batch) * a.Hkv * ((a.n + C::QT - 1) / C::QT);
    if (kv_ctas > 0x7fffffffLL || q_ctas > 0x7fffffffLL) return cudaErrorInvalidValue;
    bwd_kv_kernel<D, G><<<static_cast<unsigned>(kv_ctas), kBwdThreads, C::SMEM, stream>>>(qmap, kmap, vmap, dmap, a);
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    bwd_q_kernel<D, G><<<static_cast<unsigned>(q_ctas), kBwdThreads, C::SMEM, stream>>>(qmap, kmap, vmap, dmap, a);
    return cudaGetLastError();
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
