// PBB attention over whole sequences (the forward pass / prefill) for sm_103a.
//
// Every position t of a sequence attends to the interval [a(t), t],
// a(t) = max(0, h(floor(t/h) - 1)) (Eq. pbb_relay, the interval form of
// Eq. pbb, Sec. 3): the whole previous half-block and the causal prefix of its
// own half-block, with the single softmax of Eq. (attention). Each output row
// also gets its natural-log partition lse = ln sum exp(z) (Eq. lse), which a
// backward pass reuses.
//
// Work. A CTA takes QT consecutive positions t0 .. t0+QT-1 of all G query
// heads of one KV head: M = G*QT = 64 query rows, stacked head-major, so every
// K/V tile it streams serves all G heads (native GQA, K/V read once per CTA).
// Its keys are [a(t0), t_last]; a(t) only grows with t, so that range covers
// every row, and rows whose support starts later or ends earlier are masked in
// the tiles that cross their bounds (no dense mask exists anywhere).
//
// Data movement. One producer lane issues TMA tensor copies (128-byte swizzle,
// boxes of 64 columns): first the Q rows of the CTA, then the K/V tiles of 64
// keys into a STAGES-deep ring of full/empty mbarriers.
//
// Math. Four consumer warps own 16 query rows each and run FlashAttention-style
// tiles on mma.sync m16n8k16 (bf16 operands, fp32 accumulation): S = Q K^T from
// ldmatrix fragments of the swizzled tiles, an online softmax in the base-2
// domain (log2(e)/sqrt(d) folded into one scale; the output is rescaled only
// when a row's running maximum grows), P rounded to bf16 as the A operand of
// O += P V with V fragments from ldmatrix.trans. The epilogue divides by the
// row sums and writes O (bf16 or fp32) and lse.
//
// Every wait is bounded by the global timer; a wait that runs out records a
// timeout in this file's status word, the CTA drains its copies and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pbb_device.cuh"
#include "pbb_internal.h"

namespace pbb {

__device__ int g_fwd_status;  // first fault recorded by a forward kernel, kDevOk if none

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr unsigned long long kGuardNs = 2000000000ull;  // waits only a broken GPU can exceed
constexpr int kFwdConsumers = 4;                         // warps that compute, 16 query rows each
constexpr int kFwdThreads = (kFwdConsumers + 1) * 32;    // plus one producer warp

template <int D, int G>
struct FwdCfg {
    static constexpr int M = 16 * kFwdConsumers;        // query rows of a CTA (G heads x QT positions)
    static constexpr int QT = M / G;                    // positions of a CTA
    static constexpr int NK = 64;                       // keys per K/V tile
    static constexpr int BOXES = D / 64;                // 64-column boxes of a row
    static constexpr int KBOX = NK * 128;               // bytes of one K (or V) box
    static constexpr int QBOX = M * 128;                // bytes of one Q box
    static constexpr int STAGE = 2 * BOXES * KBOX;      // K boxes then V boxes
    static constexpr int STAGES = D == 128 ? 2 : 3;
    static constexpr int Q_OFF = STAGES * STAGE;
    static constexpr int SMEM = Q_OFF + BOXES * QBOX + 1024;  // + alignment slack
    static constexpr int KSTEPS = D / 16;               // k-steps of S = Q K^T
    static constexpr int NT_S = NK / 8;                 // 8-key n-tiles of S
    static constexpr int NT_O = D / 8;                  // 8-dim n-tiles of O
    static_assert(QT % 8 == 0, "a head's Q rows must start on a swizzle atom (8 rows)");
    static_assert(KBOX % 1024 == 0 && QBOX % 1024 == 0, "boxes keep 1024-byte alignment");
};

// Start of the PBB support of position t: a(t) = max(0, h (floor(t/h) - 1)).
__device__ __forceinline__ int support_start(int t, int h)
{
    const int m = t / h;
    return m > 0 ? h * (m - 1) : 0;
}

template <int D, int G>
__global__ void __launch_bounds__(kFwdThreads, 2)
forward_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
               const __grid_constant__ CUtensorMap vmap, const ForwardArgs a)
{
    using C = FwdCfg<D, G>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ unsigned char dsmem_raw[];
    __shared__ __align__(8) uint64_t full_bar[STAGES];
    __shared__ __align__(8) uint64_t empty_bar[STAGES];
    __shared__ __align__(8) uint64_t q_bar;
    __shared__ volatile int abort_s;
    unsigned char* dsmem = reinterpret_cast<unsigned char*>(
        (reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~static_cast<uintptr_t>(1023));

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // item -> (sequence, KV head, query tile); query tiles of a head are adjacent,
    // so CTAs running together share K/V tiles in L2
    const int nq = (a.n + C::QT - 1) / C::QT;
    const int qtile = static_cast<int>(blockIdx.x % static_cast<unsigned>(nq));
    const int pair = static_cast<int>(blockIdx.x / static_cast<unsigned>(nq));
    const int b = pair / a.Hkv, kvh = pair - b * a.Hkv;
    const int h = a.B >> 1;
    const int t0 = qtile * C::QT;
    const int tl = min(t0 + C::QT, a.n) - 1;   // last valid position of the CTA
    const int lo = support_start(t0, h);       // first key any row needs
    const int ntiles = (tl - lo + C::NK) / C::NK;
    const int a_max = support_start(tl, h);    // latest support start among the rows

    if (tid == 0) {
#pragma unroll
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], kFwdConsumers);
        }
        mbar_init(&q_bar, 1);
        fence_mbar_init();
        abort_s = 0;
    }
    __syncthreads();

    int issued = 0;  // K/V tiles issued (producer lane only)
    if (warp == kFwdConsumers) {
        // ================= producer: one lane =================
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&kmap)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&vmap)) : "memory");
            mbar_expect_tx(&q_bar, static_cast<uint32_t>(C::BOXES * C::QBOX));
            const int qrow0 = (b * a.Hq + kvh * G) * a.n + t0;
#pragma unroll
            for (int gi = 0; gi < G; ++gi)
#pragma unroll
                for (int bx = 0; bx < C::BOXES; ++bx)
                    tma_load_2d(dsmem + C::Q_OFF + bx * C::QBOX + gi * C::QT * 128, &qmap, bx * 64,
                                qrow0 + gi * a.n, &q_bar);
            const int krow0 = pair * a.n + lo;
            for (int it = 0; it < ntiles; ++it) {
                const int s = it % STAGES;
                if (it >= STAGES &&
                    !mbar_wait(&empty_bar[s], static_cast<uint32_t>((it / STAGES - 1) & 1), a.timeout_ns)) {
                    abort_s = 1;
                    atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
                    break;
                }
                if (abort_s) break;
                unsigned char* st = dsmem + s * C::STAGE;
                mbar_expect_tx(&full_bar[s], static_cast<uint32_t>(C::STAGE));
#pragma unroll
                for (int bx = 0; bx < C::BOXES; ++bx) {
                    tma_load_2d(st + bx * C::KBOX, &kmap, bx * 64, krow0 + it * C::NK, &full_bar[s]);
                    tma_load_2d(st + (C::BOXES + bx) * C::KBOX, &vmap, bx * 64, krow0 + it * C::NK, &full_bar[s]);
                }
                ++issued;
            }
        }
    } else {
        // ================= consumers: 16 query rows per warp =================
        const int g = lane >> 2, tig = lane & 3;  // fragment row group and thread in group
        const int lm = lane >> 3;                 // which 8x8 matrix this lane addresses
        const float qscale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
        // the warp's two rows per thread: r0 = 16 warp + g, r1 = r0 + 8 (CTA rows are head-major)
        const int r0 = 16 * warp + g, r1 = r0 + 8;
        const int tp0 = t0 + r0 % C::QT, tp1 = t0 + r1 % C::QT;    // their positions
        const int as0 = support_start(tp0, h), as1 = support_start(tp1, h);

        bool ok = mbar_wait(&q_bar, 0u, a.timeout_ns);
        uint32_t qa[C::KSTEPS][4];  // Q A-fragments of the warp's 16 rows
        if (ok) {
            const uint32_t qbase = smem_addr(dsmem + C::Q_OFF);
            const int row = 16 * warp + 8 * (lm & 1) + (lane & 7);
#pragma unroll
            for (int kk = 0; kk < C::KSTEPS; ++kk) {
                const int ch = 2 * kk + (lm >> 1);
                ldmatrix_x4(qa[kk], qbase + (ch >> 3) * C::QBOX + swz(row, ch & 7));
            }
        }
        float o[C::NT_O][4];
#pragma unroll
        for (int nt = 0; nt < C::NT_O; ++nt)
#pragma unroll
            for (int x = 0; x < 4; ++x) o[nt][x] = 0.f;
        float m0 = -INFINITY, m1 = -INFINITY;  // running maxima of rows r0, r1 (base-2 domain)
        float l0 = 0.f, l1 = 0.f;              // this thread's share of their running sums

        for (int it = 0; ok && it < ntiles; ++it) {
            const int s = it % STAGES;
            if (!mbar_wait(&full_bar[s], static_cast<uint32_t>((it / STAGES) & 1), a.timeout_ns)) {
                ok = false;
                break;
            }
            if (abort_s) {
                ok = false;
                break;
            }
            const uint32_t kbase = smem_addr(dsmem + s * C::STAGE);
            const uint32_t vbase = kbase + C::BOXES * C::KBOX;
            const int key0 = lo + it * C::NK;

            // ---- S = Q K^T for 16 rows x 64 keys
            float sc[C::NT_S][4];
#pragma unroll
            for (int nt = 0; nt < C::NT_S; ++nt)
#pragma unroll
                for (int x = 0; x < 4; ++x) sc[nt][x] = 0.f;
#pragma unroll
            for (int j = 0; j < C::NK / 16; ++j) {
                const int krow = 16 * j + 8 * (lm >> 1) + (lane & 7);
#pragma unroll
                for (int kk = 0; kk < C::KSTEPS; ++kk) {
                    const int ch = 2 * kk + (lm & 1);
                    uint32_t kb[4];
                    ldmatrix_x4(kb, kbase + (ch >> 3) * C::KBOX + swz(krow, ch & 7));
                    mma_bf16_16816(sc[2 * j], qa[kk], kb[0], kb[1]);
                    mma_bf16_16816(sc[2 * j + 1], qa[kk], kb[2], kb[3]);
                }
            }
            // ---- scale, mask where the tile crosses a row's bounds [a(t), t]
            const bool edge = (key0 + C::NK - 1 > t0) || (key0 < a_max);
#pragma unroll
            for (int nt = 0; nt < C::NT_S; ++nt) {
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    float z = sc[nt][x] * qscale;
                    if (edge) {
                        const int key = key0 + 8 * nt + 2 * tig + (x & 1);
                        const bool vis = (x < 2) ? (key >= as0 && key <= tp0) : (key >= as1 && key <= tp1);
                        z = vis ? z : -INFINITY;
                    }
                    sc[nt][x] = z;
                }
            }
            // ---- online softmax (base 2)
            float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
            for (int nt = 0; nt < C::NT_S; ++nt) {
                mx0 = fmaxf(mx0, fmaxf(sc[nt][0], sc[nt][1]));
                mx1 = fmaxf(mx1, fmaxf(sc[nt][2], sc[nt][3]));
            }
            mx0 = fmaxf(mx0, __shfl_xor_sync(kFull, mx0, 1));
            mx0 = fmaxf(mx0, __shfl_xor_sync(kFull, mx0, 2));
            mx1 = fmaxf(mx1, __shfl_xor_sync(kFull, mx1, 1));
            mx1 = fmaxf(mx1, __shfl_xor_sync(kFull, mx1, 2));
            const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
            if (__any_sync(kFull, (mn0 > m0) || (mn1 > m1))) {
                // a row with no visible key yet keeps m = -inf; its factor is 1 (o and l are 0)
                const float al0 = (mn0 == -INFINITY) ? 1.f : fast_exp2(m0 - mn0);
                const float al1 = (mn1 == -INFINITY) ? 1.f : fast_exp2(m1 - mn1);
                l0 *= al0;
                l1 *= al1;
#pragma unroll
                for (int nt = 0; nt < C::NT_O; ++nt) {
                    o[nt][0] *= al0;
                    o[nt][1] *= al0;
                    o[nt][2] *= al1;
                    o[nt][3] *= al1;
                }
            }
            m0 = mn0;
            m1 = mn1;
            const float b0 = (mn0 == -INFINITY) ? 0.f : mn0;
            const float b1 = (mn1 == -INFINITY) ? 0.f : mn1;
            uint32_t pa[C::NK / 16][4];  // P as bf16 A-fragments, one per 16-key k-step
#pragma unroll
            for (int kk = 0; kk < C::NK / 16; ++kk) {
                float p[2][4];
#pragma unroll
                for (int hlf = 0; hlf < 2; ++hlf) {
                    const int nt = 2 * kk + hlf;
                    p[hlf][0] = fast_exp2(sc[nt][0] - b0);
                    p[hlf][1] = fast_exp2(sc[nt][1] - b0);
                    p[hlf][2] = fast_exp2(sc[nt][2] - b1);
                    p[hlf][3] = fast_exp2(sc[nt][3] - b1);
                    l0 += p[hlf][0] + p[hlf][1];
                    l1 += p[hlf][2] + p[hlf][3];
                }
                pa[kk][0] = pack_bf16x2(p[0][0], p[0][1]);
                pa[kk][1] = pack_bf16x2(p[0][2], p[0][3]);
                pa[kk][2] = pack_bf16x2(p[1][0], p[1][1]);
                pa[kk][3] = pack_bf16x2(p[1][2], p[1][3]);
            }
            // ---- O += P V
#pragma unroll
            for (int kk = 0; kk < C::NK / 16; ++kk) {
                const int vrow = 16 * kk + 8 * (lm & 1) + (lane & 7);
#pragma unroll
                for (int j = 0; j < D / 16; ++j) {
                    const int ch = 2 * j + (lm >> 1);
                    uint32_t vb[4];
                    ldmatrix_x4_trans(vb, vbase + (ch >> 3) * C::KBOX + swz(vrow, ch & 7));
                    mma_bf16_16816(o[2 * j], pa[kk], vb[0], vb[1]);
                    mma_bf16_16816(o[2 * j + 1], pa[kk], vb[2], vb[3]);
                }
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&empty_bar[s]);
        }
        if (!ok) {
            abort_s = 1;
            atomicCAS(&g_fwd_status, kDevOk, kDevTimeout);
        } else {
            // ---- epilogue: row sums over the quad, normalise, write O and lse
            l0 += __shfl_xor_sync(kFull, l0, 1);
            l0 += __shfl_xor_sync(kFull, l0, 2);
            l1 += __shfl_xor_sync(kFull, l1, 1);
            l1 += __shfl_xor_sync(kFull, l1, 2);
            const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f;
            const float inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
            const int gi0 = r0 / C::QT, gi1 = r1 / C::QT;
            const size_t row0 = static_cast<size_t>(b * a.Hq + kvh * G + gi0) * a.n + tp0;
            const size_t row1 = static_cast<size_t>(b * a.Hq + kvh * G + gi1) * a.n + tp1;
            const bool w0 = tp0 < a.n, w1 = tp1 < a.n;
            if (a.out_f32) {
                float* out = static_cast<float*>(a.out);
#pragma unroll
                for (int nt = 0; nt < C::NT_O; ++nt) {
                    const int dim = 8 * nt + 2 * tig;
                    if (w0) *reinterpret_cast<float2*>(out + row0 * D + dim) = make_float2(o[nt][0] * inv0, o[nt][1] * inv0);
                    if (w1) *reinterpret_cast<float2*>(out + row1 * D + dim) = make_float2(o[nt][2] * inv1, o[nt][3] * inv1);
                }
            } else {
                uint32_t* out = static_cast<uint32_t*>(a.out);  // bf16 pairs
#pragma unroll
                for (int nt = 0; nt < C::NT_O; ++nt) {
                    const int dim = 8 * nt + 2 * tig;
                    if (w0) out[(row0 * D + dim) >> 1] = pack_bf16x2(o[nt][0] * inv0, o[nt][1] * inv0);
                    if (w1) out[(row1 * D + dim) >> 1] = pack_bf16x2(o[nt][2] * inv1, o[nt][3] * inv1);
                }
            }
            if (a.lse != nullptr && tig == 0) {
                // ln sum exp(z) = (m2 + log2 l) ln 2, m2 the base-2 running maximum
                constexpr float kLn2 = 0.6931471805599453f;
                if (w0) a.lse[row0] = (m0 + log2f(l0)) * kLn2;
                if (w1) a.lse[row1] = (m1 + log2f(l1)) * kLn2;
            }
        }
    }
    __syncthreads();
    if (abort_s && warp == kFwdConsumers && lane == 0) {
        // drain: wait (bounded) for the copies this CTA issued before its shared memory goes away
        mbar_wait(&q_bar, 0u, kGuardNs);
        for (int s = 0; s < STAGES && s < issued; ++s) {
            const int j = s + STAGES * ((issued - 1 - s) / STAGES);
            mbar_wait(&full_bar[s], static_cast<uint32_t>((j / STAGES) & 1), kGuardNs);
        }
    }
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

template <int D, int G>
cudaError_t launch_fwd(const ForwardArgs& a, cudaStream_t stream)
{
    using C = FwdCfg<D, G>;
    static bool attr_set[64] = {};
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 64 && !attr_set[dev]) {
        err = cudaFuncSetAttribute(forward_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (err != cudaSuccess) return err;
        attr_set[dev] = true;
    }
    CUtensorMap qmap, kmap, vmap;
    const unsigned long long qrows = static_cast<unsigned long long>(a.batch) * a.Hq * a.n;
    const unsigned long long krows = static_cast<unsigned long long>(a.batch) * a.Hkv * a.n;
    if (!rows_tensor_map(&qmap, a.q, qrows, D, C::QT) || !rows_tensor_map(&kmap, a.k, krows, D, C::NK) ||
        !rows_tensor_map(&vmap, a.v, krows, D, C::NK))
        return cudaErrorInvalidValue;
    const long long nq = (a.n + C::QT - 1) / C::QT;
    const long long grid = static_cast<long long>(a.batch) * a.Hkv * nq;
    if (grid < 1) return cudaSuccess;
    if (grid > 0x7fffffffLL) return cudaErrorInvalidValue;
    forward_kernel<D, G><<<static_cast<unsigned>(grid), kFwdThreads, C::SMEM, stream>>>(qmap, kmap, vmap, a);
    return cudaGetLastError();
}

template <int D>
cudaError_t launch_fwd_d(const ForwardArgs& a, cudaStream_t stream)
{
    switch (a.Hq / a.Hkv) {
        case 1: return launch_fwd<D, 1>(a, stream);
        case 2: return launch_fwd<D, 2>(a, stream);
        case 4: return launch_fwd<D, 4>(a, stream);
        case 8: return launch_fwd<D, 8>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_forward(const ForwardArgs& a, cudaStream_t stream)
{
    if (a.d == 64) return launch_fwd_d<64>(a, stream);
    if (a.d == 128) return launch_fwd_d<128>(a, stream);
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
