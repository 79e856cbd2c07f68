// Kernels of the PBB decode step for sm_103a.
//
// Work decomposition. The support of a sequence at position t = p + r is the
// interval [a(t), t] (Eq. pbb_relay). Apart from the current token, which
// comes from k_new/v_new, it occupies at most two contiguous runs of ring
// slots (Appendix F.1): bridge phases (p > 0, r < h) read slots h..B-1 (the
// previous block's tail, positions p-h..p-1) and then 0..r-1; the other phases
// read 0..r-1. Counting those n keys in position order, logical key i lives in
// slot (base + i) mod B with base = h for a bridge phase and 0 otherwise.
//
// The grid is (chunk, KV head, sequence). CTA `chunk` takes logical keys
// [chunk*C, chunk*C + C) of its (sequence, KV head), serves all G = Hq/Hkv
// query heads of the group (each K/V byte is read from HBM once per step),
// and CTAs past the end of a short support exit at once. Chunk 0 also appends
// the new K/V to slot r and folds the current token into its softmax state;
// slot r is never in the read set, so the append and the reads do not race.
//
// Inside a CTA one thread streams K/V tiles of TK keys into a 4-stage shared
// memory ring with 1-D bulk copies (cp.async.bulk, completion on an mbarrier);
// a tile that straddles the ring's end is fetched as two copies. Each of the 4
// warps owns a quarter of every tile and keeps its own fp32 online softmax in
// the base-2 domain (the scale log2(e)/sqrt(d) is folded into q):
//   scores: 8 lanes per key, 4 keys per warp step; a lane holds q for d/8 dims
//           of all G heads in registers and the partial dot products are
//           combined with a reduce-scatter over the 8 lanes, so each lane ends
//           with the score of one (key, head);
//   P.V:    the warp walks its keys; every lane owns d/32 output dims of all G
//           heads and reads the weights of a key as a broadcast from shared
//           memory.
// The warps' states are merged in shared memory. A single-CTA support writes
// `out` directly; otherwise each CTA stores its partial (max, sum, output) and
// the last CTA of the (sequence, KV head) to arrive (an atomic counter, no
// spinning) fuses them in chunk order with Eq. (lse) and resets the counter,
// so the result does not depend on CTA scheduling.
//
// Every wait on an mbarrier is bounded (globaltimer); when it runs out the CTA
// records kDevTimeout, waits (bounded) for its own copies still in flight and
// returns without writing its output.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "pbb_internal.h"

namespace pbb {

__device__ int g_status;  // first device-side fault recorded, kDevOk if none

namespace {

constexpr int kWarps = 4;
constexpr int kThreads = kWarps * 32;
constexpr int kStages = 4;
constexpr int kTileBytes = 8192;  // bytes of K (and of V) per stage
constexpr unsigned kFull = 0xffffffffu;

// ---------------------------------------------------------------- PTX ----

__device__ __forceinline__ uint32_t smem_addr(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint64_t* bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ bool mbar_try(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ unsigned long long global_ns()
{
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Wait for phase `parity` of `bar` to complete, giving up after `limit_ns`.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity,
                                          unsigned long long limit_ns)
{
    if (mbar_test(bar, parity)) return true;
    if (limit_ns == 0) return false;
    const unsigned long long t0 = global_ns();
    while (!mbar_try(bar, parity)) {
        if (global_ns() - t0 > limit_ns) return false;
    }
    return true;
}

// 1-D bulk copy global -> shared, completion counted in bytes on `bar`.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

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

// Within each aligned group of 8 lanes, every lane holds G partial sums (one
// per head). Afterwards lane `sub` (0..7) holds the group's full sum for head
// sub >> (3 - log2 G): each exchange step halves the values a lane keeps and
// the steps left over once one value remains are plain butterfly sums.
template <int G>
__device__ __forceinline__ float reduce_scatter8(const float (&acc)[G], int sub)
{
    float v[G];
#pragma unroll
    for (int i = 0; i < G; ++i) v[i] = acc[i];
    int cnt = G;
#pragma unroll
    for (int lvl = 4; lvl >= 1; lvl >>= 1) {
        if (cnt > 1) {
            const int half = cnt / 2;
            const bool up = (sub & lvl) != 0;
#pragma unroll
            for (int i = 0; i < half; ++i) {
                const float send = up ? v[i] : v[i + half];
                const float keep = up ? v[i + half] : v[i];
                v[i] = keep + __shfl_xor_sync(kFull, send, lvl);
            }
            cnt = half;
        } else {
            v[0] += __shfl_xor_sync(kFull, v[0], lvl);
        }
    }
    return v[0];
}

template <int N>
struct Log2 {
    static constexpr int value = (N <= 1) ? 0 : 1 + Log2<N / 2>::value;
};
template <>
struct Log2<1> {
    static constexpr int value = 0;
};

// ------------------------------------------------------------ config ----

template <int ELEM, int D, int G>
struct Cfg {
    static constexpr int ROW = D * ELEM;            // bytes of one K or V row
    static constexpr int TK = kTileBytes / ROW;     // keys per tile
    static constexpr int KW = TK / kWarps;          // keys per warp per tile
    static constexpr int STEPS = KW / 4;            // score steps (4 keys each) per tile
    static constexpr int VPL = ROW / 128;           // 16-byte vectors per lane (score phase)
    static constexpr int EPV = 16 / ELEM;           // elements per 16-byte vector
    static constexpr int DPL = D / 8;               // dims per lane (score phase)
    static constexpr int PVD = D / 32;              // dims per lane (P.V phase)
    static constexpr int REP = 3 - Log2<G>::value;  // lanes per (key, head) = 2^REP
    static constexpr int STAGE = 2 * TK * ROW;      // K tile + V tile
    static constexpr int SMEM = kStages * STAGE;
    static_assert(KW % 4 == 0 && KW >= 4, "a warp needs whole score steps");
    static_assert(VPL * EPV == DPL, "score-phase slice");
    static_assert(kWarps * G * D * 4 <= SMEM, "merge buffer must fit in the stages");
};

// ------------------------------------------------------------ kernel ----

template <int ELEM, int D, int G>
__global__ void __launch_bounds__(kThreads) decode_kernel(const DecodeArgs a)
{
    using C = Cfg<ELEM, D, G>;
    extern __shared__ __align__(128) unsigned char dsmem[];
    __shared__ __align__(8) uint64_t full_bar[kStages];
    __shared__ __align__(16) float q_s[G * D];
    __shared__ __align__(16) float p_s[kWarps][C::KW][G];
    __shared__ __align__(16) float alpha_s[kWarps][G];
    __shared__ float2 ml_s[kWarps][G];
    __shared__ int last_s;

    const int chunk = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int t = __ldg(a.pos + b);
    if (t < 0) {
        if (chunk == 0 && kvh == 0 && tid == 0) atomicCAS(&g_status, kDevOk, kDevBadPosition);
        return;
    }
    const int B = a.B, h = B >> 1;
    const int blk = t / B;
    const int r = t - blk * B;
    const bool bridge = (blk > 0) && (r < h);
    const int n = bridge ? h + r : r;  // ring keys of the support (positions a(t) .. t-1)
    const int base = bridge ? h : 0;   // slot of logical key 0
    const int nch = n > 0 ? (n + a.chunk - 1) / a.chunk : 1;
    if (chunk >= nch) return;
    const int i0 = chunk * a.chunk;
    const int i1 = min(i0 + a.chunk, n);
    const int ntiles = i1 > i0 ? (i1 - i0 + C::TK - 1) / C::TK : 0;

    const size_t head = static_cast<size_t>(b) * a.Hkv + kvh;
    const unsigned char* kring = static_cast<const unsigned char*>(a.k_ring) + head * B * C::ROW;
    const unsigned char* vring = static_cast<const unsigned char*>(a.v_ring) + head * B * C::ROW;

    if (tid == 0) {
#pragma unroll
        for (int s = 0; s < kStages; ++s) mbar_init(&full_bar[s], 1);
        fence_mbar_init();
    }
    // Scaled queries of the group, fp32: q_s[j][c] = q[b][kvh*G + j][c] * log2(e)/sqrt(d).
    {
        const float scale = 1.4426950408889634f * rsqrtf(static_cast<float>(D));
        const unsigned char* qg = static_cast<const unsigned char*>(a.q) +
                                  (static_cast<size_t>(b) * a.Hq + static_cast<size_t>(kvh) * G) * C::ROW;
        for (int e = tid; e < G * D; e += kThreads) q_s[e] = Elem<ELEM>::to_float(qg + e * ELEM) * scale;
    }
    __syncthreads();

    auto issue = [&](int it) {
        const int s = it % kStages;
        const int k0 = i0 + it * C::TK;
        const int nk = min(C::TK, i1 - k0);
        int slot = base + k0;
        if (slot >= B) slot -= B;
        const int len1 = min(nk, B - slot);
        unsigned char* sK = dsmem + s * C::STAGE;
        unsigned char* sV = sK + C::TK * C::ROW;
        mbar_expect_tx(&full_bar[s], static_cast<uint32_t>(2 * nk * C::ROW));
        bulk_g2s(sK, kring + static_cast<size_t>(slot) * C::ROW, len1 * C::ROW, &full_bar[s]);
        bulk_g2s(sV, vring + static_cast<size_t>(slot) * C::ROW, len1 * C::ROW, &full_bar[s]);
        if (len1 < nk) {  // wrapped past slot B-1: the rest starts at slot 0
            bulk_g2s(sK + len1 * C::ROW, kring, (nk - len1) * C::ROW, &full_bar[s]);
            bulk_g2s(sV + len1 * C::ROW, vring, (nk - len1) * C::ROW, &full_bar[s]);
        }
    };
    if (tid == 0) {
        const int pro = min(kStages, ntiles);
        for (int it = 0; it < pro; ++it) issue(it);
    }

    // Queries of this lane's score-phase slice: vector m covers dims (sub + 8m)*EPV ...
    const int sub = lane & 7, kq = lane >> 3;
    float qr[G][C::DPL];
#pragma unroll
    for (int j = 0; j < G; ++j)
#pragma unroll
        for (int m = 0; m < C::VPL; ++m)
#pragma unroll
            for (int x = 0; x < C::EPV; ++x)
                qr[j][m * C::EPV + x] = q_s[j * D + (sub + 8 * m) * C::EPV + x];

    const int myhead = sub >> C::REP;
    const bool primary = (sub & ((1 << C::REP) - 1)) == 0;
    float m_run = -INFINITY;  // running max of this lane's head (log2 domain)
    float l_run = 0.f;        // this lane's share of the running sum (primary lanes only)
    float o[G][C::PVD];
#pragma unroll
    for (int j = 0; j < G; ++j)
#pragma unroll
        for (int x = 0; x < C::PVD; ++x) o[j][x] = 0.f;

    if (chunk == 0) {
        // Append: slot r of both rings <- the new token's rows (bit copy).
        const uint4* kn = reinterpret_cast<const uint4*>(static_cast<const unsigned char*>(a.k_new) + head * C::ROW);
        const uint4* vn = reinterpret_cast<const uint4*>(static_cast<const unsigned char*>(a.v_new) + head * C::ROW);
        uint4* kd = reinterpret_cast<uint4*>(static_cast<unsigned char*>(a.k_ring) + (head * B + r) * C::ROW);
        uint4* vd = reinterpret_cast<uint4*>(static_cast<unsigned char*>(a.v_ring) + (head * B + r) * C::ROW);
        for (int x = tid; x < C::ROW / 16; x += kThreads) {
            kd[x] = __ldg(kn + x);
            vd[x] = __ldg(vn + x);
        }
        if (warp == 0) {  // the current token seeds warp 0's softmax state
            float kc[C::PVD], vc[C::PVD];
            const unsigned char* knb = static_cast<const unsigned char*>(a.k_new) + head * C::ROW;
            const unsigned char* vnb = static_cast<const unsigned char*>(a.v_new) + head * C::ROW;
            load_elems<ELEM, C::PVD>(knb + lane * C::PVD * ELEM, kc);
            load_elems<ELEM, C::PVD>(vnb + lane * C::PVD * ELEM, vc);
            float zc[G];
#pragma unroll
            for (int j = 0; j < G; ++j) {
                float acc = 0.f;
#pragma unroll
                for (int x = 0; x < C::PVD; ++x) acc = fmaf(q_s[j * D + lane * C::PVD + x], kc[x], acc);
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
                for (int x = 0; x < C::PVD; ++x) o[j][x] = vc[x];
        }
    }

    int it = 0;
    bool failed = false;
    for (; it < ntiles; ++it) {
        const int s = it % kStages;
        const bool ok = mbar_wait(&full_bar[s], static_cast<uint32_t>((it / kStages) & 1), a.timeout_ns);
        const int k0 = i0 + it * C::TK;
        const int nk = min(C::TK, i1 - k0);
        const int nkw = ok ? min(max(nk - warp * C::KW, 0), C::KW) : 0;
        if (nkw > 0) {
            const unsigned char* sK = dsmem + s * C::STAGE + warp * C::KW * C::ROW;
            const unsigned char* sV = dsmem + s * C::STAGE + C::TK * C::ROW + warp * C::KW * C::ROW;
            float zs[C::STEPS];
            float mx = -INFINITY;
#pragma unroll
            for (int st = 0; st < C::STEPS; ++st) {
                const int key = st * 4 + kq;
                float z = -INFINITY;
                if (st * 4 < nkw) {  // warp-uniform
                    float acc[G];
#pragma unroll
                    for (int j = 0; j < G; ++j) acc[j] = 0.f;
#pragma unroll
                    for (int m = 0; m < C::VPL; ++m) {
                        float kf[C::EPV];
                        const uint4 u = *reinterpret_cast<const uint4*>(sK + key * C::ROW + (sub + 8 * m) * 16);
                        Elem<ELEM>::vec16(u, kf);
#pragma unroll
                        for (int j = 0; j < G; ++j)
#pragma unroll
                            for (int x = 0; x < C::EPV; ++x)
                                acc[j] = fmaf(qr[j][m * C::EPV + x], kf[x], acc[j]);
                    }
                    const float zz = reduce_scatter8<G>(acc, sub);
                    z = key < nkw ? zz : -INFINITY;
                }
                zs[st] = z;
                mx = fmaxf(mx, z);
            }
            mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 8));
            mx = fmaxf(mx, __shfl_xor_sync(kFull, mx, 16));
            const float m_new = fmaxf(m_run, mx);
            const float alpha = exp2f(m_run - m_new);
            float lsum = 0.f;
#pragma unroll
            for (int st = 0; st < C::STEPS; ++st) {
                const float pz = exp2f(zs[st] - m_new);
                if (st * 4 < nkw && primary) p_s[warp][st * 4 + kq][myhead] = pz;
                lsum += pz;
            }
            l_run = l_run * alpha + (primary ? lsum : 0.f);
            m_run = m_new;
            if (primary && kq == 0) alpha_s[warp][myhead] = alpha;
            __syncwarp();
#pragma unroll
            for (int j = 0; j < G; ++j) {
                const float al = alpha_s[warp][j];
#pragma unroll
                for (int x = 0; x < C::PVD; ++x) o[j][x] *= al;
            }
#pragma unroll 4
            for (int k = 0; k < nkw; ++k) {
                float pv[G];
#pragma unroll
                for (int j = 0; j < G; ++j) pv[j] = p_s[warp][k][j];
                float vf[C::PVD];
                load_elems<ELEM, C::PVD>(sV + k * C::ROW + lane * C::PVD * ELEM, vf);
#pragma unroll
                for (int j = 0; j < G; ++j)
#pragma unroll
                    for (int x = 0; x < C::PVD; ++x) o[j][x] = fmaf(pv[j], vf[x], o[j][x]);
            }
        }
        failed = __syncthreads_or(!ok) != 0;
        if (failed) break;
        if (tid == 0 && it + kStages < ntiles) {
            fence_proxy_async();
            issue(it + kStages);
        }
    }
    if (failed) {
        if (tid == 0) {
            atomicCAS(&g_status, kDevOk, kDevTimeout);
            const int issued = min(ntiles, it + kStages);
            for (int j = it; j < issued; ++j)
                mbar_wait(&full_bar[j % kStages], static_cast<uint32_t>((j / kStages) & 1), 1000000000ull);
        }
        __syncthreads();
        return;
    }

    // ---- merge the warps' states (all copies have landed: the stages are free)
    {
        float l = l_run;
        l += __shfl_xor_sync(kFull, l, 8);
        l += __shfl_xor_sync(kFull, l, 16);
#pragma unroll
        for (int x = 1; x < (1 << C::REP); x <<= 1) l += __shfl_xor_sync(kFull, l, x);
        if (lane == (myhead << C::REP)) ml_s[warp][myhead] = make_float2(m_run, l);
    }
    float* o_s = reinterpret_cast<float*>(dsmem);  // [kWarps][G][D]
#pragma unroll
    for (int j = 0; j < G; ++j)
#pragma unroll
        for (int x = 0; x < C::PVD; ++x) o_s[(warp * G + j) * D + lane * C::PVD + x] = o[j][x];
    __syncthreads();

    const size_t part = head * a.nchunk + chunk;
    for (int e = tid; e < G * D; e += kThreads) {
        const int j = e / D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) M = fmaxf(M, ml_s[w][j].x);
        float L = 0.f, O = 0.f;
#pragma unroll
        for (int w = 0; w < kWarps; ++w) {
            const float sc = exp2f(ml_s[w][j].x - M);
            L = fmaf(ml_s[w][j].y, sc, L);
            O = fmaf(o_s[(w * G) * D + e], sc, O);
        }
        if (nch == 1) {
            a.out[(static_cast<size_t>(b) * a.Hq + static_cast<size_t>(kvh) * G) * D + e] = O / L;
        } else {
            a.part_o[part * G * D + e] = O;
            if ((e % D) == 0) reinterpret_cast<float2*>(a.part_ml)[part * G + j] = make_float2(M, L);
        }
    }
    if (nch == 1) return;

    // ---- split combine (Eq. lse): the last CTA of this (sequence, KV head) fuses all partials
    __threadfence();
    __syncthreads();
    if (tid == 0) last_s = (atomicAdd(a.counters + head, 1) == nch - 1);
    __syncthreads();
    if (!last_s) return;
    __threadfence();
    const float* po = a.part_o + head * a.nchunk * G * D;
    const float2* pml = reinterpret_cast<const float2*>(a.part_ml) + head * a.nchunk * G;
    for (int e = tid; e < G * D; e += kThreads) {
        const int j = e / D;
        float M = -INFINITY;
        for (int c = 0; c < nch; ++c) M = fmaxf(M, __ldcg(&pml[c * G + j]).x);
        float L = 0.f, O = 0.f;
        for (int c = 0; c < nch; ++c) {
            const float2 ml = __ldcg(&pml[c * G + j]);
            const float sc = exp2f(ml.x - M);
            L = fmaf(ml.y, sc, L);
            O = fmaf(__ldcg(po + c * G * D + e), sc, O);
        }
        a.out[(static_cast<size_t>(b) * a.Hq + static_cast<size_t>(kvh) * G) * D + e] = O / L;
    }
    if (tid == 0) a.counters[head] = 0;
}

// --------------------------------------------------- prefill / advance ----

// Ring of a sequence resuming at t = pos[b]: row j of the history (position
// t - B + j) goes to slot (t - B + j) mod B; negative positions write zeros.
__global__ void prefill_kernel(const uint4* __restrict__ k_hist, const uint4* __restrict__ v_hist,
                               const int32_t* __restrict__ pos, uint4* __restrict__ k_ring,
                               uint4* __restrict__ v_ring, int Hkv, int B, int row16,
                               long long total)
{
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
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < batch; i += gridDim.x * blockDim.x) pos[i] += 1;
}

// Opt the kernel in to its dynamic shared memory (above the 48 KiB default), once per device.
template <int ELEM, int D, int G>
cudaError_t ensure_smem_attr()
{
    static bool attr_set[64] = {};
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 64 && attr_set[dev]) return cudaSuccess;
    err = cudaFuncSetAttribute(decode_kernel<ELEM, D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               Cfg<ELEM, D, G>::SMEM);
    if (err == cudaSuccess && dev < 64) attr_set[dev] = true;
    return err;
}

template <int ELEM, int D, int G>
cudaError_t launch_t(const DecodeArgs& a, cudaStream_t stream)
{
    using C = Cfg<ELEM, D, G>;
    cudaError_t err = ensure_smem_attr<ELEM, D, G>();
    if (err != cudaSuccess) return err;
    const dim3 grid(a.nchunk, a.Hkv, a.batch);
    decode_kernel<ELEM, D, G><<<grid, kThreads, C::SMEM, stream>>>(a);
    return cudaGetLastError();
}

template <int ELEM, int D>
cudaError_t launch_g(const DecodeArgs& a, cudaStream_t stream)
{
    switch (a.Hq / a.Hkv) {
        case 1: return launch_t<ELEM, D, 1>(a, stream);
        case 2: return launch_t<ELEM, D, 2>(a, stream);
        case 4: return launch_t<ELEM, D, 4>(a, stream);
        case 8: return launch_t<ELEM, D, 8>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

template <int ELEM, int D, int G>
int occupancy_t()
{
    static int cache[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (dev < 64 && cache[dev] > 0) return cache[dev];
    int n = 0;
    if (ensure_smem_attr<ELEM, D, G>() != cudaSuccess) return 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, decode_kernel<ELEM, D, G>, kThreads,
                                                      Cfg<ELEM, D, G>::SMEM) != cudaSuccess)
        return 0;
    if (dev < 64) cache[dev] = n;
    return n;
}

template <int ELEM, int D>
int occupancy_g(int group)
{
    switch (group) {
        case 1: return occupancy_t<ELEM, D, 1>();
        case 2: return occupancy_t<ELEM, D, 2>();
        case 4: return occupancy_t<ELEM, D, 4>();
        case 8: return occupancy_t<ELEM, D, 8>();
        default: return 0;
    }
}

}  // namespace

int tile_keys(int elem_bytes, int d) { return kTileBytes / (elem_bytes * d); }

int decode_ctas_per_sm(int elem_bytes, int d, int group)
{
    if (elem_bytes == 2 && d == 64) return occupancy_g<2, 64>(group);
    if (elem_bytes == 2 && d == 128) return occupancy_g<2, 128>(group);
    if (elem_bytes == 4 && d == 64) return occupancy_g<4, 64>(group);
    if (elem_bytes == 4 && d == 128) return occupancy_g<4, 128>(group);
    return 0;
}

cudaError_t launch_decode(const DecodeArgs& a, int elem_bytes, cudaStream_t stream)
{
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
    prefill_kernel<<<blocks, 256, 0, stream>>>(static_cast<const uint4*>(k_hist),
                                               static_cast<const uint4*>(v_hist), pos,
                                               static_cast<uint4*>(k_ring),
                                               static_cast<uint4*>(v_ring), Hkv, B, row16, total);
    return cudaGetLastError();
}

cudaError_t launch_advance(int32_t* pos, int batch, cudaStream_t stream)
{
    if (batch == 0) return cudaSuccess;
    const int blocks = (batch + 255) / 256 < 64 ? (batch + 255) / 256 : 64;
    advance_kernel<<<blocks, 256, 0, stream>>>(pos, batch);
    return cudaGetLastError();
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
