// Internal interface between the C-ABI layer (pbb_api.cu) and the kernels
// (pbb_decode.cu). Not installed; the public interface is include/pbb.h.
#pragma once

#include <cuda.h>
#include <cuda_runtime_api.h>
#include <stddef.h>
#include <stdint.h>

#include <atomic>

namespace pbb {

// Device status codes (the word read by pbb_get_device_status).
enum DeviceStatus : int { kDevOk = 0, kDevTimeout = 1, kDevBadPosition = 2 };

struct DecodeArgs {
    const void* q;       // [batch][Hq][d]
    const void* k_new;   // [batch][Hkv][d]
    const void* v_new;   // [batch][Hkv][d]
    void* k_ring;        // [batch][Hkv][B][d]
    void* v_ring;        // [batch][Hkv][B][d]
    const int32_t* pos;  // [batch]
    float* out;          // [batch][Hq][d]
    float* part_o;       // [batch*Hkv - whole][nchunk][G][d]   split partials (unnormalised output)
    float* part_ml;      // [batch*Hkv - whole][nchunk][G][2]   split partials (max, sum), log2 domain
    int* counters;       // [batch][Hkv]                 finished chunks per (sequence, KV head)
    int* ctl;            // [2] work-queue head and finished CTAs; zero between launches
    int batch, Hq, Hkv, d, B;
    int gq;              // query heads per KV head (Hq / Hkv); the kernel's group G is gq, or 8 for gq = 6
    int pos_batch;       // sequences with their own position: sequence b reads pos[b % pos_batch]
                         // (layers of a multi-layer step are consecutive batches sharing positions)
    int window;          // 0: the PBB support [a(t), t]; w in [1, B]: the sliding window {t-w+1, ..., t}
    int whole;           // supports [0, whole) are one work item each
    int chunk;           // ring keys per work item of the later supports (a multiple of the tile)
    int nchunk;          // work items per later support = ceil((B-1)/chunk)
    int total_items;     // whole + (batch * Hkv - whole) * nchunk
    const int* order;    // null, or (whole == batch * Hkv, tensor-core kernel) the sequences in the order
                         // their supports are taken: longest first (launch_support_order)
    unsigned long long timeout_ns;
};

// Keys per shared-memory tile of a kernel instance (rows of K and of V).
int tile_keys(int elem_bytes, int d, int group);

// GQA groups the tensor-core decode kernel serves: its score tile has 8 query columns, and a
// group of 4 or 6 fills the rest with zero query rows (PBB_TC_MIN_GROUP = 8 keeps those groups
// on the CUDA-core kernel).
#ifndef PBB_TC_MIN_GROUP
#define PBB_TC_MIN_GROUP 4
#endif
inline bool tc_group(int group)
{
    return group == 8 || (group >= PBB_TC_MIN_GROUP && (group == 4 || group == 6));
}

// The kernel choice of pbb_set_kernel (PBB_KERNEL_AUTO, _CUDA_CORES or _TENSOR_CORES); returns
// the previous one.
int set_kernel_choice(int kernel);

// Whether a decode step of this shape runs the tensor-core kernel (given chunks of whole
// tiles, which plan_split makes for it).
bool tensor_core_shape(int batch, int Hkv, int d, int B, int elem_bytes, int group, int window);

// Resident CTAs per SM of the decode kernel a step of this shape runs (0 if unsupported).
int decode_ctas_per_sm(int batch, int Hkv, int elem_bytes, int d, int group, int B, int window);

// The split plan of a step (see plan_split in pbb_api.cu): supports [0, whole)
// run whole, every later one in nchunk chunks of `chunk` ring keys. window as
// in DecodeArgs (0 = PBB).
struct SplitPlan {
    int whole, chunk, nchunk;
};
SplitPlan plan_split(int batch, int Hkv, int d, int B, int elem_bytes, int group, int window);

// Whether launch_decode would run the tensor-core kernel for these arguments.
bool use_tensor_cores(const DecodeArgs& a, int elem_bytes);

// Launch the fused append + attention + combine kernel (persistent grid of at
// most SMs x resident CTAs). elem_bytes: 2 (bf16) or 4 (fp32).
cudaError_t launch_decode(const DecodeArgs& a, int elem_bytes, cudaStream_t stream);
// Writes the step's sequences into order[0, batch) by descending number of ring keys in their
// supports (one block; a counting sort on 256 length classes, the order within a class
// unspecified), for DecodeArgs::order.
cudaError_t launch_support_order(const DecodeArgs& a, int* order, cudaStream_t stream);

cudaError_t launch_prefill(const void* k_hist, const void* v_hist, const int32_t* pos, void* k_ring,
                           void* v_ring, int batch, int Hkv, int B, int row_bytes,
                           cudaStream_t stream);

cudaError_t launch_advance(int32_t* pos, int batch, cudaStream_t stream);

// Read (and clear) the device status word of the current device.
cudaError_t read_and_clear_status(int* status, cudaStream_t stream);

// 2-D bf16 tensor map over `rows` rows of d elements read in boxes of 64
// columns x box_rows rows with the 128-byte swizzle (cached; false if the
// driver's encoder is unavailable or refuses).
bool rows_tensor_map(CUtensorMap* map, const void* base, unsigned long long rows, int d, int box_rows);

// Whole-sequence forward (pbb_forward.cu).
struct ForwardArgs {
    const void* q;   // [batch][Hq][n][d] bf16
    const void* k;   // [batch][Hkv][n][d] bf16
    const void* v;   // [batch][Hkv][n][d] bf16
    void* out;       // [batch][Hq][n][d] bf16 or fp32 (out_f32)
    float* lse;      // [batch][Hq][n] or null
    int batch, Hq, Hkv, n, d, B;
    int out_f32;
    unsigned long long timeout_ns;
};
cudaError_t launch_forward(const ForwardArgs& a, cudaStream_t stream);
// The shape launch_forward runs for these arguments (nothing is launched): keys per K/V tile,
// persistent CTAs per SM and the grid.
struct ForwardPlan {
    int keys_per_tile, ctas_per_sm, grid;
};
cudaError_t plan_forward(const ForwardArgs& a, ForwardPlan* plan);
cudaError_t launch_seq_ring(const void* k, const void* v, void* k_ring, void* v_ring, int batch, int Hkv,
                            int n, int B, int row_bytes, cudaStream_t stream);
// Status word of the forward kernels (read and cleared; the caller synchronises first).
cudaError_t read_and_clear_forward_status(int* status);

// Whole-sequence backward (pbb_backward.cu).
struct BackwardArgs {
    const void* q;      // [batch][Hq][n][d] bf16
    const void* k;      // [batch][Hkv][n][d] bf16
    const void* v;      // [batch][Hkv][n][d] bf16
    const void* out;    // [batch][Hq][n][d] bf16, the forward's output
    const void* dout;   // [batch][Hq][n][d] bf16, upstream gradient
    const float* lse;   // [batch][Hq][n], the forward's log-partition
    float* delta;       // [batch][Hq][n] scratch: dO . O per row
    float* dq;          // [batch][Hq][n][d]
    float* dk;          // [batch][Hkv][n][d]
    float* dv;          // [batch][Hkv][n][d]
    int batch, Hq, Hkv, n, d, B;
    unsigned long long timeout_ns;
};
cudaError_t launch_backward(const BackwardArgs& a, cudaStream_t stream);
cudaError_t read_and_clear_backward_status(int* status);

// Per-device values worked out once: a kernel's shared-memory opt-in with its resident CTAs, the
// SM count. Slot `dev` of `cache` holds 0 until a call on that device stores the positive result
// of `make`; a result of 0 or less (a failed query) is returned without being stored. Host
// threads calling at once may each run `make`, which only issues idempotent queries and
// settings; the release store publishes those with the value. Devices at or past
// kMaxCachedDevices run `make` on every call.
constexpr int kMaxCachedDevices = 64;

template <typename F>
int cached_per_device(std::atomic<int>* cache, int dev, F make)
{
    const bool slot = dev >= 0 && dev < kMaxCachedDevices;
    if (slot) {
        const int v = cache[dev].load(std::memory_order_acquire);
        if (v > 0) return v;
    }
    const int v = make();
    if (slot && v > 0) cache[dev].store(v, std::memory_order_release);
    return v;
}

// Resident CTAs per SM of `kernel` from the resources the SM checks (registers, shared memory,
// threads), at most `want`. The runtime's occupancy calculator answers 1 for the tcgen05
// kernels even where two fit (and two did run together on GB300); the callers keep TMEM
// shared by construction (columns per CTA x want <= 512).
template <typename K>
int resident_ctas(K kernel, int threads, int dyn_smem, int want, int dev)
{
    cudaFuncAttributes fa{};
    int smem_sm = 0, regs_sm = 0, reserved = 0, threads_sm = 0;
    if (cudaFuncGetAttributes(&fa, kernel) != cudaSuccess ||
        cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&threads_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev) != cudaSuccess)
        return 1;
    const int warps = (threads + 31) / 32;
    const int regs_warp = (fa.numRegs * 32 + 255) / 256 * 256;  // allocated per warp in 256-register units
    const long long smem_cta = static_cast<long long>(dyn_smem) + fa.sharedSizeBytes + reserved;
    long long n = want;
    if (smem_sm / smem_cta < n) n = smem_sm / smem_cta;
    if (regs_warp > 0 && regs_sm / (regs_warp * warps) < n) n = regs_sm / (regs_warp * warps);
    if (threads_sm / threads < n) n = threads_sm / threads;
    return n < 1 ? 1 : static_cast<int>(n);
}

}  // namespace pbb
