/*
 * libpbb: fused decode step of Post-Boundary Bridge (PBB) local attention on
 * one GPU (sm_103a), with the sliding-window control and the whole-sequence
 * forward (prefill) over the same support.
 *
 * The operation (Sec. 3, Eq. (pbb) and Eq. (attention); Appendix F.1):
 * a sequence whose current token sits at absolute position t, with block size
 * B = 2h, block start p = B*floor(t/B) and phase r = t - p, reads the support
 *
 *     A(t) = {p, ..., t}  U  {p-h, ..., p-1} if p > 0 and r < h,
 *
 * which is the interval [a(t), t], a(t) = max(0, h(floor(t/h) - 1))
 * (Eq. pbb_relay). Each query head j of the sequence returns
 *
 *     o_j = sum_{s in A(t)} exp(z_s) v_s / sum_{s in A(t)} exp(z_s),
 *     z_s = q_j . k_s / sqrt(d),
 *
 * where K/V come from KV head j / (Hq/Hkv) (contiguous GQA grouping). K/V of
 * every KV head live in a fixed ring of B slots: position s is stored in slot
 * s mod B and no retained entry is ever moved (Appendix F.1, Proposition
 * "Relocation-free PBB cache"). One decode step writes the new token's K/V
 * into slot r and attends over the ring; the slot written is never one read.
 *
 * Conventions shared by every call below.
 *   - Layouts are dense, row-major, in this order:
 *       q      [batch][Hq][d]        query of the current token (already rotated)
 *       k_new  [batch][Hkv][d]       K of the current token
 *       v_new  [batch][Hkv][d]       V of the current token
 *       ring   [batch][Hkv][B][d]    one K ring and one V ring
 *       pos    [batch] int32         absolute position t of the current token
 *       out    [batch][Hq][d] fp32   attention output
 *     Element type: bf16 for pbb_decode_step, fp32 for pbb_decode_step_f32;
 *     the output is fp32 in both.
 *   - Every tensor pointer is a DEVICE pointer, owned by the caller, 16-byte
 *     aligned (pos: 4-byte aligned). Rings are either caller memory with the
 *     layout above or come from pbb_ring_alloc.
 *   - Calls are asynchronous on `stream` (0 = the legacy default stream) and
 *     never synchronise. Sizes: batch >= 0, Hq % Hkv == 0 with
 *     Hq/Hkv in {1, 2, 4, 6, 8}, d in {64, 128}, B even and 2 <= B <= 2^20.
 *     A group of 6 (12 query heads on 2 KV heads, the paper's models of Sec. 5)
 *     runs as a group of 8 (on either kernel) with two zero query rows that are
 *     computed and never written.
 *   - Return value: PBB_OK or a negative PBB_ERR_* code; nothing is launched
 *     when argument checking fails. Faults the device finds (a negative
 *     position, a wait that ran out) are kept in a device-side status word
 *     read by pbb_get_device_status.
 */
#ifndef PBB_H_
#define PBB_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { PBB_BF16 = 0, PBB_F32 = 1 } pbb_dtype;

enum {
    PBB_OK = 0,
    PBB_ERR_INVALID_ARG = -1,    /* null or misaligned pointer, negative size, window outside [1, B] */
    PBB_ERR_UNSUPPORTED = -2,    /* B odd/out of range, Hq % Hkv != 0, group or d not supported */
    PBB_ERR_CUDA = -3,           /* a CUDA runtime call or a launch failed */
    PBB_ERR_DEVICE_TIMEOUT = -4, /* a kernel's bounded wait on a bulk copy ran out */
    PBB_ERR_WORKSPACE = -5,      /* workspace too small while the stream is being captured */
    PBB_ERR_DEVICE_POSITION = -6, /* a kernel saw pos[b] < 0; that sequence was skipped */
    PBB_ERR_SCRATCH_LIMIT = -7    /* pbb_decode_step_noalloc: the step needs more scratch than
                                     PBB_NOALLOC_SCRATCH_BYTES */
};

/*
 * Bytes of ONE ring (K or V): batch * Hkv * B * d * element size. The pair is
 * twice this: 2 * batch * B * Hkv * d * u, Appendix F.1 (65,536 bytes at
 * batch 1, B 128, Hkv 2, d 64, bf16). Returns 0 for invalid sizes. Host only.
 */
size_t pbb_ring_bytes(int batch, int Hkv, int d, int B, pbb_dtype dtype);

/*
 * Allocate a zero-filled K ring and V ring (cudaMallocAsync on `stream`,
 * zeroed on the same stream). The caller owns both and frees them with
 * pbb_ring_free. On error nothing stays allocated and *k_ring, *v_ring are
 * set to NULL.
 */
int pbb_ring_alloc(void** k_ring, void** v_ring, int batch, int Hkv, int d, int B,
                   pbb_dtype dtype, cudaStream_t stream);

/* Free rings from pbb_ring_alloc (cudaFreeAsync on `stream`). NULL is ignored. */
int pbb_ring_free(void* k_ring, void* v_ring, cudaStream_t stream);

/*
 * Load the ring of a sequence that resumes at position t = pos[b] from its
 * history (Appendix F.1: position s goes to slot s mod B).
 *   k_hist, v_hist [batch][Hkv][B][d]: row j holds position t - B + j.
 * Every slot is written: rows whose position is negative (before the start of
 * the sequence) write zeros. The result is the ring that t sequential decode
 * steps from a zeroed ring would have left, so the next pbb_decode_step at
 * position t continues it exactly. Sequences with pos[b] < 0 are skipped and
 * flagged (PBB_ERR_DEVICE_POSITION). Bit copy; same element type as the ring.
 */
int pbb_ring_prefill(const void* k_hist, const void* v_hist, const int32_t* pos, void* k_ring,
                     void* v_ring, int batch, int Hkv, int d, int B, pbb_dtype dtype,
                     cudaStream_t stream);

/*
 * Make sure the library's workspace of (current device, `stream`) holds the
 * split partials of a step of this shape (and of every smaller batch). A
 * workspace (owned by the library, freed at exit) holds the work-queue words,
 * one counter per (sequence, KV head), the order of the sequences for a
 * longest-first step (pbb_plan_support_order) and the per-split partial (max,
 * sum, output) of Eq. (lse). Every decode step (pbb_decode_step, _f32, _layers and
 * pbb_swa_decode_step) uses the workspace of the stream it is issued on and
 * grows it on demand, which allocates and waits for the device; so call this
 * first, on the capture stream, when decode steps are to be captured in a
 * CUDA graph.
 *   - Steps on different streams use different workspaces and may overlap on
 *     the GPU. Steps on one stream run in order. A captured graph keeps the
 *     workspace of the stream it was captured on: do not replay it while steps
 *     (or replays of other graphs captured on that stream) run on other
 *     streams, and do not let that stream's workspace grow after the capture
 *     (growth frees the buffers the graph holds).
 *   - Issuing calls from several host threads is safe: the library serialises
 *     its own bookkeeping, and a growth waits for the steps already launched
 *     before it frees the old buffers.
 */
int pbb_reserve_workspace(int max_batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype, cudaStream_t stream);

/*
 * One PBB decode step for every sequence (bf16 q/k/v/ring, fp32 out).
 * For each sequence b with t = pos[b]: writes k_new/v_new[b] into slot
 * t mod B of its rings (bit copy), then computes out[b] as defined above over
 * A(t), the new token included (read from k_new/v_new, not back from the
 * ring). Precondition (Appendix F.1, sequential single-token decoding): the
 * rings hold positions t-B .. t-1 of the sequence in their slots, which holds
 * after pbb_ring_prefill at t, or after steps at t-1, t-2, ... starting from a
 * zeroed ring at t = 0. pos is read on the device and never by the host.
 * Deterministic: the same inputs give bitwise the same out and rings.
 * A step with many whole supports first launches a small kernel that sorts its
 * sequences by support length (pbb_plan_support_order); it changes no result.
 */
int pbb_decode_step(const void* q, const void* k_new, const void* v_new, void* k_ring,
                    void* v_ring, const int32_t* pos, float* out, int batch, int Hq, int Hkv,
                    int d, int B, cudaStream_t stream);

/* Same as pbb_decode_step with fp32 q, k_new, v_new and rings. */
int pbb_decode_step_f32(const float* q, const float* k_new, const float* v_new, float* k_ring,
                        float* v_ring, const int32_t* pos, float* out, int batch, int Hq,
                        int Hkv, int d, int B, cudaStream_t stream);

/*
 * One decode step of `layers` PBB local-attention layers in a single launch
 * (the paper's hybrid runs 15 local layers per token; one launch amortises the
 * launch latency that dominates small batches). Every tensor gains a leading
 * layer index, [layers][batch]...: q [layers][batch][Hq][d], k_new/v_new
 * [layers][batch][Hkv][d], rings [layers][batch][Hkv][B][d], out
 * [layers][batch][Hq][d]; pos [batch] is shared by all layers (they decode the
 * same token). Layer l of sequence b computes exactly what pbb_decode_step would
 * for that layer's tensors; the work of all layers forms one persistent grid.
 * layers * batch <= 65535; other rules as pbb_decode_step (bf16) and
 * pbb_decode_step_f32 (PBB_F32). The caller synchronises layer inputs: use this
 * where every layer's q/k/v of the token are known before the step (batched
 * evaluation of layers, or benchmarking), and per-layer calls inside a captured
 * graph otherwise.
 */
int pbb_decode_step_layers(const void* q, const void* k_new, const void* v_new, void* k_ring, void* v_ring,
                           const int32_t* pos, float* out, int layers, int batch, int Hq, int Hkv, int d, int B,
                           pbb_dtype dtype, cudaStream_t stream);

/*
 * Sliding-window attention decode step over the same rings: the control the
 * paper compares PBB with (Sec. 2.3; Sec. 3 notes that SWA with w = B can also
 * live in a B-slot ring). Identical to pbb_decode_step / pbb_decode_step_f32
 * (element type `dtype`) except for the support, which is the window
 *
 *     A_SWA(t) = {max(0, t-w+1), ..., t},   w = window, 1 <= w <= B,
 *
 * the current token included. Same ring contents and precondition: the step
 * writes k_new/v_new into slot t mod B, which holds position t-B, outside the
 * window. A ring can be switched between the two kinds of step at any
 * position. Runs on the same kernels as the PBB step (the tensor-core kernel
 * for bf16 with Hq/Hkv in {4, 6, 8} and B a multiple of 64, under the same
 * rules; its tiles start at slot multiples of 32 and mask the slots outside
 * the window's run). Returns
 * PBB_ERR_INVALID_ARG for a window outside [1, B]. pbb_reserve_workspace
 * covers window steps with window = B; for a smaller window make one step on
 * the capture stream outside any stream capture first.
 */
int pbb_swa_decode_step(const void* q, const void* k_new, const void* v_new, void* k_ring,
                        void* v_ring, const int32_t* pos, float* out, int batch, int Hq, int Hkv,
                        int d, int B, int window, pbb_dtype dtype, cudaStream_t stream);

/*
 * PBB attention over whole sequences: the forward pass of the paper's fused
 * training kernel and the prefill before decoding (Sec. 3, Eq. (attention) over
 * A(t) for every position t; Appendix "exact union and numerical checks": block
 * tiles and bridge rectangles under one softmax, native GQA, no dense mask).
 * Every position t in [0, n) of a sequence attends to [a(t), t] of the same
 * sequence, a(t) = max(0, h(floor(t/h) - 1)); positions start at 0.
 *   q    [batch][Hq][n][d]   bf16, row t = query of position t (already rotated)
 *   k, v [batch][Hkv][n][d]  bf16, row s = key / value of position s
 *   out  [batch][Hq][n][d]   out_dtype (PBB_BF16 or PBB_F32)
 *   lse  [batch][Hq][n]      fp32 ln sum_{s in A(t)} exp(q_t.k_s/sqrt(d)), the
 *                            log-partition of Eq. (lse) a backward pass reuses;
 *                            NULL to skip
 * Device pointers owned by the caller; q, k, v, out 16-byte aligned. Same
 * head-size rules as the decode step; Hq/Hkv in {1, 2, 4, 8} (a tile stacks
 * Hq/Hkv heads x 128/(Hq/Hkv) positions as 128 rows, so 6 returns
 * PBB_ERR_UNSUPPORTED); batch*Hq*n < 2^31. Runs on the
 * fifth-generation tensor cores (tcgen05, bf16 operands, fp32 accumulation in
 * tensor memory; the softmax weights are rounded to bf16 before P.V), one
 * persistent CTA per SM. Asynchronous on `stream`; a bounded wait that runs out
 * is reported by pbb_get_device_status as PBB_ERR_DEVICE_TIMEOUT.
 */
int pbb_forward(const void* q, const void* k, const void* v, void* out, float* lse, int batch, int Hq,
                int Hkv, int n, int d, int B, pbb_dtype out_dtype, cudaStream_t stream);

/*
 * The launch shape pbb_forward would use for these sizes on the current device
 * (nothing is launched): *keys_per_tile, the keys of one K/V tile (128 for
 * B >= 512; 32 at d = 64 and 64 at d = 128 below), and *ctas_per_sm, the
 * persistent CTAs sharing an SM's tensor memory (0 when there is no work).
 * Same shape rules as pbb_forward; PBB_ERR_INVALID_ARG for null outputs.
 */
int pbb_plan_forward(int batch, int Hq, int Hkv, int n, int d, int B, int* keys_per_tile, int* ctas_per_sm);

/*
 * The query tiles (128 rows of the GQA group's heads) one persistent CTA of
 * pbb_forward works on at once for these sizes on the current device: 2 where
 * long supports with B a multiple of 256 take the paired-item kernel (two
 * consecutive query tiles of one sequence and KV head stream their union of keys
 * once, their softmaxes alternating on the tensor pipe), else 1. Negative on
 * error, with pbb_plan_forward's shape rules. Nothing is launched.
 */
int pbb_plan_forward_query_tiles(int batch, int Hq, int Hkv, int n, int d, int B);

/*
 * Gradients of pbb_forward (the backward pass of the paper's fused training
 * kernel, Sec. 3: bridge gradients flow into the previous half-block's K and V).
 * With P_ts = exp(q_t.k_s/sqrt(d) - lse_t) on A(t) and D_t = dO_t . o_t:
 *   dq_t = sum_s P_ts (dO_t.v_s - D_t) k_s / sqrt(d)
 *   dk_s = sum over t (and the group's query heads) of P_ts (dO_t.v_s - D_t) q_t / sqrt(d)
 *   dv_s = sum over t (and the group's query heads) of P_ts dO_t
 *   q, out, dout [batch][Hq][n][d] bf16   out and lse from pbb_forward of q, k, v
 *   k, v        [batch][Hkv][n][d] bf16   lse [batch][Hq][n] fp32
 *   delta       [batch][Hq][n] fp32      scratch (receives D)
 *   dq          [batch][Hq][n][d] fp32   dk, dv [batch][Hkv][n][d] fp32 (overwritten)
 * Same shape rules as pbb_forward; 16-byte aligned tensors (lse, delta 4-byte).
 * Runs on the fifth-generation tensor cores (tcgen05: S, dP and the gradients
 * accumulate in fp32 in tensor memory; bf16 operands, with P and dS rounded to
 * bf16): one pass over key tiles for dK and dV, one over query tiles for dQ,
 * each persistent with one CTA per SM. No floating-point atomics, so results
 * are bitwise deterministic. Asynchronous on `stream`; a bounded wait that runs out is
 * reported by pbb_get_device_status as PBB_ERR_DEVICE_TIMEOUT.
 */
int pbb_backward(const void* q, const void* k, const void* v, const void* out, const void* dout, const float* lse,
                 float* delta, float* dq, float* dk, float* dv, int batch, int Hq, int Hkv, int n, int d, int B,
                 cudaStream_t stream);

/*
 * Load the decode rings of sequences whose first n positions went through
 * pbb_forward (the cache-populating prefill, Appendix F.1): slot j of each ring
 * receives the position s in [n-B, n-1] with s = j (mod B), zeros where s < 0.
 * k, v [batch][Hkv][n][d] as for pbb_forward (may be NULL when n = 0). The next
 * decode step is at position n. Bit copy; element type `dtype`.
 */
int pbb_ring_from_sequence(const void* k, const void* v, int n, void* k_ring, void* v_ring, int batch,
                           int Hkv, int d, int B, pbb_dtype dtype, cudaStream_t stream);

/* pos[b] += 1 for every sequence, on the device (advances a decode loop, e.g. in a graph). */
int pbb_advance_positions(int32_t* pos, int batch, cudaStream_t stream);

/*
 * Synchronise `stream`, then return and clear the device status words (decode
 * and forward kernels) of the current device: PBB_OK, PBB_ERR_DEVICE_TIMEOUT or
 * PBB_ERR_DEVICE_POSITION (first fault recorded since the last call). Clearing also resets the split
 * counters in the workspace, which an aborted step can leave behind.
 */
int pbb_get_device_status(cudaStream_t stream);

/*
 * Limit, in nanoseconds, of every wait of a decode kernel on a bulk copy
 * (default 1e9). A wait that runs out sets PBB_ERR_DEVICE_TIMEOUT, the CTA
 * drains its copies and returns without writing its output. A limit of 0
 * makes a wait give up as soon as its data has not yet landed (for tests).
 */
int pbb_set_wait_timeout_ns(unsigned long long ns);

/*
 * Keys of the support each CTA handles (the split of the support across CTAs
 * whose partials are fused with Eq. (lse)). 0 = automatic (default): chosen
 * from the batch, Hkv, B, d and the device's SM count. A positive value is
 * rounded up to a whole number of tiles. Returns the previous setting.
 */
int pbb_set_chunk_keys(int keys);

/* Keys per CTA a PBB decode step of this shape would use on the current device (0 on error). */
int pbb_plan_chunk_keys(int batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype);

/*
 * Which kernel a decode step of this shape runs on the current device:
 * PBB_KERNEL_CUDA_CORES (packed fp32 FMAs; every shape) or PBB_KERNEL_TENSOR_CORES
 * (bf16 steps with Hq/Hkv = 8, where the scores of a 16-key block against the
 * 8 query heads form a dense mma tile, or Hq/Hkv = 4 or 6 with the tile's other
 * columns zero; needs B a multiple of 64). Window steps of the shape take the
 * same kernel. Negative on error.
 */
enum { PBB_KERNEL_AUTO = -1, PBB_KERNEL_CUDA_CORES = 0, PBB_KERNEL_TENSOR_CORES = 1 };
int pbb_plan_kernel(int batch, int Hq, int Hkv, int d, int B, pbb_dtype dtype);

/*
 * Whether a decode step of this shape (window = 0 for PBB, else the window size
 * of pbb_swa_decode_step) launches the support-ordering kernel before the decode
 * kernel on the current device: 1 or 0, negative on error. No counterpart in the
 * paper. A step on the tensor-core kernel whose supports are all whole work items,
 * with at least four of them per resident CTA, first sorts its sequences by
 * support length (one small kernel, into the stream's workspace) and then takes
 * the supports longest first, so that its CTAs finish together. The order changes
 * no result: every support is an independent work item.
 */
int pbb_plan_support_order(int batch, int Hq, int Hkv, int d, int B, int window, pbb_dtype dtype);

/*
 * Kernel choice for the decode steps that follow (process-wide, like
 * pbb_set_chunk_keys): PBB_KERNEL_AUTO (the default) lets the library choose;
 * PBB_KERNEL_CUDA_CORES runs every step on the CUDA-core kernel;
 * PBB_KERNEL_TENSOR_CORES runs every step the tensor-core kernel supports (bf16
 * PBB steps, Hq/Hkv in {4, 6, 8}, B a multiple of 64) on it whatever the batch,
 * the rest on the CUDA cores. Returns the previous choice, or
 * PBB_ERR_INVALID_ARG (and no change) for any other value.
 */
int pbb_set_kernel(int kernel);

/*
 * No counterpart in the paper: a library-usage variant for callers that cannot
 * allocate device memory while they decode (a serving runtime that owns all of
 * HBM through its own pool and forbids other allocations, or a loop that cannot
 * afford the device-wide synchronisation a cudaMalloc can bring).
 *
 * Same arguments, layouts and result as pbb_decode_step (bf16), but the split
 * scratch (per-(sequence, KV head) arrival counters and split partials) lives
 * in a fixed array of PBB_NOALLOC_SCRATCH_BYTES compiled into the library;
 * every GPU that loads the library holds that array until the process exits.
 * The call never allocates or frees memory. A step whose split needs more than
 * the array holds (more than 65,534 (sequence, KV head) pairs, or partials
 * beyond the rest of the array) returns PBB_ERR_SCRATCH_LIMIT without
 * launching; pbb_decode_step handles those shapes. Bounded waits use the
 * default limit of one second (pbb_set_wait_timeout_ns does not apply here).
 *   - The first call on each device, with that device current, looks up the
 *     array's device address (cudaGetSymbolAddress) and caches it; make that
 *     first call before any stream capture.
 *   - All calls on a device share the one array, which keeps the last call's
 *     contents; each call zeroes the counters it uses (an asynchronous memset
 *     on `stream`) before its kernel. Calls whose execution overlaps on the GPU
 *     (different streams, or concurrent host threads) race on the array: the
 *     caller must order them.
 */
#define PBB_NOALLOC_SCRATCH_BYTES (16u << 20)
int pbb_decode_step_noalloc(const void* q, const void* k_new, const void* v_new, void* k_ring,
                            void* v_ring, const int32_t* pos, float* out, int batch, int Hq,
                            int Hkv, int d, int B, cudaStream_t stream);

/*
 * No counterpart in the paper: a measurement utility. Reads every byte of
 * buf[0, bytes) once from device memory the way the decode kernels do (16 KiB
 * bulk copies into a shared-memory ring, 8 in flight, one CTA per SM; a tail
 * under 16 KiB by plain loads). Timing it gives the read-only HBM bandwidth,
 * the roof of a decode step (which reads its K/V support and writes almost
 * nothing), next to the copy (read + write) bandwidth. buf: device pointer,
 * 16-byte aligned, bytes a multiple of 16; sink: device pointer, 8-byte
 * aligned, caller-owned: the tail's words are xor-folded into it, and bit 63
 * is set if a bounded wait on a copy ran out. Asynchronous on `stream`;
 * PBB_ERR_INVALID_ARG on a null or misaligned argument, nothing launched for
 * bytes = 0.
 */
int pbb_stream_read(const void* buf, size_t bytes, unsigned long long* sink, cudaStream_t stream);

/* Static description of an error code. */
const char* pbb_error_string(int code);

#ifdef __cplusplus
}
#endif

#endif /* PBB_H_ */
