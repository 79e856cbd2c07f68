/*
 * Post-Boundary Bridge (PBB) attention (decode step and whole-sequence
 * forward): plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY. Nothing on the product path may link, load or call
 * this file: only the tests, the smoke check and the benchmark's CPU-baseline
 * leg use it. It shares no code, header or constant with the CUDA library.
 *
 * What it computes, written out from the paper's definitions, slowly and in
 * the paper's order:
 *   - the block start and phase of Eq. 1 (Sec. 2.2): p(t) = b*floor(t/b),
 *     r(t) = t - p(t);
 *   - the PBB support of Eq. (pbb) (Sec. 3): {p..t}, plus the preceding
 *     half-block {p-h..p-1} when p > 0 and r < h, with b = 2h;
 *   - single-softmax attention over that support, Eq. (attention) (Sec. 3):
 *     z_ts = q_t . k_s / sqrt(d_h),  o_t = sum e^{z} v / sum e^{z};
 *   - the relocation-free ring of Appendix F.1 (Proposition "Relocation-free
 *     PBB cache"): position s is stored in slot s mod b; and a second,
 *     ring-indexed evaluation of the same attention over the interval form
 *     [a(t), t], a(t) = max(0, h(floor(t/h) - 1)) (Eq. pbb_relay, App. A.3);
 *   - sliding-window attention over {t-w+1, ..., t} (Sec. 2.3), the pattern
 *     the paper compares PBB with, for the window-ring decode control;
 *   - PBB attention for every position of whole sequences (the forward pass /
 *     prefill of Sec. 3) with its log-partition ln sum exp(z) (Eq. lse), and
 *     its gradients with respect to q, k and v (the backward pass).
 *
 * The brute-force evaluation visits every s in [0, t] and tests the support
 * predicate in its block/bridge form; it never uses the interval form, so the
 * two forms are checked against each other only through results.
 *
 * Floating point is fp64 throughout. Inputs are widened exactly (bf16 and
 * fp32 values are exactly representable in fp64).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_OK 0
#define ORACLE_ERR_ARG (-1)
#define ORACLE_ERR_WINDOW (-2) /* a source the support needs is not in the history given */
#define ORACLE_ERR_RING (-3)   /* the ring does not hold a position the support needs */

/* Eq. 1: block start p(t) = b * floor(t / b) (t >= 0). */
static long block_start(long t, long b) { return b * (t / b); }

/* Eq. (pbb): is source s in A_PBB(t)? Block/bridge form, with h = b/2. */
int pbb_oracle_in_support(long t, long s, long b)
{
    const long h = b / 2;
    const long p = block_start(t, b);
    const long r = t - p;
    if (s < 0 || s > t) return 0;
    if (s >= p) return 1; /* causal block prefix {p, ..., t} */
    if (p > 0 && r < h && s >= p - h && s <= p - 1) return 1; /* bridge {p-h, ..., p-1} */
    return 0;
}

/* |A_PBB(t)|, counted by testing the predicate at every s in [0, t]. */
long pbb_oracle_support_count(long t, long b)
{
    long n = 0;
    for (long s = 0; s <= t; ++s) n += pbb_oracle_in_support(t, s, b);
    return n;
}

/*
 * Attention of one query vector over a list of sources (Eq. attention), fp64,
 * two passes: the maximum logit first, then the normalised weighted sum.
 * k_rows[i], v_rows[i] point at the d-vectors of the i-th source.
 */
static void softmax_attend(const double* q, const double* const* k_rows,
                           const double* const* v_rows, long n, int d,
                           double* z, double* out, double* lse)
{
    const double scale = 1.0 / sqrt((double)d);
    double m = -INFINITY;
    for (long i = 0; i < n; ++i) {
        double dot = 0.0;
        for (int c = 0; c < d; ++c) dot += q[c] * k_rows[i][c];
        z[i] = dot * scale;
        if (z[i] > m) m = z[i];
    }
    double den = 0.0;
    for (int c = 0; c < d; ++c) out[c] = 0.0;
    for (long i = 0; i < n; ++i) {
        const double w = exp(z[i] - m);
        den += w;
        for (int c = 0; c < d; ++c) out[c] += w * v_rows[i][c];
    }
    for (int c = 0; c < d; ++c) out[c] /= den;
    if (lse) *lse = m + log(den); /* ln sum_s exp(z_s), the log-partition of Eq. (lse) */
}

/*
 * One decode step for every sequence by brute force over the history.
 *
 *   q       [batch][Hq][d]          query of the token at position t[b]
 *   hist_k  [batch][Hkv][n_hist][d] K history: row j is position s0[b] + j
 *   hist_v  [batch][Hkv][n_hist][d] V history, same indexing
 *   s0, t   [batch]                 window start and current position
 *   out     [batch][Hq][d]
 *
 * Query head j reads KV head j / (Hq/Hkv) (contiguous GQA grouping). For each
 * sequence the predicate is tested at every s in [0, t]; a source it admits
 * must lie in the window, else ORACLE_ERR_WINDOW. Rows outside the support are
 * never read.
 */
int pbb_oracle_attend(const double* q, const double* hist_k, const double* hist_v,
                      const long* s0, const long* t, long n_hist, int batch, int Hq,
                      int Hkv, int d, long b, double* out, int n_threads)
{
    if (batch < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || b < 2 || (b % 2) || (Hq % Hkv) ||
        n_hist <= 0)
        return ORACLE_ERR_ARG;
    const int group = Hq / Hkv;
    int status = ORACLE_OK;
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
#pragma omp parallel for schedule(dynamic, 1)
    for (int bi = 0; bi < batch; ++bi) {
        const long tb = t[bi];
        long* src = (long*)malloc(sizeof(long) * (size_t)(b + 1));
        long n = 0;
        int bad = (tb < 0);
        for (long s = 0; s <= tb && !bad; ++s) {
            if (!pbb_oracle_in_support(tb, s, b)) continue;
            if (s < s0[bi] || s >= s0[bi] + n_hist || n >= b + 1) { bad = 1; break; }
            src[n++] = s;
        }
        if (bad) {
#pragma omp critical
            status = ORACLE_ERR_WINDOW;
            free(src);
            continue;
        }
        const double** kr = (const double**)malloc(sizeof(double*) * (size_t)n);
        const double** vr = (const double**)malloc(sizeof(double*) * (size_t)n);
        double* z = (double*)malloc(sizeof(double) * (size_t)n);
        for (int j = 0; j < Hq; ++j) {
            const int kv = j / group;
            const size_t head = ((size_t)bi * Hkv + kv) * (size_t)n_hist;
            for (long i = 0; i < n; ++i) {
                const size_t row = head + (size_t)(src[i] - s0[bi]);
                kr[i] = hist_k + row * d;
                vr[i] = hist_v + row * d;
            }
            softmax_attend(q + ((size_t)bi * Hq + j) * d, kr, vr, n, d, z,
                           out + ((size_t)bi * Hq + j) * d, NULL);
        }
        free(z);
        free(vr);
        free(kr);
        free(src);
    }
    return status;
}

/*
 * PBB attention over whole sequences (Sec. 3): every position t of a sequence
 * attends to A_PBB(t) among that sequence's positions 0..n-1 with the single
 * softmax of Eq. (attention). This is what the paper's fused forward kernel
 * computes for all t at once (the training forward, and the prefill that
 * precedes decoding); here it is evaluated one requested output row at a time.
 *
 *   q     [batch][Hq][n][d]   row t is the query of position t
 *   k, v  [batch][Hkv][n][d]  row s is the key / value of position s
 *   rows  [n_rows][3]         (sequence, query head, position t) of each row
 *   out   [n_rows][d]
 *   lse   [n_rows]            ln sum_{s in A(t)} exp(z_ts), the log-partition a
 *                             backward pass reuses (Eq. lse); NULL to skip
 *
 * Query head j reads KV head j / (Hq/Hkv). The predicate is tested at every
 * s in [0, t] (block/bridge form), as in pbb_oracle_attend.
 */
int pbb_oracle_forward_rows(const double* q, const double* k, const double* v, int batch, int Hq,
                            int Hkv, long n, int d, long b, const long* rows, long n_rows,
                            double* out, double* lse, int n_threads)
{
    if (batch < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || n <= 0 || b < 2 || (b % 2) || (Hq % Hkv) ||
        n_rows < 0)
        return ORACLE_ERR_ARG;
    for (long i = 0; i < n_rows; ++i) {
        const long* rw = rows + 3 * i;
        if (rw[0] < 0 || rw[0] >= batch || rw[1] < 0 || rw[1] >= Hq || rw[2] < 0 || rw[2] >= n)
            return ORACLE_ERR_ARG;
    }
    const int group = Hq / Hkv;
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
#pragma omp parallel for schedule(dynamic, 16)
    for (long i = 0; i < n_rows; ++i) {
        const long bi = rows[3 * i], j = rows[3 * i + 1], t = rows[3 * i + 2];
        const long kv = j / group;
        const double** kr = (const double**)malloc(sizeof(double*) * (size_t)(b + 1));
        const double** vr = (const double**)malloc(sizeof(double*) * (size_t)(b + 1));
        double* z = (double*)malloc(sizeof(double) * (size_t)(b + 1));
        const size_t head = ((size_t)bi * Hkv + (size_t)kv) * (size_t)n;
        long m = 0;
        for (long s = 0; s <= t; ++s) {
            if (!pbb_oracle_in_support(t, s, b)) continue;
            if (m < b + 1) { /* |A(t)| <= b always (Eq. pbb_cache_support) */
                kr[m] = k + (head + (size_t)s) * d;
                vr[m] = v + (head + (size_t)s) * d;
            }
            ++m;
        }
        if (m > b) m = b + 1; /* cannot happen; keeps the buffers in bounds */
        softmax_attend(q + (((size_t)bi * Hq + (size_t)j) * (size_t)n + (size_t)t) * d, kr, vr, m, d, z,
                       out + (size_t)i * d, lse ? lse + i : NULL);
        free(z);
        free(vr);
        free(kr);
    }
    return ORACLE_OK;
}

/*
 * Gradients of the whole-sequence PBB attention: the backward pass of the
 * paper's fused training kernel (Sec. 3; Appendix "exact union and numerical
 * checks", bridge gradients into the previous block's K/V included). Given the
 * upstream gradient dO of every output row, the chain rule through Eq.
 * (attention) over A_PBB(t), written out per query row t and head j:
 *   z_ts  = q_t . k_s / sqrt(d),  P_ts = exp(z_ts) / sum_{u in A(t)} exp(z_tu)
 *   dP_ts = dO_t . v_s
 *   dz_ts = P_ts (dP_ts - sum_{u in A(t)} P_tu dP_tu)
 *   dq_t += dz_ts k_s / sqrt(d)    dk_s += dz_ts q_t / sqrt(d)    dv_s += P_ts dO_t
 * for every s in A(t). K/V gradients collect every query head of the group
 * (GQA) and every position whose support holds s.
 *
 *   q, dout     [batch][Hq][n][d]       dq   [batch][Hq][n][d]
 *   k, v        [batch][Hkv][n][d]      dk, dv [batch][Hkv][n][d]
 */
int pbb_oracle_backward(const double* q, const double* k, const double* v, const double* dout, int batch,
                        int Hq, int Hkv, long n, int d, long b, double* dq, double* dk, double* dv,
                        int n_threads)
{
    if (batch < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || n <= 0 || b < 2 || (b % 2) || (Hq % Hkv))
        return ORACLE_ERR_ARG;
    const int group = Hq / Hkv;
    const double scale = 1.0 / sqrt((double)d);
    memset(dq, 0, sizeof(double) * (size_t)batch * Hq * n * d);
    memset(dk, 0, sizeof(double) * (size_t)batch * Hkv * n * d);
    memset(dv, 0, sizeof(double) * (size_t)batch * Hkv * n * d);
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
    /* one (sequence, KV head) pair per task: its dk, dv rows are written by no other task */
#pragma omp parallel for schedule(dynamic, 1)
    for (long pr = 0; pr < (long)batch * Hkv; ++pr) {
        const long bi = pr / Hkv, kv = pr % Hkv;
        long* src = (long*)malloc(sizeof(long) * (size_t)(b + 1));
        double* P = (double*)malloc(sizeof(double) * (size_t)(b + 1));
        double* dP = (double*)malloc(sizeof(double) * (size_t)(b + 1));
        const double* kh = k + (size_t)pr * n * d;
        const double* vh = v + (size_t)pr * n * d;
        double* dkh = dk + (size_t)pr * n * d;
        double* dvh = dv + (size_t)pr * n * d;
        for (int jg = 0; jg < group; ++jg) {
            const long j = kv * group + jg;
            const size_t qh = ((size_t)bi * Hq + (size_t)j) * (size_t)n;
            for (long t = 0; t < n; ++t) {
                const double* qt = q + (qh + (size_t)t) * d;
                const double* dot_ = dout + (qh + (size_t)t) * d;
                double* dqt = dq + (qh + (size_t)t) * d;
                long m = 0;
                for (long s = 0; s <= t; ++s)
                    if (pbb_oracle_in_support(t, s, b) && m < b + 1) src[m++] = s;
                /* P over the support: two passes as in softmax_attend */
                double zmax = -INFINITY;
                for (long i = 0; i < m; ++i) {
                    double z = 0.0;
                    for (int c = 0; c < d; ++c) z += qt[c] * kh[src[i] * d + c];
                    P[i] = z * scale;
                    if (P[i] > zmax) zmax = P[i];
                }
                double den = 0.0;
                for (long i = 0; i < m; ++i) {
                    P[i] = exp(P[i] - zmax);
                    den += P[i];
                }
                double sum_pdp = 0.0;
                for (long i = 0; i < m; ++i) {
                    P[i] /= den;
                    double x = 0.0;
                    for (int c = 0; c < d; ++c) x += dot_[c] * vh[src[i] * d + c];
                    dP[i] = x;
                    sum_pdp += P[i] * x;
                }
                for (long i = 0; i < m; ++i) {
                    const double dz = P[i] * (dP[i] - sum_pdp);
                    const double* ks = kh + src[i] * d;
                    double* dks = dkh + src[i] * d;
                    double* dvs = dvh + src[i] * d;
                    for (int c = 0; c < d; ++c) {
                        dqt[c] += dz * ks[c] * scale;
                        dks[c] += dz * qt[c] * scale;
                        dvs[c] += P[i] * dot_[c];
                    }
                }
            }
        }
        free(dP);
        free(P);
        free(src);
    }
    return ORACLE_OK;
}

/*
 * Sliding-window attention, the comparison pattern of the paper (Sec. 2.3,
 * Proposition "Sliding-window relay"): A_SWA(t) = {max(0, t-w+1), ..., t}, the
 * window w counting the current position. Same brute-force evaluation as
 * pbb_oracle_attend (predicate at every s in [0, t], fp64, two passes).
 */
int pbb_oracle_in_window(long t, long s, long w)
{
    return s >= 0 && s <= t && s >= t - w + 1;
}

long pbb_oracle_window_count(long t, long w)
{
    long n = 0;
    for (long s = 0; s <= t; ++s) n += pbb_oracle_in_window(t, s, w);
    return n;
}

int pbb_oracle_attend_window(const double* q, const double* hist_k, const double* hist_v,
                             const long* s0, const long* t, long n_hist, int batch, int Hq,
                             int Hkv, int d, long w, double* out, int n_threads)
{
    if (batch < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || w < 1 || (Hq % Hkv) || n_hist <= 0)
        return ORACLE_ERR_ARG;
    const int group = Hq / Hkv;
    int status = ORACLE_OK;
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
#pragma omp parallel for schedule(dynamic, 1)
    for (int bi = 0; bi < batch; ++bi) {
        const long tb = t[bi];
        long* src = (long*)malloc(sizeof(long) * (size_t)(w + 1));
        long n = 0;
        int bad = (tb < 0);
        for (long s = 0; s <= tb && !bad; ++s) {
            if (!pbb_oracle_in_window(tb, s, w)) continue;
            if (s < s0[bi] || s >= s0[bi] + n_hist || n >= w + 1) { bad = 1; break; }
            src[n++] = s;
        }
        if (bad) {
#pragma omp critical
            status = ORACLE_ERR_WINDOW;
            free(src);
            continue;
        }
        const double** kr = (const double**)malloc(sizeof(double*) * (size_t)n);
        const double** vr = (const double**)malloc(sizeof(double*) * (size_t)n);
        double* z = (double*)malloc(sizeof(double) * (size_t)n);
        for (int j = 0; j < Hq; ++j) {
            const int kv = j / group;
            const size_t head = ((size_t)bi * Hkv + kv) * (size_t)n_hist;
            for (long i = 0; i < n; ++i) {
                const size_t row = head + (size_t)(src[i] - s0[bi]);
                kr[i] = hist_k + row * d;
                vr[i] = hist_v + row * d;
            }
            softmax_attend(q + ((size_t)bi * Hq + j) * d, kr, vr, n, d, z,
                           out + ((size_t)bi * Hq + j) * d, NULL);
        }
        free(z);
        free(vr);
        free(kr);
        free(src);
    }
    return status;
}

/* ---- ring simulator (Appendix F.1) --------------------------------------- */

/*
 * Write the rows of position t[b] into slot t[b] mod b of every KV head's ring.
 *   ring     [batch][Hkv][b][row_bytes]   raw element bits (bf16 or fp32)
 *   tags     [batch][b]                   position held by each slot, -1 = never written
 *   new_rows [batch][Hkv][row_bytes]
 * Sequences with t[b] < 0 are skipped.
 */
void pbb_oracle_ring_append(uint8_t* ring, long* tags, const uint8_t* new_rows,
                            const long* t, int batch, int Hkv, long b, long row_bytes)
{
    for (int bi = 0; bi < batch; ++bi) {
        if (t[bi] < 0) continue;
        const long slot = t[bi] % b;
        for (int kv = 0; kv < Hkv; ++kv) {
            uint8_t* dst = ring + (((size_t)bi * Hkv + kv) * (size_t)b + (size_t)slot) * row_bytes;
            memcpy(dst, new_rows + ((size_t)bi * Hkv + kv) * row_bytes, (size_t)row_bytes);
        }
        tags[(size_t)bi * b + slot] = t[bi];
    }
}

/*
 * Replay a history window into the ring, oldest first: row j of hist is
 * position s0[b] + j, j < n_hist; negative positions are skipped.
 *   hist [batch][Hkv][n_hist][row_bytes]
 */
void pbb_oracle_ring_replay(uint8_t* ring, long* tags, const uint8_t* hist, const long* s0,
                            long n_hist, int batch, int Hkv, long b, long row_bytes)
{
    for (int bi = 0; bi < batch; ++bi) {
        for (long j = 0; j < n_hist; ++j) {
            const long s = s0[bi] + j;
            if (s < 0) continue;
            const long slot = s % b;
            for (int kv = 0; kv < Hkv; ++kv) {
                const uint8_t* src = hist + (((size_t)bi * Hkv + kv) * (size_t)n_hist + (size_t)j) * row_bytes;
                uint8_t* dst = ring + (((size_t)bi * Hkv + kv) * (size_t)b + (size_t)slot) * row_bytes;
                memcpy(dst, src, (size_t)row_bytes);
            }
            tags[(size_t)bi * b + slot] = s;
        }
    }
}

/* Exact widening of one stored element to fp64: bf16 (2 bytes) or fp32 (4 bytes). */
static double widen(const uint8_t* p, int elem_bytes)
{
    float f;
    if (elem_bytes == 2) {
        uint16_t h;
        memcpy(&h, p, 2);
        const uint32_t w = (uint32_t)h << 16; /* bf16 is the high half of an fp32 */
        memcpy(&f, &w, 4);
    } else {
        memcpy(&f, p, 4);
    }
    return (double)f;
}

/*
 * Second evaluation of the same attention, read from the ring simulator over
 * the interval form [a(t), t], a(t) = max(0, h(floor(t/h) - 1)) (Eq. pbb_relay).
 * Every source must be present (tags[s mod b] == s), else ORACLE_ERR_RING.
 * The ring must already hold position t (append first, then attend).
 *   q [batch][Hq][d] fp64; ring_k, ring_v as in pbb_oracle_ring_append.
 */
int pbb_oracle_attend_ring(const double* q, const uint8_t* ring_k, const uint8_t* ring_v,
                           const long* tags, int elem_bytes, const long* t, int batch,
                           int Hq, int Hkv, int d, long b, double* out, int n_threads)
{
    if (batch < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || b < 2 || (b % 2) || (Hq % Hkv) ||
        (elem_bytes != 2 && elem_bytes != 4))
        return ORACLE_ERR_ARG;
    const long h = b / 2;
    const int group = Hq / Hkv;
    const long row_bytes = (long)d * elem_bytes;
    int status = ORACLE_OK;
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
#pragma omp parallel for schedule(dynamic, 1)
    for (int bi = 0; bi < batch; ++bi) {
        const long tb = t[bi];
        long a = h * (tb / h - 1);
        if (a < 0) a = 0;
        const long n = tb - a + 1;
        int bad = (tb < 0);
        for (long s = a; s <= tb && !bad; ++s)
            if (tags[(size_t)bi * b + (size_t)(s % b)] != s) bad = 1;
        if (bad) {
#pragma omp critical
            status = ORACLE_ERR_RING;
            continue;
        }
        double* kbuf = (double*)malloc(sizeof(double) * (size_t)n * d);
        double* vbuf = (double*)malloc(sizeof(double) * (size_t)n * d);
        const double** kr = (const double**)malloc(sizeof(double*) * (size_t)n);
        const double** vr = (const double**)malloc(sizeof(double*) * (size_t)n);
        double* z = (double*)malloc(sizeof(double) * (size_t)n);
        for (int kv = 0; kv < Hkv; ++kv) {
            for (long i = 0; i < n; ++i) {
                const long slot = (a + i) % b;
                const uint8_t* kp = ring_k + (((size_t)bi * Hkv + kv) * (size_t)b + (size_t)slot) * row_bytes;
                const uint8_t* vp = ring_v + (((size_t)bi * Hkv + kv) * (size_t)b + (size_t)slot) * row_bytes;
                for (int c = 0; c < d; ++c) {
                    kbuf[i * d + c] = widen(kp + (size_t)c * elem_bytes, elem_bytes);
                    vbuf[i * d + c] = widen(vp + (size_t)c * elem_bytes, elem_bytes);
                }
                kr[i] = kbuf + i * d;
                vr[i] = vbuf + i * d;
            }
            for (int g = 0; g < group; ++g) {
                const int j = kv * group + g;
                softmax_attend(q + ((size_t)bi * Hq + j) * d, kr, vr, n, d, z,
                               out + ((size_t)bi * Hq + j) * d, NULL);
            }
        }
        free(z);
        free(vr);
        free(kr);
        free(vbuf);
        free(kbuf);
    }
    return status;
}

/* Number of OpenMP threads a parallel region of the oracle uses. */
int pbb_oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
