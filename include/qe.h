/*
 * qe.h -- C ABI of libqe.so: QuantEase layer-wise quantization on one GB300
 * (Behdin et al., "QuantEase: Optimization-based Quantization for Language
 * Models", arXiv 2309.01885).
 *
 * Problem (Sec. 2.1, Eq. layerwise-main): for a linear layer with weights
 * W (q x p: q output channels, p input features) and calibration inputs
 * X (p x n), find What on a per-row uniform b-bit grid Q_i minimising
 *     f(What) = || W X - What X ||_F^2 = tr((W - What) Sigma (W - What)^T),
 * Sigma = X X^T.  The solver is cyclic coordinate descent with the closed-form
 * quantized update of Lemma 1, organised as the accelerated Algorithm 3.
 *
 * Conventions for every entry point:
 *  - All array arguments are DEVICE pointers owned by the caller, unless a
 *    parameter says otherwise.  The library never frees caller memory.
 *  - Matrices are row-major with an explicit leading dimension (elements).
 *  - Calls are stream-ordered and asynchronous on `stream` (a cudaStream_t;
 *    NULL = legacy default stream).  Argument errors are returned
 *    synchronously before anything is enqueued.  Errors found on the device
 *    (non-finite input, a device-side wait that gave up) are latched in a
 *    per-device error word and reported by qe_sync_status().
 *  - Scratch memory: taken from opts->workspace when given (at least
 *    qe_workspace_size() bytes, 256-byte aligned), otherwise allocated with
 *    cudaMallocAsync / cudaFreeAsync on `stream` inside the call.
 *  - Thread safety: distinct streams may be used from distinct host threads.
 */
#ifndef QE_H
#define QE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t; declared here so the header needs no CUDA headers. */
typedef struct CUstream_st *qe_stream_t;

typedef enum {
    QE_OK = 0,
    QE_ERR_INVALID_ARG = 1,   /* bad size, pointer, alignment or option */
    QE_ERR_CUDA = 2,          /* a CUDA runtime/driver call failed */
    QE_ERR_OOM = 3,           /* workspace allocation failed or too small */
    QE_ERR_NUMERIC = 4,       /* non-finite value in W or Sigma (device-detected) */
    QE_ERR_TIMEOUT = 5,       /* a bounded device-side wait gave up (device-detected) */
    QE_ERR_UNSUPPORTED = 6    /* option or layout not implemented */
} qe_status;

typedef enum { QE_F32 = 0, QE_BF16 = 1 } qe_dtype;

typedef enum {
    QE_FEATURE_MAJOR = 0,     /* X is p x n row-major: the paper's X (Sec. 2.1) */
    QE_TOKEN_MAJOR = 1        /* X is n x p row-major: activations as a model emits them */
} qe_xlayout;

/* Kernel classes an optional qe_timer can time (bit k of its mask = class k). */
typedef enum {
    QE_KERNEL_PINIT_GEMM = 0,     /* P = W (I + Sigma_bar), once per call */
    QE_KERNEL_RESIDUAL_GEMM = 1,  /* R = P - What Sigma_bar (+ the fused objective) */
    QE_KERNEL_TRAIL_GEMM = 2,     /* per column block: Delta' Sigma_bar correction (split-K) */
    QE_KERNEL_CD_BLOCK = 3,       /* per column block: the in-block coordinate updates */
    QE_KERNEL_CD_LISTS = 4,       /* the sweeps driven by change lists (one persistent launch) */
    QE_KERNEL_COUNT = 5
} qe_kernel;

/* Opaque set of CUDA event pairs; see qe_timer_create. */
typedef struct qe_timer qe_timer;

typedef struct {
    /* Column block width B of the blocked CD sweep: 0 = default (256); 64, 128 or 256. */
    int block_width;
    /* Relax heuristic of Sec. 3.2: with R > 0, sweep t (counted from 1) with
     * t mod R = 0 and t < iters keeps every live coordinate at beta~ of Lemma 1
     * unquantized (a column with Sigma_jj <= 0 stays on its level); the last
     * sweep always quantizes.  obj[t] of a relaxed sweep is f of the relaxed
     * weights, and its sweep_codes record their nearest levels.  0 = off;
     * negative is QE_ERR_INVALID_ARG; the outlier variant returns
     * QE_ERR_UNSUPPORTED for R != 0. */
    int relax_period;
    /* Structured outliers (Sec. 4.3): 1 = H keeps whole columns, the floor(s/q)
     * of largest l2 norm, in place of the s largest entries (outlier variant
     * only; must be 0 for qe_quantize_layer). */
    int structured_outliers;
    /* Outlier variant: power-method iterations for lambda_max(Sigma), 0 = default 64. */
    int power_iters;
    /* How the cross-block term Delta'[:, other blocks] Sigma_bar[:, block] of a
     * sweep is formed (no paper counterpart: both forms compute the same sums of
     * Eq. cd-update-closed-2).  Sweeps 1 .. dense_sweeps multiply the dense
     * change matrix on the tensor cores; later sweeps, where few codes change,
     * walk per-row lists of the changed columns and add their fp32 Sigma_bar
     * rows.  0 = default: the adaptive schedule of switch_below; n > 0: sweeps
     * 1 .. n dense, lists from sweep n + 1; a value >= iters keeps the dense
     * form throughout;
     * negative is QE_ERR_INVALID_ARG.  Ignored by the outlier variant. */
    int dense_sweeps;
    /* List sweeps: the rows of a CTA step through the column blocks together
     * (sharing each packed Sigma_bar block) while they made more than this many
     * changes per row in the previous sweep, then each row runs on its own.
     * Both modes take the same decisions in the same order; only the speed
     * differs.  0 = default (64); -1 = always together; below -1 is
     * QE_ERR_INVALID_ARG.  The outlier variant applies it to its per-iteration
     * sweeps after the first. */
    int free_changes;
    /* Grouped grids (the paper notes that grouping can be incorporated into the
     * per-channel grid of Sec. 2.1): G > 0 gives every row one scale and
     * zero-point per group of G consecutive columns, and the call's `scales` /
     * `zeros` hold q x ceil(p / G) values, row-major ([i * groups + j / G]).
     * 0 (or G >= p) = one grid per row.  G must be a multiple of the block width
     * (QE_ERR_INVALID_ARG otherwise); relax_period != 0 or the outlier variant
     * return QE_ERR_UNSUPPORTED with G < p. */
    int group_size;
    /* Optional warm start (Sec. 3.1: the descent may start from another method's solution):
     * q x p codes (leading dimension p) on the grid this call computes.  NULL = start at W. */
    const uint8_t *init_codes;
    /* Optional output: iters x q x p codes after every sweep (for parity checks). */
    uint8_t *sweep_codes;
    /* Optional output: one double, ||W X||_F^2, the denominator of the relative
     * calibration error of Sec. 3.4 (target W - H for the outlier variant). */
    double *wx_norm2;
    /* Optional caller workspace (device, 256-byte aligned) and its size. */
    void *workspace;
    size_t workspace_bytes;
    /* Optional: record CUDA events around the launches of the timed kernel classes. */
    qe_timer *timer;
    /* Adaptive sweep schedule, used when dense_sweeps = 0 (no paper counterpart:
     * it only picks which of the two forms above computes each sweep's sums).
     * The sweeps after the first take the dense tensor-core form until a sweep
     * changes fewer than switch_below codes; the change lists take the rest.
     * The choice is made on the device from the change counts, so the call
     * stays asynchronous: both forms of such a sweep are enqueued and the one
     * not chosen returns at once.  0 = automatic: when the fp32 Sigma_bar rows
     * (4 p^2 bytes) fit in three quarters of the GPU's L2, lists from sweep 2
     * (their gathers hit L2); otherwise the threshold of a cost model (a dense
     * sweep's 6 q p^2 flops of plane products against a gather of 4 p bytes
     * from DRAM per change, the next sweep changing about 0.7 times as many
     * codes).  > 0 forces the adaptive schedule with this threshold; negative is
     * QE_ERR_INVALID_ARG.  Ignored by the outlier variant. */
    int64_t switch_below;
    /* Optional output (device, iters bytes): how each sweep of qe_quantize_layer
     * formed its cross-block sums: 0 = the sequential form (sweep 1, a relaxed
     * sweep and the sweep after one), 1 = the dense tensor-core form, 2 = the
     * change lists.  NULL = not recorded.  Ignored by the outlier variant. */
    uint8_t *sweep_forms;
    /* Test hook of the failure path (no paper counterpart): 1 = qe_quantize_layer
     * (without init_codes; ignored by the outlier variant) runs up to its first
     * in-block kernel, which issues no copy of its packed
     * Sigma_bar block and waits for it with a 5 ms limit.  The wait gives up,
     * QE_ERR_TIMEOUT is latched for qe_sync_status, and the call returns QE_OK
     * without further work (codes, scales, zeros and obj are not all written).
     * Nothing is left in flight, so the next call runs normally.  0 = off. */
    int wait_test;
    /* Near-tie refinement (no paper counterpart: it makes the binary32 kernels
     * take the decisions exact arithmetic takes).  A coordinate update rounds
     * beta~ / s + z (Lemma 1) to the nearest level; where that binary32 value
     * lies within tie_eps grid steps of a midpoint between two levels, the
     * decision is taken again from beta~ recomputed from the row's current
     * codes, W (and H) and Sigma: every term exact, the sum in double-float
     * (about 48 significant bits).  0 = default (1e-5, about four times the
     * largest binary32 error measured on the benchmark layers); negative =
     * off.
     * Not applied in relaxed sweeps or the sweep after one. */
    float tie_eps;
} qe_opts;

/*
 * Sigma = X X^T (Lemma 1; the memory-footprint paragraph of Sec. 3.2 keeps it
 * resident), fp32 output, p x p row-major, leading dimension p.
 *   X          device, bf16 or fp32; layout QE_FEATURE_MAJOR (p x n, leading
 *              dimension ldx >= n) or QE_TOKEN_MAJOR (n x p, ldx >= p).
 *   accumulate 0: Sigma = X X^T;  1: Sigma += X X^T (stream n in chunks).
 * The result is exactly symmetric.  bf16 X runs on tcgen05 tensor cores with
 * fp32 accumulation; fp32 X on fp32 FMA.  Errors: QE_ERR_INVALID_ARG for
 * p < 1, n < 0, a short leading dimension or NULL pointers.
 */
qe_status qe_build_sigma(const void *X, qe_dtype x_dtype, qe_xlayout layout,
                         int64_t p, int64_t n, int64_t ldx, float *Sigma,
                         int accumulate, qe_stream_t stream);

/*
 * QuantEase for one layer (Algorithm 3, Sec. 3.2, blocked by columns).
 *   W        device q x p, bf16 or fp32, leading dimension ldw >= p.
 *   Sigma    device p x p fp32, symmetric PSD (e.g. from qe_build_sigma).
 *            Columns with Sigma_jj <= 0 (X_j = 0, footnote of Lemma 1) drop
 *            out of the objective and get the nearest level of W_ij.
 *   bits     b in [2, 8]: 2^b levels per row.
 *   iters    K >= 1 cyclic sweeps over j = 1..p (Sec. 3.1).
 *   codes    out, device q x p uint8 (leading dimension p): What_ij = s_i (c_ij - z_i).
 *   scales   out, device q floats s_i;  zeros: out, device q floats z_i
 *            (integer-valued).  Grid: asymmetric per-row min/max with 0 in
 *            range, s = (max - min)/(2^b - 1), z = round(-min/s), evaluated
 *            in binary32 (Sec. 2.1: evenly spaced levels, as in GPTQ).
 *   obj      out, device iters doubles: f after each sweep.
 *   opts     may be NULL (all defaults).
 * Each coordinate takes the nearest level of the closed-form minimiser
 * (Lemma 1); ties in rounding go to the even integer of beta/s + z.
 */
qe_status qe_quantize_layer(const void *W, qe_dtype w_dtype, int64_t q, int64_t p,
                            int64_t ldw, const float *Sigma, int bits, int iters,
                            const qe_opts *opts, uint8_t *codes, float *scales,
                            float *zeros, double *obj, qe_stream_t stream);

/*
 * Outlier-aware QuantEase (Sec. 4, Eq. main-outlier, Algorithm 4): What on
 * the grid plus a sparse full-precision H with ||H||_0 <= s_budget.
 *   H = P_s(W) initially; the grid is computed from W without those entries
 *   (Sec. 4.3); every iteration runs one CD sweep with target W - H, then one
 *   IHT step H <- P_s(H - eta grad_H g), eta = 1/(2 lambda_max(Sigma)) with
 *   lambda_max from opts->power_iters power-method steps (Sec. 4.3).
 *   P_s keeps the s_budget largest |entries|; ties go to the smaller
 *   row-major index i*p + j; exact zeros are never kept.
 *   With opts->structured_outliers = 1 (Sec. 4.3, "Structured Outliers") P_s
 *   keeps instead the floor(s_budget / q) columns of largest l2 norm (ties:
 *   smaller column index; a column of zeros is never kept), and the grid
 *   leaves out the starting columns; every entry of a kept column is kept.
 *   H_val, H_idx  out, device s_budget floats / int64: the kept values and
 *                 their linear indices i*p + j in ascending order.
 *   H_nnz         out, device int64: number of kept entries (<= s_budget;
 *                 q x the kept columns when structured).
 *   obj           out, device iters doubles: g after the IHT step of each iteration.
 *   obj_cd        out (may be NULL), device iters doubles: g after the CD sweep.
 * Other arguments as qe_quantize_layer.
 */
qe_status qe_quantize_layer_outlier(const void *W, qe_dtype w_dtype, int64_t q,
                                    int64_t p, int64_t ldw, const float *Sigma,
                                    int bits, int iters, int64_t s_budget,
                                    const qe_opts *opts, uint8_t *codes,
                                    float *scales, float *zeros, float *H_val,
                                    int64_t *H_idx, int64_t *H_nnz, double *obj,
                                    double *obj_cd, qe_stream_t stream);

/*
 * Sigma = X X^T (Lemma 1) for bf16 X held in HOST memory, streamed to the GPU
 * in chunks of tokens.  (Beyond Lemma 1 the paper has no counterpart: this is
 * how calibration activations that live on the host reach the GPU.)
 *   X          host, bf16, feature-major p x n, leading dimension ldx >= n
 *              (elements).  Page-locked memory (cudaHostAlloc/Register) lets
 *              the copies run asynchronously; pageable memory is still correct.
 *   Sigma      device, fp32 p x p as in qe_build_sigma; accumulate as there.
 *   staging    device, 16-byte aligned, holding nbuf = staging_bytes /
 *              (p * chunk * 2) chunk buffers, at least 2 (at most 64 are used).
 *              Caller-owned; it may be reused across calls.
 *   chunk      tokens per copy, a positive multiple of 64 (wide chunks copy
 *              faster: rows of chunk * 2 bytes are the copy's unit).
 * Chunks are copied on an internal per-device copy stream into the nbuf
 * buffers in turn, the turn carrying over from one call to the next, while
 * earlier chunks accumulate on `stream`; a buffer is refilled only after the
 * GEMM that read it (also one of an earlier call) has finished.  So the copies
 * of one call overlap work queued on `stream` before it: with nbuf >= the
 * chunks of one call they all arrive during that work, and with nbuf >= twice
 * that (e.g. chunk = n, two buffers) consecutive calls' copies run back to
 * back, each call's while the previous one computes.  The call
 * returns once all work is enqueued; X must stay unchanged and allocated until
 * Sigma is complete on `stream`.  Calls are serialized per device while they
 * enqueue (the copy stream and its events are shared).
 * Errors: QE_ERR_INVALID_ARG for bad sizes or pointers, a chunk that is not a
 * positive multiple of 64, or a staging area that is too small or misaligned
 * (before anything is enqueued); QE_ERR_CUDA when a copy, event or launch fails.
 */
qe_status qe_build_sigma_host(const void *X, int64_t p, int64_t n, int64_t ldx, float *Sigma,
                              int accumulate, void *staging, size_t staging_bytes, int64_t chunk,
                              qe_stream_t stream);

/*
 * Sigma = X X^T like qe_build_sigma, but the call never allocates device
 * memory.  (The paper has no counterpart: this is a deployment variant.)
 *
 * For callers that cannot let a library allocate: processes whose device
 * memory is handed out entirely by their own allocator, latency-critical
 * loops that must stay off the allocator, and platforms without
 * stream-ordered allocation.  Where qe_build_sigma allocates a staging buffer
 * (bf16 X that is token-major, or feature-major with an unaligned base or a
 * leading dimension that is not a multiple of 8), this entry point stages
 * through a fixed array of QE_STATIC_SCRATCH_BYTES that belongs to the
 * library's device image: every GPU that loads the library holds it until the
 * process exits.  Other inputs need no staging and run as in qe_build_sigma.
 *
 *   Arguments, layouts and the result are those of qe_build_sigma.
 *   Limit: a staged X needs p <= QE_STATIC_SCRATCH_BYTES / 128 (= 65536 for
 *   8 MiB); larger p returns QE_ERR_INVALID_ARG before anything is enqueued.
 *   First call per device: looks up the array's device address (with that
 *   device current) and caches it; make that first call before any stream
 *   capture.  The cached address is not looked up again: resetting the device
 *   (cudaDeviceReset) after the first call and then calling again is not
 *   supported (the same holds for the device error word every entry point
 *   caches, see qe_sync_status).
 *   Every call shares the array: calls that overlap on the GPU (other streams,
 *   other host threads) race.  Each call clears the part of the array it relies
 *   on being zero.
 */
#define QE_STATIC_SCRATCH_BYTES (8u << 20)
qe_status qe_build_sigma_static(const void *X, qe_dtype x_dtype, qe_xlayout layout,
                                int64_t p, int64_t n, int64_t ldx, float *Sigma,
                                int accumulate, qe_stream_t stream);

/* Bytes of scratch qe_quantize_layer (outlier = 0) or qe_quantize_layer_outlier
 * (outlier = 1) needs for this shape and options; written to *bytes. */
qe_status qe_workspace_size(int64_t q, int64_t p, int outlier, const qe_opts *opts,
                            size_t *bytes);

/*
 * Kernel timing (profiling aid; the paper has no counterpart).  A timer holds
 * `capacity` pairs of CUDA events created on the current device.  Passed in
 * qe_opts, it makes the call record one pair on the call's stream around each
 * launch whose class bit is set in `kernel_mask`, until the pairs run out
 * (later launches go untimed).  Recording adds no synchronisation;
 * qe_timer_read waits for the recorded events and returns the number of timed
 * launches of `kernel` and their summed duration in milliseconds.  Not
 * thread-safe: one timer per host thread.
 */
qe_status qe_timer_create(unsigned kernel_mask, int capacity, qe_timer **timer);
qe_status qe_timer_read(qe_timer *timer, int kernel, int *launches, double *total_ms);
qe_status qe_timer_reset(qe_timer *timer);
qe_status qe_timer_destroy(qe_timer *timer);

/*
 * Bit-packed codes, the storage form of a quantized layer (the paper fixes the
 * codes as integers 0 .. 2^b - 1, Sec. 2.1, and leaves their storage open).
 * Row i of `out` is a little-endian bit stream: code j occupies bits
 * [j bits, (j + 1) bits), least significant bit first, of the row's
 * ceil(p bits / 8) bytes; the padding bits of the last byte are zero.
 *   codes  device, q x p uint8, leading dimension ldc >= p; only the low `bits`
 *          bits of each code are stored (qe_quantize_layer's codes fit).
 *   out    device, q rows of ldo >= ceil(p bits / 8) bytes (bytes beyond that
 *          are not written).
 * qe_unpack_codes is the inverse.  Both are stream-ordered; QE_ERR_INVALID_ARG
 * for NULL pointers, q or p < 1, bits outside 1 .. 8 or a short leading
 * dimension (before anything is enqueued); QE_ERR_CUDA when the launch fails.
 */
qe_status qe_pack_codes(const uint8_t *codes, int64_t q, int64_t p, int64_t ldc, int bits, uint8_t *out,
                        int64_t ldo, qe_stream_t stream);
qe_status qe_unpack_codes(const uint8_t *packed, int64_t q, int64_t p, int64_t ldp, int bits, uint8_t *codes,
                          int64_t ldc, qe_stream_t stream);

/*
 * P_s of the IHT step (Sec. 4.3, Eq. iht-update) on its own: of the N entries
 * of T, keep the s of largest magnitude.  Exact zeros are never kept; among
 * entries of equal magnitude at the threshold the smaller index goes first.
 * The operator qe_quantize_layer_outlier applies once per iteration.
 *   T          device, N fp32 values (any alignment; 16-byte aligned is faster).
 *   s          0 <= s <= N.
 *   idx, val   device, s int64 / s fp32 (may be NULL when s = 0): the kept
 *              indices in ascending order and their values T[idx[k]].
 *   nnz        device, one int64: the number kept (min(s, nonzeros of T)).
 *   workspace  device scratch of qe_hard_threshold_workspace(N) bytes,
 *              256-byte aligned, owned by the caller, not used across calls.
 * Stream-ordered.  QE_ERR_INVALID_ARG for NULL pointers, N < 1 or N >= 2^32,
 * s outside 0 .. N, or a short or misaligned workspace (before anything is
 * enqueued); QE_ERR_CUDA when a launch fails.
 */
qe_status qe_hard_threshold_workspace(int64_t N, size_t *bytes);
qe_status qe_hard_threshold(const float *T, int64_t N, int64_t s, int64_t *idx, float *val, int64_t *nnz,
                            void *workspace, size_t workspace_bytes, qe_stream_t stream);

/* Waits for `stream`, then returns and clears the error latched on the current
 * device (QE_ERR_NUMERIC / QE_ERR_TIMEOUT), or QE_ERR_CUDA if the stream failed.
 * The error word is a file-scope device variable whose address the library looks
 * up once per device and caches; calling the library on a device after a
 * cudaDeviceReset of that device is not supported. */
qe_status qe_sync_status(qe_stream_t stream);

/* Static description of a status code. */
const char *qe_status_string(qe_status status);

/* ABI version: major * 10000 + minor * 100 + patch. */
int qe_version(void);

#ifdef __cplusplus
}
#endif

#endif /* QE_H */
