// Argument blocks and launchers of the streaming / sequential kernels of libqe.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace qe {

// In-block sequential CD over one column block [b0, b0 + bw).
struct CdArgs {
    int64_t q, p;
    int64_t b0;
    int bw;
    float *R;                       // residual in grid-step units: (P - What Sigma_bar) / s + z
    int64_t ldr;
    int store_base;                 // write the staged block values back to R (rolling window)
    const float *part;              // split-K partials [nsplit][q][ldpart] (t-units)
    int nsplit;
    int64_t part_stride, ldpart;
    // Change lists (rolling window): per row and column block, the changes of
    // that block's most recent visit, entry = column offset | (int16 Delta' << 16).
    const float *sbar;              // non-NULL: correction from the lists x fp32 Sigma_bar rows
    int64_t lds;                    // leading dimension of sbar
    int nblk;                       // column blocks per row
    int *lcnt;                      // [q][nblk] entry counts
    uint32_t *lent;                 // [q][nblk][B] entries; non-NULL: record this visit's changes
    const float *tri;               // packed diagonal blocks of Sigma_bar (launch_pack_diag)
    const float *scale, *zero;      // per row, or per row and group: [i * ngroups + column / gsize]
    int64_t gsize, ngroups;         // columns per group (p when not grouped) and groups per row
    int grouped;                    // grouped grids: the Delta' planes carry s_g Delta' (absolute) and
                                    // the split partials are absolute (divided by the block's scale)
    const float *d;                 // Sigma_jj (objective change of each decision)
    double *rowdf;                  // per-row objective change accumulator, or NULL
    float maxq;
    int first_sweep;                // What_start is R itself (not on the grid)
    int frac;                       // Delta' real-valued (every coordinate moves): three planes, in-block
                                    // sequential kernel
    const float *vstart;            // non-NULL: What_start in grid units, leading dimension ldv (the
                                    // values a relaxed sweep left)
    float *vout;                    // non-NULL: relaxed sweep (relax heuristic, Sec. 3.2): a live column
                                    // takes beta~ itself, written here; codes get its nearest level
    int64_t ldv;
    int write_qf;                   // also write C - z (needed by the residual GEMM)
    uint8_t *codes;                 // in: codes at sweep start (unless first_sweep); out: new codes
    int64_t ldc;
    __nv_bfloat16 *qf;              // out: C - z
    int64_t ldq;
    __nv_bfloat16 *dp;              // out: Delta' hi plane (mid / lo planes dp_plane_rows apart), or NULL
    int64_t ldd, dp_plane_rows;
    int dp_f16;                     // 1: Delta' is an integer: one fp16 plane (the fp16 window GEMM);
                                    // 2: real Delta' (first sweep) times dp_scale in two fp16 planes
    float dp_scale;
    unsigned *err;
    // optional gate: the launch does its work only when *gate == gate_run (the
    // adaptive sweep schedule enqueues both forms of a sweep and runs one)
    const int *gate;
    int gate_run;
    // test hook of the failure path (in-block kernels): skip_copy = 1 issues no copy
    // of the packed Sigma_bar block, so the bounded wait for it gives up after
    // wait_ns (0 = the library's limit) and latches a timeout; nothing is in flight
    int skip_copy;
    unsigned long long wait_ns;
    // Near-tie refinement: a decision whose beta~ (binary32, grid units) lies within
    // tie_eps of a rounding midpoint between two levels is taken again from beta~
    // recomputed in binary64 from the row's current state (Lemma 1):
    //   beta~_j = T_j + sum_{k != j} (T_k - What_k) Sigma_kj / Sigma_jj,  T = W (- H).
    // 0 = off (relaxed sweeps and the sweep after one, whose start is real-valued).
    float tie_eps;
    const float *S;                 // Sigma as given (p x p, leading dimension lds_full)
    int64_t lds_full;
    const void *W;                  // the layer (bf16 or fp32, leading dimension ldw)
    int w_bf16;
    int64_t ldw;
    const float *Hd;                // outlier variant: dense H (target W - H, leading dimension ldh), or NULL
    int64_t ldh;
    // change-driven kernel with the refinement: rows with near-tie notes go to this
    // queue (entries, then two B-float rows per entry: final and start codes) and are
    // finished by the check kernel; tq_cnt[0] counts entries, tq_cnt[1] check CTAs done
    // (both zero between launches: the check kernel's last CTA resets them)
    struct TieEntry *tq;
    float *tq_rows;
    unsigned *tq_cnt;
};

// One queued row of the change-driven kernel's near-tie check.
struct TieEntry {
    int64_t i;              // the row
    double df;              // its objective change (warp-summed)
    int nev;                // notes (columns within tie_eps of a midpoint), ev[0 .. min(nev, 8))
    int ev[8];
    int pad[3];
};

// Objective / reference-norm reduction.
struct ObjArgs {
    int64_t q, p;
    const void *W;
    int w_bf16;
    int64_t ldw;
    const float *H;                 // dense outlier matrix or NULL
    int64_t ldh;
    const uint8_t *codes;           // NULL: reference norm sum (W-H)_ij d_j R_ij
    int64_t ldc;
    const float *scale, *zero, *d;
    const float *R;                 // residual (or P for the reference norm)
    int64_t ldr;
};

// Per row (gsize = p) or per row and group of gsize columns: scale / zero [q][ceil(p / gsize)].
cudaError_t launch_grid(const void *W, int w_bf16, int64_t ldw, const float *H, int64_t ldh, int64_t q,
                        int64_t p, int64_t gsize, int bits, float *scale, float *zero, unsigned *err,
                        cudaStream_t s);
cudaError_t launch_sigma_norm(const float *S, int64_t lds, int64_t p, float *d, __nv_bfloat16 *snt,
                              int64_t ldn, unsigned *err, cudaStream_t s);
// Sigma_bar^T in two fp16 planes (rows [0, p) hi, [p, 2p) lo; leading dimension ldn, zero-padded),
// each row j scaled by a power of two; cscale[j] = the factor that undoes it.
cudaError_t launch_sigma_planes_h2(const float *S, int64_t lds, int64_t p, const float *d, __half *snh, int64_t ldn,
                                   float *cscale, cudaStream_t s);
// bf16 W (q x p) as one fp16 plane (leading dimension ld), each row scaled by a power of two;
// rscale[i] = the factor that undoes it.
cudaError_t launch_w_plane_h1(const void *W, int64_t ldw, int64_t q, int64_t p, __half *wh, int64_t ld, float *rscale,
                              cudaStream_t s);
// fp32 Sigma_bar, row k = the coupling of column k to every column (ld columns, zero-padded).
cudaError_t launch_sigma_bar_rows(const float *S, int64_t lds, int64_t p, const float *d, float *sbar,
                                  int64_t ld, cudaStream_t s);
cudaError_t launch_make_planes(const void *W, int w_bf16, int64_t ldw, int64_t q, int64_t p,
                               int split, __nv_bfloat16 *out, int64_t ldo, cudaStream_t s);
cudaError_t launch_init_residual(const void *W, int w_bf16, int64_t ldw, const float *H, int64_t ldh,
                                 int64_t q, int64_t p, int64_t gsize, const float *scale, const float *zero,
                                 float *R, int64_t ldr, cudaStream_t s);
// obj[out] = obj[prev] + sum_i rowdf[i]; rowdf is zeroed.  prev may be NULL (0).  With a
// gate, only when *gate == gate_run.
cudaError_t launch_obj_step(double *rowdf, int64_t q, const double *prev, double *out, cudaStream_t s,
                            const int *gate = nullptr, int gate_run = 0);
// The adaptive sweep schedule's switch: counts the entries of the change lists
// (the changes of the sweep just finished, n = q * nblk counts) and sets *flag = 1
// when they are fewer than `below`; a set flag stays set (no work then).  counter:
// one 8-byte device word of scratch.
// *form = *flag ? 2 : 1 (which form of the adaptive schedule ran the sweep just enqueued).
cudaError_t launch_record_form(const int *flag, uint8_t *form, cudaStream_t s);
cudaError_t launch_list_switch(const int *lcnt, int64_t n, int64_t below, unsigned long long *counter, int *flag,
                               cudaStream_t s);
// C - z (one exact fp16 plane), or with grouped grids s_g (C - z_g) in three bf16 planes
// (rows [0, q), [q, 2q), [2q, 3q)); gsize = p: per-row grids.
cudaError_t launch_codes_to_qf(const uint8_t *codes, int64_t ldc, const float *scale, const float *zero,
                               int64_t q, int64_t p, int64_t gsize, int grouped, __nv_bfloat16 *qf,
                               int64_t ldq, cudaStream_t s);
cudaError_t launch_cd_block(int B, const CdArgs &a, int nsm, cudaStream_t s);
// The near-tie check after a change-driven launch with the refinement (a.tq set):
// every queued row's notes against beta~ recomputed exactly, a row with a wrong
// decision decided again, and the queued rows' results written.
cudaError_t launch_cd_tie_check(int B, const CdArgs &a, int nsm, cudaStream_t s);
// Sweeps [t_begin, t_end) with the change-list correction in one persistent launch
// (a.sbar, a.lcnt, a.lent set; a.b0 / a.bw / a.part unused); the objective change of
// sweep t and row i goes to rowdf_t[(t - t_begin) q + i]; sweep_codes (optional) gets
// the codes after each sweep at [t][q][p].  A CTA runs a sweep in the free mode when
// its rows made at most free_max_changes changes each (on average) in the previous
// sweep; first_lockstep = 1 forces the lockstep mode for the first sweep, 2 marks
// R as refreshed since the lists were left (they give only the previous sweep's
// change counts; the window starts empty, every row is visited).  flush: end
// with R the exact residual of the final codes (each block's base takes the changes
// its last visit did not see).
cudaError_t launch_cd_rows_lists(int B, const CdArgs &a, int t_begin, int t_end, double *rowdf_t,
                                 uint8_t *sweep_codes, int first_lockstep, int free_max_changes, int flush,
                                 int nsm, cudaStream_t s);
// obj[t] = obj[t-1] + sum_i rowdf_t[t][i] for t < nt, starting from *prev (or 0).  With a
// gate, only when *gate == gate_run.
cudaError_t launch_obj_prefix(const double *rowdf_t, int64_t q, int nt, const double *prev, double *out,
                              cudaStream_t s, const int *gate = nullptr, int gate_run = 0);
int64_t packed_diag_floats(int64_t p, int B);
cudaError_t launch_pack_diag(const __nv_bfloat16 *snt, int64_t ldn, int64_t p, int B, float *out,
                             cudaStream_t s);
int objective_blocks(int64_t q);
// fp64 partials written by the residual GEMM's fused objective (8 per 128 x 256 tile)
inline int64_t rfull_partials(int64_t q, int64_t p) { return ((q + 127) / 128) * ((p + 255) / 256) * 8; }
cudaError_t launch_sum_partials(const double *partial, int n, double *out, cudaStream_t s);
cudaError_t launch_objective(const ObjArgs &a, double *partial, double *out, cudaStream_t s);

}  // namespace qe
