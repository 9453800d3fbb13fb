/*
 * QuantEase oracle: a plain, slow, binary64 CPU restatement of the layer-wise
 * quantization method of Behdin et al., "QuantEase: Optimization-based
 * Quantization for Language Models" (arXiv 2309.01885).
 *
 * TEST INFRASTRUCTURE ONLY. This file is compiled into its own shared library
 * (oracle/_build/libqe_oracle.so) that only the test-suite, the smoke check and
 * the CPU-baseline leg of bench.py load. It shares no code, header, table or
 * constant with the CUDA library, and the product path never calls it.
 *
 * Conventions (Sec. 2.1): matrices are row-major; W is q x p (q output channels,
 * p input features), X is p x n, Sigma = X X^T is p x p.  All arithmetic is
 * binary64, except the per-row grid (scale, zero-point): its zero-point is an
 * integer decided by a division, and that decision is taken in binary32 here as
 * in the GPU path, so that both sides decide it identically.
 *
 * Every function below is pinned by the CPU tests in tests/test_oracle_*.py
 * (brute-force 1-D argmin, exhaustive search on tiny layers, monotone
 * objective, Algorithm 1 == Algorithm 3, diagonal Sigma == round-to-nearest,
 * direct ||WX - W^X||^2, eigvalsh for lambda_max, a full sort for P_s, and
 * the IHT descent of Lemma 3, and for the relax heuristic one Gauss-Seidel
 * step of the normal equations per relaxed sweep).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Host threads of the OpenMP row loops (for timing only): n > 0 sets the count;
 * returns the count in effect before the call. */
int qo_threads(int n)
{
#ifdef _OPENMP
    const int old = omp_get_max_threads();
    if (n > 0)
        omp_set_num_threads(n);
    return old;
#else
    (void)n;
    return 1;
#endif
}

/* ------------------------------------------------------------------------- */
/* Quantization grid and operator                                            */
/* ------------------------------------------------------------------------- */

/*
 * Per-channel uniform grid Q_i (Sec. 2.1: evenly spaced levels, the grid GPTQ uses):
 * levels s_i * (c - z_i), c = 0 .. 2^b - 1, asymmetric min/max over row i with
 * 0 always inside the range; an all-zero row gets the range [-1, 1].
 * excl (q*p bytes, may be NULL) removes entries from the pool; with 0 always in
 * the range this is the same as setting them to 0 (Sec. 4.3, outliers removed
 * from the quantization pool).  Evaluated in binary32 (see file header).
 * Grouped grids (a grid per row and group of gsize consecutive columns, the
 * grouping the paper notes can be incorporated): the same rule over each
 * group's columns; scale / zero are q x ceil(p / gsize), row-major.  gsize = p
 * is the per-row grid.
 */
void qo_grid_groups(const double *W, int64_t q, int64_t p, int64_t gsize, int bits,
                    const uint8_t *excl, float *scale, float *zero)
{
    const float maxq = (float)((1 << bits) - 1);
    const int64_t ng = (p + gsize - 1) / gsize;
    for (int64_t i = 0; i < q; ++i)
        for (int64_t g = 0; g < ng; ++g) {
            float lo = 0.0f, hi = 0.0f;
            const int64_t j1 = (g + 1) * gsize < p ? (g + 1) * gsize : p;
            for (int64_t j = g * gsize; j < j1; ++j) {
                if (excl && excl[i * p + j])
                    continue;
                float w = (float)W[i * p + j];
                if (w < lo) lo = w;
                if (w > hi) hi = w;
            }
            if (lo == 0.0f && hi == 0.0f) {
                lo = -1.0f;
                hi = 1.0f;
            }
            float s = (hi - lo) / maxq;
            float z = nearbyintf(-lo / s);
            scale[i * ng + g] = s;
            zero[i * ng + g] = z;
        }
}

void qo_grid(const double *W, int64_t q, int64_t p, int bits,
             const uint8_t *excl, float *scale, float *zero)
{
    qo_grid_groups(W, q, p, p, bits, excl, scale, zero);
}

/*
 * q_i of Eq. (eq:quant): the nearest level to x.  With levels s (c - z) and
 * s > 0, |x - s (c - z)| is minimised over integers c by the integer nearest
 * to x / s + z, clamped to [0, 2^b - 1] (a convex 1-D distance).  Exact ties
 * go to the even integer (round-half-to-even).  Returns the code c.
 */
static int qo_code(double x, double s, double z, int maxq)
{
    double c = nearbyint(x / s + z);
    if (c < 0.0) c = 0.0;
    if (c > (double)maxq) c = (double)maxq;
    return (int)c;
}

static double qo_level(int c, double s, double z)
{
    return s * ((double)c - z);
}

/* Round-to-nearest of a whole matrix on the (grouped) grid. */
void qo_rtn_groups(const double *W, int64_t q, int64_t p, int64_t gsize, const float *scale,
                   const float *zero, int bits, uint8_t *codes)
{
    const int maxq = (1 << bits) - 1;
    const int64_t ng = (p + gsize - 1) / gsize;
    for (int64_t i = 0; i < q; ++i)
        for (int64_t j = 0; j < p; ++j)
            codes[i * p + j] = (uint8_t)qo_code(W[i * p + j], scale[i * ng + j / gsize],
                                                zero[i * ng + j / gsize], maxq);
}

void qo_rtn(const double *W, int64_t q, int64_t p, const float *scale,
            const float *zero, int bits, uint8_t *codes)
{
    qo_rtn_groups(W, q, p, p, scale, zero, bits, codes);
}

/* ------------------------------------------------------------------------- */
/* Sigma and objective                                                       */
/* ------------------------------------------------------------------------- */

/* Sigma = X X^T (Lemma 1), X p x n row-major, Sigma p x p. */
void qo_sigma(const double *X, int64_t p, int64_t n, double *S)
{
#pragma omp parallel for schedule(dynamic)
    for (int64_t a = 0; a < p; ++a) {
        for (int64_t b = a; b < p; ++b) {
            double acc = 0.0;
            for (int64_t k = 0; k < n; ++k)
                acc += X[a * n + k] * X[b * n + k];
            S[a * p + b] = acc;
            S[b * p + a] = acc;
        }
    }
}

/* A bfloat16 bit pattern is the upper half of a binary32: promote it exactly. */
static double qo_bf16(uint16_t h)
{
    const uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * Selected entries of Sigma = X X^T (Lemma 1): out[m] = sum_k X[a[m]][k] X[b[m]][k]
 * for X given as bfloat16 bit patterns, row-major with leading dimension ldx.
 * For checking a Sigma too large to form here entry by entry.
 */
void qo_sigma_pairs_bf16(const uint16_t *X, int64_t n, int64_t ldx, const int64_t *a,
                         const int64_t *b, int64_t npairs, double *out)
{
#pragma omp parallel for schedule(dynamic)
    for (int64_t m = 0; m < npairs; ++m) {
        const uint16_t *xa = X + a[m] * ldx, *xb = X + b[m] * ldx;
        double acc = 0.0;
        for (int64_t k = 0; k < n; ++k)
            acc += qo_bf16(xa[k]) * qo_bf16(xb[k]);
        out[m] = acc;
    }
}

/*
 * Sigma as the CD routines read it: binary64, or binary32 promoted exactly row
 * by row (for layers whose binary64 Sigma would not fit in host memory).  The
 * arithmetic is binary64 either way.
 */
typedef struct {
    const double *d;
    const float *f;
    int64_t p;
} qo_sig;

/* Row j of Sigma in binary64: a pointer into S->d, or buf filled from S->f. */
static const double *qo_srow(const qo_sig *S, int64_t j, double *buf)
{
    if (S->d)
        return S->d + j * S->p;
    const float *r = S->f + j * S->p;
    for (int64_t k = 0; k < S->p; ++k)
        buf[k] = (double)r[k];
    return buf;
}

/* Scratch row for qo_srow (only a binary32 Sigma needs one). */
static double *qo_sbuf(const qo_sig *S)
{
    return S->d ? NULL : (double *)malloc((size_t)S->p * sizeof(double));
}

/* d^T Sigma d for one row d (the per-row term of f = tr(D Sigma D^T), proof of Lemma 1). */
static double qo_quad(const double *d, const qo_sig *S, int64_t p, double *buf)
{
    double f = 0.0;
    for (int64_t a = 0; a < p; ++a) {
        if (d[a] == 0.0)
            continue;
        const double *Sa = qo_srow(S, a, buf);
        double t = 0.0;
        for (int64_t b = 0; b < p; ++b)
            t += Sa[b] * d[b];
        f += d[a] * t;
    }
    return f;
}

/*
 * Per-row objective f_i = (T_i - What_i) Sigma (T_i - What_i)^T of Eq.
 * (layerwise-main), What = s (codes - z) plus the optional dense H (Eq.
 * main-outlier: g = ||W X - (What + H) X||^2).  rows_out[i] = f_i.
 */
void qo_objective_rows_groups(const double *W, const double *H, const uint8_t *codes,
                              const float *scale, const float *zero, int64_t q, int64_t p,
                              int64_t gsize, const double *S, double *rows_out)
{
    const qo_sig Sg = {S, NULL, p};
    const int64_t ng = (p + gsize - 1) / gsize;
#pragma omp parallel for schedule(dynamic)
    for (int64_t i = 0; i < q; ++i) {
        double *d = (double *)malloc((size_t)p * sizeof(double));
        for (int64_t j = 0; j < p; ++j) {
            double wh = qo_level(codes[i * p + j], scale[i * ng + j / gsize], zero[i * ng + j / gsize]);
            d[j] = W[i * p + j] - wh - (H ? H[i * p + j] : 0.0);
        }
        rows_out[i] = qo_quad(d, &Sg, p, NULL);
        free(d);
    }
}

void qo_objective_rows(const double *W, const double *H, const uint8_t *codes,
                       const float *scale, const float *zero, int64_t q, int64_t p,
                       const double *S, double *rows_out)
{
    qo_objective_rows_groups(W, H, codes, scale, zero, q, p, p, S, rows_out);
}

/* ------------------------------------------------------------------------- */
/* Algorithm 1 (basic QuantEase, rank-1 bookkeeping of What Sigma)           */
/* ------------------------------------------------------------------------- */

/*
 * One cyclic sweep j = 1..p of Algorithm 1 on one row (rows are independent,
 * Sec. 3.2 "Parallelization over i").
 *   Wh   : current row of What (in/out)
 *   WS   : (What Sigma)_i,:  kept current by the rank-1 updates of Eq. (rank1-update)
 *   TS   : (T Sigma)_i,: for the fixed target T (T = W, or W - H in Algorithm 4)
 *   tgt  : the target row T_i (used for dead columns only)
 * For each column j: u = [(What Sigma)_ij - Sigma_jj What_ij - (T Sigma)_ij] / Sigma_jj
 * (so -u is beta~ of Lemma 1), remove the old column (part A), set
 * What_ij = q_i(-u), add the new column (part B).
 * A dead column (Sigma_jj <= 0, i.e. X_j,: = 0, footnote of Lemma 1) drops out
 * of the objective; it is set to the nearest level of the target and fixed.
 * forced (p codes, may be NULL): use these codes instead of q_i(-u) (teacher
 * forcing; beta~ is still recorded).  beta (p, may be NULL) receives beta~.
 * relax != 0: the relax heuristic of Sec. 3.2, What_ij = beta~ itself (no
 * quantization, forced ignored); codes[j] then records q_i(beta~), the nearest
 * level, as a view of the relaxed row.  Dead columns stay on their level.
 */
static void qo_sweep_row(const qo_sig *S, int64_t p, const float *srow, const float *zrow, int64_t gsize,
                         int maxq, const double *tgt, const double *TS, double *Wh, double *WS,
                         const uint8_t *forced, uint8_t *codes, double *beta, double *buf,
                         int relax)
{
    for (int64_t j = 0; j < p; ++j) {
        const double s = srow[j / gsize], z = zrow[j / gsize];
        const double *Sj = qo_srow(S, j, buf);
        const double djj = Sj[j];
        int c;
        if (djj > 0.0) {
            double u = (WS[j] - djj * Wh[j] - TS[j]) / djj;
            double b = -u;
            double old = Wh[j];
            for (int64_t k = 0; k < p; ++k)          /* part (A) */
                WS[k] -= old * Sj[k];
            if (relax) {
                c = qo_code(b, s, z, maxq);
                Wh[j] = b;
            } else {
                c = forced ? (int)forced[j] : qo_code(b, s, z, maxq);
                Wh[j] = qo_level(c, s, z);
            }
            for (int64_t k = 0; k < p; ++k)          /* part (B) */
                WS[k] += Wh[j] * Sj[k];
            if (beta) beta[j] = b;
        } else {
            c = forced ? (int)forced[j] : qo_code(tgt[j], s, z, maxq);
            Wh[j] = qo_level(c, s, z);
            if (beta) beta[j] = tgt[j];
        }
        codes[j] = (uint8_t)c;
    }
}

/* y = x Sigma for a row vector x. */
static void qo_row_times_sigma(const double *x, const qo_sig *S, int64_t p, double *y, double *buf)
{
    for (int64_t k = 0; k < p; ++k)
        y[k] = 0.0;
    for (int64_t l = 0; l < p; ++l) {
        if (x[l] == 0.0)
            continue;
        const double *Sl = qo_srow(S, l, buf);
        for (int64_t k = 0; k < p; ++k)
            y[k] += x[l] * Sl[k];
    }
}

/*
 * Relax heuristic of Sec. 3.2 (a reading of "every other third iteration"):
 * with period R > 0, sweep t (counted from 1) is relaxed when t mod R = 0 and
 * t < iters, so the last sweep always quantizes.  R = 0: never.
 */
static int qo_relaxed(int relax_period, int t1, int iters)
{
    return relax_period > 0 && t1 % relax_period == 0 && t1 < iters;
}

/*
 * Algorithm 1.  Start: What = W (Sec. 3.1), or the levels of init_codes.
 *   codes       q*p   out: codes after the last sweep
 *   obj_rows    iters*q out (may be NULL): f_i after each sweep
 *   sweep_codes iters*q*p out (may be NULL): codes after each sweep
 *   forced      iters*q*p in (may be NULL): teacher-forced codes per sweep
 *   beta        iters*q*p out (may be NULL): beta~ of every update (in a relaxed
 *               sweep, the relaxed row itself)
 *   relax_period  the relax heuristic (qo_relaxed); 0 = off
 */
static int qo_alg1_core(const double *W, int64_t q, int64_t p, const qo_sig *S,
                        const float *scale, const float *zero, int64_t gsize, int bits, int iters,
                        const uint8_t *init_codes, const uint8_t *forced,
                        uint8_t *codes, double *obj_rows, uint8_t *sweep_codes,
                        double *beta, int relax_period)
{
    const int maxq = (1 << bits) - 1;
    const int64_t ng = (p + gsize - 1) / gsize;
    int err = 0;
#pragma omp parallel for schedule(dynamic)
    for (int64_t i = 0; i < q; ++i) {
        double *Wh = (double *)malloc((size_t)p * sizeof(double));
        double *WS = (double *)malloc((size_t)p * sizeof(double));
        double *TS = (double *)malloc((size_t)p * sizeof(double));
        double *d = (double *)malloc((size_t)p * sizeof(double));
        double *buf = qo_sbuf(S);
        if (!Wh || !WS || !TS || !d || (!S->d && !buf)) {
            err = 1;
        } else {
            const double *Wi = W + i * p;
            const float *srow = scale + i * ng, *zrow = zero + i * ng;
            for (int64_t j = 0; j < p; ++j)
                Wh[j] = init_codes ? qo_level(init_codes[i * p + j], srow[j / gsize], zrow[j / gsize]) : Wi[j];
            qo_row_times_sigma(Wh, S, p, WS, buf);
            qo_row_times_sigma(Wi, S, p, TS, buf);
            for (int t = 0; t < iters; ++t) {
                const size_t off = ((size_t)t * (size_t)q + (size_t)i) * (size_t)p;
                qo_sweep_row(S, p, srow, zrow, gsize, maxq, Wi, TS, Wh, WS,
                             forced ? forced + off : NULL, codes + i * p,
                             beta ? beta + off : NULL, buf,
                             qo_relaxed(relax_period, t + 1, iters));
                if (sweep_codes)
                    memcpy(sweep_codes + off, codes + i * p, (size_t)p);
                if (obj_rows) {
                    for (int64_t j = 0; j < p; ++j)
                        d[j] = Wi[j] - Wh[j];
                    obj_rows[(size_t)t * (size_t)q + (size_t)i] = qo_quad(d, S, p, buf);
                }
            }
        }
        free(Wh); free(WS); free(TS); free(d); free(buf);
    }
    return err;
}

int qo_quantease_alg1(const double *W, int64_t q, int64_t p, const double *S,
                      const float *scale, const float *zero, int bits, int iters,
                      const uint8_t *init_codes, const uint8_t *forced,
                      uint8_t *codes, double *obj_rows, uint8_t *sweep_codes,
                      double *beta, int relax_period)
{
    const qo_sig Sg = {S, NULL, p};
    return qo_alg1_core(W, q, p, &Sg, scale, zero, p, bits, iters, init_codes, forced, codes,
                        obj_rows, sweep_codes, beta, relax_period);
}

/* Algorithm 1 on grouped grids: scale / zero are q x ceil(p / gsize) (qo_grid_groups). */
int qo_quantease_alg1_groups(const double *W, int64_t q, int64_t p, const double *S, int64_t gsize,
                             const float *scale, const float *zero, int bits, int iters,
                             const uint8_t *init_codes, const uint8_t *forced,
                             uint8_t *codes, double *obj_rows, uint8_t *sweep_codes,
                             double *beta, int relax_period)
{
    const qo_sig Sg = {S, NULL, p};
    return qo_alg1_core(W, q, p, &Sg, scale, zero, gsize, bits, iters, init_codes, forced, codes,
                        obj_rows, sweep_codes, beta, relax_period);
}

/* Algorithm 1 with Sigma given in binary32 (promoted exactly; same arithmetic). */
int qo_quantease_alg1_f32(const double *W, int64_t q, int64_t p, const float *S,
                          const float *scale, const float *zero, int bits, int iters,
                          const uint8_t *init_codes, const uint8_t *forced,
                          uint8_t *codes, double *obj_rows, uint8_t *sweep_codes,
                          double *beta, int relax_period)
{
    const qo_sig Sg = {NULL, S, p};
    return qo_alg1_core(W, q, p, &Sg, scale, zero, p, bits, iters, init_codes, forced, codes,
                        obj_rows, sweep_codes, beta, relax_period);
}

/* ------------------------------------------------------------------------- */
/* Algorithm 3 (accelerated QuantEase with partial update)                   */
/* ------------------------------------------------------------------------- */

/*
 * Algorithm 3, written independently of Algorithm 1 as a second form that must
 * agree with it in exact arithmetic (Sec. 3.2, Eq. cd-update-closed-2):
 *   Sn_:,j = Sigma_:,j / Sigma_jj;  P = W Sn (diagonal still 1);  then Sn_jj = 0.
 *   per sweep: dW = What;  Ph = What Sn;
 *     per column j: beta = P_:,j - Ph_:,j + dW_:,1:j Sn_1:j,j;  What_:,j = q(beta);
 *                   dW_:,j -= What_:,j.
 * Dead columns (Sigma_jj <= 0) are set to the nearest level of W and fixed.
 * In a relaxed sweep (qo_relaxed) What_:,j = beta itself, as in Algorithm 1.
 */
int qo_quantease_alg3(const double *W, int64_t q, int64_t p, const double *S,
                      const float *scale, const float *zero, int bits, int iters,
                      uint8_t *codes, double *obj_rows, int relax_period)
{
    const int maxq = (1 << bits) - 1;
    const qo_sig Sg = {S, NULL, p};
    double *Sn = (double *)malloc((size_t)p * (size_t)p * sizeof(double));
    if (!Sn)
        return 1;
    for (int64_t k = 0; k < p; ++k)
        for (int64_t j = 0; j < p; ++j) {
            double djj = S[j * p + j];
            Sn[k * p + j] = djj > 0.0 ? S[k * p + j] / djj : 0.0;
        }
    int err = 0;
#pragma omp parallel for schedule(dynamic)
    for (int64_t i = 0; i < q; ++i) {
        double *P = (double *)malloc((size_t)p * sizeof(double));
        double *Ph = (double *)malloc((size_t)p * sizeof(double));
        double *Wh = (double *)malloc((size_t)p * sizeof(double));
        double *dW = (double *)malloc((size_t)p * sizeof(double));
        if (!P || !Ph || !Wh || !dW) {
            err = 1;
        } else {
            const double *Wi = W + i * p;
            const double s = scale[i], z = zero[i];
            /* P = W Sn with the unit diagonal, before the diagonal is zeroed */
            for (int64_t j = 0; j < p; ++j) {
                double acc = 0.0;
                for (int64_t k = 0; k < p; ++k)
                    acc += Wi[k] * Sn[k * p + j];
                P[j] = acc;
            }
            for (int64_t j = 0; j < p; ++j)
                Wh[j] = Wi[j];
            for (int t = 0; t < iters; ++t) {
                const int relax = qo_relaxed(relax_period, t + 1, iters);
                for (int64_t j = 0; j < p; ++j)
                    dW[j] = Wh[j];
                /* Ph = What Sn with Sn_jj = 0 */
                for (int64_t j = 0; j < p; ++j) {
                    double acc = 0.0;
                    for (int64_t k = 0; k < p; ++k)
                        if (k != j)
                            acc += Wh[k] * Sn[k * p + j];
                    Ph[j] = acc;
                }
                for (int64_t j = 0; j < p; ++j) {
                    int c;
                    double b = 0.0;
                    const int live = S[j * p + j] > 0.0;
                    if (live) {
                        b = P[j] - Ph[j];
                        for (int64_t k = 0; k < j; ++k)   /* k = j adds Sn_jj = 0 */
                            b += dW[k] * Sn[k * p + j];
                        c = qo_code(b, s, z, maxq);
                    } else {
                        c = qo_code(Wi[j], s, z, maxq);
                    }
                    Wh[j] = (relax && live) ? b : qo_level(c, s, z);
                    dW[j] -= Wh[j];
                    codes[i * p + j] = (uint8_t)c;
                }
                if (obj_rows) {
                    double *d = Ph; /* reuse */
                    for (int64_t j = 0; j < p; ++j)
                        d[j] = Wi[j] - Wh[j];
                    obj_rows[(size_t)t * (size_t)q + (size_t)i] = qo_quad(d, &Sg, p, NULL);
                }
            }
        }
        free(P); free(Ph); free(Wh); free(dW);
    }
    free(Sn);
    return err;
}

/* ------------------------------------------------------------------------- */
/* Outlier-aware QuantEase (Sec. 4, Algorithm 4)                             */
/* ------------------------------------------------------------------------- */

/*
 * lambda_max(Sigma) by the power method (Sec. 4.3 names power iteration for it):
 * v0 = 1/sqrt(p) * ones;  iters times: v <- Sigma v / ||Sigma v||;
 * return the Rayleigh quotient v^T Sigma v.
 */
double qo_power_lambda(const double *S, int64_t p, int iters)
{
    double *v = (double *)malloc((size_t)p * sizeof(double));
    double *w = (double *)malloc((size_t)p * sizeof(double));
    for (int64_t k = 0; k < p; ++k)
        v[k] = 1.0 / sqrt((double)p);
    double lam = 0.0;
    for (int it = 0; it <= iters; ++it) {
        for (int64_t a = 0; a < p; ++a) {
            double acc = 0.0;
            for (int64_t b = 0; b < p; ++b)
                acc += S[a * p + b] * v[b];
            w[a] = acc;
        }
        if (it == iters) {
            lam = 0.0;
            for (int64_t a = 0; a < p; ++a)
                lam += v[a] * w[a];
            break;
        }
        double nrm = 0.0;
        for (int64_t a = 0; a < p; ++a)
            nrm += w[a] * w[a];
        nrm = sqrt(nrm);
        if (nrm == 0.0)
            break;
        for (int64_t a = 0; a < p; ++a)
            v[a] = w[a] / nrm;
    }
    free(v);
    free(w);
    return lam;
}

typedef struct {
    double key;
    int64_t idx;
} qo_kv;

static int qo_kv_cmp(const void *a, const void *b)
{
    const qo_kv *x = (const qo_kv *)a, *y = (const qo_kv *)b;
    if (x->key > y->key) return -1;      /* larger magnitude first */
    if (x->key < y->key) return 1;
    if (x->idx < y->idx) return -1;      /* tie: smaller linear index first */
    if (x->idx > y->idx) return 1;
    return 0;
}

static int qo_i64_cmp(const void *a, const void *b)
{
    int64_t x = *(const int64_t *)a, y = *(const int64_t *)b;
    return (x > y) - (x < y);
}

/*
 * P_s of Eq. (iht-update): keep the s entries of largest |T| (over all q*p
 * entries), zero the rest.  Ties at the threshold go to the smaller row-major
 * index; exact zeros are never kept.  idx_out receives the kept linear indices
 * in ascending order; returns their count (<= s).
 */
int64_t qo_topk(const double *T, int64_t N, int64_t s, int64_t *idx_out)
{
    qo_kv *kv = (qo_kv *)malloc((size_t)(N > 0 ? N : 1) * sizeof(qo_kv));
    int64_t m = 0;
    for (int64_t k = 0; k < N; ++k) {
        double a = fabs(T[k]);
        if (a > 0.0) {
            kv[m].key = a;
            kv[m].idx = k;
            ++m;
        }
    }
    qsort(kv, (size_t)m, sizeof(qo_kv), qo_kv_cmp);
    int64_t cnt = m < s ? m : s;
    for (int64_t k = 0; k < cnt; ++k)
        idx_out[k] = kv[k].idx;
    qsort(idx_out, (size_t)cnt, sizeof(int64_t), qo_i64_cmp);
    free(kv);
    return cnt;
}

/*
 * Structured outliers (Sec. 4.3, "Structured Outliers"): in place of the s
 * largest entries, keep whole columns of T: those with the floor(s / q) largest
 * l2 norms, which is the Euclidean projection onto matrices with at most that
 * many nonzero columns.  Ties go to the smaller column index and a column of
 * zeros is never kept (the rules of P_s, applied to the squared column norms,
 * summed over the rows in order).  idx_out receives the kept column indices,
 * ascending; the return value is their number.
 */
int64_t qo_topk_columns(const double *T, int64_t q, int64_t p, int64_t k, int64_t *idx_out)
{
    double *norm2 = (double *)calloc((size_t)(p > 0 ? p : 1), sizeof(double));
    for (int64_t i = 0; i < q; ++i)
        for (int64_t j = 0; j < p; ++j)
            norm2[j] += T[i * p + j] * T[i * p + j];
    const int64_t cnt = qo_topk(norm2, p, k, idx_out);
    free(norm2);
    return cnt;
}

/*
 * The kept entries of T as ascending linear indices: P_s (the s largest |T|),
 * or with `structured` every entry of the kept columns (zeros included).
 */
static int64_t qo_select(const double *T, int64_t q, int64_t p, int64_t s_budget, int structured,
                         int64_t *idx, int64_t *cols)
{
    if (!structured)
        return qo_topk(T, q * p, s_budget, idx);
    const int64_t nc = qo_topk_columns(T, q, p, s_budget / q, cols);
    for (int64_t i = 0; i < q; ++i)
        for (int64_t r = 0; r < nc; ++r)
            idx[i * nc + r] = i * p + cols[r];
    return q * nc;
}

/*
 * Algorithm 4 (outlier-aware QuantEase), block coordinate descent between What
 * and H (Sec. 4.3):
 *   H = P_s(W); grid from W without the support of H; What = W - H;
 *   eta = 1 / (2 lambda_max(Sigma));
 *   per iteration t:
 *     one sweep of Algorithm 1 on every row with target W - H;   obj_cd[t] = g
 *     G = 2 (H + What - W) Sigma;  H = P_s(H - eta G);           obj[t]    = g
 * With `structured`, P_s is the column selection of qo_topk_columns, both for
 * the start H and in the IHT step, and the grid leaves out the start columns.
 * Outputs: codes, scale, zero, dense H (q*p), obj, obj_cd (iters each), eta.
 */
int qo_quantease_outlier(const double *W, int64_t q, int64_t p, const double *S,
                         int bits, int iters, int64_t s_budget, int power_iters,
                         uint8_t *codes, float *scale, float *zero, double *H,
                         double *obj, double *obj_cd, double *eta_out,
                         int64_t *nnz_out, int structured)
{
    const int maxq = (1 << bits) - 1;
    const int64_t N = q * p;
    const qo_sig Sg = {S, NULL, p};
    int64_t *idx = (int64_t *)malloc((size_t)(s_budget > 0 ? s_budget : 1) * sizeof(int64_t));
    int64_t *cols = (int64_t *)malloc((size_t)(p > 0 ? p : 1) * sizeof(int64_t));
    uint8_t *excl = (uint8_t *)calloc((size_t)N, 1);
    double *Wh = (double *)malloc((size_t)N * sizeof(double));
    double *T = (double *)malloc((size_t)N * sizeof(double));
    double *rows = (double *)malloc((size_t)q * sizeof(double));
    if (!idx || !cols || !excl || !Wh || !T || !rows)
        return 1;

    /* H = P_s(W), grid without the support of H, What = W - H */
    int64_t nnz = qo_select(W, q, p, s_budget, structured, idx, cols);
    memset(H, 0, (size_t)N * sizeof(double));
    for (int64_t k = 0; k < nnz; ++k) {
        H[idx[k]] = W[idx[k]];
        excl[idx[k]] = 1;
    }
    qo_grid(W, q, p, bits, excl, scale, zero);
    for (int64_t k = 0; k < N; ++k)
        Wh[k] = W[k] - H[k];

    double lam = qo_power_lambda(S, p, power_iters);
    double eta = 1.0 / (2.0 * lam);
    if (eta_out)
        *eta_out = eta;

    for (int t = 0; t < iters; ++t) {
        /* CD sweep with W replaced by W - H */
#pragma omp parallel for schedule(dynamic)
        for (int64_t i = 0; i < q; ++i) {
            double *tgt = (double *)malloc((size_t)p * sizeof(double));
            double *TS = (double *)malloc((size_t)p * sizeof(double));
            double *WS = (double *)malloc((size_t)p * sizeof(double));
            for (int64_t j = 0; j < p; ++j)
                tgt[j] = W[i * p + j] - H[i * p + j];
            qo_row_times_sigma(tgt, &Sg, p, TS, NULL);
            qo_row_times_sigma(Wh + i * p, &Sg, p, WS, NULL);
            qo_sweep_row(&Sg, p, scale + i, zero + i, p, maxq, tgt, TS, Wh + i * p, WS,
                         NULL, codes + i * p, NULL, NULL, 0);
            free(tgt); free(TS); free(WS);
        }
        qo_objective_rows(W, H, codes, scale, zero, q, p, S, rows);
        double g = 0.0;
        for (int64_t i = 0; i < q; ++i)
            g += rows[i];
        if (obj_cd)
            obj_cd[t] = g;

        /* gradient step and hard thresholding */
#pragma omp parallel for schedule(dynamic)
        for (int64_t i = 0; i < q; ++i) {
            double *D = (double *)malloc((size_t)p * sizeof(double));
            double *G = (double *)malloc((size_t)p * sizeof(double));
            for (int64_t j = 0; j < p; ++j)
                D[j] = H[i * p + j] + Wh[i * p + j] - W[i * p + j];
            qo_row_times_sigma(D, &Sg, p, G, NULL);  /* G/2 = (H + What - W) Sigma */
            for (int64_t j = 0; j < p; ++j)
                T[i * p + j] = H[i * p + j] - eta * 2.0 * G[j];
            free(D); free(G);
        }
        nnz = qo_select(T, q, p, s_budget, structured, idx, cols);
        memset(H, 0, (size_t)N * sizeof(double));
        for (int64_t k = 0; k < nnz; ++k)
            H[idx[k]] = T[idx[k]];

        qo_objective_rows(W, H, codes, scale, zero, q, p, S, rows);
        g = 0.0;
        for (int64_t i = 0; i < q; ++i)
            g += rows[i];
        if (obj)
            obj[t] = g;
    }
    if (nnz_out)
        *nnz_out = nnz;
    free(idx); free(cols); free(excl); free(Wh); free(T); free(rows);
    return 0;
}

/*
 * One IHT half-step of Algorithm 4 entered from a given state: the codes on the
 * grid (scale, zero) give What, H is the current outlier matrix (dense q*p), and
 *   G = 2 (H + What - W) Sigma,   T = H - eta G,   H_new = P_s(T)
 * (the column selection of qo_topk_columns with `structured`).  Writes T (q*p)
 * and the support of H_new (ascending linear indices, at most s_budget entries;
 * H_new = T there) and returns its size.  These are the steps of the IHT half of
 * qo_quantease_outlier; a test uses them to replay another implementation's
 * iterations one at a time from that implementation's own state.
 */
int64_t qo_iht_step(const double *W, int64_t q, int64_t p, const double *S, const uint8_t *codes,
                    const float *scale, const float *zero, const double *H, double eta,
                    int64_t s_budget, int structured, double *T, int64_t *idx)
{
    const qo_sig Sg = {S, NULL, p};
    int64_t *cols = (int64_t *)malloc((size_t)(p > 0 ? p : 1) * sizeof(int64_t));
    if (!cols)
        return -1;
#pragma omp parallel for schedule(dynamic)
    for (int64_t i = 0; i < q; ++i) {
        double *D = (double *)malloc((size_t)p * sizeof(double));
        double *G = (double *)malloc((size_t)p * sizeof(double));
        for (int64_t j = 0; j < p; ++j)
            D[j] = H[i * p + j] + qo_level(codes[i * p + j], scale[i], zero[i]) - W[i * p + j];
        qo_row_times_sigma(D, &Sg, p, G, NULL);  /* G/2 = (H + What - W) Sigma */
        for (int64_t j = 0; j < p; ++j)
            T[i * p + j] = H[i * p + j] - 2.0 * eta * G[j];   /* 2 eta = eta 2 exactly */
        free(D); free(G);
    }
    const int64_t nnz = qo_select(T, q, p, s_budget, structured, idx, cols);
    free(cols);
    return nnz;
}
