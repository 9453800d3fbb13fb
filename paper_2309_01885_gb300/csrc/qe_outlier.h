// Launchers of the outlier-aware kernels (Sec. 4.3, Algorithm 4).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace qe {

// Device-side state of the radix select behind P_s.
constexpr int kTopkBins = 2048;   // digit bins of the first two passes (the third has 512)
struct TopkState {
    unsigned hist[3][kTopkBins];   // per digit pass (zeroed by the launcher)
    unsigned ticket[3];            // CTAs done with each pass
    unsigned prefix;               // key bits fixed so far
    unsigned remaining;            // keys still to take from the current bucket
    unsigned empty;
    unsigned long long count_gt;
    unsigned kstar;      // the s-th largest nonzero key (0xffffffff: nothing kept)
    unsigned need_eq;    // keys == kstar to keep, in ascending linear index
};

// part: 2 * kPowerMaxBlocks doubles (the per-CTA partial norms carried between steps).
constexpr int kPowerMaxBlocks = 1024;
cudaError_t launch_power_lambda(const float *S, int64_t lds, int64_t p, int iters, float *y0, float *y1,
                                double *part, double *lam, double *eta, int nsm, cudaStream_t s);
cudaError_t launch_iht_target(const float *H, const float *R, int64_t ld, const uint8_t *codes,
                              int64_t ldc, const float *scale, const float *zero, const float *d,
                              const double *eta, int64_t q, int64_t p, float *T, cudaStream_t s);
cudaError_t launch_flat_copy(const void *W, int w_bf16, int64_t ldw, int64_t q, int64_t p, float *T,
                             cudaStream_t s);
int64_t topk_chunks(int64_t N);
cudaError_t launch_topk(const float *T, int64_t N, int64_t s_budget, TopkState *st, unsigned *cnt_gt,
                        unsigned *cnt_eq, unsigned *sel_base, unsigned *eq_base, int64_t *H_idx,
                        float *H_val, int64_t *nnz, int nsm, cudaStream_t s);
// Structured outliers (Sec. 4.3): the k columns of T with the largest l2 norm
// (ties: smaller index; zero columns never kept), emitted as every entry of those
// columns in ascending linear order (nnz = q x kept columns).  part: colnorm_chunks(q)
// x p doubles; norm2, colval: p floats; cols: p indices; ncols: one.
int colnorm_chunks(int64_t q);
cudaError_t launch_topk_columns(const float *T, int64_t q, int64_t p, int64_t k, TopkState *st, unsigned *cnt_gt,
                                unsigned *cnt_eq, unsigned *sel_base, unsigned *eq_base, double *part,
                                float *norm2, int64_t *cols, float *colval, int64_t *ncols, int64_t *H_idx,
                                float *H_val, int64_t *nnz, int nsm, cudaStream_t s);
cudaError_t launch_scatter_rowptr(const int64_t *H_idx, const float *H_val, const int64_t *nnz,
                                  int64_t cap, int64_t q, int64_t p, float *H, int64_t ld,
                                  int64_t *rowptr, cudaStream_t s);
cudaError_t launch_spmm_refresh(const float *PW, float *P, float *R, int64_t ld, const float *sbar,
                                int64_t lds, const int64_t *H_idx, const float *H_val, const int64_t *rowptr,
                                int64_t q, int64_t p, int update_r, const float *scale, cudaStream_t s);
cudaError_t launch_dinv(const float *d, int64_t p, float *dinv, cudaStream_t s);

}  // namespace qe
