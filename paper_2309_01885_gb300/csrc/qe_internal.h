// Host-side declarations shared by the translation units of libqe.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace qe {

// Epilogues of the tensor-core GEMM  D[M x N] = sum over products of A_pa . B_pb^T.
enum EpiMode : int {
    EPI_SIGMA = 0,  // out[r][c] (=|+=) D, only c >= r, mirrored to out[c][r]
    EPI_PINIT = 1,  // out[r][c] = W[r][c] + D            (P = W (I + Sigma_bar))
    EPI_RFULL = 2,  // out[r][c] = P[r][c] / s_r - D + z_r  (R = P - What Sigma_bar in grid steps)
    EPI_TRAIL = 3   // out[split][r][c] = D               (split-K partial sums)
};

struct GemmArgs {
    int M, N;                 // extent of the output window
    int kb_begin, kb_count;   // 64-wide k-blocks covered (split evenly over gridDim.z)
    int n_prod;               // products per k-block (1..6)
    int prod_a[6], prod_b[6]; // operand plane of each product
    int a_plane_rows, b_plane_rows;  // row distance between stacked planes in the maps
    int a_row0, b_row0;       // row offsets of the operand windows
    int mode;
    int m_fast;               // grid x runs over M tiles (B slices shared within a wave)
    float *out;
    int64_t ldo;
    int64_t split_stride;     // EPI_TRAIL: elements between split slices
    const float *P;           // EPI_RFULL
    int64_t ldp;
    const float *scale;       // EPI_RFULL
    const void *W;            // EPI_PINIT
    int w_is_bf16;
    int64_t ldw;
    int accumulate;           // EPI_SIGMA
    // EPI_RFULL, optional fused objective f = sum D_ij d_j (R_ij - What_ij) with
    // What = s (codes - z) and D = W - What (- H): one fp64 partial per epilogue
    // warp and tile, at obj_part[(tile * 8) + warp - 2].
    double *obj_part;
    const uint8_t *codes;
    int64_t ldc;
    const float *zero;
    // EPI_RFULL with grouped grids: scale / zero per row and group of gsize columns
    // ([r * ngroups + c / gsize]; ngroups = 1: per row), and absolute = 1: the A operand
    // is s_g (C - z_g), so R = (P - acc) / s_g + z_g
    int64_t gsize, ngroups;
    int absolute;
    const float *dvec;
    const float *Hd;
    int64_t ldh;
    unsigned *err;
    // optional gate: the launch does its work only when *gate == gate_run (the
    // adaptive sweep schedule enqueues both forms of a sweep and runs one)
    const int *gate;
    int gate_run;
    // f16 = 1: both operands are fp16 (kind::f16 with f16 inputs) instead of bf16;
    // colscale (EPI_TRAIL, EPI_RFULL; may be NULL): output column c of the window is
    // multiplied by colscale[c] (a power of two undoing the B operand's row scaling)
    int f16;
    const float *colscale;
    float ascale;             // with colscale: a further factor (a power of two) on every output
    const float *rowscale;    // EPI_PINIT (may be NULL): output row r is multiplied by rowscale[r]
};

// The per-device error word that qe_sync_status reads and clears.
unsigned *device_error_word();

// Builds a 2-D bf16 tensor map (rows x cols, leading dimension ld elements) with
// a box of 64 columns x box_rows rows and 128-byte swizzle.  false on failure.
bool make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols,
                    uint64_t ld, uint32_t box_rows);
// The same for fp16 elements.
bool make_tmap_f16(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols,
                   uint64_t ld, uint32_t box_rows);

// Launches the tcgen05 GEMM with BN in {64, 128, 256} output columns per CTA.
// grid = (ceil(N / BN), ceil(M / 128), splits).
cudaError_t launch_tc_gemm(int BN, const CUtensorMap &ta, const CUtensorMap &tb,
                           const GemmArgs &g, int splits, cudaStream_t s);

// fp32 SIMT Sigma for fp32 X with arbitrary strides: X(feature a, token k) at
// X[a * sa + k * sk].
cudaError_t launch_sigma_f32(const float *X, int64_t p, int64_t n, int64_t sa, int64_t sk,
                             float *S, int accumulate, cudaStream_t s);

// Token-major bf16 X (n x p, ld) -> feature-major chunk (p x nc, ld_out).
cudaError_t launch_transpose_bf16(const void *X, int64_t n0, int64_t nc, int64_t p, int64_t ldx,
                                  void *out, int64_t ld_out, cudaStream_t s);

}  // namespace qe
