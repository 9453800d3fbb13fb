// Streaming and sequential kernels of the QuantEase CD path (Sec. 3.2):
// per-row grid, Sigma normalisation into bf16 hi/lo planes of Sigma_bar^T,
// the in-block sequential column updates (Lemma 1, Eq. cd-update-closed-2),
// the objective reduction, plus the fp32 SIMT Sigma and the bf16 transpose.
#include "qe_common.cuh"
#include "qe_internal.h"
#include <cuda_fp16.h>

#include "qe_kernels.h"

namespace qe {

__device__ __forceinline__ float load_elem(const void *base, int is_bf16, int64_t idx) {
    if (is_bf16) return __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(base)[idx]);
    return reinterpret_cast<const float *>(base)[idx];
}

// ---------------------------------------------------------------------------
// Grid (Sec. 2.1): asymmetric per-row min/max with 0 in range, binary32.
// One CTA of 256 threads per row.  Optional H (dense) is subtracted first, so
// that the entries held by H (exactly equal to W there) leave the pool
// (Sec. 4.3).  Non-finite entries latch ERR_NUMERIC.
// ---------------------------------------------------------------------------
// Grouped grids: CTA (i, g) takes the columns of group g only and writes entry
// i * gridDim.y + g.
__global__ void __launch_bounds__(256) k_grid(const void *W, int w_bf16, int64_t ldw, const float *H,
                                              int64_t ldh, int64_t p, int64_t gsize, float maxq, float *scale,
                                              float *zero, unsigned *err) {
    const int64_t i = blockIdx.x;
    const int64_t j0 = static_cast<int64_t>(blockIdx.y) * gsize;
    const int64_t j1 = (j0 + gsize) < p ? (j0 + gsize) : p;
    float lo = 0.0f, hi = 0.0f;
    bool bad = false;
    for (int64_t j = j0 + threadIdx.x; j < j1; j += blockDim.x) {
        float w = load_elem(W, w_bf16, i * ldw + j);
        if (!isfinite(w)) bad = true;
        if (H) w = w - H[i * ldh + j];
        lo = fminf(lo, w);
        hi = fmaxf(hi, w);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        lo = fminf(lo, __shfl_xor_sync(0xffffffffu, lo, o));
        hi = fmaxf(hi, __shfl_xor_sync(0xffffffffu, hi, o));
    }
    __shared__ float slo[8], shi[8];
    __shared__ int sbad;
    if (threadIdx.x == 0) sbad = 0;
    __syncthreads();
    if (bad) sbad = 1;
    if ((threadIdx.x & 31) == 0) {
        slo[threadIdx.x >> 5] = lo;
        shi[threadIdx.x >> 5] = hi;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int w = 1; w < (int)(blockDim.x >> 5); ++w) {
            lo = fminf(lo, slo[w]);
            hi = fmaxf(hi, shi[w]);
        }
        if (lo == 0.0f && hi == 0.0f) {
            lo = -1.0f;
            hi = 1.0f;
        }
        const float s = __fdiv_rn(__fsub_rn(hi, lo), maxq);
        const float z = rintf(__fdiv_rn(-lo, s));
        scale[i * gridDim.y + blockIdx.y] = s;
        zero[i * gridDim.y + blockIdx.y] = z;
        if (sbad) set_error(err, ERR_NUMERIC);
    }
}

// ---------------------------------------------------------------------------
// Sigma normalisation (Algorithm 3 initialisation, footnote of Lemma 1):
// d_j = Sigma_jj; a column with d_j <= 0 is dead.  SnT = Sigma_bar^T with
// SnT[j][k] = Sigma[j][k] / d_j for k != j and j, k alive, 0 otherwise; this is
// Sigma_bar[k][j] = Sigma[k][j] / Sigma_jj of the column-normalised matrix with
// zero diagonal.  Stored as three bf16 planes hi, mid, lo (rows [0, p), [p, 2p),
// [2p, 3p)) whose sum carries the 24 significant bits of the fp32 value.
// ---------------------------------------------------------------------------
__global__ void k_sigma_diag(const float *S, int64_t lds, int64_t p, float *d, unsigned *err) {
    const int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (j >= p) return;
    const float v = S[j * lds + j];
    if (!isfinite(v)) set_error(err, ERR_NUMERIC);
    d[j] = v;
}

// The hi/mid/lo split of one binary32 value.
__device__ __forceinline__ void split3(float x, __nv_bfloat16 &h, __nv_bfloat16 &m, __nv_bfloat16 &l) {
    h = __float2bfloat16_rn(x);
    const float r1 = x - __bfloat162float(h);
    m = __float2bfloat16_rn(r1);
    l = __float2bfloat16_rn(r1 - __bfloat162float(m));
}

// One CTA per row j of Sigma (grid.y), 4 consecutive columns k per thread:
// 16-byte reads of Sigma and d, 8-byte writes of each plane.
__global__ void __launch_bounds__(256) k_sigma_planes(const float *S, int64_t lds, int64_t p, const float *d,
                                                      __nv_bfloat16 *snt, int64_t ldn, unsigned *err) {
    bool bad = false;
    const bool vec = (lds % 4 == 0) && ((reinterpret_cast<uintptr_t>(S) & 15u) == 0);
    for (int64_t j = blockIdx.y; j < p; j += gridDim.y) {
        const float dj = d[j];
        const bool jalive = dj > 0.0f;
        for (int64_t k0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) * 4; k0 < p;
             k0 += (int64_t)gridDim.x * blockDim.x * 4) {
            float sv[4], dk[4];
            if (vec && k0 + 4 <= p) {
                const float4 a = *reinterpret_cast<const float4 *>(S + j * lds + k0);
                const float4 b = *reinterpret_cast<const float4 *>(d + k0);
                sv[0] = a.x; sv[1] = a.y; sv[2] = a.z; sv[3] = a.w;
                dk[0] = b.x; dk[1] = b.y; dk[2] = b.z; dk[3] = b.w;
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    sv[e] = (k0 + e < p) ? S[j * lds + k0 + e] : 0.0f;
                    dk[e] = (k0 + e < p) ? d[k0 + e] : 0.0f;
                }
            }
            __nv_bfloat16 h[4], m[4], l[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int64_t k = k0 + e;
                if (k < p && !isfinite(sv[e])) bad = true;
                float x = 0.0f;
                if (k < p && jalive && k != j && dk[e] > 0.0f) x = __fdiv_rn(sv[e], dj);
                split3(x, h[e], m[e], l[e]);
            }
            __nv_bfloat16 *r0 = snt + j * ldn + k0;
            __nv_bfloat16 *r1 = snt + (p + j) * ldn + k0;
            __nv_bfloat16 *r2 = snt + (2 * p + j) * ldn + k0;
            if (k0 + 4 <= p) {   // ldn is a multiple of 64, k0 of 4: 8-byte aligned
                *reinterpret_cast<uint2 *>(r0) = make_uint2(
                    (uint32_t)__bfloat16_as_ushort(h[0]) | ((uint32_t)__bfloat16_as_ushort(h[1]) << 16),
                    (uint32_t)__bfloat16_as_ushort(h[2]) | ((uint32_t)__bfloat16_as_ushort(h[3]) << 16));
                *reinterpret_cast<uint2 *>(r1) = make_uint2(
                    (uint32_t)__bfloat16_as_ushort(m[0]) | ((uint32_t)__bfloat16_as_ushort(m[1]) << 16),
                    (uint32_t)__bfloat16_as_ushort(m[2]) | ((uint32_t)__bfloat16_as_ushort(m[3]) << 16));
                *reinterpret_cast<uint2 *>(r2) = make_uint2(
                    (uint32_t)__bfloat16_as_ushort(l[0]) | ((uint32_t)__bfloat16_as_ushort(l[1]) << 16),
                    (uint32_t)__bfloat16_as_ushort(l[2]) | ((uint32_t)__bfloat16_as_ushort(l[3]) << 16));
            } else {
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (k0 + e < p) {
                        r0[e] = h[e];
                        r1[e] = m[e];
                        r2[e] = l[e];
                    }
            }
        }
    }
    if (bad) set_error(err, ERR_NUMERIC);
}

// Sigma_bar^T in two fp16 planes for the CD GEMMs whose other operand is an
// exact small integer (the changes Delta' of a window sweep, C - z of the
// residual refresh): row j (Sigma_bar[:, j]) is scaled by a power of two 2^e_j
// that brings its largest magnitude just under 2^15, then split as
// hi = fp16(x), lo = fp16(x - hi): 22 significant bits (relative 2^-22) at one
// product fewer than three bf16 planes; the GEMM epilogue multiplies output
// column j by cscale[j] = 2^-e_j (exact).  x is the same binary32 value the bf16
// planes and the fp32 rows hold.  One CTA per row j (grid-stride), two passes
// over the row (its largest magnitude, then the planes).
__global__ void __launch_bounds__(256) k_sigma_planes_h2(const float *S, int64_t lds, int64_t p, const float *d,
                                                         __half *snh, int64_t ldn, float *cscale) {
    __shared__ float red[8];
    for (int64_t j = blockIdx.x; j < p; j += gridDim.x) {
        const float dj = d[j];
        const bool jalive = dj > 0.0f;
        float mx = 0.0f;
        for (int64_t k = threadIdx.x; k < p; k += blockDim.x)
            if (jalive && k != j && d[k] > 0.0f) mx = fmaxf(mx, fabsf(__fdiv_rn(S[j * lds + k], dj)));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
        __syncthreads();
        mx = 0.0f;
        for (int w = 0; w < 8; ++w) mx = fmaxf(mx, red[w]);
        __syncthreads();   // red is rewritten for the next row
        // 2^e with mx 2^e in [2^14, 2^15) (finite mx; e = 0 for an all-zero row)
        int e = 0;
        if (mx > 0.0f && isfinite(mx)) e = 14 - ilogbf(mx);
        if (e > 100) e = 100;
        if (e < -100) e = -100;
        if (threadIdx.x == 0) cscale[j] = ldexpf(1.0f, -e);
        for (int64_t k = threadIdx.x; k < ldn; k += blockDim.x) {
            float x = 0.0f;
            if (k < p && jalive && k != j && d[k] > 0.0f) x = ldexpf(__fdiv_rn(S[j * lds + k], dj), e);
            const __half hi = __float2half_rn(x);
            const __half lo = __float2half_rn(x - __half2float(hi));
            snh[j * ldn + k] = hi;
            snh[(p + j) * ldn + k] = lo;
        }
    }
}

// bf16 W as one fp16 plane for the P GEMM against the fp16 planes of Sigma_bar:
// row i scaled by a power of two 2^e_i that brings its largest magnitude just
// under 2^15 (bf16's 8 significant bits fit fp16's 11, so every entry above
// 2^-14 of that maximum is exact); rscale[i] = 2^-e_i undoes it in the epilogue.
// One CTA per row (grid-stride), columns [p, ld) zero.
__global__ void __launch_bounds__(256) k_w_plane_h1(const __nv_bfloat16 *W, int64_t ldw, int64_t q, int64_t p,
                                                    __half *wh, int64_t ld, float *rscale) {
    __shared__ float red[8];
    for (int64_t i = blockIdx.x; i < q; i += gridDim.x) {
        float mx = 0.0f;
        for (int64_t k = threadIdx.x; k < p; k += blockDim.x) mx = fmaxf(mx, fabsf(__bfloat162float(W[i * ldw + k])));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
        __syncthreads();
        mx = 0.0f;
        for (int w = 0; w < 8; ++w) mx = fmaxf(mx, red[w]);
        __syncthreads();
        int e = 0;
        if (mx > 0.0f && isfinite(mx)) e = 14 - ilogbf(mx);
        if (e > 100) e = 100;
        if (e < -100) e = -100;
        if (threadIdx.x == 0) rscale[i] = ldexpf(1.0f, -e);
        for (int64_t k = threadIdx.x; k < ld; k += blockDim.x)
            wh[i * ld + k] = __float2half_rn(k < p ? ldexpf(__bfloat162float(W[i * ldw + k]), e) : 0.0f);
    }
}

cudaError_t launch_w_plane_h1(const void *W, int64_t ldw, int64_t q, int64_t p, __half *wh, int64_t ld, float *rscale,
                              cudaStream_t s) {
    const int64_t g = q < 65535 ? q : 65535;
    k_w_plane_h1<<<static_cast<unsigned>(g), 256, 0, s>>>(static_cast<const __nv_bfloat16 *>(W), ldw, q, p, wh, ld,
                                                          rscale);
    return cudaGetLastError();
}

// Sigma_bar in fp32, row-major (row k, column j): Sigma_bar[k][j] =
// Sigma[j][k] / d_j, the same binary32 value whose hi + mid + lo planes
// k_sigma_planes writes (so the change-list correction and the tensor-core
// correction multiply the same matrix).  Row k holds what a change of column k
// adds to the other columns, contiguous over j.  Columns [p, ld) are zero.
// 32 x 32 tiles transposed through shared memory; grid (ld / 32, p / 32).
__global__ void __launch_bounds__(256) k_sigma_bar_rows(const float *S, int64_t lds, int64_t p, const float *d,
                                                        float *sbar, int64_t ld) {
    __shared__ float tile[32][33];
    const int64_t j0 = static_cast<int64_t>(blockIdx.x) * 32, k0 = static_cast<int64_t>(blockIdx.y) * 32;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    // load: S[j][k] for j in [j0, j0+32) (rows), k = k0 + tx (coalesced)
    for (int r = ty; r < 32; r += 8) {
        const int64_t j = j0 + r, k = k0 + tx;
        float x = 0.0f;
        if (j < p && k < p) {
            const float dj = d[j];
            if (dj > 0.0f && k != j && d[k] > 0.0f) x = __fdiv_rn(S[j * lds + k], dj);
        }
        tile[r][tx] = x;
    }
    __syncthreads();
    // store: sbar[k][j] for k in [k0, k0+32), j = j0 + tx (coalesced)
    for (int r = ty; r < 32; r += 8) {
        const int64_t k = k0 + r, j = j0 + tx;
        if (k < p && j < ld) sbar[k * ld + j] = tile[tx][r];
    }
}

// ---------------------------------------------------------------------------
// Operand planes of a q x p matrix for the tensor-core GEMM (rows [0,q) = hi,
// [q, 2q) = mid, [2q, 3q) = lo when split).  fp32 input splits into three bf16
// planes; bf16 input is copied (exact in one plane).
// ---------------------------------------------------------------------------
__global__ void k_make_planes(const void *W, int w_bf16, int64_t ldw, int64_t q, int64_t p,
                              int split, __nv_bfloat16 *out, int64_t ldo) {
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < p;
             j += (int64_t)gridDim.x * blockDim.x) {
            const float w = load_elem(W, w_bf16, i * ldw + j);
            const __nv_bfloat16 h = __float2bfloat16_rn(w);
            out[i * ldo + j] = h;
            if (split) {
                const float r1 = w - __bfloat162float(h);
                const __nv_bfloat16 m = __float2bfloat16_rn(r1);
                out[(q + i) * ldo + j] = m;
                out[(2 * q + i) * ldo + j] = __float2bfloat16_rn(r1 - __bfloat162float(m));
            }
        }
    }
}

// The residual at the start of the first sweep, in grid-step units: with
// What = W - H, P - What Sigma_bar = (W - H)(I + Sigma_bar) - (W - H) Sigma_bar
// = W - H, stored as (W - H) / s + z.
__global__ void k_init_residual(const void *W, int w_bf16, int64_t ldw, const float *H, int64_t ldh,
                                int64_t q, int64_t p, int64_t gsize, const float *scale, const float *zero,
                                float *R, int64_t ldr) {
    const int64_t ng = ceil_div(p, gsize);   // the 4 columns of a thread lie in one group (gsize = p or % 64 == 0)
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        for (int64_t j0 = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) * 4; j0 < p;
             j0 += (int64_t)gridDim.x * blockDim.x * 4) {
            const float s = scale[i * ng + j0 / gsize], z = zero[i * ng + j0 / gsize];
            float o[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int64_t j = j0 + e;
                float w = 0.0f;
                if (j < p) {
                    w = load_elem(W, w_bf16, i * ldw + j);
                    if (H) w -= H[i * ldh + j];
                }
                o[e] = __fdiv_rn(w, s) + z;
            }
            float *rr = R + i * ldr + j0;
            if (j0 + 4 <= p) *reinterpret_cast<float4 *>(rr) = make_float4(o[0], o[1], o[2], o[3]);   // ldr % 64 == 0
            else
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    if (j0 + e < p) rr[e] = o[e];
        }
    }
}

// obj_out = obj_prev + sum_i rowdf[i] (fixed order); rowdf is cleared.
__global__ void k_obj_step(double *rowdf, int64_t q, const double *prev, double *out, const int *gate,
                           int gate_run) {
    if (gate && *gate != gate_run) return;
    __shared__ double sw[32];
    double acc = 0.0;
    for (int64_t k = threadIdx.x; k < q; k += blockDim.x) {
        acc += rowdf[k];
        rowdf[k] = 0.0;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) sw[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = prev ? *prev : 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += sw[w];
        *out = t;
    }
}

// (C - z) as bf16 (exact: |C - z| <= 255) for the R = P - s (C - z) Sigma_bar GEMM.
__global__ void k_codes_to_qf(const uint8_t *codes, int64_t ldc, const float *scale, const float *zero,
                              int64_t q, int64_t p, int64_t gsize, int grouped, __nv_bfloat16 *qf, int64_t ldq) {
    const int64_t ng = ceil_div(p, gsize);
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < p;
             j += (int64_t)gridDim.x * blockDim.x) {
            const int64_t gi = i * ng + j / gsize;
            const float cz = static_cast<float>(codes[i * ldc + j]) - zero[gi];
            if (!grouped) {   // exact in fp16: the residual GEMM takes fp16 operands
                reinterpret_cast<__half *>(qf)[i * ldq + j] = __float2half_rn(cz);
            } else {
                __nv_bfloat16 h, m, l;
                split3(scale[gi] * cz, h, m, l);
                qf[i * ldq + j] = h;
                qf[(q + i) * ldq + j] = m;
                qf[(2 * q + i) * ldq + j] = l;
            }
        }
    }
}

// ---------------------------------------------------------------------------
// In-block sequential CD (Algorithm 3 inner loop, one column block of width B).
// One warp per row i (rows are independent, Sec. 3.2); the lanes hold the
// block's columns and the decisions travel by warp shuffles.  Work in units of the
// grid step: t_ij = beta_ij / s_i + z_i, so the code is rint(clamp(t, 0, 2^b-1))
// (the nearest level, Eq. eq:quant) and the column change is
// Delta'_ij = (What_start_ij - What_new_ij) / s_i = a_ij - c_ij with
// a_ij = What_start_ij / s_i + z_i (an integer code after the first sweep).
// On entry t for column l of the block is
//     R_il / s_i + z_i + sum_split partial[split][i][l]
// (R = P - What_start Sigma_bar, partial = Delta'[:, 0:b0] Sigma_bar[0:b0, block]);
// the in-block contributions Delta'_ij Sigma_bar_jl (j < l in the block) are
// added here, right after column j is decided.
// ---------------------------------------------------------------------------
// Packed strict upper triangle of a diagonal B x B block of Sigma_bar:
// row j holds columns j+1 .. B-1 at kPackPad + tri_off(j) + (l - j - 1).  The
// kPackPad floats in front keep the harmless reads of already-decided columns
// (l <= j, see the kernels below) inside the array.
constexpr int kPackPad = 32;
__host__ __device__ constexpr int tri_off(int B, int j) { return j * B - (j * (j + 1)) / 2; }
__host__ __device__ constexpr int packed_block_floats(int B) {
    return static_cast<int>(round_up(kPackPad + B * (B - 1) / 2, 4));
}

// One diagonal block per grid row: Sigma_bar[b0 + j][b0 + l] (l > j) from the
// hi + mid + lo planes (the same values the tensor-core GEMMs use).
__global__ void k_pack_diag(const __nv_bfloat16 *snt, int64_t ldn, int64_t plane_rows, int64_t p, int B,
                            float *out) {
    const int bi = blockIdx.x, j = blockIdx.y;
    const int64_t b0 = static_cast<int64_t>(bi) * B;
    float *blk = out + static_cast<int64_t>(bi) * packed_block_floats(B);
    const int64_t pl = plane_rows * ldn;
    if (j == 0 && threadIdx.x < kPackPad) blk[threadIdx.x] = 0.0f;
    for (int l = j + 1 + threadIdx.x; l < B; l += blockDim.x) {
        float v = 0.0f;
        if (b0 + j < p && b0 + l < p) {
            const int64_t o = (b0 + l) * ldn + b0 + j;
            v = __bfloat162float(snt[o]) + __bfloat162float(snt[pl + o]) + __bfloat162float(snt[2 * pl + o]);
        }
        blk[kPackPad + tri_off(B, j) + (l - j - 1)] = v;
    }
}

template <int B>
struct CdCfg {
    static constexpr int CPL = B / 32;                    // columns owned by each lane
    static constexpr int MAX_WARPS = 32;                  // rows per CTA (one row per warp)
    static constexpr int PACK = packed_block_floats(B);
    static constexpr int SMEM = PACK * 4 + 16;            // packed block + its mbarrier
    static constexpr int MAX_SPLITS = 16;
};

// Cross-block correction from the change lists (the sparse form of the
// trailing GEMM, used once few codes change per sweep): for every column block
// (this one included) the changes of its most recent visit, each adding
// Delta'_ik Sigma_bar[k][block] to the row; Sigma_bar rows are fp32 and
// contiguous over the block, so each change is one coalesced read of B floats
// per warp.  Returns whether the row had any change in the window.  Lists of
// blocks below bmin are left out.
template <int B, bool FULL, int U = 4, bool GR = false>
__device__ __forceinline__ bool list_correction(const CdArgs &a, int64_t b0, int bw_, int64_t ii, bool row_ok,
                                                int lane, float (&ps)[B / 32], int bmin = 0) {
    constexpr int CPL = B / 32;
    const int bw = FULL ? B : bw_;
    const int64_t rb = ii * a.nblk;
    const float *sb0 = a.sbar + b0 + lane;
    bool any = false;
    for (int c0 = 0; c0 < a.nblk; c0 += 32) {
        const int cnt = (row_ok && c0 + lane < a.nblk && c0 + lane >= bmin) ? a.lcnt[rb + c0 + lane] : 0;
        unsigned m = __ballot_sync(0xffffffffu, cnt > 0);
        any = any || m != 0u;
        while (m != 0u) {
            const int sl = __ffs(m) - 1;
            m &= m - 1u;
            const int c = __shfl_sync(0xffffffffu, cnt, sl);
            const int64_t blk2 = c0 + sl;
            const uint32_t *seg = a.lent + (rb + blk2) * B;
            const float *sbk = sb0 + blk2 * B * a.lds;
            // grouped grids: the listed changes are in the grid units of their own group
            float fac = 1.0f;
            if (GR) fac = __fdiv_rn(a.scale[ii * a.ngroups + blk2 * B / a.gsize], a.scale[ii * a.ngroups + b0 / a.gsize]);
            for (int e0 = 0; e0 < c; e0 += 32) {
                const uint32_t mine = (e0 + lane < c) ? seg[e0 + lane] : 0u;
                const int ne = (c - e0) < 32 ? (c - e0) : 32;
                // U changes in flight per step (the gather is bound by loads in flight);
                // the sum still runs over the changes in list order
                int u = 0;
                for (; u + U <= ne; u += U) {
                    const float *r[U];
                    float dv[U];
#pragma unroll
                    for (int e = 0; e < U; ++e) {
                        const uint32_t ev = __shfl_sync(0xffffffffu, mine, u + e);
                        r[e] = sbk + static_cast<int64_t>(ev & 0xffffu) * a.lds;
                        dv[e] = static_cast<float>(static_cast<int16_t>(ev >> 16)) * fac;
                    }
                    float v[U][CPL];
#pragma unroll
                    for (int e = 0; e < U; ++e)
#pragma unroll
                        for (int h = 0; h < CPL; ++h)
                            v[e][h] = (FULL || 32 * h + lane < bw) ? __ldg(r[e] + 32 * h) : 0.0f;
#pragma unroll
                    for (int h = 0; h < CPL; ++h)
#pragma unroll
                        for (int e = 0; e < U; ++e) ps[h] = fmaf(dv[e], v[e][h], ps[h]);
                }
                for (; u < ne; ++u) {
                    const uint32_t e1 = __shfl_sync(0xffffffffu, mine, u);
                    const float *r1 = sbk + static_cast<int64_t>(e1 & 0xffffu) * a.lds;
                    const float d1 = static_cast<float>(static_cast<int16_t>(e1 >> 16)) * fac;
#pragma unroll
                    for (int h = 0; h < CPL; ++h)
                        if (FULL || 32 * h + lane < bw) ps[h] = fmaf(d1, __ldg(r1 + 32 * h), ps[h]);
                }
            }
        }
    }
    return any;
}

// Common prologue of both in-block kernels: start the bulk copy of the packed
// block, stage the row (t = R + sum of split partials, R already in grid-step
// units; st = start value: R itself in the first sweep, else the old code),
// optionally store t back as the block's new base (rolling window), then wait
// for the block.  Lane l holds columns 32 h + l.
template <int B, bool FULL>
__device__ __forceinline__ bool cd_prologue(const CdArgs &a, float *tri, uint64_t *bar, int64_t i,
                                            bool row_ok, int lane, float (&t)[B / 32], float (&st)[B / 32]) {
    using C = CdCfg<B>;
    constexpr int CPL = C::CPL;
    const int bw = FULL ? B : a.bw;
    const int64_t b0 = a.b0;
    if (threadIdx.x == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !a.skip_copy) {
        constexpr uint32_t bytes = C::PACK * 4;
        mbar_arrive_expect_tx(bar, bytes);
        bulk_load(tri, a.tri + (b0 / B) * C::PACK, bytes, bar);
    }
    const int64_t ii = row_ok ? i : 0;
    float r_[CPL], ps[CPL];
    uint32_t cd_[CPL];
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        const int l = 32 * h + lane;
        const bool ok = row_ok && (FULL || l < bw);
        r_[h] = ok ? a.R[ii * a.ldr + b0 + l] : 0.0f;
        cd_[h] = (ok && !a.first_sweep && !a.vstart) ? a.codes[ii * a.ldc + b0 + l] : 0u;
        ps[h] = 0.0f;
    }
#pragma unroll
    for (int sp = 0; sp < C::MAX_SPLITS; ++sp) {
        if (sp >= a.nsplit) break;
        const float *prow = a.part + sp * a.part_stride + ii * a.ldpart;
#pragma unroll
        for (int h = 0; h < CPL; ++h)
            if (row_ok && (FULL || 32 * h + lane < bw)) ps[h] += prow[32 * h + lane];
    }
    const bool changed = a.nsplit > 0;
    if (a.grouped && changed) {   // absolute partials: into the grid units of the block's group
        const float sg = a.scale[ii * a.ngroups + b0 / a.gsize];
#pragma unroll
        for (int h = 0; h < CPL; ++h) ps[h] = __fdiv_rn(ps[h], sg);
    }
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        st[h] = a.first_sweep ? r_[h]
                : (a.vstart ? ((row_ok && (FULL || 32 * h + lane < bw)) ? a.vstart[ii * a.ldv + b0 + 32 * h + lane]
                                                                         : 0.0f)
                            : static_cast<float>(cd_[h]));
        t[h] = r_[h] + ps[h];
    }
    if (a.store_base && changed) {
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            if (row_ok && (FULL || l < bw)) a.R[ii * a.ldr + b0 + l] = t[h];
        }
    }
    const unsigned long long lim = a.wait_ns ? a.wait_ns : kWaitLimitNs;
    if (!mbar_wait_bounded_ns(bar, 0u, nullptr, lim)) {
        if (lane == 0) set_error(a.err, ERR_TIMEOUT);
        // a copy that was issued may still land: thread 0 keeps the CTA (and its
        // shared memory) alive until it has, within one more limit
        if (threadIdx.x == 0 && !a.skip_copy) mbar_wait_bounded_ns(bar, 0u, nullptr, lim);
        return false;
    }
    return true;
}

// Common epilogue: codes, C - z (both skipped for unchanged columns when
// skip_same) and the Delta' plane(s).  G = false: never grouped grids (one
// scale per row, no group logic compiled in); G = true: as a.grouped says.
template <int B, bool FULL, bool RECORD, bool G = true>
__device__ __forceinline__ void cd_epilogue(const CdArgs &a, int64_t b0, int bw_, int64_t i, int lane,
                                            const float (&code)[B / 32], const float (&dlt)[B / 32],
                                            bool skip_same) {
    constexpr int CPL = B / 32;
    const int bw = FULL ? B : bw_;
    const bool grouped = G && a.grouped;
    const int64_t gi = G ? i * a.ngroups + b0 / a.gsize : i;   // the block lies in one group
    const float z = a.zero[gi];
    const float sg = grouped ? a.scale[gi] : 1.0f;
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        const int l = 32 * h + lane;
        if (!FULL && l >= bw) continue;
        const int64_t col = b0 + l;
        if (a.vout) {   // relaxed: the value itself, and its nearest level as the code
            a.vout[i * a.ldv + col] = code[h];
            a.codes[i * a.ldc + col] = static_cast<uint8_t>(rintf(fminf(fmaxf(code[h], 0.0f), a.maxq)));
        } else if (!skip_same || dlt[h] != 0.0f) {
            a.codes[i * a.ldc + col] = static_cast<uint8_t>(code[h]);
            if (a.write_qf) {
                if (!grouped) {   // exact in fp16: the residual GEMM takes fp16 operands
                    reinterpret_cast<__half *>(a.qf)[i * a.ldq + col] = __float2half_rn(code[h] - z);
                } else {   // the residual GEMM takes s_g (C - z_g), three planes
                    __nv_bfloat16 qh, qm, ql;
                    split3(sg * (code[h] - z), qh, qm, ql);
                    a.qf[i * a.ldq + col] = qh;
                    a.qf[(a.q + i) * a.ldq + col] = qm;
                    a.qf[(2 * a.q + i) * a.ldq + col] = ql;
                }
            }
        }
        if (!a.dp) continue;
        // grouped: the trailing GEMM sums changes of several groups, so it takes them
        // absolute (s_g Delta'), which is not an integer: three planes
        const float dv = grouped ? sg * dlt[h] : dlt[h];
        if (a.dp_f16 == 1) {   // an integer change, exact in fp16, for the fp16 window GEMM
            reinterpret_cast<__half *>(a.dp)[i * a.ldd + col] = __float2half_rn(dv);
            continue;
        }
        if (a.dp_f16 == 2) {   // a real change (first sweep), scaled by a power of two: fp16 hi / lo
            const float x = dv * a.dp_scale;
            const __half hi = __float2half_rn(x);
            reinterpret_cast<__half *>(a.dp)[i * a.ldd + col] = hi;
            reinterpret_cast<__half *>(a.dp)[(a.dp_plane_rows + i) * a.ldd + col] = __float2half_rn(x - __half2float(hi));
            continue;
        }
        const __nv_bfloat16 hi = __float2bfloat16_rn(dv);
        a.dp[i * a.ldd + col] = hi;
        if (a.frac || grouped) {   // Delta' is not an integer: three planes
            const float r1 = dv - __bfloat162float(hi);
            const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
            a.dp[(a.dp_plane_rows + i) * a.ldd + col] = mid;
            a.dp[(2 * a.dp_plane_rows + i) * a.ldd + col] = __float2bfloat16_rn(r1 - __bfloat162float(mid));
        }
    }
    if (RECORD) {   // this visit's changes replace the block's list (ascending columns)
        __syncwarp();
        const int64_t seg = i * a.nblk + b0 / B;
        uint32_t *ent = a.lent + seg * B;
        int n = 0;
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            const bool ch = (FULL || l < bw) && dlt[h] != 0.0f;
            const unsigned m = __ballot_sync(0xffffffffu, ch);
            if (ch) {
                const int16_t dv = static_cast<int16_t>(__float2int_rn(dlt[h]));
                ent[n + __popc(m & ((1u << lane) - 1u))] =
                    static_cast<uint32_t>(l) | (static_cast<uint32_t>(static_cast<uint16_t>(dv)) << 16);
            }
            n += __popc(m);
        }
        if (lane == 0) a.lcnt[seg] = n;
    }
}

__device__ __forceinline__ double warp_sum(double x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

// ---- near-tie refinement ------------------------------------------------------
// A decision rounds beta~ / s + z (binary32, grid units) to the nearest level; it
// can only come out differently from exact arithmetic when that value lies within
// the binary32 error of a midpoint between two levels.  Such decisions (within
// a.tie_eps, far above that error) are taken again from beta~ recomputed from
// the row's current state, Lemma 1:
//   beta~_j = T_j + sum_{k != j} (T_k - What_k) Sigma_kj / Sigma_jj,  T = W (- H),
// with What_k = s (c_k - z) of the code column k holds at that moment (this
// sweep's for k < j, the previous sweep's for k > j; in the first sweep the
// columns after j still hold T).  One warp-wide pass over the row: every term
// exact, the sum in double-float arithmetic (about 48 significant bits), the
// last steps in binary64, so the decision is that of exact arithmetic except
// within about 1e-9 grid steps of a midpoint.

__device__ __forceinline__ float tie_w(const CdArgs &a, int64_t i, int64_t k) {
    return a.w_bf16 ? __bfloat162float(static_cast<const __nv_bfloat16 *>(a.W)[i * a.ldw + k])
                    : static_cast<const float *>(a.W)[i * a.ldw + k];
}

// beta~ / s + z of column b0 + j of row i, from the row's current
// state.  blk: the warp's shared row with the block's current codes (decided in
// this visit before j, start codes after j; unused after j in the first sweep).
// Warp-collective (every lane calls it; the result is the same in every lane).
// The columns outside the block are read from global memory in 16-byte pieces,
// several pieces per lane in flight, so a pass over a long row takes few round
// trips.  Compiled only into the kernels' refinement variants.
// Error-free transformations (Knuth's two-sum; the fma two-product), for the
// refinement's sums in double-float arithmetic: about 48 significant bits on the
// fp32 pipes (GB300's binary64 rate is a small fraction of its binary32 rate).
__device__ __forceinline__ void ef_two_sum(float a, float b, float &s, float &e) {
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

// (hi, lo) += (t - hs - sg (c - zg)) * sjk in double-float; t, hs, sg, zg, sjk are
// binary32 values and c - zg an exact small integer, so every operand is exact.
__device__ __forceinline__ void df_term(float &hi, float &lo, float t, float hs, float sg, float m, float sjk) {
    const float w1 = __fmul_rn(sg, m);
    const float w2 = fmaf(sg, m, -w1);            // sg m = w1 + w2 exactly
    float u1, u2, d1, e1;
    ef_two_sum(t, -hs, u1, u2);                   // t - hs = u1 + u2 exactly
    ef_two_sum(u1, -w1, d1, e1);
    const float d2 = __fadd_rn(e1, __fsub_rn(u2, w2));
    const float p1 = __fmul_rn(d1, sjk);
    const float p2 = fmaf(d2, sjk, fmaf(d1, sjk, -p1));
    float s1, s2;
    ef_two_sum(hi, p1, s1, s2);
    s2 = __fadd_rn(s2, __fadd_rn(lo, p2));
    hi = __fadd_rn(s1, s2);
    lo = __fsub_rn(s2, __fsub_rn(hi, s1));
}

__device__ __forceinline__ double tie_beta(const CdArgs *ap, int64_t i, int64_t b0, int bw, int j, int lane,
                                        const float *blk) {
    const CdArgs &a = *ap;
    const int64_t jg = b0 + j;
    const float *Srow = a.S + jg * a.lds_full;
    const int64_t kend = a.first_sweep ? b0 : a.p;   // first sweep: later columns still hold T
    const float *sc = a.scale + i * a.ngroups;
    const float *zc = a.zero + i * a.ngroups;
    const bool grouped = a.ngroups > 1;
    const uint32_t gs = static_cast<uint32_t>(a.gsize);
    const uint8_t *crow = a.codes + i * a.ldc;
    const float *hrow = a.Hd ? a.Hd + i * a.ldh : nullptr;
    // Pull the row's data toward L2 first, every line at once (prefetches hold no
    // register), so the summing loop below waits on L2 rather than on DRAM.
    for (int64_t k = 32 * lane; k < kend; k += 32 * 32) prefetch_l2(Srow + k);
    for (int64_t k = 128 * lane; k < kend; k += 128 * 32) prefetch_l2(crow + k);
    if (a.w_bf16) {
        for (int64_t k = 64 * lane; k < kend; k += 64 * 32)
            prefetch_l2(static_cast<const __nv_bfloat16 *>(a.W) + i * a.ldw + k);
    } else {
        for (int64_t k = 32 * lane; k < kend; k += 32 * 32) prefetch_l2(static_cast<const float *>(a.W) + i * a.ldw + k);
    }
    if (hrow)
        for (int64_t k = 32 * lane; k < kend; k += 32 * 32) prefetch_l2(hrow + k);
    float hi = 0.0f, lo = 0.0f;   // the lane's sum, double-float
    // the block's own columns from the shared row
    for (int l = lane; l < bw; l += 32) {
        if (l == j || (a.first_sweep && l > j)) continue;
        const int64_t k = b0 + l;
        const uint32_t g = grouped ? static_cast<uint32_t>(k) / gs : 0u;
        df_term(hi, lo, tie_w(a, i, k), hrow ? hrow[k] : 0.0f, sc[g], blk[l] - zc[g], Srow[k]);
    }
    // the columns outside the block from the row's codes in global memory
    const bool vec = (a.lds_full % 4) == 0 && (a.ldc % 4) == 0 && (a.ldw % 4) == 0 && (!hrow || (a.ldh % 4) == 0) &&
                     ((reinterpret_cast<uintptr_t>(a.S) & 15u) == 0) &&
                     ((reinterpret_cast<uintptr_t>(a.codes) & 3u) == 0) &&
                     ((reinterpret_cast<uintptr_t>(a.W) & (a.w_bf16 ? 7u : 15u)) == 0) &&
                     (!hrow || (reinterpret_cast<uintptr_t>(a.Hd) & 15u) == 0) && (b0 % 4) == 0;
    if (vec) {
#pragma unroll 2
        for (int64_t k = 4 * lane; k < kend; k += 128) {
            if (k >= b0 && k < b0 + bw) continue;   // 4-aligned pieces never straddle the block
            const float4 s4 = *reinterpret_cast<const float4 *>(Srow + k);
            const uint32_t c4 = *reinterpret_cast<const uint32_t *>(crow + k);
            float wv[4];
            if (a.w_bf16) {
                const uint2 r = *reinterpret_cast<const uint2 *>(static_cast<const __nv_bfloat16 *>(a.W) + i * a.ldw + k);
                const __nv_bfloat162 w01 = *reinterpret_cast<const __nv_bfloat162 *>(&r.x);
                const __nv_bfloat162 w23 = *reinterpret_cast<const __nv_bfloat162 *>(&r.y);
                wv[0] = __low2float(w01); wv[1] = __high2float(w01);
                wv[2] = __low2float(w23); wv[3] = __high2float(w23);
            } else {
                const float4 w4 = *reinterpret_cast<const float4 *>(static_cast<const float *>(a.W) + i * a.ldw + k);
                wv[0] = w4.x; wv[1] = w4.y; wv[2] = w4.z; wv[3] = w4.w;
            }
            float hv[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            if (hrow) {
                const float4 h4 = *reinterpret_cast<const float4 *>(hrow + k);
                hv[0] = h4.x; hv[1] = h4.y; hv[2] = h4.z; hv[3] = h4.w;
            }
            const float sv[4] = {s4.x, s4.y, s4.z, s4.w};
            const uint32_t g = grouped ? static_cast<uint32_t>(k) / gs : 0u;   // 4 columns share a group
            const float sg = sc[g], zg = zc[g];
#pragma unroll
            for (int e = 0; e < 4; ++e)
                df_term(hi, lo, wv[e], hv[e], sg, static_cast<float>((c4 >> (8 * e)) & 0xffu) - zg, sv[e]);
        }
    } else {
        for (int64_t k = lane; k < kend; k += 32) {
            if (k >= b0 && k < b0 + bw) continue;
            const uint32_t g = grouped ? static_cast<uint32_t>(k) / gs : 0u;
            df_term(hi, lo, tie_w(a, i, k), hrow ? hrow[k] : 0.0f, sc[g], static_cast<float>(crow[k]) - zc[g], Srow[k]);
        }
    }
    const double acc = warp_sum(static_cast<double>(hi) + static_cast<double>(lo));
    double tj = static_cast<double>(tie_w(a, i, jg));
    if (hrow) tj -= static_cast<double>(hrow[jg]);
    const double dj = static_cast<double>(Srow[jg]);
    const uint32_t g = grouped ? static_cast<uint32_t>(jg) / gs : 0u;
    const double beta = dj > 0.0 ? tj + acc / dj : tj;
    return beta / static_cast<double>(sc[g]) + static_cast<double>(zc[g]);
}

// The level of t in binary64 (round half to even, clamped to 0 .. maxq).
__device__ __forceinline__ float tie_code(double t, float maxq) {
    return static_cast<float>(rint(fmin(fmax(t, 0.0), static_cast<double>(maxq))));
}

// Sequential in-block kernel (sweeps where every column moves by a real
// amount: the first sweep, a relaxed sweep and the sweep after one).
// One warp per row; column j = 32 h + jj is decided by lane jj, which keeps
// its code and change Delta'; the change (db, the same in every lane after the
// shuffle) times Sigma_bar[j][l] is added to every later column l.  Lanes whose
// column is already decided (l <= j) absorb harmless updates, so no lane test
// is needed; an unchanged column (db == 0) skips the updates.
// RELAX: the relax heuristic (Sec. 3.2): a live column (Sigma_jj > 0) takes
// beta~ itself instead of its nearest level; a dead one stays on its level.
// DF: the objective change of each decision (Lemma 1 along one coordinate)
// goes to rowdf, as in the change-driven kernels: the deciding lane only stores
// beta~ of its column (in grid units) to the warp's row of shared memory, and
// the changes are formed after the sweep over the block, so the sequential
// chain waits on no load.
template <int B, bool FULL, bool RELAX, bool DF, bool TIE = false>
__global__ void __launch_bounds__(1024) k_cd_block_seq(const __grid_constant__ CdArgs a) {
    using C = CdCfg<B>;
    constexpr int CPL = C::CPL;
    extern __shared__ __align__(16) float cd_smem[];
    float *tri = cd_smem;
    uint64_t *bar = reinterpret_cast<uint64_t *>(cd_smem + C::PACK);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *tdec = cd_smem + C::PACK + 4 + warp * B;   // DF: beta~ at each decision (after the barrier)
    // the codes decided in this visit and a snapshot of the lanes' values, for the
    // near-tie refinement (after the DF rows)
    float *cdec = cd_smem + C::PACK + 4 + (DF ? (blockDim.x >> 5) * B : 0) + 2 * warp * B;
    float *snap = cdec + B;
    const int64_t i = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + warp;
    const bool row_ok = i < a.q;
    float t[CPL], st[CPL];
    if (!cd_prologue<B, FULL>(a, tri, bar, i, row_ok, lane, t, st)) return;
    if (!row_ok) return;
    const int bw = FULL ? B : a.bw;
    const float maxq = a.maxq;
    uint32_t live = 0u;   // bit h: this lane's column 32 h + lane has Sigma_jj > 0
    if (RELAX) {
#pragma unroll
        for (int h = 0; h < CPL; ++h)
            if ((FULL || 32 * h + lane < bw) && a.d[a.b0 + 32 * h + lane] > 0.0f) live |= 1u << h;
    }
    // near-tie refinement: only in the first sweep (RELAX and a real-valued start turn it off)
    const bool tie = TIE && !RELAX && a.tie_eps > 0.0f && a.first_sweep && !a.vstart;
    float code[CPL], dlt[CPL];
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        code[h] = 0.0f;
        dlt[h] = 0.0f;
    }
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        // The word's 32 columns in order.  The deciding lane notes whether its value
        // sat within tie_eps of a midpoint (off the sequential chain); after the word,
        // the first such column is decided again from the binary64 beta~: the lanes
        // restore the values of the snapshot taken before the pass, replay the
        // decisions before that column (the same arithmetic, so the same results),
        // decide it exactly and resume after it.
        int start = 0;
        while (true) {
            if (tie) {
#pragma unroll
                for (int g = h; g < CPL; ++g) snap[32 * g + lane] = t[g];
            }
            bool mynear = false;
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
                if (jj < start) continue;
                const int j = 32 * h + jj;
                if (!FULL && j >= bw) break;
                const float cq = rintf(fminf(fmaxf(t[h], 0.0f), maxq));
                const float c = (RELAX && ((live >> h) & 1u)) ? t[h] : cq;
                const float dl = st[h] - c;
                if (lane == jj) {
                    code[h] = c;
                    dlt[h] = dl;
                    if (DF) tdec[j] = t[h];
                    if (tie) {
                        cdec[j] = c;
                        mynear = fabsf(fabsf(t[h] - cq) - 0.5f) < a.tie_eps;
                    }
                }
                const float db = __shfl_sync(0xffffffffu, dl, jj);
                if (db != 0.0f) {
                    const float *row = tri + kPackPad + tri_off(B, j) - (j + 1);
#pragma unroll
                    for (int g = h; g < CPL; ++g) t[g] = fmaf(db, row[32 * g + lane], t[g]);
                }
            }
            if (!tie) break;
            const unsigned nb = __ballot_sync(0xffffffffu, mynear);
            if (nb == 0u) break;
            const int jt = __ffs(nb) - 1;
            __syncwarp();
#pragma unroll
            for (int g = h; g < CPL; ++g) t[g] = snap[32 * g + lane];
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {   // replay the columns before jt
                if (jj < start) continue;
                if (jj >= jt) break;
                const int j = 32 * h + jj;
                const float c = rintf(fminf(fmaxf(t[h], 0.0f), maxq));
                const float dl = st[h] - c;
                const float db = __shfl_sync(0xffffffffu, dl, jj);
                if (db != 0.0f) {
                    const float *row = tri + kPackPad + tri_off(B, j) - (j + 1);
#pragma unroll
                    for (int g = h; g < CPL; ++g) t[g] = fmaf(db, row[32 * g + lane], t[g]);
                }
            }
            // column 32 h + jt from the binary64 beta~ of the row's state
            const int j = 32 * h + jt;
            const double te = tie_beta(&a, i, a.b0, bw, j, lane, cdec);
            const float c = tie_code(te, maxq);
            const float dl = __shfl_sync(0xffffffffu, st[h], jt) - c;
            if (lane == jt) {
                code[h] = c;
                dlt[h] = dl;
                if (DF) tdec[j] = static_cast<float>(te);
                cdec[j] = c;
            }
            if (dl != 0.0f) {
                const float *row = tri + kPackPad + tri_off(B, j) - (j + 1);
#pragma unroll
                for (int g = h; g < CPL; ++g) t[g] = fmaf(dl, row[32 * g + lane], t[g]);
            }
            start = jt + 1;
            if (start >= 32 || (!FULL && 32 * h + start >= bw)) break;
        }
    }
    if (DF) {
        __syncwarp();
        const float sc = a.scale[i * a.ngroups + a.b0 / a.gsize];
        const float s2 = sc * sc;
        double dfacc = 0.0;
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            if (!FULL && l >= bw) continue;
            const float dj = a.d[a.b0 + l];
            if (dj > 0.0f) {
                const float tv = tdec[l];
                const float e1 = code[h] - tv, e0 = st[h] - tv;
                dfacc += static_cast<double>(dj * s2 * (e1 * e1 - e0 * e0));
            }
        }
        dfacc = warp_sum(dfacc);
        if (lane == 0) a.rowdf[i] += dfacc;
    }
    cd_epilogue<B, FULL, false>(a, a.b0, a.bw, i, lane, code, dlt, false);
}

// Change-driven in-block kernel (every sweep after the first), exactly
// equivalent to the sequential order: a column whose code does not change
// alters no other column, so all remaining columns are quantized at once, the
// first one that changes is found by a warp ballot, its change is applied to
// the columns after it, and the pass resumes right after it.  The cost is
// (number of changed columns + 1) data-parallel passes.
// The change-driven decisions of one row over one block (shared by the
// per-block and the persistent kernels): quantize every column not yet final,
// find the first one whose code changes (warp ballot), add its change times
// its row of the block's Sigma_bar (packed triangle `tri`) to the columns
// after it, and resume right after it.  dfacc (per lane) collects the exact
// objective change of each applied decision (Lemma 1: along one coordinate
// f(u) = Sigma_jj (u - beta)^2 + const, here u = s (code - z), beta = s (t - z)).
//   GROWS = false: the coupling rows come from the packed triangle in shared
//   memory; GROWS = true: from the fp32 Sigma_bar rows in global memory
//   (`grow` = &Sigma_bar[b0][b0], leading dimension lds; the same values).
// With `ax` (near-tie refinement on, ax->tie_eps > 0; row i, block start b0;
// tie_blk: B floats of the warp's shared memory), a
// column whose beta~ lies within tie_eps of a midpoint also stops the pass: its
// decision is taken from the binary64 beta~ of the row's state at that point
// (columns before it final, after it at their start codes), and the pass goes on
// from it as from any other column.
template <int B, bool FULL, bool GROWS = false, bool TIE = false>
__device__ __forceinline__ int chg_decide(const float *tri, const float *d_blk, int bw_, float maxq, float s2,
                                          bool want_df, int lane, float (&t)[B / 32], const float (&st)[B / 32],
                                          float (&code)[B / 32], float (&dlt)[B / 32], double &dfacc,
                                          const float *grow = nullptr, int64_t lds = 0,
                                          const CdArgs *ax = nullptr, int64_t i = 0, int64_t b0 = 0,
                                          float *tie_blk = nullptr) {
    constexpr int CPL = B / 32;
    const int bw = FULL ? B : bw_;
    const bool tie = TIE && ax != nullptr && tie_blk != nullptr && ax->tie_eps > 0.0f;
    const float eps = tie ? ax->tie_eps : 0.0f;
#pragma unroll
    for (int h = 0; h < CPL; ++h) code[h] = st[h];
    // dlt (= st - code, exact for these small integers) is formed once at the end, so
    // it holds no registers during the passes
    int pos = 0;                                       // first column not yet final
    int nchg = 0;
    while (pos < bw) {
        int jstar = -1;
        bool jtie = false;
        // values of this lane's column in the word that holds the first change
        // (captured with a compile-time h, so the arrays stay in registers)
        float v = 0.0f, tv = 0.0f, cv = 0.0f, sv = 0.0f;
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            const bool active = l >= pos && (FULL || l < bw);
            const float c = rintf(fminf(fmaxf(t[h], 0.0f), maxq));
            const float dl = st[h] - c;
            if (active) code[h] = c;
            // within eps of a midpoint: |t - nearest level| within eps of 1/2 (a clamped
            // t just beyond the end levels also passes; deciding it exactly is harmless)
            const bool nt = tie && active && fabsf(fabsf(t[h] - c) - 0.5f) < eps;
            const unsigned m = __ballot_sync(0xffffffffu, active && (dl != 0.0f || nt));
            if (jstar < 0 && m != 0u) {
                jstar = 32 * h + (__ffs(m) - 1);
                if (TIE) jtie = tie && ((__ballot_sync(0xffffffffu, nt) >> (jstar & 31)) & 1u);
                v = dl;
                tv = t[h];
                cv = c;
                sv = st[h];
            }
        }
        if (jstar < 0) break;
        if (TIE && jtie) {
            // binary64 beta~ of column jstar: the block's columns from this warp's shared
            // row (final before jstar, start after), the rest from global memory
#pragma unroll
            for (int h = 0; h < CPL; ++h)
                if (FULL || 32 * h + lane < bw) tie_blk[32 * h + lane] = (32 * h + lane < jstar) ? code[h] : st[h];
            __syncwarp();
            const double te = tie_beta(ax, i, b0, bw, jstar, lane, tie_blk);
            __syncwarp();
            const float ce = tie_code(te, maxq);
            const float se = __shfl_sync(0xffffffffu, sv, jstar & 31);
            const float de = se - ce;
#pragma unroll
            for (int h = 0; h < CPL; ++h)
                if (32 * h + lane == jstar) code[h] = ce;
            if (de == 0.0f) {   // no change: the columns after it keep their provisional decisions
                pos = jstar + 1;
                continue;
            }
            v = de;
            tv = static_cast<float>(te);
            cv = ce;
            sv = se;
        }
        if (want_df && lane == (jstar & 31)) {
            const float dj = d_blk[jstar];
            if (dj > 0.0f) {
                const float e1 = cv - tv, e0 = sv - tv;
                dfacc += static_cast<double>(dj * s2 * (e1 * e1 - e0 * e0));
            }
        }
        const float db = __shfl_sync(0xffffffffu, v, jstar & 31);
        if (GROWS) {
            const float *row = grow + jstar * lds + lane;
            float rv[CPL];
#pragma unroll
            for (int g = 0; g < CPL; ++g) rv[g] = (FULL || 32 * g + lane < bw) ? __ldg(row + 32 * g) : 0.0f;
#pragma unroll
            for (int g = 0; g < CPL; ++g) t[g] = fmaf(db, rv[g], t[g]);
        } else {
            const float *row = tri + kPackPad + tri_off(B, jstar) - (jstar + 1);
#pragma unroll
            for (int g = 0; g < CPL; ++g) t[g] = fmaf(db, row[32 * g + lane], t[g]);
        }
        pos = jstar + 1;
        ++nchg;
    }
#pragma unroll
    for (int h = 0; h < CPL; ++h) dlt[h] = st[h] - code[h];
    return nchg;
}

// ---- refinement of the per-block change-driven kernel, CTA-wide -----------------
// The rows of a CTA first decide in binary32 as usual, noting every final
// decision whose t lies within tie_eps of a midpoint; then the whole CTA checks
// those decisions one at a time, each against beta~ recomputed from the row's
// state at that decision (one pass over the row by every thread of the CTA,
// double-float sums); a row whose decision was wrong decides again from the
// block's start with that column forced to its exact code, noting only the
// near-ties after it, and the check repeats.  A row checks its first kMaxEv notes
// of a visit and forces at most kMaxForced decisions (at tie_eps = 1e-5 a
// 256-column visit has one note in about eighty).
constexpr int kMaxEv = 8;      // near-tie notes per row and block visit
constexpr int kMaxForced = 4;  // exact decisions forced per row and block visit

// chg_decide's binary32 passes with notes: columns fj[0 .. nf) take the codes
// fc[..]; every decision after column rec_from whose t lay within eps of a
// midpoint goes to ev (ascending), *nev counting past kMaxEv on overflow.  A
// change here updates only the columns after it, so every column keeps the t it
// was decided on, and the notes are taken once at the end.
template <int B, bool FULL>
__device__ __forceinline__ void chg_decide_rec(const float *tri, const float *d_blk, int bw_, float maxq, float s2,
                                               bool want_df, int lane, float (&t)[B / 32], const float (&st)[B / 32],
                                               float (&code)[B / 32], float (&dlt)[B / 32], double &dfacc, float eps,
                                               const int *fj, const float *fc, int nf, int rec_from, int *ev,
                                               int *nev) {
    constexpr int CPL = B / 32;
    const int bw = FULL ? B : bw_;
#pragma unroll
    for (int h = 0; h < CPL; ++h) code[h] = st[h];
    int pos = 0;
    while (pos < bw) {
        int jstar = -1;
        float v = 0.0f, tv = 0.0f, cv = 0.0f, sv = 0.0f;
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            const bool active = l >= pos && (FULL || l < bw);
            float c = rintf(fminf(fmaxf(t[h], 0.0f), maxq));
            if (nf > 0)
                for (int f = 0; f < nf; ++f)
                    if (fj[f] == l) c = fc[f];
            const float dl = st[h] - c;
            if (active) code[h] = c;
            const unsigned m = __ballot_sync(0xffffffffu, active && dl != 0.0f);
            if (jstar < 0 && m != 0u) {
                jstar = 32 * h + (__ffs(m) - 1);
                v = dl;
                tv = t[h];
                cv = c;
                sv = st[h];
            }
        }
        if (jstar < 0) break;
        if (want_df && lane == (jstar & 31)) {
            const float dj = d_blk[jstar];
            if (dj > 0.0f) {
                const float e1 = cv - tv, e0 = sv - tv;
                dfacc += static_cast<double>(dj * s2 * (e1 * e1 - e0 * e0));
            }
        }
        const float db = __shfl_sync(0xffffffffu, v, jstar & 31);
        const float *row = tri + kPackPad + tri_off(B, jstar) - (jstar + 1);
#pragma unroll
        for (int g = 0; g < CPL; ++g)
            if (32 * g + lane > jstar) t[g] = fmaf(db, row[32 * g + lane], t[g]);
        pos = jstar + 1;
    }
    // the notes: every column's t is the one it was decided on
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        const int l = 32 * h + lane;
        bool nt = (FULL || l < bw) && l > rec_from && fabsf(fabsf(t[h] - rintf(fminf(fmaxf(t[h], 0.0f), maxq))) - 0.5f) < eps;
        for (int f = 0; f < nf; ++f)
            if (fj[f] == l) nt = false;
        unsigned mn = __ballot_sync(0xffffffffu, nt);
        if (mn != 0u && lane == 0) {
            int n = *nev;
            while (mn != 0u) {
                const int b = __ffs(mn) - 1;
                mn &= mn - 1u;
                if (n < kMaxEv) ev[n] = 32 * h + b;
                ++n;
            }
            *nev = n;
        }
    }
    __syncwarp();
#pragma unroll
    for (int h = 0; h < CPL; ++h) dlt[h] = st[h] - code[h];
}

// CTA-wide: beta~ / s + z of column b0 + j of row i at its decision: the block's
// columns before j from cr (final codes), after j from sr (start codes), the rest
// from the codes in global memory.  Every thread of the CTA calls it; red holds
// 34 doubles of shared memory.  Returns the same value in every thread.
__device__ __forceinline__ double coop_tie_beta(const CdArgs &a, int64_t i, int64_t b0, int bw, int j,
                                                const float *cr, const float *sr, double *red) {
    const int tid = threadIdx.x, nth = blockDim.x;
    const int64_t jg = b0 + j;
    const float *Srow = a.S + jg * a.lds_full;
    const float *sc = a.scale + i * a.ngroups;
    const float *zc = a.zero + i * a.ngroups;
    const bool grouped = a.ngroups > 1;
    const uint32_t gs = static_cast<uint32_t>(a.gsize);
    const uint8_t *crow = a.codes + i * a.ldc;
    const float *hrow = a.Hd ? a.Hd + i * a.ldh : nullptr;
    float hi = 0.0f, lo = 0.0f;
    // U columns per thread in flight: all their loads are issued before the sums
    constexpr int U = 8;
    for (int64_t k0 = tid; k0 < a.p; k0 += static_cast<int64_t>(nth) * U) {
        float cv[U], wv[U], hv[U], sv[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t k = k0 + static_cast<int64_t>(u) * nth;
            cv[u] = wv[u] = hv[u] = sv[u] = 0.0f;
            if (k < a.p) {
                if (k >= b0 && k < b0 + bw) {
                    const int l = static_cast<int>(k - b0);
                    cv[u] = l < j ? cr[l] : sr[l];
                } else {
                    cv[u] = static_cast<float>(crow[k]);
                }
                wv[u] = tie_w(a, i, k);
                if (hrow) hv[u] = hrow[k];
                sv[u] = (k == jg) ? 0.0f : Srow[k];   // column j itself is left out
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t k = k0 + static_cast<int64_t>(u) * nth;
            if (k >= a.p) continue;
            const uint32_t g = grouped ? static_cast<uint32_t>(k) / gs : 0u;
            df_term(hi, lo, wv[u], hv[u], sc[g], cv[u] - zc[g], sv[u]);
        }
    }
    double acc = warp_sum(static_cast<double>(hi) + static_cast<double>(lo));
    if ((tid & 31) == 0) red[tid >> 5] = acc;
    __syncthreads();
    if (tid == 0) {
        double sum = 0.0;
        for (int w = 0; w < (nth >> 5); ++w) sum += red[w];
        double tj = static_cast<double>(tie_w(a, i, jg));
        if (hrow) tj -= static_cast<double>(hrow[jg]);
        const double dj = static_cast<double>(Srow[jg]);
        const uint32_t g = grouped ? static_cast<uint32_t>(jg) / gs : 0u;
        const double beta = dj > 0.0 ? tj + sum / dj : tj;
        red[32] = beta / static_cast<double>(sc[g]) + static_cast<double>(zc[g]);
    }
    __syncthreads();
    return red[32];
}

// Shared memory of the refinement variant after the packed block, per warp.
struct TieWarp {
    int ev[kMaxEv];
    int fj[kMaxForced];
    float fc[kMaxForced];
    int nev, nf, wrong_j;
    float wrong_c;
};

template <int B>
__host__ __device__ constexpr int tie_cta_bytes(int warps) {
    return warps * (2 * B * 4 + static_cast<int>(sizeof(TieWarp))) + 34 * 8;
}

// Change-driven in-block kernel (every sweep after the first), exactly
// equivalent to the sequential order: a column whose code does not change
// alters no other column, so the cost is (number of changed columns + 1)
// data-parallel passes (chg_decide).
template <int B, bool FULL, bool TIE = false>
__global__ void __launch_bounds__(1024, 1) k_cd_block_chg(const __grid_constant__ CdArgs a) {
    if (a.gate && *a.gate != a.gate_run) return;   // uniform: the list form of the sweep runs
    using C = CdCfg<B>;
    constexpr int CPL = C::CPL;
    extern __shared__ __align__(16) float cd_smem[];
    float *tri = cd_smem;
    uint64_t *bar = reinterpret_cast<uint64_t *>(cd_smem + C::PACK);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t i = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + warp;
    const bool row_ok = i < a.q;
    float t[CPL], st[CPL];
    float code[CPL], dlt[CPL];
    double dfacc = 0.0;
    if constexpr (TIE) {
        // refinement variant: binary32 decisions with notes, checked CTA-wide
        const int nw = static_cast<int>(blockDim.x >> 5);
        float *cr = cd_smem + C::PACK + 4;                  // [nw][B] final codes
        float *sr = cr + nw * B;                            // [nw][B] start codes
        TieWarp *tw = reinterpret_cast<TieWarp *>(sr + nw * B);
        double *red = reinterpret_cast<double *>(tw + nw);
        const bool ok = cd_prologue<B, FULL>(a, tri, bar, i, row_ok, lane, t, st);
        if (__syncthreads_or(!ok)) return;   // a wait gave up somewhere: every warp leaves
        const int bw = FULL ? B : a.bw;
        const float s = row_ok ? a.scale[i * a.ngroups + a.b0 / a.gsize] : 1.0f;
        TieWarp &me = tw[warp];
        if (lane == 0) {
            me.nev = 0;
            me.nf = 0;
            me.wrong_j = -1;
        }
        __syncwarp();
        if (row_ok)
            chg_decide_rec<B, FULL>(tri, a.d + a.b0, a.bw, a.maxq, s * s, a.rowdf != nullptr, lane, t, st, code, dlt,
                                    dfacc, a.tie_eps, me.fj, me.fc, 0, -1, me.ev, &me.nev);
        // a row without notes is final: it writes its results now, without waiting
        const bool noted = row_ok && me.nev > 0;
        if (row_ok && !noted) {
            if (a.rowdf) {
                dfacc = warp_sum(dfacc);
                if (lane == 0) a.rowdf[i] += dfacc;
            }
            if (a.lent)
                cd_epilogue<B, FULL, true>(a, a.b0, a.bw, i, lane, code, dlt, true);
            else
                cd_epilogue<B, FULL, false>(a, a.b0, a.bw, i, lane, code, dlt, true);
        }
        if (noted) {
#pragma unroll
            for (int h = 0; h < CPL; ++h) {
                cr[warp * B + 32 * h + lane] = code[h];
                sr[warp * B + 32 * h + lane] = st[h];
            }
        }
        if (__syncthreads_count(noted && lane == 0) == 0) return;   // no notes in this CTA
        for (int round = 0; round <= kMaxForced; ++round) {
            __syncthreads();
            // check the notes, row by row, in order; the first wrong one stops its row's checks
            bool any = false;
            for (int w = 0; w < nw; ++w) {
                const int64_t iw = static_cast<int64_t>(blockIdx.x) * nw + w;
                if (iw >= a.q) break;
                // (more than kMaxEv notes: the first kMaxEv, in column order, are checked)
                const int n = tw[w].nev < kMaxEv ? tw[w].nev : kMaxEv;
                for (int e = 0; e < n; ++e) {
                    const int j = tw[w].ev[e];
                    const double te = coop_tie_beta(a, iw, a.b0, bw, j, cr + w * B, sr + w * B, red);
                    const float ce = tie_code(te, a.maxq);
                    const bool wrong = ce != cr[w * B + j];
                    if (wrong) {
                        if (threadIdx.x == 0) {
                            tw[w].wrong_j = j;
                            tw[w].wrong_c = ce;
                        }
                        any = true;
                        break;
                    }
                }
            }
            __syncthreads();
            if (!any) break;
            if (lane == 0 && me.wrong_j == -1) me.nev = 0;   // this row's notes all held
            // rows with a wrong decision decide again from the block's start (R holds it)
            if (row_ok && me.wrong_j != -1) {
                const int wj = me.wrong_j;
                __syncwarp();
#pragma unroll
                for (int h = 0; h < CPL; ++h) {
                    const int l = 32 * h + lane;
                    t[h] = (FULL || l < bw) ? a.R[i * a.ldr + a.b0 + l] : 0.0f;
                }
                dfacc = 0.0;
                // force the exact code (a row whose kMaxForced forced decisions are used
                // up keeps its last decisions: in practice never reached)
                if (lane == 0) {
                    if (me.nf < kMaxForced) {
                        me.fj[me.nf] = wj;
                        me.fc[me.nf] = me.wrong_c;
                        me.nf += 1;
                    }
                    me.nev = 0;
                    me.wrong_j = -1;
                }
                __syncwarp();
                chg_decide_rec<B, FULL>(tri, a.d + a.b0, a.bw, a.maxq, s * s, a.rowdf != nullptr, lane, t, st, code,
                                        dlt, dfacc, a.tie_eps, me.fj, me.fc, me.nf, wj, me.ev, &me.nev);
                if (round == kMaxForced && lane == 0) me.nev = 0;
                __syncwarp();
#pragma unroll
                for (int h = 0; h < CPL; ++h) {
                    cr[warp * B + 32 * h + lane] = code[h];
                    sr[warp * B + 32 * h + lane] = st[h];
                }
            }
        }
        if (!noted) return;   // written above
    } else {
        if (!cd_prologue<B, FULL>(a, tri, bar, i, row_ok, lane, t, st)) return;
        if (!row_ok) return;
        const float s = a.scale[i * a.ngroups + a.b0 / a.gsize];
        chg_decide<B, FULL>(tri, a.d + a.b0, a.bw, a.maxq, s * s, a.rowdf != nullptr, lane, t, st, code, dlt, dfacc);
    }
    if (a.rowdf) {
        dfacc = warp_sum(dfacc);
        if (lane == 0) a.rowdf[i] += dfacc;
    }
    if (a.lent)
        cd_epilogue<B, FULL, true>(a, a.b0, a.bw, i, lane, code, dlt, true);
    else
        cd_epilogue<B, FULL, false>(a, a.b0, a.bw, i, lane, code, dlt, true);
}

// One block of one row in the persistent list kernel (R and the codes stream with
// evict-first hints, so that L2 keeps the Sigma_bar rows the gathers re-read): stage t = R + the
// change-list correction (storing it back as the block's base when the window
// held a change), wait for the block's packed Sigma_bar, decide, write back.
// Returns false when the wait gave up.
template <int B, bool FULL, bool LATE, bool GR = false, bool TIE = false>
__device__ __forceinline__ bool rows_block(const CdArgs &a, int64_t b0, int bw_, const float *tri, uint64_t *bar,
                                           uint32_t parity, int64_t i, bool row_ok, int lane, float s2_row,
                                           double &dfacc, int &nchg, float *tie_blk) {
    constexpr int CPL = B / 32;
    const int bw = FULL ? B : bw_;
    const int64_t ii = row_ok ? i : 0;
    float s2 = s2_row;   // grouped grids: the scale of the block's group
    if (GR) {
        const float sb = a.scale[ii * a.ngroups + b0 / a.gsize];
        s2 = sb * sb;
    }
    float ps[CPL], st[CPL], t[CPL];
#pragma unroll
    for (int h = 0; h < CPL; ++h) ps[h] = 0.0f;
    bool changed;
    if (LATE) {
        // few listed changes: issue the block's base and codes first, so their
        // latency overlaps the count / entry / gather chain
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            const bool ok = row_ok && (FULL || l < bw);
            t[h] = ok ? __ldcs(a.R + ii * a.ldr + b0 + l) : 0.0f;
            st[h] = ok ? static_cast<float>(__ldcs(a.codes + ii * a.ldc + b0 + l)) : 0.0f;
        }
        changed = list_correction<B, FULL, 2, GR>(a, b0, bw, ii, row_ok, lane, ps);
#pragma unroll
        for (int h = 0; h < CPL; ++h) t[h] += ps[h];
    } else {
        // the gathers first (many changes: they hold the registers), then base and codes
        changed = list_correction<B, FULL, 4, GR>(a, b0, bw, ii, row_ok, lane, ps);
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            const bool ok = row_ok && (FULL || l < bw);
            t[h] = (ok ? __ldcs(a.R + ii * a.ldr + b0 + l) : 0.0f) + ps[h];
            st[h] = ok ? static_cast<float>(__ldcs(a.codes + ii * a.ldc + b0 + l)) : 0.0f;
        }
    }
    if (changed) {
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            if (row_ok && (FULL || l < bw)) __stcs(a.R + ii * a.ldr + b0 + l, t[h]);
        }
    }
    if (!LATE && !mbar_wait_bounded(bar, parity, nullptr)) return false;
    if (!row_ok) return true;
    float code[CPL], dlt[CPL];
    nchg += chg_decide<B, FULL, LATE, TIE>(tri, a.d + b0, bw, a.maxq, s2, true, lane, t, st, code, dlt, dfacc,
                                      a.sbar + b0 * a.lds + b0, a.lds, &a, i, b0, tie_blk);
    cd_epilogue<B, FULL, true, GR>(a, b0, bw, i, lane, code, dlt, true);
    return true;
}

// Free-mode shared memory of one warp of the persistent list kernel: the row's
// window (kWinCap entries) and a staging area for the Sigma_bar row segments of
// the correction, filled by cp.async so that many segments are in flight
// without holding registers.
constexpr int kFreeWarpBytes = 8192;
constexpr int kWinCap = 128;
constexpr int kStageFloats = (kFreeWarpBytes - 4 * kWinCap) / 4;

// Window of one row: the entries of all its change lists (the changes of every
// block's most recent visit) in ascending global column, each as
// column | Delta' << 16 (p <= 65536).  All lists of 32 blocks are read in one
// gather.  Returns the number of entries, or -1 when there are more than
// kWinCap (the lists in global memory serve then).
template <int B>
__device__ __forceinline__ int build_window(const CdArgs &a, int64_t i, int lane, uint32_t *win) {
    const int64_t rb = i * a.nblk;
    int wn = 0;
    for (int c0 = 0; c0 < a.nblk; c0 += 32) {
        const int cnt = (c0 + lane < a.nblk) ? a.lcnt[rb + c0 + lane] : 0;
        int incl = cnt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        const int tot = __shfl_sync(0xffffffffu, incl, 31);
        if (tot == 0) continue;
        if (wn + tot > kWinCap) return -1;
        uint32_t e[kWinCap / 32];
#pragma unroll
        for (int k = 0; k < kWinCap / 32; ++k) {
            const int x = 32 * k + lane;   // entry number within the chunk
            // its block: how many blocks have an inclusive count <= x
            int pos = 0;
#pragma unroll
            for (int st = 16; st > 0; st >>= 1) {
                const int v = __shfl_sync(0xffffffffu, incl, pos + st - 1);
                if (v <= x) pos += st;
            }
            const int excl = __shfl_sync(0xffffffffu, incl - cnt, pos);
            e[k] = 0u;
            if (x < tot) {
                const uint32_t raw = a.lent[(rb + c0 + pos) * B + (x - excl)];
                e[k] = (static_cast<uint32_t>((c0 + pos) * B) + (raw & 0xffffu)) | (raw & 0xffff0000u);
            }
        }
#pragma unroll
        for (int k = 0; k < kWinCap / 32; ++k)
            if (32 * k + lane < tot) win[wn + 32 * k + lane] = e[k];
        wn += tot;
    }
    __syncwarp();
    return wn;
}

// One block of one row in the free mode with the shared-memory window: the same
// steps as rows_block (the correction adds the same changes in the same order,
// so the same sums), then this block's entries in the window are replaced by
// the changes just made.  The lists in global memory are written as well, so a
// window that outgrows kWinCap (wn = -1) hands over to them.
template <int B, bool FULL, bool GR = false, bool TIE = false>
__device__ __forceinline__ void rows_block_win(const CdArgs &a, int64_t b0, int bw_, int64_t i, int lane,
                                               float s2_row, double &dfacc, int &nchg, uint32_t *win, float *stg,
                                               int &wn) {
    constexpr int CPL = B / 32;
    constexpr int NST = kStageFloats / B;       // segments per staged batch
    constexpr int SEG16 = B / 4;                // 16-byte pieces per segment
    const int bw = FULL ? B : bw_;
    float s2 = s2_row, sblk = 1.0f;   // grouped grids: the scale of the block's group
    if (GR) {
        sblk = a.scale[i * a.ngroups + b0 / a.gsize];
        s2 = sblk * sblk;
    }
    float ps[CPL], st[CPL], t[CPL];
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        const int l = 32 * h + lane;
        const bool ok = FULL || l < bw;
        t[h] = ok ? __ldcs(a.R + i * a.ldr + b0 + l) : 0.0f;
        st[h] = ok ? static_cast<float>(__ldcs(a.codes + i * a.ldc + b0 + l)) : 0.0f;
        ps[h] = 0.0f;
    }
    const float *sb = a.sbar + b0;
    for (int u0 = 0; u0 < wn; u0 += NST) {
        const int nb = (wn - u0) < NST ? (wn - u0) : NST;
        for (int x = lane; x < nb * SEG16; x += 32) {
            const int e = x / SEG16, c = x % SEG16;
            if (FULL || 4 * c < bw)
                cp_async16(stg + e * B + 4 * c, sb + static_cast<int64_t>(win[u0 + e] & 0xffffu) * a.lds + 4 * c);
        }
        cp_async_wait_all();
        __syncwarp();
        for (int e = 0; e < nb; ++e) {
            // grouped grids: the change is in the grid units of its own group (the same
            // factor list_correction applies per list)
            float fac = 1.0f;
            if (GR) fac = __fdiv_rn(a.scale[i * a.ngroups + (win[u0 + e] & 0xffffu) / a.gsize], sblk);
            const float dv = static_cast<float>(static_cast<int16_t>(win[u0 + e] >> 16)) * fac;
#pragma unroll
            for (int h = 0; h < CPL; ++h)
                if (FULL || 32 * h + lane < bw) ps[h] = fmaf(dv, stg[e * B + 32 * h + lane], ps[h]);
        }
        __syncwarp();
    }
#pragma unroll
    for (int h = 0; h < CPL; ++h) t[h] += ps[h];
    if (wn > 0) {
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            const int l = 32 * h + lane;
            if (FULL || l < bw) __stcs(a.R + i * a.ldr + b0 + l, t[h]);
        }
    }
    float code[CPL], dlt[CPL];
    nchg += chg_decide<B, FULL, true, TIE>(nullptr, a.d + b0, bw, a.maxq, s2, true, lane, t, st, code, dlt, dfacc,
                                      a.sbar + b0 * a.lds + b0, a.lds, &a, i, b0, stg);
    cd_epilogue<B, FULL, true, GR>(a, b0, bw, i, lane, code, dlt, true);
    // window = [entries left of the block (k1)] [this visit's changes (nn)] [entries right of it]
    int k1 = 0, k2 = 0;
#pragma unroll
    for (int k = 0; k < kWinCap / 32; ++k) {
        const int x = 32 * k + lane;
        const int64_t col = x < wn ? static_cast<int64_t>(win[x] & 0xffffu) : INT64_MAX;
        k1 += __popc(__ballot_sync(0xffffffffu, col < b0));
        k2 += __popc(__ballot_sync(0xffffffffu, col < b0 + bw));
    }
    int nn = 0;
#pragma unroll
    for (int h = 0; h < CPL; ++h)
        nn += __popc(__ballot_sync(0xffffffffu, (FULL || 32 * h + lane < bw) && dlt[h] != 0.0f));
    const int wn2 = k1 + nn + (wn - k2);
    if (wn2 > kWinCap) {
        wn = -1;
        return;
    }
    uint32_t tail[kWinCap / 32];
#pragma unroll
    for (int k = 0; k < kWinCap / 32; ++k) {
        const int x = k2 + 32 * k + lane;
        tail[k] = x < wn ? win[x] : 0u;
    }
    __syncwarp();
#pragma unroll
    for (int k = 0; k < kWinCap / 32; ++k)
        if (k2 + 32 * k + lane < wn) win[k1 + nn + 32 * k + lane] = tail[k];
    int r = 0;
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        const int l = 32 * h + lane;
        const bool ch = (FULL || l < bw) && dlt[h] != 0.0f;
        const unsigned m = __ballot_sync(0xffffffffu, ch);
        if (ch) {
            const int16_t dv = static_cast<int16_t>(__float2int_rn(dlt[h]));
            win[k1 + r + __popc(m & ((1u << lane) - 1u))] =
                static_cast<uint32_t>(b0 + l) | (static_cast<uint32_t>(static_cast<uint16_t>(dv)) << 16);
        }
        r += __popc(m);
    }
    __syncwarp();
    wn = wn2;
}

// Rolling-window sweeps t_begin .. t_end-1 with the change-list correction,
// persistent over column blocks and sweeps.  With the correction taken from
// each row's own change lists, rows need nothing from one another (rows are
// independent given Sigma, Sec. 3.2), so a CTA keeps its rows (one per warp)
// for all its sweeps.  Each sweep, a CTA picks one of two modes from the
// number of changes its rows made in the previous sweep (the entries of the
// lists at sweep start):
//   lockstep: the warps step through the blocks together to share the packed
//     Sigma_bar block in shared memory, whose bulk copy overlaps the gathers
//     (many in-block changes per row: early sweeps);
//   free: every warp runs through the blocks on its own and reads the coupling
//     row of each in-block change from the fp32 Sigma_bar in global memory
//     (few changes: no block barriers, no copies).  A CTA that goes free stays
//     free for its remaining sweeps (correct at any density), so its warps no
//     longer meet between sweeps, and a row at a fixed point skips its sweeps.
// first_lockstep = 1 forces lockstep for the first sweep (its lists are empty
// after a residual refresh although many codes are about to change).
// first_lockstep = 2 (fresh): R was refreshed since the sweep that left the
// lists (the outlier variant's target moved), so the lists only give that
// sweep's change counts: the first sweep picks its mode from them, each row
// clears its own lists (the window starts empty) and visits its blocks even at
// a fixed point.
// Per sweep and row the objective change goes to rowdf_t[t - t_begin][i]; with
// sweep_codes the row's codes after each sweep are copied out.  flush: after the
// last sweep every block's base takes the changes of the lists of its own and
// later blocks (the ones its last visit did not see), so R is the exact residual
// of the final codes.
constexpr int kRowsMaxWarps = 28;   // rows per CTA of the persistent kernel (896 threads: 72 registers)

template <int B, bool GR, bool TIE = false>
__global__ void __launch_bounds__(32 * kRowsMaxWarps, 1) k_cd_rows_lists(const __grid_constant__ CdArgs a, int t_begin, int t_end,
                                                           double *rowdf_t, uint8_t *sweep_codes,
                                                           int first_lockstep, int free_max_changes, int flush) {
    if (a.gate && *a.gate != a.gate_run) return;   // uniform: the dense form of the sweep runs
    using C = CdCfg<B>;
    extern __shared__ __align__(16) float cd_smem[];
    float *tri = cd_smem;
    uint64_t *bar = reinterpret_cast<uint64_t *>(cd_smem + C::PACK);
    __shared__ int s_bad;
    __shared__ int s_chg[kRowsMaxWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nwarps = static_cast<int>(blockDim.x >> 5);
    const int64_t i = static_cast<int64_t>(blockIdx.x) * nwarps + warp;
    const bool row_ok = i < a.q;
    if (threadIdx.x == 0) {
        mbar_init(bar, 1);
        fence_mbar_init();
        s_bad = 0;
    }
    const float s = row_ok ? a.scale[i] : 1.0f;
    const float s2 = s * s;
    // changes of this row in the previous sweep = entries of its lists now
    int prev = 0;
    if (row_ok) {
        for (int c0 = 0; c0 < a.nblk; c0 += 32) {
            int cnt = (c0 + lane < a.nblk) ? a.lcnt[i * a.nblk + c0 + lane] : 0;
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
            prev += cnt;
        }
    }
    const bool fresh = first_lockstep == 2;
    if (fresh && row_ok) {
        __syncwarp();
        for (int c = lane; c < a.nblk; c += 32) a.lcnt[i * a.nblk + c] = 0;
        __syncwarp();
    }
    uint32_t use = 0;
    bool free_run = false;   // CTA-uniform; once set, the warps run their remaining sweeps alone
    for (int t = t_begin; t < t_end; ++t) {
        const bool forced_lockstep = first_lockstep == 1 && t == t_begin;
        if (!free_run) {
            if (lane == 0) s_chg[warp] = prev;
            __syncthreads();
            int cta = 0;
            for (int w = 0; w < nwarps; ++w) cta += s_chg[w];
            free_run = !forced_lockstep &&
                       static_cast<int64_t>(cta) <= static_cast<int64_t>(free_max_changes) * nwarps;
            // the free mode reuses the shared memory of the packed block and its barrier
            if (free_run && threadIdx.x == 0) mbar_inval(bar);
            __syncthreads();   // s_chg is rewritten at the next sweep
        }
        double dfacc = 0.0;
        int nchg = 0;
        if (free_run) {
            // A row whose previous sweep changed nothing is at a fixed point: its window
            // is empty, so every block stages the values it decided on last time.
            // With at most kWinCap changes the window lives in the warp's shared memory
            // (the packed block is no longer needed once the CTA runs free).
            if (row_ok && (prev > 0 || (fresh && t == t_begin))) {
                uint32_t *win = reinterpret_cast<uint32_t *>(reinterpret_cast<char *>(cd_smem) + warp * kFreeWarpBytes);
                float *stg = reinterpret_cast<float *>(win + kWinCap);
                int wn = (prev <= kWinCap && a.p <= 65536) ? build_window<B>(a, i, lane, win) : -1;
                for (int64_t b0 = 0; b0 < a.p; b0 += B) {
                    const int bw = static_cast<int>((a.p - b0) < B ? (a.p - b0) : B);
                    if (wn >= 0) {
                        if (bw == B)
                            rows_block_win<B, true, GR, TIE>(a, b0, bw, i, lane, s2, dfacc, nchg, win, stg, wn);
                        else
                            rows_block_win<B, false, GR, TIE>(a, b0, bw, i, lane, s2, dfacc, nchg, win, stg, wn);
                    } else if (bw == B) {
                        rows_block<B, true, true, GR, TIE>(a, b0, bw, tri, bar, 0u, i, row_ok, lane, s2, dfacc, nchg, stg);
                    } else {
                        rows_block<B, false, true, GR, TIE>(a, b0, bw, tri, bar, 0u, i, row_ok, lane, s2, dfacc, nchg, stg);
                    }
                }
            }
        } else {
            for (int64_t b0 = 0; b0 < a.p; b0 += B) {
                const int bw = static_cast<int>((a.p - b0) < B ? (a.p - b0) : B);
                if (threadIdx.x == 0) {
                    constexpr uint32_t bytes = C::PACK * 4;
                    mbar_arrive_expect_tx(bar, bytes);
                    bulk_load(tri, a.tri + (b0 / B) * C::PACK, bytes, bar);
                }
                // the warp's row for the near-tie refinement, after the packed block
                float *tblk = cd_smem + C::PACK + 4 + warp * B;
                const bool ok =
                    bw == B
                        ? rows_block<B, true, false, GR, TIE>(a, b0, bw, tri, bar, use & 1u, i, row_ok, lane, s2, dfacc, nchg,
                                                     tblk)
                        : rows_block<B, false, false, GR, TIE>(a, b0, bw, tri, bar, use & 1u, i, row_ok, lane, s2, dfacc,
                                                      nchg, tblk);
                ++use;
                if (!ok) {
                    set_error(a.err, ERR_TIMEOUT);
                    s_bad = 1;
                }
                // every warp is done with this block's Sigma_bar before the next copy replaces it
                __syncthreads();
                if (s_bad) {
                    // the copy may still land: keep the CTA until it has (bounded)
                    if (threadIdx.x == 0) mbar_wait_bounded(bar, (use - 1) & 1u, nullptr);
                    return;
                }
            }
        }
        prev = nchg;
        dfacc = warp_sum(dfacc);
        if (row_ok) {
            if (lane == 0) rowdf_t[static_cast<int64_t>(t - t_begin) * a.q + i] = dfacc;
            if (sweep_codes) {
                __syncwarp();
                const uint8_t *src = a.codes + i * a.ldc;
                uint8_t *dst = sweep_codes + (static_cast<int64_t>(t) * a.q + i) * a.p;
                for (int64_t j = lane; j < a.p; j += 32) dst[j] = src[j];
            }
        }
    }
    if (flush && row_ok) {
        constexpr int CPL = B / 32;
        __syncwarp();
        for (int64_t b0 = 0; b0 < a.p; b0 += B) {
            const int bw = static_cast<int>((a.p - b0) < B ? (a.p - b0) : B);
            float ps[CPL];
#pragma unroll
            for (int h = 0; h < CPL; ++h) ps[h] = 0.0f;
            const int bmin = static_cast<int>(b0 / B);
            const bool any = bw == B ? list_correction<B, true, 4, GR>(a, b0, bw, i, true, lane, ps, bmin)
                                     : list_correction<B, false, 4, GR>(a, b0, bw, i, true, lane, ps, bmin);
            if (!any) continue;
#pragma unroll
            for (int h = 0; h < CPL; ++h) {
                const int l = 32 * h + lane;
                if (l < bw) a.R[i * a.ldr + b0 + l] += ps[h];
            }
        }
    }
}

// obj[t] = obj[t-1] + sum_i rowdf_t[t][i] for nt <= 32 sweeps; prev may be NULL (0).
// Warp t sums sweep t (lane-strided, then a fixed butterfly: a fixed order); one
// thread then runs the prefix over the sweeps.
__global__ void k_obj_prefix(const double *rowdf_t, int64_t q, int nt, const double *prev, double *out,
                             const int *gate, int gate_run) {
    if (gate && *gate != gate_run) return;
    __shared__ double sw[32];
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (w < nt) {
        double acc = 0.0;
        for (int64_t k = lane; k < q; k += 32) acc += rowdf_t[static_cast<int64_t>(w) * q + k];
        acc = warp_sum(acc);
        if (lane == 0) sw[w] = acc;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double run = prev ? *prev : 0.0;
        for (int t = 0; t < nt; ++t) {
            run += sw[t];
            out[t] = run;
        }
    }
}

template <int B, bool FULL, bool SEQ, bool RELAX = false, bool DF = false, bool TIE = false>
static cudaError_t launch_cd_block_b(const CdArgs &a, int nsm, cudaStream_t s) {
    using C = CdCfg<B>;
    if (a.nsplit > C::MAX_SPLITS) return cudaErrorInvalidValue;
    auto kern = SEQ ? k_cd_block_seq<B, FULL, RELAX, DF, TIE> : k_cd_block_chg<B, FULL, TIE>;
    // one CTA per SM when the rows allow it (the packed block is shared by the CTA's rows)
    int64_t warps = ceil_div(a.q, nsm);
    if (warps > C::MAX_WARPS) warps = C::MAX_WARPS;
    if (warps < 1) warps = 1;
    // the sequential kernel keeps one row of beta~ per warp (DF), and one row of the
    // codes decided in the visit and one snapshot row (near-tie refinement), after the
    // packed block
    // (the change-driven kernel keeps one row per warp for the refinement)
    const int rows = static_cast<int>(warps) * B * 4;
    const int smem = SEQ ? (C::PACK + 4) * 4 + (DF ? rows : 0) + (TIE ? 2 * rows : 0)
                         : (C::PACK + 4) * 4 + (TIE ? tie_cta_bytes<B>(static_cast<int>(warps)) : 0);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const unsigned grid = static_cast<unsigned>(ceil_div(a.q, warps));
    kern<<<grid, static_cast<unsigned>(32 * warps), smem, s>>>(a);
    return cudaGetLastError();
}

template <int B, bool FULL>
static cudaError_t launch_cd_block_f(const CdArgs &a, int nsm, cudaStream_t s) {
    // the refinement variants: change-driven kernel, and the first sweep's sequential kernel
    const bool tie = a.tie_eps > 0.0f;
    if (!a.frac)
        return tie ? launch_cd_block_b<B, FULL, false, false, false, true>(a, nsm, s)
                   : launch_cd_block_b<B, FULL, false>(a, nsm, s);
    if (a.vout) return a.rowdf ? launch_cd_block_b<B, FULL, true, true, true>(a, nsm, s) : cudaErrorInvalidValue;
    if (tie && a.first_sweep && !a.vstart)
        return a.rowdf ? launch_cd_block_b<B, FULL, true, false, true, true>(a, nsm, s)
                       : launch_cd_block_b<B, FULL, true, false, false, true>(a, nsm, s);
    return a.rowdf ? launch_cd_block_b<B, FULL, true, false, true>(a, nsm, s)
                   : launch_cd_block_b<B, FULL, true, false, false>(a, nsm, s);
}

template <int B>
static cudaError_t launch_cd_block_w(const CdArgs &a, int nsm, cudaStream_t s) {
    return a.bw == B ? launch_cd_block_f<B, true>(a, nsm, s) : launch_cd_block_f<B, false>(a, nsm, s);
}

cudaError_t launch_cd_block(int B, const CdArgs &a, int nsm, cudaStream_t s) {
    switch (B) {
        case 64: return launch_cd_block_w<64>(a, nsm, s);
        case 128: return launch_cd_block_w<128>(a, nsm, s);
        case 256: return launch_cd_block_w<256>(a, nsm, s);
        default: return cudaErrorInvalidValue;
    }
}

int64_t packed_diag_floats(int64_t p, int B) { return ceil_div(p, B) * packed_block_floats(B); }

template <int B, bool GR, bool TIE>
static cudaError_t launch_cd_rows_b(const CdArgs &a, int t_begin, int t_end, double *rowdf_t,
                                   uint8_t *sweep_codes, int first_lockstep, int free_max_changes, int flush,
                                   int nsm, cudaStream_t s) {
    using C = CdCfg<B>;
    int64_t warps = ceil_div(a.q, nsm);
    if (warps > kRowsMaxWarps) warps = kRowsMaxWarps;
    if (warps < 1) warps = 1;
    // the packed block and one row per warp for the near-tie refinement (lockstep), or
    // one free-mode area per warp, whichever is larger
    const int64_t lock = C::SMEM + (TIE ? warps * B * 4 : 0);
    const int smem = static_cast<int>(warps * kFreeWarpBytes > lock ? warps * kFreeWarpBytes : lock);
    cudaError_t e = cudaFuncSetAttribute(k_cd_rows_lists<B, GR, TIE>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const unsigned grid = static_cast<unsigned>(ceil_div(a.q, warps));
    k_cd_rows_lists<B, GR, TIE><<<grid, static_cast<unsigned>(32 * warps), smem, s>>>(
        a, t_begin, t_end, rowdf_t, sweep_codes, first_lockstep, free_max_changes, flush);
    return cudaGetLastError();
}

cudaError_t launch_cd_rows_lists(int B, const CdArgs &a, int t_begin, int t_end, double *rowdf_t,
                                 uint8_t *sweep_codes, int first_lockstep, int free_max_changes, int flush,
                                 int nsm, cudaStream_t s) {
    if (!a.sbar || !a.lent || !a.lcnt || a.first_sweep || t_end <= t_begin) return cudaErrorInvalidValue;
    const int f = first_lockstep, m = free_max_changes, fl = flush;
#define QE_ROWS(BB)                                                                                            \
    (a.grouped ? (a.tie_eps > 0.0f ? launch_cd_rows_b<BB, true, true>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s)   \
                                   : launch_cd_rows_b<BB, true, false>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s)) \
               : (a.tie_eps > 0.0f ? launch_cd_rows_b<BB, false, true>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s)  \
                                   : launch_cd_rows_b<BB, false, false>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s)))
    switch (B) {
        case 64: return QE_ROWS(64);
        case 128: return QE_ROWS(128);
        case 256: return QE_ROWS(256);
        default: return cudaErrorInvalidValue;
    }
#undef QE_ROWS
}

cudaError_t launch_obj_prefix(const double *rowdf_t, int64_t q, int nt, const double *prev, double *out,
                              cudaStream_t s, const int *gate, int gate_run) {
    if (nt < 1 || nt > 32) return cudaErrorInvalidValue;
    k_obj_prefix<<<1, 32 * nt, 0, s>>>(rowdf_t, q, nt, prev, out, gate, gate_run);
    return cudaGetLastError();
}

// Sum of the list entry counts (the changes of the sweep just finished), per CTA
// then one 64-bit atomic add per CTA (integer sums: the order does not matter).
__global__ void __launch_bounds__(256) k_count_changes(const int *lcnt, int64_t n, const int *flag,
                                                       unsigned long long *counter) {
    if (*flag) return;
    __shared__ unsigned long long sw[8];
    unsigned long long acc = 0;
    for (int64_t k = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; k < n;
         k += static_cast<int64_t>(gridDim.x) * blockDim.x)
        acc += static_cast<unsigned long long>(lcnt[k]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) sw[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long t = 0;
        for (int w = 0; w < 8; ++w) t += sw[w];
        if (t) atomicAdd(counter, t);
    }
}

__global__ void k_switch_decide(unsigned long long *counter, long long below, int *flag) {
    if (*flag == 0 && *counter < static_cast<unsigned long long>(below)) *flag = 1;
    *counter = 0ull;
}

__global__ void k_record_form(const int *flag, uint8_t *form) { *form = *flag ? 2 : 1; }

cudaError_t launch_record_form(const int *flag, uint8_t *form, cudaStream_t s) {
    k_record_form<<<1, 1, 0, s>>>(flag, form);
    return cudaGetLastError();
}

cudaError_t launch_list_switch(const int *lcnt, int64_t n, int64_t below, unsigned long long *counter, int *flag,
                               cudaStream_t s) {
    if (n < 1 || below < 0) return cudaErrorInvalidValue;
    int64_t blocks = ceil_div(n, 256 * 16);
    if (blocks > 1024) blocks = 1024;
    k_count_changes<<<static_cast<unsigned>(blocks), 256, 0, s>>>(lcnt, n, flag, counter);
    k_switch_decide<<<1, 1, 0, s>>>(counter, static_cast<long long>(below), flag);
    return cudaGetLastError();
}

cudaError_t launch_pack_diag(const __nv_bfloat16 *snt, int64_t ldn, int64_t p, int B, float *out,
                             cudaStream_t s) {
    dim3 grid(static_cast<unsigned>(ceil_div(p, B)), static_cast<unsigned>(B));
    k_pack_diag<<<grid, 128, 0, s>>>(snt, ldn, p, p, B, out);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Objective (proof of Lemma 1; Eq. main-outlier): with D = W - H - What and
// R = P - What Sigma_bar current,  (D Sigma)_ij = d_j (R_ij - What_ij), so
//     f = sum_ij D_ij d_j (R_ij - What_ij).
// With codes == NULL it computes sum_ij (W - H)_ij d_j P_ij = ||(W - H) X||^2.
// Per-CTA partial sums (fp64), reduced in a fixed order by k_sum_partials.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_objective(const ObjArgs a, double *partial) {
    double acc = 0.0;
    for (int64_t i = blockIdx.x; i < a.q; i += gridDim.x) {
        const float s = a.codes ? a.scale[i] : 0.0f;
        const float z = a.codes ? a.zero[i] : 0.0f;
        for (int64_t j = threadIdx.x; j < a.p; j += blockDim.x) {
            const float dj = a.d[j];
            if (!(dj > 0.0f)) continue;
            float t = load_elem(a.W, a.w_bf16, i * a.ldw + j);
            if (a.H) t -= a.H[i * a.ldh + j];
            const float r = a.R[i * a.ldr + j];
            float term;
            if (a.codes) {   // R in grid-step units: R_abs - What = s (R - code)
                const float cj = static_cast<float>(a.codes[i * a.ldc + j]);
                const float wh = s * (cj - z);
                term = (t - wh) * dj * (s * (r - cj));
            } else {
                term = t * dj * r;
            }
            acc += static_cast<double>(term);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    __shared__ double sw[8];
    if ((threadIdx.x & 31) == 0) sw[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += sw[w];
        partial[blockIdx.x] = t;
    }
}

// The same with 4 consecutive columns per thread (p and the leading dimensions
// multiples of 4, 16-byte aligned rows; 8-byte for bf16 W): the 4 fp32 terms are
// added in fp32 before the fp64 accumulation (a quarter of the fp64 operations).
__global__ void __launch_bounds__(256) k_objective4(const ObjArgs a, double *partial) {
    double acc = 0.0;
    for (int64_t i = blockIdx.x; i < a.q; i += gridDim.x) {
        const float s = a.codes ? a.scale[i] : 0.0f;
        const float z = a.codes ? a.zero[i] : 0.0f;
        for (int64_t j = 4 * threadIdx.x; j < a.p; j += 4 * blockDim.x) {
            const float4 dv = *reinterpret_cast<const float4 *>(a.d + j);
            float t[4];
            if (a.w_bf16) {
                const uint2 u = *reinterpret_cast<const uint2 *>(static_cast<const __nv_bfloat16 *>(a.W) + i * a.ldw + j);
                t[0] = __uint_as_float(u.x << 16);
                t[1] = __uint_as_float(u.x & 0xffff0000u);
                t[2] = __uint_as_float(u.y << 16);
                t[3] = __uint_as_float(u.y & 0xffff0000u);
            } else {
                const float4 w = *reinterpret_cast<const float4 *>(static_cast<const float *>(a.W) + i * a.ldw + j);
                t[0] = w.x;
                t[1] = w.y;
                t[2] = w.z;
                t[3] = w.w;
            }
            if (a.H) {
                const float4 h = *reinterpret_cast<const float4 *>(a.H + i * a.ldh + j);
                t[0] -= h.x;
                t[1] -= h.y;
                t[2] -= h.z;
                t[3] -= h.w;
            }
            const float4 rv = *reinterpret_cast<const float4 *>(a.R + i * a.ldr + j);
            const float r[4] = {rv.x, rv.y, rv.z, rv.w};
            const float dj[4] = {dv.x, dv.y, dv.z, dv.w};
            float c[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            if (a.codes) {
                const uchar4 cv = *reinterpret_cast<const uchar4 *>(a.codes + i * a.ldc + j);
                c[0] = cv.x;
                c[1] = cv.y;
                c[2] = cv.z;
                c[3] = cv.w;
            }
            float sum = 0.0f;
#pragma unroll
            for (int x = 0; x < 4; ++x) {
                if (!(dj[x] > 0.0f)) continue;
                float term;
                if (a.codes) {   // R in grid-step units: R_abs - What = s (R - code)
                    const float wh = s * (c[x] - z);
                    term = (t[x] - wh) * dj[x] * (s * (r[x] - c[x]));
                } else {
                    term = t[x] * dj[x] * r[x];
                }
                sum += term;
            }
            acc += static_cast<double>(sum);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    __shared__ double sw[8];
    if ((threadIdx.x & 31) == 0) sw[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += sw[w];
        partial[blockIdx.x] = t;
    }
}

__global__ void k_sum_partials(const double *partial, int n, double *out) {
    __shared__ double sw[32];
    double acc = 0.0;
    for (int k = threadIdx.x; k < n; k += blockDim.x) acc += partial[k];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if ((threadIdx.x & 31) == 0) sw[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += sw[w];
        *out = t;
    }
}

// ---------------------------------------------------------------------------
// Sigma for fp32 X on fp32 FMA (64 x 64 tiles on or above the diagonal,
// mirrored).  X(a, k) = X[a * sa + k * sk] covers both layouts.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_sigma_f32(const float *X, int64_t p, int64_t n, int64_t sa,
                                                   int64_t sk, float *S, int accumulate) {
    const int ti = blockIdx.y, tj = blockIdx.x;
    if (tj < ti) return;
    __shared__ float As[16][68], Bs[16][68];
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    const int64_t a0 = static_cast<int64_t>(ti) * 64, b0 = static_cast<int64_t>(tj) * 64;
    float acc[4][4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = 0.0f;
    const bool kfast = (sk == 1);
    for (int64_t k0 = 0; k0 < n; k0 += 16) {
        for (int e = threadIdx.x; e < 1024; e += 256) {
            int kk, rr;
            if (kfast) {
                kk = e & 15;
                rr = e >> 4;
            } else {
                rr = e & 63;
                kk = e >> 6;
            }
            const int64_t k = k0 + kk, ra = a0 + rr, rb = b0 + rr;
            As[kk][rr] = (k < n && ra < p) ? X[ra * sa + k * sk] : 0.0f;
            Bs[kk][rr] = (k < n && rb < p) ? X[rb * sa + k * sk] : 0.0f;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk) {
            float av[4], bv[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) av[u] = As[kk][ty * 4 + u];
#pragma unroll
            for (int v = 0; v < 4; ++v) bv[v] = Bs[kk][tx * 4 + v];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(av[u], bv[v], acc[u][v]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int64_t r = a0 + ty * 4 + u, c = b0 + tx * 4 + v;
            if (r < p && c < p && c >= r) {
                float val = acc[u][v];
                if (accumulate) val += S[r * p + c];
                S[r * p + c] = val;
                if (c != r) S[c * p + r] = val;
            }
        }
}

cudaError_t launch_sigma_f32(const float *X, int64_t p, int64_t n, int64_t sa, int64_t sk, float *S,
                             int accumulate, cudaStream_t s) {
    const unsigned t = static_cast<unsigned>(ceil_div(p, 64));
    k_sigma_f32<<<dim3(t, t), 256, 0, s>>>(X, p, n, sa, sk, S, accumulate);
    return cudaGetLastError();
}

// Token-major bf16 X (rows n0 .. n0+nc of an n x p matrix) -> feature-major p x nc.
__global__ void k_transpose_bf16(const __nv_bfloat16 *X, int64_t n0, int64_t nc, int64_t p,
                                 int64_t ldx, __nv_bfloat16 *out, int64_t ldo) {
    __shared__ __nv_bfloat16 tile[32][33];
    const int64_t kb = static_cast<int64_t>(blockIdx.x) * 32, fb = static_cast<int64_t>(blockIdx.y) * 32;
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int64_t k = kb + r, f = fb + threadIdx.x;
        tile[r][threadIdx.x] = (k < nc && f < p) ? X[(n0 + k) * ldx + f] : __float2bfloat16_rn(0.0f);
    }
    __syncthreads();
    for (int r = threadIdx.y; r < 32; r += blockDim.y) {
        const int64_t f = fb + r, k = kb + threadIdx.x;
        if (f < p && k < nc) out[f * ldo + k] = tile[threadIdx.x][r];
    }
}

cudaError_t launch_transpose_bf16(const void *X, int64_t n0, int64_t nc, int64_t p, int64_t ldx,
                                  void *out, int64_t ld_out, cudaStream_t s) {
    dim3 grid(static_cast<unsigned>(ceil_div(nc, 32)), static_cast<unsigned>(ceil_div(p, 32)));
    k_transpose_bf16<<<grid, dim3(32, 8), 0, s>>>(reinterpret_cast<const __nv_bfloat16 *>(X), n0, nc,
                                                  p, ldx, reinterpret_cast<__nv_bfloat16 *>(out),
                                                  ld_out);
    return cudaGetLastError();
}

// ---- launchers -------------------------------------------------------------
static inline dim3 row_grid(int64_t rows, int64_t cols) {
    const int64_t bx = ceil_div(cols, 256) < 16 ? ceil_div(cols, 256) : 16;
    return dim3(static_cast<unsigned>(bx > 0 ? bx : 1), static_cast<unsigned>(rows < 65535 ? rows : 65535));
}

// for kernels that take 4 consecutive columns per thread
static inline dim3 row_grid4(int64_t rows, int64_t cols) { return row_grid(rows, ceil_div(cols, 4)); }

cudaError_t launch_grid(const void *W, int w_bf16, int64_t ldw, const float *H, int64_t ldh, int64_t q,
                        int64_t p, int64_t gsize, int bits, float *scale, float *zero, unsigned *err,
                        cudaStream_t s) {
    const dim3 grid(static_cast<unsigned>(q), static_cast<unsigned>(ceil_div(p, gsize)));
    k_grid<<<grid, 256, 0, s>>>(W, w_bf16, ldw, H, ldh, p, gsize, static_cast<float>((1 << bits) - 1), scale,
                                zero, err);
    return cudaGetLastError();
}

cudaError_t launch_sigma_norm(const float *S, int64_t lds, int64_t p, float *d, __nv_bfloat16 *snt,
                              int64_t ldn, unsigned *err, cudaStream_t s) {
    k_sigma_diag<<<static_cast<unsigned>(ceil_div(p, 256)), 256, 0, s>>>(S, lds, p, d, err);
    k_sigma_planes<<<row_grid4(p, p), 256, 0, s>>>(S, lds, p, d, snt, ldn, err);
    return cudaGetLastError();
}

cudaError_t launch_sigma_planes_h2(const float *S, int64_t lds, int64_t p, const float *d, __half *snh, int64_t ldn,
                                   float *cscale, cudaStream_t s) {
    const int64_t g = p < 65535 ? p : 65535;
    k_sigma_planes_h2<<<static_cast<unsigned>(g), 256, 0, s>>>(S, lds, p, d, snh, ldn, cscale);
    return cudaGetLastError();
}

cudaError_t launch_sigma_bar_rows(const float *S, int64_t lds, int64_t p, const float *d, float *sbar,
                                  int64_t ld, cudaStream_t s) {
    const dim3 grid(static_cast<unsigned>(ceil_div(ld, 32)), static_cast<unsigned>(ceil_div(p, 32)));
    k_sigma_bar_rows<<<grid, 256, 0, s>>>(S, lds, p, d, sbar, ld);
    return cudaGetLastError();
}

cudaError_t launch_make_planes(const void *W, int w_bf16, int64_t ldw, int64_t q, int64_t p,
                               int split, __nv_bfloat16 *out, int64_t ldo, cudaStream_t s) {
    k_make_planes<<<row_grid(q, p), 256, 0, s>>>(W, w_bf16, ldw, q, p, split, out, ldo);
    return cudaGetLastError();
}

cudaError_t launch_init_residual(const void *W, int w_bf16, int64_t ldw, const float *H, int64_t ldh,
                                 int64_t q, int64_t p, int64_t gsize, const float *scale, const float *zero,
                                 float *R, int64_t ldr, cudaStream_t s) {
    k_init_residual<<<row_grid4(q, p), 256, 0, s>>>(W, w_bf16, ldw, H, ldh, q, p, gsize, scale, zero, R, ldr);
    return cudaGetLastError();
}

cudaError_t launch_obj_step(double *rowdf, int64_t q, const double *prev, double *out, cudaStream_t s,
                            const int *gate, int gate_run) {
    k_obj_step<<<1, 1024, 0, s>>>(rowdf, q, prev, out, gate, gate_run);
    return cudaGetLastError();
}

cudaError_t launch_codes_to_qf(const uint8_t *codes, int64_t ldc, const float *scale, const float *zero,
                               int64_t q, int64_t p, int64_t gsize, int grouped, __nv_bfloat16 *qf,
                               int64_t ldq, cudaStream_t s) {
    k_codes_to_qf<<<row_grid(q, p), 256, 0, s>>>(codes, ldc, scale, zero, q, p, gsize, grouped, qf, ldq);
    return cudaGetLastError();
}




int objective_blocks(int64_t q) { return static_cast<int>(q < 1024 ? q : 1024); }

cudaError_t launch_sum_partials(const double *partial, int n, double *out, cudaStream_t s) {
    k_sum_partials<<<1, 256, 0, s>>>(partial, n, out);
    return cudaGetLastError();
}

cudaError_t launch_objective(const ObjArgs &a, double *partial, double *out, cudaStream_t s) {
    const int nb = objective_blocks(a.q);
    const auto al = [](const void *ptr, unsigned m) { return (reinterpret_cast<uintptr_t>(ptr) & m) == 0; };
    const bool vec = a.p % 4 == 0 && a.ldw % 4 == 0 && a.ldr % 4 == 0 && (!a.H || (a.ldh % 4 == 0 && al(a.H, 15))) &&
                     (!a.codes || (a.ldc % 4 == 0 && al(a.codes, 3))) && al(a.W, a.w_bf16 ? 7 : 15) && al(a.R, 15) &&
                     al(a.d, 15);
    if (vec)
        k_objective4<<<nb, 256, 0, s>>>(a, partial);
    else
        k_objective<<<nb, 256, 0, s>>>(a, partial);
    k_sum_partials<<<1, 256, 0, s>>>(partial, nb, out);
    return cudaGetLastError();
}

}  // namespace qe
