// Streaming and sequential kernels of the QuantEase CD path (Sec. 3.2):
// per-row grid, Sigma normalisation into bf16 hi/lo planes of Sigma_bar^T,
// the in-block sequential column updates (Lemma 1, Eq. cd-update-closed-2),
// the objective reduction, plus the fp32 SIMT Sigma and the bf16 transpose.
#include "qe_common.cuh"
#include "qe_internal.h"
#include <cuda_fp16.h>

#include "qe_kernels.h"
#include "qe_sweep.cuh"

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
        // max_k |S_jk| / d_j over the live k != j: a correctly rounded division by d_j > 0
        // keeps the order, so the largest |S_jk| is divided once (16-byte loads where the
        // row allows)
        float mx = 0.0f;
        if (jalive) {
            const float *row = S + j * lds;
            int64_t k = 0;
            if ((lds & 3) == 0 && (reinterpret_cast<uintptr_t>(S) & 15u) == 0 &&
                (reinterpret_cast<uintptr_t>(d) & 15u) == 0) {
                const int64_t p4 = p >> 2;
                for (int64_t k4 = threadIdx.x; k4 < p4; k4 += blockDim.x) {
                    const float4 v = reinterpret_cast<const float4 *>(row)[k4];
                    const float4 dd = reinterpret_cast<const float4 *>(d)[k4];
                    const int64_t kb = 4 * k4;
                    if (kb != j && dd.x > 0.0f) mx = fmaxf(mx, fabsf(v.x));
                    if (kb + 1 != j && dd.y > 0.0f) mx = fmaxf(mx, fabsf(v.y));
                    if (kb + 2 != j && dd.z > 0.0f) mx = fmaxf(mx, fabsf(v.z));
                    if (kb + 3 != j && dd.w > 0.0f) mx = fmaxf(mx, fabsf(v.w));
                }
                k = 4 * p4;
            }
            for (k += threadIdx.x; k < p; k += blockDim.x)
                if (k != j && d[k] > 0.0f) mx = fmaxf(mx, fabsf(row[k]));
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = mx;
        __syncthreads();
        mx = 0.0f;
        for (int w = 0; w < 8; ++w) mx = fmaxf(mx, red[w]);
        __syncthreads();   // red is rewritten for the next row
        if (jalive) mx = __fdiv_rn(mx, dj);
        // 2^e with mx 2^e in [2^14, 2^15) (finite mx; e = 0 for an all-zero row)
        int e = 0;
        if (mx > 0.0f && isfinite(mx)) e = 14 - ilogbf(mx);
        if (e > 100) e = 100;
        if (e < -100) e = -100;
        if (threadIdx.x == 0) cscale[j] = ldexpf(1.0f, -e);
        if ((ldn & 3) == 0 && (lds & 3) == 0 && (reinterpret_cast<uintptr_t>(S) & 15u) == 0 &&
            (reinterpret_cast<uintptr_t>(d) & 15u) == 0 && (reinterpret_cast<uintptr_t>(snh) & 7u) == 0) {
            // four columns per thread: 16-byte loads, 8-byte stores of each plane
            const float *row = S + j * lds;
            for (int64_t k4 = threadIdx.x; k4 < (ldn >> 2); k4 += blockDim.x) {
                const int64_t kb = 4 * k4;
                float v[4] = {0.0f, 0.0f, 0.0f, 0.0f}, dd[4] = {0.0f, 0.0f, 0.0f, 0.0f};
                if (jalive && kb + 3 < p) {
                    const float4 v4 = reinterpret_cast<const float4 *>(row)[k4];
                    const float4 d4 = reinterpret_cast<const float4 *>(d)[k4];
                    v[0] = v4.x; v[1] = v4.y; v[2] = v4.z; v[3] = v4.w;
                    dd[0] = d4.x; dd[1] = d4.y; dd[2] = d4.z; dd[3] = d4.w;
                } else if (jalive) {
                    for (int u = 0; u < 4; ++u)
                        if (kb + u < p) {
                            v[u] = row[kb + u];
                            dd[u] = d[kb + u];
                        }
                }
                __half hi[4], lo[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    float x = 0.0f;
                    if (kb + u < p && jalive && kb + u != j && dd[u] > 0.0f) x = ldexpf(__fdiv_rn(v[u], dj), e);
                    hi[u] = __float2half_rn(x);
                    lo[u] = __float2half_rn(x - __half2float(hi[u]));
                }
                const __half2 h01 = __halves2half2(hi[0], hi[1]), h23 = __halves2half2(hi[2], hi[3]);
                const __half2 l01 = __halves2half2(lo[0], lo[1]), l23 = __halves2half2(lo[2], lo[3]);
                uint2 ph, pl;
                ph.x = *reinterpret_cast<const unsigned *>(&h01);
                ph.y = *reinterpret_cast<const unsigned *>(&h23);
                pl.x = *reinterpret_cast<const unsigned *>(&l01);
                pl.y = *reinterpret_cast<const unsigned *>(&l23);
                *reinterpret_cast<uint2 *>(snh + j * ldn + kb) = ph;
                *reinterpret_cast<uint2 *>(snh + (p + j) * ldn + kb) = pl;
            }
        } else {
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

template <int B>
static cudaError_t launch_cd_block_w(const CdArgs &a, int nsm, cudaStream_t s) {
    const bool full = a.bw == B;
    if (a.frac)   // real-valued changes: the sequential kernel
        return full ? launch_cd_block_k<B, true, true>(a, nsm, s) : launch_cd_block_k<B, true, false>(a, nsm, s);
    return full ? launch_cd_block_k<B, false, true>(a, nsm, s) : launch_cd_block_k<B, false, false>(a, nsm, s);
}

cudaError_t launch_cd_tie_check(int B, const CdArgs &a, int nsm, cudaStream_t s) {
    const bool full = a.bw == B;
    switch (B) {
        case 64: return full ? launch_cd_tie_check_k<64, true>(a, nsm, s) : launch_cd_tie_check_k<64, false>(a, nsm, s);
        case 128: return full ? launch_cd_tie_check_k<128, true>(a, nsm, s) : launch_cd_tie_check_k<128, false>(a, nsm, s);
        case 256: return full ? launch_cd_tie_check_k<256, true>(a, nsm, s) : launch_cd_tie_check_k<256, false>(a, nsm, s);
        default: return cudaErrorInvalidValue;
    }
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

cudaError_t launch_cd_rows_lists(int B, const CdArgs &a, int t_begin, int t_end, double *rowdf_t,
                                 uint8_t *sweep_codes, int first_lockstep, int free_max_changes, int flush,
                                 int nsm, cudaStream_t s) {
    if (!a.sbar || !a.lent || !a.lcnt || a.first_sweep || t_end <= t_begin) return cudaErrorInvalidValue;
    const int f = first_lockstep, m = free_max_changes, fl = flush;
    switch (B) {
        case 64: return launch_cd_rows_k<64>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s);
        case 128: return launch_cd_rows_k<128>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s);
        case 256: return launch_cd_rows_k<256>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s);
        default: return cudaErrorInvalidValue;
    }
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
