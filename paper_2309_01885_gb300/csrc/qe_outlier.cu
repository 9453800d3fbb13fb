// Kernels of the outlier-aware variant (Sec. 4.3, Algorithm 4): lambda_max by
// the power method, the IHT target T = H - eta grad_H g, the hard-thresholding
// operator P_s as a radix select + stable compaction, and the sparse refresh
// P = P_W - H (I + Sigma_bar).
#include "qe_common.cuh"
#include "qe_outlier.h"

namespace qe {

// ---- block reductions ------------------------------------------------------
__device__ __forceinline__ double block_sum(double v, double *sh) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) sh[w] = v;
    __syncthreads();
    double t = 0.0;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) t += sh[k];
    return t;
}

// Exclusive scan of one unsigned value per thread over the CTA (blockDim <= 1024).
__device__ __forceinline__ unsigned block_excl_scan(unsigned v, unsigned *sh, unsigned *total) {
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    unsigned x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const unsigned y = __shfl_up_sync(0xffffffffu, x, o);
        if (l >= o) x += y;
    }
    __syncthreads();
    if (l == 31) sh[w] = x;
    __syncthreads();
    if (w == 0) {
        const int nw = blockDim.x >> 5;
        unsigned s = (l < nw) ? sh[l] : 0u;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const unsigned y = __shfl_up_sync(0xffffffffu, s, o);
            if (l >= o) s += y;
        }
        if (l < nw) sh[l] = s;
    }
    __syncthreads();
    const unsigned warp_base = (w > 0) ? sh[w - 1] : 0u;
    if (total) *total = sh[(blockDim.x >> 5) - 1];
    return warp_base + x - v;
}

// ---- power method (Sec. 4.3: lambda_max(X X^T) by power iteration) ----------
// y_out = Sigma (y_in / ||y_in||).  ||y_in||^2 is the sum of the per-CTA
// partials the previous step left in part_in (nparts of them, added in a fixed
// order, so the result is reproducible), or is computed here when part_in is
// NULL (the first step); each CTA leaves the sum of the squares of the y_out
// values it wrote in part_out[blockIdx.x].  One warp per row of Sigma; eight
// independent partial sums and four 16-byte row loads in flight per lane (a
// dependent chain of single loads made this step latency-bound) when the rows
// are 16-byte aligned.
__global__ void __launch_bounds__(256) k_power_step(const float *S, int64_t lds, int64_t p,
                                                    const float *y_in, const double *part_in, int nparts,
                                                    float *y_out, double *part_out) {
    __shared__ double sh[8];
    double n2 = 0.0;
    if (part_in) {
        for (int k = threadIdx.x; k < nparts; k += blockDim.x) n2 += part_in[k];
    } else {
        for (int64_t k = threadIdx.x; k < p; k += blockDim.x) n2 += (double)y_in[k] * y_in[k];
    }
    n2 = block_sum(n2, sh);
    const float inv = n2 > 0.0 ? static_cast<float>(1.0 / sqrt(n2)) : 0.0f;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool vec = (lds % 4 == 0) && ((reinterpret_cast<uintptr_t>(S) & 15u) == 0) &&
                     ((reinterpret_cast<uintptr_t>(y_in) & 15u) == 0);
    double own2 = 0.0;
    for (int64_t a = (int64_t)blockIdx.x * 8 + warp; a < p; a += (int64_t)gridDim.x * 8) {
        const float *row = S + a * lds;
        float acc[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) acc[u] = 0.0f;
        int64_t b0 = 0;
        if (vec) {
            const int64_t n4 = p / 4;
            const float4 *r4 = reinterpret_cast<const float4 *>(row);
            const float4 *y4 = reinterpret_cast<const float4 *>(y_in);
            // four 16-byte loads of the row in flight per lane; accumulators 0-3 take pieces
            // lane, lane + 64, ... and 4-7 pieces lane + 32, lane + 96, ..., in order
            for (int64_t b = lane; b < n4; b += 128) {
                float4 x[4], v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const bool in = b + 32 * u < n4;
                    x[u] = in ? r4[b + 32 * u] : make_float4(0.f, 0.f, 0.f, 0.f);
                    v[u] = in ? y4[b + 32 * u] : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int k = 4 * (u & 1);
                    acc[k] = fmaf(x[u].x, v[u].x, acc[k]);
                    acc[k + 1] = fmaf(x[u].y, v[u].y, acc[k + 1]);
                    acc[k + 2] = fmaf(x[u].z, v[u].z, acc[k + 2]);
                    acc[k + 3] = fmaf(x[u].w, v[u].w, acc[k + 3]);
                }
            }
            b0 = n4 * 4;
        }
        for (int64_t b = b0 + lane; b < p; b += 32) acc[0] = fmaf(row[b], y_in[b], acc[0]);
        float t = ((acc[0] + acc[1]) + (acc[2] + acc[3])) + ((acc[4] + acc[5]) + (acc[6] + acc[7]));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
        if (lane == 0) {
            const float ya = t * inv;
            y_out[a] = ya;
            own2 += (double)ya * ya;
        }
    }
    own2 = block_sum(own2, sh);
    if (threadIdx.x == 0) part_out[blockIdx.x] = own2;
}

__global__ void __launch_bounds__(256) k_power_final(const float *y, const float *z, int64_t p,
                                                     double *lam, double *eta) {
    __shared__ double sh[8];
    double n2 = 0.0, dz = 0.0;
    for (int64_t k = threadIdx.x; k < p; k += blockDim.x) {
        n2 += (double)y[k] * y[k];
        dz += (double)y[k] * z[k];
    }
    n2 = block_sum(n2, sh);
    dz = block_sum(dz, sh);
    if (threadIdx.x == 0) {
        const double l = n2 > 0.0 ? dz / sqrt(n2) : 0.0;
        *lam = l;
        *eta = l > 0.0 ? 1.0 / (2.0 * l) : 0.0;
    }
}

__global__ void k_fill(float *y, int64_t n, float v) {
    const int64_t k = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (k < n) y[k] = v;
}

// ---- IHT target (Eq. iht-update, Algorithm 4) --------------------------------
// grad_H g = 2 (H + What - W) Sigma = -2 D Sigma and (D Sigma)_ij = d_j (R_ij - What_ij),
// so T = H - eta grad = H + 2 eta d_j (R_ij - What_ij).  T is written flat (ld = p).
__global__ void k_iht_target(const float *H, const float *R, int64_t ld, const uint8_t *codes,
                             int64_t ldc, const float *scale, const float *zero, const float *d,
                             const double *eta, int64_t q, int64_t p, float *T) {
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        const float e2 = static_cast<float>(2.0 * (*eta));
        const float s = scale[i];
        for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < p;
             j += (int64_t)gridDim.x * blockDim.x) {
            const float dj = d[j] > 0.0f ? d[j] : 0.0f;
            // R in grid-step units: R_abs - What = s (R - code)
            const float cj = static_cast<float>(codes[i * ldc + j]);
            T[i * p + j] = H[i * ld + j] + e2 * dj * (s * (R[i * ld + j] - cj));
        }
    }
}

// The same with 4 consecutive columns per thread (16-byte loads of H, R, d and T,
// 4-byte loads of the codes; p, ld and ldc multiples of 4 and aligned rows), a CTA
// covering 1024 columns of gridDim.y-strided rows.
__global__ void __launch_bounds__(256) k_iht_target4(const float *H, const float *R, int64_t ld,
                                                     const uint8_t *codes, int64_t ldc, const float *scale,
                                                     const float *d, const double *eta, int64_t q, int64_t p,
                                                     float *T) {
    const int64_t j = (blockIdx.x * (int64_t)blockDim.x + threadIdx.x) * 4;
    if (j >= p) return;
    const float e2 = static_cast<float>(2.0 * (*eta));
    const float4 dv = *reinterpret_cast<const float4 *>(d + j);
    const float dj[4] = {dv.x > 0.0f ? dv.x : 0.0f, dv.y > 0.0f ? dv.y : 0.0f, dv.z > 0.0f ? dv.z : 0.0f,
                         dv.w > 0.0f ? dv.w : 0.0f};
#pragma unroll 2
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        const float s = scale[i];
        const float4 h = *reinterpret_cast<const float4 *>(H + i * ld + j);
        const float4 r = *reinterpret_cast<const float4 *>(R + i * ld + j);
        const uchar4 c = *reinterpret_cast<const uchar4 *>(codes + i * ldc + j);
        float4 o;
        o.x = h.x + e2 * dj[0] * (s * (r.x - static_cast<float>(c.x)));
        o.y = h.y + e2 * dj[1] * (s * (r.y - static_cast<float>(c.y)));
        o.z = h.z + e2 * dj[2] * (s * (r.z - static_cast<float>(c.z)));
        o.w = h.w + e2 * dj[3] * (s * (r.w - static_cast<float>(c.w)));
        *reinterpret_cast<float4 *>(T + i * p + j) = o;
    }
}

// Flat copy of a q x p matrix (bf16 / fp32, leading dimension ldw) into T (ld = p).
__global__ void k_flat_copy(const void *W, int w_bf16, int64_t ldw, int64_t q, int64_t p, float *T) {
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        for (int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; j < p;
             j += (int64_t)gridDim.x * blockDim.x) {
            const float w = w_bf16 ? __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(W)[i * ldw + j])
                                   : reinterpret_cast<const float *>(W)[i * ldw + j];
            T[i * p + j] = w;
        }
    }
}

// ---- P_s: radix select of the s-th largest nonzero |T| ----------------------
// Keys are the binary32 magnitudes (sign bit cleared): for non-negative floats
// the unsigned bit pattern orders like the value.  Three digit passes (bits
// 30..20, 19..9, 8..0) find kstar; then exactly count_gt keys are > kstar and
// need_eq keys == kstar are taken in ascending linear index (the tie rule).
__device__ __forceinline__ unsigned mag_key(float v) { return __float_as_uint(v) & 0x7fffffffu; }

constexpr int kHistThreads = 256;
__host__ __device__ constexpr int topk_shift(int pass) { return pass == 0 ? 20 : (pass == 1 ? 9 : 0); }
__host__ __device__ constexpr int topk_bins(int pass) { return pass == 2 ? 512 : kTopkBins; }
// Key bits fixed before the pass.
__host__ __device__ constexpr unsigned topk_fixed(int pass) { return pass == 0 ? 0u : (pass == 1 ? 0x7ff00000u : 0x7ffffe00u); }

// One digit pass.  Each CTA histograms its grid-stride share of T (16-byte loads
// when T is 16-byte aligned) in shared memory and adds it to st->hist[PASS]; the
// CTA that finishes last (ticket) picks the digit of the s-th largest key: the
// digit bins are scanned from the top, each thread owning a run of R consecutive
// bins, and the one thread whose run holds the crossing fixes the digit.
template <int PASS>
__global__ void __launch_bounds__(kHistThreads) k_topk_hist(const float *T, int64_t N, TopkState *st,
                                                            int64_t s_budget) {
    constexpr int kShift = topk_shift(PASS), kBins = topk_bins(PASS), R = kBins / kHistThreads;
    constexpr unsigned kFixed = topk_fixed(PASS), kMask = static_cast<unsigned>(kBins - 1);
    __shared__ unsigned h[kBins];
    __shared__ unsigned sh[32];
    __shared__ unsigned last;
#pragma unroll
    for (int j = 0; j < R; ++j) h[threadIdx.x + j * kHistThreads] = 0;
    __syncthreads();
    const unsigned prefix = PASS == 0 ? 0u : st->prefix;
    const int64_t stride = (int64_t)gridDim.x * kHistThreads;
    const int64_t t0 = blockIdx.x * (int64_t)kHistThreads + threadIdx.x;
    int64_t tail = 0;
    if ((reinterpret_cast<uintptr_t>(T) & 15u) == 0) {
        const int64_t N4 = N >> 2;
        const float4 *T4 = reinterpret_cast<const float4 *>(T);
#pragma unroll 4
        for (int64_t e = t0; e < N4; e += stride) {
            const float4 v = T4[e];
            const unsigned k[4] = {mag_key(v.x), mag_key(v.y), mag_key(v.z), mag_key(v.w)};
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (k[u] != 0u && ((k[u] ^ prefix) & kFixed) == 0u) atomicAdd(&h[(k[u] >> kShift) & kMask], 1u);
        }
        tail = N4 << 2;
    }
    for (int64_t e = tail + t0; e < N; e += stride) {
        const unsigned k = mag_key(T[e]);
        if (k != 0u && ((k ^ prefix) & kFixed) == 0u) atomicAdd(&h[(k >> kShift) & kMask], 1u);
    }
    __syncthreads();
    unsigned *gh = st->hist[PASS];
#pragma unroll
    for (int j = 0; j < R; ++j) {
        const int b = threadIdx.x + j * kHistThreads;
        if (h[b]) atomicAdd(&gh[b], h[b]);
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) last = (atomicAdd(&st->ticket[PASS], 1u) == gridDim.x - 1) ? 1u : 0u;
    __syncthreads();
    if (!last) return;
    __threadfence();
    // The last CTA: thread t owns the bins of descending rank [t R, t R + R).
    unsigned c[R];
    unsigned mine = 0;
#pragma unroll
    for (int j = 0; j < R; ++j) {
        c[j] = __ldcg(&gh[kBins - 1 - (threadIdx.x * R + j)]);
        mine += c[j];
    }
    unsigned total;
    const unsigned before = block_excl_scan(mine, sh, &total);
    unsigned remaining, empty;
    if (PASS == 0) {
        const unsigned long long want = (unsigned long long)s_budget < total ? (unsigned long long)s_budget : total;
        remaining = static_cast<unsigned>(want);
        empty = want == 0 ? 1u : 0u;
        if (threadIdx.x == 0) st->empty = empty;
    } else {
        remaining = st->remaining;
        empty = st->empty;
    }
    __syncthreads();
    if (empty) {
        if (threadIdx.x == 0 && PASS == 2) {
            st->kstar = 0xffffffffu;
            st->need_eq = 0u;
        }
        return;
    }
    if (before < remaining && before + mine >= remaining) {
        unsigned cum = before, run = before;
        int jj = R - 1;
        bool found = false;
#pragma unroll
        for (int j = 0; j < R; ++j) {   // the first bin of the run at which the running sum reaches remaining
            if (!found && run + c[j] >= remaining) {
                jj = j;
                cum = run;
                found = true;
            }
            run += c[j];
        }
        const unsigned digit = static_cast<unsigned>(kBins - 1 - (threadIdx.x * R + jj));
        const unsigned pre = prefix | (digit << kShift);
        st->prefix = pre;
        st->count_gt += cum;
        st->remaining = remaining - cum;
        if (PASS == 2) {
            st->kstar = pre;
            st->need_eq = remaining - cum;
        }
    }
}

constexpr int kChunk = 4096;   // elements per CTA in the compaction (256 threads x 16)

// The 16 consecutive keys of thread threadIdx.x in chunk blockIdx.x (0 past N).
__device__ __forceinline__ void chunk_keys(const float *T, int64_t N, bool vec, float v[16]) {
    const int64_t base = (int64_t)blockIdx.x * kChunk + threadIdx.x * 16;
    if (vec && base + 16 <= N) {
        const float4 *p4 = reinterpret_cast<const float4 *>(T + base);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const float4 x = p4[u];
            v[4 * u] = x.x;
            v[4 * u + 1] = x.y;
            v[4 * u + 2] = x.z;
            v[4 * u + 3] = x.w;
        }
    } else {
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = (base + u < N) ? T[base + u] : 0.0f;
    }
}

__global__ void __launch_bounds__(256) k_topk_count(const float *T, int64_t N, const TopkState *st,
                                                    unsigned *cnt_gt, unsigned *cnt_eq) {
    __shared__ unsigned sh[32];
    const unsigned kstar = st->kstar;
    float v[16];
    chunk_keys(T, N, (reinterpret_cast<uintptr_t>(T) & 15u) == 0, v);
    unsigned g = 0, q = 0;
#pragma unroll
    for (int u = 0; u < 16; ++u) {
        const unsigned k = mag_key(v[u]);
        if (k == 0u) continue;
        g += (k > kstar) ? 1u : 0u;
        q += (k == kstar) ? 1u : 0u;
    }
    unsigned tg, tq;
    block_excl_scan(g, sh, &tg);
    block_excl_scan(q, sh, &tq);
    if (threadIdx.x == 0) {
        cnt_gt[blockIdx.x] = tg;
        cnt_eq[blockIdx.x] = tq;
    }
}

// One CTA: exclusive scans over the chunks.  sel_base[c] = first output slot of
// chunk c, eq_base[c] = number of keys == kstar in chunks before c.
__global__ void __launch_bounds__(1024) k_topk_scan(const unsigned *cnt_gt, const unsigned *cnt_eq,
                                                    int nchunks, const TopkState *st, unsigned *sel_base,
                                                    unsigned *eq_base, int64_t *nnz_out) {
    __shared__ unsigned sh[32];
    const unsigned need = st->need_eq;
    unsigned carry_eq = 0, carry_sel = 0;
    for (int c0 = 0; c0 < nchunks; c0 += blockDim.x) {
        const int c = c0 + threadIdx.x;
        const unsigned ge = (c < nchunks) ? cnt_gt[c] : 0u;
        const unsigned qe_ = (c < nchunks) ? cnt_eq[c] : 0u;
        unsigned tq;
        const unsigned eqb = carry_eq + block_excl_scan(qe_, sh, &tq);
        unsigned take = 0;
        if (need > eqb) take = (need - eqb) < qe_ ? (need - eqb) : qe_;
        const unsigned sel = ge + take;
        unsigned ts;
        const unsigned sb = carry_sel + block_excl_scan(sel, sh, &ts);
        if (c < nchunks) {
            sel_base[c] = sb;
            eq_base[c] = eqb;
        }
        carry_eq += tq;
        carry_sel += ts;
        __syncthreads();
    }
    if (threadIdx.x == 0) *nnz_out = static_cast<int64_t>(carry_sel);
}

__global__ void __launch_bounds__(256) k_topk_emit(const float *T, int64_t N, const TopkState *st,
                                                   const unsigned *sel_base, const unsigned *eq_base,
                                                   int64_t *H_idx, float *H_val) {
    __shared__ unsigned sh[32];
    const unsigned kstar = st->kstar, need = st->need_eq;
    float v[16];
    chunk_keys(T, N, (reinterpret_cast<uintptr_t>(T) & 15u) == 0, v);
    unsigned ng = 0, nq = 0;
#pragma unroll
    for (int u = 0; u < 16; ++u) {
        const unsigned k = mag_key(v[u]);
        if (k == 0u) continue;
        ng += (k > kstar) ? 1u : 0u;
        nq += (k == kstar) ? 1u : 0u;
    }
    const unsigned eq0 = eq_base[blockIdx.x] + block_excl_scan(nq, sh, nullptr);
    unsigned take = 0;
    if (need > eq0) take = (need - eq0) < nq ? (need - eq0) : nq;
    unsigned out = sel_base[blockIdx.x] + block_excl_scan(ng + take, sh, nullptr);
    if (ng + take == 0u) return;
    const int64_t base = (int64_t)blockIdx.x * kChunk + threadIdx.x * 16;
    unsigned eqseen = 0;
#pragma unroll
    for (int u = 0; u < 16; ++u) {
        const unsigned k = mag_key(v[u]);
        if (k == 0u) continue;
        bool keep = k > kstar;
        if (k == kstar) {
            keep = eqseen < take;
            ++eqseen;
        }
        if (keep) {
            H_idx[out] = base + u;
            H_val[out] = v[u];
            ++out;
        }
    }
}

// ---- structured outliers (Sec. 4.3): keep whole columns -----------------------
// Squared column norms of the flat q x p matrix T, summed in fp64 over row
// chunks (part[rc][j]) and then over the chunks in order, rounded to fp32 keys
// for the radix select.
__global__ void __launch_bounds__(256) k_colnorm_partial(const float *T, int64_t q, int64_t p, int64_t rows_per,
                                                         double *part) {
    const int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (j >= p) return;
    const int64_t i0 = blockIdx.y * rows_per;
    const int64_t i1 = (i0 + rows_per) < q ? (i0 + rows_per) : q;
    double acc = 0.0;
    for (int64_t i = i0; i < i1; ++i) {
        const double v = T[i * p + j];
        acc += v * v;
    }
    part[blockIdx.y * p + j] = acc;
}

__global__ void k_colnorm_final(const double *part, int nrc, int64_t p, float *norm2) {
    const int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (j >= p) return;
    double acc = 0.0;
    for (int rc = 0; rc < nrc; ++rc) acc += part[rc * p + j];
    norm2[j] = static_cast<float>(acc);
}

// Every entry of the kept columns, as ascending linear indices: row i, kept
// column r -> slot i * ncols + r (the kept columns are ascending).
__global__ void k_col_emit(const float *T, int64_t q, int64_t p, const int64_t *cols, const int64_t *ncols_p,
                           int64_t *H_idx, float *H_val, int64_t *H_nnz) {
    const int64_t nc = *ncols_p;
    const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (t == 0) *H_nnz = q * nc;
    if (nc == 0 || t >= q * nc) return;
    const int64_t i = t / nc, r = t % nc;
    const int64_t e = i * p + cols[r];
    H_idx[t] = e;
    H_val[t] = T[e];
}

// Dense H from the kept entries (H zeroed before).
__global__ void k_scatter(const int64_t *H_idx, const float *H_val, const int64_t *nnz, int64_t cap,
                          int64_t p, float *H, int64_t ld) {
    const int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (t >= cap || t >= *nnz) return;
    const int64_t e = H_idx[t];
    H[(e / p) * ld + (e % p)] = H_val[t];
}

// rowptr[i] = first kept entry with linear index >= i * p (entries are sorted).
__global__ void k_rowptr(const int64_t *H_idx, const int64_t *nnz, int64_t q, int64_t p,
                         int64_t *rowptr) {
    const int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (i > q) return;
    const int64_t key = i * p;
    int64_t lo = 0, hi = *nnz;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (H_idx[mid] < key) lo = mid + 1;
        else hi = mid;
    }
    rowptr[i] = lo;
}

// Close this thread's current group of cp.async copies / wait until at most N of
// its committed groups are still in flight (the copies always complete).
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait_group() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// 4 bytes global -> shared (the columns of a piece cut by p).
__device__ __forceinline__ void cp_async4(void *dst, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)),
                 "l"(static_cast<unsigned long long>(__cvta_generic_to_global(src)))
                 : "memory");
}

// P_new = P_W - H (I + Sigma_bar) for row i; R += (P_new - P_old) / s_i when
// update_r (R in grid-step units); P = P_new.  Sigma_bar comes as fp32 rows
// (sbar[k][j] = Sigma_jk / d_j, zero on the diagonal and for dead columns: the
// binary32 values the tensor-core planes split), so the identity adds 1 at
// j = k.  One CTA per (row, tile of kSpmmCols columns); thread t owns
// kSpmmPieces pieces of 4 columns, piece u at u * 4 * kSpmmThreads + 4 t (so a
// warp's piece is 512 contiguous bytes: coalesced, and free of shared-memory
// bank conflicts).  The row's kept entries are staged in shared memory
// kSpmmChunk at a time; each thread copies its own pieces of the next
// kSpmmDepth - 1 entries' Sigma_bar rows into a ring in shared memory by
// cp.async (many rows in flight without registers, no thread waits for
// another) and adds the entries one after another in their sorted order.
// Rows are 16-byte aligned (ld, lds multiples of 4); a piece cut by p goes
// column by column.
constexpr int kSpmmThreads = 256;
constexpr int kSpmmPieces = 4;
constexpr int kSpmmPer = 4 * kSpmmPieces;
constexpr int kSpmmCols = kSpmmThreads * kSpmmPer;
constexpr int kSpmmChunk = 256;
constexpr int kSpmmDepth = 4;
constexpr int kSpmmSmem = kSpmmDepth * kSpmmCols * 4;

__global__ void __launch_bounds__(kSpmmThreads) k_spmm_refresh(const float *PW, float *P, float *R, int64_t ld,
                                                               const float *sbar, int64_t lds,
                                                               const int64_t *H_idx, const float *H_val,
                                                               const int64_t *rowptr, int64_t p, int update_r,
                                                               const float *scale) {
    __shared__ int sk[kSpmmChunk];
    __shared__ float sv[kSpmmChunk];
    __shared__ int so[kSpmmChunk];   // owner thread << 4 | slot of column k in this tile, or -1
    extern __shared__ __align__(16) float ring[];   // [kSpmmDepth][kSpmmPieces][kSpmmThreads][4]
    const int64_t i = blockIdx.x;
    const int64_t j0 = static_cast<int64_t>(blockIdx.y) * kSpmmCols + 4 * threadIdx.x;
    int ncol[kSpmmPieces];   // columns of piece u inside the layer (0 .. 4)
#pragma unroll
    for (int u = 0; u < kSpmmPieces; ++u) {
        const int64_t j = j0 + u * 4 * kSpmmThreads;
        ncol[u] = j >= p ? 0 : static_cast<int>((p - j) < 4 ? (p - j) : 4);
    }
    const int64_t e0 = rowptr[i], e1 = rowptr[i + 1];
    float acc[kSpmmPer];
#pragma unroll
    for (int u = 0; u < kSpmmPieces; ++u) {
        const int64_t j = j0 + u * 4 * kSpmmThreads;
        float4 v = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        if (ncol[u] == 4) {
            v = __ldcs(reinterpret_cast<const float4 *>(PW + i * ld + j));   // streamed
        } else {
            if (ncol[u] > 0) v.x = __ldcs(PW + i * ld + j);
            if (ncol[u] > 1) v.y = __ldcs(PW + i * ld + j + 1);
            if (ncol[u] > 2) v.z = __ldcs(PW + i * ld + j + 2);
        }
        acc[4 * u] = v.x;
        acc[4 * u + 1] = v.y;
        acc[4 * u + 2] = v.z;
        acc[4 * u + 3] = v.w;
    }
    float *mine = ring + 4 * threadIdx.x;
    for (int64_t c0 = e0; c0 < e1; c0 += kSpmmChunk) {
        const int n = static_cast<int>((e1 - c0) < kSpmmChunk ? (e1 - c0) : kSpmmChunk);
        __syncthreads();   // the previous chunk is consumed
        if (static_cast<int>(threadIdx.x) < n) {
            const int k = static_cast<int>(H_idx[c0 + threadIdx.x] - i * p);
            sk[threadIdx.x] = k;
            sv[threadIdx.x] = H_val[c0 + threadIdx.x];
            const int64_t kk = k - static_cast<int64_t>(blockIdx.y) * kSpmmCols;
            int own = -1;
            if (kk >= 0 && kk < kSpmmCols) {
                const int u = static_cast<int>(kk) / (4 * kSpmmThreads), w = static_cast<int>(kk) % (4 * kSpmmThreads);
                own = ((w >> 2) << 4) | (4 * u + (w & 3));
            }
            so[threadIdx.x] = own;
        }
        __syncthreads();
        // entry e goes to slot e % kSpmmDepth; one commit group per entry (empty past n)
        auto issue = [&](int e) {
            if (e < n) {
                const float *src = sbar + static_cast<int64_t>(sk[e]) * lds + j0;
                float *dst = mine + (e % kSpmmDepth) * kSpmmCols;
#pragma unroll
                for (int u = 0; u < kSpmmPieces; ++u) {
                    const int off = u * 4 * kSpmmThreads;
                    if (ncol[u] == 4) {
                        cp_async16(dst + off, src + off);
                    } else {
#pragma unroll
                        for (int x = 0; x < 3; ++x)
                            if (x < ncol[u]) cp_async4(dst + off + x, src + off + x);
                    }
                }
            }
            cp_async_commit();
        };
#pragma unroll
        for (int e = 0; e < kSpmmDepth - 1; ++e) issue(e);
        for (int e = 0; e < n; ++e) {
            issue(e + kSpmmDepth - 1);
            cp_async_wait_group<kSpmmDepth - 1>();   // entry e has landed
            const float hv = sv[e];
            const float *seg = mine + (e % kSpmmDepth) * kSpmmCols;
            // every column adds -h Sigma_bar[k][j] (columns past p take values never
            // stored); Sigma_bar[k][k] = 0, so the identity's -h at column k follows as one
            // more step of the same chain, in the thread that owns the column
#pragma unroll
            for (int u = 0; u < kSpmmPieces; ++u) {
                const float4 v = *reinterpret_cast<const float4 *>(seg + u * 4 * kSpmmThreads);
                acc[4 * u] = fmaf(-hv, v.x, acc[4 * u]);
                acc[4 * u + 1] = fmaf(-hv, v.y, acc[4 * u + 1]);
                acc[4 * u + 2] = fmaf(-hv, v.z, acc[4 * u + 2]);
                acc[4 * u + 3] = fmaf(-hv, v.w, acc[4 * u + 3]);
            }
            const int own = so[e];
            if ((own >> 4) == static_cast<int>(threadIdx.x)) {
                const int sl = own & 15;
#pragma unroll
                for (int z = 0; z < kSpmmPer; ++z) {
                    const float y = fmaf(-hv, 1.0f, acc[z]);
                    acc[z] = (z == sl) ? y : acc[z];
                }
            }
        }
        cp_async_wait_group<0>();
    }
    const float s = update_r ? scale[i] : 1.0f;
#pragma unroll
    for (int u = 0; u < kSpmmPieces; ++u) {
        const int64_t j = j0 + u * 4 * kSpmmThreads;
        if (ncol[u] == 4) {
            float4 *pp = reinterpret_cast<float4 *>(P + i * ld + j);
            const float4 pn = make_float4(acc[4 * u], acc[4 * u + 1], acc[4 * u + 2], acc[4 * u + 3]);
            if (update_r) {
                float4 *rp = reinterpret_cast<float4 *>(R + i * ld + j);
                const float4 po = __ldcs(pp);
                float4 r = __ldcs(rp);
                r.x += __fdiv_rn(pn.x - po.x, s);
                r.y += __fdiv_rn(pn.y - po.y, s);
                r.z += __fdiv_rn(pn.z - po.z, s);
                r.w += __fdiv_rn(pn.w - po.w, s);
                __stcs(rp, r);
            }
            __stcs(pp, pn);
        } else {
#pragma unroll
            for (int x = 0; x < 3; ++x) {
                if (x >= ncol[u]) break;
                float *pp = P + i * ld + j + x;
                if (update_r) __stcs(R + i * ld + j + x, __ldcs(R + i * ld + j + x) + __fdiv_rn(acc[4 * u + x] - __ldcs(pp), s));
                __stcs(pp, acc[4 * u + x]);
            }
        }
    }
}

__global__ void k_dinv(const float *d, int64_t p, float *dinv) {
    const int64_t j = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
    if (j < p) dinv[j] = d[j] > 0.0f ? 1.0f / d[j] : 0.0f;
}

// ---- launchers --------------------------------------------------------------
static inline bool aligned16(const void *ptr) { return (reinterpret_cast<uintptr_t>(ptr) & 15u) == 0; }

static inline dim3 rows_grid(int64_t rows, int64_t cols) {
    int64_t bx = ceil_div(cols, 256);
    if (bx > 16) bx = 16;
    if (bx < 1) bx = 1;
    return dim3(static_cast<unsigned>(bx), static_cast<unsigned>(rows < 65535 ? rows : 65535));
}

cudaError_t launch_power_lambda(const float *S, int64_t lds, int64_t p, int iters, float *y0, float *y1,
                                double *part, double *lam, double *eta, int nsm, cudaStream_t s) {
    k_fill<<<static_cast<unsigned>(ceil_div(p, 256)), 256, 0, s>>>(y0, p, 1.0f);
    int64_t blocks = ceil_div(p, 8);
    if (blocks > nsm * 4) blocks = nsm * 4;
    if (blocks > kPowerMaxBlocks) blocks = kPowerMaxBlocks;
    float *a = y0, *b = y1;
    const double *pin = nullptr;
    double *pout = part;
    for (int it = 0; it <= iters; ++it) {
        k_power_step<<<static_cast<unsigned>(blocks), 256, 0, s>>>(S, lds, p, a, pin, static_cast<int>(blocks), b,
                                                                   pout);
        if (it < iters) {
            float *t = a;
            a = b;
            b = t;
            pin = pout;
            pout = (pout == part) ? part + kPowerMaxBlocks : part;
        }
    }
    // a = y_iters, b = Sigma (y_iters / ||y_iters||)
    k_power_final<<<1, 256, 0, s>>>(a, b, p, lam, eta);
    return cudaGetLastError();
}

cudaError_t launch_iht_target(const float *H, const float *R, int64_t ld, const uint8_t *codes,
                              int64_t ldc, const float *scale, const float *zero, const float *d,
                              const double *eta, int64_t q, int64_t p, float *T, cudaStream_t s) {
    const bool vec = p % 4 == 0 && ld % 4 == 0 && ldc % 4 == 0 && aligned16(H) && aligned16(R) && aligned16(T) &&
                     aligned16(d) && (reinterpret_cast<uintptr_t>(codes) & 3u) == 0;
    if (vec) {
        const dim3 grid(static_cast<unsigned>(ceil_div(p, 1024)), static_cast<unsigned>(q < 1024 ? q : 1024));
        k_iht_target4<<<grid, 256, 0, s>>>(H, R, ld, codes, ldc, scale, d, eta, q, p, T);
    } else {
        k_iht_target<<<rows_grid(q, p), 256, 0, s>>>(H, R, ld, codes, ldc, scale, zero, d, eta, q, p, T);
    }
    return cudaGetLastError();
}

cudaError_t launch_flat_copy(const void *W, int w_bf16, int64_t ldw, int64_t q, int64_t p, float *T,
                             cudaStream_t s) {
    k_flat_copy<<<rows_grid(q, p), 256, 0, s>>>(W, w_bf16, ldw, q, p, T);
    return cudaGetLastError();
}

int64_t topk_chunks(int64_t N) { return ceil_div(N, kChunk); }

cudaError_t launch_topk(const float *T, int64_t N, int64_t s_budget, TopkState *st, unsigned *cnt_gt,
                        unsigned *cnt_eq, unsigned *sel_base, unsigned *eq_base, int64_t *H_idx,
                        float *H_val, int64_t *nnz, int nsm, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(st, 0, sizeof(TopkState), s);
    if (e != cudaSuccess) return e;
    int64_t hb = ceil_div(N, 256 * 16);
    if (hb > nsm * 4) hb = nsm * 4;
    if (hb < 1) hb = 1;
    k_topk_hist<0><<<static_cast<unsigned>(hb), kHistThreads, 0, s>>>(T, N, st, s_budget);
    k_topk_hist<1><<<static_cast<unsigned>(hb), kHistThreads, 0, s>>>(T, N, st, s_budget);
    k_topk_hist<2><<<static_cast<unsigned>(hb), kHistThreads, 0, s>>>(T, N, st, s_budget);
    const int64_t nch = topk_chunks(N);
    k_topk_count<<<static_cast<unsigned>(nch), 256, 0, s>>>(T, N, st, cnt_gt, cnt_eq);
    k_topk_scan<<<1, 1024, 0, s>>>(cnt_gt, cnt_eq, static_cast<int>(nch), st, sel_base, eq_base, nnz);
    k_topk_emit<<<static_cast<unsigned>(nch), 256, 0, s>>>(T, N, st, sel_base, eq_base, H_idx, H_val);
    return cudaGetLastError();
}

int colnorm_chunks(int64_t q) { return static_cast<int>(q < 64 * 64 ? ceil_div(q, 64) : 64); }

cudaError_t launch_topk_columns(const float *T, int64_t q, int64_t p, int64_t k, TopkState *st, unsigned *cnt_gt,
                                unsigned *cnt_eq, unsigned *sel_base, unsigned *eq_base, double *part,
                                float *norm2, int64_t *cols, float *colval, int64_t *ncols, int64_t *H_idx,
                                float *H_val, int64_t *nnz, int nsm, cudaStream_t s) {
    const int nrc = colnorm_chunks(q);
    const int64_t rows_per = ceil_div(q, nrc);
    const dim3 g1(static_cast<unsigned>(ceil_div(p, 256)), static_cast<unsigned>(nrc));
    k_colnorm_partial<<<g1, 256, 0, s>>>(T, q, p, rows_per, part);
    k_colnorm_final<<<static_cast<unsigned>(ceil_div(p, 256)), 256, 0, s>>>(part, nrc, p, norm2);
    cudaError_t e = launch_topk(norm2, p, k, st, cnt_gt, cnt_eq, sel_base, eq_base, cols, colval, ncols, nsm, s);
    if (e != cudaSuccess) return e;
    const int64_t cap = q * k;
    k_col_emit<<<static_cast<unsigned>(ceil_div(cap > 0 ? cap : 1, 256)), 256, 0, s>>>(T, q, p, cols, ncols, H_idx,
                                                                                     H_val, nnz);
    return cudaGetLastError();
}

cudaError_t launch_scatter_rowptr(const int64_t *H_idx, const float *H_val, const int64_t *nnz,
                                  int64_t cap, int64_t q, int64_t p, float *H, int64_t ld,
                                  int64_t *rowptr, cudaStream_t s) {
    if (cap > 0)
        k_scatter<<<static_cast<unsigned>(ceil_div(cap, 256)), 256, 0, s>>>(H_idx, H_val, nnz, cap, p, H,
                                                                             ld);
    k_rowptr<<<static_cast<unsigned>(ceil_div(q + 1, 256)), 256, 0, s>>>(H_idx, nnz, q, p, rowptr);
    return cudaGetLastError();
}

cudaError_t launch_spmm_refresh(const float *PW, float *P, float *R, int64_t ld, const float *sbar,
                                int64_t lds, const int64_t *H_idx, const float *H_val, const int64_t *rowptr,
                                int64_t q, int64_t p, int update_r, const float *scale, cudaStream_t s) {
    if (ld % 4 != 0 || lds % 4 != 0) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_spmm_refresh, cudaFuncAttributeMaxDynamicSharedMemorySize, kSpmmSmem);
    if (e != cudaSuccess) return e;
    const dim3 grid(static_cast<unsigned>(q), static_cast<unsigned>(ceil_div(p, kSpmmCols)));
    k_spmm_refresh<<<grid, kSpmmThreads, kSpmmSmem, s>>>(PW, P, R, ld, sbar, lds, H_idx, H_val, rowptr, p,
                                                         update_r, scale);
    return cudaGetLastError();
}

cudaError_t launch_dinv(const float *d, int64_t p, float *dinv, cudaStream_t s) {
    k_dinv<<<static_cast<unsigned>(ceil_div(p, 256)), 256, 0, s>>>(d, p, dinv);
    return cudaGetLastError();
}

}  // namespace qe
