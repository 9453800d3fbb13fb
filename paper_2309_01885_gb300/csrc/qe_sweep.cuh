// Column-block CD sweep kernels (Algorithm 3 inner loop, Sec. 3.2: the in-block
// sequential and change-driven kernels and the persistent change-list kernel)
// and their launch templates.  The explicit instantiations are spread over the
// qe_sweep_*.cu translation units, one kernel family and block width each, so
// that they compile in parallel; qe_cd.cu dispatches on the block width.
#pragma once

#include "qe_common.cuh"
#include "qe_internal.h"
#include <cuda_fp16.h>

#include "qe_kernels.h"

namespace qe {

// The hi/mid/lo split of one binary32 value.
__device__ __forceinline__ void split3(float x, __nv_bfloat16 &h, __nv_bfloat16 &m, __nv_bfloat16 &l) {
    h = __float2bfloat16_rn(x);
    const float r1 = x - __bfloat162float(h);
    m = __float2bfloat16_rn(r1);
    l = __float2bfloat16_rn(r1 - __bfloat162float(m));
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

// Pull toward L2 what an exact recompute of beta~ for row i reads (the row's codes,
// weights and H; Sigma's row jg): every line at once, from `nth` threads of which
// this is number `tid`.  Prefetches hold no register, so a recompute that comes
// later waits on L2 rather than on DRAM.
__device__ __forceinline__ void tie_prefetch_row(const CdArgs &a, int64_t i, int tid, int nth) {
    const uint8_t *crow = a.codes + i * a.ldc;
    for (int64_t k = 128 * static_cast<int64_t>(tid); k < a.p; k += 128 * static_cast<int64_t>(nth)) prefetch_l2(crow + k);
    if (a.w_bf16) {
        const __nv_bfloat16 *w = static_cast<const __nv_bfloat16 *>(a.W) + i * a.ldw;
        for (int64_t k = 64 * static_cast<int64_t>(tid); k < a.p; k += 64 * static_cast<int64_t>(nth)) prefetch_l2(w + k);
    } else {
        const float *w = static_cast<const float *>(a.W) + i * a.ldw;
        for (int64_t k = 32 * static_cast<int64_t>(tid); k < a.p; k += 32 * static_cast<int64_t>(nth)) prefetch_l2(w + k);
    }
    if (a.Hd)
        for (int64_t k = 32 * static_cast<int64_t>(tid); k < a.p; k += 32 * static_cast<int64_t>(nth))
            prefetch_l2(a.Hd + i * a.ldh + k);
}
__device__ __forceinline__ void tie_prefetch_srow(const CdArgs &a, int64_t jg, int tid, int nth) {
    const float *Srow = a.S + jg * a.lds_full;
    for (int64_t k = 32 * static_cast<int64_t>(tid); k < a.p; k += 32 * static_cast<int64_t>(nth)) prefetch_l2(Srow + k);
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
    int nchg = 0;
    int pos = 0;                                       // first column not yet final
    while (true) {
        // Word by word (lane l of word h is column 32 h + l): a change alters only the
        // columns after it, so once a word has no change left its decisions are final
        // and the passes go on with the next word alone.  A near-tie column (refinement
        // on) ends the scan; it is decided below and the scan resumes after it.
        int jt = -1;
#pragma unroll
        for (int h = 0; h < CPL; ++h) {
            if (jt >= 0 || 32 * h + 31 < pos) continue;   // (warp-uniform)
            const bool inb = FULL || 32 * h + lane < bw;
            int lo = pos > 32 * h ? pos - 32 * h : 0;  // first lane of word h not yet final
            while (true) {
                const bool active = lane >= lo && inb;
                const float c = rintf(fminf(fmaxf(t[h], 0.0f), maxq));
                const float dl = st[h] - c;
                if (active) code[h] = c;
                // within eps of a midpoint: |t - nearest level| within eps of 1/2 (a clamped
                // t just beyond the end levels also passes; deciding it exactly is harmless)
                const bool nt = tie && active && fabsf(fabsf(t[h] - c) - 0.5f) < eps;
                const unsigned m = __ballot_sync(0xffffffffu, active && (dl != 0.0f || nt));
                if (m == 0u) break;
                const int jl = __ffs(m) - 1;
                const int jstar = 32 * h + jl;
                if (TIE && ((__ballot_sync(0xffffffffu, nt) >> jl) & 1u)) {
                    jt = jstar;
                    break;
                }
                if (want_df && lane == jl) {
                    const float dj = d_blk[jstar];
                    if (dj > 0.0f) {
                        const float e1 = c - t[h], e0 = st[h] - t[h];
                        dfacc += static_cast<double>(dj * s2 * (e1 * e1 - e0 * e0));
                    }
                }
                const float db = __shfl_sync(0xffffffffu, dl, jl);
                // the change times its coupling row, added to the columns after it: the
                // rest of this word and every later word
                if (GROWS) {
                    const float *row = grow + jstar * lds + lane;
                    float rv[CPL];
#pragma unroll
                    for (int g = h; g < CPL; ++g)
                        rv[g] = (FULL || 32 * g + lane < bw) && (g > h || lane > jl) ? __ldg(row + 32 * g) : 0.0f;
                    if (lane > jl) t[h] = fmaf(db, rv[h], t[h]);
#pragma unroll
                    for (int g = h + 1; g < CPL; ++g) t[g] = fmaf(db, rv[g], t[g]);
                } else {
                    const float *row = tri + kPackPad + tri_off(B, jstar) - (jstar + 1);
                    if (lane > jl) t[h] = fmaf(db, row[32 * h + lane], t[h]);
#pragma unroll
                    for (int g = h + 1; g < CPL; ++g) t[g] = fmaf(db, row[32 * g + lane], t[g]);
                }
                lo = jl + 1;
                ++nchg;
            }
        }
        if constexpr (!TIE) {
            break;
        } else {
            if (jt < 0) break;
            // binary64 beta~ of the near-tie column jt: the block's columns from this warp's
            // shared row (final before jt, start after), the rest from global memory
#pragma unroll
            for (int g = 0; g < CPL; ++g)
                if (FULL || 32 * g + lane < bw) tie_blk[32 * g + lane] = (32 * g + lane < jt) ? code[g] : st[g];
            __syncwarp();
            const double te = tie_beta(ax, i, b0, bw, jt, lane, tie_blk);
            __syncwarp();
            const float ce = tie_code(te, maxq);
            float se = 0.0f;
#pragma unroll
            for (int g = 0; g < CPL; ++g)
                if (g == (jt >> 5)) se = __shfl_sync(0xffffffffu, st[g], jt & 31);
            const float de = se - ce;
#pragma unroll
            for (int g = 0; g < CPL; ++g)
                if (32 * g + lane == jt) code[g] = ce;
            pos = jt + 1;
            if (de == 0.0f) continue;   // no change: the columns after it keep their provisional decisions
            if (want_df && lane == (jt & 31)) {
                const float dj = d_blk[jt];
                if (dj > 0.0f) {
                    const float tv = static_cast<float>(te);
                    const float e1 = ce - tv, e0 = se - tv;
                    dfacc += static_cast<double>(dj * s2 * (e1 * e1 - e0 * e0));
                }
            }
            if (GROWS) {
                const float *row = grow + jt * lds + lane;
#pragma unroll
                for (int g = 0; g < CPL; ++g)
                    if ((FULL || 32 * g + lane < bw) && 32 * g + lane > jt) t[g] = fmaf(de, __ldg(row + 32 * g), t[g]);
            } else {
                const float *row = tri + kPackPad + tri_off(B, jt) - (jt + 1);
#pragma unroll
                for (int g = 0; g < CPL; ++g)
                    if (32 * g + lane > jt) t[g] = fmaf(de, row[32 * g + lane], t[g]);
            }
            ++nchg;
        }
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
    // word by word, as in chg_decide: a finished word's decisions are final
#pragma unroll
    for (int h = 0; h < CPL; ++h) {
        const int l = 32 * h + lane;
        const bool inb = FULL || l < bw;
        int lo = 0;
        while (true) {
            const bool active = lane >= lo && inb;
            float c = rintf(fminf(fmaxf(t[h], 0.0f), maxq));
            if (nf > 0)
                for (int f = 0; f < nf; ++f)
                    if (fj[f] == l) c = fc[f];
            const float dl = st[h] - c;
            if (active) code[h] = c;
            const unsigned m = __ballot_sync(0xffffffffu, active && dl != 0.0f);
            if (m == 0u) break;
            const int jl = __ffs(m) - 1;
            const int jstar = 32 * h + jl;
            if (want_df && lane == jl) {
                const float dj = d_blk[jstar];
                if (dj > 0.0f) {
                    const float e1 = c - t[h], e0 = st[h] - t[h];
                    dfacc += static_cast<double>(dj * s2 * (e1 * e1 - e0 * e0));
                }
            }
            const float db = __shfl_sync(0xffffffffu, dl, jl);
            const float *row = tri + kPackPad + tri_off(B, jstar) - (jstar + 1);
            if (lane > jl) t[h] = fmaf(db, row[32 * h + lane], t[h]);
#pragma unroll
            for (int g = h + 1; g < CPL; ++g) t[g] = fmaf(db, row[32 * g + lane], t[g]);
            lo = jl + 1;
        }
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

// Notes of one warp's row in shared memory (the refinement variants).
struct TieWarp {
    int ev[kMaxEv];
    int fj[kMaxForced];
    float fc[kMaxForced];
    int nev, nf, wrong_j;
    float wrong_c;
};
static_assert(kMaxEv == 8, "TieEntry holds 8 notes");

template <int B, bool FULL>
__device__ __forceinline__ void chg_write(const CdArgs &a, int64_t i, int lane, const float (&code)[B / 32],
                                          const float (&dlt)[B / 32]) {
    if (a.lent)
        cd_epilogue<B, FULL, true>(a, a.b0, a.bw, i, lane, code, dlt, true);
    else
        cd_epilogue<B, FULL, false>(a, a.b0, a.bw, i, lane, code, dlt, true);
}

// Change-driven in-block kernel (every sweep after the first), exactly
// equivalent to the sequential order: a column whose code does not change
// alters no other column, so the cost is (number of changed columns + 1)
// data-parallel passes (chg_decide).  With the refinement (TIE) the decisions
// are binary32 with notes of the near ties; a row without notes writes its
// results, a row with notes goes to the queue that k_cd_tie_check finishes.
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
    if (!cd_prologue<B, FULL>(a, tri, bar, i, row_ok, lane, t, st)) return;
    if (!row_ok) return;
    const float s = a.scale[i * a.ngroups + a.b0 / a.gsize];
    if constexpr (TIE) {
        TieWarp &me = reinterpret_cast<TieWarp *>(cd_smem + C::PACK + 4)[warp];
        if (lane == 0) me.nev = 0;
        __syncwarp();
        chg_decide_rec<B, FULL>(tri, a.d + a.b0, a.bw, a.maxq, s * s, a.rowdf != nullptr, lane, t, st, code, dlt,
                                dfacc, a.tie_eps, me.fj, me.fc, 0, -1, me.ev, &me.nev);
        const int nev = me.nev;
        if (nev > 0) {
            // the row waits for the check kernel: its notes, final and start codes to the queue,
            // and what the check reads starts toward L2
            int slot = 0;
            if (lane == 0) slot = static_cast<int>(atomicAdd(a.tq_cnt, 1u));
            slot = __shfl_sync(0xffffffffu, slot, 0);
            const double dfw = warp_sum(dfacc);
            TieEntry &e = a.tq[slot];
            if (lane == 0) {
                e.i = i;
                e.df = dfw;
                e.nev = nev;
            }
            if (lane < kMaxEv) e.ev[lane] = me.ev[lane];
            float *cr = a.tq_rows + static_cast<int64_t>(slot) * 2 * B, *sr = cr + B;
#pragma unroll
            for (int h = 0; h < CPL; ++h) {
                cr[32 * h + lane] = code[h];
                sr[32 * h + lane] = st[h];
            }
            tie_prefetch_row(a, i, lane, 32);
            const int ne = nev < kMaxEv ? nev : kMaxEv;
            for (int k = 0; k < ne; ++k) tie_prefetch_srow(a, a.b0 + me.ev[k], lane, 32);
            return;
        }
    } else {
        chg_decide<B, FULL>(tri, a.d + a.b0, a.bw, a.maxq, s * s, a.rowdf != nullptr, lane, t, st, code, dlt, dfacc);
    }
    if (a.rowdf) {
        dfacc = warp_sum(dfacc);
        if (lane == 0) a.rowdf[i] += dfacc;
    }
    chg_write<B, FULL>(a, i, lane, code, dlt);
}

// Shared memory of the check kernel: the packed block (copied only when a row must
// decide again) and its barrier, the entry's final and start codes, the forced
// decisions and notes, the reduction slots of the CTA-wide recompute.
template <int B>
__host__ __device__ constexpr int tie_check_smem_bytes() {
    return (CdCfg<B>::PACK + 4) * 4 + 2 * B * 4 + static_cast<int>(sizeof(TieWarp)) + 34 * 8;
}

// The near-tie check after a change-driven launch (same arguments): each CTA takes
// queued rows in turn.  A row's notes are checked in column order against beta~
// recomputed exactly by the whole CTA (coop_tie_beta, over the row's state at that
// decision: columns before it final, after it at their start codes); at the first
// wrong one the row decides again from the block's start (R holds it) with that
// column forced, and its new notes are checked in the next round (at most
// kMaxForced forced decisions; a row that uses them up keeps its last decisions, in
// practice never reached).  Then the row's results are written.  The last CTA out
// resets the queue's counters.
template <int B, bool FULL>
__global__ void __launch_bounds__(1024, 1) k_cd_tie_check(const __grid_constant__ CdArgs a) {
    if (a.gate && *a.gate != a.gate_run) return;   // uniform: the list form of the sweep runs
    using C = CdCfg<B>;
    constexpr int CPL = C::CPL;
    extern __shared__ __align__(16) float cd_smem[];
    float *tri = cd_smem;
    uint64_t *bar = reinterpret_cast<uint64_t *>(cd_smem + C::PACK);
    float *cr = cd_smem + C::PACK + 4, *sr = cr + B;
    TieWarp *me = reinterpret_cast<TieWarp *>(sr + B);
    double *red = reinterpret_cast<double *>(me + 1);
    __shared__ int s_copy;   // 0: block not copied, 1: copied and landed, -1: the wait gave up
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int bw = FULL ? B : a.bw;
    const int n = static_cast<int>(a.tq_cnt[0]);
    if (threadIdx.x == 0) {
        s_copy = 0;
        mbar_init(bar, 1);
        fence_mbar_init();
    }
    __syncthreads();
    const unsigned long long lim = a.wait_ns ? a.wait_ns : kWaitLimitNs;
    for (int e = blockIdx.x; e < n && s_copy >= 0; e += gridDim.x) {
        const TieEntry &E = a.tq[e];
        const int64_t i = E.i;
        const float *gcr = a.tq_rows + static_cast<int64_t>(e) * 2 * B;
        for (int l = threadIdx.x; l < B; l += blockDim.x) {
            cr[l] = gcr[l];
            sr[l] = gcr[B + l];
        }
        if (threadIdx.x == 0) {
            me->nev = E.nev;
            for (int k = 0; k < kMaxEv; ++k) me->ev[k] = E.ev[k];
            me->nf = 0;
            me->wrong_j = -1;
        }
        double df = E.df;
        __syncthreads();
        for (int round = 0; round <= kMaxForced; ++round) {
            // the notes in column order; the first wrong one stops the checks
            const int ne = me->nev < kMaxEv ? me->nev : kMaxEv;
            bool wrong = false;
            for (int k = 0; k < ne && !wrong; ++k) {
                const int j = me->ev[k];
                const double te = coop_tie_beta(a, i, a.b0, bw, j, cr, sr, red);
                const float ce = tie_code(te, a.maxq);
                if (ce != cr[j]) {
                    wrong = true;
                    if (threadIdx.x == 0) {
                        me->wrong_j = j;
                        me->wrong_c = ce;
                    }
                }
            }
            if (!wrong) break;
            // the packed block, once per CTA, for the rows that decide again
            if (s_copy == 0) {
                if (threadIdx.x == 0 && !a.skip_copy) {
                    constexpr uint32_t bytes = C::PACK * 4;
                    mbar_arrive_expect_tx(bar, bytes);
                    bulk_load(tri, a.tri + (a.b0 / B) * C::PACK, bytes, bar);
                }
                const bool ok = mbar_wait_bounded_ns(bar, 0u, nullptr, lim);
                __syncthreads();   // every thread has read s_copy == 0 and waited
                if (threadIdx.x == 0) {
                    s_copy = ok ? 1 : -1;
                    if (!ok) set_error(a.err, ERR_TIMEOUT);
                }
                __syncthreads();
                if (s_copy < 0) break;
            }
            if (warp == 0) {
                __syncwarp();
                const int wj = me->wrong_j;
                __syncwarp();
                if (lane == 0) {
                    if (me->nf < kMaxForced) {
                        me->fj[me->nf] = wj;
                        me->fc[me->nf] = me->wrong_c;
                        me->nf += 1;
                    }
                    me->nev = 0;
                    me->wrong_j = -1;
                }
                __syncwarp();
                float t[CPL], st[CPL], code[CPL], dlt[CPL];
#pragma unroll
                for (int h = 0; h < CPL; ++h) {
                    const int l = 32 * h + lane;
                    t[h] = (FULL || l < bw) ? a.R[i * a.ldr + a.b0 + l] : 0.0f;
                    st[h] = sr[l];
                }
                const float s = a.scale[i * a.ngroups + a.b0 / a.gsize];
                double dfacc = 0.0;
                chg_decide_rec<B, FULL>(tri, a.d + a.b0, a.bw, a.maxq, s * s, a.rowdf != nullptr, lane, t, st, code,
                                        dlt, dfacc, a.tie_eps, me->fj, me->fc, me->nf, wj, me->ev, &me->nev);
                if (round == kMaxForced && lane == 0) me->nev = 0;
                df = warp_sum(dfacc);
#pragma unroll
                for (int h = 0; h < CPL; ++h) cr[32 * h + lane] = code[h];
                __syncwarp();
            }
            __syncthreads();
        }
        if (s_copy < 0) break;
        // the row's results
        if (warp == 0) {
            float code[CPL], dlt[CPL];
#pragma unroll
            for (int h = 0; h < CPL; ++h) {
                const int l = 32 * h + lane;
                code[h] = cr[l];
                dlt[h] = sr[l] - code[h];
            }
            if (a.rowdf && lane == 0) a.rowdf[i] += df;
            chg_write<B, FULL>(a, i, lane, code, dlt);
        }
        __syncthreads();   // cr, sr and the notes are rewritten for the next row
    }
    if (threadIdx.x == 0) {
        // an issued copy has landed before the CTA leaves (bounded once more after a
        // wait that gave up)
        if (s_copy < 0 && !a.skip_copy) mbar_wait_bounded_ns(bar, 0u, nullptr, lim);
        // the last CTA out resets the queue for the next launch
        __threadfence();
        if (atomicAdd(a.tq_cnt + 1, 1u) == gridDim.x - 1) {
            a.tq_cnt[0] = 0u;
            a.tq_cnt[1] = 0u;
            __threadfence();
        }
    }
}

template <int B, bool FULL>
static cudaError_t launch_cd_tie_check_b(const CdArgs &a, int nsm, cudaStream_t s) {
    constexpr int smem = tie_check_smem_bytes<B>();
    cudaError_t e = cudaFuncSetAttribute(k_cd_tie_check<B, FULL>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    k_cd_tie_check<B, FULL><<<static_cast<unsigned>(nsm), 1024, smem, s>>>(a);
    return cudaGetLastError();
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

template <int B, bool FULL, bool SEQ, bool RELAX = false, bool DF = false, bool TIE = false>
static cudaError_t launch_cd_block_b(const CdArgs &a, int nsm, cudaStream_t s) {
    using C = CdCfg<B>;
    if (a.nsplit > C::MAX_SPLITS) return cudaErrorInvalidValue;
    auto kern = [] {
        if constexpr (SEQ) return k_cd_block_seq<B, FULL, RELAX, DF, TIE>;
        else return k_cd_block_chg<B, FULL, TIE>;
    }();
    // one CTA per SM when the rows allow it (the packed block is shared by the CTA's rows)
    int64_t warps = ceil_div(a.q, nsm);
    if (warps > C::MAX_WARPS) warps = C::MAX_WARPS;
    if (warps < 1) warps = 1;
    // the sequential kernel keeps one row of beta~ per warp (DF), and one row of the
    // codes decided in the visit and one snapshot row (near-tie refinement), after the
    // packed block; the change-driven kernel the notes of each warp's row
    const int rows = static_cast<int>(warps) * B * 4;
    const int smem = SEQ ? (C::PACK + 4) * 4 + (DF ? rows : 0) + (TIE ? 2 * rows : 0)
                         : (C::PACK + 4) * 4 + (TIE ? static_cast<int>(warps) * static_cast<int>(sizeof(TieWarp)) : 0);
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    const unsigned grid = static_cast<unsigned>(ceil_div(a.q, warps));
    kern<<<grid, static_cast<unsigned>(32 * warps), smem, s>>>(a);
    return cudaGetLastError();
}

// The near-tie check after a change-driven launch with the refinement.
template <int B, bool FULL>
static cudaError_t launch_cd_tie_check_f(const CdArgs &a, int nsm, cudaStream_t s) {
    if (!a.tq || !a.tq_rows || !a.tq_cnt) return cudaErrorInvalidValue;
    return launch_cd_tie_check_b<B, FULL>(a, nsm, s);
}

// The change-driven kernel (integer changes, !a.frac), with or without the
// near-tie refinement.
template <int B, bool FULL>
static cudaError_t launch_cd_block_chg_f(const CdArgs &a, int nsm, cudaStream_t s) {
    return a.tie_eps > 0.0f ? launch_cd_block_b<B, FULL, false, false, false, true>(a, nsm, s)
                            : launch_cd_block_b<B, FULL, false>(a, nsm, s);
}

// The sequential kernel (real-valued changes: the first sweep, relaxed sweeps and
// the sweep after one); the refinement variant serves the first sweep.
template <int B, bool FULL>
static cudaError_t launch_cd_block_seq_f(const CdArgs &a, int nsm, cudaStream_t s) {
    const bool tie = a.tie_eps > 0.0f;
    if (a.vout) return a.rowdf ? launch_cd_block_b<B, FULL, true, true, true>(a, nsm, s) : cudaErrorInvalidValue;
    if (tie && a.first_sweep && !a.vstart)
        return a.rowdf ? launch_cd_block_b<B, FULL, true, false, true, true>(a, nsm, s)
                       : launch_cd_block_b<B, FULL, true, false, false, true>(a, nsm, s);
    return a.rowdf ? launch_cd_block_b<B, FULL, true, false, true>(a, nsm, s)
                   : launch_cd_block_b<B, FULL, true, false, false>(a, nsm, s);
}

// One kernel family at block width B (SEQ: sequential, else change-driven), for a
// full block (FULL) or the ragged last one.  Instantiated in the qe_sweep_*.cu units.
template <int B, bool SEQ, bool FULL>
cudaError_t launch_cd_block_k(const CdArgs &a, int nsm, cudaStream_t s) {
    if constexpr (SEQ)
        return launch_cd_block_seq_f<B, FULL>(a, nsm, s);
    else
        return launch_cd_block_chg_f<B, FULL>(a, nsm, s);
}

// The near-tie check at block width B (instantiated with the change-driven kernel).
template <int B, bool FULL>
cudaError_t launch_cd_tie_check_k(const CdArgs &a, int nsm, cudaStream_t s) {
    return launch_cd_tie_check_f<B, FULL>(a, nsm, s);
}

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

// The persistent change-list kernel at block width B (grouped grids or not, with or
// without the near-tie refinement).  Instantiated in the qe_sweep_*.cu units.
template <int B>
cudaError_t launch_cd_rows_k(const CdArgs &a, int t_begin, int t_end, double *rowdf_t, uint8_t *sweep_codes,
                             int f, int m, int fl, int nsm, cudaStream_t s) {
    if (a.grouped)
        return a.tie_eps > 0.0f ? launch_cd_rows_b<B, true, true>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s)
                                : launch_cd_rows_b<B, true, false>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s);
    return a.tie_eps > 0.0f ? launch_cd_rows_b<B, false, true>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s)
                            : launch_cd_rows_b<B, false, false>(a, t_begin, t_end, rowdf_t, sweep_codes, f, m, fl, nsm, s);
}

#define QE_SWEEP_ROWS_SIG (const CdArgs &, int, int, double *, uint8_t *, int, int, int, int, cudaStream_t)
#define QE_SWEEP_BLOCK_SIG (const CdArgs &, int, cudaStream_t)
#ifndef QE_SWEEP_INSTANTIATE
extern template cudaError_t launch_cd_block_k<64, true, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<128, true, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<256, true, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<64, true, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<128, true, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<256, true, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<64, false, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<128, false, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<256, false, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<64, false, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<128, false, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_block_k<256, false, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_tie_check_k<64, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_tie_check_k<64, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_tie_check_k<128, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_tie_check_k<128, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_tie_check_k<256, true> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_tie_check_k<256, false> QE_SWEEP_BLOCK_SIG;
extern template cudaError_t launch_cd_rows_k<64> QE_SWEEP_ROWS_SIG;
extern template cudaError_t launch_cd_rows_k<128> QE_SWEEP_ROWS_SIG;
extern template cudaError_t launch_cd_rows_k<256> QE_SWEEP_ROWS_SIG;
#endif

}  // namespace qe
