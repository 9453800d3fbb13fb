// Tensor-core GEMM of libqe: D[M x N] = sum_t A_{pa(t)} . B_{pb(t)}^T over K, on
// tcgen05 (bf16 x bf16 -> fp32 accumulators in TMEM), operands fed by TMA in
// 128-byte-swizzled K-major tiles.  One kernel serves four contractions of the
// method, selected by the epilogue:
//   Sigma = X X^T                         (Lemma 1; upper tiles + mirror)
//   P = W (I + Sigma_bar)                 (Algorithm 3, "P = W Sigma^norm")
//   R = (P - s (C - z) Sigma_bar) / s + z  (Algorithm 3, "P_hat = What Sigma^norm"), grid steps
//   partial_k = Delta' Sigma_bar[0:b0, block]  (Eq. cd-update-closed-2, the
//                                          dW_{:,1:j} Sigma^norm_{1:j,j} term,
//                                          deferred per column block, split-K)
// fp32 accuracy for the Sigma_bar products comes from splitting an fp32 operand
// into three bf16 planes (hi + mid + lo, 24 significant bits) and summing the
// cross products down to 2^-16 relative order in the same accumulator (planes
// are stacked along rows in one tensor map).
//
// Warp roles (320 threads): warp 0 lane 0 issues TMA, warp 1 lane 0 issues MMA
// (warp 1 owns the TMEM allocation: two accumulation buffers), warps 2..9 fold
// the chunk partial sums into fp32 registers and run the epilogue (warp w reads
// TMEM lanes 32 (w mod 4) .. +31 = output rows, half of the columns each).
#include <cudaTypedefs.h>

#include "qe_common.cuh"
#include "qe_internal.h"

namespace qe {

template <int BN>
struct GemmCfg {
    static constexpr int BM = 128;
    static constexpr int BK = 64;                       // 64 bf16 = one 128-byte swizzle row
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int STAGES = (BN == 256) ? 4 : (BN == 128) ? 6 : 8;
    static constexpr int TMEM_COLS = 2 * BN;           // two accumulation buffers
    static constexpr int HALF = BN / 2;                // columns per epilogue thread
    static constexpr int THREADS = 320;                // producer, MMA, 8 epilogue warps
    static constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 + 256;
    static_assert(BN == 64 || BN == 128 || BN == 256, "BN");
    static_assert(SMEM_BYTES <= 232448, "smem");
    static_assert(8 * 32 * (HALF + 4) * 4 <= STAGES * STAGE_BYTES, "epilogue staging fits the ring");
};

// Virtual K steps (k-block x operand-plane product) accumulated in one TMEM
// buffer before the epilogue warps fold it into fp32 registers.  The tensor-core
// accumulator loses up to about one unit in the last place per accumulate, with
// a bias toward zero (measured: ~1e-5 relative after 256 accumulates), so long K
// is summed as short chunks (4 MMA per step -> 16 accumulates per chunk, a
// relative bias of ~1e-6) whose partial sums are added with round-to-nearest
// fp32 on the CUDA cores.  Folding every 2 steps cost 9% of Sigma's time in TMEM
// traffic; every 8 steps gains ~1% more for twice the bias.
constexpr int kChunkSteps = 4;

// Sigma's tile order.  Only the tiles on or above the diagonal run (the mirror
// writes the rest).  They are taken in groups of kSigmaGroupM consecutive tile
// rows; inside a group the tile row runs fastest, then the tile column, from the
// first column that reaches the group's diagonal.  A wave of CTAs then covers a
// compact patch of tiles: at a given k-step it reads a few hundred kilobytes of
// distinct rows of X, where row-by-row order (one tile row against 152 tile
// columns) read several megabytes per k-step and left the GEMM waiting on DRAM
// for wide layers.
constexpr int kSigmaGroupM = 8;

// Tiles of group gi (tile rows [gi * kSigmaGroupM, ...)), counting from the
// first tile column whose BN columns reach the group's first row.
__host__ __device__ __forceinline__ int64_t sigma_group_tiles(int gi, int mt, int nt, int BN) {
    const int mlo = gi * kSigmaGroupM;
    const int gm = (mt - mlo) < kSigmaGroupM ? (mt - mlo) : kSigmaGroupM;
    const int ns = static_cast<int>((static_cast<int64_t>(mlo) * 128) / BN);
    return static_cast<int64_t>(gm) * (nt - ns);
}

__host__ __device__ __forceinline__ int64_t sigma_tiles(int mt, int nt, int BN) {
    int64_t t = 0;
    for (int gi = 0; gi * kSigmaGroupM < mt; ++gi) t += sigma_group_tiles(gi, mt, nt, BN);
    return t;
}

// Linear tile id -> (tile row, tile column) in the grouped order.
__host__ __device__ __forceinline__ void sigma_tile(int64_t id, int mt, int nt, int BN, int &m, int &n) {
    int gi = 0;
    for (;;) {
        const int64_t t = sigma_group_tiles(gi, mt, nt, BN);
        if (id < t || (gi + 1) * kSigmaGroupM >= mt) break;
        id -= t;
        ++gi;
    }
    const int mlo = gi * kSigmaGroupM;
    const int gm = (mt - mlo) < kSigmaGroupM ? (mt - mlo) : kSigmaGroupM;
    const int ns = static_cast<int>((static_cast<int64_t>(mlo) * 128) / BN);
    m = mlo + static_cast<int>(id % gm);
    n = ns + static_cast<int>(id / gm);
}

__device__ __forceinline__ float load_w(const GemmArgs &g, int64_t r, int64_t c) {
    if (g.w_is_bf16)
        return __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(g.W)[r * g.ldw + c]);
    return reinterpret_cast<const float *>(g.W)[r * g.ldw + c];
}

// Epilogue for one thread: output row r, columns [c0, c0 + 32) of the window.
// `objacc` collects the fused objective terms of EPI_RFULL (when requested).
// GR: grouped grids possible (per-group scales, the absolute residual form); the
// per-row kernel is compiled without them.
template <bool GR>
__device__ __forceinline__ void epilogue_row(const GemmArgs &g, int r, int c0, const float (&v)[32],
                                             int split, double &objacc) {
    if (r >= g.M) return;
    const int64_t rr = r;
    switch (g.mode) {
        case EPI_SIGMA: {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const int c = c0 + i;
                if (c < g.N && c >= r) {
                    float *a = g.out + rr * g.ldo + c;
                    float *b = g.out + static_cast<int64_t>(c) * g.ldo + r;
                    if (g.accumulate) {
                        const float nv = *a + v[i];
                        *a = nv;
                        if (c != r) *b = nv;
                    } else {
                        *a = v[i];
                        if (c != r) *b = v[i];
                    }
                }
            }
            break;
        }
        case EPI_PINIT: {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                const int c = c0 + i;
                if (c < g.N) g.out[rr * g.ldo + c] = load_w(g, rr, c) + v[i];
            }
            break;
        }
        case EPI_RFULL: {
            // R in grid-step units: (P - s (C - z) Sigma_bar) / s + z = P / s - acc + z; with
            // grouped grids (absolute) acc = s_g (C - z_g) Sigma_bar, R = (P - acc) / s_g + z_g
            // (the 32 columns lie in one group)
            const int64_t gi = (GR && g.ngroups > 1) ? rr * g.ngroups + c0 / g.gsize : rr;
            const float s = g.scale[gi];
            const float zz = g.zero[gi];
            const float *prow = g.P + rr * g.ldp;
            float *orow = g.out + rr * g.ldo;
            float o[32];
            const bool full = c0 + 32 <= g.N;
            if (GR && g.absolute) {
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const int c = c0 + i;
                    o[i] = 0.0f;
                    if (c < g.N) orow[c] = o[i] = __fdiv_rn(prow[c] - v[i], s) + zz;
                }
            } else if (full && ((g.ldo | g.ldp) & 3) == 0) {
#pragma unroll
                for (int i = 0; i < 32; i += 4) {
                    const float4 pv = *reinterpret_cast<const float4 *>(prow + c0 + i);
                    o[i] = (__fdiv_rn(pv.x, s) - v[i + 0]) + zz;
                    o[i + 1] = (__fdiv_rn(pv.y, s) - v[i + 1]) + zz;
                    o[i + 2] = (__fdiv_rn(pv.z, s) - v[i + 2]) + zz;
                    o[i + 3] = (__fdiv_rn(pv.w, s) - v[i + 3]) + zz;
                    *reinterpret_cast<float4 *>(orow + c0 + i) = make_float4(o[i], o[i + 1], o[i + 2], o[i + 3]);
                }
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const int c = c0 + i;
                    o[i] = 0.0f;
                    if (c < g.N) orow[c] = o[i] = (__fdiv_rn(prow[c], s) - v[i]) + zz;
                }
            }
            if (g.obj_part) {
                // (D Sigma)_ij = d_j (R_ij - What_ij) = d_j s (R'_ij - C_ij) with R' = R / s + z:
                // f = sum D_ij d_j s (R'_ij - C_ij)
                const float z = zz;
                float part = 0.0f;
                const bool vec = full && g.w_is_bf16 && (g.ldw % 8) == 0 && (g.ldc % 16) == 0 &&
                                 (g.Hd == nullptr || (g.ldh % 4) == 0);
                if (vec) {
                    const uint4 *wp = reinterpret_cast<const uint4 *>(
                        reinterpret_cast<const __nv_bfloat16 *>(g.W) + rr * g.ldw + c0);
                    const uint4 *cp = reinterpret_cast<const uint4 *>(g.codes + rr * g.ldc + c0);
                    const float4 *dp = reinterpret_cast<const float4 *>(g.dvec + c0);
                    const float4 *hp = g.Hd ? reinterpret_cast<const float4 *>(g.Hd + rr * g.ldh + c0) : nullptr;
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        union { uint4 v; uint8_t b[16]; } cu;
                        cu.v = cp[h];
#pragma unroll
                        for (int w8 = 0; w8 < 2; ++w8) {
                            union { uint4 v; __nv_bfloat16 e[8]; } wu;
                            wu.v = wp[2 * h + w8];
#pragma unroll
                            for (int q4 = 0; q4 < 2; ++q4) {
                                const float4 d4 = dp[4 * h + 2 * w8 + q4];
                                const float dd[4] = {d4.x, d4.y, d4.z, d4.w};
                                const float4 h4 = hp ? hp[4 * h + 2 * w8 + q4] : make_float4(0.f, 0.f, 0.f, 0.f);
                                const float hh[4] = {h4.x, h4.y, h4.z, h4.w};
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    const int i = 16 * h + 8 * w8 + 4 * q4 + e;
                                    const float cj = static_cast<float>(cu.b[i - 16 * h]);
                                    const float wh = s * (cj - z);
                                    const float t = (__bfloat162float(wu.e[4 * q4 + e]) - wh) - hh[e];
                                    const float dj = dd[e] > 0.0f ? dd[e] : 0.0f;
                                    part += t * dj * (s * (o[i] - cj));
                                }
                            }
                        }
                    }
                } else {
#pragma unroll
                    for (int i = 0; i < 32; ++i) {
                        const int c = c0 + i;
                        if (c < g.N) {
                            const float dj = g.dvec[c];
                            if (dj > 0.0f) {
                                const float cj = static_cast<float>(g.codes[rr * g.ldc + c]);
                                const float wh = s * (cj - z);
                                float t = load_w(g, rr, c) - wh;
                                if (g.Hd) t -= g.Hd[rr * g.ldh + c];
                                part += t * dj * (s * (o[i] - cj));
                            }
                        }
                    }
                }
                objacc += static_cast<double>(part);
            }
            break;
        }
        case EPI_TRAIL: {
            float *orow = g.out + static_cast<int64_t>(split) * g.split_stride + rr * g.ldo;
            if (c0 + 32 <= g.N && (g.ldo & 3) == 0 && (g.split_stride & 3) == 0) {
#pragma unroll
                for (int i = 0; i < 32; i += 4)
                    *reinterpret_cast<float4 *>(orow + c0 + i) =
                        make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (c0 + i < g.N) orow[c0 + i] = v[i];
            }
            break;
        }
        default:
            break;
    }
}

template <int N>
__device__ __forceinline__ void ld_fv(const float *p, float *v) {
    if constexpr (N == 4) {
        const float4 t = *reinterpret_cast<const float4 *>(p);
        v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
    } else if constexpr (N == 2) {
        const float2 t = *reinterpret_cast<const float2 *>(p);
        v[0] = t.x; v[1] = t.y;
    } else {
        v[0] = *p;
    }
}

template <int N>
__device__ __forceinline__ void st_fv(float *p, const float *v) {
    if constexpr (N == 4) *reinterpret_cast<float4 *>(p) = make_float4(v[0], v[1], v[2], v[3]);
    else if constexpr (N == 2) *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
    else *p = v[0];
}

// Epilogue of the P, residual and trailing GEMMs.  Each epilogue thread holds one
// row of the tile, so writing from registers would touch 32 rows per warp
// access; instead the warp's 32 rows x HALF columns go through shared memory
// (the operand ring is idle once the last chunk has been folded) and are then
// processed row by row with the lanes across the columns: every global load and
// store becomes one contiguous access.  `objacc` collects the fused objective of
// EPI_RFULL (when requested).
template <int HALF>
__device__ __forceinline__ void epilogue_rows(const GemmArgs &g, float *stg, int r0, int c0, int lane,
                                              const float (&acc)[HALF], int split, double &objacc) {
    constexpr int LD = HALF + 4;          // padded row: spreads the column-wise writes over the banks
    constexpr int VEC = HALF / 32;        // columns per lane
#pragma unroll
    for (int i = 0; i < HALF; i += 4)
        *reinterpret_cast<float4 *>(stg + lane * LD + i) = make_float4(acc[i], acc[i + 1], acc[i + 2], acc[i + 3]);
    __syncwarp();
    const int cl = c0 + VEC * lane;
    const bool full = cl + VEC <= g.N;
    for (int rr = 0; rr < 32; ++rr) {
        const int r = r0 + rr;
        if (r >= g.M) break;
        const int64_t rw = r;
        float v[VEC];
        ld_fv<VEC>(stg + rr * LD + VEC * lane, v);
        if (g.colscale) {
#pragma unroll
            for (int e = 0; e < VEC; ++e) v[e] *= (cl + e < g.N) ? g.colscale[cl + e] * g.ascale : 1.0f;
        }
        if (g.rowscale) {
            const float rs = g.rowscale[rw];
#pragma unroll
            for (int e = 0; e < VEC; ++e) v[e] *= rs;
        }
        if (g.mode == EPI_TRAIL) {
            float *orow = g.out + static_cast<int64_t>(split) * g.split_stride + rw * g.ldo;
            if (full) st_fv<VEC>(orow + cl, v);
            else
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    if (cl + e < g.N) orow[cl + e] = v[e];
        } else if (g.mode == EPI_PINIT) {
            float *orow = g.out + rw * g.ldo;
            float o[VEC];
#pragma unroll
            for (int e = 0; e < VEC; ++e) o[e] = (cl + e < g.N) ? load_w(g, rw, cl + e) + v[e] : 0.0f;
            if (full) st_fv<VEC>(orow + cl, o);
            else
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    if (cl + e < g.N) orow[cl + e] = o[e];
        } else {   // EPI_RFULL: R in grid-step units, P / s - acc + z
            const float sc = g.scale[r];
            const float zz = g.zero[r];
            const float *prow = g.P + rw * g.ldp;
            float *orow = g.out + rw * g.ldo;
            float pv[VEC], o[VEC];
            if (full) ld_fv<VEC>(prow + cl, pv);
            else
#pragma unroll
                for (int e = 0; e < VEC; ++e) pv[e] = (cl + e < g.N) ? prow[cl + e] : 0.0f;
#pragma unroll
            for (int e = 0; e < VEC; ++e) o[e] = (__fdiv_rn(pv[e], sc) - v[e]) + zz;
            if (full) st_fv<VEC>(orow + cl, o);
            else
#pragma unroll
                for (int e = 0; e < VEC; ++e)
                    if (cl + e < g.N) orow[cl + e] = o[e];
            if (g.obj_part) {
                // (D Sigma)_ij = d_j (R_ij - What_ij) = d_j s (R'_ij - C_ij) with R' = R / s + z:
                // f = sum D_ij d_j s (R'_ij - C_ij), D = W - What (- H)
                float part = 0.0f;
                if constexpr (VEC == 4) {
                    // 4 columns per lane: W as 4 bf16 (8 bytes), codes as one word, d and H as float4
                    const bool vec = full && g.w_is_bf16 && (g.ldw % 4) == 0 && (g.ldc % 4) == 0 &&
                                     ((reinterpret_cast<uintptr_t>(g.W) & 7u) == 0) &&
                                     ((reinterpret_cast<uintptr_t>(g.codes) & 3u) == 0) &&
                                     (g.Hd == nullptr || (g.ldh % 4) == 0);
                    if (vec) {
                        const uint2 wraw = *reinterpret_cast<const uint2 *>(
                            reinterpret_cast<const __nv_bfloat16 *>(g.W) + rw * g.ldw + cl);
                        const uint32_t craw = *reinterpret_cast<const uint32_t *>(g.codes + rw * g.ldc + cl);
                        float dv[4], hv[4] = {0.f, 0.f, 0.f, 0.f};
                        ld_fv<4>(g.dvec + cl, dv);
                        if (g.Hd) ld_fv<4>(g.Hd + rw * g.ldh + cl, hv);
                        const __nv_bfloat162 w01 = *reinterpret_cast<const __nv_bfloat162 *>(&wraw.x);
                        const __nv_bfloat162 w23 = *reinterpret_cast<const __nv_bfloat162 *>(&wraw.y);
                        const float wv[4] = {__low2float(w01), __high2float(w01), __low2float(w23), __high2float(w23)};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const float cj = static_cast<float>((craw >> (8 * e)) & 0xffu);
                            const float wh = sc * (cj - zz);
                            const float t = (wv[e] - wh) - hv[e];
                            const float dj = dv[e] > 0.0f ? dv[e] : 0.0f;
                            part += t * dj * (sc * (o[e] - cj));
                        }
                        objacc += static_cast<double>(part);
                        continue;
                    }
                }
#pragma unroll
                for (int e = 0; e < VEC; ++e) {
                    const int c = cl + e;
                    if (c < g.N) {
                        const float dj = g.dvec[c];
                        if (dj > 0.0f) {
                            const float cj = static_cast<float>(g.codes[rw * g.ldc + c]);
                            const float wh = sc * (cj - zz);
                            float t = load_w(g, rw, c) - wh;
                            if (g.Hd) t -= g.Hd[rw * g.ldh + c];
                            part += t * dj * (sc * (o[e] - cj));
                        }
                    }
                }
                objacc += static_cast<double>(part);
            }
        }
    }
}

template <int BN, bool GR>
__global__ void __launch_bounds__(320, 1)
    k_tc_gemm(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
              const GemmArgs g) {
    using C = GemmCfg<BN>;
    if (g.gate && *g.gate != g.gate_run) return;   // uniform: the other form of the sweep runs
    extern __shared__ uint8_t smem_raw[];
    const uint32_t pad = (1024u - (smem_u32(smem_raw) & 1023u)) & 1023u;
    uint8_t *smem = smem_raw + pad;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem + C::STAGES * C::STAGE_BYTES);
    uint64_t *empty = full + C::STAGES;
    uint64_t *acc_full = empty + C::STAGES;   // [2]: chunk accumulated in buffer b
    uint64_t *acc_empty = acc_full + 2;       // [2]: buffer b drained by the epilogue
    uint64_t *drain = acc_empty + 2;          // every MMA this CTA issued has completed
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(drain + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    // m_fast: consecutive CTAs walk down M, so a wave shares a few B column
    // slices (each read once from DRAM) instead of sweeping all of B.  Sigma:
    // the 1-D grid runs over the tiles on or above the diagonal in groups of
    // kSigmaGroupM tile rows (sigma_tile).
    int m0, n0;
    if (g.mode == EPI_SIGMA) {
        int mt_, nt_;
        sigma_tile(static_cast<int64_t>(blockIdx.x), static_cast<int>(ceil_div(g.M, C::BM)),
                   static_cast<int>(ceil_div(g.N, BN)), BN, mt_, nt_);
        m0 = mt_ * C::BM;
        n0 = nt_ * BN;
    } else {
        m0 = (g.m_fast ? blockIdx.x : blockIdx.y) * C::BM;
        n0 = (g.m_fast ? blockIdx.y : blockIdx.x) * BN;
    }
    // Sigma: a tile whose every element lies strictly below the diagonal is
    // produced by the mirror of its transpose (uniform exit, before any barrier).
    if (g.mode == EPI_SIGMA && n0 + BN <= m0) return;

    const int split = blockIdx.z;
    const int splits = gridDim.z;
    const int kb_lo = g.kb_begin + static_cast<int>((static_cast<long long>(g.kb_count) * split) / splits);
    const int kb_hi =
        g.kb_begin + static_cast<int>((static_cast<long long>(g.kb_count) * (split + 1)) / splits);
    const int nsteps = (kb_hi - kb_lo) * g.n_prod;
    const int nchunks = (nsteps + kChunkSteps - 1) / kChunkSteps;

    if (threadIdx.x == 0) {
        for (int s = 0; s < C::STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], 256);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tensormap(&ta);
        prefetch_tensormap(&tb);
    }
    if (warp == 1) tmem_alloc(tmem_slot, C::TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ---- TMA producer ----
            int st = 0;
            for (; st < nsteps; ++st) {
                const int s = st % C::STAGES;
                const uint32_t ph = (st / C::STAGES) & 1u;
                if (!mbar_wait_bounded(&empty[s], ph ^ 1u, abort_flag)) {
                    *abort_flag = 1;
                    set_error(g.err, ERR_TIMEOUT);
                    break;
                }
                const int kb = kb_lo + st / g.n_prod;
                const int t = st % g.n_prod;
                uint8_t *sa = smem + s * C::STAGE_BYTES;
                uint8_t *sb = sa + C::A_BYTES;
                mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);
                tma_load_2d(&ta, sa, &full[s], kb * C::BK, g.a_row0 + m0 + g.prod_a[t] * g.a_plane_rows);
                tma_load_2d(&tb, sb, &full[s], kb * C::BK, g.b_row0 + n0 + g.prod_b[t] * g.b_plane_rows);
            }
            // Drain: the last load into each stage has landed before the CTA releases
            // its shared memory (a wait that gave up elsewhere leaves loads unconsumed;
            // on the normal path these phases are complete and each test passes at once).
            for (int k = (st > C::STAGES ? st - C::STAGES : 0); k < st; ++k)
                mbar_wait_bounded(&full[k % C::STAGES], (k / C::STAGES) & 1u, nullptr);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---- MMA issuer: chunk c accumulates into TMEM buffer c & 1 ----
            const uint32_t idesc = g.f16 ? idesc_f16_f32(C::BM, BN) : idesc_bf16_f32(C::BM, BN);
            int st = 0;
            for (int c = 0; c < nchunks && !*abort_flag; ++c) {
                const int buf = c & 1;
                if (c >= 2 && !mbar_wait_bounded(&acc_empty[buf], ((c >> 1) - 1) & 1u, abort_flag)) {
                    *abort_flag = 1;
                    set_error(g.err, ERR_TIMEOUT);
                    break;
                }
                tc_fence_after();
                const uint32_t dst = tmem + static_cast<uint32_t>(buf * BN);
                const int st_end = (st + kChunkSteps < nsteps) ? st + kChunkSteps : nsteps;
                for (int first = 1; st < st_end; ++st, first = 0) {
                    const int s = st % C::STAGES;
                    const uint32_t ph = (st / C::STAGES) & 1u;
                    if (!mbar_wait_bounded(&full[s], ph, abort_flag)) {
                        *abort_flag = 1;
                        set_error(g.err, ERR_TIMEOUT);
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(smem + s * C::STAGE_BYTES);
                    const uint64_t da = smem_desc_k128(sa);
                    const uint64_t db = smem_desc_k128(sa + C::A_BYTES);
#pragma unroll
                    for (int k = 0; k < C::BK / 16; ++k)
                        mma_bf16_ss(dst, da + 2u * k, db + 2u * k, idesc, (first && k == 0) ? 0u : 1u);
                    mma_commit(&empty[s]);
                }
                mma_commit(&acc_full[buf]);   // arrives when this chunk's MMAs complete
            }
            // Drain: every MMA issued so far has completed before TMEM is released (on
            // the normal path they have by the time the epilogue folds the last chunk).
            mma_commit(drain);
            mbar_wait_bounded(drain, 0u, nullptr);
        }
    } else {
        // ---- epilogue warps 2..9: fold chunks into fp32 registers, then store ----
        const int quad = warp & 3;                    // TMEM lanes 32*quad .. +31
        const int half = (warp - 2) >> 2;             // columns [half*BN/2, +BN/2)
        const uint32_t tl = tmem + (static_cast<uint32_t>(quad * 32) << 16) +
                            static_cast<uint32_t>(half * C::HALF);
        float acc[C::HALF];
#pragma unroll
        for (int i = 0; i < C::HALF; ++i) acc[i] = 0.0f;
        bool ok = true;
        for (int c = 0; c < nchunks; ++c) {
            const int buf = c & 1;
            if (!mbar_wait_bounded(&acc_full[buf], (c >> 1) & 1u, abort_flag)) {
                ok = false;
                if (lane == 0) set_error(g.err, ERR_TIMEOUT);
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
#pragma unroll
            for (int q = 0; q < C::HALF / 32; ++q) {
                float v[32];
                tmem_ld_32x32b_x32(tl + static_cast<uint32_t>(buf * BN + q * 32), v);
#pragma unroll
                for (int i = 0; i < 32; ++i) acc[q * 32 + i] += v[i];
            }
            tc_fence_before();
            mbar_arrive(&acc_empty[buf]);
        }
        double objacc = 0.0;
        if (ok && *abort_flag == 0) {
            // Sigma (mirrored writes) and the residual refresh (already vectorized along the
            // thread's row, and its fused objective reads several arrays per element) write
            // from registers; P and the trailing partials go row-wise through shared memory
            if (g.mode == EPI_SIGMA || g.mode == EPI_RFULL) {
                const int r = m0 + quad * 32 + lane;
#pragma unroll
                for (int q = 0; q < C::HALF / 32; ++q) {
                    const int c0 = n0 + half * C::HALF + q * 32;
                    if (c0 < g.N) {
                        float v[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = acc[q * 32 + i];
                        if (g.colscale) {
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] *= (c0 + i < g.N) ? g.colscale[c0 + i] * g.ascale : 1.0f;
                        }
                        epilogue_row<GR>(g, r, c0, v, split, objacc);
                    }
                }
            } else {
                // every MMA has completed (the last chunk was folded), so the operand
                // ring is free: 8 warps x 32 rows x (HALF + 4) floats fit in it
                float *stg = reinterpret_cast<float *>(smem) + (warp - 2) * 32 * (C::HALF + 4);
                epilogue_rows<C::HALF>(g, stg, m0 + quad * 32, n0 + half * C::HALF, lane, acc, split, objacc);
            }
        }
        if (g.obj_part) {   // one fp64 partial per epilogue warp, reduced later in a fixed order
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) objacc += __shfl_xor_sync(0xffffffffu, objacc, o);
            if (lane == 0)
                g.obj_part[(static_cast<int64_t>(blockIdx.y) * gridDim.x + blockIdx.x) * 8 + (warp - 2)] = objacc;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) tmem_dealloc(tmem, C::TMEM_COLS);
}

// ---- host side ---------------------------------------------------------------
static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

static bool get_encode() {
    if (g_encode) return true;
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult qres;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &qres) != cudaSuccess ||
        qres != cudaDriverEntryPointSuccess || fn == nullptr)
        return false;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return true;
}

bool make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols, uint64_t ld,
                    uint32_t box_rows) {
    if (!get_encode()) return false;
    if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || ((ld * 2) & 15u) != 0) return false;
    if (rows == 0 || cols == 0 || box_rows == 0 || box_rows > 256) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {ld * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estr[2] = {1, 1};
    const CUresult r =
        g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides,
                 box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_tmap_f16(CUtensorMap *map, const void *base, uint64_t rows, uint64_t cols, uint64_t ld,
                   uint32_t box_rows) {
    if (!get_encode()) return false;
    if ((reinterpret_cast<uintptr_t>(base) & 15u) != 0 || ((ld * 2) & 15u) != 0) return false;
    if (rows == 0 || cols == 0 || box_rows == 0 || box_rows > 256) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {ld * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t estr[2] = {1, 1};
    const CUresult r =
        g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(base), dims, strides,
                 box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <int BN, bool GR>
static cudaError_t launch_bn(const CUtensorMap &ta, const CUtensorMap &tb, const GemmArgs &g,
                             int splits, cudaStream_t s) {
    using C = GemmCfg<BN>;
    cudaError_t e = cudaFuncSetAttribute(k_tc_gemm<BN, GR>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    const unsigned nt = static_cast<unsigned>(ceil_div(g.N, BN)), mt = static_cast<unsigned>(ceil_div(g.M, C::BM));
    dim3 grid(g.m_fast ? mt : nt, g.m_fast ? nt : mt, static_cast<unsigned>(splits));
    if (g.mode == EPI_SIGMA) {
        const int64_t tiles = sigma_tiles(static_cast<int>(mt), static_cast<int>(nt), BN);
        if (tiles > 0x7fffffffll) return cudaErrorInvalidValue;
        grid = dim3(static_cast<unsigned>(tiles), 1, static_cast<unsigned>(splits));
    }
    k_tc_gemm<BN, GR><<<grid, C::THREADS, C::SMEM_BYTES, s>>>(ta, tb, g);
    return cudaGetLastError();
}

cudaError_t launch_tc_gemm(int BN, const CUtensorMap &ta, const CUtensorMap &tb, const GemmArgs &g,
                           int splits, cudaStream_t s) {
    if (g.M <= 0 || g.N <= 0 || splits < 1 || g.n_prod < 1 || g.n_prod > 6)
        return cudaErrorInvalidValue;
    if (g.mode != EPI_SIGMA && (g.m_fast ? ceil_div(g.N, BN) : ceil_div(g.M, 128)) > 65535) return cudaErrorInvalidValue;
    if (splits > 65535) return cudaErrorInvalidValue;
    switch (BN) {
        case 64: return launch_bn<64, false>(ta, tb, g, splits, s);
        case 128: return launch_bn<128, false>(ta, tb, g, splits, s);
        case 256:   // grouped grids only reach the residual GEMM, which runs 128 x 256 tiles
            return (g.ngroups > 1 || g.absolute) ? launch_bn<256, true>(ta, tb, g, splits, s)
                                                 : launch_bn<256, false>(ta, tb, g, splits, s);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace qe
