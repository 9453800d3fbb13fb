// C ABI of libqe (include/qe.h): argument checks, workspace layout and the
// stream-ordered schedule of the QuantEase kernels.
//
// qe_quantize_layer, per layer (Algorithm 3 of Sec. 3.2, blocked by columns):
//   grid(W) -> s, z;  Sigma -> d, Sigma_bar^T planes;  P = W (I + Sigma_bar);
//   R = W (the first sweep starts at What = W, Sec. 3.1);
//   per sweep:  per column block [b0, b0+B):
//                   partial = Delta'[:, 0:b0] Sigma_bar[0:b0, block]   (tcgen05, split-K)
//                   sequential in-block updates -> codes, C - z, Delta'
//               R = P - s (C - z) Sigma_bar                           (tcgen05)
//               f = sum D_ij d_j (R_ij - What_ij)                     (reduction)
// qe_quantize_layer_outlier adds, per iteration (Algorithm 4 of Sec. 4.3):
//   T = H + 2 eta d_j (R - What);  H = P_s(T);  P = P_W - H (I + Sigma_bar);
//   R += P_new - P_old.
#include <math.h>
#include <stdio.h>
#include <string.h>

#include <vector>

#include "../../include/qe.h"
#include "qe_common.cuh"
#include "qe_internal.h"
#include "qe_kernels.h"
#include "qe_outlier.h"

namespace qe {

__device__ unsigned g_err_word;

static unsigned *error_word() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    static unsigned *cache[64] = {};
    if (!cache[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_err_word) == cudaSuccess) cache[dev] = static_cast<unsigned *>(p);
    }
    return cache[dev];
}

unsigned *device_error_word() { return error_word(); }

static int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 148;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
        return 148;
    return n;
}

constexpr int kDefaultBlock = 256;
constexpr int kDefaultPowerIters = 64;
constexpr int kDefaultDenseSweeps = 1;
constexpr int kSweepChunk = 32;          // list-mode sweeps per persistent launch
constexpr int kFreeMaxChanges = 64;      // changes per row in the previous sweep below which a CTA runs free
constexpr int kMaxSplits = 16;           // split-K pieces of a trailing GEMM (partial buffers)
constexpr int kMinStepsPerSplit = 48;    // k-steps (k-blocks x plane products) per split-K piece

// Split-K pieces of a trailing GEMM with mt tile rows and kb k-blocks of nprod
// products: the count whose CTAs (one per SM) fill their waves best, less a
// small charge per piece for the partial sums it writes and the in-block
// prologue reads back; every piece keeps at least kMinStepsPerSplit k-steps.
// (A wide layer with 116 tile rows on 152 SMs runs 5 pieces in 4 full waves
// instead of one wave three quarters full.)
static int choose_splits(int64_t mt, int kb, int nprod, int nsm) {
    int cap = (kb * nprod) / kMinStepsPerSplit;
    if (cap > kb) cap = kb;
    if (cap > kMaxSplits) cap = kMaxSplits;
    if (cap < 1) cap = 1;
    int best = 1;
    double bv = -1.0;
    for (int S = 1; S <= cap; ++S) {
        const int64_t ctas = S * mt;
        const int64_t waves = ceil_div(ctas, nsm);
        const double v = static_cast<double>(ctas) / static_cast<double>(waves * nsm) - 0.01 * S;
        if (v > bv + 1e-12) {
            bv = v;
            best = S;
        }
    }
    return best;
}

// ---- workspace layout -----------------------------------------------------------
struct Plan {
    int64_t q = 0, p = 0, ld = 0;
    int B = kDefaultBlock, smax = 1;
    int64_t gsize = 0, ngroups = 1;   // grid columns per group (p: per row), groups per row
    bool grouped = false;
    size_t snt = 0, snh = 0, cscale = 0, wh = 0, rscale = 0, d = 0, dinv = 0, tri = 0, P = 0, R = 0, wpl = 0, qf = 0, dp = 0, part = 0, objp = 0,
           rowdf = 0, objbase = 0, sbar = 0, lcnt = 0, lent = 0, rowdft = 0, sw = 0, tq = 0, tqrows = 0, tqcnt = 0;
    int64_t nblk = 0;
    size_t PW = 0, H = 0, T = 0, st = 0, cg = 0, ce = 0, sb = 0, eb = 0, y0 = 0, y1 = 0, lam = 0,
           eta = 0, rowptr = 0, cpart = 0, cnorm = 0, ccols = 0, cval = 0, cn = 0, ppart = 0;
    size_t total = 0;
};

static size_t take(size_t &cur, size_t bytes) {
    const size_t o = cur;
    cur += static_cast<size_t>(round_up(static_cast<int64_t>(bytes > 0 ? bytes : 1), 256));
    return o;
}

static Plan make_plan(int64_t q, int64_t p, int B, bool outlier, int wpl_planes, int nsm, int64_t group = 0) {
    Plan pl;
    pl.q = q;
    pl.p = p;
    pl.grouped = group > 0 && group < p;
    pl.gsize = pl.grouped ? group : p;
    pl.ngroups = ceil_div(p, pl.gsize);
    pl.ld = round_up(p, 64);
    pl.B = B;
    pl.nblk = ceil_div(p, B);
    (void)nsm;
    pl.smax = kMaxSplits;
    const size_t qld = static_cast<size_t>(q) * pl.ld;
    size_t cur = 0;
    pl.snt = take(cur, static_cast<size_t>(3 * p) * pl.ld * 2);
    pl.snh = take(cur, static_cast<size_t>(2 * p) * pl.ld * 2);   // fp16 hi / lo, rows scaled by powers of two
    pl.cscale = take(cur, p * 4);
    pl.wh = take(cur, qld * 2);     // bf16 W as one row-scaled fp16 plane (the P GEMM)
    pl.rscale = take(cur, q * 4);
    pl.d = take(cur, p * 4);
    pl.dinv = take(cur, p * 4);
    pl.tri = take(cur, static_cast<size_t>(packed_diag_floats(p, B)) * 4);
    pl.P = take(cur, qld * 4);
    pl.R = take(cur, qld * 4);
    pl.wpl = take(cur, wpl_planes > 0 ? qld * 2 * wpl_planes : 0);
    pl.qf = take(cur, qld * 2 * (pl.grouped ? 3 : 1));   // grouped: s_g (C - z_g) in three planes
    pl.dp = take(cur, qld * 2 * 3);
    pl.part = take(cur, static_cast<size_t>(pl.smax) * q * B * 4);
    pl.objp = take(cur, static_cast<size_t>(rfull_partials(q, p) > objective_blocks(q) ? rfull_partials(q, p)
                                                                                    : objective_blocks(q)) * 8);
    pl.rowdf = take(cur, static_cast<size_t>(q) * 8);
    pl.objbase = take(cur, 8);
    {   // change lists and fp32 Sigma_bar rows of the change-list sweeps
        pl.sbar = take(cur, static_cast<size_t>(p) * pl.ld * 4);
        pl.lcnt = take(cur, static_cast<size_t>(q) * pl.nblk * 4);
        pl.lent = take(cur, static_cast<size_t>(q) * pl.nblk * B * 4);
        pl.rowdft = take(cur, static_cast<size_t>(q) * kSweepChunk * 8);
        pl.sw = take(cur, 16);   // adaptive schedule: switch flag (int) and change counter (u64)
    }
    // the change-driven kernel's near-tie queue: an entry and two rows of B floats per row
    pl.tq = take(cur, static_cast<size_t>(q) * sizeof(TieEntry));
    pl.tqrows = take(cur, static_cast<size_t>(q) * 2 * B * 4);
    pl.tqcnt = take(cur, 16);
    if (outlier) {
        const int64_t N = q * p;
        const int64_t nch = topk_chunks(N);
        pl.PW = take(cur, qld * 4);
        pl.H = take(cur, qld * 4);
        pl.T = take(cur, static_cast<size_t>(N) * 4);
        pl.st = take(cur, sizeof(TopkState));
        pl.cg = take(cur, nch * 4);
        pl.ce = take(cur, nch * 4);
        pl.sb = take(cur, nch * 4);
        pl.eb = take(cur, nch * 4);
        pl.y0 = take(cur, p * 4);
        pl.y1 = take(cur, p * 4);
        pl.lam = take(cur, 8);
        pl.ppart = take(cur, 2 * kPowerMaxBlocks * 8);
        pl.eta = take(cur, 8);
        pl.rowptr = take(cur, (q + 1) * 8);
        // structured outliers: column norms and the kept columns
        pl.cpart = take(cur, static_cast<size_t>(colnorm_chunks(q)) * p * 8);
        pl.cnorm = take(cur, p * 4);
        pl.ccols = take(cur, p * 8);
        pl.cval = take(cur, p * 4);
        pl.cn = take(cur, 8);
    }
    pl.total = cur;
    return pl;
}

}  // namespace qe

// ---- kernel timer (C ABI type) ----------------------------------------------------------
struct qe_timer {
    unsigned mask = 0;
    int used = 0;
    std::vector<cudaEvent_t> start, stop;
    std::vector<int> kind;
};

namespace qe {

// Records an event pair around one launch of class `k` when the timer asks for it.
class Timed {
  public:
    Timed(qe_timer *t, int k, cudaStream_t s) : t_(nullptr), s_(s) {
        if (t && (t->mask & (1u << k)) && t->used < static_cast<int>(t->start.size())) {
            t_ = t;
            idx_ = t->used++;
            t->kind[idx_] = k;
            cudaEventRecord(t->start[idx_], s);
        }
    }
    ~Timed() {
        if (t_) cudaEventRecord(t_->stop[idx_], s_);
    }

  private:
    qe_timer *t_;
    cudaStream_t s_;
    int idx_ = 0;
};

// ---- per-call context ----------------------------------------------------------------
struct Ctx {
    cudaStream_t s = nullptr;
    qe_timer *timer = nullptr;
    unsigned *err = nullptr;
    int nsm = 148;
    Plan pl;
    uint8_t *ws = nullptr;
    bool own = false;
    __nv_bfloat16 *snt = nullptr, *wpl = nullptr, *qf = nullptr, *dp = nullptr;
    __half *snh = nullptr, *wh = nullptr;
    float *cscale = nullptr, *rscale = nullptr;
    float *d = nullptr, *dinv = nullptr, *tri = nullptr, *P = nullptr, *R = nullptr, *part = nullptr;
    double *objp = nullptr, *rowdf = nullptr, *objbase = nullptr;
    float *sbar = nullptr;
    int *lcnt = nullptr;
    uint32_t *lent = nullptr;
    double *rowdft = nullptr;
    int *swflag = nullptr;
    unsigned long long *swcount = nullptr;
    TieEntry *tq = nullptr;
    float *tqrows = nullptr;
    unsigned *tqcnt = nullptr;
    float *PW = nullptr, *H = nullptr, *T = nullptr, *y0 = nullptr, *y1 = nullptr;
    TopkState *st = nullptr;
    unsigned *cg = nullptr, *ce = nullptr, *sb = nullptr, *eb = nullptr;
    double *lam = nullptr, *eta = nullptr, *ppart = nullptr;
    int64_t *rowptr = nullptr;
    double *cpart = nullptr;
    float *cnorm = nullptr, *cval = nullptr;
    int64_t *ccols = nullptr, *cn = nullptr;
    CUtensorMap tm_snt256, tm_snt64, tm_snt128, tm_qf, tm_dp, tm_wa;
    // the fp16 forms: Sigma_bar^T in two planes, C - z and the integer changes Delta'
    CUtensorMap tm_snh256, tm_snh64, tm_snh128, tm_qf16, tm_dp16;
    int wa_planes = 1;
    // near-tie refinement: the layer's inputs as given (and H for the outlier variant)
    float tie_eps = 0.0f;
    const float *Sig = nullptr;
    const void *Wl = nullptr;
    int wbf16 = 0;
    int64_t ldw = 0;
    const float *Hr = nullptr;

    ~Ctx() {
        if (own && ws) cudaFreeAsync(ws, s);
    }
};

template <typename T>
static T *at(uint8_t *ws, size_t off) {
    return reinterpret_cast<T *>(ws + off);
}

static qe_status setup_ctx(Ctx &c, const Plan &pl, const qe_opts *o, cudaStream_t s) {
    c.s = s;
    c.timer = o ? o->timer : nullptr;
    c.pl = pl;
    c.err = error_word();
    if (!c.err) return QE_ERR_CUDA;
    if (o && o->workspace) {
        if (o->workspace_bytes < pl.total || (reinterpret_cast<uintptr_t>(o->workspace) & 255u))
            return QE_ERR_OOM;
        c.ws = static_cast<uint8_t *>(o->workspace);
    } else {
        void *p = nullptr;
        if (cudaMallocAsync(&p, pl.total, s) != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_OOM;
        }
        c.ws = static_cast<uint8_t *>(p);
        c.own = true;
    }
    uint8_t *w = c.ws;
    c.snt = at<__nv_bfloat16>(w, pl.snt);
    c.snh = at<__half>(w, pl.snh);
    c.cscale = at<float>(w, pl.cscale);
    c.wh = at<__half>(w, pl.wh);
    c.rscale = at<float>(w, pl.rscale);
    c.d = at<float>(w, pl.d);
    c.dinv = at<float>(w, pl.dinv);
    c.tri = at<float>(w, pl.tri);
    c.P = at<float>(w, pl.P);
    c.R = at<float>(w, pl.R);
    c.wpl = at<__nv_bfloat16>(w, pl.wpl);
    c.qf = at<__nv_bfloat16>(w, pl.qf);
    c.dp = at<__nv_bfloat16>(w, pl.dp);
    c.part = at<float>(w, pl.part);
    c.objp = at<double>(w, pl.objp);
    c.rowdf = at<double>(w, pl.rowdf);
    c.objbase = at<double>(w, pl.objbase);
    if (pl.sbar) {
        c.sbar = at<float>(w, pl.sbar);
        c.lcnt = at<int>(w, pl.lcnt);
        c.lent = at<uint32_t>(w, pl.lent);
        c.rowdft = at<double>(w, pl.rowdft);
        c.swflag = at<int>(w, pl.sw);
        c.swcount = at<unsigned long long>(w, pl.sw + 8);
    }
    c.tq = at<TieEntry>(w, pl.tq);
    c.tqrows = at<float>(w, pl.tqrows);
    c.tqcnt = at<unsigned>(w, pl.tqcnt);
    // the queue's counters start at zero (every check launch leaves them so; this
    // clears what an aborted call left)
    if (cudaMemsetAsync(c.tqcnt, 0, 16, s) != cudaSuccess) {
        cudaGetLastError();
        return QE_ERR_CUDA;
    }
    if (pl.PW) {
        c.PW = at<float>(w, pl.PW);
        c.H = at<float>(w, pl.H);
        c.T = at<float>(w, pl.T);
        c.st = at<TopkState>(w, pl.st);
        c.cg = at<unsigned>(w, pl.cg);
        c.ce = at<unsigned>(w, pl.ce);
        c.sb = at<unsigned>(w, pl.sb);
        c.eb = at<unsigned>(w, pl.eb);
        c.y0 = at<float>(w, pl.y0);
        c.y1 = at<float>(w, pl.y1);
        c.lam = at<double>(w, pl.lam);
        c.ppart = at<double>(w, pl.ppart);
        c.eta = at<double>(w, pl.eta);
        c.rowptr = at<int64_t>(w, pl.rowptr);
        c.cpart = at<double>(w, pl.cpart);
        c.cnorm = at<float>(w, pl.cnorm);
        c.ccols = at<int64_t>(w, pl.ccols);
        c.cval = at<float>(w, pl.cval);
        c.cn = at<int64_t>(w, pl.cn);
    }
    const uint64_t q = pl.q, p = pl.p, ld = pl.ld;
    if (!make_tmap_bf16(&c.tm_snt256, c.snt, 3 * p, p, ld, 256) ||
        !make_tmap_bf16(&c.tm_snt64, c.snt, 3 * p, p, ld, 64) ||
        !make_tmap_bf16(&c.tm_snt128, c.snt, 3 * p, p, ld, 128) ||
        !make_tmap_bf16(&c.tm_qf, c.qf, pl.grouped ? 3 * q : q, p, ld, 128) ||
        !make_tmap_bf16(&c.tm_dp, c.dp, 3 * q, p, ld, 128) ||
        !make_tmap_f16(&c.tm_snh256, c.snh, 2 * p, p, ld, 256) || !make_tmap_f16(&c.tm_snh64, c.snh, 2 * p, p, ld, 64) ||
        !make_tmap_f16(&c.tm_snh128, c.snh, 2 * p, p, ld, 128) || !make_tmap_f16(&c.tm_qf16, c.qf, q, p, ld, 128) ||
        !make_tmap_f16(&c.tm_dp16, c.dp, 2 * q, p, ld, 128))
        return QE_ERR_CUDA;
    return QE_OK;
}

#define QE_CK(x)                                     \
    do {                                             \
        if ((x) != cudaSuccess) {                    \
            cudaGetLastError();                      \
            return QE_ERR_CUDA;                      \
        }                                            \
    } while (0)

static GemmArgs gemm_args(const Ctx &c, int M, int N, int kb_count, int mode) {
    GemmArgs g;
    memset(&g, 0, sizeof(g));
    g.M = M;
    g.N = N;
    g.kb_begin = 0;
    g.kb_count = kb_count;
    g.mode = mode;
    g.err = c.err;
    return g;
}

// Plane products of A (1 exact plane, or hi/mid/lo) times B = Sigma_bar^T (hi/mid/lo):
// every pair whose order is at least 2^-16 relative (plane k carries ~2^-8k).
static void set_prods(GemmArgs &g, int a_planes) {
    static const int one[3][2] = {{0, 0}, {0, 1}, {0, 2}};
    static const int three[6][2] = {{0, 0}, {0, 1}, {1, 0}, {0, 2}, {1, 1}, {2, 0}};
    g.n_prod = (a_planes == 3) ? 6 : 3;
    for (int t = 0; t < g.n_prod; ++t) {
        g.prod_a[t] = (a_planes == 3) ? three[t][0] : one[t][0];
        g.prod_b[t] = (a_planes == 3) ? three[t][1] : one[t][1];
    }
}

// An exact fp16 A (C - z, or integer changes) times the two fp16 planes of Sigma_bar^T.
static void set_prods_h2(GemmArgs &g, const Ctx &c, int64_t col0) {
    g.n_prod = 2;
    g.prod_a[0] = 0;
    g.prod_b[0] = 0;
    g.prod_a[1] = 0;
    g.prod_b[1] = 1;
    g.f16 = 1;
    g.colscale = c.cscale + col0;
    g.ascale = 1.0f;
}

// A real A (the first sweep's changes, times 2^sh) in two fp16 planes times the two
// fp16 planes of Sigma_bar^T: hi.hi, hi.lo, lo.hi (lo.lo is below 2^-22 relative).
static void set_prods_h2r(GemmArgs &g, const Ctx &c, int64_t col0, int sh) {
    static const int pa[3] = {0, 0, 1}, pb[3] = {0, 1, 0};
    g.n_prod = 3;
    for (int k = 0; k < 3; ++k) {
        g.prod_a[k] = pa[k];
        g.prod_b[k] = pb[k];
    }
    g.f16 = 1;
    g.colscale = c.cscale + col0;
    g.ascale = ldexpf(1.0f, -sh);
}

// Sigma -> d, Sigma_bar^T planes; W operand planes; P = W (I + Sigma_bar) into `Pout`.
static qe_status prepare(Ctx &c, const void *W, int wbf16, int64_t ldw, const float *Sigma, float *Pout) {
    const int64_t q = c.pl.q, p = c.pl.p, ld = c.pl.ld;
    QE_CK(launch_sigma_norm(Sigma, p, p, c.d, c.snt, ld, c.err, c.s));
    QE_CK(launch_dinv(c.d, p, c.dinv, c.s));
    QE_CK(launch_pack_diag(c.snt, ld, p, c.pl.B, c.tri, c.s));
    QE_CK(launch_sigma_planes_h2(Sigma, p, p, c.d, c.snh, ld, c.cscale, c.s));
    if (c.sbar) QE_CK(launch_sigma_bar_rows(Sigma, p, p, c.d, c.sbar, ld, c.s));
    // bf16 W: one row-scaled fp16 plane against the two fp16 planes of Sigma_bar
    // (2 products); fp32 W: three bf16 planes against three (6 products)
    const bool h1 = wbf16 != 0;
    if (h1) {
        QE_CK(launch_w_plane_h1(W, ldw, q, p, c.wh, ld, c.rscale, c.s));
        if (!make_tmap_f16(&c.tm_wa, c.wh, q, p, ld, 128)) return QE_ERR_CUDA;
        c.wa_planes = 1;
    } else {
        c.wa_planes = wbf16 ? 1 : 3;
        QE_CK(launch_make_planes(W, wbf16, ldw, q, p, c.wa_planes == 3, c.wpl, ld, c.s));
        if (!make_tmap_bf16(&c.tm_wa, c.wpl, c.wa_planes * q, p, ld, 128)) return QE_ERR_CUDA;
    }
    GemmArgs g = gemm_args(c, static_cast<int>(q), static_cast<int>(p), static_cast<int>(ceil_div(p, 64)),
                           EPI_PINIT);
    if (h1) {
        set_prods_h2(g, c, 0);
        g.rowscale = c.rscale;
    } else {
        set_prods(g, c.wa_planes);
    }
    g.m_fast = 1;
    g.a_plane_rows = static_cast<int>(q);
    g.b_plane_rows = static_cast<int>(p);
    g.out = Pout;
    g.ldo = ld;
    g.W = W;
    g.w_is_bf16 = wbf16;
    g.ldw = ldw;
    {
        Timed tm(c.timer, QE_KERNEL_PINIT_GEMM, c.s);
        QE_CK(launch_tc_gemm(256, c.tm_wa, h1 ? c.tm_snh256 : c.tm_snt256, g, 1, c.s));
    }
    return QE_OK;
}

// R = P - s (C - z) Sigma_bar from the current codes (C - z held in qf).  With
// `obj`, the epilogue also reduces f = sum D_ij d_j (R_ij - What_ij) for the
// codes in `codes` (D = W - What - H) and k_sum_partials writes it to *obj.
struct ObjFuse {
    double *obj;
    const void *W;
    int wbf16;
    int64_t ldw;
    const uint8_t *codes;
    const float *H;
};

static qe_status residual(Ctx &c, const float *scales, const float *zeros, const ObjFuse *f = nullptr) {
    const int64_t q = c.pl.q, p = c.pl.p, ld = c.pl.ld;
    GemmArgs g = gemm_args(c, static_cast<int>(q), static_cast<int>(p), static_cast<int>(ceil_div(p, 64)),
                           EPI_RFULL);
    if (c.pl.grouped) set_prods(g, 3);
    else set_prods_h2(g, c, 0);   // C - z is an exact small integer
    g.gsize = c.pl.gsize;
    g.ngroups = c.pl.ngroups;
    g.absolute = c.pl.grouped ? 1 : 0;
    g.m_fast = 1;
    g.a_plane_rows = static_cast<int>(q);
    g.b_plane_rows = static_cast<int>(p);
    g.out = c.R;
    g.ldo = ld;
    g.P = c.P;
    g.ldp = ld;
    g.scale = scales;
    g.zero = zeros;   // R is kept in grid-step units: the epilogue adds z
    if (f) {
        g.obj_part = c.objp;
        g.W = f->W;
        g.w_is_bf16 = f->wbf16;
        g.ldw = f->ldw;
        g.codes = f->codes;
        g.ldc = p;
        g.dvec = c.d;
        g.Hd = f->H;
        g.ldh = ld;
    }
    {
        Timed tm(c.timer, QE_KERNEL_RESIDUAL_GEMM, c.s);
        if (c.pl.grouped) QE_CK(launch_tc_gemm(256, c.tm_qf, c.tm_snt256, g, 1, c.s));
        else QE_CK(launch_tc_gemm(256, c.tm_qf16, c.tm_snh256, g, 1, c.s));
    }
    if (f) QE_CK(launch_sum_partials(c.objp, static_cast<int>(rfull_partials(q, p)), f->obj, c.s));
    return QE_OK;
}

// One cyclic sweep j = 1..p, blocked by B columns.
//   classic (window == 0): block b gets the deferred correction
//       Delta'[:, 0:b0] Sigma_bar[0:b0, block] on top of R (the sweep-start
//       residual), which a residual GEMM refreshes after the sweep.
//   rolling window (window > 0): R holds each block's value from its last
//       visit; the correction covers the `window` most recent column changes
//       (this sweep's for columns < b0, the previous sweep's for columns >= b0,
//       all of them in dp), the staged values become the new base, and the
//       objective changes of the decisions accumulate in rowdf.  window = -1
//       means the first window sweep after a residual refresh: only columns < b0.
//       Every window visit also records its changes in the block's change list,
//       from which the later sweeps (k_cd_rows_lists) take the correction.
// src: where What at the sweep start comes from: W itself (the first sweep, R
// then holds it), the codes, or the real values a relaxed sweep left (kept in
// the change-list entry buffer, unused while such sweeps run).  relax: the
// relax heuristic of Sec. 3.2 (the sweep keeps beta~ unquantized).  When the
// changes are real-valued (src != SRC_CODES or relax) they take three bf16
// planes and the in-block sequential kernel.
// Near-tie refinement fields of a CD launch.
static void set_tie(const Ctx &c, CdArgs &a, bool on) {
    a.tie_eps = on ? c.tie_eps : 0.0f;
    a.S = c.Sig;
    a.lds_full = c.pl.p;
    a.W = c.Wl;
    a.w_bf16 = c.wbf16;
    a.ldw = c.ldw;
    a.Hd = c.Hr;
    a.ldh = c.pl.ld;
}

enum { SRC_W = 0, SRC_CODES = 1, SRC_V = 2 };

static float *relaxed_values(const Ctx &c) { return reinterpret_cast<float *>(c.lent); }

static qe_status sweep(Ctx &c, uint8_t *codes, const float *scales, const float *zeros, int bits,
                       int src, bool relax, int window, const int *gate = nullptr, bool wait_test = false) {
    const int64_t q = c.pl.q, p = c.pl.p, ld = c.pl.ld;
    const int B = c.pl.B;
    const bool frac = src != SRC_CODES || relax;
    // window sweeps over integer changes run their trailing GEMMs in fp16; so does the
    // first sweep from W, whose changes |a - c| <= 2^bits - 1 (a = W / s + z and the
    // code both lie in [0, 2^bits - 1]) are scaled by 2^(14 - bits) into two fp16 planes
    const bool h2 = window != 0 && !frac && !c.pl.grouped;
    const bool h2r = frac && src == SRC_W && !relax && !c.pl.grouped;
    const int sh = 14 - bits;
    for (int64_t b0 = 0; b0 < p; b0 += B) {
        const int bw = static_cast<int>((p - b0) < B ? (p - b0) : B);
        const int64_t kcols = (window > 0) ? p : b0;
        int nsplit = 0;
        if (kcols > 0) {
            const int kb = static_cast<int>(ceil_div(kcols, 64));
            GemmArgs g = gemm_args(c, static_cast<int>(q), bw, kb, EPI_TRAIL);
            if (h2) set_prods_h2(g, c, b0);   // integer changes: fp16 A, two fp16 planes of Sigma_bar^T
            else if (h2r) set_prods_h2r(g, c, b0, sh);
            else set_prods(g, (frac || c.pl.grouped) ? 3 : 1);
            int S = choose_splits(ceil_div(q, 128), kb, g.n_prod, c.nsm);
            if (S > c.pl.smax) S = c.pl.smax;
            g.a_plane_rows = static_cast<int>(q);
            g.b_plane_rows = static_cast<int>(p);
            g.b_row0 = static_cast<int>(b0);
            g.out = c.part;
            g.ldo = B;
            g.split_stride = q * B;
            g.gate = gate;
            Timed tm(c.timer, QE_KERNEL_TRAIL_GEMM, c.s);
            if (h2 || h2r)
                QE_CK(launch_tc_gemm(B, c.tm_dp16, B == 64 ? c.tm_snh64 : (B == 128 ? c.tm_snh128 : c.tm_snh256), g,
                                     S, c.s));
            else
                QE_CK(launch_tc_gemm(B, c.tm_dp, B == 64 ? c.tm_snt64 : (B == 128 ? c.tm_snt128 : c.tm_snt256), g,
                                     S, c.s));
            nsplit = S;
        }
        CdArgs a;
        memset(&a, 0, sizeof(a));
        a.q = q;
        a.p = p;
        a.b0 = b0;
        a.bw = bw;
        a.R = c.R;
        a.ldr = ld;
        a.store_base = window != 0 ? 1 : 0;
        a.part = c.part;
        a.nsplit = nsplit;
        a.part_stride = q * B;
        a.ldpart = B;
        a.tri = c.tri;
        a.scale = scales;
        a.zero = zeros;
        a.gsize = c.pl.gsize;
        a.ngroups = c.pl.ngroups;
        a.grouped = c.pl.grouped ? 1 : 0;
        a.d = c.d;
        a.rowdf = window != 0 ? c.rowdf : nullptr;
        a.maxq = static_cast<float>((1 << bits) - 1);
        a.first_sweep = src == SRC_W ? 1 : 0;
        a.frac = frac ? 1 : 0;
        a.vstart = src == SRC_V ? relaxed_values(c) : nullptr;
        a.vout = relax ? relaxed_values(c) : nullptr;
        a.ldv = ld;
        a.write_qf = window != 0 ? 0 : 1;
        a.codes = codes;
        a.ldc = p;
        a.qf = c.qf;
        a.ldq = ld;
        a.dp = c.dp;
        a.nblk = static_cast<int>(c.pl.nblk);
        a.lcnt = c.lcnt;
        if (window != 0 && !frac) a.lent = c.lent;
        a.ldd = ld;
        a.dp_plane_rows = q;
        a.dp_f16 = h2 ? 1 : (h2r ? 2 : 0);
        a.dp_scale = ldexpf(1.0f, sh);
        a.err = c.err;
        a.gate = gate;
        a.tq = c.tq;
        a.tq_rows = c.tqrows;
        a.tq_cnt = c.tqcnt;
        // relaxed sweeps and the sweep after one start from real values: no refinement
        set_tie(c, a, !relax && src != SRC_V);
        if (wait_test) {   // the failure-path test hook: the first block waits for a copy never issued
            a.skip_copy = 1;
            a.wait_ns = 5000000ull;
            QE_CK(launch_cd_block(B, a, c.nsm, c.s));
            return QE_OK;
        }
        Timed tm(c.timer, QE_KERNEL_CD_BLOCK, c.s);
        QE_CK(launch_cd_block(B, a, c.nsm, c.s));
        // the change-driven kernel with the refinement leaves its noted rows to the check
        if (!frac && a.tie_eps > 0.0f) QE_CK(launch_cd_tie_check(B, a, c.nsm, c.s));
    }
    return QE_OK;
}

// Arguments of the persistent change-list kernel (block fields unused).
static CdArgs list_args(const Ctx &c, uint8_t *codes, const float *scales, const float *zeros, int bits) {
    CdArgs a;
    memset(&a, 0, sizeof(a));
    a.q = c.pl.q;
    a.p = c.pl.p;
    a.R = c.R;
    a.ldr = c.pl.ld;
    a.tri = c.tri;
    a.scale = scales;
    a.zero = zeros;
    a.gsize = c.pl.gsize;
    a.ngroups = c.pl.ngroups;
    a.grouped = c.pl.grouped ? 1 : 0;
    a.d = c.d;
    a.maxq = static_cast<float>((1 << bits) - 1);
    a.codes = codes;
    a.ldc = c.pl.p;
    a.qf = c.qf;
    a.ldq = c.pl.ld;
    a.sbar = c.sbar;
    a.lds = c.pl.ld;
    a.nblk = static_cast<int>(c.pl.nblk);
    a.lcnt = c.lcnt;
    a.lent = c.lent;
    a.err = c.err;
    set_tie(c, a, true);
    return a;
}

static qe_status objective(Ctx &c, const void *W, int wbf16, int64_t ldw, const float *H,
                           const uint8_t *codes, const float *scales, const float *zeros,
                           const float *Rsrc, double *out) {
    ObjArgs a;
    memset(&a, 0, sizeof(a));
    a.q = c.pl.q;
    a.p = c.pl.p;
    a.W = W;
    a.w_bf16 = wbf16;
    a.ldw = ldw;
    a.H = H;
    a.ldh = c.pl.ld;
    a.codes = codes;
    a.ldc = c.pl.p;
    a.scale = scales;
    a.zero = zeros;
    a.d = c.d;
    a.R = Rsrc;
    a.ldr = c.pl.ld;
    QE_CK(launch_objective(a, c.objp, out, c.s));
    return QE_OK;
}

static int block_width(const qe_opts *o) {
    return (o && o->block_width) ? o->block_width : kDefaultBlock;
}

static int dense_sweeps(const qe_opts *o) {
    return (o && o->dense_sweeps) ? o->dense_sweeps : kDefaultDenseSweeps;
}

static int relax_period(const qe_opts *o) { return o ? o->relax_period : 0; }

constexpr float kDefaultTieEps = 1e-5f;
static float tie_eps(const qe_opts *o) {
    if (!o || o->tie_eps == 0.0f) return kDefaultTieEps;
    return o->tie_eps > 0.0f ? o->tie_eps : 0.0f;
}

// Whether the fp32 Sigma_bar rows that the list sweeps gather (4 p ld bytes) fit
// in three quarters of this GPU's L2.
static bool sbar_rows_fit_l2(int64_t p, int64_t ld) {
    int dev = 0, l2 = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, dev) != cudaSuccess ||
        l2 <= 0) {
        cudaGetLastError();
        l2 = 128 << 20;
    }
    return 4.0 * static_cast<double>(p) * static_cast<double>(ld) <= 0.75 * static_cast<double>(l2);
}

// The adaptive schedule's switch threshold for layers whose Sigma_bar rows exceed
// L2: a dense sweep costs its window GEMMs, 2 q p^2 flops of two fp16 products each
// (~1.2 PFLOP/s on 152 SMs as measured on the 15360 x 14848 layer), plus an
// in-block pass with its near-tie checks (~35 ps per coordinate); a list sweep
// gathers one Sigma_bar row of 4 p bytes per change (~4.75 TB/s measured on the
// same layer); the next sweep makes about 0.8 times the changes of the one just
// finished.
static int64_t switch_below_model(int64_t q, int64_t p, int nsm) {
    const double qd = static_cast<double>(q), pd = static_cast<double>(p);
    const double t_dense = 4.0 * qd * pd * pd / (1.2e15 * nsm / 152.0) + 3.5e-11 * qd * pd;
    const double t_change = 4.0 * pd / 4.75e12;
    const double below = t_dense / t_change / 0.8;
    return below > 9.0e18 ? static_cast<int64_t>(9.0e18) : static_cast<int64_t>(below);
}

static int free_changes(const qe_opts *o) {
    return (o && o->free_changes) ? o->free_changes : kFreeMaxChanges;
}

// structured: the call accepts structured_outliers = 1 (the outlier variant,
// which has no relax heuristic)
static qe_status check_opts(const qe_opts *o, bool structured = false) {
    if (!o) return QE_OK;
    if (o->relax_period < 0) return QE_ERR_INVALID_ARG;
    if (o->relax_period != 0 && structured) return QE_ERR_UNSUPPORTED;
    if (o->structured_outliers != 0 && !(structured && o->structured_outliers == 1)) return QE_ERR_UNSUPPORTED;
    if (o->block_width != 0 && o->block_width != 64 && o->block_width != 128 && o->block_width != 256)
        return QE_ERR_UNSUPPORTED;
    if (o->power_iters < 0 || o->dense_sweeps < 0 || o->free_changes < -1 || o->group_size < 0 ||
        o->switch_below < 0)
        return QE_ERR_INVALID_ARG;
    if (o->workspace && o->workspace_bytes == 0) return QE_ERR_INVALID_ARG;
    if (o->wait_test < 0 || o->wait_test > 1) return QE_ERR_INVALID_ARG;
    if (!(o->tie_eps == o->tie_eps) || o->tie_eps > 0.25f) return QE_ERR_INVALID_ARG;   // NaN or too wide
    if (o->group_size > 0) {
        // groups hold whole column blocks; no relax heuristic, no outlier variant with groups
        if (o->group_size % block_width(o) != 0) return QE_ERR_INVALID_ARG;
        if (structured || o->relax_period != 0) return QE_ERR_UNSUPPORTED;
    }
    return QE_OK;
}

static int64_t group_size(const qe_opts *o) { return o ? o->group_size : 0; }

static qe_status check_layer(const void *W, qe_dtype wt, int64_t q, int64_t p, int64_t ldw,
                             const float *Sigma, int bits, int iters, const uint8_t *codes,
                             const float *scales, const float *zeros, const double *obj) {
    if (!W || !Sigma || !codes || !scales || !zeros || !obj) return QE_ERR_INVALID_ARG;
    if (wt != QE_F32 && wt != QE_BF16) return QE_ERR_INVALID_ARG;
    if (q < 1 || p < 1 || q > (1ll << 30) || p > (1ll << 30) || ldw < p) return QE_ERR_INVALID_ARG;
    if (bits < 2 || bits > 8 || iters < 1) return QE_ERR_INVALID_ARG;
    return QE_OK;
}

}  // namespace qe

using namespace qe;

extern "C" {

int qe_version(void) { return 10000; }

const char *qe_status_string(qe_status st) {
    switch (st) {
        case QE_OK: return "ok";
        case QE_ERR_INVALID_ARG: return "invalid argument";
        case QE_ERR_CUDA: return "CUDA error";
        case QE_ERR_OOM: return "workspace allocation failed or too small";
        case QE_ERR_NUMERIC: return "non-finite value in W or Sigma";
        case QE_ERR_TIMEOUT: return "a device-side wait gave up";
        case QE_ERR_UNSUPPORTED: return "option or layout not implemented";
        default: return "unknown status";
    }
}

qe_status qe_timer_create(unsigned kernel_mask, int capacity, qe_timer **timer) {
    if (!timer || capacity < 1 || capacity > (1 << 20)) return QE_ERR_INVALID_ARG;
    qe_timer *t = new qe_timer();
    t->mask = kernel_mask;
    t->start.assign(capacity, nullptr);
    t->stop.assign(capacity, nullptr);
    t->kind.assign(capacity, -1);
    for (int k = 0; k < capacity; ++k) {
        if (cudaEventCreate(&t->start[k]) != cudaSuccess || cudaEventCreate(&t->stop[k]) != cudaSuccess) {
            cudaGetLastError();
            qe_timer_destroy(t);
            return QE_ERR_CUDA;
        }
    }
    *timer = t;
    return QE_OK;
}

qe_status qe_timer_read(qe_timer *timer, int kernel, int *launches, double *total_ms) {
    if (!timer || !launches || !total_ms || kernel < 0 || kernel >= QE_KERNEL_COUNT) return QE_ERR_INVALID_ARG;
    int n = 0;
    double ms = 0.0;
    for (int k = 0; k < timer->used; ++k) {
        if (timer->kind[k] != kernel) continue;
        float e = 0.0f;
        if (cudaEventSynchronize(timer->stop[k]) != cudaSuccess ||
            cudaEventElapsedTime(&e, timer->start[k], timer->stop[k]) != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
        ms += e;
        ++n;
    }
    *launches = n;
    *total_ms = ms;
    return QE_OK;
}

qe_status qe_timer_reset(qe_timer *timer) {
    if (!timer) return QE_ERR_INVALID_ARG;
    timer->used = 0;
    return QE_OK;
}

qe_status qe_timer_destroy(qe_timer *timer) {
    if (!timer) return QE_ERR_INVALID_ARG;
    for (size_t k = 0; k < timer->start.size(); ++k) {
        if (timer->start[k]) cudaEventDestroy(timer->start[k]);
        if (timer->stop[k]) cudaEventDestroy(timer->stop[k]);
    }
    delete timer;
    return QE_OK;
}

qe_status qe_sync_status(qe_stream_t stream) {
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) {
        cudaGetLastError();
        return QE_ERR_CUDA;
    }
    unsigned *e = error_word();
    if (!e) return QE_ERR_CUDA;
    unsigned v = 0;
    if (cudaMemcpyAsync(&v, e, sizeof(v), cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemsetAsync(e, 0, sizeof(unsigned), s) != cudaSuccess || cudaStreamSynchronize(s) != cudaSuccess) {
        cudaGetLastError();
        return QE_ERR_CUDA;
    }
    if (v & ERR_TIMEOUT) return QE_ERR_TIMEOUT;
    if (v & ERR_NUMERIC) return QE_ERR_NUMERIC;
    return QE_OK;
}

qe_status qe_workspace_size(int64_t q, int64_t p, int outlier, const qe_opts *opts, size_t *bytes) {
    if (!bytes || q < 1 || p < 1) return QE_ERR_INVALID_ARG;
    const qe_status st = check_opts(opts, outlier != 0);
    if (st != QE_OK) return st;
    const Plan pl = make_plan(q, p, block_width(opts), outlier != 0, 3, sm_count(), group_size(opts));
    *bytes = pl.total;
    return QE_OK;
}

qe_status qe_build_sigma(const void *X, qe_dtype x_dtype, qe_xlayout layout, int64_t p, int64_t n,
                         int64_t ldx, float *Sigma, int accumulate, qe_stream_t stream) {
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (!X || !Sigma || p < 1 || n < 0 || p > (1ll << 30)) return QE_ERR_INVALID_ARG;
    if (x_dtype != QE_F32 && x_dtype != QE_BF16) return QE_ERR_INVALID_ARG;
    if (layout != QE_FEATURE_MAJOR && layout != QE_TOKEN_MAJOR) return QE_ERR_INVALID_ARG;
    if (layout == QE_FEATURE_MAJOR ? ldx < n : ldx < p) return QE_ERR_INVALID_ARG;
    if (n == 0) {
        if (!accumulate) QE_CK(cudaMemsetAsync(Sigma, 0, static_cast<size_t>(p) * p * 4, s));
        return QE_OK;
    }
    unsigned *err = error_word();
    if (!err) return QE_ERR_CUDA;
    if (x_dtype == QE_F32) {
        const float *Xf = static_cast<const float *>(X);
        if (layout == QE_FEATURE_MAJOR) QE_CK(launch_sigma_f32(Xf, p, n, ldx, 1, Sigma, accumulate, s));
        else QE_CK(launch_sigma_f32(Xf, p, n, 1, ldx, Sigma, accumulate, s));
        return QE_OK;
    }
    GemmArgs g;
    memset(&g, 0, sizeof(g));
    g.M = static_cast<int>(p);
    g.N = static_cast<int>(p);
    g.n_prod = 1;
    g.mode = EPI_SIGMA;
    g.out = Sigma;
    g.ldo = p;
    g.err = err;
    const bool direct = layout == QE_FEATURE_MAJOR && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0) &&
                        (ldx % 8 == 0);
    if (direct) {
        CUtensorMap ta, tb;
        if (!make_tmap_bf16(&ta, X, p, n, ldx, 128) || !make_tmap_bf16(&tb, X, p, n, ldx, 256))
            return QE_ERR_CUDA;
        g.kb_count = static_cast<int>(ceil_div(n, 64));
        g.accumulate = accumulate;
        QE_CK(launch_tc_gemm(256, ta, tb, g, 1, s));
        return QE_OK;
    }
    // Token-major or unaligned bf16 X: stage feature-major chunks of tokens.
    const int64_t nc = n < 8192 ? round_up(n, 64) : 8192;
    void *buf = nullptr;
    if (cudaMallocAsync(&buf, static_cast<size_t>(p) * nc * 2, s) != cudaSuccess) {
        cudaGetLastError();
        return QE_ERR_OOM;
    }
    qe_status st = QE_OK;
    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, buf, p, nc, nc, 128) || !make_tmap_bf16(&tb, buf, p, nc, nc, 256)) st = QE_ERR_CUDA;
    for (int64_t n0 = 0; st == QE_OK && n0 < n; n0 += nc) {
        const int64_t len = (n - n0) < nc ? (n - n0) : nc;
        cudaError_t e;
        if (layout == QE_TOKEN_MAJOR) {
            e = launch_transpose_bf16(X, n0, len, p, ldx, buf, nc, s);
        } else {
            e = cudaMemcpy2DAsync(buf, nc * 2, static_cast<const __nv_bfloat16 *>(X) + n0, ldx * 2, len * 2,
                                  p, cudaMemcpyDeviceToDevice, s);
        }
        if (e == cudaSuccess && len < nc)  // zero the unused tail of the chunk
            e = cudaMemset2DAsync(static_cast<__nv_bfloat16 *>(buf) + len, nc * 2, 0, (nc - len) * 2, p, s);
        g.kb_count = static_cast<int>(ceil_div(len, 64));
        g.accumulate = (n0 > 0) ? 1 : accumulate;
        if (e == cudaSuccess) e = launch_tc_gemm(256, ta, tb, g, 1, s);
        if (e != cudaSuccess) {
            cudaGetLastError();
            st = QE_ERR_CUDA;
        }
    }
    cudaFreeAsync(buf, s);
    return st;
}

qe_status qe_quantize_layer(const void *W, qe_dtype w_dtype, int64_t q, int64_t p, int64_t ldw,
                            const float *Sigma, int bits, int iters, const qe_opts *opts,
                            uint8_t *codes, float *scales, float *zeros, double *obj, qe_stream_t stream) {
    qe_status st = check_layer(W, w_dtype, q, p, ldw, Sigma, bits, iters, codes, scales, zeros, obj);
    if (st != QE_OK) return st;
    if ((st = check_opts(opts)) != QE_OK) return st;
    const int wbf16 = (w_dtype == QE_BF16);
    Ctx c;
    c.nsm = sm_count();
    const Plan pl = make_plan(q, p, block_width(opts), false, wbf16 ? 1 : 3, c.nsm, group_size(opts));
    if ((st = setup_ctx(c, pl, opts, reinterpret_cast<cudaStream_t>(stream))) != QE_OK) return st;
    c.tie_eps = tie_eps(opts);
    c.Sig = Sigma;
    c.Wl = W;
    c.wbf16 = wbf16;
    c.ldw = ldw;

    QE_CK(launch_grid(W, wbf16, ldw, nullptr, 0, q, p, pl.gsize, bits, scales, zeros, c.err, c.s));
    if ((st = prepare(c, W, wbf16, ldw, Sigma, c.P)) != QE_OK) return st;
    if (opts && opts->wx_norm2)
        if ((st = objective(c, W, wbf16, ldw, nullptr, nullptr, nullptr, nullptr, c.P, opts->wx_norm2)) != QE_OK)
            return st;
    // Sweep 1 starts at What = W (Sec. 3.1) and changes every coordinate by a
    // real amount: the classic schedule with a residual refresh (which also
    // yields obj[0]).  Later sweeps change few codes, by integers: the rolling
    // window schedule with the objective updated decision by decision.  A
    // relaxed sweep (relax heuristic, Sec. 3.2) and the sweep after it move
    // every coordinate by a real amount again: they run as sequential in-block
    // sweeps between two residual refreshes.
    const bool warm = opts && opts->init_codes;
    const int rp = relax_period(opts);
    auto relaxed = [&](int t) { return rp > 0 && (t + 1) % rp == 0 && t + 1 < iters; };
    const size_t plane0 = static_cast<size_t>(q) * pl.ld * 2;
    // after a residual refresh R holds every change so far: empty window, no list entries
    auto restart = [&](int planes) -> qe_status {
        QE_CK(cudaMemsetAsync(c.dp, 0, plane0 * planes, c.s));
        QE_CK(cudaMemsetAsync(c.lcnt, 0, static_cast<size_t>(q) * pl.nblk * 4, c.s));
        QE_CK(cudaMemsetAsync(c.rowdf, 0, static_cast<size_t>(q) * 8, c.s));
        return QE_OK;
    };
    auto refresh = [&]() -> qe_status {
        QE_CK(launch_codes_to_qf(codes, p, scales, zeros, q, p, pl.gsize, pl.grouped, c.qf, pl.ld, c.s));
        return residual(c, scales, zeros);
    };
    auto record = [&](int t) -> qe_status {
        if (opts && opts->sweep_codes)
            QE_CK(cudaMemcpyAsync(opts->sweep_codes + static_cast<size_t>(t) * q * p, codes,
                                  static_cast<size_t>(q) * p, cudaMemcpyDeviceToDevice, c.s));
        return QE_OK;
    };
    // sweep_forms[t0 .. t0 + n) = form (0 sequential, 1 dense, 2 lists)
    auto form = [&](int t0, int n, int f) -> qe_status {
        if (opts && opts->sweep_forms && n > 0) QE_CK(cudaMemsetAsync(opts->sweep_forms + t0, f, n, c.s));
        return QE_OK;
    };
    int t = 0, src = SRC_CODES;
    if (warm) {
        QE_CK(cudaMemcpyAsync(codes, opts->init_codes, static_cast<size_t>(q) * p, cudaMemcpyDeviceToDevice, c.s));
        QE_CK(launch_codes_to_qf(codes, p, scales, zeros, q, p, pl.gsize, pl.grouped, c.qf, pl.ld, c.s));
        const ObjFuse f{c.objbase, W, wbf16, ldw, codes, nullptr};
        if ((st = residual(c, scales, zeros, &f)) != QE_OK) return st;
    } else {
        QE_CK(launch_init_residual(W, wbf16, ldw, nullptr, 0, q, p, pl.gsize, scales, zeros, c.R, pl.ld, c.s));
        QE_CK(cudaMemsetAsync(c.objbase, 0, 8, c.s));   // f(W) = 0
        src = SRC_W;
        if (opts && opts->wait_test) return sweep(c, codes, scales, zeros, bits, SRC_W, false, 0, nullptr, true);
        if (!relaxed(0)) {
            if ((st = sweep(c, codes, scales, zeros, bits, SRC_W, false, 0)) != QE_OK) return st;
            const ObjFuse f{obj, W, wbf16, ldw, codes, nullptr};
            if ((st = residual(c, scales, zeros, &f)) != QE_OK) return st;
            if ((st = record(0)) != QE_OK) return st;
            if ((st = form(0, 1, 0)) != QE_OK) return st;
            t = 1;
            src = SRC_CODES;
        }
    }
    if ((st = restart(src == SRC_CODES ? 1 : 3)) != QE_OK) return st;
    bool exact = true;   // R is the residual of the current What and no list has entries
    bool chain = false;  // the last sweep was a sequential one (its three-plane changes are in dp)
    const int dense = dense_sweeps(opts);
    // adaptive schedule (dense_sweeps = 0): dense sweeps until one changes fewer than
    // `below` codes, decided on the device after each sweep
    bool adaptive = false;
    int64_t below = 0;
    if (!(opts && opts->dense_sweeps > 0)) {
        if (opts && opts->switch_below > 0) {
            adaptive = true;
            below = opts->switch_below;
        } else if (!sbar_rows_fit_l2(p, pl.ld)) {
            adaptive = true;
            below = switch_below_model(q, p, c.nsm);
        }
    }
    while (t < iters) {
        const bool rx = relaxed(t);
        if (rx || src != SRC_CODES) {
            if (!exact && !chain) {   // from the change lists: refresh R from the codes
                if ((st = refresh()) != QE_OK) return st;
                if ((st = restart(3)) != QE_OK) return st;
                exact = true;
            }
            if ((st = sweep(c, codes, scales, zeros, bits, src, rx, exact ? -1 : 1)) != QE_OK) return st;
            QE_CK(launch_obj_step(c.rowdf, q, t == 0 ? c.objbase : obj + t - 1, obj + t, c.s));
            if ((st = record(t)) != QE_OK) return st;
            if ((st = form(t, 1, 0)) != QE_OK) return st;
            ++t;
            src = rx ? SRC_V : SRC_CODES;
            exact = false;
            chain = true;
            if (src == SRC_CODES && t < iters) {   // back on the grid
                if ((st = refresh()) != QE_OK) return st;
                if ((st = restart(1)) != QE_OK) return st;
                exact = true;
                chain = false;
            }
            continue;
        }
        // quantized sweeps up to the next relaxed one: sweeps 1 .. dense use the
        // tensor-core correction (one launch pair per block), later ones the change
        // lists, persistent over blocks and sweeps
        int tend = t;
        while (tend < iters && !relaxed(tend)) ++tend;
        if (adaptive && t < tend) {
            // both forms of every sweep are enqueued; the flag (reset here, where the
            // lists are empty or hold one sweep's changes) runs the dense form until
            // the switch sets it, then the list form (one launch per sweep)
            QE_CK(cudaMemsetAsync(c.swflag, 0, 16, c.s));   // flag and change counter
            for (; t < tend; ++t) {
                const double *prev_obj = t == 0 ? c.objbase : obj + t - 1;
                if ((st = sweep(c, codes, scales, zeros, bits, SRC_CODES, false, exact ? -1 : 1, c.swflag)) != QE_OK)
                    return st;
                QE_CK(launch_obj_step(c.rowdf, q, prev_obj, obj + t, c.s, c.swflag, 0));
                CdArgs a = list_args(c, codes, scales, zeros, bits);
                a.gate = c.swflag;
                a.gate_run = 1;
                {
                    Timed tm(c.timer, QE_KERNEL_CD_LISTS, c.s);
                    QE_CK(launch_cd_rows_lists(pl.B, a, t, t + 1, c.rowdft, nullptr, 0, free_changes(opts), 0, c.nsm,
                                               c.s));
                }
                QE_CK(launch_obj_prefix(c.rowdft, q, 1, prev_obj, obj + t, c.s, c.swflag, 1));
                if ((st = record(t)) != QE_OK) return st;
                if (opts && opts->sweep_forms) QE_CK(launch_record_form(c.swflag, opts->sweep_forms + t, c.s));
                if (t + 1 < tend) QE_CK(launch_list_switch(c.lcnt, q * pl.nblk, below, c.swcount, c.swflag, c.s));
                exact = false;
                chain = false;
            }
            continue;
        }
        for (; t < tend && t < dense; ++t) {
            if ((st = sweep(c, codes, scales, zeros, bits, SRC_CODES, false, exact ? -1 : 1)) != QE_OK) return st;
            QE_CK(launch_obj_step(c.rowdf, q, t == 0 ? c.objbase : obj + t - 1, obj + t, c.s));
            if ((st = record(t)) != QE_OK) return st;
            if ((st = form(t, 1, 1)) != QE_OK) return st;
            exact = false;
            chain = false;
        }
        while (t < tend) {
            const int te = (tend - t) < kSweepChunk ? tend : t + kSweepChunk;
            CdArgs a = list_args(c, codes, scales, zeros, bits);
            {
                Timed tm(c.timer, QE_KERNEL_CD_LISTS, c.s);
                // with empty lists (after a refresh) the first sweep steps in lockstep
                QE_CK(launch_cd_rows_lists(pl.B, a, t, te, c.rowdft, opts ? opts->sweep_codes : nullptr,
                                           exact ? 1 : 0, free_changes(opts), 0, c.nsm, c.s));
            }
            QE_CK(launch_obj_prefix(c.rowdft, q, te - t, t == 0 ? c.objbase : obj + t - 1, obj + t, c.s));
            if ((st = form(t, te - t, 2)) != QE_OK) return st;
            t = te;
            exact = false;
            chain = false;
        }
    }
    return QE_OK;
}

qe_status qe_quantize_layer_outlier(const void *W, qe_dtype w_dtype, int64_t q, int64_t p, int64_t ldw,
                                    const float *Sigma, int bits, int iters, int64_t s_budget,
                                    const qe_opts *opts, uint8_t *codes, float *scales, float *zeros,
                                    float *H_val, int64_t *H_idx, int64_t *H_nnz, double *obj,
                                    double *obj_cd, qe_stream_t stream) {
    qe_status st = check_layer(W, w_dtype, q, p, ldw, Sigma, bits, iters, codes, scales, zeros, obj);
    if (st != QE_OK) return st;
    if ((st = check_opts(opts, true)) != QE_OK) return st;
    const bool structured = opts && opts->structured_outliers == 1;
    const int64_t N = q * p;
    if (s_budget < 0 || s_budget > N || N >= (1ll << 32) || !H_nnz) return QE_ERR_INVALID_ARG;
    if (s_budget > 0 && (!H_val || !H_idx)) return QE_ERR_INVALID_ARG;
    const int wbf16 = (w_dtype == QE_BF16);
    const int power_iters = (opts && opts->power_iters > 0) ? opts->power_iters : kDefaultPowerIters;
    Ctx c;
    c.nsm = sm_count();
    const Plan pl = make_plan(q, p, block_width(opts), true, wbf16 ? 1 : 3, c.nsm);
    if ((st = setup_ctx(c, pl, opts, reinterpret_cast<cudaStream_t>(stream))) != QE_OK) return st;
    const int64_t ld = pl.ld;
    c.tie_eps = tie_eps(opts);
    c.Sig = Sigma;
    c.Wl = W;
    c.wbf16 = wbf16;
    c.ldw = ldw;
    c.Hr = c.H;   // the target of every sweep is W - H (dense H, leading dimension ld)

    // P_s: the s largest |T|, or with structured outliers the floor(s/q) columns of
    // largest l2 norm (Sec. 4.3, "Structured Outliers")
    auto select = [&](const float *T) -> cudaError_t {
        if (structured)
            return launch_topk_columns(T, q, p, s_budget / q, c.st, c.cg, c.ce, c.sb, c.eb, c.cpart, c.cnorm,
                                       c.ccols, c.cval, c.cn, H_idx, H_val, H_nnz, c.nsm, c.s);
        return launch_topk(T, N, s_budget, c.st, c.cg, c.ce, c.sb, c.eb, H_idx, H_val, H_nnz, c.nsm, c.s);
    };
    // H = P_s(W); the grid ignores those entries (Sec. 4.3)
    QE_CK(launch_flat_copy(W, wbf16, ldw, q, p, c.T, c.s));
    QE_CK(select(c.T));
    QE_CK(cudaMemsetAsync(c.H, 0, static_cast<size_t>(q) * ld * 4, c.s));
    QE_CK(launch_scatter_rowptr(H_idx, H_val, H_nnz, s_budget, q, p, c.H, ld, c.rowptr, c.s));
    QE_CK(launch_grid(W, wbf16, ldw, c.H, ld, q, p, p, bits, scales, zeros, c.err, c.s));
    // P_W = W (I + Sigma_bar), eta = 1 / (2 lambda_max), P = P_W - H (I + Sigma_bar)
    if ((st = prepare(c, W, wbf16, ldw, Sigma, c.PW)) != QE_OK) return st;
    QE_CK(launch_power_lambda(Sigma, p, p, power_iters, c.y0, c.y1, c.ppart, c.lam, c.eta, c.nsm, c.s));
    QE_CK(launch_spmm_refresh(c.PW, c.P, c.R, ld, c.sbar, ld, H_idx, H_val, c.rowptr, q, p, 0, scales,
                              c.s));
    if (opts && opts->wx_norm2)
        if ((st = objective(c, W, wbf16, ldw, c.H, nullptr, nullptr, nullptr, c.P, opts->wx_norm2)) != QE_OK)
            return st;
    const bool warm = opts && opts->init_codes;
    if (warm) {
        QE_CK(cudaMemcpyAsync(codes, opts->init_codes, static_cast<size_t>(q) * p, cudaMemcpyDeviceToDevice, c.s));
        QE_CK(launch_codes_to_qf(codes, p, scales, zeros, q, p, p, 0, c.qf, ld, c.s));
        if ((st = residual(c, scales, zeros)) != QE_OK) return st;
    } else {
        QE_CK(launch_init_residual(W, wbf16, ldw, c.H, ld, q, p, p, scales, zeros, c.R, ld, c.s));
    }
    // g of a warm start, the base of the first sweep's objective changes
    if (warm && obj_cd)
        if ((st = objective(c, W, wbf16, ldw, c.H, codes, scales, zeros, c.R, c.objbase)) != QE_OK) return st;
    for (int t = 0; t < iters; ++t) {
        if (t == 0 && !warm) {
            // sweep 1 from What = W: the blocked classic sweep, then the residual GEMM
            // (with g fused)
            if ((st = sweep(c, codes, scales, zeros, bits, SRC_W, false, 0)) != QE_OK) return st;
            const ObjFuse f{obj_cd ? obj_cd + t : nullptr, W, wbf16, ldw, codes, c.H};
            if ((st = residual(c, scales, zeros, obj_cd ? &f : nullptr)) != QE_OK) return st;
        } else {
            // R is exact and the target W - H stays fixed during the sweep: one
            // change-list sweep whose window starts empty (each block corrected by
            // this sweep's changes left of it), which ends by flushing the window into
            // R; g after it = g before + the objective changes of its decisions.  The
            // first such sweep of the call starts in lockstep; later ones take their
            // mode from the change counts the previous sweep left in the lists.
            const bool first_list = t == (warm ? 0 : 1);
            if (first_list) QE_CK(cudaMemsetAsync(c.lcnt, 0, static_cast<size_t>(q) * pl.nblk * 4, c.s));
            CdArgs a = list_args(c, codes, scales, zeros, bits);
            {
                Timed tm(c.timer, QE_KERNEL_CD_LISTS, c.s);
                QE_CK(launch_cd_rows_lists(pl.B, a, t, t + 1, c.rowdft, nullptr, first_list ? 1 : 2,
                                           free_changes(opts), 1, c.nsm, c.s));
            }
            if (obj_cd) QE_CK(launch_obj_prefix(c.rowdft, q, 1, t == 0 ? c.objbase : obj + t - 1, obj_cd + t, c.s));
        }
        // IHT step: T = H + 2 eta d (R - What); H = P_s(T)
        QE_CK(launch_iht_target(c.H, c.R, ld, codes, p, scales, zeros, c.d, c.eta, q, p, c.T, c.s));
        QE_CK(select(c.T));
        QE_CK(cudaMemsetAsync(c.H, 0, static_cast<size_t>(q) * ld * 4, c.s));
        QE_CK(launch_scatter_rowptr(H_idx, H_val, H_nnz, s_budget, q, p, c.H, ld, c.rowptr, c.s));
        // P = P_W - H (I + Sigma_bar); R += P_new - P_old  (R = P - What Sigma_bar stays current)
        QE_CK(launch_spmm_refresh(c.PW, c.P, c.R, ld, c.sbar, ld, H_idx, H_val, c.rowptr, q, p, 1, scales,
                                  c.s));
        if ((st = objective(c, W, wbf16, ldw, c.H, codes, scales, zeros, c.R, obj + t)) != QE_OK) return st;
        if (opts && opts->sweep_codes)
            QE_CK(cudaMemcpyAsync(opts->sweep_codes + static_cast<size_t>(t) * q * p, codes,
                                  static_cast<size_t>(q) * p, cudaMemcpyDeviceToDevice, c.s));
    }
    return QE_OK;
}

}  // extern "C"
