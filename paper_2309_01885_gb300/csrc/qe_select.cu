// P_s, the hard-thresholding operator of the IHT step (Sec. 4.3, Eq. iht-update),
// as an entry point of its own: the radix select + stable compaction that the
// outlier-aware variant runs once per iteration, on a caller's flat fp32 array.
#include "../../include/qe.h"
#include "qe_common.cuh"
#include "qe_outlier.h"

namespace qe {
namespace {

struct SelectPlan {
    size_t st, cg, ce, sb, eb, total;
};

size_t aligned(size_t &cur, size_t bytes) {
    const size_t o = cur;
    cur += (bytes + 255) / 256 * 256;
    return o;
}

SelectPlan select_plan(int64_t N) {
    SelectPlan pl{};
    size_t cur = 0;
    const size_t nch = static_cast<size_t>(topk_chunks(N > 0 ? N : 1));
    pl.st = aligned(cur, sizeof(TopkState));
    pl.cg = aligned(cur, nch * 4);
    pl.ce = aligned(cur, nch * 4);
    pl.sb = aligned(cur, nch * 4);
    pl.eb = aligned(cur, nch * 4);
    pl.total = cur;
    return pl;
}

}  // namespace
}  // namespace qe

using namespace qe;

extern "C" {

qe_status qe_hard_threshold_workspace(int64_t N, size_t *bytes) {
    if (!bytes || N < 1 || N >= (1ll << 32)) return QE_ERR_INVALID_ARG;
    *bytes = select_plan(N).total;
    return QE_OK;
}

qe_status qe_hard_threshold(const float *T, int64_t N, int64_t s, int64_t *idx, float *val, int64_t *nnz,
                            void *workspace, size_t workspace_bytes, qe_stream_t stream) {
    if (!T || !nnz || !workspace || N < 1 || N >= (1ll << 32) || s < 0 || s > N) return QE_ERR_INVALID_ARG;
    if (s > 0 && (!idx || !val)) return QE_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return QE_ERR_INVALID_ARG;
    const SelectPlan pl = select_plan(N);
    if (workspace_bytes < pl.total) return QE_ERR_INVALID_ARG;
    int dev = 0, nsm = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return QE_ERR_CUDA;
    uint8_t *w = static_cast<uint8_t *>(workspace);
    const cudaError_t e =
        launch_topk(T, N, s, reinterpret_cast<TopkState *>(w + pl.st), reinterpret_cast<unsigned *>(w + pl.cg),
                    reinterpret_cast<unsigned *>(w + pl.ce), reinterpret_cast<unsigned *>(w + pl.sb),
                    reinterpret_cast<unsigned *>(w + pl.eb), idx, val, nnz, nsm,
                    reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? QE_OK : QE_ERR_CUDA;
}

}  // extern "C"
