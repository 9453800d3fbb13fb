// qe_build_sigma_static: Sigma = X X^T without any device allocation.
//
// qe_build_sigma stages token-major (or unaligned) bf16 X through a scratch
// buffer it allocates with cudaMallocAsync.  Some callers cannot let a library
// allocate at all: a process whose device memory is handed out entirely by
// its own allocator, a latency-critical loop that must not touch the
// allocator, or a platform without stream-ordered allocation.  This variant
// stages through a fixed array that is part of the library's device image
// instead, so the call itself never allocates.
//
// The array is a file-scope __device__ object: every GPU that loads the
// library holds its QE_STATIC_SCRATCH_BYTES until the process exits.  Host
// code must not pass the symbol itself to a kernel or a copy (on the host it
// names a host-side stand-in, not device memory); the device address is
// looked up once per device with cudaGetSymbolAddress, on the first call made
// with that device current, and cached.  All calls share the array, so calls
// that overlap on the GPU (different streams, or different host threads) race.
#include <mutex>

#include "../../include/qe.h"
#include "qe_common.cuh"
#include "qe_internal.h"

namespace qe {
namespace {

static __device__ __align__(256) unsigned char g_static_scratch[QE_STATIC_SCRATCH_BYTES];

std::mutex g_scratch_mu;
void *g_scratch_ptr[64] = {};

// Device address of g_static_scratch on the current device (looked up once).
qe_status static_scratch(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return QE_ERR_CUDA;
    }
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_static_scratch);
        if (e != cudaSuccess || p == nullptr) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return QE_OK;
}

}  // namespace
}  // namespace qe

using namespace qe;

extern "C" qe_status qe_build_sigma_static(const void *X, qe_dtype x_dtype, qe_xlayout layout, int64_t p,
                                           int64_t n, int64_t ldx, float *Sigma, int accumulate,
                                           qe_stream_t stream) {
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (!X || !Sigma || p < 1 || n < 0 || p > (1ll << 30)) return QE_ERR_INVALID_ARG;
    if (x_dtype != QE_F32 && x_dtype != QE_BF16) return QE_ERR_INVALID_ARG;
    if (layout != QE_FEATURE_MAJOR && layout != QE_TOKEN_MAJOR) return QE_ERR_INVALID_ARG;
    if (layout == QE_FEATURE_MAJOR ? ldx < n : ldx < p) return QE_ERR_INVALID_ARG;
    const bool direct = x_dtype == QE_F32 ||
                        (layout == QE_FEATURE_MAJOR && ((reinterpret_cast<uintptr_t>(X) & 15u) == 0) &&
                         (ldx % 8 == 0));
    // the staging chunk is p x nc bf16 with nc a positive multiple of 64 tokens
    const int64_t max_nc = static_cast<int64_t>(QE_STATIC_SCRATCH_BYTES) / (2 * p) / 64 * 64;
    if (!direct && max_nc < 64) return QE_ERR_INVALID_ARG;
    if (n == 0) {
        if (!accumulate && cudaMemsetAsync(Sigma, 0, static_cast<size_t>(p) * p * 4, s) != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
        return QE_OK;
    }
    void *scratch = nullptr;
    qe_status st = static_scratch(&scratch);
    if (st != QE_OK) return st;
    unsigned *err = device_error_word();   // timeouts latch where qe_sync_status reads them
    if (!err) return QE_ERR_CUDA;
    if (x_dtype == QE_F32) {
        const float *Xf = static_cast<const float *>(X);
        const cudaError_t e = layout == QE_FEATURE_MAJOR ? launch_sigma_f32(Xf, p, n, ldx, 1, Sigma, accumulate, s)
                                                         : launch_sigma_f32(Xf, p, n, 1, ldx, Sigma, accumulate, s);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
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
    if (direct) {
        CUtensorMap ta, tb;
        if (!make_tmap_bf16(&ta, X, p, n, ldx, 128) || !make_tmap_bf16(&tb, X, p, n, ldx, 256)) return QE_ERR_CUDA;
        g.kb_count = static_cast<int>(ceil_div(n, 64));
        g.accumulate = accumulate;
        if (launch_tc_gemm(256, ta, tb, g, 1, s) != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
        return QE_OK;
    }
    // stage feature-major chunks of tokens through the fixed array
    int64_t nc = max_nc < 8192 ? max_nc : 8192;
    if (nc > round_up(n, 64)) nc = round_up(n, 64);
    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, scratch, p, nc, nc, 128) || !make_tmap_bf16(&tb, scratch, p, nc, nc, 256))
        return QE_ERR_CUDA;
    for (int64_t n0 = 0; n0 < n; n0 += nc) {
        const int64_t len = (n - n0) < nc ? (n - n0) : nc;
        cudaError_t e;
        if (layout == QE_TOKEN_MAJOR) {
            e = launch_transpose_bf16(X, n0, len, p, ldx, scratch, nc, s);
        } else {
            e = cudaMemcpy2DAsync(scratch, nc * 2, static_cast<const __nv_bfloat16 *>(X) + n0, ldx * 2, len * 2, p,
                                  cudaMemcpyDeviceToDevice, s);
        }
        // the array keeps the previous call's tokens: clear the unused tail of a short chunk
        if (e == cudaSuccess && len < nc)
            e = cudaMemset2DAsync(static_cast<__nv_bfloat16 *>(scratch) + len, nc * 2, 0, (nc - len) * 2, p, s);
        g.kb_count = static_cast<int>(ceil_div(len, 64));
        g.accumulate = (n0 > 0) ? 1 : accumulate;
        if (e == cudaSuccess) e = launch_tc_gemm(256, ta, tb, g, 1, s);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
    }
    return QE_OK;
}
