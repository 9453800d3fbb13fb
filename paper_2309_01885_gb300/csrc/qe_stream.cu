// qe_build_sigma_host: Sigma = X X^T (Lemma 1) for bf16 X in host memory,
// streamed to the device in token chunks through caller-provided chunk
// buffers (two or more).  The host-to-device copies run on a per-device copy
// stream and overlap the tensor-core GEMMs that accumulate earlier chunks (and
// any work queued before the call on the caller's stream: with as many
// buffers as chunks, a whole X arrives while the previous layer computes).
#include <mutex>

#include "../../include/qe.h"
#include "qe_common.cuh"
#include "qe_internal.h"

namespace qe {
namespace {

constexpr int kMaxBuffers = 64;

// Per-device copy stream and the events that hand the chunk buffers back and forth:
// copied[b]: buffer b holds its chunk; freed[b]: the GEMM that read buffer b is done.
// next: the buffer the next chunk goes to; the rotation carries over from call to
// call, so with more buffers than chunks per call a call's copies go to buffers that
// an earlier call's GEMMs released long before, and the copy stream never waits.
struct CopyState {
    cudaStream_t copy = nullptr;
    int nev = 0;
    int next = 0;
    cudaEvent_t copied[kMaxBuffers] = {};
    cudaEvent_t freed[kMaxBuffers] = {};
};

std::mutex g_copy_mu;
CopyState g_copy[64];

qe_status copy_state(int dev, int nbuf, CopyState **out) {
    CopyState &c = g_copy[dev];
    if (!c.copy && cudaStreamCreateWithFlags(&c.copy, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        c.copy = nullptr;
        return QE_ERR_CUDA;
    }
    for (; c.nev < nbuf; ++c.nev) {
        if (cudaEventCreateWithFlags(&c.copied[c.nev], cudaEventDisableTiming) != cudaSuccess ||
            cudaEventCreateWithFlags(&c.freed[c.nev], cudaEventDisableTiming) != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
    }
    *out = &c;
    return QE_OK;
}

}  // namespace
}  // namespace qe

using namespace qe;

extern "C" qe_status qe_build_sigma_host(const void *X, int64_t p, int64_t n, int64_t ldx, float *Sigma,
                                         int accumulate, void *staging, size_t staging_bytes, int64_t chunk,
                                         qe_stream_t stream) {
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    if (!X || !Sigma || !staging || p < 1 || n < 0 || p > (1ll << 30) || ldx < n) return QE_ERR_INVALID_ARG;
    if (chunk < 64 || chunk % 64 != 0 || chunk > (1ll << 30)) return QE_ERR_INVALID_ARG;
    const size_t buf_bytes = static_cast<size_t>(p) * static_cast<size_t>(chunk) * 2;
    if (staging_bytes < 2 * buf_bytes || (reinterpret_cast<uintptr_t>(staging) & 15u) != 0)
        return QE_ERR_INVALID_ARG;
    if (n == 0) {
        if (!accumulate && cudaMemsetAsync(Sigma, 0, static_cast<size_t>(p) * p * 4, s) != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
        return QE_OK;
    }
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) {
        cudaGetLastError();
        return QE_ERR_CUDA;
    }
    unsigned *err = device_error_word();
    if (!err) return QE_ERR_CUDA;
    // as many chunk buffers as the staging area holds (at most kMaxBuffers)
    const int64_t fit = static_cast<int64_t>(staging_bytes / buf_bytes);
    const int nbuf = static_cast<int>(fit < kMaxBuffers ? fit : kMaxBuffers);
    std::lock_guard<std::mutex> lock(g_copy_mu);
    CopyState *cs = nullptr;
    qe_status st = copy_state(dev, nbuf, &cs);
    if (st != QE_OK) return st;
    GemmArgs g;
    memset(&g, 0, sizeof(g));
    g.M = static_cast<int>(p);
    g.N = static_cast<int>(p);
    g.n_prod = 1;
    g.mode = EPI_SIGMA;
    g.out = Sigma;
    g.ldo = p;
    g.err = err;
    const __nv_bfloat16 *Xh = static_cast<const __nv_bfloat16 *>(X);
    for (int64_t n0 = 0; n0 < n; n0 += chunk) {
        const int b = cs->next % nbuf;
        cs->next = (b + 1) % nbuf;
        uint8_t *buf = static_cast<uint8_t *>(staging) + static_cast<size_t>(b) * buf_bytes;
        CUtensorMap ta, tb;
        if (!make_tmap_bf16(&ta, buf, p, chunk, chunk, 128) || !make_tmap_bf16(&tb, buf, p, chunk, chunk, 256))
            return QE_ERR_CUDA;
        const int64_t len = (n - n0) < chunk ? (n - n0) : chunk;
        const int64_t rlen = round_up(len, 64);
        cudaError_t e = cudaStreamWaitEvent(cs->copy, cs->freed[b], 0);
        if (e == cudaSuccess)
            e = cudaMemcpy2DAsync(buf, chunk * 2, Xh + n0, ldx * 2, len * 2, p, cudaMemcpyHostToDevice, cs->copy);
        if (e == cudaSuccess && rlen > len)   // the GEMM reads whole 64-token blocks
            e = cudaMemset2DAsync(buf + len * 2, chunk * 2, 0, (rlen - len) * 2, p, cs->copy);
        if (e == cudaSuccess) e = cudaEventRecord(cs->copied[b], cs->copy);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, cs->copied[b], 0);
        g.kb_count = static_cast<int>(rlen / 64);
        g.accumulate = (n0 > 0) ? 1 : accumulate;
        if (e == cudaSuccess) e = launch_tc_gemm(256, ta, tb, g, 1, s);
        if (e == cudaSuccess) e = cudaEventRecord(cs->freed[b], s);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return QE_ERR_CUDA;
        }
    }
    return QE_OK;
}
