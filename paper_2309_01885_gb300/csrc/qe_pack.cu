// Bit-packed codes: the storage form of a quantized layer (the paper leaves the
// format open; Sec. 2.1 only fixes the codes as integers 0 .. 2^b - 1).  Row i
// is a little-endian bit stream: code j occupies bits [j b, (j + 1) b) of the
// row's bytes, least significant bit first.  Both kernels move one 32-bit word
// of the stream per thread (coalesced), so they are HBM-bound: q p bytes of
// codes against q p b / 8 bytes of stream.
#include "../../include/qe.h"
#include "qe_common.cuh"
#include "qe_internal.h"

namespace qe {
namespace {

// Word w of row i: bits [32 w, 32 w + 32) gather codes floor(32 w / b) ..
// floor((32 w + 31) / b) (a code may straddle two words).
__global__ void __launch_bounds__(256) k_pack_codes(const uint8_t *codes, int64_t q, int64_t p, int64_t ldc,
                                                    int bits, uint8_t *out, int64_t ldo, int64_t nbytes) {
    const int64_t w = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (4 * w >= nbytes) return;
    const uint32_t mask = (1u << bits) - 1u;
    const int64_t bit0 = 32 * w;
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        const uint8_t *row = codes + i * ldc;
        uint32_t word = 0u;
        for (int64_t j = bit0 / bits; j < p && j * bits < bit0 + 32; ++j) {
            const uint32_t c = row[j] & mask;
            const int64_t sh = j * bits - bit0;   // -bits < sh < 32
            word |= sh >= 0 ? (c << sh) : (c >> (-sh));
        }
        uint8_t *o = out + i * ldo + 4 * w;
        for (int k = 0; k < 4 && 4 * w + k < nbytes; ++k) o[k] = static_cast<uint8_t>(word >> (8 * k));
    }
}

__global__ void __launch_bounds__(256) k_unpack_codes(const uint8_t *packed, int64_t q, int64_t p, int64_t ldp,
                                                      int bits, uint8_t *codes, int64_t ldc, int64_t nbytes) {
    const int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (j >= p) return;
    const int64_t b0 = j * bits;
    // the code's bits lie in the bytes b0 / 8 and (b0 + bits - 1) / 8 (at most two)
    const int64_t k0 = b0 >> 3;
    for (int64_t i = blockIdx.y; i < q; i += gridDim.y) {
        const uint8_t *row = packed + i * ldp;
        uint32_t v = row[k0];
        if (k0 + 1 < nbytes) v |= static_cast<uint32_t>(row[k0 + 1]) << 8;
        codes[i * ldc + j] = static_cast<uint8_t>((v >> (b0 & 7)) & ((1u << bits) - 1u));
    }
}

}  // namespace
}  // namespace qe

using namespace qe;

extern "C" {

qe_status qe_pack_codes(const uint8_t *codes, int64_t q, int64_t p, int64_t ldc, int bits, uint8_t *out,
                        int64_t ldo, qe_stream_t stream) {
    if (!codes || !out || q < 1 || p < 1 || bits < 1 || bits > 8 || ldc < p) return QE_ERR_INVALID_ARG;
    const int64_t nbytes = (p * bits + 7) / 8;
    if (ldo < nbytes) return QE_ERR_INVALID_ARG;
    const dim3 grid(static_cast<unsigned>(ceil_div(ceil_div(nbytes, 4), 256)), static_cast<unsigned>(q < 65535 ? q : 65535));
    k_pack_codes<<<grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(codes, q, p, ldc, bits, out, ldo, nbytes);
    if (cudaGetLastError() != cudaSuccess) return QE_ERR_CUDA;
    return QE_OK;
}

qe_status qe_unpack_codes(const uint8_t *packed, int64_t q, int64_t p, int64_t ldp, int bits, uint8_t *codes,
                          int64_t ldc, qe_stream_t stream) {
    if (!packed || !codes || q < 1 || p < 1 || bits < 1 || bits > 8 || ldc < p) return QE_ERR_INVALID_ARG;
    const int64_t nbytes = (p * bits + 7) / 8;
    if (ldp < nbytes) return QE_ERR_INVALID_ARG;
    const dim3 grid(static_cast<unsigned>(ceil_div(p, 256)), static_cast<unsigned>(q < 65535 ? q : 65535));
    k_unpack_codes<<<grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(packed, q, p, ldp, bits, codes, ldc,
                                                                            nbytes);
    if (cudaGetLastError() != cudaSuccess) return QE_ERR_CUDA;
    return QE_OK;
}

}  // extern "C"
