// Explicit instantiation of the sequential in-block kernel at block width 256 for
// the ragged last block of a layer whose width is not a multiple of 256.
#define QE_SWEEP_INSTANTIATE
#include "qe_sweep.cuh"

namespace qe {
template cudaError_t launch_cd_block_k<256, true, false> QE_SWEEP_BLOCK_SIG;
}  // namespace qe
