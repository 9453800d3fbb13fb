// Explicit instantiations of the sequential in-block kernel (real-valued changes:
// first, relaxed and post-relax sweeps) at block widths 64 and 128.
#define QE_SWEEP_INSTANTIATE
#include "qe_sweep.cuh"

namespace qe {
template cudaError_t launch_cd_block_k<64, true, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_block_k<64, true, false> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_block_k<128, true, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_block_k<128, true, false> QE_SWEEP_BLOCK_SIG;
}  // namespace qe
