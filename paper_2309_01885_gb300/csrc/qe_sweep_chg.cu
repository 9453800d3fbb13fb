// Explicit instantiations of the change-driven in-block kernel (integer changes:
// dense window sweeps) and of its near-tie check at block widths 64 and 128.
#define QE_SWEEP_INSTANTIATE
#include "qe_sweep.cuh"

namespace qe {
template cudaError_t launch_cd_block_k<64, false, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_block_k<64, false, false> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_block_k<128, false, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_block_k<128, false, false> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_tie_check_k<64, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_tie_check_k<64, false> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_tie_check_k<128, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_tie_check_k<128, false> QE_SWEEP_BLOCK_SIG;
}  // namespace qe
