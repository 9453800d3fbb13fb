// Explicit instantiations of the change-driven in-block kernel (integer changes:
// dense window sweeps) and of its near-tie check at block width 256 (the default).
#define QE_SWEEP_INSTANTIATE
#include "qe_sweep.cuh"

namespace qe {
template cudaError_t launch_cd_block_k<256, false, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_block_k<256, false, false> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_tie_check_k<256, true> QE_SWEEP_BLOCK_SIG;
template cudaError_t launch_cd_tie_check_k<256, false> QE_SWEEP_BLOCK_SIG;
}  // namespace qe
