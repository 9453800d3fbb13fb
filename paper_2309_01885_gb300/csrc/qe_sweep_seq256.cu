// Explicit instantiation of the sequential in-block kernel (real-valued changes:
// first, relaxed and post-relax sweeps) at block width 256 (the default), full blocks.
#define QE_SWEEP_INSTANTIATE
#include "qe_sweep.cuh"

namespace qe {
template cudaError_t launch_cd_block_k<256, true, true> QE_SWEEP_BLOCK_SIG;
}  // namespace qe
