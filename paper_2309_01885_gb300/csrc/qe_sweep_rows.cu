// Explicit instantiations of the persistent change-list kernel at block widths 64
// and 128.
#define QE_SWEEP_INSTANTIATE
#include "qe_sweep.cuh"

namespace qe {
template cudaError_t launch_cd_rows_k<64> QE_SWEEP_ROWS_SIG;
template cudaError_t launch_cd_rows_k<128> QE_SWEEP_ROWS_SIG;
}  // namespace qe
