// Explicit instantiation of the persistent change-list kernel at block width 256
// (the default).
#define QE_SWEEP_INSTANTIATE
#include "qe_sweep.cuh"

namespace qe {
template cudaError_t launch_cd_rows_k<256> QE_SWEEP_ROWS_SIG;
}  // namespace qe
