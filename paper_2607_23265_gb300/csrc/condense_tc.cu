// Condensed tokens Z_m = W_m X_m on the tcgen05 tensor cores (placeholder
// until the tensor-core kernel lands; the CUDA-core path serves meanwhile).
#include "wz_internal.cuh"

namespace wz {

bool tensor_path_available() { return false; }

cudaError_t launch_condense_tc(const Ctx &, cudaStream_t) { return cudaErrorNotSupported; }

}  // namespace wz
