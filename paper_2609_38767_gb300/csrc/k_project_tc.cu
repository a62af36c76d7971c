// k_project_tc.cu -- placeholder until the tensor-core projection lands.
#include "tda_internal.cuh"

namespace tda {
bool project_tc_supported(const tda_layer_desc&, const void*, const void*) { return false; }
cudaError_t launch_project_tc(const tda_layer_desc&, const void*, const void*, int64_t, float*, int64_t,
                              unsigned int*, cudaStream_t) {
    return cudaErrorNotSupported;
}
}  // namespace tda
