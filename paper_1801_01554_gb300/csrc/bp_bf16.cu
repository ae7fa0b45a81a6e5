// bfloat16 tensor-core path (placeholder until the tcgen05 kernels land).
#include "bp_bf16.h"

namespace bp {

bp_status bf16_check_shape(const int*, int, int) { return BP_ESHAPE; }
const char* bf16_last_message() { return "the bfloat16 path is not built yet"; }
bp_status bf16_create(const int*, int, int, int, float*, float*, float*, Bf16Net**) {
    return BP_ESHAPE;
}
void bf16_destroy(Bf16Net*) {}
void bf16_set_flags(Bf16Net*, int*) {}
cudaError_t bf16_refresh_weights(Bf16Net*, cudaStream_t) { return cudaErrorNotSupported; }
cudaError_t bf16_forward(Bf16Net*, const void*, int, void*, cudaStream_t) {
    return cudaErrorNotSupported;
}
cudaError_t bf16_backward(Bf16Net*, const void*, const void*, int, float*, bool, cudaStream_t) {
    return cudaErrorNotSupported;
}
cudaError_t bf16_update(Bf16Net*, float, float, float, cudaStream_t) {
    return cudaErrorNotSupported;
}
cudaError_t bf16_train(Bf16Net*, const void*, const void*, int, int, float*, float, float, float,
                       bool, cudaStream_t) {
    return cudaErrorNotSupported;
}

}  // namespace bp
