// Placeholder until the tcgen05 TF32 kernel lands: reports "not handled" so
// weight_grad_dense falls back to the float32 kernel.
#include "common.cuh"

namespace csrt {
int gemm_tc_tf32(const float *, const float *, int32_t, int32_t, int32_t, float *, void *, size_t, cudaStream_t,
                 bool *handled) {
    *handled = false;
    return CSRT_OK;
}
}  // namespace csrt
