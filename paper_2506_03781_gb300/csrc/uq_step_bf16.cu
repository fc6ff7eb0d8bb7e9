// Fused optimisation step with bf16 dL/dW^ and W^ (uq_train_step_bf16): the
// same kernel as uq_step.cu (uq_step.cuh), instantiated for bf16 input
// gradients and bf16 output weights, in a translation unit of its own so
// that the two variants compile in parallel.
#include <cstdint>

namespace uq {
// bounded-wait flag of this translation unit's step kernels (uq_check_device)
static __device__ unsigned int g_step_err = 0;
}  // namespace uq

#include "uq_step.cuh"

namespace uq {

cudaError_t launch_step_bf16(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const uint16_t* gup,
                             float lr_f, float lr_b, int mode, uint16_t* what, cudaStream_t st) {
    return step_q<true>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
}

cudaError_t step_bf16_error(bool clear, unsigned int* flag) {
    unsigned int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_step_err, sizeof(v));
    if (e != cudaSuccess) return e;
    *flag = v;
    if (clear && v) {
        const unsigned int z = 0;
        e = cudaMemcpyToSymbol(g_step_err, &z, sizeof(z));
    }
    return e;
}

}  // namespace uq
