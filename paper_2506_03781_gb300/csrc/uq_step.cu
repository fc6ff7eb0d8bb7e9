// Fused optimisation step with fp32 dL/dW^ and W^ (uq_train_step); the
// kernel itself is in uq_step.cuh.
#include <cstdint>

namespace uq {
// bounded-wait flag of this translation unit's step kernels (uq_check_device)
static __device__ unsigned int g_step_err = 0;
}  // namespace uq

#include "uq_step.cuh"

namespace uq {

static int step_units(const Shape& sh) { return sh.n_in / (sh.g == 32 ? 256 : 512); }

bool step_path_ok(const Shape& sh) {
    if (!stream_path_ok(sh)) return false;
    return step_units(sh) <= kWarps * kMaxCluster;
}

cudaError_t launch_step(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const float* gup, float lr_f,
                        float lr_b, int mode, float* what, cudaStream_t st) {
    return step_q<false>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
}

cudaError_t step_error(bool clear, unsigned int* flag) {
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
