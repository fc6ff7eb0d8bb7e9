// Internal interface between the C-ABI front end (uq_api.cu, which validates
// arguments) and the kernel translation units (which pick a template
// instantiation and launch).  Each launcher returns the cudaError_t of its
// launch.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/uq_api.h"

namespace uq {

struct Shape {
    int64_t out;
    int n_in;
    int q;
    int g;
    int wdtype;     // uq_wdtype
};

cudaError_t launch_fwd(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode,
                       float* what, cudaStream_t st);
cudaError_t launch_bwd(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                       uq_grads gr, cudaStream_t st, int filter = UQ_FILTER_STE);
cudaError_t launch_export(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                          uint32_t* planes, float* astar, float* zstar, cudaStream_t st);
// The same export with alpha*, z_B* written as IEEE half (bits), rounded to nearest even.
cudaError_t launch_export_half(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                               uint32_t* planes, uint16_t* astar, uint16_t* zstar, cudaStream_t st);
cudaError_t launch_init(const Shape& sh, const void* W, int G, int T, int clip, uq_params p, uint8_t* codes,
                        cudaStream_t st);

// Persistent TMA-pipelined kernels (uq_stream.cu): used when stream_path_ok.
bool stream_path_ok(const Shape& sh);
cudaError_t launch_fwd_stream(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode,
                              float* what, cudaStream_t st);
cudaError_t launch_bwd_stream(const Shape& sh, const void* W, uq_params p, const uint8_t* codes,
                              const float* gup, uq_grads gr, cudaStream_t st, int filter = UQ_FILTER_STE);
// Fused optimisation step (uq_step.cu): backward of step t, SGD update,
// forward of step t + 1 in `mode` (a FWD_* value).  step_path_ok tells
// whether the shape is one the fused kernel handles.
bool step_path_ok(const Shape& sh);
cudaError_t launch_step(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const float* gup, float lr_f,
                        float lr_b, int mode, float* what, cudaStream_t st);
// Reads (and optionally clears) the fused step kernel's bounded-wait flag.
cudaError_t step_error(bool clear, unsigned int* flag);
// The fused step with bf16 dL/dW^ and W^ (uq_step_bf16.cu), and its flag.
cudaError_t launch_step_bf16(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const uint16_t* gup,
                             float lr_f, float lr_b, int mode, uint16_t* what, cudaStream_t st);
cudaError_t step_bf16_error(bool clear, unsigned int* flag);
// BCQ matrix-vector product from the exported bit-planes (uq_gemv.cu); `work`
// holds gemv_workspace_floats(out, in, batch) floats of per-tile partials.
int64_t gemv_workspace_floats(int64_t out, int64_t n_in, int batch);
// The library's own scratch for the product (uq_bcq_gemv_noalloc): its size in
// floats, and its device address on the current device (looked up once per device).
int64_t gemv_static_workspace_floats();
cudaError_t gemv_static_workspace(float** work);
// Reads (and optionally clears) the flag the product's tensor-copy staging sets
// when a bounded wait runs out.
cudaError_t gemv_error(bool clear, unsigned int* flag);
cudaError_t launch_gemv(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in, int q,
                        int g, const void* x, int xdtype, int batch, float* y, float* work, cudaStream_t st);
// UniQuan with OmniQuant's maps (uq_omni.cu); omni_ok: the group sizes it takes.
bool omni_ok(const Shape& sh);
cudaError_t launch_omni_fwd(const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes, int mode, float* what,
                            cudaStream_t st);
cudaError_t launch_omni_bwd(const Shape& sh, const void* W, uq_params_omni p, const uint8_t* codes, const float* gup,
                            uq_grads_omni gr, cudaStream_t st);
// Reads (and optionally clears) the OmniQuant-map kernels' bounded-wait flag.
cudaError_t omni_error(bool clear, unsigned int* flag);
cudaError_t awq_error(bool clear, unsigned int* flag);
cudaError_t launch_omni_scales(const Shape& sh, const void* W, const float* beta, const float* gamma, float* delta,
                               float* zo, cudaStream_t st);
// UniQuan with AWQ's maps (uq_awq.cu); awq_ok: the group sizes it takes;
// awq_workspace_floats: floats of per-row-range ds_A partials the backward needs.
bool awq_ok(const Shape& sh);
int64_t awq_workspace_floats(const Shape& sh);
cudaError_t launch_awq_fwd(const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes, int mode, float* what,
                           cudaStream_t st);
cudaError_t launch_awq_bwd(const Shape& sh, const void* W, uq_params_awq p, const uint8_t* codes, const float* gup,
                           uq_grads_awq gr, float* work, cudaStream_t st);
// Launches the bounded-wait self-test (one warp, a wait that runs out).
cudaError_t launch_wait_selftest(cudaStream_t st);
// Streaming multiprocessors of the current device (cached per device).
int sm_count();
// Reads (and optionally clears) the flag a pipelined kernel sets when a
// bounded wait runs out.
cudaError_t stream_error(bool clear, unsigned int* flag);

// Forward modes (see uq_api.h): full mapping, local remap step, keep codes.
enum { FWD_FULL = 0, FWD_REMAP = 1, FWD_KEEP = 2 };

}  // namespace uq
