// C-ABI front end: argument validation, error reporting, dispatch to the
// kernel launchers.  Nothing here allocates device memory or keeps a
// pointer beyond the call.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <cstdint>

#include "uq_launch.h"

namespace {

thread_local char g_err[512] = "";

uq_status fail(uq_status st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return st;
}

uq_status ok() {
    g_err[0] = '\0';
    return UQ_OK;
}

constexpr int64_t kMaxIn = int64_t(1) << 24;   // row lengths whose 32-bit per-row offsets stay exact

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Checks shape, q, g, W dtype.  Returns UQ_OK or an error status.
uq_status check_shape(int64_t out, int64_t in, int q, int g, int wdtype) {
    if (q < 1 || q > 4) return fail(UQ_ERR_UNSUPPORTED, "q=%d: bit-widths 1..4 are supported", q);
    if (out < 1 || in < 1) return fail(UQ_ERR_ARG, "empty matrix: out=%lld in=%lld", (long long)out, (long long)in);
    if (out > 0x7fffffffLL) return fail(UQ_ERR_ARG, "out=%lld exceeds 2^31-1 rows", (long long)out);
    if (g < 32 || g % 32 != 0) return fail(UQ_ERR_ARG, "g=%d must be a positive multiple of 32", g);
    if (in % g != 0) return fail(UQ_ERR_ARG, "in=%lld is not a multiple of g=%d", (long long)in, g);
    if (!(g == 32 || g == 64 || g % 128 == 0))
        return fail(UQ_ERR_UNSUPPORTED, "g=%d: supported group sizes are 32, 64 and multiples of 128", g);
    if (in > kMaxIn) return fail(UQ_ERR_UNSUPPORTED, "in=%lld exceeds %lld", (long long)in, (long long)kMaxIn);
    if (wdtype != UQ_W_F32 && wdtype != UQ_W_BF16) return fail(UQ_ERR_ARG, "unknown weight dtype %d", wdtype);
    return UQ_OK;
}

uq_status check_ptr(const void* p, const char* name) {
    if (p == nullptr) return fail(UQ_ERR_ARG, "%s is NULL", name);
    if (!aligned16(p)) return fail(UQ_ERR_ALIGN, "%s=%p is not 16-byte aligned", name, p);
    return UQ_OK;
}

#define UQ_TRY(expr)                      \
    do {                                  \
        uq_status _s = (expr);            \
        if (_s != UQ_OK) return _s;       \
    } while (0)

uq_status cuda_status(cudaError_t e, const char* what) {
    if (e != cudaSuccess) return fail(UQ_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
    return ok();
}

// The product cuts the columns into tiles of 512; a row's groups must either
// tile a column tile exactly (g divides 512) or be made of whole tiles (512
// divides g), so that every group boundary falls on a lane boundary the
// kernels know at compile time.
uq_status check_gemv_group(int g) {
    if (512 % g != 0 && g % 512 != 0)
        return fail(UQ_ERR_UNSUPPORTED,
                    "g=%d: the BCQ product needs g to divide 512 or to be a multiple of 512 (32, 64, 128, 256, "
                    "512, 1024, ...)",
                    g);
    return UQ_OK;
}

}  // namespace

extern "C" {

int uq_abi_version(void) { return 1; }

const char* uq_last_error(void) { return g_err; }

uq_status uq_init_params(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, int G, int T,
                         uq_clip clip, uq_params p, uint8_t* codes, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    if (g > 32768) return fail(UQ_ERR_UNSUPPORTED, "initialization supports g <= 32768 (g=%d)", g);
    if (G < 1) return fail(UQ_ERR_ARG, "G=%d must be >= 1", G);
    if (T < 0) return fail(UQ_ERR_ARG, "T=%d must be >= 0", T);
    if (clip != UQ_CLIP_FIXED_MIN && clip != UQ_CLIP_FIXED_MAX && clip != UQ_CLIP_BALANCED)
        return fail(UQ_ERR_ARG, "unknown clipping strategy %d", (int)clip);
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.s, "params.s"));
    UQ_TRY(check_ptr(p.sr, "params.sr"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    return cuda_status(uq::launch_init(sh, W, G, T, (int)clip, p, codes, (cudaStream_t)stream), "uq_init_params");
}

uq_status uq_quantize_fwd(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, uq_params p,
                          uint8_t* codes, uq_map map, int64_t step, int p_period, float* W_hat, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    if (map != UQ_MAP_FULL && map != UQ_MAP_LOCAL_PERIODIC) return fail(UQ_ERR_ARG, "unknown mapping %d", (int)map);
    if (p_period < 1) return fail(UQ_ERR_ARG, "p_period=%d must be >= 1", p_period);
    if (step < 0) return fail(UQ_ERR_ARG, "step=%lld must be >= 0", (long long)step);
    const int mode = map == UQ_MAP_FULL ? uq::FWD_FULL : (step % p_period == 0 ? uq::FWD_REMAP : uq::FWD_KEEP);
    if (mode != uq::FWD_KEEP) {
        UQ_TRY(check_ptr(W, "W"));
        UQ_TRY(check_ptr(p.s, "params.s"));
        UQ_TRY(check_ptr(p.sr, "params.sr"));
    }
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(W_hat, "W_hat"));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    return cuda_status(uq::launch_fwd(sh, W, p, codes, mode, W_hat, (cudaStream_t)stream), "uq_quantize_fwd");
}

uq_status uq_quantize_bwd(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, uq_params p,
                          const uint8_t* codes, const float* dL_dWhat, uq_grads gr, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.s, "params.s"));
    UQ_TRY(check_ptr(p.sr, "params.sr"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(dL_dWhat, "dL_dWhat"));
    UQ_TRY(check_ptr(gr.ddelta, "grads.ddelta"));
    UQ_TRY(check_ptr(gr.dzu, "grads.dzu"));
    UQ_TRY(check_ptr(gr.ds, "grads.ds"));
    UQ_TRY(check_ptr(gr.dsr, "grads.dsr"));
    UQ_TRY(check_ptr(gr.dalpha, "grads.dalpha"));
    UQ_TRY(check_ptr(gr.dzb, "grads.dzb"));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    return cuda_status(uq::launch_bwd(sh, W, p, codes, dL_dWhat, gr, (cudaStream_t)stream), "uq_quantize_bwd");
}

uq_status uq_quantize_bwd_ex(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, uq_params p,
                             const uint8_t* codes, const float* dL_dWhat, uq_grads gr, uq_filter filter,
                             void* stream) {
    if (filter != UQ_FILTER_STE && filter != UQ_FILTER_ELEMENT)
        return fail(UQ_ERR_ARG, "unknown gradient filter %d", (int)filter);
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.s, "params.s"));
    UQ_TRY(check_ptr(p.sr, "params.sr"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(dL_dWhat, "dL_dWhat"));
    UQ_TRY(check_ptr(gr.ddelta, "grads.ddelta"));
    UQ_TRY(check_ptr(gr.dzu, "grads.dzu"));
    UQ_TRY(check_ptr(gr.ds, "grads.ds"));
    UQ_TRY(check_ptr(gr.dsr, "grads.dsr"));
    UQ_TRY(check_ptr(gr.dalpha, "grads.dalpha"));
    UQ_TRY(check_ptr(gr.dzb, "grads.dzb"));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    return cuda_status(uq::launch_bwd(sh, W, p, codes, dL_dWhat, gr, (cudaStream_t)stream, (int)filter),
                       "uq_quantize_bwd_ex");
}

uq_status uq_export_bcq_half(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, uq_params p,
                             const uint8_t* codes, uq_export_mode mode, uint32_t* bitplanes, uint16_t* alpha_star,
                             uint16_t* zb_star, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    if (mode != UQ_EXPORT_REUSE_CODES && mode != UQ_EXPORT_REMAP_EQ4)
        return fail(UQ_ERR_ARG, "unknown export mode %d", (int)mode);
    if (mode == UQ_EXPORT_REMAP_EQ4) UQ_TRY(check_ptr(W, "W"));
    else UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(bitplanes, "bitplanes"));
    UQ_TRY(check_ptr(alpha_star, "alpha_star"));
    UQ_TRY(check_ptr(zb_star, "zb_star"));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    return cuda_status(uq::launch_export_half(sh, W, p, codes, (int)mode, bitplanes, alpha_star, zb_star,
                                              (cudaStream_t)stream),
                       "uq_export_bcq_half");
}

uq_status uq_train_step(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, uq_params p,
                        uint8_t* codes, const float* dL_dWhat, float lr_F, float lr_B, uq_map map, int64_t step,
                        int p_period, float* W_hat, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    if (map != UQ_MAP_FULL && map != UQ_MAP_LOCAL_PERIODIC) return fail(UQ_ERR_ARG, "unknown mapping %d", (int)map);
    if (p_period < 1) return fail(UQ_ERR_ARG, "p_period=%d must be >= 1", p_period);
    if (step < 0 || step == INT64_MAX) return fail(UQ_ERR_ARG, "step=%lld must be in [0, 2^63 - 1)", (long long)step);
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    if (!uq::step_path_ok(sh))
        return fail(UQ_ERR_UNSUPPORTED,
                    "the fused step handles g in {32, 64, 128} with in a multiple of %d and at most %d (g=%d in=%lld); "
                    "use uq_quantize_bwd and uq_quantize_fwd",
                    g == 32 ? 256 : 512, g == 32 ? 16384 : 32768, g, (long long)in);
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.s, "params.s"));
    UQ_TRY(check_ptr(p.sr, "params.sr"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(dL_dWhat, "dL_dWhat"));
    UQ_TRY(check_ptr(W_hat, "W_hat"));
    const int64_t next = step + 1;
    const int mode = map == UQ_MAP_FULL ? uq::FWD_FULL : (next % p_period == 0 ? uq::FWD_REMAP : uq::FWD_KEEP);
    return cuda_status(uq::launch_step(sh, W, p, codes, dL_dWhat, lr_F, lr_B, mode, W_hat, (cudaStream_t)stream),
                       "uq_train_step");
}

uq_status uq_train_step_bf16(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, uq_params p,
                             uint8_t* codes, const uint16_t* dL_dWhat, float lr_F, float lr_B, uq_map map,
                             int64_t step, int p_period, uint16_t* W_hat, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    if (map != UQ_MAP_FULL && map != UQ_MAP_LOCAL_PERIODIC) return fail(UQ_ERR_ARG, "unknown mapping %d", (int)map);
    if (p_period < 1) return fail(UQ_ERR_ARG, "p_period=%d must be >= 1", p_period);
    if (step < 0 || step == INT64_MAX) return fail(UQ_ERR_ARG, "step=%lld must be in [0, 2^63 - 1)", (long long)step);
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    if (!uq::step_path_ok(sh))
        return fail(UQ_ERR_UNSUPPORTED,
                    "the fused step handles g in {32, 64, 128} with in a multiple of %d and at most %d (g=%d in=%lld)",
                    g == 32 ? 256 : 512, g == 32 ? 16384 : 32768, g, (long long)in);
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.s, "params.s"));
    UQ_TRY(check_ptr(p.sr, "params.sr"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(dL_dWhat, "dL_dWhat"));
    UQ_TRY(check_ptr(W_hat, "W_hat"));
    const int64_t next = step + 1;
    const int mode = map == UQ_MAP_FULL ? uq::FWD_FULL : (next % p_period == 0 ? uq::FWD_REMAP : uq::FWD_KEEP);
    return cuda_status(
        uq::launch_step_bf16(sh, W, p, codes, dL_dWhat, lr_F, lr_B, mode, W_hat, (cudaStream_t)stream),
        "uq_train_step_bf16");
}

uq_status uq_quantize_fwd_omni(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                               uq_params_omni p, uint8_t* codes, uq_map map, int64_t step, int p_period,
                               float* W_hat, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    if (!uq::omni_ok(sh)) return fail(UQ_ERR_UNSUPPORTED, "g=%d: the OmniQuant maps take g in {32, 64, 128, 256, 512}", g);
    if (map != UQ_MAP_FULL && map != UQ_MAP_LOCAL_PERIODIC) return fail(UQ_ERR_ARG, "unknown mapping %d", (int)map);
    if (p_period < 1) return fail(UQ_ERR_ARG, "p_period=%d must be >= 1", p_period);
    if (step < 0) return fail(UQ_ERR_ARG, "step=%lld must be >= 0", (long long)step);
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.beta, "params.beta"));
    UQ_TRY(check_ptr(p.gamma, "params.gamma"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(W_hat, "W_hat"));
    const int mode = map == UQ_MAP_FULL ? uq::FWD_FULL : (step % p_period == 0 ? uq::FWD_REMAP : uq::FWD_KEEP);
    return cuda_status(uq::launch_omni_fwd(sh, W, p, codes, mode, W_hat, (cudaStream_t)stream), "uq_quantize_fwd_omni");
}

uq_status uq_quantize_bwd_omni(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                               uq_params_omni p, const uint8_t* codes, const float* dL_dWhat, uq_grads_omni gr,
                               void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    if (!uq::omni_ok(sh)) return fail(UQ_ERR_UNSUPPORTED, "g=%d: the OmniQuant maps take g in {32, 64, 128, 256, 512}", g);
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.beta, "params.beta"));
    UQ_TRY(check_ptr(p.gamma, "params.gamma"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(dL_dWhat, "dL_dWhat"));
    UQ_TRY(check_ptr(gr.dbeta, "grads.dbeta"));
    UQ_TRY(check_ptr(gr.dgamma, "grads.dgamma"));
    UQ_TRY(check_ptr(gr.dalpha, "grads.dalpha"));
    UQ_TRY(check_ptr(gr.dzb, "grads.dzb"));
    return cuda_status(uq::launch_omni_bwd(sh, W, p, codes, dL_dWhat, gr, (cudaStream_t)stream), "uq_quantize_bwd_omni");
}

uq_status uq_omni_scales(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, const float* beta,
                         const float* gamma, float* delta, float* zo, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    if (!uq::omni_ok(sh)) return fail(UQ_ERR_UNSUPPORTED, "g=%d: the OmniQuant maps take g in {32, 64, 128, 256, 512}", g);
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(beta, "beta"));
    UQ_TRY(check_ptr(gamma, "gamma"));
    UQ_TRY(check_ptr(delta, "delta"));
    UQ_TRY(check_ptr(zo, "zo"));
    return cuda_status(uq::launch_omni_scales(sh, W, beta, gamma, delta, zo, (cudaStream_t)stream), "uq_omni_scales");
}

uq_status uq_quantize_fwd_awq(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                              uq_params_awq p, uint8_t* codes, uq_map map, int64_t step, int p_period, float* W_hat,
                              void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    if (!uq::awq_ok(sh)) return fail(UQ_ERR_UNSUPPORTED, "g=%d: the AWQ maps take g in {32, 64, 128, 256, 512}", g);
    if (map != UQ_MAP_FULL && map != UQ_MAP_LOCAL_PERIODIC) return fail(UQ_ERR_ARG, "unknown mapping %d", (int)map);
    if (p_period < 1) return fail(UQ_ERR_ARG, "p_period=%d must be >= 1", p_period);
    if (step < 0) return fail(UQ_ERR_ARG, "step=%lld must be >= 0", (long long)step);
    const int mode = map == UQ_MAP_FULL ? uq::FWD_FULL : (step % p_period == 0 ? uq::FWD_REMAP : uq::FWD_KEEP);
    if (mode != uq::FWD_KEEP) UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.sa, "params.sa"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.za, "params.za"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(W_hat, "W_hat"));
    return cuda_status(uq::launch_awq_fwd(sh, W, p, codes, mode, W_hat, (cudaStream_t)stream), "uq_quantize_fwd_awq");
}

int64_t uq_awq_bwd_workspace_bytes(int64_t out, int64_t in, int q, int g) {
    if (q < 1 || q > 4 || out < 1 || in < 1 || g < 32 || in % g != 0 || in > kMaxIn || out > 0x7fffffffLL) return -1;
    const uq::Shape sh{out, (int)in, q, g, UQ_W_BF16};
    if (!uq::awq_ok(sh)) return -1;
    return uq::awq_workspace_floats(sh) * (int64_t)sizeof(float);
}

uq_status uq_quantize_bwd_awq(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                              uq_params_awq p, const uint8_t* codes, const float* dL_dWhat, uq_grads_awq gr,
                              float* workspace, int64_t workspace_bytes, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    if (!uq::awq_ok(sh)) return fail(UQ_ERR_UNSUPPORTED, "g=%d: the AWQ maps take g in {32, 64, 128, 256, 512}", g);
    UQ_TRY(check_ptr(W, "W"));
    UQ_TRY(check_ptr(p.sa, "params.sa"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.za, "params.za"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(dL_dWhat, "dL_dWhat"));
    UQ_TRY(check_ptr(gr.dsa, "grads.dsa"));
    UQ_TRY(check_ptr(gr.ddelta, "grads.ddelta"));
    UQ_TRY(check_ptr(gr.dza, "grads.dza"));
    UQ_TRY(check_ptr(gr.dalpha, "grads.dalpha"));
    UQ_TRY(check_ptr(gr.dzb, "grads.dzb"));
    UQ_TRY(check_ptr(workspace, "workspace"));
    const int64_t need = uq::awq_workspace_floats(sh) * (int64_t)sizeof(float);
    if (workspace_bytes < need)
        return fail(UQ_ERR_ARG, "workspace of %lld bytes; the backward needs %lld (uq_awq_bwd_workspace_bytes)",
                    (long long)workspace_bytes, (long long)need);
    return cuda_status(uq::launch_awq_bwd(sh, W, p, codes, dL_dWhat, gr, workspace, (cudaStream_t)stream),
                       "uq_quantize_bwd_awq");
}

uq_status uq_export_bcq(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g, uq_params p,
                        const uint8_t* codes, uq_export_mode mode, uint32_t* bitplanes, float* alpha_star,
                        float* zb_star, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, wdtype));
    if (mode != UQ_EXPORT_REUSE_CODES && mode != UQ_EXPORT_REMAP_EQ4)
        return fail(UQ_ERR_ARG, "unknown export mode %d", (int)mode);
    if (mode == UQ_EXPORT_REMAP_EQ4) UQ_TRY(check_ptr(W, "W"));
    else UQ_TRY(check_ptr(codes, "codes"));
    UQ_TRY(check_ptr(p.delta, "params.delta"));
    UQ_TRY(check_ptr(p.zu, "params.zu"));
    UQ_TRY(check_ptr(p.alpha, "params.alpha"));
    UQ_TRY(check_ptr(p.zb, "params.zb"));
    UQ_TRY(check_ptr(bitplanes, "bitplanes"));
    UQ_TRY(check_ptr(alpha_star, "alpha_star"));
    UQ_TRY(check_ptr(zb_star, "zb_star"));
    const uq::Shape sh{out, (int)in, q, g, (int)wdtype};
    return cuda_status(uq::launch_export(sh, W, p, codes, (int)mode, bitplanes, alpha_star, zb_star,
                                         (cudaStream_t)stream),
                       "uq_export_bcq");
}

int64_t uq_bcq_gemv_workspace_bytes(int64_t out, int64_t in, int batch) {
    if (out < 1 || in < 32 || in % 32 != 0 || in > kMaxIn || batch < 1 || batch > 64) return -1;
    return uq::gemv_workspace_floats(out, in, batch) * (int64_t)sizeof(float);
}

uq_status uq_bcq_gemv(const uint32_t* bitplanes, const float* alpha_star, const float* zb_star, int64_t out,
                      int64_t in, int q, int g, const void* x, uq_wdtype xdtype, int batch, float* y, float* workspace,
                      int64_t workspace_bytes, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, xdtype));
    UQ_TRY(check_gemv_group(g));
    if (batch < 1 || batch > 64) return fail(UQ_ERR_ARG, "batch=%d must be in 1..64", batch);
    UQ_TRY(check_ptr(bitplanes, "bitplanes"));
    UQ_TRY(check_ptr(alpha_star, "alpha_star"));
    UQ_TRY(check_ptr(zb_star, "zb_star"));
    UQ_TRY(check_ptr(x, "x"));
    UQ_TRY(check_ptr(y, "y"));
    UQ_TRY(check_ptr(workspace, "workspace"));
    const int64_t need = uq_bcq_gemv_workspace_bytes(out, in, batch);
    if (workspace_bytes < need)
        return fail(UQ_ERR_ARG, "workspace of %lld bytes; this product needs %lld (uq_bcq_gemv_workspace_bytes)",
                    (long long)workspace_bytes, (long long)need);
    return cuda_status(uq::launch_gemv(bitplanes, alpha_star, zb_star, out, (int)in, q, g, x, (int)xdtype, batch, y,
                                       workspace, (cudaStream_t)stream),
                       "uq_bcq_gemv");
}

uq_status uq_bcq_gemv_noalloc(const uint32_t* bitplanes, const float* alpha_star, const float* zb_star,
                              int64_t out, int64_t in, int q, int g, const void* x, uq_wdtype xdtype, int batch,
                              float* y, void* stream) {
    UQ_TRY(check_shape(out, in, q, g, xdtype));
    UQ_TRY(check_gemv_group(g));
    if (batch < 1 || batch > 64) return fail(UQ_ERR_ARG, "batch=%d must be in 1..64", batch);
    UQ_TRY(check_ptr(bitplanes, "bitplanes"));
    UQ_TRY(check_ptr(alpha_star, "alpha_star"));
    UQ_TRY(check_ptr(zb_star, "zb_star"));
    UQ_TRY(check_ptr(x, "x"));
    UQ_TRY(check_ptr(y, "y"));
    const int64_t need = uq::gemv_workspace_floats(out, in, batch);
    const int64_t have = uq::gemv_static_workspace_floats();
    if (need > have)
        return fail(UQ_ERR_UNSUPPORTED,
                    "this product needs %lld floats of scratch (ceil(in/512) * batch * out); the built-in scratch "
                    "holds %lld: pass a workspace to uq_bcq_gemv instead",
                    (long long)need, (long long)have);
    float* work = nullptr;
    const cudaError_t e = uq::gemv_static_workspace(&work);
    if (e != cudaSuccess) return cuda_status(e, "uq_bcq_gemv_noalloc: looking up the built-in scratch");
    return cuda_status(uq::launch_gemv(bitplanes, alpha_star, zb_star, out, (int)in, q, g, x, (int)xdtype, batch, y,
                                       work, (cudaStream_t)stream),
                       "uq_bcq_gemv_noalloc");
}

uq_status uq_check_device(void* stream) {
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return fail(UQ_ERR_CUDA, "uq_check_device: %s", cudaGetErrorString(e));
    unsigned int flag = 0, flag_step = 0, flag_omni = 0, flag_awq = 0, flag_gemv = 0;
    e = uq::stream_error(true, &flag);
    if (e == cudaSuccess) e = uq::step_error(true, &flag_step);
    if (e == cudaSuccess) {
        unsigned int flag_step_bf16 = 0;
        e = uq::step_bf16_error(true, &flag_step_bf16);
        flag_step |= flag_step_bf16;
    }
    if (e == cudaSuccess) e = uq::omni_error(true, &flag_omni);
    if (e == cudaSuccess) e = uq::awq_error(true, &flag_awq);
    if (e == cudaSuccess) e = uq::gemv_error(true, &flag_gemv);
    if (e != cudaSuccess) return fail(UQ_ERR_CUDA, "uq_check_device: %s", cudaGetErrorString(e));
    flag |= (flag_step << 4) | (flag_omni << 8) | (flag_awq << 12) | (flag_gemv << 16);
    const unsigned int drain_bits = 0x88888u;   // kDrainTimeoutBit of each kernel family
    if (flag & drain_bits)
        return fail(UQ_ERR_CUDA, "a bounded wait ran out on the device (flag %u): a kernel gave up waiting "
                                 "for its own data copies, and its wait for the copies still in flight ran out "
                                 "too, so a block may have exited with copies landing in its shared memory",
                    flag);
    if (flag) return fail(UQ_ERR_CUDA, "a bounded wait ran out on the device (flag %u): a kernel gave up waiting "
                                       "for its own data copies", flag);
    return ok();
}

uq_status uq_selftest_wait_timeout(void* stream) {
    return cuda_status(uq::launch_wait_selftest((cudaStream_t)stream), "uq_selftest_wait_timeout");
}

}  // extern "C"
