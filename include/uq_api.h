/*
 * uq_api.h -- C ABI of the GB300 (sm_103a) UniQuan_F weight quantizer.
 *
 * UniQuan_F (arXiv 2506.03781) quantizes each group of g weights of a
 * weight matrix W [out, in] with
 *     w^ = Q*_IF(w) = D_R( M*_B( T_F(w; Delta, z_U, s, s_r); alpha, z_B ); Delta, z_U )   (Eq. 3)
 *   T_F  (Eq. 1)       x   = w / (Delta * s * s_r) + z_U
 *   M_B  (Sec. 2.3)    code of the nearest of the 2^q BCQ levels  l(c) = c . alpha + z_B
 *   M*_B (Algorithm 4) every p steps, nearest among the current level and its two
 *                      neighbours in the sorted level list; codes kept in between
 *   D_R  (Sec. 3.1)    w^  = Delta * (l(c) - z_U)
 * and trains Delta, z_U, s, s_r, alpha, z_B by SGD through a straight-through
 * estimator with gradient filtering (App. C.1).  After training, Theorem 1
 * folds D_R into the BCQ parameters (alpha* = Delta alpha,
 * z_B* = Delta (z_B - z_U)) and the binary codes are exported as bit-planes
 * (the last two steps of Algorithm 1; Eq. 4).
 *
 * Conventions common to every entry point
 * ---------------------------------------
 * Memory.  Every pointer argument is DEVICE memory owned by the caller
 *   (except the return value of uq_last_error).  The library never allocates,
 *   frees or keeps a pointer after a call returns.
 * Device.  Work is launched on the calling thread's current CUDA device;
 *   every pointer and the stream must belong to that device.
 * Asynchrony.  Work is enqueued on `stream` (a cudaStream_t; NULL = the
 *   legacy default stream) and the call returns without synchronising.
 *   UQ_OK means "validated and launched"; execution errors surface on the
 *   stream as usual.
 * Layouts (row-major, contiguous, no padding):
 *   W       [out, in]      fp32 (UQ_W_F32) or bf16 (UQ_W_BF16), read only
 *   s       [out, in]      fp32   per-element FlexRound scale
 *   s_r     [out]          fp32   per-row scale
 *   Delta, z_U, z_B [out, in/g] fp32   per-group parameters
 *   alpha   [out, in/g, q] fp32   alpha_1 first
 *   codes   [out, in]      uint8  code word: bit (j-1) set <=> c_j = +1; bits
 *                                 at or above q are ignored on input and
 *                                 written as zero
 *   W_hat, dL/dW_hat, ds [out, in] fp32
 *   bit-planes [q, out, in/32] uint32: bit b of planes[j][r][t] is c_{j+1}
 *                                 of column 32 t + b (1 <=> +1)
 * Shapes.  1 <= q <= 4; g in {32, 64} or g a multiple of 128; in a multiple
 *   of g; 1 <= out <= 2^31 - 1; in <= 2^24.
 * Alignment.  Every pointer must be 16-byte aligned.
 * Errors.  Arguments are checked before anything is launched; on error the
 *   call returns a non-zero uq_status, launches nothing, writes nothing, and
 *   uq_last_error() describes the problem.  UQ_ERR_CUDA reports a failed
 *   launch (cudaGetLastError after the launch).  No entry point aborts,
 *   exits or traps the device.
 * Determinism.  No output is accumulated with atomics (the only atomic is
 *   the OR into the library's timeout flag); a call repeated on the same
 *   inputs gives bitwise-identical outputs.
 * Numerics.  Every value that decides an integer (x, the levels, the
 *   distances, the filter test) is computed in IEEE fp32 with the operation
 *   order written at each entry point, no FMA contraction; gradients are
 *   accumulated in fp32.
 */
#ifndef UQ_API_H
#define UQ_API_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    UQ_OK = 0,
    UQ_ERR_ARG = 1,          /* null pointer, bad shape, bad enum value      */
    UQ_ERR_UNSUPPORTED = 2,  /* valid per the method but not built (q, g)    */
    UQ_ERR_ALIGN = 3,        /* a pointer is not 16-byte aligned             */
    UQ_ERR_CUDA = 4          /* the CUDA runtime reported an error           */
} uq_status;

typedef enum { UQ_W_F32 = 0, UQ_W_BF16 = 1 } uq_wdtype;

/* Clipping strategies of the unified initialization (App. E.2). */
typedef enum { UQ_CLIP_FIXED_MIN = 0, UQ_CLIP_FIXED_MAX = 1, UQ_CLIP_BALANCED = 2 } uq_clip;

/* Mapping: full nearest level every call (Eq. 2, "UniQuan_F-0"), or the
 * local and periodic mapping M*_B of Algorithm 4 (Eq. 3). */
typedef enum { UQ_MAP_FULL = 0, UQ_MAP_LOCAL_PERIODIC = 1 } uq_map;

/* Export: reuse the codes of the last quantizer call (for which Theorem 1
 * makes R_B(C; Theta_B*) equal the quantizer output), or recompute them
 * from the original weights by Eq. 4. */
typedef enum { UQ_EXPORT_REUSE_CODES = 0, UQ_EXPORT_REMAP_EQ4 = 1 } uq_export_mode;

/* Gradient filter (App. C.1): cut only the straight-through path of a
 * filtered element (the library's reading, used by uq_quantize_bwd), or drop
 * the filtered element from every gradient (the alternative reading). */
typedef enum { UQ_FILTER_STE = 0, UQ_FILTER_ELEMENT = 1 } uq_filter;

/* The learnable parameters Theta_IF = Theta_F u Theta_B (Eq. 1, Sec. 2.3). */
typedef struct {
    float* delta;   /* [out, in/g]    Delta                                */
    float* zu;      /* [out, in/g]    z_U                                  */
    float* s;       /* [out, in]      s   (element-wise scale)             */
    float* sr;      /* [out]          s_r (row-wise scale)                 */
    float* alpha;   /* [out, in/g, q] alpha                                */
    float* zb;      /* [out, in/g]    z_B                                  */
} uq_params;

/* Gradients of the loss w.r.t. each parameter, same shapes as uq_params. */
typedef struct {
    float* ddelta;
    float* dzu;
    float* ds;
    float* dsr;
    float* dalpha;
    float* dzb;
} uq_grads;

/* UniQuan with OmniQuant's transformation (App. E, extensibility): per
 * group the learnable clipping factors beta, gamma of T_O / D_O, and the
 * BCQ parameters alpha, z_B.  All [out, in/g] (alpha [out, in/g, q]). */
typedef struct {
    float* beta;
    float* gamma;
    float* alpha;
    float* zb;
} uq_params_omni;

typedef struct {
    float* dbeta;
    float* dgamma;
    float* dalpha;
    float* dzb;
} uq_grads_omni;

/* UniQuan with AWQ's transformation (App. E, extensibility): sa [in] one
 * scale per column (shared by every row), delta and za [out, in/g] per
 * group, and the BCQ parameters alpha [out, in/g, q], zb [out, in/g]. */
typedef struct {
    float* sa;
    float* delta;
    float* za;
    float* alpha;
    float* zb;
} uq_params_awq;

typedef struct {
    float* dsa;
    float* ddelta;
    float* dza;
    float* dalpha;
    float* dzb;
} uq_grads_awq;

/*
 * uq_init_params -- unified initialization (Algorithm 2 with the general
 * alternating update of Algorithm 3 and the clipping strategies of App. E.2).
 *
 * For every group: w_m, w_M = min, max of the group; z_B starts at
 * (2^q - 1)/2, s = 1, s_r = 1.  For gamma_i = float(i)/float(G), i = 1..G:
 *   Delta' = (gamma (w_M - w_m)) / (2^q - 1)   (w_M - w_m floored at 1e-12)
 *   z'_U   = -w_m/Delta' | (2^q-1) - w_M/Delta' | -(gamma w_m)/Delta'   (clip)
 *   x      = T_F(w) with s = s_r = 1
 *   greedy start: r = x - z_B; for j: c_j = sign(r) (0 -> +1),
 *                 alpha_j = mean |r| (fp64 sum), r -= c_j alpha_j
 *   T rounds of: alpha <- (C^T C)^{-1} C^T (x - z_B)  (fp64; unchanged when
 *                C^T C is singular), C <- nearest level, and if G == 1
 *                z_B <- mean(x - C alpha) (fp64)
 *   e' = sum (w - w^)^2 in fp64 with the full mapping; kept if e' < e.
 * Writes delta, zu, alpha, zb for every group, s = 1 for every element,
 * sr = 1 for every row, and the codes of the full mapping under the kept
 * parameters.  G >= 1, T >= 0, g <= 32768.  Not on the per-step path.
 * W is read only; every params pointer and `codes` is written.
 */
uq_status uq_init_params(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                         int G, int T, uq_clip clip, uq_params params, uint8_t* codes, void* stream);

/*
 * uq_quantize_fwd -- the quantizer Q*_IF (Eq. 3) or Q_IF (Eq. 2).
 *
 * map == UQ_MAP_FULL: every element is mapped to the nearest of all 2^q
 *   levels: codes is written (not read), W_hat is written.
 * map == UQ_MAP_LOCAL_PERIODIC and step % p_period == 0 (a remap step,
 *   Algorithm 4): for each element with current rank d in the ascending
 *   level order of its group, the nearest of ranks d, max(d-1,0),
 *   min(d+1,2^q-1) (examined in that order, replaced only when strictly
 *   nearer) is taken; codes is read and rewritten, W_hat written.
 * map == UQ_MAP_LOCAL_PERIODIC and step % p_period != 0: codes is kept (not
 *   written) and W_hat = D_R(l(code)) with the current alpha, z_B; W, s and
 *   s_r are not read (they may be NULL).
 * Arithmetic (fp32): den = (Delta * s) * s_r; x = w / den + z_U;
 *   l(c) = ((c_1 a_1 + c_2 a_2) + ... + c_q a_q) + z_B; levels sorted
 *   ascending, equal values by ascending code word; full mapping ties go to
 *   the lower rank; W_hat = Delta * (l(c) - z_U).
 * params.delta/zu/alpha/zb are read; s, sr read on remap/full calls.
 * step >= 0, p_period >= 1.
 */
uq_status uq_quantize_fwd(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                          uq_params params, uint8_t* codes, uq_map map, int64_t step, int p_period,
                          float* W_hat, void* stream);

/*
 * uq_quantize_bwd -- gradients through Eq. 3 with the straight-through
 * estimator and gradient filtering of App. C.1, given G = dL/dW_hat.
 *
 * The codes are those of the forward call this backward belongs to.  With
 * u = w / ((Delta s) s_r), x = u + z_U, m = l(code), tau = min_j |alpha_j|
 * and f = (|x - m| <= tau) (fp32 decision):
 *   ds_i     = -G_i Delta f_i u_i / s_i
 *   dDelta   = sum_{i in group} G_i ((m_i - z_U) - f_i u_i)
 *   dz_U     = sum G_i Delta (f_i - 1)
 *   dz_B     = sum G_i Delta
 *   dalpha_j = sum G_i Delta c_ij
 *   ds_r     = -sum_{i in row} G_i Delta f_i u_i / s_r
 * Every grads pointer is written (overwritten, not accumulated).  Group
 * sums are reduced inside each group's warp(s) and row sums inside the
 * row's thread block: no atomics.
 */
uq_status uq_quantize_bwd(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                          uq_params params, const uint8_t* codes, const float* dL_dWhat,
                          uq_grads grads, void* stream);

/*
 * uq_quantize_bwd_ex -- uq_quantize_bwd with a choice of gradient filter:
 * UQ_FILTER_STE is exactly uq_quantize_bwd; with UQ_FILTER_ELEMENT every
 * term of an element with |x - l(c)| > tau is dropped (G_i replaced by
 * f_i G_i in every sum, so dz_U is zero).  Same arguments, layouts and
 * numerics otherwise; an unknown filter is UQ_ERR_ARG.
 */
uq_status uq_quantize_bwd_ex(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                             uq_params params, const uint8_t* codes, const float* dL_dWhat, uq_grads grads,
                             uq_filter filter, void* stream);

/*
 * uq_train_step -- one optimisation step of Algorithm 1's inner loop, fused
 * into one kernel: the backward of step `step` (exactly the gradients
 * uq_quantize_bwd defines, not written out), the SGD update of every
 * parameter in place (FlexRound trains Theta_F by SGD, Sec. 3.1; one
 * learning rate for Theta_F = {Delta, z_U, s, s_r} and one for
 * Theta_B = {alpha, z_B}, hyperparameter table of App. C.1: 0.005 and
 * 0.0005), then the forward of step + 1 (as uq_quantize_fwd with step + 1)
 * with the updated parameters.
 *
 * codes: in, the codes the forward of `step` produced; out, the codes of
 *   step + 1 (under UQ_MAP_LOCAL_PERIODIC rewritten only when
 *   (step + 1) % p_period == 0).
 * dL_dWhat: [out, in] fp32, the gradient of that forward's W_hat.
 * params: read, then overwritten with theta - lr * grad, evaluated in fp32
 *   as fl(theta - fl(lr * grad)); each gradient is formed as in
 *   uq_quantize_bwd (ds_r from the row's partial sums in a fixed order).
 * W_hat: [out, in] fp32, written with W^ of step + 1.
 * Shapes: g in {32, 64, 128}, in a multiple of 512 (256 for g = 32) and at
 *   most 32768 (16384 for g = 32); other shapes return UQ_ERR_UNSUPPORTED
 *   (the separate entry points cover them).  step in [0, 2^63 - 1),
 *   p_period >= 1.  Outputs must not overlap the inputs other than the
 *   in/out codes and params.  Deterministic: the same inputs give the same
 *   bits.  The paper has no fused kernel; the step itself is its own.
 */
uq_status uq_train_step(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                        uq_params params, uint8_t* codes, const float* dL_dWhat, float lr_F, float lr_B,
                        uq_map map, int64_t step, int p_period, float* W_hat, void* stream);

/*
 * uq_train_step_bf16 -- uq_train_step for a block computed in bf16 (the
 * reconstruction loop of Algorithm 1 back-propagates through the block in
 * its compute type): the same step, parameters and codes bit for bit as
 * uq_train_step given the same dL_dWhat values, except that
 *   dL_dWhat: [out, in] bf16 bits (uint16), read exactly (each value is the
 *     fp32 number those bits denote);
 *   W_hat: [out, in] bf16 bits (uint16), written with W^ of step + 1 as
 *     computed in fp32 by uq_train_step, rounded to the nearest bf16 (ties
 *     to even).
 * So the caller's block consumes W^ and produces dL/dW^ in its own type
 * without a conversion pass over the weights.  Arguments, shapes and errors
 * otherwise as uq_train_step.
 */
uq_status uq_train_step_bf16(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                             uq_params params, uint8_t* codes, const uint16_t* dL_dWhat, float lr_F, float lr_B,
                             uq_map map, int64_t step, int p_period, uint16_t* W_hat, void* stream);

/*
 * uq_quantize_fwd_omni -- the UniQuan quantizer with OmniQuant's maps
 * (App. E, extensibility) in place of FlexRound's:
 *   T_O(w) = w / Delta_O + z_O,  D_O(w~) = Delta_O (w~ - z_O),
 *   Delta_O = (gamma w_M - beta w_m) / (2^q - 1),  z_O = -round(beta w_m / Delta_O)
 * with w_m, w_M the smallest and largest weight of the group.  fp32 order:
 * num = gamma * w_M - beta * w_m (each product rounded), Delta_O = num /
 * (2^q - 1), z_O = -rint((beta * w_m) / Delta_O) (half to even),
 * x = w / Delta_O + z_O, W_hat = Delta_O * (l(c) - z_O).  The mapping, the
 * level order and every tie rule are those of uq_quantize_fwd (map, step,
 * p_period likewise; W is read on every call, also on keep steps).
 * g in {32, 64, 128, 256, 512}, else UQ_ERR_UNSUPPORTED.  Delta_O must come
 * out positive (gamma w_M > beta w_m); the caller keeps it so.
 */
uq_status uq_quantize_fwd_omni(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                               uq_params_omni params, uint8_t* codes, uq_map map, int64_t step, int p_period,
                               float* W_hat, void* stream);

/*
 * uq_quantize_bwd_omni -- gradients through uq_quantize_fwd_omni with the
 * straight-through estimator and the gradient filter of App. C.1
 * (tau = min_j |alpha_j|, f = |x - l(c)| <= tau), and the rounding in z_O
 * passed straight through.  With u = w / Delta_O and per group
 *   A = sum G ((l(c) - z_O) - f u),  B = -Delta_O sum G (1 - f):
 *   dbeta  = A (-w_m / (2^q-1)) + B dz/dbeta,
 *   dgamma = A ( w_M / (2^q-1)) + B dz/dgamma,
 *   dz/dbeta = -(w_m / Delta_O - beta w_m (dDelta/dbeta) / Delta_O^2),
 *   dz/dgamma = beta w_m (dDelta/dgamma) / Delta_O^2,
 *   dalpha_j = Delta_O sum G c_j,  dz_B = Delta_O sum G.
 * Every grads pointer is written (overwritten).  Group sums are reduced
 * inside the group's lanes; fp32; deterministic.  Shapes as the forward.
 */
uq_status uq_quantize_bwd_omni(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                               uq_params_omni params, const uint8_t* codes, const float* dL_dWhat,
                               uq_grads_omni grads, void* stream);

/*
 * uq_omni_scales -- Delta_O and z_O of every group (the fp32 values the
 * forward uses), written to delta [out, in/g] and zo [out, in/g].  With them
 * the export of the OmniQuant-unified quantizer is uq_export_bcq with
 * params.delta = delta and params.zu = zo (D_O has D_R's form, so Theorem 1
 * gives alpha* = Delta_O alpha, z_B* = Delta_O (z_B - z_O)).
 */
uq_status uq_omni_scales(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                         const float* beta, const float* gamma, float* delta, float* zo, void* stream);

/*
 * uq_quantize_fwd_awq -- the UniQuan quantizer with AWQ's maps (App. E,
 * extensibility): T_A(w) = (w s_A) / Delta_A + z_A and
 * D_A(w~) = Delta_A (w~ - z_A) / s_A (the printed D_A subtracts z_O; read
 * as z_A).  fp32 order: x = ((w * s_A) / Delta_A) + z_A,
 * W_hat = (Delta_A * (l(c) - z_A)) / s_A.  Mapping, level order and tie
 * rules as uq_quantize_fwd (map, step, p_period likewise; W is not read on
 * keep steps).  g in {32, 64, 128, 256, 512}, else UQ_ERR_UNSUPPORTED.
 * The export is uq_export_bcq with params.delta = delta, params.zu = za
 * (alpha* = Delta_A alpha, z_B* = Delta_A (z_B - z_A)); the column scale
 * 1 / s_A stays outside the BCQ weights (applied to the activations).
 */
uq_status uq_quantize_fwd_awq(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                              uq_params_awq params, uint8_t* codes, uq_map map, int64_t step, int p_period,
                              float* W_hat, void* stream);

/*
 * uq_quantize_bwd_awq -- gradients through uq_quantize_fwd_awq with the
 * straight-through estimator and the gradient filter of App. C.1.  With
 * u = w s / Delta and f = |x - l(c)| <= min_j |alpha_j|:
 *   dDelta = sum G ((l(c) - z) - f u) / s,   dz_A = -Delta sum G (1 - f) / s,
 *   ds_A[col] = sum over the rows of G (f w - Delta (l(c) - z) / s) / s,
 *   dalpha_j = Delta sum G c_j / s,          dz_B = Delta sum G / s.
 * ds_A sums over every row of its column: per-row-range partials go to
 * `workspace` (caller-owned device memory of at least
 * uq_awq_bwd_workspace_bytes(out, in, q, g) bytes, overwritten) and are
 * summed in a fixed order (eight contiguous slices of the ranges, each in
 * range order, then the slices in order).  fp32, deterministic.  A too
 * small workspace is
 * UQ_ERR_ARG.
 */
uq_status uq_quantize_bwd_awq(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                              uq_params_awq params, const uint8_t* codes, const float* dL_dWhat,
                              uq_grads_awq grads, float* workspace, int64_t workspace_bytes, void* stream);

/* Bytes of workspace uq_quantize_bwd_awq needs (or -1 for an invalid shape).
 * It depends on the current device's SM count; query it on that device. */
int64_t uq_awq_bwd_workspace_bytes(int64_t out, int64_t in, int q, int g);

/*
 * uq_export_bcq -- Theorem 1 and the final binary codes (the last two
 * steps of Algorithm 1).
 *
 * alpha_star[r, k, j] = Delta * alpha_j and zb_star[r, k] = Delta * (z_B - z_U)
 * (fp32, z_B - z_U first).  The code matrix is the stored codes
 * (UQ_EXPORT_REUSE_CODES; W may be NULL) or, for UQ_EXPORT_REMAP_EQ4, the
 * nearest level of Theta_B* to each original weight w (Eq. 4, same sorting
 * and tie rule as the full mapping; codes may be NULL).  Writes
 * bitplanes [q, out, in/32], alpha_star [out, in/g, q], zb_star [out, in/g].
 * params.s and params.sr are not used (may be NULL).
 */
uq_status uq_export_bcq(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                        uq_params params, const uint8_t* codes, uq_export_mode mode,
                        uint32_t* bitplanes, float* alpha_star, float* zb_star, void* stream);

/*
 * uq_export_bcq_half -- uq_export_bcq with alpha* and z_B* stored as 16-bit
 * reals (the storage App. F.1 counts: g k + 16 (k + 1) bits per group): the
 * fp32 values uq_export_bcq computes, rounded to IEEE half precision (nearest
 * even; overflow to infinity), written as raw half bits to alpha_star
 * [out, in/g, q] and zb_star [out, in/g] (uint16).  Bit-planes as
 * uq_export_bcq.
 */
uq_status uq_export_bcq_half(const void* W, uq_wdtype wdtype, int64_t out, int64_t in, int q, int g,
                             uq_params params, const uint8_t* codes, uq_export_mode mode, uint32_t* bitplanes,
                             uint16_t* alpha_star, uint16_t* zb_star, void* stream);

/*
 * uq_bcq_gemv -- the BCQ matrix-vector product of deployment, computed from
 * the exported format alone: y[b, r] = sum_i W~[r, i] x[b, i] with
 * W~[r, i] = sum_j alpha_star[r, k, j] c_j + zb_star[r, k], k = i / g, and
 * c_j = +1 where bit (i % 32) of bitplanes[j, r, i / 32] is set, else -1
 * (R_B(C; Theta_B*) of Sec. 2.3; by Theorem 1 this is the quantizer's W^,
 * so no Delta or z_U is needed at inference; bit-plane storage of App. F.1).
 *
 * bitplanes [q, out, in/32] uint32, alpha_star [out, in/g, q] and
 * zb_star [out, in/g] fp32 as uq_export_bcq writes them; x [batch, in]
 * (xdtype fp32 or bf16), y [batch, out] fp32, both row-major.  The columns
 * are split into tiles: 1024 columns (32 per lane) when in is a multiple of
 * 1024 and g <= 256, else 512.  Each tile's contribution is formed from
 * per-8-column partial sums of x (one table lookup per plane byte) and
 * written to `workspace` (caller-owned device memory of at least
 * uq_bcq_gemv_workspace_bytes(out, in, batch) bytes, overwritten), then the
 * tiles are summed in order into y.  fp32 throughout, fixed order for a
 * given shape: deterministic, and within a small multiple of the fp32 unit
 * roundoff of sum_i (sum_j |alpha*_j| + |z*|) |x_i| of the exact product
 * (the two tilings add in different orders, both within that bound).
 * Shapes as uq_quantize_fwd, except that g must divide 512 or be a multiple
 * of 512 (32, 64, 128, 256, 512, 1024, ...; any other g, e.g. 384 or 640, is
 * UQ_ERR_UNSUPPORTED); 1 <= batch <= 64 (each token re-reads the planes).
 * The 1024-column tiles, and the 512-column ones when in is a multiple of
 * 512 and g <= 128, are staged with TMA tensor maps that the call encodes on
 * the host (through the runtime's driver entry point; stack memory only,
 * nothing is allocated); any other shape, or a driver without the encoder,
 * takes per-thread asynchronous copies (same arithmetic as the 512-column
 * tensor-map path).  The 1024-column product is launched as a programmatic
 * dependent of the preceding work on the stream: it is scheduled early but
 * reads and writes nothing before that work has completed, so stream order
 * is kept.
 * Reads every input, writes y and the workspace.  A too small workspace is
 * UQ_ERR_ARG.
 */
uq_status uq_bcq_gemv(const uint32_t* bitplanes, const float* alpha_star, const float* zb_star, int64_t out,
                      int64_t in, int q, int g, const void* x, uq_wdtype xdtype, int batch, float* y,
                      float* workspace, int64_t workspace_bytes, void* stream);

/* Bytes of workspace uq_bcq_gemv needs for this shape (ceil(in/512) * batch
 * * out floats), or -1 if the shape or batch is invalid.  Host only. */
int64_t uq_bcq_gemv_workspace_bytes(int64_t out, int64_t in, int batch);

/*
 * uq_bcq_gemv_noalloc -- the same product as uq_bcq_gemv (same arguments
 * minus the workspace, same results bit for bit), for callers that cannot
 * allocate device memory: code that runs where every byte of the GPU is
 * owned by someone else's allocator, or where an allocation call is not
 * allowed at all (it may block the whole device, or the host runtime simply
 * gives the caller no way to reach it).  The paper has no counterpart; this
 * is a convenience of the library.
 *
 * Instead of a workspace it uses scratch built into the library: 4 MiB
 * (1,048,576 floats) in a static device array, which every GPU that loads
 * the library holds until the process exits.  A shape whose partials need
 * more (ceil(in/512) * batch * out floats, e.g. more than 2 tokens of an
 * 8192 x 28672 matrix) is rejected with UQ_ERR_UNSUPPORTED before anything
 * is launched.  Nothing is allocated and nothing is freed: no cudaMalloc,
 * no cudaFree, no library routine that allocates.
 *
 * The first call on a device looks up the scratch's device address (once,
 * with that device current) and caches it with the identifier of the
 * device's context; make that first call before any stream capture.  After
 * cudaDeviceReset the device gets a new context and the array a possibly
 * different address, so the first call in the new context looks it up again
 * (and must also come before any capture).  All calls share the one scratch array and it keeps the
 * last call's contents: each call overwrites every word it reads before
 * reading it, so nothing needs clearing, but two calls whose work overlaps
 * on the GPU (for instance on two streams) race on it and may give wrong
 * results.  Order such calls on one stream.
 */
uq_status uq_bcq_gemv_noalloc(const uint32_t* bitplanes, const float* alpha_star, const float* zb_star,
                              int64_t out, int64_t in, int q, int g, const void* x, uq_wdtype xdtype, int batch,
                              float* y, void* stream);

/*
 * uq_check_device -- waits for `stream` to finish, then reports whether a
 * pipelined kernel of this library gave up waiting for its own data copies
 * since the last check (every wait on an mbarrier is bounded to about one
 * second of GPU clock; when one runs out the warp stops computing and a
 * device-side indicator is set instead of hanging).  Clears the indicator.
 * UQ_OK if none ran out; UQ_ERR_CUDA if one did or the synchronisation
 * failed.  Needs no arguments beyond the stream; allocates nothing.
 */
uq_status uq_check_device(void* stream);

/*
 * uq_selftest_wait_timeout -- exercises the bounded-wait path without any
 * fault: launches one warp that waits on a shared-memory mbarrier nothing
 * arrives at; after about 2^24 GPU clock cycles (~8 ms) the wait gives up,
 * sets the same device indicator as a pipelined kernel would, and the warp
 * returns.  The next uq_check_device() then returns UQ_ERR_CUDA (and clears
 * the indicator); the context stays usable.  For tests of the failure path.
 * The paper has no counterpart.
 */
uq_status uq_selftest_wait_timeout(void* stream);

/* Message for the last non-OK status returned on the calling thread (never
 * NULL; "" if none).  Owned by the library, valid until the next call on
 * the same thread. */
const char* uq_last_error(void);

/* Version of this ABI (incremented on any incompatible change). */
int uq_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* UQ_API_H */
