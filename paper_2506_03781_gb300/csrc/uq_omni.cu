// UniQuan with OmniQuant's transformation (App. E, extensibility): the
// same BCQ mapping, levels and gradient filter as UniQuan_F, with
//   T_O(w) = w / Delta_O + z_O,   D_O(w~) = Delta_O (w~ - z_O),
//   Delta_O = (gamma w_M - beta w_m) / (2^q - 1),  z_O = -round(beta w_m / Delta_O)
// per group, beta and gamma learnable, w_m / w_M the group's smallest and
// largest weight (round half to even; the rounding is passed straight through
// in the backward, as OmniQuant trains its zero point).
//
// Work decomposition as in the general-path kernels (uq_common.cuh): thread
// blocks of 8 warps own R whole rows, a warp's unit is NG whole groups with
// LPG lanes per group; here every lane holds all of its group elements in
// registers at once (NV <= 4 vectors of 4, g <= 512), so the group's min and
// max are a lane-local reduction plus log2(LPG) shuffles, and every lane of
// the group forms Delta_O and z_O itself.  No element-wise scale: HBM traffic
// per element (bf16 W) is 2 + 1 read, 4 + 1 written for a remap step and
// 2 + 1 + 4 read for the backward.
//
// Shapes the pipelined UniQuan_F kernels take (g in {32, 64, 128}, rows of
// whole work units) run on the same persistent TMA-pipelined skeleton
// (uq_pipe.cuh): every warp streams its (row block, unit) items through a
// ring of shared-memory stages -- the weights, the code words (and dL/dW^ for
// the backward), and the unit's beta, gamma, z_B, alpha -- with bounded
// mbarrier waits (a wait that runs out sets g_omni_err, reported by
// uq_check_device).  Other shapes use the kernels above, which load straight
// into registers.
#include "uq_common.cuh"
#include "uq_launch.h"
#include "uq_pipe.cuh"

namespace uq {

#ifndef UQ_OMNI_MIN_BLOCKS
#define UQ_OMNI_MIN_BLOCKS 3
#endif

// Delta_O and z_O of a group from the lanes' weights (all LPG lanes of the
// group call it together; lanes of absent groups pass +inf / -inf).
template <int Q, int LPG>
__device__ __forceinline__ void omni_scales(float lmin, float lmax, float beta, float gamma, float& wm, float& wM,
                                            float& delta, float& zo) {
#pragma unroll
    for (int off = LPG / 2; off >= 1; off >>= 1) {
        lmin = fminf(lmin, __shfl_xor_sync(kFull, lmin, off));
        lmax = fmaxf(lmax, __shfl_xor_sync(kFull, lmax, off));
    }
    wm = lmin;
    wM = lmax;
    const float num = __fsub_rn(__fmul_rn(gamma, wM), __fmul_rn(beta, wm));
    delta = __fdiv_rn(num, (float)((1 << Q) - 1));
    zo = -rintf(__fdiv_rn(__fmul_rn(beta, wm), delta));
}

template <int Q, typename WT, int LPG, int MODE>
__global__ void __launch_bounds__(kThreads, UQ_OMNI_MIN_BLOCKS)
omni_fwd_kernel(const void* __restrict__ W, const float* __restrict__ BETA, const float* __restrict__ GAMMA,
                const float* __restrict__ ALPHA, const float* __restrict__ ZB, uint8_t* __restrict__ CODES,
                float* __restrict__ WHAT, float* __restrict__ DOUT, float* __restrict__ ZOUT, int64_t out, int n_in,
                int g, int R) {
    constexpr int L = 1 << Q;
    constexpr int NG = 32 / LPG;
    __shared__ MapTab<Q, NG> tabs[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    MapTab<Q, NG>& t = tabs[warp];
    const int WPR = kWarps / R;
    const int64_t row = (int64_t)blockIdx.x * R + warp / WPR;
    if (row >= out) return;                       // no block barrier in this kernel
    const int wr = warp % WPR;
    const int Gr = n_in / g;
    const int units = (Gr + NG - 1) / NG;
    const int nv = g / (4 * LPG);                 // 1..4
    const int sub = lane / LPG, li = lane % LPG;
    const int64_t rbase = row * (int64_t)n_in;

    for (int u = wr; u < units; u += WPR) {
        const int gi = u * NG + sub;
        const bool ok = gi < Gr;
        const int64_t grp = row * Gr + gi;
        const int64_t ebase = rbase + (int64_t)gi * g + 4 * li;
        float w[4][4];
        uint32_t cv[4] = {0u, 0u, 0u, 0u};
        float lmin = INFINITY, lmax = -INFINITY;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            if (ok && v < nv) {
                const int64_t e = ebase + 4 * LPG * v;
                WT::unpack(WT::load(W, e), w[v]);
                if (MODE != FWD_FULL && WHAT != nullptr) cv[v] = *reinterpret_cast<const uint32_t*>(CODES + e);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    lmin = fminf(lmin, w[v][k]);
                    lmax = fmaxf(lmax, w[v][k]);
                }
            }
        }
        float wm, wM, dl, zo;
        omni_scales<Q, LPG>(lmin, lmax, ok ? __ldg(BETA + grp) : 1.f, ok ? __ldg(GAMMA + grp) : 1.f, wm, wM, dl, zo);
        if (WHAT == nullptr) {                    // scales only (uq_omni_scales)
            if (ok && li == 0) {
                DOUT[grp] = dl;
                ZOUT[grp] = zo;
            }
            continue;
        }
        __syncwarp();
        unit_levels<Q, NG>(t, (float*)nullptr, lane, ALPHA, ZB, row * Gr + u * NG, min(NG, Gr - u * NG));
        if (MODE == FWD_REMAP) unit_sort<Q, NG, true>(t, lane);
        else if (MODE == FWD_FULL) unit_sort<Q, NG, false>(t, lane);
        float srt[L];
        if (MODE == FWD_FULL) {
#pragma unroll
            for (int r = 0; r < L; ++r) srt[r] = t.srt[sub][r];
        }
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            if (!(ok && v < nv)) continue;
            const int64_t e = ebase + 4 * LPG * v;
            float o[4];
            uint32_t nc = 0;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float x = __fadd_rn(__fdiv_rn(w[v][k], dl), zo);
                float m;
                uint32_t code;
                if (MODE == FWD_KEEP) {
                    code = (cv[v] >> (8 * k)) & (L - 1);
                    m = t.lv[sub][code];
                } else if (MODE == FWD_REMAP) {
                    const int c = (cv[v] >> (8 * k)) & (L - 1);
                    const float4 nb = t.nb[sub][c];
                    const uint32_t packed = __float_as_uint(nb.w);
                    float best = fabsf(__fsub_rn(x, nb.y));
                    m = nb.y;
                    code = c;
                    const float dlo = fabsf(__fsub_rn(x, nb.x));
                    if (dlo < best) { best = dlo; m = nb.x; code = packed & 0xffu; }
                    const float dhi = fabsf(__fsub_rn(x, nb.z));
                    if (dhi < best) { m = nb.z; code = (packed >> 8) & 0xffu; }
                } else {
                    const int r = nearest_rank<L>(x, srt, m);
                    code = t.cor[sub][r];
                }
                o[k] = __fmul_rn(dl, __fsub_rn(m, zo));
                nc |= code << (8 * k);
            }
            if (MODE != FWD_KEEP) *reinterpret_cast<uint32_t*>(CODES + e) = nc;
            *reinterpret_cast<float4*>(WHAT + e) = make_float4(o[0], o[1], o[2], o[3]);
        }
    }
}

template <int Q, typename WT, int LPG>
__global__ void __launch_bounds__(kThreads, UQ_OMNI_MIN_BLOCKS)
omni_bwd_kernel(const void* __restrict__ W, const float* __restrict__ BETA, const float* __restrict__ GAMMA,
                const float* __restrict__ ALPHA, const float* __restrict__ ZB, const uint8_t* __restrict__ CODES,
                const float* __restrict__ GUP, float* __restrict__ DBETA, float* __restrict__ DGAMMA,
                float* __restrict__ DALPHA, float* __restrict__ DZB, int64_t out, int n_in, int g, int R) {
    constexpr int L = 1 << Q;
    constexpr int NG = 32 / LPG;
    using SR8 = SegReduce<LPG>;
    __shared__ LvTab<Q, NG> tabs[kWarps];
    __shared__ float tau_s[kWarps][NG];
    __shared__ float sums[kWarps][NG][8];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    LvTab<Q, NG>& t = tabs[warp];
    const int WPR = kWarps / R;
    const int64_t row = (int64_t)blockIdx.x * R + warp / WPR;
    if (row >= out) return;                       // no block barrier in this kernel
    const int wr = warp % WPR;
    const int Gr = n_in / g;
    const int units = (Gr + NG - 1) / NG;
    const int nv = g / (4 * LPG);
    const int sub = lane / LPG, li = lane % LPG;
    const int64_t rbase = row * (int64_t)n_in;

    for (int u = wr; u < units; u += WPR) {
        const int gi = u * NG + sub;
        const bool ok = gi < Gr;
        const int64_t grp = row * Gr + gi;
        const int64_t ebase = rbase + (int64_t)gi * g + 4 * li;
        float w[4][4], G[4][4];
        uint32_t cv[4] = {0u, 0u, 0u, 0u};
        float lmin = INFINITY, lmax = -INFINITY;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            if (ok && v < nv) {
                const int64_t e = ebase + 4 * LPG * v;
                WT::unpack(WT::load(W, e), w[v]);
                f4_to(ldg4(GUP + e), G[v]);
                cv[v] = __ldg(reinterpret_cast<const unsigned int*>(CODES + e));
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    lmin = fminf(lmin, w[v][k]);
                    lmax = fmaxf(lmax, w[v][k]);
                }
            }
        }
        const float beta = ok ? __ldg(BETA + grp) : 1.f, gamma = ok ? __ldg(GAMMA + grp) : 1.f;
        float wm, wM, dl, zo;
        omni_scales<Q, LPG>(lmin, lmax, beta, gamma, wm, wM, dl, zo);
        __syncwarp();                             // previous unit is done with the tables
        unit_levels<Q, NG>(t, tau_s[warp], lane, ALPHA, ZB, row * Gr + u * NG, min(NG, Gr - u * NG));
        const float tau = tau_s[warp][sub];
        float acc[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = 0.f;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            if (!(ok && v < nv)) continue;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int c = (cv[v] >> (8 * k)) & (L - 1);
                const float m = t.lv[sub][c];
                const float uu = __fdiv_rn(w[v][k], dl);
                const float x = __fadd_rn(uu, zo);
                const bool f = fabsf(__fsub_rn(x, m)) <= tau;
                const float gk = G[v][k];
                acc[0] += gk * ((m - zo) - (f ? uu : 0.f));
                acc[1] += f ? 0.f : gk;
                acc[2] += gk;
#pragma unroll
                for (int j = 0; j < Q; ++j) acc[4 + j] += ((c >> j) & 1) ? gk : -gk;
            }
        }
        const int slot0 = SR8::run(acc, lane);
        if (SR8::writer(lane)) {
#pragma unroll
            for (int i = 0; i < SR8::NOUT; ++i) sums[warp][sub][slot0 + i] = acc[i];
        }
        __syncwarp();
        if (ok && li == 0) {
            const float* sg = sums[warp][sub];
            const float A = sg[0];                                   // dL/dDelta with z_O held
            const float B = -(dl * sg[1]);                           // dL/dz_O
            const float l1 = (float)(L - 1);
            const float dDb = -wm / l1, dDg = wM / l1;
            const float bw = beta * wm;
            const float dzb = -(wm / dl - bw * dDb / (dl * dl));
            const float dzg = bw * dDg / (dl * dl);
            DBETA[grp] = A * dDb + B * dzb;
            DGAMMA[grp] = A * dDg + B * dzg;
            DZB[grp] = dl * sg[2];
#pragma unroll
            for (int j = 0; j < Q; ++j) DALPHA[grp * Q + j] = dl * sg[4 + j];
        }
        __syncwarp();                             // sums of this unit are read
    }
}

// ---------------------------------------------------------------------------
// Pipelined kernels (g in {32, 64, 128})
// ---------------------------------------------------------------------------

__device__ unsigned int g_omni_err = 0;

#ifndef UQ_OMNI_FWD_STAGE_BYTES
#define UQ_OMNI_FWD_STAGE_BYTES 5632
#endif
#ifndef UQ_OMNI_BWD_STAGE_BYTES
#define UQ_OMNI_BWD_STAGE_BYTES 11520
#endif

// Stage layouts: weights (no s), code words unless the full mapping, dL/dW^
// for the backward; the unit's beta in the Delta slot, gamma in the z_U slot.
template <int Q, typename WT, int G_, int MODE>
using OmniFwdStage = Stage<Q, WT, G_, true, false, MODE != FWD_FULL, UQ_OMNI_FWD_STAGE_BYTES, false>;
template <int Q, typename WT, int G_>
using OmniBwdStage = Stage<Q, WT, G_, true, true, true, UQ_OMNI_BWD_STAGE_BYTES, false>;

template <typename St, int KIND>
struct OmniTag {};

template <int Q, typename St>
__device__ __forceinline__ void omni_issue(const Items& it, const Cursor& c, int s, uint32_t bar, unsigned char* wsm,
                                           const void* W, const float* GUP, const uint8_t* CODES, const float* BETA,
                                           const float* GAMMA, const float* ZB, const float* ALPHA, int64_t out,
                                           int n_in, int Gr) {
    const int64_t row = it.row(c.k);
    if (row >= out) { tma::bar_arrive(bar); return; }
    const int64_t e0 = row * n_in + (int64_t)it.unit(c.j) * St::UE;
    const int64_t g0 = row * Gr + (int64_t)it.unit(c.j) * St::NG;
    const uint32_t d = tma::smem_addr(wsm + (size_t)s * St::BYTES);
    tma::fence_async_smem();
    tma::bar_arrive_tx(bar, St::TX);
    tma::copy_g2s(d + St::OFF_W, static_cast<const unsigned char*>(W) + e0 * St::WBYTES, St::SZ_W, bar);
    if constexpr (St::SZ_G > 0) tma::copy_g2s(d + St::OFF_G, GUP + e0, St::SZ_G, bar);
    if constexpr (St::SZ_C > 0) tma::copy_g2s(d + St::OFF_C, CODES + e0, St::SZ_C, bar);
    tma::copy_g2s(d + St::OFF_D, BETA + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_Z, GAMMA + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_B, ZB + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_A, ALPHA + g0 * Q, St::SZ_A, bar);
}

template <int Q, typename WT, int G_, int MODE>
__global__ void __launch_bounds__(kThreads, 3)
omni_stream_fwd_kernel(const void* __restrict__ W, const float* __restrict__ BETA, const float* __restrict__ GAMMA,
                       const float* __restrict__ ALPHA, const float* __restrict__ ZB, uint8_t* __restrict__ CODES,
                       float* __restrict__ WHAT, int64_t out, int n_in, int R, int n_rb) {
    using St = OmniFwdStage<Q, WT, G_, MODE>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NV = St::NV, UE = St::UE, NST = St::NST;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][NST];
    __shared__ MapTab<Q, NG> tabs[kWarps];
    constexpr int NIV = MODE == FWD_REMAP ? NG : 1;              // remap intervals only on remap steps
    __shared__ float4 ivs[kWarps][NIV][L];
    __shared__ float dzs[kWarps][2][NIV];                        // Delta_O, z_O per group slot
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / LPG, li = lane % LPG;
    const int U = n_in / UE, Gr = n_in / G_;
    const Items it(U, R, n_rb, warp);
    unsigned char* wsm = smem + (size_t)warp * St::WARP_BYTES;
    MapTab<Q, NG>& t = tabs[warp];

    if (lane == 0) {
        for (int s = 0; s < NST; ++s) tma::bar_init(tma::smem_addr(&bars[warp][s]), 1);
        tma::bar_init_fence();
    }
    __syncwarp();
    auto issue = [&](const Cursor& c, int s) {          // lane 0 only
        omni_issue<Q, St>(it, c, s, tma::smem_addr(&bars[warp][s]), wsm, W, nullptr, CODES, BETA, GAMMA, ZB, ALPHA,
                          out, n_in, Gr);
    };
    const bool ok = pipe_run<NST>(it, bars[warp], lane, &g_omni_err, 1u, issue,
                                  [&](const Cursor& cc, int s) {
        const int64_t row = it.row(cc.k);
        if (row < out) {
            const unsigned char* st = wsm + (size_t)s * St::BYTES;
            const float* pbeta = reinterpret_cast<const float*>(st + St::OFF_D);
            const float* pgam = reinterpret_cast<const float*>(st + St::OFF_Z);
            const float* pb = reinterpret_cast<const float*>(st + St::OFF_B);
            const float* pa = reinterpret_cast<const float*>(st + St::OFF_A);
            float w[NV][4];
            float lmin = INFINITY, lmax = -INFINITY;
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w[v]);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    lmin = fminf(lmin, w[v][k]);
                    lmax = fmaxf(lmax, w[v][k]);
                }
            }
            float wm, wM, dl, zo;
            omni_scales<Q, LPG>(lmin, lmax, pbeta[sub], pgam[sub], wm, wM, dl, zo);
#pragma unroll
            for (int e = lane; e < NG * L; e += 32) {
                const int kk = e / L, c = e % L;
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[kk * Q + jj];
                t.lv[kk][c] = level_of<Q>(c, a, pb[kk]);
            }
            __syncwarp();
            if constexpr (MODE == FWD_REMAP) {
                if (li == 0) {
                    dzs[warp][0][sub] = dl;
                    dzs[warp][1][sub] = zo;
                }
                unit_sort<Q, NG, false>(t, lane);
                unit_remap_iv<Q, NG>(t, ivs[warp], lane, dzs[warp][0], dzs[warp][1]);
            } else if constexpr (MODE == FWD_FULL) {
                unit_sort<Q, NG, false>(t, lane);
            }
            const int64_t ebase = row * n_in + (int64_t)it.unit(cc.j) * UE;
            float srt[L];
            if constexpr (MODE == FWD_FULL) {
#pragma unroll
                for (int r = 0; r < L; ++r) srt[r] = t.srt[sub][r];
            }
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                uint32_t cv = 0u;
                if constexpr (MODE != FWD_FULL) cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                float o[4];
                uint32_t nc = 0;
                if constexpr (MODE == FWD_REMAP) {
                    // x = w / Delta_O + z_O: the interval test with s = s_r = 1
                    const float one[4] = {1.f, 1.f, 1.f, 1.f};
                    nc = remap_vec4<Q, NG>(w[v], one, cv, t, ivs[warp], sub, dl, 1.f, zo, o);
                } else {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        float m;
                        uint32_t code;
                        if constexpr (MODE == FWD_KEEP) {
                            code = (cv >> (8 * k)) & (L - 1);
                            m = t.lv[sub][code];
                        } else {
                            const float x = __fadd_rn(__fdiv_rn(w[v][k], dl), zo);
                            const int r = nearest_rank<L>(x, srt, m);
                            code = t.cor[sub][r];
                        }
                        o[k] = __fmul_rn(dl, __fsub_rn(m, zo));
                        nc |= code << (8 * k);
                    }
                }
                if constexpr (MODE != FWD_KEEP) *reinterpret_cast<uint32_t*>(CODES + ebase + el) = nc;
                *reinterpret_cast<float4*>(WHAT + ebase + el) = make_float4(o[0], o[1], o[2], o[3]);
            }
        }
                                  });
    if (!ok) return;                                 // no block barrier in this kernel
}

template <int Q, typename WT, int G_>
__global__ void __launch_bounds__(kThreads, 2)
omni_stream_bwd_kernel(const void* __restrict__ W, const float* __restrict__ BETA, const float* __restrict__ GAMMA,
                       const float* __restrict__ ALPHA, const float* __restrict__ ZB, const uint8_t* __restrict__ CODES,
                       const float* __restrict__ GUP, float* __restrict__ DBETA, float* __restrict__ DGAMMA,
                       float* __restrict__ DALPHA, float* __restrict__ DZB, int64_t out, int n_in, int R, int n_rb) {
    using St = OmniBwdStage<Q, WT, G_>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NV = St::NV, UE = St::UE, NST = St::NST;
    using SR8 = SegReduce<LPG>;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][NST];
    __shared__ float lvs[kWarps][NG][L];
    __shared__ float sums[kWarps][NG][8];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / LPG, li = lane % LPG;
    const int U = n_in / UE, Gr = n_in / G_;
    const Items it(U, R, n_rb, warp);
    unsigned char* wsm = smem + (size_t)warp * St::WARP_BYTES;

    if (lane == 0) {
        for (int s = 0; s < NST; ++s) tma::bar_init(tma::smem_addr(&bars[warp][s]), 1);
        tma::bar_init_fence();
    }
    __syncwarp();
    auto issue = [&](const Cursor& c, int s) {          // lane 0 only
        omni_issue<Q, St>(it, c, s, tma::smem_addr(&bars[warp][s]), wsm, W, GUP, CODES, BETA, GAMMA, ZB, ALPHA, out,
                          n_in, Gr);
    };
    const bool ok = pipe_run<NST>(it, bars[warp], lane, &g_omni_err, 1u, issue,
                                  [&](const Cursor& cc, int s) {
        const int64_t row = it.row(cc.k);
        if (row < out) {
            const unsigned char* st = wsm + (size_t)s * St::BYTES;
            const float* pbeta = reinterpret_cast<const float*>(st + St::OFF_D);
            const float* pgam = reinterpret_cast<const float*>(st + St::OFF_Z);
            const float* pb = reinterpret_cast<const float*>(st + St::OFF_B);
            const float* pa = reinterpret_cast<const float*>(st + St::OFF_A);
            float w[NV][4];
            float lmin = INFINITY, lmax = -INFINITY;
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w[v]);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    lmin = fminf(lmin, w[v][k]);
                    lmax = fmaxf(lmax, w[v][k]);
                }
            }
            const float beta = pbeta[sub], gamma = pgam[sub];
            float wm, wM, dl, zo;
            omni_scales<Q, LPG>(lmin, lmax, beta, gamma, wm, wM, dl, zo);
#pragma unroll
            for (int e = lane; e < NG * L; e += 32) {
                const int kk = e / L, c = e % L;
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[kk * Q + jj];
                lvs[warp][kk][c] = level_of<Q>(c, a, pb[kk]);
            }
            __syncwarp();
            // tau of the lane's own group, on every lane
            float tau = fabsf(pa[sub * Q]);
#pragma unroll
            for (int jj = 1; jj < Q; ++jj) tau = fminf(tau, fabsf(pa[sub * Q + jj]));
            // x = w / Delta_O + z_O: one reciprocal of Delta_O per group, the
            // filter proven equal to the IEEE one (shared_div_filter4)
            const float rdl = rcp_approx(dl);
            const float eg = bwd_margin(zo, pb[sub], pa + sub * Q, Q, dl);
            float acc[8];
#pragma unroll
            for (int q8 = 0; q8 < 8; ++q8) acc[q8] = 0.f;
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                float G[4];
                f4_to(*reinterpret_cast<const float4*>(st + St::OFF_G + el * 4), G);
                const uint32_t cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                float m4[4], uv[4];
                bool fv[4];
#pragma unroll
                for (int k = 0; k < 4; ++k) m4[k] = lvs[warp][sub][(cv >> (8 * k)) & (L - 1)];
                shared_div_filter4(w[v], dl, rdl, zo, m4, tau, eg, uv, fv);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int c = (cv >> (8 * k)) & (L - 1);
                    const float m = m4[k];
                    const float uu = uv[k];
                    const bool f = fv[k];
                    const float gk = G[k];
                    acc[0] += gk * ((m - zo) - (f ? uu : 0.f));
                    acc[1] += f ? 0.f : gk;
                    acc[2] += gk;
#pragma unroll
                    for (int j = 0; j < Q; ++j)                  // P_j: dalpha_j = Delta (2 P_j - S)
                        if ((c >> j) & 1) acc[4 + j] += gk;
                }
            }
            const int slot0 = SR8::run(acc, lane);
            if (SR8::writer(lane)) {
#pragma unroll
                for (int i2 = 0; i2 < SR8::NOUT; ++i2) sums[warp][sub][slot0 + i2] = acc[i2];
            }
            __syncwarp();
            if (li == 0) {
                const int64_t grp = row * Gr + (int64_t)it.unit(cc.j) * NG + sub;
                const float* sg = sums[warp][sub];
                const float A = sg[0];
                const float B = -(dl * sg[1]);
                const float l1 = (float)(L - 1);
                const float dDb = -wm / l1, dDg = wM / l1;
                const float bw = beta * wm;
                const float dzb = -(wm / dl - bw * dDb / (dl * dl));
                const float dzg = bw * dDg / (dl * dl);
                DBETA[grp] = A * dDb + B * dzb;
                DGAMMA[grp] = A * dDg + B * dzg;
                DZB[grp] = dl * sg[2];
#pragma unroll
                for (int j = 0; j < Q; ++j) DALPHA[grp * Q + j] = dl * __fmaf_rn(2.f, sg[4 + j], -sg[2]);
            }
        }
                                  });
    if (!ok) return;                                 // no block barrier in this kernel
}

template <int Q, typename WT, int G_, int MODE>
static cudaError_t run_omni_stream_fwd(const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes, float* what,
                                       cudaStream_t st) {
    using St = OmniFwdStage<Q, WT, G_, MODE>;
    const int U = sh.n_in / St::UE;
    const int R = rows_per_block(U);
    const int n_rb = (int)((sh.out + R - 1) / R);
    const size_t dyn = (size_t)kWarps * St::WARP_BYTES;
    auto kern = omni_stream_fwd_kernel<Q, WT, G_, MODE>;
    int grid = 0;
    cudaError_t e = grid_for<OmniTag<St, MODE>>(kern, dyn, n_rb, grid);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, dyn, st>>>(W, p.beta, p.gamma, p.alpha, p.zb, codes, what, sh.out, sh.n_in, R, n_rb);
    return cudaGetLastError();
}

template <int Q, typename WT, int G_>
static cudaError_t run_omni_stream_bwd(const Shape& sh, const void* W, uq_params_omni p, const uint8_t* codes,
                                       const float* gup, uq_grads_omni gr, cudaStream_t st) {
    using St = OmniBwdStage<Q, WT, G_>;
    const int U = sh.n_in / St::UE;
    const int R = rows_per_block(U);
    const int n_rb = (int)((sh.out + R - 1) / R);
    const size_t dyn = (size_t)kWarps * St::WARP_BYTES;
    auto kern = omni_stream_bwd_kernel<Q, WT, G_>;
    int grid = 0;
    cudaError_t e = grid_for<OmniTag<St, 9>>(kern, dyn, n_rb, grid);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, dyn, st>>>(W, p.beta, p.gamma, p.alpha, p.zb, codes, gup, gr.dbeta, gr.dgamma, gr.dalpha,
                                      gr.dzb, sh.out, sh.n_in, R, n_rb);
    return cudaGetLastError();
}

template <int Q, typename WT, int G_>
static cudaError_t omni_stream_g(bool bwd, int mode, const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes,
                                 float* what, const float* gup, uq_grads_omni gr, cudaStream_t st) {
    if (bwd) return run_omni_stream_bwd<Q, WT, G_>(sh, W, p, codes, gup, gr, st);
    if (mode == FWD_KEEP) return run_omni_stream_fwd<Q, WT, G_, FWD_KEEP>(sh, W, p, codes, what, st);
    if (mode == FWD_REMAP) return run_omni_stream_fwd<Q, WT, G_, FWD_REMAP>(sh, W, p, codes, what, st);
    return run_omni_stream_fwd<Q, WT, G_, FWD_FULL>(sh, W, p, codes, what, st);
}

template <int Q, typename WT>
static cudaError_t omni_stream_w(bool bwd, int mode, const Shape& sh, const void* W, uq_params_omni p,
                                 uint8_t* codes, float* what, const float* gup, uq_grads_omni gr, cudaStream_t st) {
    if (sh.g == 32) return omni_stream_g<Q, WT, 32>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
    if (sh.g == 64) return omni_stream_g<Q, WT, 64>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
    return omni_stream_g<Q, WT, 128>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
}

template <int Q>
static cudaError_t omni_stream_q(bool bwd, int mode, const Shape& sh, const void* W, uq_params_omni p,
                                 uint8_t* codes, float* what, const float* gup, uq_grads_omni gr, cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return omni_stream_w<Q, WBF16>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
    return omni_stream_w<Q, WF32>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
}

static cudaError_t omni_stream(bool bwd, int mode, const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes,
                               float* what, const float* gup, uq_grads_omni gr, cudaStream_t st) {
    switch (sh.q) {
        case 1: return omni_stream_q<1>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
        case 2: return omni_stream_q<2>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
        case 3: return omni_stream_q<3>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
        default: return omni_stream_q<4>(bwd, mode, sh, W, p, codes, what, gup, gr, st);
    }
}

cudaError_t omni_error(bool clear, unsigned int* flag) {
    unsigned int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_omni_err, sizeof(v));
    if (e != cudaSuccess) return e;
    *flag = v;
    if (clear && v) {
        const unsigned int z = 0;
        e = cudaMemcpyToSymbol(g_omni_err, &z, sizeof(z));
    }
    return e;
}

bool omni_ok(const Shape& sh) { return sh.g == 32 || sh.g == 64 || sh.g == 128 || sh.g == 256 || sh.g == 512; }

template <int Q, typename WT, int LPG, int MODE>
static cudaError_t run_omni_fwd(const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes, float* what,
                                float* dout, float* zout, cudaStream_t st) {
    constexpr int NG = 32 / LPG;
    const int Gr = sh.n_in / sh.g;
    const int R = rows_per_block((Gr + NG - 1) / NG);
    const int64_t blocks = (sh.out + R - 1) / R;
    omni_fwd_kernel<Q, WT, LPG, MODE><<<dim3((unsigned)blocks), kThreads, 0, st>>>(
        W, p.beta, p.gamma, p.alpha, p.zb, codes, what, dout, zout, sh.out, sh.n_in, sh.g, R);
    return cudaGetLastError();
}

template <int Q, typename WT, int LPG>
static cudaError_t run_omni_bwd(const Shape& sh, const void* W, uq_params_omni p, const uint8_t* codes,
                                const float* gup, uq_grads_omni gr, cudaStream_t st) {
    constexpr int NG = 32 / LPG;
    const int Gr = sh.n_in / sh.g;
    const int R = rows_per_block((Gr + NG - 1) / NG);
    const int64_t blocks = (sh.out + R - 1) / R;
    omni_bwd_kernel<Q, WT, LPG><<<dim3((unsigned)blocks), kThreads, 0, st>>>(
        W, p.beta, p.gamma, p.alpha, p.zb, codes, gup, gr.dbeta, gr.dgamma, gr.dalpha, gr.dzb, sh.out, sh.n_in,
        sh.g, R);
    return cudaGetLastError();
}

// kind: 0 forward (mode), 1 backward, 2 scales only
template <int Q, typename WT, int LPG>
static cudaError_t omni_lpg(int kind, int mode, const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes,
                            float* what, const float* gup, uq_grads_omni gr, float* dout, float* zout,
                            cudaStream_t st) {
    if (kind == 1) return run_omni_bwd<Q, WT, LPG>(sh, W, p, codes, gup, gr, st);
    if (kind == 2) return run_omni_fwd<Q, WT, LPG, FWD_FULL>(sh, W, p, nullptr, nullptr, dout, zout, st);
    if (mode == FWD_KEEP) return run_omni_fwd<Q, WT, LPG, FWD_KEEP>(sh, W, p, codes, what, nullptr, nullptr, st);
    if (mode == FWD_REMAP) return run_omni_fwd<Q, WT, LPG, FWD_REMAP>(sh, W, p, codes, what, nullptr, nullptr, st);
    return run_omni_fwd<Q, WT, LPG, FWD_FULL>(sh, W, p, codes, what, nullptr, nullptr, st);
}

template <int Q, typename WT>
static cudaError_t omni_g(int kind, int mode, const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes,
                          float* what, const float* gup, uq_grads_omni gr, float* dout, float* zout, cudaStream_t st) {
    switch (lanes_per_group(sh.g)) {
        case 4: return omni_lpg<Q, WT, 4>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
        case 8: return omni_lpg<Q, WT, 8>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
        case 16: return omni_lpg<Q, WT, 16>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
        default: return omni_lpg<Q, WT, 32>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
    }
}

template <int Q>
static cudaError_t omni_w(int kind, int mode, const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes,
                          float* what, const float* gup, uq_grads_omni gr, float* dout, float* zout, cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return omni_g<Q, WBF16>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
    return omni_g<Q, WF32>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
}

static cudaError_t omni_dispatch(int kind, int mode, const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes,
                                 float* what, const float* gup, uq_grads_omni gr, float* dout, float* zout,
                                 cudaStream_t st) {
    switch (sh.q) {
        case 1: return omni_w<1>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
        case 2: return omni_w<2>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
        case 3: return omni_w<3>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
        default: return omni_w<4>(kind, mode, sh, W, p, codes, what, gup, gr, dout, zout, st);
    }
}

cudaError_t launch_omni_fwd(const Shape& sh, const void* W, uq_params_omni p, uint8_t* codes, int mode, float* what,
                            cudaStream_t st) {
    if (stream_path_ok(sh)) return omni_stream(false, mode, sh, W, p, codes, what, nullptr, uq_grads_omni{}, st);
    return omni_dispatch(0, mode, sh, W, p, codes, what, nullptr, uq_grads_omni{}, nullptr, nullptr, st);
}

cudaError_t launch_omni_bwd(const Shape& sh, const void* W, uq_params_omni p, const uint8_t* codes, const float* gup,
                            uq_grads_omni gr, cudaStream_t st) {
    if (stream_path_ok(sh))
        return omni_stream(true, 0, sh, W, p, const_cast<uint8_t*>(codes), nullptr, gup, gr, st);
    return omni_dispatch(1, 0, sh, W, p, const_cast<uint8_t*>(codes), nullptr, gup, gr, nullptr, nullptr, st);
}

cudaError_t launch_omni_scales(const Shape& sh, const void* W, const float* beta, const float* gamma, float* delta,
                               float* zo, cudaStream_t st) {
    uq_params_omni p{const_cast<float*>(beta), const_cast<float*>(gamma), nullptr, nullptr};
    return omni_dispatch(2, 0, sh, W, p, nullptr, nullptr, nullptr, uq_grads_omni{}, delta, zo, st);
}

}  // namespace uq
