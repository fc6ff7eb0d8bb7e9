// Backward of the quantizer: straight-through estimator with gradient
// filtering (App. C.1) through Eq. 3.
//
// Per element (NV vectors of 4 per lane and group, see uq_common.cuh):
// recompute x = T_F(w) and m = l(code), filter f = |x - m| <= tau (fp32
// decision), write ds = -(Delta G f u) / s.  Per group, with G = dL/dW^:
//   S0 = sum G ((m - z_U) - f u)   -> dDelta = S0
//   S1 = sum_{f = 0} G             -> dz_U   = -Delta S1
//   S2 = sum G                     -> dz_B   =  Delta S2
//   S3 = sum G f u                 -> row partial Delta S3 of ds_r
//   S4+j = sum G c_j               -> dalpha_j = Delta S4+j
// are reduced over the group's LPG lanes (SegReduce, no atomics); groups of
// more than 512 elements accumulate over several vector chunks first.
// ds_r = -(sum over the row of Delta S3) / s_r, summed per row in warp and
// lane order.  HBM traffic per element (bf16 W): 2 + 4 + 1 + 4 read, 4
// written.
#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

// Minimum resident blocks per SM the register allocation is bounded for.
#ifndef UQ_BWD_MIN_BLOCKS
#define UQ_BWD_MIN_BLOCKS 3
#endif

// ELEM: the whole-element filter (a filtered element drops out of every
// gradient); otherwise the filter cuts the straight-through path only.
template <int Q, typename WT, int LPG, bool ELEM>
__global__ void __launch_bounds__(kThreads, UQ_BWD_MIN_BLOCKS)
bwd_kernel(const void* __restrict__ W, const float* __restrict__ S, const float* __restrict__ SR,
           const float* __restrict__ DELTA, const float* __restrict__ ZU, const float* __restrict__ ALPHA,
           const float* __restrict__ ZB, const uint8_t* __restrict__ CODES, const float* __restrict__ GUP,
           float* __restrict__ DS, float* __restrict__ DSR, float* __restrict__ DDELTA, float* __restrict__ DZU,
           float* __restrict__ DZB, float* __restrict__ DALPHA, int64_t out, int n_in, int g, int R) {
    constexpr int L = 1 << Q;
    constexpr int NG = 32 / LPG;                 // groups per unit
    using SR8 = SegReduce<LPG>;
    __shared__ LvTab<Q, NG> tabs[kWarps];
    __shared__ float tau_s[kWarps][NG];
    __shared__ float red[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    LvTab<Q, NG>& t = tabs[warp];
    const int WPR = kWarps / R;
    const int64_t row = (int64_t)blockIdx.x * R + warp / WPR;
    const int wr = warp % WPR;
    const int Gr = n_in / g;
    const int units = (Gr + NG - 1) / NG;
    const int nv = g / (4 * LPG);                // vectors per lane and group
    const int sub = lane / LPG, li = lane % LPG;
    float prow = 0.f;                            // this lane's share of sum Delta S3 over the row

    if (row < out) {
        const float sr = __ldg(SR + row);
        const int64_t rbase = row * (int64_t)n_in;
        for (int u = wr; u < units; u += WPR) {
            const int gi = u * NG + sub;
            const bool ok = gi < Gr;
            const int64_t grp = row * Gr + gi;
            const int64_t ebase = rbase + (int64_t)gi * g + 4 * li;
            float dl = 0.f, zu = 0.f;
            typename WT::raw wr4[4];
            float4 sv[4], gv[4];
            uint32_t cv[4];
            auto load_chunk = [&](int c0) {
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    if (ok && c0 + v < nv) {
                        const int64_t e = ebase + 4 * LPG * (c0 + v);
                        wr4[v] = WT::load(W, e);
                        sv[v] = ldg4(S + e);
                        gv[v] = ldg4(GUP + e);
                        cv[v] = __ldg(reinterpret_cast<const unsigned int*>(CODES + e));
                    }
                }
            };
            load_chunk(0);
            if (ok) {
                dl = __ldg(DELTA + grp);
                zu = __ldg(ZU + grp);
            }
            __syncwarp();                        // previous unit is done with the tables
            unit_levels<Q, NG>(t, tau_s[warp], lane, ALPHA, ZB, row * Gr + u * NG, min(NG, Gr - u * NG));
            const float tau = tau_s[warp][sub];
            float acc[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = 0.f;
            for (int c0 = 0; c0 < nv; c0 += 4) {
                if (c0 > 0) load_chunk(c0);
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    if (!(ok && c0 + v < nv)) continue;
                    float w[4], s[4], G[4], ds[4];
                    WT::unpack(wr4[v], w);
                    f4_to(sv[v], s);
                    f4_to(gv[v], G);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int c = (cv[v] >> (8 * k)) & (L - 1);
                        const float m = t.lv[sub][c];
                        float uu;
                        const float x = transform_x(w[k], s[k], dl, sr, zu, uu);
                        const bool f = fabsf(__fsub_rn(x, m)) <= tau;
                        const float fu = f ? uu : 0.f;
                        const float gk = (ELEM && !f) ? 0.f : G[k];
                        const float gfu = gk * fu;
                        ds[k] = -__fdividef(dl * gfu, s[k]);
                        acc[0] += gk * ((m - zu) - fu);
                        acc[1] += f ? 0.f : gk;
                        acc[2] += gk;
                        acc[3] += gfu;
#pragma unroll
                        for (int j = 0; j < Q; ++j) acc[4 + j] += ((c >> j) & 1) ? gk : -gk;
                    }
                    *reinterpret_cast<float4*>(DS + ebase + 4 * LPG * (c0 + v)) = make_float4(ds[0], ds[1], ds[2], ds[3]);
                }
            }
            const int slot0 = SR8::run(acc, lane);
            if (ok && SR8::writer(lane)) {
#pragma unroll
                for (int i = 0; i < SR8::NOUT; ++i) {
                    const int slot = slot0 + i;
                    const float tot = acc[i];
                    if (slot == 0) DDELTA[grp] = tot;
                    else if (slot == 1) DZU[grp] = -(dl * tot);
                    else if (slot == 2) DZB[grp] = dl * tot;
                    else if (slot == 3) prow += dl * tot;
                    else if (slot - 4 < Q) DALPHA[grp * Q + (slot - 4)] = dl * tot;
                }
            }
        }
    }

    // ds_r: the row's lane shares, summed in lane order, then in warp order.
    prow = warp_sum(prow);
    if (lane == 0) red[warp] = prow;
    __syncthreads();
    if (threadIdx.x < R) {
        const int64_t r = (int64_t)blockIdx.x * R + threadIdx.x;
        if (r < out) {
            float s = red[threadIdx.x * WPR];
            for (int w = 1; w < WPR; ++w) s += red[threadIdx.x * WPR + w];
            DSR[r] = -s / __ldg(SR + r);
        }
    }
}

template <int Q, typename WT, int LPG, bool ELEM>
static cudaError_t run_bwd(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                           uq_grads gr, cudaStream_t st) {
    constexpr int NG = 32 / LPG;
    const int Gr = sh.n_in / sh.g;
    const int R = rows_per_block((Gr + NG - 1) / NG);
    const int64_t blocks = (sh.out + R - 1) / R;
    bwd_kernel<Q, WT, LPG, ELEM><<<dim3((unsigned)blocks), kThreads, 0, st>>>(
        W, p.s, p.sr, p.delta, p.zu, p.alpha, p.zb, codes, gup, gr.ds, gr.dsr, gr.ddelta, gr.dzu, gr.dzb, gr.dalpha,
        sh.out, sh.n_in, sh.g, R);
    return cudaGetLastError();
}

template <int Q, typename WT, bool ELEM>
static cudaError_t bwd_gf(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                          uq_grads gr, cudaStream_t st) {
    switch (lanes_per_group(sh.g)) {
        case 4: return run_bwd<Q, WT, 4, ELEM>(sh, W, p, codes, gup, gr, st);
        case 8: return run_bwd<Q, WT, 8, ELEM>(sh, W, p, codes, gup, gr, st);
        case 16: return run_bwd<Q, WT, 16, ELEM>(sh, W, p, codes, gup, gr, st);
        default: return run_bwd<Q, WT, 32, ELEM>(sh, W, p, codes, gup, gr, st);
    }
}

template <int Q>
static cudaError_t bwd_w(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                         uq_grads gr, int filter, cudaStream_t st) {
    const bool elem = filter == UQ_FILTER_ELEMENT;
    if (sh.wdtype == UQ_W_BF16)
        return elem ? bwd_gf<Q, WBF16, true>(sh, W, p, codes, gup, gr, st)
                    : bwd_gf<Q, WBF16, false>(sh, W, p, codes, gup, gr, st);
    return elem ? bwd_gf<Q, WF32, true>(sh, W, p, codes, gup, gr, st)
                : bwd_gf<Q, WF32, false>(sh, W, p, codes, gup, gr, st);
}

cudaError_t launch_bwd(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                       uq_grads gr, cudaStream_t st, int filter) {
    if (stream_path_ok(sh)) return launch_bwd_stream(sh, W, p, codes, gup, gr, st, filter);
    switch (sh.q) {
        case 1: return bwd_w<1>(sh, W, p, codes, gup, gr, filter, st);
        case 2: return bwd_w<2>(sh, W, p, codes, gup, gr, filter, st);
        case 3: return bwd_w<3>(sh, W, p, codes, gup, gr, filter, st);
        default: return bwd_w<4>(sh, W, p, codes, gup, gr, filter, st);
    }
}

}  // namespace uq
