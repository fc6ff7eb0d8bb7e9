// Backward of the quantizer: straight-through estimator with gradient
// filtering (App. C.1) through Eq. 3, one thread block per row.
//
// Per element (4 per lane per warp-step): recompute x = T_F(w) and
// m = l(code), filter f = |x - m| <= tau (fp32 decision), write ds.  Per
// group: 3 + q partial sums (dDelta, dz_U, dz_B, dalpha_j) are reduced over
// the group's lanes by a segmented butterfly (no atomics); for g > 128 the
// per-warp-step partials of a row go to shared memory and are summed per
// group in warp-step order after the row is done.  ds_r: per-lane partials,
// warp sums, then the 8 warp sums in warp order.
// HBM traffic per element (bf16 W): 2 + 4 + 1 + 4 read, 4 written.
#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

template <int Q, typename WT, int GPS>
__global__ void __launch_bounds__(kThreads)
bwd_kernel(const void* __restrict__ W, const float* __restrict__ S, const float* __restrict__ SR,
           const float* __restrict__ DELTA, const float* __restrict__ ZU, const float* __restrict__ ALPHA,
           const float* __restrict__ ZB, const uint8_t* __restrict__ CODES, const float* __restrict__ GUP,
           float* __restrict__ DS, float* __restrict__ DSR, float* __restrict__ DDELTA, float* __restrict__ DZU,
           float* __restrict__ DZB, float* __restrict__ DALPHA, int n_in, int g) {
    constexpr int L = 1 << Q;
    constexpr int WB = kSlots / GPS;
    constexpr int SH = GPS == 4 ? 3 : (GPS == 2 ? 4 : 5);
    constexpr int SEGL = 32 / GPS;              // lanes per group within a warp-step
    constexpr int NSUM = 3 + Q;                 // dDelta, dz_U, dz_B, dalpha_1..q
    __shared__ GroupTables<Q> tabs[kWarps];
    __shared__ float red[kWarps];
    extern __shared__ float part[];             // [n_ws][8] when g > 128
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    GroupTables<Q>& t = tabs[warp];
    const int64_t row = blockIdx.x;
    const int n_ws = (n_in + kStep - 1) / kStep;
    const int Gr = n_in / g;
    const int64_t eoff = row * (int64_t)n_in;
    const int64_t goff = row * (int64_t)Gr;
    const float sr = __ldg(SR + row);
    const bool big = g > kStep;
    float pacc = 0.f;                           // sum of G Delta f u over this lane's elements

    for (int base = warp; base < n_ws; base += kWarps * WB) {
        typename WT::raw wraw[WB];
        float4 sv[WB], gv[WB];
        uint32_t cv[WB];
        float dl[WB], zu[WB];
        bool ok[WB];
        int col[WB];
#pragma unroll
        for (int b = 0; b < WB; ++b) {
            const int ws = base + b * kWarps;
            col[b] = ws * kStep + lane * kVec;
            ok[b] = ws < n_ws && col[b] < n_in;
            if (ok[b]) {
                const int64_t grp = goff + (ws * kStep) / g + (lane >> SH);
                dl[b] = __ldg(DELTA + grp);
                zu[b] = __ldg(ZU + grp);
                wraw[b] = WT::load(W, eoff + col[b]);
                sv[b] = ldg4(S + eoff + col[b]);
                gv[b] = ldg4(GUP + eoff + col[b]);
                cv[b] = __ldg(reinterpret_cast<const unsigned int*>(CODES + eoff + col[b]));
            }
        }
        auto grp_of_slot = [&](int k) -> int64_t {
            return goff + ((base + (k / GPS) * kWarps) * kStep) / g + (k % GPS);
        };
        auto ok_of_slot = [&](int k) -> bool {
            const int ws = base + (k / GPS) * kWarps;
            return ws < n_ws && (ws * kStep) / g + (k % GPS) < Gr;
        };
        __syncwarp();
        build_tables<Q, false, false>(t, lane, ALPHA, ZB, grp_of_slot, ok_of_slot);

#pragma unroll
        for (int b = 0; b < WB; ++b) {
            const int ws = base + b * kWarps;
            if (ws >= n_ws) break;                      // warp-uniform
            const int k = b * GPS + (lane >> SH);
            float acc[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = 0.f;
            if (ok[b]) {
                float w[4], s[4], G[4], ds[4];
                WT::unpack(wraw[b], w);
                f4_to(sv[b], s);
                f4_to(gv[b], G);
                const float tau = t.tau[k];
                const float d = dl[b], z = zu[b];
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    const int c = (cv[b] >> (8 * v)) & (L - 1);
                    const float m = t.lv[k][c];
                    float u;
                    const float x = transform_x(w[v], s[v], d, sr, z, u);
                    const bool f = fabsf(__fsub_rn(x, m)) <= tau;
                    const float gb = G[v] * d;                   // dL/dw~
                    const float fu = f ? u : 0.f;
                    ds[v] = __fdividef(-(gb * fu), s[v]);
                    acc[0] += G[v] * ((m - z) - fu);
                    acc[1] += f ? 0.f : -gb;
                    acc[2] += gb;
#pragma unroll
                    for (int j = 0; j < Q; ++j) acc[3 + j] += ((c >> j) & 1) ? gb : -gb;
                    pacc += gb * fu;
                }
                *reinterpret_cast<float4*>(DS + eoff + col[b]) = make_float4(ds[0], ds[1], ds[2], ds[3]);
            }
            int slot;
            const float tot = seg_reduce8<SEGL>(acc, lane, slot);
            const bool writer = (lane & (SEGL / 8 - 1)) == 0 && slot < NSUM;
            if (!big) {
                const int gi = (ws * kStep) / g + (lane >> SH);
                if (writer && gi < Gr) {
                    const int64_t grp = goff + gi;
                    float* dst = slot == 0 ? DDELTA + grp : slot == 1 ? DZU + grp : slot == 2 ? DZB + grp
                                                                                : DALPHA + grp * Q + (slot - 3);
                    *dst = tot;
                }
            } else if (writer) {
                part[ws * 8 + slot] = tot;
            }
        }
    }

    pacc = warp_sum(pacc);
    if (lane == 0) red[warp] = pacc;
    __syncthreads();
    if (threadIdx.x == 0) {
        float s = red[0];
#pragma unroll
        for (int w = 1; w < kWarps; ++w) s += red[w];
        DSR[row] = -s / sr;
    }
    if (big) {
        const int spg = g / kStep;                  // warp-steps per group
        for (int idx = threadIdx.x; idx < Gr * NSUM; idx += kThreads) {
            const int gi = idx / NSUM, slot = idx % NSUM;
            float s = part[(gi * spg) * 8 + slot];
            for (int st = 1; st < spg; ++st) s += part[(gi * spg + st) * 8 + slot];
            const int64_t grp = goff + gi;
            float* dst = slot == 0 ? DDELTA + grp : slot == 1 ? DZU + grp : slot == 2 ? DZB + grp
                                                                        : DALPHA + grp * Q + (slot - 3);
            *dst = s;
        }
    }
}

template <int Q, typename WT, int GPS>
static cudaError_t run_bwd(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                           uq_grads gr, cudaStream_t st) {
    const int n_ws = (sh.n_in + kStep - 1) / kStep;
    const size_t dyn = sh.g > kStep ? (size_t)n_ws * 8 * sizeof(float) : 0;
    auto kern = bwd_kernel<Q, WT, GPS>;
    if (dyn > 32 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e != cudaSuccess) return e;
    }
    kern<<<dim3((unsigned)sh.out), kThreads, dyn, st>>>(W, p.s, p.sr, p.delta, p.zu, p.alpha, p.zb, codes, gup,
                                                        gr.ds, gr.dsr, gr.ddelta, gr.dzu, gr.dzb, gr.dalpha,
                                                        sh.n_in, sh.g);
    return cudaGetLastError();
}

template <int Q, typename WT>
static cudaError_t bwd_g(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                         uq_grads gr, cudaStream_t st) {
    if (sh.g == 32) return run_bwd<Q, WT, 4>(sh, W, p, codes, gup, gr, st);
    if (sh.g == 64) return run_bwd<Q, WT, 2>(sh, W, p, codes, gup, gr, st);
    return run_bwd<Q, WT, 1>(sh, W, p, codes, gup, gr, st);
}

template <int Q>
static cudaError_t bwd_w(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                         uq_grads gr, cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return bwd_g<Q, WBF16>(sh, W, p, codes, gup, gr, st);
    return bwd_g<Q, WF32>(sh, W, p, codes, gup, gr, st);
}

cudaError_t launch_bwd(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                       uq_grads gr, cudaStream_t st) {
    switch (sh.q) {
        case 1: return bwd_w<1>(sh, W, p, codes, gup, gr, st);
        case 2: return bwd_w<2>(sh, W, p, codes, gup, gr, st);
        case 3: return bwd_w<3>(sh, W, p, codes, gup, gr, st);
        default: return bwd_w<4>(sh, W, p, codes, gup, gr, st);
    }
}

}  // namespace uq
