// Export: unification theorem (Theorem 1) and bit-plane packing of the
// final binary codes (Algorithm 1, lines 10-11), one thread block per row.
//
// alpha* = Delta alpha, z_B* = Delta (z_B - z_U) per group.  The codes are
// the stored ones (REUSE) or the nearest level of Theta_B* to each original
// weight (Eq. 4).  Packing: a lane holds 4 consecutive code words; for each
// 32-column word of a warp-step, one shuffle gives every lane the code of
// its column and one __ballot_sync per bit j yields the 32-bit word of
// plane j.  HBM traffic per element: 1 (or 2 for Eq. 4 with bf16 W) read,
// q/8 written, plus (q+1)*4/g each way for the group parameters.
#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

template <int Q, typename WT, int GPS, bool EQ4>
__global__ void __launch_bounds__(kThreads)
export_kernel(const void* __restrict__ W, const float* __restrict__ DELTA, const float* __restrict__ ZU,
              const float* __restrict__ ALPHA, const float* __restrict__ ZB, const uint8_t* __restrict__ CODES,
              uint32_t* __restrict__ PLANES, float* __restrict__ ASTAR, float* __restrict__ ZSTAR, int64_t out,
              int n_in, int g) {
    constexpr int L = 1 << Q;
    constexpr int WB = kSlots / GPS;
    constexpr int SH = GPS == 4 ? 3 : (GPS == 2 ? 4 : 5);
    constexpr uint32_t kMask = (uint32_t(L - 1) * 0x01010101u);
    __shared__ GroupTables<Q> tabs[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    GroupTables<Q>& t = tabs[warp];
    const int64_t row = blockIdx.x;
    const int n_ws = (n_in + kStep - 1) / kStep;
    const int Gr = n_in / g;
    const int words = n_in / 32;
    const int64_t eoff = row * (int64_t)n_in;
    const int64_t goff = row * (int64_t)Gr;

    // Theorem 1 for every group of the row.
    for (int gi = threadIdx.x; gi < Gr; gi += kThreads) {
        const int64_t grp = goff + gi;
        const float d = __ldg(DELTA + grp);
#pragma unroll
        for (int j = 0; j < Q; ++j) ASTAR[grp * Q + j] = __fmul_rn(d, __ldg(ALPHA + grp * Q + j));
        ZSTAR[grp] = __fmul_rn(d, __fsub_rn(__ldg(ZB + grp), __ldg(ZU + grp)));
    }

    for (int base = warp; base < n_ws; base += kWarps * WB) {
        uint32_t cw[WB];
        typename WT::raw wraw[WB];
        bool ok[WB];
        int col[WB];
#pragma unroll
        for (int b = 0; b < WB; ++b) {
            const int ws = base + b * kWarps;
            col[b] = ws * kStep + lane * kVec;
            ok[b] = ws < n_ws && col[b] < n_in;
            cw[b] = 0;
            if (ok[b]) {
                if constexpr (EQ4) wraw[b] = WT::load(W, eoff + col[b]);
                else cw[b] = __ldg(reinterpret_cast<const unsigned int*>(CODES + eoff + col[b])) & kMask;
            }
        }
        if constexpr (EQ4) {
            // Levels of Theta_B*: the same fp32 alpha*, z_B* as written above.
            auto ok_of_slot = [&](int k) -> bool {
                const int ws = base + (k / GPS) * kWarps;
                return ws < n_ws && (ws * kStep) / g + (k % GPS) < Gr;
            };
            __syncwarp();
            constexpr int E = kSlots * L;
#pragma unroll
            for (int e = lane; e < E; e += 32) {
                const int k = e / L, c = e % L;
                float lvv = 0.f;
                if (ok_of_slot(k)) {
                    const int64_t grp = goff + ((base + (k / GPS) * kWarps) * kStep) / g + (k % GPS);
                    const float d = __ldg(DELTA + grp);
                    float a[Q];
#pragma unroll
                    for (int j = 0; j < Q; ++j) a[j] = __fmul_rn(d, __ldg(ALPHA + grp * Q + j));
                    lvv = level_of<Q>(c, a, __fmul_rn(d, __fsub_rn(__ldg(ZB + grp), __ldg(ZU + grp))));
                }
                t.lv[k][c] = lvv;
            }
            __syncwarp();
#pragma unroll
            for (int e = lane; e < E; e += 32) {
                const int k = e / L, c = e % L;
                const float v = t.lv[k][c];
                int r = 0;
#pragma unroll
                for (int c2 = 0; c2 < L; ++c2) {
                    const float v2 = t.lv[k][c2];
                    r += (v2 < v) || (v2 == v && c2 < c);
                }
                t.srt[k][r] = v;
                t.cor[k][r] = static_cast<uint8_t>(c);
            }
            __syncwarp();
#pragma unroll
            for (int b = 0; b < WB; ++b) {
                if (!ok[b]) continue;
                const int k = b * GPS + (lane >> SH);
                float srt[L], w[4];
#pragma unroll
                for (int r = 0; r < L; ++r) srt[r] = t.srt[k][r];
                WT::unpack(wraw[b], w);
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    float m;
                    const int r = nearest_rank<L>(w[v], srt, m);
                    cw[b] |= uint32_t(t.cor[k][r]) << (8 * v);
                }
            }
        }
#pragma unroll
        for (int b = 0; b < WB; ++b) {
            const int ws = base + b * kWarps;
            if (ws >= n_ws) break;                           // warp-uniform
            uint32_t mine = 0;
#pragma unroll
            for (int tw = 0; tw < 4; ++tw) {
                // column 32*tw + lane of this warp-step lives in lane 8*tw + lane/4, byte lane%4
                const uint32_t v = (__shfl_sync(kFull, cw[b], 8 * tw + (lane >> 2)) >> (8 * (lane & 3))) & 0xffu;
#pragma unroll
                for (int j = 0; j < Q; ++j) {
                    const uint32_t word = __ballot_sync(kFull, (v >> j) & 1u);
                    if (lane == j * 4 + tw) mine = word;
                }
            }
            if (lane < 4 * Q) {
                const int j = lane >> 2, tw = lane & 3;
                const int wcol = ws * kStep + tw * 32;
                if (wcol < n_in) PLANES[((int64_t)j * out + row) * words + ws * 4 + tw] = mine;
            }
        }
    }
}

template <int Q, typename WT, int GPS, bool EQ4>
static cudaError_t run_export(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, uint32_t* planes,
                              float* astar, float* zstar, cudaStream_t st) {
    export_kernel<Q, WT, GPS, EQ4><<<dim3((unsigned)sh.out), kThreads, 0, st>>>(
        W, p.delta, p.zu, p.alpha, p.zb, codes, planes, astar, zstar, sh.out, sh.n_in, sh.g);
    return cudaGetLastError();
}

template <int Q, typename WT, bool EQ4>
static cudaError_t export_g(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, uint32_t* planes,
                            float* astar, float* zstar, cudaStream_t st) {
    if (sh.g == 32) return run_export<Q, WT, 4, EQ4>(sh, W, p, codes, planes, astar, zstar, st);
    if (sh.g == 64) return run_export<Q, WT, 2, EQ4>(sh, W, p, codes, planes, astar, zstar, st);
    return run_export<Q, WT, 1, EQ4>(sh, W, p, codes, planes, astar, zstar, st);
}

template <int Q>
static cudaError_t export_q(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                            uint32_t* planes, float* astar, float* zstar, cudaStream_t st) {
    if (mode == UQ_EXPORT_REUSE_CODES) return export_g<Q, WF32, false>(sh, W, p, codes, planes, astar, zstar, st);
    if (sh.wdtype == UQ_W_BF16) return export_g<Q, WBF16, true>(sh, W, p, codes, planes, astar, zstar, st);
    return export_g<Q, WF32, true>(sh, W, p, codes, planes, astar, zstar, st);
}

cudaError_t launch_export(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                          uint32_t* planes, float* astar, float* zstar, cudaStream_t st) {
    switch (sh.q) {
        case 1: return export_q<1>(sh, W, p, codes, mode, planes, astar, zstar, st);
        case 2: return export_q<2>(sh, W, p, codes, mode, planes, astar, zstar, st);
        case 3: return export_q<3>(sh, W, p, codes, mode, planes, astar, zstar, st);
        default: return export_q<4>(sh, W, p, codes, mode, planes, astar, zstar, st);
    }
}

}  // namespace uq
