// Forward quantizer: Q*_IF (Eq. 3, local and periodic mapping of
// Algorithm 4) and Q_IF (Eq. 2, full mapping).
//
// Per warp and work unit (NG whole groups, see uq_common.cuh): the lanes
// issue their vector loads (W, s, codes) first, then build the unit's group
// tables in shared memory (levels by code word; for mapping steps also the
// sorted order and the local-mapping neighbour triples), then map and
// reconstruct their elements.  HBM traffic per element (bf16 W): remap step
// 2 + 4 + 1 read, 4 + 1 written; keep step 1 read, 4 written; full mapping
// 2 + 4 read, 4 + 1 written.
#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

// Minimum resident blocks per SM the register allocation is bounded for.
#ifndef UQ_FWD_MIN_BLOCKS
#define UQ_FWD_MIN_BLOCKS 3
#endif

template <int Q, typename WT, int LPG>
__global__ void __launch_bounds__(kThreads, UQ_FWD_MIN_BLOCKS)
fwd_kernel(const void* __restrict__ W, const float* __restrict__ S, const float* __restrict__ SR,
           const float* __restrict__ DELTA, const float* __restrict__ ZU, const float* __restrict__ ALPHA,
           const float* __restrict__ ZB, uint8_t* __restrict__ CODES, float* __restrict__ WHAT, int64_t out,
           int n_in, int g, int R, int mode) {
    constexpr int L = 1 << Q;
    constexpr int NG = 32 / LPG;
    __shared__ MapTab<Q, NG> tabs[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    MapTab<Q, NG>& t = tabs[warp];
    const int WPR = kWarps / R;
    const int64_t row = (int64_t)blockIdx.x * R + warp / WPR;
    if (row >= out) return;                      // no block barrier in this kernel
    const int wr = warp % WPR;
    const int Gr = n_in / g;
    const int units = (Gr + NG - 1) / NG;
    const int nv = g / (4 * LPG);
    const int sub = lane / LPG, li = lane % LPG;
    const bool need_x = mode != FWD_KEEP;
    const float sr = need_x ? __ldg(SR + row) : 0.f;
    const int64_t rbase = row * (int64_t)n_in;

    for (int u = wr; u < units; u += WPR) {
        const int gi = u * NG + sub;
        const bool ok = gi < Gr;
        const int64_t grp = row * Gr + gi;
        const int64_t ebase = rbase + (int64_t)gi * g + 4 * li;
        typename WT::raw wr4[4];
        float4 sv[4];
        uint32_t cv[4];
        auto load_chunk = [&](int c0) {
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                if (ok && c0 + v < nv) {
                    const int64_t e = ebase + 4 * LPG * (c0 + v);
                    if (need_x) {
                        wr4[v] = WT::load(W, e);
                        sv[v] = ldg4(S + e);
                    }
                    if (mode != FWD_FULL) cv[v] = *reinterpret_cast<const uint32_t*>(CODES + e);
                }
            }
        };
        load_chunk(0);
        float dl = 0.f, zu = 0.f;
        if (ok) {
            dl = __ldg(DELTA + grp);
            zu = __ldg(ZU + grp);
        }
        __syncwarp();
        unit_levels<Q, NG>(t, (float*)nullptr, lane, ALPHA, ZB, row * Gr + u * NG, min(NG, Gr - u * NG));
        if (mode == FWD_REMAP) unit_sort<Q, NG, true>(t, lane);
        else if (mode == FWD_FULL) unit_sort<Q, NG, false>(t, lane);
        float srt[L];
        if (mode == FWD_FULL) {
#pragma unroll
            for (int r = 0; r < L; ++r) srt[r] = t.srt[sub][r];
        }
        for (int c0 = 0; c0 < nv; c0 += 4) {
            if (c0 > 0) load_chunk(c0);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                if (!(ok && c0 + v < nv)) continue;
                const int64_t e = ebase + 4 * LPG * (c0 + v);
                float o[4];
                uint32_t nc = 0;
                if (mode == FWD_KEEP) {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const int c = (cv[v] >> (8 * k)) & (L - 1);
                        o[k] = __fmul_rn(dl, __fsub_rn(t.lv[sub][c], zu));
                    }
                } else {
                    float w[4], s[4];
                    WT::unpack(wr4[v], w);
                    f4_to(sv[v], s);
                    if (mode == FWD_REMAP) {
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const int c = (cv[v] >> (8 * k)) & (L - 1);
                            const float4 nb = t.nb[sub][c];
                            float uu;
                            const float x = transform_x(w[k], s[k], dl, sr, zu, uu);
                            const uint32_t packed = __float_as_uint(nb.w);
                            float best = fabsf(__fsub_rn(x, nb.y));
                            float m = nb.y;
                            uint32_t code = c;
                            const float dlo = fabsf(__fsub_rn(x, nb.x));
                            if (dlo < best) { best = dlo; m = nb.x; code = packed & 0xffu; }
                            const float dhi = fabsf(__fsub_rn(x, nb.z));
                            if (dhi < best) { m = nb.z; code = (packed >> 8) & 0xffu; }
                            o[k] = __fmul_rn(dl, __fsub_rn(m, zu));
                            nc |= code << (8 * k);
                        }
                    } else {
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            float uu, m;
                            const float x = transform_x(w[k], s[k], dl, sr, zu, uu);
                            const int r = nearest_rank<L>(x, srt, m);
                            o[k] = __fmul_rn(dl, __fsub_rn(m, zu));
                            nc |= uint32_t(t.cor[sub][r]) << (8 * k);
                        }
                    }
                    *reinterpret_cast<uint32_t*>(CODES + e) = nc;
                }
                *reinterpret_cast<float4*>(WHAT + e) = make_float4(o[0], o[1], o[2], o[3]);
            }
        }
    }
}

template <int Q, typename WT, int LPG>
static cudaError_t run_fwd(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                           cudaStream_t st) {
    constexpr int NG = 32 / LPG;
    const int Gr = sh.n_in / sh.g;
    const int R = rows_per_block((Gr + NG - 1) / NG);
    const int64_t blocks = (sh.out + R - 1) / R;
    fwd_kernel<Q, WT, LPG><<<dim3((unsigned)blocks), kThreads, 0, st>>>(
        W, p.s, p.sr, p.delta, p.zu, p.alpha, p.zb, codes, what, sh.out, sh.n_in, sh.g, R, mode);
    return cudaGetLastError();
}

template <int Q, typename WT>
static cudaError_t fwd_g(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                         cudaStream_t st) {
    switch (lanes_per_group(sh.g)) {
        case 4: return run_fwd<Q, WT, 4>(sh, W, p, codes, mode, what, st);
        case 8: return run_fwd<Q, WT, 8>(sh, W, p, codes, mode, what, st);
        case 16: return run_fwd<Q, WT, 16>(sh, W, p, codes, mode, what, st);
        default: return run_fwd<Q, WT, 32>(sh, W, p, codes, mode, what, st);
    }
}

template <int Q>
static cudaError_t fwd_w(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                         cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return fwd_g<Q, WBF16>(sh, W, p, codes, mode, what, st);
    return fwd_g<Q, WF32>(sh, W, p, codes, mode, what, st);
}

cudaError_t launch_fwd(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                       cudaStream_t st) {
    if (stream_path_ok(sh)) return launch_fwd_stream(sh, W, p, codes, mode, what, st);
    switch (sh.q) {
        case 1: return fwd_w<1>(sh, W, p, codes, mode, what, st);
        case 2: return fwd_w<2>(sh, W, p, codes, mode, what, st);
        case 3: return fwd_w<3>(sh, W, p, codes, mode, what, st);
        default: return fwd_w<4>(sh, W, p, codes, mode, what, st);
    }
}

}  // namespace uq
