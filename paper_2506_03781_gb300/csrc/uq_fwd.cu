// Forward quantizer: Q*_IF (Eq. 3, local and periodic mapping of
// Algorithm 4) and Q_IF (Eq. 2, full mapping), one thread block per row.
//
// Per warp and batch of warp-steps: the lanes issue their vector loads
// (W, s, codes, Delta, z_U) first, then build the batch's group tables in
// shared memory (levels, sorted order, neighbour triples), then map and
// reconstruct 4 elements each.  HBM traffic per element (bf16 W): remap
// step 2 + 4 + 1 read, 4 + 1 written; keep step 1 read, 4 written.
#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

template <int Q, typename WT, int GPS>
__global__ void __launch_bounds__(kThreads)
fwd_kernel(const void* __restrict__ W, const float* __restrict__ S, const float* __restrict__ SR,
           const float* __restrict__ DELTA, const float* __restrict__ ZU, const float* __restrict__ ALPHA,
           const float* __restrict__ ZB, uint8_t* __restrict__ CODES, float* __restrict__ WHAT,
           int n_in, int g, int mode) {
    constexpr int L = 1 << Q;
    constexpr int WB = kSlots / GPS;                      // warp-steps per batch
    constexpr int SH = GPS == 4 ? 3 : (GPS == 2 ? 4 : 5); // lane -> group within a warp-step
    __shared__ GroupTables<Q> tabs[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    GroupTables<Q>& t = tabs[warp];
    const int64_t row = blockIdx.x;
    const int n_ws = (n_in + kStep - 1) / kStep;
    const int Gr = n_in / g;
    const int64_t eoff = row * (int64_t)n_in;
    const int64_t goff = row * (int64_t)Gr;
    const bool need_x = mode != FWD_KEEP;
    const float sr = need_x ? __ldg(SR + row) : 0.f;

    for (int base = warp; base < n_ws; base += kWarps * WB) {
        typename WT::raw wraw[WB];
        float4 sv[WB];
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
                if (need_x) {
                    wraw[b] = WT::load(W, eoff + col[b]);
                    sv[b] = ldg4(S + eoff + col[b]);
                }
                if (mode != FWD_FULL) cv[b] = *reinterpret_cast<const uint32_t*>(CODES + eoff + col[b]);
            }
        }
        auto grp_of_slot = [&](int k) -> int64_t {
            return goff + ((base + (k / GPS) * kWarps) * kStep) / g + (k % GPS);
        };
        auto ok_of_slot = [&](int k) -> bool {
            const int ws = base + (k / GPS) * kWarps;
            return ws < n_ws && (ws * kStep) / g + (k % GPS) < Gr;
        };
        __syncwarp();   // the previous batch is done with the tables
        if (mode == FWD_FULL) build_tables<Q, true, false>(t, lane, ALPHA, ZB, grp_of_slot, ok_of_slot);
        else if (mode == FWD_REMAP) build_tables<Q, true, true>(t, lane, ALPHA, ZB, grp_of_slot, ok_of_slot);
        else build_tables<Q, false, false>(t, lane, ALPHA, ZB, grp_of_slot, ok_of_slot);

#pragma unroll
        for (int b = 0; b < WB; ++b) {
            if (!ok[b]) continue;
            const int k = b * GPS + (lane >> SH);
            float o[4];
            uint32_t nc = 0;
            if (mode == FWD_KEEP) {
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    const int c = (cv[b] >> (8 * v)) & (L - 1);
                    o[v] = __fmul_rn(dl[b], __fsub_rn(t.lv[k][c], zu[b]));
                }
            } else {
                float w[4], s[4];
                WT::unpack(wraw[b], w);
                f4_to(sv[b], s);
                if (mode == FWD_REMAP) {
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        const int c = (cv[b] >> (8 * v)) & (L - 1);
                        const float4 nb = t.nb[k][c];
                        float u;
                        const float x = transform_x(w[v], s[v], dl[b], sr, zu[b], u);
                        const uint32_t packed = __float_as_uint(nb.w);
                        float best = fabsf(__fsub_rn(x, nb.y));
                        float m = nb.y;
                        uint32_t code = c;
                        const float dlo = fabsf(__fsub_rn(x, nb.x));
                        if (dlo < best) { best = dlo; m = nb.x; code = packed & 0xffu; }
                        const float dhi = fabsf(__fsub_rn(x, nb.z));
                        if (dhi < best) { best = dhi; m = nb.z; code = (packed >> 8) & 0xffu; }
                        o[v] = __fmul_rn(dl[b], __fsub_rn(m, zu[b]));
                        nc |= code << (8 * v);
                    }
                } else {
                    float srt[L];
#pragma unroll
                    for (int r = 0; r < L; ++r) srt[r] = t.srt[k][r];
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        float u, m;
                        const float x = transform_x(w[v], s[v], dl[b], sr, zu[b], u);
                        const int r = nearest_rank<L>(x, srt, m);
                        o[v] = __fmul_rn(dl[b], __fsub_rn(m, zu[b]));
                        nc |= uint32_t(t.cor[k][r]) << (8 * v);
                    }
                }
                *reinterpret_cast<uint32_t*>(CODES + eoff + col[b]) = nc;
            }
            *reinterpret_cast<float4*>(WHAT + eoff + col[b]) = make_float4(o[0], o[1], o[2], o[3]);
        }
    }
}

template <int Q, typename WT, int GPS>
static cudaError_t run_fwd(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                           cudaStream_t st) {
    fwd_kernel<Q, WT, GPS><<<dim3((unsigned)sh.out), kThreads, 0, st>>>(
        W, p.s, p.sr, p.delta, p.zu, p.alpha, p.zb, codes, what, sh.n_in, sh.g, mode);
    return cudaGetLastError();
}

template <int Q, typename WT>
static cudaError_t fwd_g(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                         cudaStream_t st) {
    if (sh.g == 32) return run_fwd<Q, WT, 4>(sh, W, p, codes, mode, what, st);
    if (sh.g == 64) return run_fwd<Q, WT, 2>(sh, W, p, codes, mode, what, st);
    return run_fwd<Q, WT, 1>(sh, W, p, codes, mode, what, st);
}

template <int Q>
static cudaError_t fwd_w(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                         cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return fwd_g<Q, WBF16>(sh, W, p, codes, mode, what, st);
    return fwd_g<Q, WF32>(sh, W, p, codes, mode, what, st);
}

cudaError_t launch_fwd(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                       cudaStream_t st) {
    switch (sh.q) {
        case 1: return fwd_w<1>(sh, W, p, codes, mode, what, st);
        case 2: return fwd_w<2>(sh, W, p, codes, mode, what, st);
        case 3: return fwd_w<3>(sh, W, p, codes, mode, what, st);
        default: return fwd_w<4>(sh, W, p, codes, mode, what, st);
    }
}

}  // namespace uq
