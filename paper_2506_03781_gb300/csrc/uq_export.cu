// Export: unification theorem (Theorem 1) and bit-plane packing of the
// final binary codes (the last two steps of Algorithm 1).
//
// alpha* = Delta alpha, z_B* = Delta (z_B - z_U) per group.  The codes are
// the stored ones (REUSE) or the nearest level of Theta_B* to each original
// weight (Eq. 4).  One thread owns 32 consecutive columns of a row (one
// 32-bit word of every bit-plane): it reads their 32 code bytes with two
// 16-byte loads and gathers bit j of four bytes at a time with the
// carry-free product ((x >> j) & 0x01010101) * 0x01020408, whose top byte
// holds the four bits in order.  Consecutive threads write consecutive
// words.  HBM traffic per element: 1 (codes) or 2-4 (weights) read, q/8
// written, plus the group parameters.
#include <cuda_fp16.h>

#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

// alpha*, z_B* as fp32, or as IEEE half bits rounded to nearest even (the
// 16-bit reals of the storage count of App. F.1).
struct OutF32 {
    using T = float;
    static __device__ __forceinline__ T cvt(float v) { return v; }
};
struct OutF16 {
    using T = uint16_t;
    static __device__ __forceinline__ T cvt(float v) { return __half_as_ushort(__float2half_rn(v)); }
};

__device__ __forceinline__ uint32_t gather_bit(uint32_t four_codes, int j) {
    return (((four_codes >> j) & 0x01010101u) * 0x01020408u) >> 24;
}

template <int Q, typename WT, bool EQ4, typename OT>
__global__ void __launch_bounds__(kThreads)
export_kernel(const void* __restrict__ W, const float* __restrict__ DELTA, const float* __restrict__ ZU,
              const float* __restrict__ ALPHA, const float* __restrict__ ZB, const uint8_t* __restrict__ CODES,
              uint32_t* __restrict__ PLANES, typename OT::T* __restrict__ ASTAR, typename OT::T* __restrict__ ZSTAR,
              int64_t out, int n_in, int g) {
    constexpr int L = 1 << Q;
    constexpr uint32_t kMask = uint32_t(L - 1) * 0x01010101u;
    const int words = n_in / 32;
    const int Gr = n_in / g;
    const int64_t nthr = (int64_t)gridDim.x * blockDim.x;
    const int64_t tid = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;

    // Theorem 1 for every group.
    for (int64_t grp = tid; grp < out * Gr; grp += nthr) {
        const float d = __ldg(DELTA + grp);
#pragma unroll
        for (int j = 0; j < Q; ++j) ASTAR[grp * Q + j] = OT::cvt(__fmul_rn(d, __ldg(ALPHA + grp * Q + j)));
        ZSTAR[grp] = OT::cvt(__fmul_rn(d, __fsub_rn(__ldg(ZB + grp), __ldg(ZU + grp))));
    }

    if constexpr (!EQ4) {
        if ((words & 3) == 0) {
            // Four words per thread (128 columns): eight 16-byte loads of code
            // bytes in flight, one 16-byte store of four words per plane.
            const int quads = words >> 2;
            const int64_t qstep_rows = nthr / quads;
            const int qstep_cols = (int)(nthr - qstep_rows * quads);
            int64_t qrow = tid / quads;
            int qcol = (int)(tid - qrow * quads);
            for (int64_t ch = tid; ch < out * quads; ch += nthr) {
                const uint4* src = reinterpret_cast<const uint4*>(CODES + qrow * n_in + (int64_t)qcol * 128);
                uint4 a[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) a[k] = __ldg(src + k);
#pragma unroll
                for (int j = 0; j < Q; ++j) {
                    uint32_t wq[4];
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        const uint4 x = a[2 * h], y = a[2 * h + 1];
                        wq[h] = gather_bit(x.x & kMask, j) | (gather_bit(x.y & kMask, j) << 4) |
                                (gather_bit(x.z & kMask, j) << 8) | (gather_bit(x.w & kMask, j) << 12) |
                                (gather_bit(y.x & kMask, j) << 16) | (gather_bit(y.y & kMask, j) << 20) |
                                (gather_bit(y.z & kMask, j) << 24) | (gather_bit(y.w & kMask, j) << 28);
                    }
                    *reinterpret_cast<uint4*>(PLANES + ((int64_t)j * out + qrow) * words + (int64_t)qcol * 4) =
                        make_uint4(wq[0], wq[1], wq[2], wq[3]);
                }
                qrow += qstep_rows;
                qcol += qstep_cols;
                if (qcol >= quads) { qcol -= quads; ++qrow; }
            }
            return;
        }
    }

    // (row, wcol) of chunk ch = row * words + wcol, advanced by nthr chunks
    // per iteration without dividing inside the loop.
    const int64_t step_rows = nthr / words;
    const int step_cols = (int)(nthr - step_rows * words);
    int64_t row = tid / words;
    int wcol = (int)(tid - row * words);
    for (int64_t ch = tid; ch < out * words; ch += nthr) {
        const int64_t e0 = row * n_in + (int64_t)wcol * 32;
        uint32_t cw[8];
        if constexpr (!EQ4) {
            const uint4 a = __ldg(reinterpret_cast<const uint4*>(CODES + e0));
            const uint4 b = __ldg(reinterpret_cast<const uint4*>(CODES + e0 + 16));
            cw[0] = a.x & kMask; cw[1] = a.y & kMask; cw[2] = a.z & kMask; cw[3] = a.w & kMask;
            cw[4] = b.x & kMask; cw[5] = b.y & kMask; cw[6] = b.z & kMask; cw[7] = b.w & kMask;
        } else {
            // Levels of Theta_B* of this chunk's group (the fp32 values written above).
            const int64_t grp = row * Gr + (wcol * 32) / g;
            const float d = __ldg(DELTA + grp);
            float a[Q];
#pragma unroll
            for (int j = 0; j < Q; ++j) a[j] = __fmul_rn(d, __ldg(ALPHA + grp * Q + j));
            const float zs = __fmul_rn(d, __fsub_rn(__ldg(ZB + grp), __ldg(ZU + grp)));
            float lv[L];
            int rk[L];
#pragma unroll
            for (int c = 0; c < L; ++c) lv[c] = level_of<Q>(c, a, zs);
#pragma unroll
            for (int c = 0; c < L; ++c) {
                int r = 0;
#pragma unroll
                for (int c2 = 0; c2 < L; ++c2) r += (lv[c2] < lv[c]) || (lv[c2] == lv[c] && c2 < c);
                rk[c] = r;
            }
#pragma unroll
            for (int v = 0; v < 8; ++v) {
                float w[4];
                WT::unpack(WT::load(W, e0 + 4 * v), w);
                uint32_t packed = 0;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    // nearest level, ties to the lower rank (same result as a scan of the sorted levels)
                    float best = fabsf(__fsub_rn(w[k], lv[0]));
                    int bc = 0, br = rk[0];
#pragma unroll
                    for (int c = 1; c < L; ++c) {
                        const float dd = fabsf(__fsub_rn(w[k], lv[c]));
                        if (dd < best || (dd == best && rk[c] < br)) { best = dd; bc = c; br = rk[c]; }
                    }
                    packed |= uint32_t(bc) << (8 * k);
                }
                cw[v] = packed;
            }
        }
#pragma unroll
        for (int j = 0; j < Q; ++j) {
            uint32_t word = 0;
#pragma unroll
            for (int v = 0; v < 8; ++v) word |= gather_bit(cw[v], j) << (4 * v);
            PLANES[((int64_t)j * out + row) * words + wcol] = word;
        }
        row += step_rows;
        wcol += step_cols;
        if (wcol >= words) { wcol -= words; ++row; }
    }
}

static int export_grid(int64_t work) {
    const int sms = sm_count();
    const int64_t want = (work + kThreads - 1) / kThreads;
    const int64_t cap = (int64_t)sms * 8;
    return (int)(want < cap ? (want < 1 ? 1 : want) : cap);
}

template <int Q, typename WT, bool EQ4, typename OT>
static cudaError_t run_export(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, uint32_t* planes,
                              typename OT::T* astar, typename OT::T* zstar, cudaStream_t st) {
    const int64_t words = sh.n_in / 32;
    const int grid = export_grid(sh.out * (!EQ4 && (words & 3) == 0 ? words / 4 : words));
    export_kernel<Q, WT, EQ4, OT><<<grid, kThreads, 0, st>>>(W, p.delta, p.zu, p.alpha, p.zb, codes, planes, astar,
                                                             zstar, sh.out, sh.n_in, sh.g);
    return cudaGetLastError();
}

template <int Q, typename OT>
static cudaError_t export_q(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                            uint32_t* planes, typename OT::T* astar, typename OT::T* zstar, cudaStream_t st) {
    if (mode == UQ_EXPORT_REUSE_CODES)
        return run_export<Q, WF32, false, OT>(sh, W, p, codes, planes, astar, zstar, st);
    if (sh.wdtype == UQ_W_BF16) return run_export<Q, WBF16, true, OT>(sh, W, p, codes, planes, astar, zstar, st);
    return run_export<Q, WF32, true, OT>(sh, W, p, codes, planes, astar, zstar, st);
}

template <typename OT>
static cudaError_t export_any(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                              uint32_t* planes, typename OT::T* astar, typename OT::T* zstar, cudaStream_t st) {
    switch (sh.q) {
        case 1: return export_q<1, OT>(sh, W, p, codes, mode, planes, astar, zstar, st);
        case 2: return export_q<2, OT>(sh, W, p, codes, mode, planes, astar, zstar, st);
        case 3: return export_q<3, OT>(sh, W, p, codes, mode, planes, astar, zstar, st);
        default: return export_q<4, OT>(sh, W, p, codes, mode, planes, astar, zstar, st);
    }
}

cudaError_t launch_export(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                          uint32_t* planes, float* astar, float* zstar, cudaStream_t st) {
    return export_any<OutF32>(sh, W, p, codes, mode, planes, astar, zstar, st);
}

cudaError_t launch_export_half(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, int mode,
                               uint32_t* planes, uint16_t* astar, uint16_t* zstar, cudaStream_t st) {
    return export_any<OutF16>(sh, W, p, codes, mode, planes, astar, zstar, st);
}

}  // namespace uq
