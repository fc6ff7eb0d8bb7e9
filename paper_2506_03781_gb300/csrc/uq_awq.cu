// UniQuan with AWQ's transformation (App. E, extensibility): the BCQ
// mapping, levels and gradient filter of UniQuan_F with
//   T_A(w) = (w s_A) / Delta_A + z_A,   D_A(w~) = Delta_A (w~ - z_A) / s_A,
// s_A one scale per column (shared by every row), Delta_A and z_A per group.
//
// Decomposition: column stripes x row ranges.  Thread block (cb, rb) has 8
// warps; warp w owns work unit cb * 8 + w (NG whole groups, the lane mapping
// of uq_common.cuh, every lane holding all of its group elements: g <= 512)
// and walks the rows of range rb one after the other.  The unit's s_A is
// loaded once.  The backward writes the per-row group gradients directly and
// accumulates ds_A of its columns over its rows in registers; the range's
// partials go to a workspace [row range][in] and a second kernel sums them in
// range order.  Deterministic, no atomics.  HBM traffic per element (bf16 W):
// forward remap 2 + 1 read, 4 + 1 written; backward 2 + 1 + 4 read.  The
// forward steps that map run on the pipelined skeleton instead (below) for
// g in {32, 64, 128} and rows of whole work units.
#include "uq_common.cuh"
#include "uq_launch.h"
#include "uq_pipe.cuh"

namespace uq {

#ifndef UQ_AWQ_MIN_BLOCKS
#define UQ_AWQ_MIN_BLOCKS 3
#endif
#ifndef UQ_AWQ_BWD_MIN_BLOCKS
#define UQ_AWQ_BWD_MIN_BLOCKS 2          // the backward also keeps the unit's s_A and ds_A partials in registers
#endif

constexpr int kAwqTargetBlocksPerSm = 4;

template <int Q, typename WT, int LPG, int MODE>
__global__ void __launch_bounds__(kThreads, UQ_AWQ_MIN_BLOCKS)
awq_fwd_kernel(const void* __restrict__ W, const float* __restrict__ SA, const float* __restrict__ DELTA,
               const float* __restrict__ ZA, const float* __restrict__ ALPHA, const float* __restrict__ ZB,
               uint8_t* __restrict__ CODES, float* __restrict__ WHAT, int64_t out, int n_in, int g,
               int64_t rows_per_range) {
    constexpr int L = 1 << Q;
    constexpr int NG = 32 / LPG;
    __shared__ MapTab<Q, NG> tabs[kWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    MapTab<Q, NG>& t = tabs[warp];
    const int Gr = n_in / g;
    const int u = blockIdx.x * kWarps + warp;
    if (u * NG >= Gr) return;                     // no block barrier in this kernel
    const int64_t r0 = (int64_t)blockIdx.y * rows_per_range;
    const int64_t r1 = r0 + rows_per_range < out ? r0 + rows_per_range : out;
    const int nv = g / (4 * LPG);
    const int sub = lane / LPG, li = lane % LPG;
    const int gi = u * NG + sub;
    const bool ok = gi < Gr;
    const int64_t cbase = (int64_t)gi * g + 4 * li;       // first column of this lane's vector 0
    float s[4][4];
#pragma unroll
    for (int v = 0; v < 4; ++v)
        if (ok && v < nv) f4_to(ldg4(SA + cbase + 4 * LPG * v), s[v]);

    for (int64_t row = r0; row < r1; ++row) {
        const int64_t grp = row * Gr + gi;
        const int64_t ebase = row * (int64_t)n_in + cbase;
        float w[4][4];
        uint32_t cv[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            if (ok && v < nv) {
                const int64_t e = ebase + 4 * LPG * v;
                if (MODE != FWD_KEEP) WT::unpack(WT::load(W, e), w[v]);
                if (MODE != FWD_FULL) cv[v] = *reinterpret_cast<const uint32_t*>(CODES + e);
            }
        }
        const float dl = ok ? __ldg(DELTA + grp) : 1.f, za = ok ? __ldg(ZA + grp) : 0.f;
        __syncwarp();                             // previous row is done with the tables
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
                float m;
                uint32_t code;
                if (MODE == FWD_KEEP) {
                    code = (cv[v] >> (8 * k)) & (L - 1);
                    m = t.lv[sub][code];
                } else {
                    const float x = __fadd_rn(__fdiv_rn(__fmul_rn(w[v][k], s[v][k]), dl), za);
                    if (MODE == FWD_REMAP) {
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
                }
                o[k] = __fdiv_rn(__fmul_rn(dl, __fsub_rn(m, za)), s[v][k]);
                nc |= code << (8 * k);
            }
            if (MODE != FWD_KEEP) *reinterpret_cast<uint32_t*>(CODES + e) = nc;
            *reinterpret_cast<float4*>(WHAT + e) = make_float4(o[0], o[1], o[2], o[3]);
        }
    }
}

template <int Q, typename WT, int LPG>
__global__ void __launch_bounds__(kThreads, UQ_AWQ_BWD_MIN_BLOCKS)
awq_bwd_kernel(const void* __restrict__ W, const float* __restrict__ SA, const float* __restrict__ DELTA,
               const float* __restrict__ ZA, const float* __restrict__ ALPHA, const float* __restrict__ ZB,
               const uint8_t* __restrict__ CODES, const float* __restrict__ GUP, float* __restrict__ DDELTA,
               float* __restrict__ DZA, float* __restrict__ DALPHA, float* __restrict__ DZB,
               float* __restrict__ PART, int64_t out, int n_in, int g, int64_t rows_per_range) {
    constexpr int L = 1 << Q;
    constexpr int NG = 32 / LPG;
    using SR8 = SegReduce<LPG>;
    __shared__ LvTab<Q, NG> tabs[kWarps];
    __shared__ float tau_s[kWarps][NG];
    __shared__ float amag_s[kWarps][NG];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    LvTab<Q, NG>& t = tabs[warp];
    const int Gr = n_in / g;
    const int u = blockIdx.x * kWarps + warp;
    if (u * NG >= Gr) return;                     // no block barrier in this kernel
    const int64_t r0 = (int64_t)blockIdx.y * rows_per_range;
    const int64_t r1 = r0 + rows_per_range < out ? r0 + rows_per_range : out;
    const int nv = g / (4 * LPG);
    const int sub = lane / LPG, li = lane % LPG;
    const int gi = u * NG + sub;
    const bool ok = gi < Gr;
    const int64_t cbase = (int64_t)gi * g + 4 * li;
    // s_A of the unit's columns and its reciprocal, once: only x (the filter
    // decision) needs the exact division; the gradient values take 1/s_A.
    float s[4][4], rs[4][4], dsa[4][4];
#pragma unroll
    for (int v = 0; v < 4; ++v) {
#pragma unroll
        for (int k = 0; k < 4; ++k) dsa[v][k] = 0.f;
        if (ok && v < nv) {
            f4_to(ldg4(SA + cbase + 4 * LPG * v), s[v]);
#pragma unroll
            for (int k = 0; k < 4; ++k) rs[v][k] = 1.f / s[v][k];
        }
    }

    for (int64_t row = r0; row < r1; ++row) {
        const int64_t grp = row * Gr + gi;
        const int64_t ebase = row * (int64_t)n_in + cbase;
        float w[4][4], G[4][4];
        uint32_t cv[4] = {0u, 0u, 0u, 0u};
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            if (ok && v < nv) {
                const int64_t e = ebase + 4 * LPG * v;
                WT::unpack(WT::load(W, e), w[v]);
                f4_to(ldg4(GUP + e), G[v]);
                cv[v] = __ldg(reinterpret_cast<const unsigned int*>(CODES + e));
            }
        }
        const float dl = ok ? __ldg(DELTA + grp) : 1.f, za = ok ? __ldg(ZA + grp) : 0.f;
        __syncwarp();                             // previous row is done with the tables
        unit_levels<Q, NG>(t, tau_s[warp], lane, ALPHA, ZB, row * Gr + u * NG, min(NG, Gr - u * NG), amag_s[warp]);
        const float tau = tau_s[warp][sub];
        // x = (w s_A) / Delta_A + z_A: one reciprocal of Delta_A per group, the
        // filter proven equal to the IEEE one (shared_div_filter4)
        const float rdl = rcp_approx(dl);
        const float eg = ok ? bwd_margin_of(__fadd_rn(fabsf(za), amag_s[warp][sub]), dl) : 0.f;
        float acc[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = 0.f;
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            if (!(ok && v < nv)) continue;
            float ws[4], m4[4], uv[4];
            bool fv[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                ws[k] = __fmul_rn(w[v][k], s[v][k]);
                m4[k] = t.lv[sub][(cv[v] >> (8 * k)) & (L - 1)];
            }
            shared_div_filter4(ws, dl, rdl, za, m4, tau, eg, uv, fv);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int c = (cv[v] >> (8 * k)) & (L - 1);
                const float m = m4[k];
                const float uu = uv[k];
                const bool f = fv[k];
                const float gs = G[v][k] * rs[v][k];
                const float mz = m - za;
                acc[0] += gs * (mz - (f ? uu : 0.f));
                acc[1] += f ? 0.f : gs;
                acc[2] += gs;
#pragma unroll
                for (int j = 0; j < Q; ++j) acc[4 + j] += ((c >> j) & 1) ? gs : -gs;
                dsa[v][k] += gs * ((f ? w[v][k] : 0.f) - dl * mz * rs[v][k]);
            }
        }
        const int slot0 = SR8::run(acc, lane);
        if (ok && SR8::writer(lane)) {
#pragma unroll
            for (int i = 0; i < SR8::NOUT; ++i) {
                const int slot = slot0 + i;
                const float tot = acc[i];
                if (slot == 0) DDELTA[grp] = tot;
                else if (slot == 1) DZA[grp] = -(dl * tot);
                else if (slot == 2) DZB[grp] = dl * tot;
                else if (slot >= 4 && slot - 4 < Q) DALPHA[grp * Q + (slot - 4)] = dl * tot;
            }
        }
    }
    // this row range's ds_A partials of the unit's columns
    float* prow = PART + (int64_t)blockIdx.y * n_in + cbase;
#pragma unroll
    for (int v = 0; v < 4; ++v)
        if (ok && v < nv)
            *reinterpret_cast<float4*>(prow + 4 * LPG * v) = make_float4(dsa[v][0], dsa[v][1], dsa[v][2], dsa[v][3]);
}

// ---------------------------------------------------------------------------
// Pipelined forward (g in {32, 64, 128}, rows of whole work units)
// ---------------------------------------------------------------------------
//
// The persistent TMA-pipelined skeleton of uq_pipe.cuh: every warp streams
// its (row block, unit) items through a ring of shared-memory stages, with
// bounded mbarrier waits (a wait that runs out sets g_awq_err, reported by
// uq_check_device).  A stage holds the weights (not on keep steps), s_A of
// the unit's columns in the s slot (the same for every row, so it comes from
// L2 after the first rows), the code words (not for the full mapping) and
// Delta_A, z_A, z_B, alpha in the Delta, z_U, z_B, alpha slots.  Only the
// steps that map (remap, full) use it.

__device__ unsigned int g_awq_err = 0;

#ifndef UQ_AWQ_FWD_STAGE_BYTES
#define UQ_AWQ_FWD_STAGE_BYTES 5632
#endif

template <int Q, typename WT, int G_, int MODE>
using AwqFwdStage = Stage<Q, WT, G_, MODE != FWD_KEEP, false, MODE != FWD_FULL, UQ_AWQ_FWD_STAGE_BYTES, true>;

template <typename St, int KIND>
struct AwqTag {};

template <int Q, typename St>
__device__ __forceinline__ void awq_issue(const Items& it, const Cursor& c, int s, uint32_t bar, unsigned char* wsm,
                                          const void* W, const float* SA, const uint8_t* CODES, const float* DELTA,
                                          const float* ZA, const float* ZB, const float* ALPHA, int64_t out, int n_in,
                                          int Gr) {
    const int64_t row = it.row(c.k);
    if (row >= out) { tma::bar_arrive(bar); return; }
    const int64_t col0 = (int64_t)it.unit(c.j) * St::UE;
    const int64_t e0 = row * n_in + col0;
    const int64_t g0 = row * Gr + (int64_t)it.unit(c.j) * St::NG;
    const uint32_t d = tma::smem_addr(wsm + (size_t)s * St::BYTES);
    tma::fence_async_smem();
    tma::bar_arrive_tx(bar, St::TX);
    if constexpr (St::SZ_W > 0)
        tma::copy_g2s(d + St::OFF_W, static_cast<const unsigned char*>(W) + e0 * St::WBYTES, St::SZ_W, bar);
    tma::copy_g2s(d + St::OFF_S, SA + col0, St::SZ_S, bar);
    if constexpr (St::SZ_C > 0) tma::copy_g2s(d + St::OFF_C, CODES + e0, St::SZ_C, bar);
    tma::copy_g2s(d + St::OFF_D, DELTA + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_Z, ZA + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_B, ZB + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_A, ALPHA + g0 * Q, St::SZ_A, bar);
}

template <int Q, typename WT, int G_, int MODE>
__global__ void __launch_bounds__(kThreads, 3)
awq_stream_fwd_kernel(const void* __restrict__ W, const float* __restrict__ SA, const float* __restrict__ DELTA,
                      const float* __restrict__ ZA, const float* __restrict__ ALPHA, const float* __restrict__ ZB,
                      uint8_t* __restrict__ CODES, float* __restrict__ WHAT, int64_t out, int n_in, int R, int n_rb) {
    using St = AwqFwdStage<Q, WT, G_, MODE>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NV = St::NV, UE = St::UE, NST = St::NST;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][NST];
    __shared__ MapTab<Q, NG> tabs[kWarps];
    constexpr int NIV = MODE == FWD_REMAP ? NG : 1;              // remap intervals only on remap steps
    __shared__ float4 ivs[kWarps][NIV][L];
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
        awq_issue<Q, St>(it, c, s, tma::smem_addr(&bars[warp][s]), wsm, W, SA, CODES, DELTA, ZA, ZB, ALPHA, out, n_in,
                         Gr);
    };
    const bool ok = pipe_run<NST>(it, bars[warp], lane, &g_awq_err, 1u, issue,
                                  [&](const Cursor& cc, int s) {
        const int64_t row = it.row(cc.k);
        if (row < out) {
            const unsigned char* st = wsm + (size_t)s * St::BYTES;
            const float* pd = reinterpret_cast<const float*>(st + St::OFF_D);
            const float* pz = reinterpret_cast<const float*>(st + St::OFF_Z);
            const float* pb = reinterpret_cast<const float*>(st + St::OFF_B);
            const float* pa = reinterpret_cast<const float*>(st + St::OFF_A);
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
                unit_sort<Q, NG, false>(t, lane);
                unit_remap_iv<Q, NG>(t, ivs[warp], lane, pd, pz);
            } else if constexpr (MODE == FWD_FULL) {
                unit_sort<Q, NG, false>(t, lane);
            }
            const float dl = pd[sub], za = pz[sub];
            const int64_t ebase = row * n_in + (int64_t)it.unit(cc.j) * UE;
            float srt[L];
            if constexpr (MODE == FWD_FULL) {
#pragma unroll
                for (int r = 0; r < L; ++r) srt[r] = t.srt[sub][r];
            }
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                float s4[4], w[4];
                f4_to(*reinterpret_cast<const float4*>(st + St::OFF_S + el * 4), s4);
                if constexpr (MODE != FWD_KEEP)
                    WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w);
                uint32_t cv = 0u;
                if constexpr (MODE != FWD_FULL) cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                float o[4];
                uint32_t nc = 0;
                if constexpr (MODE == FWD_REMAP) {
                    // x = (w s_A) / Delta_A + z_A: the interval test on the numerator w s_A
                    // with s = s_r = 1; W^ = (Delta_A (l - z_A)) / s_A
                    const float one[4] = {1.f, 1.f, 1.f, 1.f};
                    float nu[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) nu[k] = __fmul_rn(w[k], s4[k]);
                    nc = remap_vec4<Q, NG>(nu, one, cv, t, ivs[warp], sub, dl, 1.f, za, o);
#pragma unroll
                    for (int k = 0; k < 4; ++k) o[k] = __fdiv_rn(o[k], s4[k]);
                } else {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        float m;
                        uint32_t code;
                        if constexpr (MODE == FWD_KEEP) {
                            code = (cv >> (8 * k)) & (L - 1);
                            m = t.lv[sub][code];
                        } else {
                            const float x = __fadd_rn(__fdiv_rn(__fmul_rn(w[k], s4[k]), dl), za);
                            const int r = nearest_rank<L>(x, srt, m);
                            code = t.cor[sub][r];
                        }
                        o[k] = __fdiv_rn(__fmul_rn(dl, __fsub_rn(m, za)), s4[k]);
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

template <int Q, typename WT, int G_, int MODE>
static cudaError_t run_awq_stream_fwd(const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes, float* what,
                                      cudaStream_t st) {
    using St = AwqFwdStage<Q, WT, G_, MODE>;
    const int U = sh.n_in / St::UE;
    const int R = rows_per_block(U);
    const int n_rb = (int)((sh.out + R - 1) / R);
    const size_t dyn = (size_t)kWarps * St::WARP_BYTES;
    auto kern = awq_stream_fwd_kernel<Q, WT, G_, MODE>;
    int grid = 0;
    cudaError_t e = grid_for<AwqTag<St, MODE>>(kern, dyn, n_rb, grid);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, dyn, st>>>(W, p.sa, p.delta, p.za, p.alpha, p.zb, codes, what, sh.out, sh.n_in, R, n_rb);
    return cudaGetLastError();
}

template <int Q, typename WT, int G_>
static cudaError_t awq_stream_fwd_g(int mode, const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes,
                                    float* what, cudaStream_t st) {
    if (mode == FWD_REMAP) return run_awq_stream_fwd<Q, WT, G_, FWD_REMAP>(sh, W, p, codes, what, st);
    return run_awq_stream_fwd<Q, WT, G_, FWD_FULL>(sh, W, p, codes, what, st);
}

template <int Q, typename WT>
static cudaError_t awq_stream_fwd(int mode, const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes,
                                  float* what, cudaStream_t st) {
    if (sh.g == 32) return awq_stream_fwd_g<Q, WT, 32>(mode, sh, W, p, codes, what, st);
    if (sh.g == 64) return awq_stream_fwd_g<Q, WT, 64>(mode, sh, W, p, codes, what, st);
    return awq_stream_fwd_g<Q, WT, 128>(mode, sh, W, p, codes, what, st);
}

// ---------------------------------------------------------------------------
// Pipelined backward (rows of at most kWarps work units)
// ---------------------------------------------------------------------------
//
// ds_A sums down each column.  When a row holds at most kWarps work units,
// every warp of a block owns one fixed unit (one set of columns) for the
// whole kernel, so its ds_A partials and 1/s_A stay in registers across all
// of its rows; at the end each (block, row slot) writes one row of partials
// to the workspace [grid * R][in], summed by awq_colsum_kernel in a fixed
// order (contiguous slices of the rows in order, then the slices in order).
// Deterministic for a given grid.  The stage holds W, s_A of the unit's
// columns (s slot), dL/dW^, the codes and Delta_A, z_A, z_B, alpha.

constexpr int kAwqStreamBwdBlocksPerSm = 2;
#ifndef UQ_AWQ_BWD_STAGE_BYTES
#define UQ_AWQ_BWD_STAGE_BYTES 11520
#endif

template <int Q, typename WT, int G_>
using AwqBwdStage = Stage<Q, WT, G_, true, true, true, UQ_AWQ_BWD_STAGE_BYTES, true>;

static bool awq_stream_bwd_ok(const Shape& sh) {
    if (!stream_path_ok(sh)) return false;
    return sh.n_in / (sh.g == 32 ? 256 : 512) <= kWarps;
}

// Rows per block, row blocks and the grid of the pipelined backward (the
// grid is bounded by the SM count only, so the workspace size is known).
static void awq_stream_bwd_grid(const Shape& sh, int& R, int& n_rb, int& grid) {
    const int U = sh.n_in / (sh.g == 32 ? 256 : 512);
    R = rows_per_block(U);
    n_rb = (int)((sh.out + R - 1) / R);
    const int cap = sm_count() * kAwqStreamBwdBlocksPerSm;
    grid = n_rb < cap ? n_rb : cap;
}

template <int Q, typename St>
__device__ __forceinline__ void awq_bwd_issue(const Items& it, const Cursor& c, int s, uint32_t bar,
                                              unsigned char* wsm, const void* W, const float* SA, const float* GUP,
                                              const uint8_t* CODES, const float* DELTA, const float* ZA,
                                              const float* ZB, const float* ALPHA, int64_t out, int n_in, int Gr) {
    const int64_t row = it.row(c.k);
    if (row >= out) { tma::bar_arrive(bar); return; }
    const int64_t col0 = (int64_t)it.unit(c.j) * St::UE;
    const int64_t e0 = row * n_in + col0;
    const int64_t g0 = row * Gr + (int64_t)it.unit(c.j) * St::NG;
    const uint32_t d = tma::smem_addr(wsm + (size_t)s * St::BYTES);
    tma::fence_async_smem();
    tma::bar_arrive_tx(bar, St::TX);
    tma::copy_g2s(d + St::OFF_W, static_cast<const unsigned char*>(W) + e0 * St::WBYTES, St::SZ_W, bar);
    tma::copy_g2s(d + St::OFF_S, SA + col0, St::SZ_S, bar);
    tma::copy_g2s(d + St::OFF_G, GUP + e0, St::SZ_G, bar);
    tma::copy_g2s(d + St::OFF_C, CODES + e0, St::SZ_C, bar);
    tma::copy_g2s(d + St::OFF_D, DELTA + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_Z, ZA + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_B, ZB + g0, St::SZ_P, bar);
    tma::copy_g2s(d + St::OFF_A, ALPHA + g0 * Q, St::SZ_A, bar);
}

template <int Q, typename WT, int G_>
__global__ void __launch_bounds__(kThreads, kAwqStreamBwdBlocksPerSm)
awq_stream_bwd_kernel(const void* __restrict__ W, const float* __restrict__ SA, const float* __restrict__ DELTA,
                      const float* __restrict__ ZA, const float* __restrict__ ALPHA, const float* __restrict__ ZB,
                      const uint8_t* __restrict__ CODES, const float* __restrict__ GUP, float* __restrict__ DDELTA,
                      float* __restrict__ DZA, float* __restrict__ DALPHA, float* __restrict__ DZB,
                      float* __restrict__ PART, int64_t out, int n_in, int R, int n_rb) {
    using St = AwqBwdStage<Q, WT, G_>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NV = St::NV, UE = St::UE, NST = St::NST;
    using SR8 = SegReduce<LPG>;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][NST];
    __shared__ float2 tabs[kWarps][NG][L];          // (l(c), l(c) - z_A) per group slot and code word
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / LPG, li = lane % LPG;
    const int U = n_in / UE, Gr = n_in / G_;
    const Items it(U, R, n_rb, warp);               // n_w <= 1: the warp's unit is it.unit(0)
    unsigned char* wsm = smem + (size_t)warp * St::WARP_BYTES;

    if (lane == 0) {
        for (int s = 0; s < NST; ++s) tma::bar_init(tma::smem_addr(&bars[warp][s]), 1);
        tma::bar_init_fence();
    }
    __syncwarp();
    auto issue = [&](const Cursor& c, int s) {          // lane 0 only
        awq_bwd_issue<Q, St>(it, c, s, tma::smem_addr(&bars[warp][s]), wsm, W, SA, GUP, CODES, DELTA, ZA, ZB, ALPHA,
                             out, n_in, Gr);
    };
    float rs[NV][4], dsa[NV][4];
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int k = 0; k < 4; ++k) { rs[v][k] = 0.f; dsa[v][k] = 0.f; }
    bool have_rs = false;
    const bool ok = pipe_run<NST>(it, bars[warp], lane, &g_awq_err, 2u, issue,
                                  [&](const Cursor& cc, int s) {
        const int64_t row = it.row(cc.k);
        if (row < out) {
            const unsigned char* st = wsm + (size_t)s * St::BYTES;
            const float* pd = reinterpret_cast<const float*>(st + St::OFF_D);
            const float* pz = reinterpret_cast<const float*>(st + St::OFF_Z);
            const float* pb = reinterpret_cast<const float*>(st + St::OFF_B);
            const float* pa = reinterpret_cast<const float*>(st + St::OFF_A);
            if (!have_rs) {                              // 1/s_A of the warp's columns, once
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    float s4[4];
                    f4_to(*reinterpret_cast<const float4*>(st + St::OFF_S + (sub * G_ + 4 * li + 4 * LPG * v) * 4), s4);
#pragma unroll
                    for (int k = 0; k < 4; ++k) rs[v][k] = __fdiv_rn(1.f, s4[k]);
                }
                have_rs = true;
            }
#pragma unroll
            for (int e = lane; e < NG * L; e += 32) {
                const int kk = e / L, c = e % L;
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[kk * Q + jj];
                const float lvc = level_of<Q>(c, a, pb[kk]);
                tabs[warp][kk][c] = make_float2(lvc, lvc - pz[kk]);
            }
            __syncwarp();
            const float dl = pd[sub], za = pz[sub];
            // tau and the filter margin of the lane's own group, on every lane
            float tau, eg;
            {
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[sub * Q + jj];
                tau = fabsf(a[0]);
#pragma unroll
                for (int jj = 1; jj < Q; ++jj) tau = fminf(tau, fabsf(a[jj]));
                eg = bwd_margin(za, pb[sub], a, Q, dl);
            }
            const float rdl = rcp_approx(dl);
            float acc[8];
#pragma unroll
            for (int q8 = 0; q8 < 8; ++q8) acc[q8] = 0.f;
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                float w[4], s4[4], G[4], ws[4], m4[4], uv[4];
                float2 mm[4];
                bool fv[4];
                WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w);
                f4_to(*reinterpret_cast<const float4*>(st + St::OFF_S + el * 4), s4);
                f4_to(*reinterpret_cast<const float4*>(st + St::OFF_G + el * 4), G);
                const uint32_t cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    ws[k] = __fmul_rn(w[k], s4[k]);
                    mm[k] = tabs[warp][sub][(cv >> (8 * k)) & (L - 1)];
                    m4[k] = mm[k].x;
                }
                shared_div_filter4(ws, dl, rdl, za, m4, tau, eg, uv, fv);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int c = (cv >> (8 * k)) & (L - 1);
                    const bool f = fv[k];
                    const float gs = G[k] * rs[v][k];
                    const float mz = mm[k].y;
                    acc[0] += gs * (mz - (f ? uv[k] : 0.f));
                    acc[1] += f ? 0.f : gs;
                    acc[2] += gs;
#pragma unroll
                    for (int j = 0; j < Q; ++j)                  // P_j: dalpha_j = Delta (2 P_j - S)
                        if ((c >> j) & 1) acc[4 + j] += gs;
                    dsa[v][k] += gs * ((f ? w[k] : 0.f) - dl * mz * rs[v][k]);
                }
            }
            const int slot0 = SR8::run(acc, lane);
            const float S = seg_slot2<LPG>(acc, lane);
            if (SR8::writer(lane)) {
                const int64_t grp = row * Gr + (int64_t)it.unit(cc.j) * NG + sub;
                // one select chain and one store per slot (slot 3 is unused here)
#pragma unroll
                for (int q8 = 0; q8 < SR8::NOUT; ++q8) {
                    const int slot = slot0 + q8;
                    const float tot = acc[q8];
                    const float dt = dl * tot;
                    const float val = slot == 0 ? tot : slot == 1 ? -dt : slot == 2 ? dt : dl * __fmaf_rn(2.f, tot, -S);
                    float* dst = slot == 0 ? DDELTA + grp
                                 : slot == 1 ? DZA + grp
                                 : slot == 2 ? DZB + grp
                                 : DALPHA + grp * Q + (slot >= 4 ? slot - 4 : 0);
                    if (slot != 3 && slot < 4 + Q) *dst = val;
                }
            }
        }
                                  });
    if (!ok) return;                                 // no block barrier in this kernel
    // this (block, row slot)'s ds_A partials of the warp's columns (zeros if it had no row)
    if (it.n_w > 0) {
        float* prow = PART + ((int64_t)blockIdx.x * R + it.row_sub) * n_in + (int64_t)it.unit(0) * UE;
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int el = sub * G_ + 4 * li + 4 * LPG * v;
            *reinterpret_cast<float4*>(prow + el) = make_float4(dsa[v][0], dsa[v][1], dsa[v][2], dsa[v][3]);
        }
    }
}

cudaError_t awq_error(bool clear, unsigned int* flag) {
    unsigned int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_awq_err, sizeof(v));
    if (e != cudaSuccess) return e;
    *flag = v;
    if (clear && v != 0) {
        const unsigned int z = 0;
        e = cudaMemcpyToSymbol(g_awq_err, &z, sizeof(z));
    }
    return e;
}

// ds_A[col] = sum over the row ranges of PART[range, col] in a fixed order:
// a block owns 32 columns; its 8 warps each sum one contiguous slice of the
// ranges (ascending, one coalesced 128-byte row piece per load), and the 8
// slice sums are added in slice order.  Deterministic, no atomics.
constexpr int kColsumSlices = 8;
__global__ void __launch_bounds__(32 * kColsumSlices)
awq_colsum_kernel(const float* __restrict__ PART, float* __restrict__ DSA, int n_in, int ranges) {
    __shared__ float part[kColsumSlices][32];
    const int lane = threadIdx.x & 31, slice = threadIdx.x >> 5;
    const int c = blockIdx.x * 32 + lane;
    const int per = (ranges + kColsumSlices - 1) / kColsumSlices;
    const int r0 = slice * per, r1 = r0 + per < ranges ? r0 + per : ranges;
    float acc = 0.f;
    if (c < n_in)
        for (int r = r0; r < r1; ++r) acc += __ldg(PART + (int64_t)r * n_in + c);
    part[slice][lane] = acc;
    __syncthreads();
    if (slice == 0 && c < n_in) {
        float tot = part[0][lane];
#pragma unroll
        for (int k = 1; k < kColsumSlices; ++k) tot += part[k][lane];
        DSA[c] = tot;
    }
}

bool awq_ok(const Shape& sh) { return sh.g == 32 || sh.g == 64 || sh.g == 128 || sh.g == 256 || sh.g == 512; }

// Row ranges: enough blocks (column stripes x ranges) for about
// kAwqTargetBlocksPerSm blocks per SM, at least one row per range.
static void awq_grid(const Shape& sh, int lpg, unsigned& col_blocks, int64_t& ranges, int64_t& rows_per_range) {
    const int NG = 32 / lpg;
    const int units = (sh.n_in / sh.g + NG - 1) / NG;
    col_blocks = (unsigned)((units + kWarps - 1) / kWarps);
    int64_t want = ((int64_t)sm_count() * kAwqTargetBlocksPerSm + col_blocks - 1) / col_blocks;
    if (want > sh.out) want = sh.out;
    if (want < 1) want = 1;
    rows_per_range = (sh.out + want - 1) / want;
    ranges = (sh.out + rows_per_range - 1) / rows_per_range;
}

int64_t awq_workspace_floats(const Shape& sh) {
    if (awq_stream_bwd_ok(sh)) {
        int R, n_rb, grid;
        awq_stream_bwd_grid(sh, R, n_rb, grid);
        return (int64_t)grid * R * sh.n_in;
    }
    unsigned cb;
    int64_t ranges, rpr;
    awq_grid(sh, lanes_per_group(sh.g), cb, ranges, rpr);
    return ranges * (int64_t)sh.n_in;
}

template <int Q, typename WT, int G_>
static cudaError_t run_awq_stream_bwd(const Shape& sh, const void* W, uq_params_awq p, const uint8_t* codes,
                                      const float* gup, uq_grads_awq gr, float* work, cudaStream_t st) {
    using St = AwqBwdStage<Q, WT, G_>;
    int R, n_rb, grid, unused = 0;
    awq_stream_bwd_grid(sh, R, n_rb, grid);
    const size_t dyn = (size_t)kWarps * St::WARP_BYTES;
    auto kern = awq_stream_bwd_kernel<Q, WT, G_>;
    cudaError_t e = grid_for<AwqTag<St, 9>>(kern, dyn, n_rb, unused);    // shared-memory attribute (once)
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, dyn, st>>>(W, p.sa, p.delta, p.za, p.alpha, p.zb, codes, gup, gr.ddelta, gr.dza,
                                      gr.dalpha, gr.dzb, work, sh.out, sh.n_in, R, n_rb);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    awq_colsum_kernel<<<(sh.n_in + 31) / 32, 32 * kColsumSlices, 0, st>>>(work, gr.dsa, sh.n_in, grid * R);
    return cudaGetLastError();
}

template <int Q, typename WT>
static cudaError_t awq_stream_bwd(const Shape& sh, const void* W, uq_params_awq p, const uint8_t* codes,
                                  const float* gup, uq_grads_awq gr, float* work, cudaStream_t st) {
    if (sh.g == 32) return run_awq_stream_bwd<Q, WT, 32>(sh, W, p, codes, gup, gr, work, st);
    if (sh.g == 64) return run_awq_stream_bwd<Q, WT, 64>(sh, W, p, codes, gup, gr, work, st);
    return run_awq_stream_bwd<Q, WT, 128>(sh, W, p, codes, gup, gr, work, st);
}

template <int Q, typename WT, int LPG>
static cudaError_t awq_lpg(bool bwd, int mode, const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes,
                           float* what, const float* gup, uq_grads_awq gr, float* work, cudaStream_t st) {
    unsigned cb;
    int64_t ranges, rpr;
    awq_grid(sh, LPG, cb, ranges, rpr);
    const dim3 grid(cb, (unsigned)ranges);
    if (bwd) {
        awq_bwd_kernel<Q, WT, LPG><<<grid, kThreads, 0, st>>>(W, p.sa, p.delta, p.za, p.alpha, p.zb, codes, gup,
                                                             gr.ddelta, gr.dza, gr.dalpha, gr.dzb, work, sh.out,
                                                             sh.n_in, sh.g, rpr);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        awq_colsum_kernel<<<(sh.n_in + 31) / 32, 32 * kColsumSlices, 0, st>>>(work, gr.dsa, sh.n_in, (int)ranges);
        return cudaGetLastError();
    }
    if (mode == FWD_KEEP)
        awq_fwd_kernel<Q, WT, LPG, FWD_KEEP><<<grid, kThreads, 0, st>>>(W, p.sa, p.delta, p.za, p.alpha, p.zb, codes,
                                                                        what, sh.out, sh.n_in, sh.g, rpr);
    else if (mode == FWD_REMAP)
        awq_fwd_kernel<Q, WT, LPG, FWD_REMAP><<<grid, kThreads, 0, st>>>(W, p.sa, p.delta, p.za, p.alpha, p.zb, codes,
                                                                         what, sh.out, sh.n_in, sh.g, rpr);
    else
        awq_fwd_kernel<Q, WT, LPG, FWD_FULL><<<grid, kThreads, 0, st>>>(W, p.sa, p.delta, p.za, p.alpha, p.zb, codes,
                                                                        what, sh.out, sh.n_in, sh.g, rpr);
    return cudaGetLastError();
}

template <int Q, typename WT>
static cudaError_t awq_g(bool bwd, int mode, const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes,
                         float* what, const float* gup, uq_grads_awq gr, float* work, cudaStream_t st) {
    switch (lanes_per_group(sh.g)) {
        case 4: return awq_lpg<Q, WT, 4>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
        case 8: return awq_lpg<Q, WT, 8>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
        case 16: return awq_lpg<Q, WT, 16>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
        default: return awq_lpg<Q, WT, 32>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
    }
}

template <int Q>
static cudaError_t awq_w(bool bwd, int mode, const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes,
                         float* what, const float* gup, uq_grads_awq gr, float* work, cudaStream_t st) {
    // Steps that map (remap, full) take the pipelined kernel on its shapes; the
    // keep step reads no weights, and the register kernel, which holds s_A
    // across a warp's rows, beats restaging s_A for every unit.
    if (bwd && awq_stream_bwd_ok(sh)) {
        if (sh.wdtype == UQ_W_BF16) return awq_stream_bwd<Q, WBF16>(sh, W, p, codes, gup, gr, work, st);
        return awq_stream_bwd<Q, WF32>(sh, W, p, codes, gup, gr, work, st);
    }
    if (!bwd && mode != FWD_KEEP && stream_path_ok(sh)) {
        if (sh.wdtype == UQ_W_BF16) return awq_stream_fwd<Q, WBF16>(mode, sh, W, p, codes, what, st);
        return awq_stream_fwd<Q, WF32>(mode, sh, W, p, codes, what, st);
    }
    if (sh.wdtype == UQ_W_BF16) return awq_g<Q, WBF16>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
    return awq_g<Q, WF32>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
}

static cudaError_t awq_dispatch(bool bwd, int mode, const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes,
                                float* what, const float* gup, uq_grads_awq gr, float* work, cudaStream_t st) {
    switch (sh.q) {
        case 1: return awq_w<1>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
        case 2: return awq_w<2>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
        case 3: return awq_w<3>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
        default: return awq_w<4>(bwd, mode, sh, W, p, codes, what, gup, gr, work, st);
    }
}

cudaError_t launch_awq_fwd(const Shape& sh, const void* W, uq_params_awq p, uint8_t* codes, int mode, float* what,
                           cudaStream_t st) {
    return awq_dispatch(false, mode, sh, W, p, codes, what, nullptr, uq_grads_awq{}, nullptr, st);
}

cudaError_t launch_awq_bwd(const Shape& sh, const void* W, uq_params_awq p, const uint8_t* codes, const float* gup,
                           uq_grads_awq gr, float* work, cudaStream_t st) {
    return awq_dispatch(true, 0, sh, W, p, const_cast<uint8_t*>(codes), nullptr, gup, gr, work, st);
}

}  // namespace uq
