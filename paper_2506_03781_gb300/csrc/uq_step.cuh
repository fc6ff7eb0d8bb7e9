#pragma once

// The fused optimisation step kernel and its launch templates, included by
// uq_step.cu (fp32 dL/dW^ and W^) and uq_step_bf16.cu (bf16 dL/dW^ and W^).
// The including file defines `static __device__ unsigned int g_step_err`,
// its own bounded-wait flag, before including this header.
//
// Fused optimisation step: the backward of step t, the SGD update of
// Theta_IF, and the forward of step t + 1, in one persistent kernel (one
// pass of the inner loop of Algorithm 1 as the quantizer sees it; SGD as
// FlexRound trains Theta_F, Sec. 3.1; learning rates per parameter set as
// in the hyperparameter table of App. C.1).
//
// The forward of step t + 1 needs the updated row scale s_r', which needs
// the whole row's ds_r, so a row cannot be finished piecewise.  Each warp
// therefore owns ONE work unit (NG whole groups, the lane mapping of
// uq_common.cuh) of a row block and keeps that unit's staged data in shared
// memory across both phases:
//
//   phase A  (bwd at t)  from the stage: x, filter, the per-element ds and
//            s' = s - lr_F ds (written to HBM and over s in the stage), the
//            group sums, and the group updates Delta', z_U', alpha', z_B'
//            (written to HBM and over the staged parameters); the warp's
//            share of ds_r goes to shared memory;
//   barrier  the partials of the row are summed in a fixed order and every
//            warp of the row forms the same s_r' = s_r - lr_F ds_r;
//   phase B  (fwd at t + 1) from the same stage: T_F with the updated
//            parameters, the mapping, W^ and codes to HBM.
//
// W, s and the codes therefore cross HBM once per step.  Rows of up to 8
// units belong to one thread block (R rows per block when a row has fewer
// units than the block has warps); longer rows are split over a thread
// block cluster of csize <= 8 blocks, whose ds_r partials are read through
// distributed shared memory after a cluster barrier.  Each warp keeps two
// stages: the row block in use and the next one, whose copies are in flight
// meanwhile.  Every mbarrier wait is bounded; a wait that runs out sets
// g_step_err (reported by uq_check_device), and the warp stops computing
// but keeps taking part in the barriers, then waits (bounded again) for the
// copies it still has in flight before it returns.
#include <cooperative_groups.h>
#include <cuda_bf16.h>

#include <atomic>

#include "uq_common.cuh"
#include "uq_launch.h"
#include "uq_pipe.cuh"

namespace uq {

// Two fp32 values rounded to bf16 (nearest even), packed low word first.
__device__ __forceinline__ uint32_t bf16x2_rn(float a, float b) {
    return uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(a))) |
           (uint32_t(__bfloat16_as_ushort(__float2bfloat16_rn(b))) << 16);
}

namespace cg = cooperative_groups;

#ifndef UQ_STEP_STAGE_BYTES
#define UQ_STEP_STAGE_BYTES 11520
#endif
#ifndef UQ_STEP_MIN_BLOCKS
#define UQ_STEP_MIN_BLOCKS 2
#endif

constexpr int kMaxCluster = 8;     // portable cluster size limit

template <int Q, int NG>
union StepTab {
    float2 a[NG][1 << Q];          // phase A: (l(c), l(c) - z_U) per group slot and code word
    MapTab<Q, NG> b;               // phase B: levels, sorted order, local-mapping neighbours
};

__device__ __forceinline__ void step_sync(int csize) {
    if (csize > 1) cg::this_cluster().sync();
    else __syncthreads();
}

// BIO: dL/dW^ is read as bf16 and W^ written as bf16 (round to nearest
// even of the fp32 value); otherwise both are fp32.
template <int Q, typename WT, int G_, int MODEB, bool BIO>
__global__ void __launch_bounds__(kThreads, UQ_STEP_MIN_BLOCKS)
step_kernel(const void* __restrict__ W, float* S, float* SR, float* DELTA, float* ZU, float* ALPHA, float* ZB,
            uint8_t* CODES, const void* __restrict__ GUP, void* __restrict__ WHAT, float lr_f, float lr_b,
            int64_t out, int n_in, int R, int csize) {
    using St = Stage<Q, WT, G_, true, true, true, UQ_STEP_STAGE_BYTES, true, BIO ? 2 : 4>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NV = St::NV, UE = St::UE;
    constexpr uint32_t TX = St::TX;
    using SR8 = SegReduce<LPG>;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][2];
    __shared__ StepTab<Q, NG> tabs[kWarps];
    __shared__ float red[2][kWarps];              // ds_r partials (Delta S3 sums) of row blocks k, k + 1

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / LPG, li = lane % LPG;
    const int U = n_in / UE, Gr = n_in / G_;
    const int crank = csize > 1 ? (int)cg::this_cluster().block_rank() : 0;
    const int64_t cid = blockIdx.x / csize, ncl = gridDim.x / csize;
    const int WPR = kWarps / R;                   // warps per row (all 8 when csize > 1, R = 1)
    const int row_sub = warp / WPR;
    const int unit = crank * kWarps + warp % WPR;
    const bool has_unit = unit < U;
    // Row blocks of this cluster (the same count in every block of it) and
    // this warp's items: the row blocks whose row exists.
    const int64_t n_rb = (out + R - 1) / R;
    const int64_t n_blocks = cid < n_rb ? (n_rb - cid + ncl - 1) / ncl : 0;
    const int64_t n_rb_sub = (out - row_sub + R - 1) / R;
    const int64_t n_items = (has_unit && n_rb_sub > cid) ? (n_rb_sub - cid + ncl - 1) / ncl : 0;
    unsigned char* wsm = smem + (size_t)warp * 2 * St::BYTES;
    StepTab<Q, NG>& t = tabs[warp];

    if (lane == 0) {
        tma::bar_init(tma::smem_addr(&bars[warp][0]), 1);
        tma::bar_init(tma::smem_addr(&bars[warp][1]), 1);
        tma::bar_init_fence();
    }
    __syncthreads();

    // The eight copies of a unit, one per lane 0..7: source base, bytes per
    // element (per group for the parameters), size and stage offset, from a
    // per-block table, so the lanes start their copies side by side.
    __shared__ struct StepCopy {
        const unsigned char* base;
        uint32_t per, size, off, grp;
    } cps[8];
    if (threadIdx.x < 8) {
        const int i = threadIdx.x;
        const unsigned char* b[8] = {static_cast<const unsigned char*>(W), reinterpret_cast<const unsigned char*>(S),
                                     static_cast<const unsigned char*>(GUP), CODES,
                                     reinterpret_cast<const unsigned char*>(DELTA), reinterpret_cast<const unsigned char*>(ZU),
                                     reinterpret_cast<const unsigned char*>(ZB), reinterpret_cast<const unsigned char*>(ALPHA)};
        const uint32_t per[8] = {(uint32_t)St::WBYTES, 4u, (uint32_t)St::GB, 1u, 4u, 4u, 4u, 4u * Q};
        const uint32_t size[8] = {St::SZ_W, St::SZ_S, St::SZ_G, St::SZ_C, St::SZ_P, St::SZ_P, St::SZ_P, St::SZ_A};
        const uint32_t off[8] = {St::OFF_W, St::OFF_S, St::OFF_G, St::OFF_C, St::OFF_D, St::OFF_Z, St::OFF_B, St::OFF_A};
        cps[i] = StepCopy{b[i], per[i], size[i], off[i], i >= 4 ? 1u : 0u};
    }
    __syncthreads();

    auto row_of = [&](int64_t k) { return (cid + k * ncl) * R + row_sub; };
    // issued by the whole warp (k < n_items): lane 0 arms the stage's
    // mbarrier with the unit's bytes, then lanes 0..7 each start one copy
    auto issue = [&](int64_t k) {
        const int s = (int)(k & 1);
        const uint32_t bar = tma::smem_addr(&bars[warp][s]);
        if (lane == 0) tma::bar_arrive_tx(bar, TX);
        __syncwarp();
        if (lane < 8) {
            const int64_t row = row_of(k);
            const StepCopy cp = cps[lane];
            const int64_t idx = cp.grp ? row * Gr + (int64_t)unit * NG : row * n_in + (int64_t)unit * UE;
            tma::fence_async_smem();
            tma::copy_g2s(tma::smem_addr(wsm + (size_t)s * St::BYTES) + cp.off, cp.base + idx * cp.per, cp.size, bar);
        }
    };
    int64_t next_issue = 0, next_wait = 0;        // items issued / waited for (every lane)
    while (next_issue < 2 && next_issue < n_items) issue(next_issue++);

    bool alive = true;
    for (int64_t k = 0; k < n_blocks; ++k) {
        const int64_t row = row_of(k);
        const bool mine = k < n_items;
        unsigned char* st = wsm + (size_t)(k & 1) * St::BYTES;
        float* pd = reinterpret_cast<float*>(st + St::OFF_D);
        float* pz = reinterpret_cast<float*>(st + St::OFF_Z);
        float* pb = reinterpret_cast<float*>(st + St::OFF_B);
        float* pa = reinterpret_cast<float*>(st + St::OFF_A);
        float sr = 1.f, prow = 0.f;
        if (mine && alive) {
            // one verdict for the whole warp (lanes poll the mbarrier separately)
            if (__all_sync(kFull, tma::bar_wait(tma::smem_addr(&bars[warp][k & 1]), (uint32_t)((k >> 1) & 1)))) {
                next_wait = k + 1;
            } else {
                alive = false;
                if (lane == 0) atomicOr(&g_step_err, 1u);
            }
        }
        if (mine && alive) {
            // ---- phase A: backward of step t and the update of s and the group parameters ----
            sr = SR[row];                          // this row's s_r is rewritten only after the barrier below
#pragma unroll
            for (int e = lane; e < NG * L; e += 32) {
                const int kk = e / L, c = e % L;
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[kk * Q + jj];
                const float lvc = level_of<Q>(c, a, pb[kk]);
                t.a[kk][c] = make_float2(lvc, lvc - pz[kk]);
            }
            __syncwarp();
            const float dl = pd[sub], zu = pz[sub];
            // tau and the filter margin of the lane's own group, on every lane
            float tau, eg;
            {
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[sub * Q + jj];
                tau = fabsf(a[0]);
#pragma unroll
                for (int jj = 1; jj < Q; ++jj) tau = fminf(tau, fabsf(a[jj]));
                eg = bwd_margin(zu, pb[sub], a, Q, __fmul_rn(__fmul_rn(dl, dl), sr));
            }
            const float kds = __fmul_rn(__fmul_rn(dl, dl), sr);         // Delta / s = r kds, r = 1 / den
            const int64_t ebase = row * n_in + (int64_t)unit * UE;
            float acc[8];
#pragma unroll
            for (int q8 = 0; q8 < 8; ++q8) acc[q8] = 0.f;
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                float w[4], s4[4], G[4], sn[4];
                WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w);
                float4* sp = reinterpret_cast<float4*>(st + St::OFF_S + el * 4);
                f4_to(*sp, s4);
                if constexpr (BIO) WBF16::unpack(*reinterpret_cast<const uint2*>(st + St::OFF_G + el * 2), G);
                else f4_to(*reinterpret_cast<const float4*>(st + St::OFF_G + el * 4), G);
                const uint32_t cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                float ds[4];
                bwd_vec4<Q, false>(w, s4, G, cv, t.a[sub], dl, sr, zu, tau, eg, kds, ds, acc);
#pragma unroll
                for (int kq = 0; kq < 4; ++kq) sn[kq] = __fsub_rn(s4[kq], __fmul_rn(lr_f, ds[kq]));
                const float4 s_new = make_float4(sn[0], sn[1], sn[2], sn[3]);
                *reinterpret_cast<float4*>(S + ebase + el) = s_new;
                *sp = s_new;                       // the forward of step t + 1 reads s' from the stage
            }
            __syncwarp();                          // every lane has read the old staged parameters
            const int slot0 = SR8::run(acc, lane);
            const float S = seg_slot2<LPG>(acc, lane);
            if (SR8::writer(lane)) {
                const int64_t grp = row * Gr + (int64_t)unit * NG + sub;
#pragma unroll
                // one select chain and one update per slot (the lanes of a warp hold
                // different slots): slot 0 dDelta = tot, 1 dz_U = -(Delta tot),
                // 2 dz_B = Delta tot, 3 Delta S3 of the group (ds_r), 4 + j
                // dalpha_j = Delta (2 P_j - S)
#pragma unroll
                for (int q8 = 0; q8 < SR8::NOUT; ++q8) {
                    const int slot = slot0 + q8;
                    const float tot = acc[q8];
                    const float dt = dl * tot;
                    const int j = slot >= 4 ? slot - 4 : 0;
                    const float gr = slot == 0 ? tot : slot == 1 ? -dt : slot == 2 ? dt : dl * __fmaf_rn(2.f, tot, -S);
                    const float lr = slot <= 1 ? lr_f : lr_b;
                    float* sp_ = slot == 0 ? pd + sub : slot == 1 ? pz + sub : slot == 2 ? pb + sub : pa + sub * Q + j;
                    float* gp = slot == 0 ? DELTA + grp : slot == 1 ? ZU + grp : slot == 2 ? ZB + grp : ALPHA + grp * Q + j;
                    prow = slot == 3 ? prow + dt : prow;
                    if (slot != 3 && slot < 4 + Q) {
                        const float v = __fsub_rn(*sp_, __fmul_rn(lr, gr));
                        *sp_ = v;
                        *gp = v;
                    }
                }
            }
        }
        prow = warp_sum(prow);
        if (lane == 0) red[k & 1][warp] = prow;
        step_sync(csize);                          // every ds_r partial of row block k is in shared memory
        if (mine && alive) {
            // ---- s_r' of the row: partials summed in (block rank, warp) order, the same in every block ----
            float tot = 0.f;
            if (csize > 1) {
                cg::cluster_group cl = cg::this_cluster();
                for (int c = 0; c < csize; ++c) {
                    const float* rr = cl.map_shared_rank(&red[k & 1][0], c);
#pragma unroll
                    for (int w = 0; w < kWarps; ++w) tot += rr[w];
                }
            } else {
                for (int w = 0; w < WPR; ++w) tot += red[k & 1][row_sub * WPR + w];
            }
            const float dsr = -tot / sr;
            const float sr_new = __fsub_rn(sr, __fmul_rn(lr_f, dsr));
            if (unit == 0 && lane == 0) SR[row] = sr_new;

            // ---- phase B: forward of step t + 1 from the stage ----
#pragma unroll
            for (int e = lane; e < NG * L; e += 32) {
                const int kk = e / L, c = e % L;
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[kk * Q + jj];
                t.b.lv[kk][c] = level_of<Q>(c, a, pb[kk]);
            }
            __syncwarp();
            if constexpr (MODEB == FWD_REMAP) unit_sort<Q, NG, true>(t.b, lane);
            else if constexpr (MODEB == FWD_FULL) unit_sort<Q, NG, false>(t.b, lane);
            const float dl = pd[sub], zu = pz[sub];
            const int64_t ebase = row * n_in + (int64_t)unit * UE;
            float srt[L];
            if constexpr (MODEB == FWD_FULL) {
#pragma unroll
                for (int r = 0; r < L; ++r) srt[r] = t.b.srt[sub][r];
            }
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                const uint32_t cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                float o[4];
                if constexpr (MODEB == FWD_KEEP) {
#pragma unroll
                    for (int kq = 0; kq < 4; ++kq) {
                        const int c = (cv >> (8 * kq)) & (L - 1);
                        o[kq] = __fmul_rn(dl, __fsub_rn(t.b.lv[sub][c], zu));
                    }
                } else {
                    float w[4], s4[4];
                    uint32_t nc = 0;
                    WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w);
                    f4_to(*reinterpret_cast<const float4*>(st + St::OFF_S + el * 4), s4);
                    if constexpr (MODEB == FWD_REMAP) {
#pragma unroll
                        for (int kq = 0; kq < 4; ++kq) {
                            const int c = (cv >> (8 * kq)) & (L - 1);
                            const float4 nb = t.b.nb[sub][c];
                            float uu;
                            const float x = transform_x(w[kq], s4[kq], dl, sr_new, zu, uu);
                            const uint32_t packed = __float_as_uint(nb.w);
                            float best = fabsf(__fsub_rn(x, nb.y));
                            float m = nb.y;
                            uint32_t code = c;
                            const float dlo = fabsf(__fsub_rn(x, nb.x));
                            if (dlo < best) { best = dlo; m = nb.x; code = packed & 0xffu; }
                            const float dhi = fabsf(__fsub_rn(x, nb.z));
                            if (dhi < best) { m = nb.z; code = (packed >> 8) & 0xffu; }
                            o[kq] = __fmul_rn(dl, __fsub_rn(m, zu));
                            nc |= code << (8 * kq);
                        }
                    } else {
#pragma unroll
                        for (int kq = 0; kq < 4; ++kq) {
                            float uu, m;
                            const float x = transform_x(w[kq], s4[kq], dl, sr_new, zu, uu);
                            const int r = nearest_rank<L>(x, srt, m);
                            o[kq] = __fmul_rn(dl, __fsub_rn(m, zu));
                            nc |= uint32_t(t.b.cor[sub][r]) << (8 * kq);
                        }
                    }
                    *reinterpret_cast<uint32_t*>(CODES + ebase + el) = nc;
                }
                if constexpr (BIO)
                    *reinterpret_cast<uint2*>(static_cast<uint16_t*>(WHAT) + ebase + el) =
                        make_uint2(bf16x2_rn(o[0], o[1]), bf16x2_rn(o[2], o[3]));
                else
                    *reinterpret_cast<float4*>(static_cast<float*>(WHAT) + ebase + el) =
                        make_float4(o[0], o[1], o[2], o[3]);
            }
            // the stage's generic writes (s', parameters) before the next bulk copy into it
            tma::fence_async_smem();
        }
        __syncwarp();
        if (alive && next_issue < n_items) issue(next_issue++);
    }
    if (!alive && lane == 0) {
        // copies this warp issued but never waited for land before the block exits
        for (int64_t k = next_wait; k < next_issue; ++k)
            if (!tma::bar_wait(tma::smem_addr(&bars[warp][k & 1]), (uint32_t)((k >> 1) & 1))) {
                atomicOr(&g_step_err, kDrainTimeoutBit);   // copies may still be in flight
                break;
            }
    }
    if (csize > 1) cg::this_cluster().sync();      // no block leaves while another may read its partials
}

// ---------------------------------------------------------------------------
// Launch templates
// ---------------------------------------------------------------------------

constexpr int kMaxDevicesStep = 64;

template <int Q, typename WT, int G_, int MODEB, bool BIO>
static cudaError_t run_step(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const void* gup,
                            float lr_f, float lr_b, void* what, cudaStream_t st) {
    using St = Stage<Q, WT, G_, true, true, true, UQ_STEP_STAGE_BYTES, true, BIO ? 2 : 4>;
    const int U = sh.n_in / St::UE;
    const int csize = U <= kWarps ? 1 : (U + kWarps - 1) / kWarps;
    const int R = csize == 1 ? rows_per_block(U) : 1;
    const int64_t n_rb = (sh.out + R - 1) / R;
    const size_t dyn = (size_t)kWarps * 2 * St::BYTES;
    auto kern = step_kernel<Q, WT, G_, MODEB, BIO>;
    // occupancy per device and cluster size (blocks per SM for csize == 1, clusters on the GPU otherwise)
    static std::atomic<int> cache[kMaxDevicesStep][kMaxCluster + 1] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::atomic<int>* slot = (dev >= 0 && dev < kMaxDevicesStep) ? &cache[dev][csize] : nullptr;
    int cap = slot ? slot->load(std::memory_order_relaxed) : 0;

    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = dyn;
    cfg.stream = st;
    if (csize > 1) {
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = csize;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
    }
    if (cap == 0) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e != cudaSuccess) return e;
        if (csize == 1) {
            int per_sm = 0;
            e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, dyn);
            if (e != cudaSuccess) return e;
            cap = sm_count() * (per_sm < 1 ? 1 : per_sm);
        } else {
            cfg.gridDim = dim3(csize);
            int ncl = 0;
            e = cudaOccupancyMaxActiveClusters(&ncl, kern, &cfg);
            if (e != cudaSuccess) return e;
            cap = ncl < 1 ? 1 : ncl;
        }
        if (slot) slot->store(cap, std::memory_order_relaxed);
    }
    const int64_t units = csize == 1 ? n_rb : sh.out;     // row blocks, or clusters' rows
    const int64_t n_grp = units < cap ? units : cap;       // blocks (csize == 1) or clusters
    cfg.gridDim = dim3((unsigned)(n_grp * csize));
    return cudaLaunchKernelEx(&cfg, kern, W, p.s, p.sr, p.delta, p.zu, p.alpha, p.zb, codes, gup, what, lr_f, lr_b,
                              sh.out, sh.n_in, R, csize);
}

template <int Q, typename WT, int G_, bool BIO>
static cudaError_t step_mode(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const void* gup,
                             float lr_f, float lr_b, int mode, void* what, cudaStream_t st) {
    if (mode == FWD_KEEP) return run_step<Q, WT, G_, FWD_KEEP, BIO>(sh, W, p, codes, gup, lr_f, lr_b, what, st);
    if (mode == FWD_REMAP) return run_step<Q, WT, G_, FWD_REMAP, BIO>(sh, W, p, codes, gup, lr_f, lr_b, what, st);
    return run_step<Q, WT, G_, FWD_FULL, BIO>(sh, W, p, codes, gup, lr_f, lr_b, what, st);
}

template <int Q, typename WT, bool BIO>
static cudaError_t step_g(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const void* gup,
                          float lr_f, float lr_b, int mode, void* what, cudaStream_t st) {
    if (sh.g == 32) return step_mode<Q, WT, 32, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
    if (sh.g == 64) return step_mode<Q, WT, 64, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
    return step_mode<Q, WT, 128, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
}

template <int Q, bool BIO>
static cudaError_t step_w(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const void* gup,
                          float lr_f, float lr_b, int mode, void* what, cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return step_g<Q, WBF16, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
    return step_g<Q, WF32, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
}

// Every q for one I/O type (the translation unit that includes this header
// instantiates one of them).
template <bool BIO>
static cudaError_t step_q(const Shape& sh, const void* W, uq_params p, uint8_t* codes, const void* gup, float lr_f,
                          float lr_b, int mode, void* what, cudaStream_t st) {
    switch (sh.q) {
        case 1: return step_w<1, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
        case 2: return step_w<2, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
        case 3: return step_w<3, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
        default: return step_w<4, BIO>(sh, W, p, codes, gup, lr_f, lr_b, mode, what, st);
    }
}

}  // namespace uq
