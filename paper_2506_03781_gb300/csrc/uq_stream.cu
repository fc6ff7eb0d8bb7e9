// Persistent, TMA-pipelined forward and backward kernels (the fast path for
// g in {32, 64, 128} and rows that split into whole work units).
//
// Each warp runs its own pipeline over its work units (NG whole groups =
// UE contiguous elements of one row, the lane mapping of uq_common.cuh):
// one bulk copy (cp.async.bulk, completion counted on an mbarrier) per input
// stream of a unit -- weights, s, dL/dW^, code words and the unit's group
// parameters -- goes into one of NST shared-memory stages (issued by lane 0
// in the forwards, by lanes 0..7 side by side in the backward), and the warp
// computes from shared memory while the copies of the next units are in
// flight.  Thread blocks are persistent: block b handles row blocks
// b, b + gridDim.x, ...; within a row block the warps split the row's units
// as in the non-pipelined kernels.  Every mbarrier wait is bounded (about one second of
// GPU clock); a wait that runs out sets g_stream_err, which
// uq_check_device() reports, and the warp stops computing.  The backward
// kernel's ds_r partials wait in a shared-memory ring of kRowRing row
// blocks, summed in warp order after one block barrier per ring.
#include <atomic>

#include "uq_common.cuh"
#include "uq_launch.h"
#include "uq_pipe.cuh"

namespace uq {

__device__ unsigned int g_stream_err = 0;

// Shared memory per warp for its stages, and the resident blocks per SM the
// register allocation is bounded for (backward; forward).
#ifndef UQ_BWD_STAGE_BYTES
#define UQ_BWD_STAGE_BYTES 11520
#endif
#ifndef UQ_FWD_STAGE_BYTES
#define UQ_FWD_STAGE_BYTES 5632
#endif
#ifndef UQ_KEEP_STAGE_BYTES
#define UQ_KEEP_STAGE_BYTES 9728
#endif
#ifndef UQ_STREAM_BWD_MIN_BLOCKS
#define UQ_STREAM_BWD_MIN_BLOCKS 2
#endif
#ifndef UQ_STREAM_FWD_MIN_BLOCKS
#define UQ_STREAM_FWD_MIN_BLOCKS 4
#endif
constexpr int kRowRing = 32;             // row blocks whose ds_r partials wait in shared memory
// Rows of at least this many work units take the backward's branch-per-array
// gradient stores: 526 vs 598 us on 8192 x 28672 (56 units per row), while
// the select chain wins on shorter rows (153 vs 160 us on 14336 x 4096,
// 516 vs 546 us on 28672 x 8192).
constexpr int kBranchyUnits = 32;

// ---------------------------------------------------------------------------
// Backward
// ---------------------------------------------------------------------------

// ELEM: the whole-element filter (a filtered element drops out of every
// gradient); otherwise the filter cuts the straight-through path only.
// branchy (warp-uniform): write the group gradients with a branch per output
// array instead of the select chain (the launcher's choice for long rows).
template <int Q, typename WT, int G_, bool ELEM>
__global__ void __launch_bounds__(kThreads, UQ_STREAM_BWD_MIN_BLOCKS)
bwd_stream_kernel(const void* __restrict__ W, const float* __restrict__ S, const float* __restrict__ SR,
                  const float* __restrict__ DELTA, const float* __restrict__ ZU, const float* __restrict__ ALPHA,
                  const float* __restrict__ ZB, const uint8_t* __restrict__ CODES, const float* __restrict__ GUP,
                  float* __restrict__ DS, float* __restrict__ DSR, float* __restrict__ DDELTA,
                  float* __restrict__ DZU, float* __restrict__ DZB, float* __restrict__ DALPHA, int64_t out,
                  int n_in, int R, int n_rb, int branchy) {
    using St = Stage<Q, WT, G_, true, true, true, UQ_BWD_STAGE_BYTES>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NV = St::NV, UE = St::UE, NST = St::NST;
    constexpr uint32_t TX = St::TX;
    using SR8 = SegReduce<LPG>;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][NST];
    __shared__ float2 tabs[kWarps][NG][L];          // (l(c), l(c) - z_U) per group slot and code word
    __shared__ float red[kRowRing][kWarps];       // per row block and warp: sum of Delta S3
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / LPG, li = lane % LPG;
    const int U = n_in / UE, Gr = n_in / G_;
    const Items it(U, R, n_rb, warp);
    unsigned char* wsm = smem + (size_t)warp * St::WARP_BYTES;
    float2 (*t)[L] = tabs[warp];

    if (lane == 0) {
        for (int s = 0; s < NST; ++s) tma::bar_init(tma::smem_addr(&bars[warp][s]), 1);
        tma::bar_init_fence();
    }
    __syncthreads();

    // The eight copies of a unit, one per lane 0..7: source base, bytes per
    // element (per group for the parameters), size and stage offset, from a
    // per-block table, so the lanes start their copies side by side.
    __shared__ struct CopySpec {
        const unsigned char* base;
        uint32_t per, size, off, grp;
    } cps[8];
    if (threadIdx.x < 8) {
        const int i = threadIdx.x;
        const unsigned char* b[8] = {static_cast<const unsigned char*>(W), reinterpret_cast<const unsigned char*>(S),
                                     reinterpret_cast<const unsigned char*>(GUP), CODES,
                                     reinterpret_cast<const unsigned char*>(DELTA), reinterpret_cast<const unsigned char*>(ZU),
                                     reinterpret_cast<const unsigned char*>(ZB), reinterpret_cast<const unsigned char*>(ALPHA)};
        const uint32_t per[8] = {(uint32_t)St::WBYTES, 4u, 4u, 1u, 4u, 4u, 4u, 4u * Q};
        const uint32_t size[8] = {St::SZ_W, St::SZ_S, St::SZ_G, St::SZ_C, St::SZ_P, St::SZ_P, St::SZ_P, St::SZ_A};
        const uint32_t off[8] = {St::OFF_W, St::OFF_S, St::OFF_G, St::OFF_C, St::OFF_D, St::OFF_Z, St::OFF_B, St::OFF_A};
        cps[i] = CopySpec{b[i], per[i], size[i], off[i], i >= 4 ? 1u : 0u};
    }
    __syncthreads();
    // issued by the whole warp: lane 0 arms the stage's mbarrier with the
    // unit's bytes, then lanes 0..7 each start one copy
    auto issue = [&](const Cursor& c, int s) {
        const uint32_t bar = tma::smem_addr(&bars[warp][s]);
        const int64_t row = it.row(c.k);
        if (row >= out) {
            if (lane == 0) tma::bar_arrive(bar);
            return;
        }
        if (lane == 0) tma::bar_arrive_tx(bar, TX);
        __syncwarp();
        if (lane < 8) {
            const CopySpec cp = cps[lane];
            const int64_t idx = cp.grp ? row * Gr + (int64_t)it.unit(c.j) * NG : row * n_in + (int64_t)it.unit(c.j) * UE;
            const uint32_t d = tma::smem_addr(wsm + (size_t)s * St::BYTES);
            tma::fence_async_smem();
            tma::copy_g2s(d + cp.off, cp.base + idx * cp.per, cp.size, bar);
        }
    };
    Cursor ic;                                            // next item to issue (every lane)
    long long issued = 0;
    for (int s = 0; s < NST && issued < it.total; ++s, ++issued) {
        issue(ic, s);
        ic.next(it.n_w);
    }

    bool alive = true;
    long long waited = 0;                                 // items whose copies have landed
    Ring<NST> ring;
    const int n_mine = it.n_blocks;
    for (int k = 0; k < n_mine; ++k) {
        const int64_t rb = (int64_t)blockIdx.x + (int64_t)k * gridDim.x;
        const int64_t row = rb * R + it.row_sub;
        const bool row_ok = row < out;
        const float sr = row_ok ? __ldg(SR + row) : 1.f;
        float prow = 0.f;
        for (int j = 0; j < it.n_w; ++j) {
            const int s = ring.s;
            if (alive) {
                // one verdict for the whole warp (lanes poll the mbarrier separately)
                if (__all_sync(kFull, tma::bar_wait(tma::smem_addr(&bars[warp][s]), ring.parity))) {
                    ++waited;
                } else {
                    alive = false;
                    if (lane == 0) atomicOr(&g_stream_err, 1u);
                }
            }
            if (alive && row_ok) {
                const unsigned char* st = wsm + (size_t)s * St::BYTES;
                const float* pd = reinterpret_cast<const float*>(st + St::OFF_D);
                const float* pz = reinterpret_cast<const float*>(st + St::OFF_Z);
                const float* pb = reinterpret_cast<const float*>(st + St::OFF_B);
                const float* pa = reinterpret_cast<const float*>(st + St::OFF_A);
                // levels and tau of the unit's groups, from the staged parameters
#pragma unroll
                for (int e = lane; e < NG * L; e += 32) {
                    const int kk = e / L, c = e % L;
                    float a[Q];
#pragma unroll
                    for (int jj = 0; jj < Q; ++jj) a[jj] = pa[kk * Q + jj];
                    const float lvc = level_of<Q>(c, a, pb[kk]);
                    t[kk][c] = make_float2(lvc, lvc - pz[kk]);
                }
                __syncwarp();
                const float dl = pd[sub], zu = pz[sub];
                // tau and the filter margin of the lane's own group, on every lane
                // (no divergent branch, no shared-memory round trip)
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
                const float kds = __fmul_rn(__fmul_rn(dl, dl), sr);     // Delta / s = r kds, r = 1 / den
                const int unit = it.unit(j);
                const int64_t ebase = row * n_in + (int64_t)unit * UE;
                float acc[8];
#pragma unroll
                for (int q8 = 0; q8 < 8; ++q8) acc[q8] = 0.f;
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int el = sub * G_ + 4 * li + 4 * LPG * v;
                    float w[4], s4[4], G[4], ds[4];
                    WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w);
                    f4_to(*reinterpret_cast<const float4*>(st + St::OFF_S + el * 4), s4);
                    f4_to(*reinterpret_cast<const float4*>(st + St::OFF_G + el * 4), G);
                    const uint32_t cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                    bwd_vec4<Q, ELEM>(w, s4, G, cv, t[sub], dl, sr, zu, tau, eg, kds, ds, acc);
                    *reinterpret_cast<float4*>(DS + ebase + el) = make_float4(ds[0], ds[1], ds[2], ds[3]);
                }
                const int slot0 = SR8::run(acc, lane);
                const float S = seg_slot2<LPG>(acc, lane);
                if (SR8::writer(lane)) {
                    const int64_t grp = row * Gr + (int64_t)unit * NG + sub;
                    if (!branchy) {
                        // one select chain and one store per slot instead of a branch per
                        // output array (the lanes of a warp hold different slots)
#pragma unroll
                        for (int q8 = 0; q8 < SR8::NOUT; ++q8) {
                            const int slot = slot0 + q8;
                            const float tot = acc[q8];
                            const float dt = dl * tot;
                            const float val =
                                slot == 0 ? tot : slot == 1 ? -dt : slot == 2 ? dt : dl * __fmaf_rn(2.f, tot, -S);
                            float* dst = slot == 0 ? DDELTA + grp
                                         : slot == 1 ? DZU + grp
                                         : slot == 2 ? DZB + grp
                                         : DALPHA + grp * Q + (slot >= 4 ? slot - 4 : 0);
                            prow = slot == 3 ? prow + dt : prow;
                            if (slot != 3 && slot < 4 + Q) *dst = val;
                        }
                    } else {
                        // a branch per output array: measured faster on rows of many units
#pragma unroll
                        for (int q8 = 0; q8 < SR8::NOUT; ++q8) {
                            const int slot = slot0 + q8;
                            const float tot = acc[q8];
                            if (slot == 0) DDELTA[grp] = tot;
                            else if (slot == 1) DZU[grp] = -(dl * tot);
                            else if (slot == 2) DZB[grp] = dl * tot;
                            else if (slot == 3) prow += dl * tot;
                            else if (slot - 4 < Q) DALPHA[grp * Q + (slot - 4)] = dl * __fmaf_rn(2.f, tot, -S);
                        }
                    }
                }
            }
            __syncwarp();                                // stage s and the tables are free again
            if (alive && issued < it.total) {
                issue(ic, s);
                ic.next(it.n_w);
                ++issued;
            }
            ring.next();
        }
        prow = warp_sum(prow);
        if (lane == 0) red[k % kRowRing][warp] = prow;
        // ds_r of the last kRowRing row blocks, once the ring is full or at the end
        if (k % kRowRing == kRowRing - 1 || k == n_mine - 1) {
            __syncthreads();
            const int k0 = k - k % kRowRing;
            const int WPR = kWarps / R;
            for (int idx = threadIdx.x; idx < (k - k0 + 1) * R; idx += kThreads) {
                const int kk = k0 + idx / R, rsub = idx % R;
                const int64_t r = ((int64_t)blockIdx.x + (int64_t)kk * gridDim.x) * R + rsub;
                if (r < out) {
                    const float* rr = red[kk % kRowRing];
                    float s = rr[rsub * WPR];
                    for (int w = 1; w < WPR; ++w) s += rr[rsub * WPR + w];
                    DSR[r] = -s / __ldg(SR + r);
                }
            }
            __syncthreads();
        }
    }
    if (!alive && lane == 0 && !drain(bars[warp], waited, issued)) atomicOr(&g_stream_err, kDrainTimeoutBit);
}

// ---------------------------------------------------------------------------
// Forward
// ---------------------------------------------------------------------------

template <int Q, typename WT, int G_, int MODE>
__global__ void __launch_bounds__(kThreads, UQ_STREAM_FWD_MIN_BLOCKS)
fwd_stream_kernel(const void* __restrict__ W, const float* __restrict__ S, const float* __restrict__ SR,
                  const float* __restrict__ DELTA, const float* __restrict__ ZU, const float* __restrict__ ALPHA,
                  const float* __restrict__ ZB, uint8_t* __restrict__ CODES, float* __restrict__ WHAT,
                  int64_t out, int n_in, int R, int n_rb) {
    static_assert(MODE != FWD_KEEP, "the keep step runs keep_stream_kernel");
    constexpr int mode = MODE;
    constexpr bool need_c = MODE != FWD_FULL;
    using St = Stage<Q, WT, G_, true, false, need_c, UQ_FWD_STAGE_BYTES>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NV = St::NV, UE = St::UE, NST = St::NST;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][NST];
    __shared__ MapTab<Q, NG> tabs[kWarps];
    constexpr int NIV = mode == FWD_REMAP ? NG : 1;              // remap intervals only on remap steps
    __shared__ float4 ivs[kWarps][NIV][L];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / LPG, li = lane % LPG;
    const int U = n_in / UE, Gr = n_in / G_;
    const Items it(U, R, n_rb, warp);
    unsigned char* wsm = smem + (size_t)warp * St::WARP_BYTES;
    MapTab<Q, NG>& t = tabs[warp];
    constexpr uint32_t TX = St::TX;

    if (lane == 0) {
        for (int s = 0; s < NST; ++s) tma::bar_init(tma::smem_addr(&bars[warp][s]), 1);
        tma::bar_init_fence();
    }
    __syncwarp();

    auto issue = [&](const Cursor& c, int s) {           // lane 0 only
        const uint32_t bar = tma::smem_addr(&bars[warp][s]);
        const int64_t row = it.row(c.k);
        if (row >= out) { tma::bar_arrive(bar); return; }
        const int64_t e0 = row * n_in + (int64_t)it.unit(c.j) * UE;
        const int64_t g0 = row * Gr + (int64_t)it.unit(c.j) * NG;
        const uint32_t d = tma::smem_addr(wsm + (size_t)s * St::BYTES);
        tma::fence_async_smem();
        tma::bar_arrive_tx(bar, TX);
        tma::copy_g2s(d + St::OFF_W, static_cast<const unsigned char*>(W) + e0 * St::WBYTES, St::SZ_W, bar);
        tma::copy_g2s(d + St::OFF_S, S + e0, St::SZ_S, bar);
        if constexpr (need_c) tma::copy_g2s(d + St::OFF_C, CODES + e0, St::SZ_C, bar);
        tma::copy_g2s(d + St::OFF_D, DELTA + g0, St::SZ_P, bar);
        tma::copy_g2s(d + St::OFF_Z, ZU + g0, St::SZ_P, bar);
        tma::copy_g2s(d + St::OFF_B, ZB + g0, St::SZ_P, bar);
        tma::copy_g2s(d + St::OFF_A, ALPHA + g0 * Q, St::SZ_A, bar);
    };

    const bool ok = pipe_run<NST>(it, bars[warp], lane, &g_stream_err, 1u, issue,
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
            if constexpr (mode == FWD_REMAP) {
                unit_sort<Q, NG, false>(t, lane);
                unit_remap_iv<Q, NG>(t, ivs[warp], lane, pd, pz);
            } else if constexpr (mode == FWD_FULL) {
                unit_sort<Q, NG, false>(t, lane);
            }
            const float dl = pd[sub], zu = pz[sub];
            const float sr = __ldg(SR + row);
            const int64_t ebase = row * n_in + (int64_t)it.unit(cc.j) * UE;
            float srt[L];
            if constexpr (mode == FWD_FULL) {
#pragma unroll
                for (int r = 0; r < L; ++r) srt[r] = t.srt[sub][r];
            }
#pragma unroll
            for (int v = 0; v < NV; ++v) {
                const int el = sub * G_ + 4 * li + 4 * LPG * v;
                float o[4];
                uint32_t nc = 0;
                uint32_t cv = 0u;
                if constexpr (need_c) cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                {
                    float w[4], s4[4];
                    WT::unpack(*reinterpret_cast<const typename WT::raw*>(st + St::OFF_W + el * St::WBYTES), w);
                    f4_to(*reinterpret_cast<const float4*>(st + St::OFF_S + el * 4), s4);
                    if constexpr (mode == FWD_REMAP) {
                        nc = remap_vec4<Q, NG>(w, s4, cv, t, ivs[warp], sub, dl, sr, zu, o);
                    } else {
#pragma unroll
                        for (int kq = 0; kq < 4; ++kq) {
                            float uu, m;
                            const float x = transform_x(w[kq], s4[kq], dl, sr, zu, uu);
                            const int r = nearest_rank<L>(x, srt, m);
                            o[kq] = __fmul_rn(dl, __fsub_rn(m, zu));
                            nc |= uint32_t(t.cor[sub][r]) << (8 * kq);
                        }
                    }
                    *reinterpret_cast<uint32_t*>(CODES + ebase + el) = nc;
                }
                *reinterpret_cast<float4*>(WHAT + ebase + el) = make_float4(o[0], o[1], o[2], o[3]);
            }
        }
                                  });
    if (!ok) return;                                 // no block barrier in this kernel
}

// ---------------------------------------------------------------------------
// Forward of the steps that keep the codes (M*_B off its remap step)
// ---------------------------------------------------------------------------
//
// W^ = Delta (l(code) - z_U) reads only the code bytes and the group
// parameters, so a work unit holds little data for the pipeline's per-item
// cost (the copies lane 0 issues, the bounded wait, the level table).  A work
// item here is KU adjacent units of one row: its codes (KU UE bytes) and the
// parameters of its KU NG groups arrive in five bulk copies, and the warp
// maps them with the lane layout of one unit, KU times.  Per element:
// W^ = fl(Delta fl(l(c) - z_U)), l(c) = level_of(c) of the element's group.

// Largest number of groups in one keep item (bounds the per-warp level table).
constexpr int kKeepMaxGroups = 16;

template <int Q, int G_, int KU>
struct KeepStage {
    using U1 = Stage<Q, WBF16, G_, false, false, true, UQ_KEEP_STAGE_BYTES>;    // lane mapping of one unit
    static constexpr int LPG = U1::LPG, NG = U1::NG, NV = U1::NV, UE = U1::UE;
    static constexpr int NGK = KU * NG;                 // groups per item
    static constexpr int SZ_C = KU * UE, SZ_P = NGK * 4, SZ_A = NGK * Q * 4;
    static constexpr int OFF_C = 0, OFF_D = SZ_C, OFF_Z = OFF_D + SZ_P, OFF_B = OFF_Z + SZ_P, OFF_A = OFF_B + SZ_P;
    static constexpr int BYTES = align_up(OFF_A + SZ_A, 128);
    static constexpr uint32_t TX = SZ_C + 3 * SZ_P + SZ_A;
    static constexpr int FIT = UQ_KEEP_STAGE_BYTES / BYTES;
    static constexpr int NST = FIT < 2 ? 2 : (FIT > kMaxStages ? kMaxStages : FIT);
    static constexpr int WARP_BYTES = NST * BYTES;
    static_assert(NGK <= kKeepMaxGroups, "level table");
    static_assert(SZ_C % 16 == 0 && SZ_P % 16 == 0 && SZ_A % 16 == 0, "bulk copy sizes must be multiples of 16");
};

template <int Q, int G_, int KU>
__global__ void __launch_bounds__(kThreads, UQ_STREAM_FWD_MIN_BLOCKS)
keep_stream_kernel(const float* __restrict__ DELTA, const float* __restrict__ ZU, const float* __restrict__ ALPHA,
                   const float* __restrict__ ZB, const uint8_t* __restrict__ CODES, float* __restrict__ WHAT,
                   int64_t out, int n_in, int R, int n_rb) {
    using St = KeepStage<Q, G_, KU>;
    constexpr int L = 1 << Q, LPG = St::LPG, NG = St::NG, NGK = St::NGK, NV = St::NV, UE = St::UE, NST = St::NST;
    extern __shared__ __align__(128) unsigned char smem[];
    __shared__ __align__(8) unsigned long long bars[kWarps][NST];
    __shared__ float lvs[kWarps][NGK][L];               // levels of the item's groups
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / LPG, li = lane % LPG;
    const int Gr = n_in / G_;
    const Items it(n_in / (KU * UE), R, n_rb, warp);
    unsigned char* wsm = smem + (size_t)warp * St::WARP_BYTES;
    float (*lv)[L] = lvs[warp];

    if (lane == 0) {
        for (int s = 0; s < NST; ++s) tma::bar_init(tma::smem_addr(&bars[warp][s]), 1);
        tma::bar_init_fence();
    }
    __syncwarp();

    auto issue = [&](const Cursor& c, int s) {           // lane 0 only
        const uint32_t bar = tma::smem_addr(&bars[warp][s]);
        const int64_t row = it.row(c.k);
        if (row >= out) { tma::bar_arrive(bar); return; }
        const int64_t e0 = row * n_in + (int64_t)it.unit(c.j) * (KU * UE);
        const int64_t g0 = row * Gr + (int64_t)it.unit(c.j) * NGK;
        const uint32_t d = tma::smem_addr(wsm + (size_t)s * St::BYTES);
        tma::fence_async_smem();
        tma::bar_arrive_tx(bar, St::TX);
        tma::copy_g2s(d + St::OFF_C, CODES + e0, St::SZ_C, bar);
        tma::copy_g2s(d + St::OFF_D, DELTA + g0, St::SZ_P, bar);
        tma::copy_g2s(d + St::OFF_Z, ZU + g0, St::SZ_P, bar);
        tma::copy_g2s(d + St::OFF_B, ZB + g0, St::SZ_P, bar);
        tma::copy_g2s(d + St::OFF_A, ALPHA + g0 * Q, St::SZ_A, bar);
    };

    const bool ok = pipe_run<NST>(it, bars[warp], lane, &g_stream_err, 1u, issue,
                                  [&](const Cursor& cc, int s) {
        const int64_t row = it.row(cc.k);
        if (row < out) {
            const unsigned char* st = wsm + (size_t)s * St::BYTES;
            const float* pd = reinterpret_cast<const float*>(st + St::OFF_D);
            const float* pz = reinterpret_cast<const float*>(st + St::OFF_Z);
            const float* pb = reinterpret_cast<const float*>(st + St::OFF_B);
            const float* pa = reinterpret_cast<const float*>(st + St::OFF_A);
#pragma unroll
            for (int e = lane; e < NGK * L; e += 32) {
                const int kk = e / L, c = e % L;
                float a[Q];
#pragma unroll
                for (int jj = 0; jj < Q; ++jj) a[jj] = pa[kk * Q + jj];
                lv[kk][c] = level_of<Q>(c, a, pb[kk]);
            }
            __syncwarp();
            const int64_t ebase = row * n_in + (int64_t)it.unit(cc.j) * (KU * UE);
#pragma unroll
            for (int ku = 0; ku < KU; ++ku) {
                const int gi = ku * NG + sub;
                const float dl = pd[gi], zu = pz[gi];
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int el = ku * UE + sub * G_ + 4 * li + 4 * LPG * v;
                    const uint32_t cv = *reinterpret_cast<const uint32_t*>(st + St::OFF_C + el);
                    float o[4];
#pragma unroll
                    for (int kq = 0; kq < 4; ++kq) o[kq] = __fmul_rn(dl, __fsub_rn(lv[gi][(cv >> (8 * kq)) & (L - 1)], zu));
                    // streaming store (evict-first): 57.3 -> 55.2 us on 14336 x 4096; the
                    // same hint on the other kernels' outputs changed nothing
                    __stcs(reinterpret_cast<float4*>(WHAT + ebase + el), make_float4(o[0], o[1], o[2], o[3]));
                }
            }
        }
                                  });
    if (!ok) return;                                 // no block barrier in this kernel
}

// ---------------------------------------------------------------------------
// Launchers
// ---------------------------------------------------------------------------

int sm_count() {
    static std::atomic<int> cached[kMaxDevices] = {};
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    if (dev >= 0 && dev < kMaxDevices) {
        const int c = cached[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) return 1;
    if (dev >= 0 && dev < kMaxDevices) cached[dev].store(n, std::memory_order_relaxed);
    return n;
}

bool stream_path_ok(const Shape& sh) {
    if (!(sh.g == 32 || sh.g == 64 || sh.g == 128)) return false;
    const int ue = sh.g == 32 ? 256 : 512;
    return sh.n_in % ue == 0;
}

template <typename St, bool ELEM>
struct BwdTag {};

template <int Q, typename WT, int G_, bool ELEM>
static cudaError_t run_bwd_stream(const Shape& sh, const void* W, uq_params p, const uint8_t* codes,
                                  const float* gup, uq_grads gr, cudaStream_t st) {
    using St = Stage<Q, WT, G_, true, true, true, UQ_BWD_STAGE_BYTES>;
    const int U = sh.n_in / St::UE;
    const int R = rows_per_block(U);
    const int n_rb = (int)((sh.out + R - 1) / R);
    const size_t dyn = (size_t)kWarps * St::WARP_BYTES;
    auto kern = bwd_stream_kernel<Q, WT, G_, ELEM>;
    int grid = 0;
    // one occupancy cache (and shared-memory opt-in) per kernel variant
    cudaError_t e = grid_for<BwdTag<St, ELEM>>(kern, dyn, n_rb, grid);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, dyn, st>>>(W, p.s, p.sr, p.delta, p.zu, p.alpha, p.zb, codes, gup, gr.ds, gr.dsr,
                                      gr.ddelta, gr.dzu, gr.dzb, gr.dalpha, sh.out, sh.n_in, R, n_rb,
                                      U >= kBranchyUnits ? 1 : 0);
    return cudaGetLastError();
}

template <int Q, typename WT, int G_, int MODE>
static cudaError_t run_fwd_stream_mode(const Shape& sh, const void* W, uq_params p, uint8_t* codes, float* what,
                                       cudaStream_t st) {
    using St = Stage<Q, WT, G_, true, false, MODE != FWD_FULL, UQ_FWD_STAGE_BYTES>;
    const int U = sh.n_in / St::UE;
    const int R = rows_per_block(U);
    const int n_rb = (int)((sh.out + R - 1) / R);
    const size_t dyn = (size_t)kWarps * St::WARP_BYTES;
    auto kern = fwd_stream_kernel<Q, WT, G_, MODE>;
    int grid = 0;
    cudaError_t e = grid_for<St>(kern, dyn, n_rb, grid);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, dyn, st>>>(W, p.s, p.sr, p.delta, p.zu, p.alpha, p.zb, codes, what, sh.out, sh.n_in, R,
                                      n_rb);
    return cudaGetLastError();
}

template <int Q, int G_, int KU>
static cudaError_t run_keep_stream(const Shape& sh, uq_params p, const uint8_t* codes, float* what, cudaStream_t st) {
    using St = KeepStage<Q, G_, KU>;
    const int U = sh.n_in / (KU * St::UE);
    const int R = rows_per_block(U);
    const int n_rb = (int)((sh.out + R - 1) / R);
    const size_t dyn = (size_t)kWarps * St::WARP_BYTES;
    auto kern = keep_stream_kernel<Q, G_, KU>;
    int grid = 0;
    cudaError_t e = grid_for<St>(kern, dyn, n_rb, grid);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, dyn, st>>>(p.delta, p.zu, p.alpha, p.zb, codes, what, sh.out, sh.n_in, R, n_rb);
    return cudaGetLastError();
}

// Units per keep item: as many adjacent units (up to 4 and kKeepMaxGroups
// groups) as divide a row's units.
template <int Q, int G_>
static cudaError_t keep_stream(const Shape& sh, uq_params p, const uint8_t* codes, float* what, cudaStream_t st) {
    constexpr int UE = KeepStage<Q, G_, 1>::UE, NG = KeepStage<Q, G_, 1>::NG;
    constexpr int KMAX = kKeepMaxGroups / NG >= 4 ? 4 : 2;     // NG is 4 or 8
    const int U = sh.n_in / UE;
    if (U % KMAX == 0) return run_keep_stream<Q, G_, KMAX>(sh, p, codes, what, st);
    if (KMAX == 4 && U % 2 == 0) return run_keep_stream<Q, G_, 2>(sh, p, codes, what, st);
    return run_keep_stream<Q, G_, 1>(sh, p, codes, what, st);
}

template <int Q, typename WT, int G_>
static cudaError_t run_fwd_stream(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode,
                                  float* what, cudaStream_t st) {
    if (mode == FWD_KEEP) return keep_stream<Q, G_>(sh, p, codes, what, st);
    if (mode == FWD_REMAP) return run_fwd_stream_mode<Q, WT, G_, FWD_REMAP>(sh, W, p, codes, what, st);
    return run_fwd_stream_mode<Q, WT, G_, FWD_FULL>(sh, W, p, codes, what, st);
}

template <int Q, typename WT, bool ELEM>
static cudaError_t bwd_stream_gf(const Shape& sh, const void* W, uq_params p, const uint8_t* codes,
                                 const float* gup, uq_grads gr, cudaStream_t st) {
    if (sh.g == 32) return run_bwd_stream<Q, WT, 32, ELEM>(sh, W, p, codes, gup, gr, st);
    if (sh.g == 64) return run_bwd_stream<Q, WT, 64, ELEM>(sh, W, p, codes, gup, gr, st);
    return run_bwd_stream<Q, WT, 128, ELEM>(sh, W, p, codes, gup, gr, st);
}

template <int Q, typename WT>
static cudaError_t bwd_stream_g(const Shape& sh, const void* W, uq_params p, const uint8_t* codes,
                                const float* gup, uq_grads gr, int filter, cudaStream_t st) {
    if (filter == UQ_FILTER_ELEMENT) return bwd_stream_gf<Q, WT, true>(sh, W, p, codes, gup, gr, st);
    return bwd_stream_gf<Q, WT, false>(sh, W, p, codes, gup, gr, st);
}

template <int Q, typename WT>
static cudaError_t fwd_stream_g(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode,
                                float* what, cudaStream_t st) {
    if (sh.g == 32) return run_fwd_stream<Q, WT, 32>(sh, W, p, codes, mode, what, st);
    if (sh.g == 64) return run_fwd_stream<Q, WT, 64>(sh, W, p, codes, mode, what, st);
    return run_fwd_stream<Q, WT, 128>(sh, W, p, codes, mode, what, st);
}

template <int Q>
static cudaError_t bwd_stream_w(const Shape& sh, const void* W, uq_params p, const uint8_t* codes,
                                const float* gup, uq_grads gr, int filter, cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return bwd_stream_g<Q, WBF16>(sh, W, p, codes, gup, gr, filter, st);
    return bwd_stream_g<Q, WF32>(sh, W, p, codes, gup, gr, filter, st);
}

template <int Q>
static cudaError_t fwd_stream_w(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode,
                                float* what, cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return fwd_stream_g<Q, WBF16>(sh, W, p, codes, mode, what, st);
    return fwd_stream_g<Q, WF32>(sh, W, p, codes, mode, what, st);
}

cudaError_t launch_bwd_stream(const Shape& sh, const void* W, uq_params p, const uint8_t* codes, const float* gup,
                              uq_grads gr, cudaStream_t st, int filter) {
    switch (sh.q) {
        case 1: return bwd_stream_w<1>(sh, W, p, codes, gup, gr, filter, st);
        case 2: return bwd_stream_w<2>(sh, W, p, codes, gup, gr, filter, st);
        case 3: return bwd_stream_w<3>(sh, W, p, codes, gup, gr, filter, st);
        default: return bwd_stream_w<4>(sh, W, p, codes, gup, gr, filter, st);
    }
}

cudaError_t launch_fwd_stream(const Shape& sh, const void* W, uq_params p, uint8_t* codes, int mode, float* what,
                              cudaStream_t st) {
    switch (sh.q) {
        case 1: return fwd_stream_w<1>(sh, W, p, codes, mode, what, st);
        case 2: return fwd_stream_w<2>(sh, W, p, codes, mode, what, st);
        case 3: return fwd_stream_w<3>(sh, W, p, codes, mode, what, st);
        default: return fwd_stream_w<4>(sh, W, p, codes, mode, what, st);
    }
}

// Self-test of the bounded wait: one warp waits on an mbarrier that nothing
// ever arrives at; the wait runs out after `limit` cycles and sets the same
// device flag a pipelined kernel sets, then the warp returns.
__global__ void wait_selftest_kernel(long long limit) {
    __shared__ __align__(8) unsigned long long bar;
    const uint32_t b = tma::smem_addr(&bar);
    if (threadIdx.x == 0) {
        tma::bar_init(b, 1);
        tma::bar_init_fence();
    }
    __syncwarp();
    const bool done = tma::bar_wait(b, 0u, limit);
    if (!done && threadIdx.x == 0) atomicOr(&g_stream_err, 2u);
}

cudaError_t launch_wait_selftest(cudaStream_t st) {
    wait_selftest_kernel<<<1, 32, 0, st>>>(1ll << 24);     // ~8 ms at 2 GHz
    return cudaGetLastError();
}

cudaError_t stream_error(bool clear, unsigned int* flag) {
    unsigned int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_stream_err, sizeof(v));
    if (e != cudaSuccess) return e;
    *flag = v;
    if (clear && v) {
        const unsigned int z = 0;
        e = cudaMemcpyToSymbol(g_stream_err, &z, sizeof(z));
    }
    return e;
}

}  // namespace uq
