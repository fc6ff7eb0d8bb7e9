// Device helpers shared by the UniQuan_F kernels (sm_103a).
//
// Work decomposition of the per-step kernels (forward, backward): thread
// blocks of 8 warps own R whole rows (R = 1 for long rows, up to 8 when a
// row has fewer work units than warps).  A warp's work unit is a set of
// whole groups: NG = 32/LPG groups, LPG lanes per group, each lane owning
// vectors of 4 consecutive elements at element offsets 4*(lane%LPG) +
// 4*LPG*v of its group (v = 0..NV-1, NV = g/(4*LPG)).  One warp instruction
// for a given v therefore reads 4*LPG contiguous elements of each of the NG
// groups -- whole 128-byte segments of the fp32 streams -- and a group's
// partial sums live on LPG neighbouring lanes only.  LPG = 4 for g = 32
// (NV = 2) and g = 64, LPG = g/16 for g = 128, 256, and LPG = 32 with
// NV = g/128 for the other multiples of 128.  Every value that decides an integer is computed with explicitly
// rounded intrinsics (__fadd_rn, __fmul_rn, __fdiv_rn): no FMA contraction,
// IEEE division, the operation order written in uq_api.h.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/uq_api.h"

namespace uq {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr unsigned kFull = 0xffffffffu;

// Weight-storage adaptors: 4 consecutive weights per lane.
struct WF32 {
    using raw = float4;
    static __device__ __forceinline__ raw load(const void* base, int64_t i) {
        return __ldg(reinterpret_cast<const float4*>(static_cast<const float*>(base) + i));
    }
    static __device__ __forceinline__ void unpack(const raw& r, float v[4]) {
        v[0] = r.x; v[1] = r.y; v[2] = r.z; v[3] = r.w;
    }
};

struct WBF16 {
    using raw = uint2;   // 4 x bf16, element k in bits [16k, 16k+16) (little endian)
    static __device__ __forceinline__ raw load(const void* base, int64_t i) {
        return __ldg(reinterpret_cast<const uint2*>(static_cast<const uint16_t*>(base) + i));
    }
    static __device__ __forceinline__ void unpack(const raw& r, float v[4]) {
        v[0] = __uint_as_float(r.x << 16);
        v[1] = __uint_as_float(r.x & 0xffff0000u);
        v[2] = __uint_as_float(r.y << 16);
        v[3] = __uint_as_float(r.y & 0xffff0000u);
    }
};

__device__ __forceinline__ float4 ldg4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }
__device__ __forceinline__ void f4_to(const float4& r, float v[4]) { v[0] = r.x; v[1] = r.y; v[2] = r.z; v[3] = r.w; }

// T_F (Eq. 1): den = (Delta * s) * s_r; u = w / den; x = u + z_U.
__device__ __forceinline__ float transform_x(float w, float s, float delta, float sr, float zu, float& u) {
    const float den = __fmul_rn(__fmul_rn(delta, s), sr);
    u = __fdiv_rn(w, den);
    return __fadd_rn(u, zu);
}

// BCQ level of code word c (Sec. 2.3): ((c_1 a_1 + c_2 a_2) + ... ) + z_B.
template <int Q>
__device__ __forceinline__ float level_of(int c, const float a[Q], float zb) {
    float acc = (c & 1) ? a[0] : -a[0];
#pragma unroll
    for (int j = 1; j < Q; ++j) acc = __fadd_rn(acc, ((c >> j) & 1) ? a[j] : -a[j]);
    return __fadd_rn(acc, zb);
}

// Full mapping M_B over the sorted levels held in registers: argmin over
// ranks of |x - l|, first (lowest) rank wins ties.  Returns the rank; m is
// the chosen level.
template <int L>
__device__ __forceinline__ int nearest_rank(float x, const float srt[L], float& m) {
    float best = fabsf(__fsub_rn(x, srt[0]));
    int br = 0;
    m = srt[0];
#pragma unroll
    for (int r = 1; r < L; ++r) {
        const float d = fabsf(__fsub_rn(x, srt[r]));
        if (d < best) { best = d; br = r; m = srt[r]; }
    }
    return br;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
    return v;
}

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
    return v;
}


// ---------------------------------------------------------------------------
// Unit-mapped tables (NS group slots per warp)
// ---------------------------------------------------------------------------

template <int Q, int NS>
struct LvTab {                       // levels by code word and tau per slot
    static constexpr int L = 1 << Q;
    float lv[NS][L];
    float tau[NS];
};

template <int Q, int NS>
struct MapTab {                      // + sorted order and local-mapping neighbours
    static constexpr int L = 1 << Q;
    float lv[NS][L];
    float srt[NS][L];
    float4 nb[NS][L];
    uint8_t cor[NS][L];
    uint8_t rk[NS][L];
};

// Levels l(c) of the NS groups grp0 + k (k < n_ok), tau = min_j |alpha_j| and,
// if amag is given, sum_j |alpha_j| + |z_B| (a bound on every |l(c)|).
// Whole warp; ends with __syncwarp().
template <int Q, int NS, typename TAB>
__device__ __forceinline__ void unit_levels(TAB& t, float* tau, int lane, const float* __restrict__ alpha,
                                            const float* __restrict__ zb, int64_t grp0, int n_ok,
                                            float* amag = nullptr) {
    constexpr int L = 1 << Q;
    constexpr int E = NS * L;
#pragma unroll
    for (int e = lane; e < E; e += 32) {
        const int k = e / L, c = e % L;
        float lvv = 0.f;
        if (k < n_ok) {
            const int64_t grp = grp0 + k;
            float a[Q];
#pragma unroll
            for (int j = 0; j < Q; ++j) a[j] = __ldg(alpha + grp * Q + j);
            const float zbv = __ldg(zb + grp);
            lvv = level_of<Q>(c, a, zbv);
            if (tau != nullptr && c == 0) {
                float m = fabsf(a[0]);
#pragma unroll
                for (int j = 1; j < Q; ++j) m = fminf(m, fabsf(a[j]));
                tau[k] = m;
                if (amag != nullptr) {
                    float s = fabsf(zbv);
#pragma unroll
                    for (int j = 0; j < Q; ++j) s = __fadd_rn(s, fabsf(a[j]));
                    amag[k] = s;
                }
            }
        }
        t.lv[k][c] = lvv;
    }
    __syncwarp();
}

// Sorted order (ascending, ties by code word) and, if NB, the neighbour
// triples of the local mapping.  Requires t.lv; ends with __syncwarp().
template <int Q, int NS, bool NB>
__device__ __forceinline__ void unit_sort(MapTab<Q, NS>& t, int lane) {
    constexpr int L = 1 << Q;
    constexpr int E = NS * L;
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
        t.rk[k][c] = static_cast<uint8_t>(r);
    }
    __syncwarp();
    if constexpr (NB) {
#pragma unroll
        for (int e = lane; e < E; e += 32) {
            const int k = e / L, c = e % L;
            const int r = t.rk[k][c];
            const int rl = r > 0 ? r - 1 : 0;
            const int rh = r < L - 1 ? r + 1 : L - 1;
            const uint32_t packed = uint32_t(t.cor[k][rl]) | (uint32_t(t.cor[k][rh]) << 8);
            t.nb[k][c] = make_float4(t.srt[k][rl], t.lv[k][c], t.srt[k][rh], __uint_as_float(packed));
        }
        __syncwarp();
    }
}

// Reduce-scatter of 8 partial sums over LPG consecutive lanes (LPG = 2..32).
// The first min(3, log2 LPG) butterfly levels halve the live values while
// exchanging the other half with the partner lane; remaining levels sum the
// last value.  On return v[0..NOUT) hold the segment totals of slots
// slot0 .. slot0+NOUT-1; lanes with (lane % LPG) a multiple of LPG/8 (all
// lanes if LPG <= 8) hold distinct slots.  Fixed order: deterministic.
template <int LPG>
struct SegReduce {
    static constexpr int HALV = LPG >= 8 ? 3 : (LPG == 4 ? 2 : 1);
    static constexpr int NOUT = 8 >> HALV;
    static __device__ __forceinline__ int run(float v[8], int lane) {
        int base = 0;
#pragma unroll
        for (int lvl = 0; lvl < HALV; ++lvl) {
            const int off = LPG >> (lvl + 1);
            const int h = 4 >> lvl;
            const bool up = (lane & off) != 0;
#pragma unroll
            for (int i = 0; i < h; ++i) {
                const float send = up ? v[i] : v[i + h];
                const float keep = up ? v[i + h] : v[i];
                v[i] = keep + __shfl_xor_sync(kFull, send, off);
            }
            base += up ? h : 0;
        }
#pragma unroll
        for (int off = LPG >> (HALV + 1); off >= 1; off >>= 1) v[0] += __shfl_xor_sync(kFull, v[0], off);
        return base;
    }
    static __device__ __forceinline__ bool writer(int lane) {
        return LPG <= 8 ? true : ((lane % LPG) % (LPG / 8)) == 0;
    }
};

// ---------------------------------------------------------------------------
// Backward terms of the pipelined kernels (App. C.1 filter, Eq. 1, Eq. 3)
// ---------------------------------------------------------------------------
//
// The filter f = (|x - w~| <= tau) decides an integer-like outcome, so it is
// always taken on the IEEE value x = fl(fl(w / den) + z_U).  The gradient
// values only need u = w / den to a few ulps.  The pipelined backward
// therefore forms u from the hardware reciprocal estimate of den (PTX
// rcp.approx.ftz.f32, relative error at most 2^-23 for normal results) and
// takes the filter from it only where that is provably the IEEE decision:
//
//   with u' = fl(w r), x' = fl(u' + z_U), d' = fl(x' - w~): |u' - u| <=
//   2^-22 |u'| (the reciprocal's 2^-23 plus one rounding on each side), and
//   one rounding of each sum on each side adds 2^-23 of its magnitude, so
//   |d' - d| <= 2^-21 |x'| + 2^-22 |z_U| + 2^-23 |w~| to first order
//   (subnormal results add at most 2^-148).
//
// With E = 2^-18 |x'| + 2^-19 (|z_U| + sum_j |alpha_j| + |z_B|) + 2^-126 (at
// least eight times that bound, since |w~| <= sum_j |alpha_j| + |z_B|), a
// vector of 4 elements whose every ||d'| - tau| exceeds E, with every |den|
// below 2^125 (so that r is a normal number), gets the same filter as the
// IEEE path.  Any other vector -- one element near the filter boundary, a
// den outside that range, an infinity or a NaN anywhere (every comparison
// with them is false) -- is recomputed with the IEEE division.  Either way
// every decision equals that of x computed by transform_x.
//
// The same reciprocal gives 1/s = r (Delta s_r), so ds = -G Delta f u / s =
// -(G f u) (r k) with k = (Delta Delta) s_r per group and row; a group whose
// k is not a normal number below 2^125 takes the IEEE path for every vector
// (eg = infinity below).

__device__ __forceinline__ float rcp_approx(float x) {
    float r;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
    return r;
}

// Per group: the part of E that does not depend on the element, or infinity
// when the reciprocal path may not be used for the group (k out of range).
// mag = |z_U| + sum_j |alpha_j| + |z_B|.
__device__ __forceinline__ float bwd_margin_of(float mag, float k) {
    const bool k_ok = fabsf(k) < 0x1p125f && fabsf(k) >= 0x1p-125f;
    return k_ok ? __fmaf_rn(mag, 0x1p-19f, 0x1p-126f) : __int_as_float(0x7f800000);
}
__device__ __forceinline__ float bwd_margin(float zu, float zb, const float* alpha, int q, float k) {
    float m = __fadd_rn(fabsf(zu), fabsf(zb));
    for (int j = 0; j < q; ++j) m = __fadd_rn(m, fabsf(alpha[j]));
    return bwd_margin_of(m, k);
}

// Backward of 4 consecutive elements of one group.  tab[c] = (l(c), l(c) -
// z_U) for code word c.  Writes ds (dL/ds), and accumulates
//   acc[0] += G (w~ - z_U - f u)      (dDelta)
//   acc[1] += G (1 - f)               (dz_U / -Delta)
//   acc[2] += G                       (dz_B / Delta; S)
//   acc[3] += G f u                   (Delta-free part of ds_r)
//   acc[4 + j] += G where bit j of c is set (P_j; dalpha_j = Delta (2 P_j - S))
// ELEM: the whole-element filter (G -> f G in every term).
template <int Q, bool ELEM>
__device__ __forceinline__ void bwd_vec4(const float w[4], const float s4[4], const float G[4], uint32_t cv,
                                         const float2* __restrict__ tab, float dl, float sr, float zu, float tau,
                                         float eg, float k, float ds[4], float acc[8]) {
    constexpr int L = 1 << Q;
    float2 mm[4];
    float u[4], d[4], rk[4];
    bool sure = true;
#pragma unroll
    for (int kq = 0; kq < 4; ++kq) {
        mm[kq] = tab[(cv >> (8 * kq)) & (L - 1)];
        const float den = __fmul_rn(__fmul_rn(dl, s4[kq]), sr);
        const float r = rcp_approx(den);
        u[kq] = __fmul_rn(w[kq], r);
        const float x = __fadd_rn(u[kq], zu);
        d[kq] = __fsub_rn(x, mm[kq].x);
        rk[kq] = __fmul_rn(r, k);
        const float E = __fmaf_rn(fabsf(x), 0x1p-18f, eg);
        sure = sure & (fabsf(__fsub_rn(fabsf(d[kq]), tau)) > E) & (fabsf(den) < 0x1p125f);
    }
    if (!sure) {
#pragma unroll
        for (int kq = 0; kq < 4; ++kq) {
            const float x = transform_x(w[kq], s4[kq], dl, sr, zu, u[kq]);
            d[kq] = __fsub_rn(x, mm[kq].x);
            rk[kq] = __fdividef(dl, s4[kq]);
        }
    }
#pragma unroll
    for (int kq = 0; kq < 4; ++kq) {
        const int c = (cv >> (8 * kq)) & (L - 1);
        const bool f = fabsf(d[kq]) <= tau;
        const float fu = f ? u[kq] : 0.f;
        const float gk = (ELEM && !f) ? 0.f : G[kq];
        const float gfu = __fmul_rn(gk, fu);
        ds[kq] = -__fmul_rn(gfu, rk[kq]);
        acc[0] = __fmaf_rn(gk, __fsub_rn(mm[kq].y, fu), acc[0]);
        acc[1] = f ? acc[1] : __fadd_rn(acc[1], gk);
        acc[2] = __fadd_rn(acc[2], gk);
        acc[3] = __fadd_rn(acc[3], gfu);
#pragma unroll
        for (int j = 0; j < Q; ++j)
            if ((c >> j) & 1) acc[4 + j] = __fadd_rn(acc[4 + j], gk);
    }
}

// ---------------------------------------------------------------------------
// Local remap step (Algorithm 4) from the reciprocal, with a proof
// ---------------------------------------------------------------------------
//
// On a remap step the code word c of an element is kept unless the level
// below it (rank r - 1) or above it (rank r + 1) is strictly nearer to the
// IEEE value x = fl(fl(w / den) + z_U) (the tie rules of the exact path).
// Used by the pipelined forward; the fused step keeps the exact path (the
// interval test made its register-bound kernel no faster).
// Per group slot k and code word c, unit_remap_iv stores iv = (a, b, w^, 0):
//   a = mid(l_lo, l_c) + m_lo, b = mid(l_c, l_hi) - m_hi  (fp32), with
//   mid(p, q) = 0.5 (p + q) and m = 2^-18 (|mid| + |z_U| + M) + 2^-126,
//   M = max |level| of the group; a = -inf when l_lo == l_c and b = +inf
//   when l_hi == l_c (equal levels never win: ties keep c);
//   w^ = Delta (l_c - z_U), the output of a kept code.
// remap_vec4 forms x' = fl(fl(w r) + z_U) from the reciprocal estimate r of
// den (as bwd_vec4 does; |x' - x| <= 2^-21 |x'| + 2^-22 |z_U| + 2^-148) and
// keeps an element's code when its x' lies in (a, b) and |den| < 2^125
// (for the same element slot of every lane of the warp: the verdict is
// taken per warp).  Then each x lies more than m / 2 from the
// midpoint on a finite side, where the fp32 distances to the two levels
// differ by more than m - 2^-22 M > 0, or beyond the level on that side
// (the far level is then never strictly nearer: rounding is monotonic); so
// the exact path keeps c as well.  Every other element slot -- an element
// near a midpoint, one whose code moves, a den out of range, an infinity or
// a NaN (all comparisons false) -- takes the exact path: transform_x and
// the three distances.
template <int Q, int NS>
__device__ __forceinline__ void unit_remap_iv(const MapTab<Q, NS>& t, float4 (*iv)[1 << Q], int lane,
                                              const float* pd, const float* pz) {
    constexpr int L = 1 << Q;
    constexpr int E = NS * L;
#pragma unroll
    for (int e = lane; e < E; e += 32) {
        const int k = e / L, c = e % L;
        const int r = t.rk[k][c];
        const int rl = r > 0 ? r - 1 : 0, rh = r < L - 1 ? r + 1 : L - 1;
        const float y = t.lv[k][c], lo = t.srt[k][rl], hi = t.srt[k][rh];
        const float zu = pz[k];
        const float M = fmaxf(fabsf(t.srt[k][0]), fabsf(t.srt[k][L - 1]));
        const float base = __fadd_rn(fabsf(zu), M);
        const float ml = __fmul_rn(0.5f, __fadd_rn(lo, y));
        const float mh = __fmul_rn(0.5f, __fadd_rn(y, hi));
        const float a = lo == y ? -__int_as_float(0x7f800000)
                                : __fadd_rn(ml, __fmaf_rn(__fadd_rn(fabsf(ml), base), 0x1p-18f, 0x1p-126f));
        const float b = hi == y ? __int_as_float(0x7f800000)
                                : __fsub_rn(mh, __fmaf_rn(__fadd_rn(fabsf(mh), base), 0x1p-18f, 0x1p-126f));
        iv[k][c] = make_float4(a, b, __fmul_rn(pd[k], __fsub_rn(y, zu)), 0.f);
    }
    __syncwarp();
}

// Remap step of 4 consecutive elements of group slot `sub`: W^ into o[],
// returns the 4 new code words packed as bytes (bits above q cleared).
// Every lane of the warp must call it (the fallback verdicts are warp-wide).
template <int Q, int NS>
__device__ __forceinline__ uint32_t remap_vec4(const float w[4], const float s4[4], uint32_t cv,
                                               const MapTab<Q, NS>& t, const float4 (*iv)[1 << Q], int sub,
                                               float dl, float sr, float zu, float o[4]) {
    constexpr int L = 1 << Q;
    uint32_t nc = 0;
#pragma unroll
    for (int kq = 0; kq < 4; ++kq) {
        const int c = (cv >> (8 * kq)) & (L - 1);
        const float4 v = iv[sub][c];
        const float den = __fmul_rn(__fmul_rn(dl, s4[kq]), sr);
        const float xa = __fadd_rn(__fmul_rn(w[kq], rcp_approx(den)), zu);
        const bool sure = (xa > v.x) & (xa < v.y) & (fabsf(den) < 0x1p125f);
        uint32_t code = c;
        o[kq] = v.z;
        // One verdict per element slot and warp: the warp redoes element kq of
        // its lanes with the exact path when any of them is unsure (the exact
        // path gives the same result where the interval already decided).
        if (__any_sync(kFull, !sure)) {
            const int r = t.rk[sub][c];
            const int rl = r > 0 ? r - 1 : 0, rh = r < L - 1 ? r + 1 : L - 1;
            float uu;
            const float x = transform_x(w[kq], s4[kq], dl, sr, zu, uu);
            float m = t.lv[sub][c];
            float best = fabsf(__fsub_rn(x, m));
            const float lo = t.srt[sub][rl];
            const float dlo = fabsf(__fsub_rn(x, lo));
            if (dlo < best) { best = dlo; m = lo; code = t.cor[sub][rl]; }
            const float hi = t.srt[sub][rh];
            const float dhi = fabsf(__fsub_rn(x, hi));
            if (dhi < best) { m = hi; code = t.cor[sub][rh]; }
            o[kq] = __fmul_rn(dl, __fsub_rn(m, zu));
        }
        nc |= code << (8 * kq);
    }
    return nc;
}

// Filter decisions of 4 elements whose x = nu / dv + z share the divisor dv
// (OmniQuant's Delta_O, AWQ's Delta_A; App. E): u = nu / dv from r =
// rcp_approx(dv) where the margin test above proves the decision equal to
// that of the IEEE quotient, else (the whole vector) from __fdiv_rn.  m[k] =
// w~ of element k; eg = bwd_margin(z, z_B, alpha, q, dv), which is infinity
// unless dv is a normal number below 2^125.  Returns u (for the gradient
// values) and f.
__device__ __forceinline__ void shared_div_filter4(const float nu[4], float dv, float r, float z, const float m[4],
                                                   float tau, float eg, float u[4], bool f[4]) {
    float d[4];
    bool sure = true;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        u[k] = __fmul_rn(nu[k], r);
        const float x = __fadd_rn(u[k], z);
        d[k] = __fsub_rn(x, m[k]);
        const float E = __fmaf_rn(fabsf(x), 0x1p-18f, eg);
        sure = sure & (fabsf(__fsub_rn(fabsf(d[k]), tau)) > E);
    }
    if (!sure) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            u[k] = __fdiv_rn(nu[k], dv);
            d[k] = __fsub_rn(__fadd_rn(u[k], z), m[k]);
        }
    }
#pragma unroll
    for (int k = 0; k < 4; ++k) f[k] = fabsf(d[k]) <= tau;
}

// After SegReduce<LPG>::run over the bwd_vec4 accumulators (LPG 4 or 8):
// S = slot 2's total, fetched from the lane that holds it.
template <int LPG>
__device__ __forceinline__ float seg_slot2(const float v[8], int lane) {
    static_assert(LPG == 4 || LPG == 8, "slot 2 sits in v[0] of lane 2 / NOUT");
    return __shfl_sync(kFull, v[0], (lane & ~(LPG - 1)) | (2 / SegReduce<LPG>::NOUT));
}

// Rows per block for the unit mapping: the largest power of two R <= 8 with
// R * units_per_row <= 8 (at least 1).
__host__ __device__ inline int rows_per_block(int units_per_row) {
    int R = 1;
    while (R < kWarps && 2 * R * units_per_row <= kWarps) R *= 2;
    return R;
}

// LPG for a group size: 4 for g = 32 (NV = 2) and g = 64, g/16 for g = 128
// and 256, else 32 (g = 512: NV = 4; larger multiples of 128: NV = g/128).
__host__ __device__ inline int lanes_per_group(int g) {
    return g <= 64 ? 4 : (g == 128 || g == 256) ? g / 16 : 32;
}

}  // namespace uq
