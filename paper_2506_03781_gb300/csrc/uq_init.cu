// Unified initialization (Algorithm 2) with the clipping strategies of
// App. E.2 and the general alternating update of Algorithm 3: one lane per
// group for g <= 128 (init_lane_kernel), one warp per group for larger
// groups (init_kernel); the group's transformed weights x and code words
// kept in shared memory.  Runs once before training; not on the per-step
// path.  A round of the alternating update that moves no code (and not z_B)
// is a fixed point: the remaining rounds are skipped, which changes nothing.
//
// Sums that feed alpha and z_B are taken in fp64 (the group's fp32 values
// are summed exactly in practice); the normal equations C^T C alpha =
// C^T (x - z_B) have an integer matrix, so singularity is decided exactly
// by an integer determinant and the system is solved in fp64 by Gaussian
// elimination with partial pivoting.
#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

constexpr int kInitMaxWarps = 8;

template <int Q>
struct InitTab {
    static constexpr int L = 1 << Q;
    float lv[L];
    float srt[L];
    uint8_t cor[L];
};

// Sorted levels of (a, zb) into registers of every lane (via the warp's table).
template <int Q>
__device__ __forceinline__ void sorted_levels(InitTab<Q>& tb, int lane, const float a[Q], float zb,
                                              float srt[1 << Q]) {
    constexpr int L = 1 << Q;
    __syncwarp();
    if (lane < L) tb.lv[lane] = level_of<Q>(lane, a, zb);
    __syncwarp();
    if (lane < L) {
        const float v = tb.lv[lane];
        int r = 0;
#pragma unroll
        for (int c2 = 0; c2 < L; ++c2) {
            const float v2 = tb.lv[c2];
            r += (v2 < v) || (v2 == v && c2 < lane);
        }
        tb.srt[r] = v;
        tb.cor[r] = static_cast<uint8_t>(lane);
    }
    __syncwarp();
#pragma unroll
    for (int r = 0; r < L; ++r) srt[r] = tb.srt[r];
}

// Exact singularity test of the integer matrix C^T C.  C^T C is a Gram
// matrix of +-1 columns, so |det| <= g^q <= 2^60 (Hadamard); the cofactor
// expansion below is evaluated with wrapping 64-bit unsigned arithmetic,
// which is exact modulo 2^64 and hence exact.
template <int Q>
__device__ __forceinline__ bool int_singular(const long long Min[Q][Q]) {
    using u64 = unsigned long long;
    u64 M[Q][Q];
#pragma unroll
    for (int i = 0; i < Q; ++i)
#pragma unroll
        for (int j = 0; j < Q; ++j) M[i][j] = (u64)Min[i][j];
    auto det3 = [&](int r0, int r1, int r2, int c0, int c1, int c2) -> u64 {
        return M[r0][c0] * (M[r1][c1] * M[r2][c2] - M[r1][c2] * M[r2][c1])
             - M[r0][c1] * (M[r1][c0] * M[r2][c2] - M[r1][c2] * M[r2][c0])
             + M[r0][c2] * (M[r1][c0] * M[r2][c1] - M[r1][c1] * M[r2][c0]);
    };
    u64 det;
    if constexpr (Q == 1) {
        det = M[0][0];
    } else if constexpr (Q == 2) {
        det = M[0][0] * M[1][1] - M[0][1] * M[1][0];
    } else if constexpr (Q == 3) {
        det = det3(0, 1, 2, 0, 1, 2);
    } else {
        det = M[0][0] * det3(1, 2, 3, 1, 2, 3) - M[0][1] * det3(1, 2, 3, 0, 2, 3)
            + M[0][2] * det3(1, 2, 3, 0, 1, 3) - M[0][3] * det3(1, 2, 3, 0, 1, 2);
    }
    return det == 0ull;
}

// Solves A x = b in fp64: Gaussian elimination with partial pivoting (first
// largest |pivot| wins) and back substitution, every product and difference
// rounded separately (no FMA contraction).  The exact solution is often an
// fp32 rounding tie (short dyadic values), so the rounding order is fixed.
template <int Q>
__device__ __forceinline__ void solve_fp64(const long long Ain[Q][Q], const double bin[Q], double x[Q]) {
    double A[Q][Q], b[Q];
#pragma unroll
    for (int i = 0; i < Q; ++i) {
        b[i] = bin[i];
#pragma unroll
        for (int j = 0; j < Q; ++j) A[i][j] = (double)Ain[i][j];
    }
#pragma unroll
    for (int k = 0; k < Q; ++k) {
        int p = k;
        double piv = fabs(A[k][k]);
#pragma unroll
        for (int i = k + 1; i < Q; ++i)
            if (fabs(A[i][k]) > piv) { piv = fabs(A[i][k]); p = i; }
#pragma unroll
        for (int i = k + 1; i < Q; ++i) {
            if (i == p) {
#pragma unroll
                for (int j = 0; j < Q; ++j) { const double tmp = A[k][j]; A[k][j] = A[i][j]; A[i][j] = tmp; }
                const double tb = b[k]; b[k] = b[i]; b[i] = tb;
            }
        }
#pragma unroll
        for (int i = k + 1; i < Q; ++i) {
            const double f = __ddiv_rn(A[i][k], A[k][k]);
#pragma unroll
            for (int j = k; j < Q; ++j) A[i][j] = __dsub_rn(A[i][j], __dmul_rn(f, A[k][j]));
            b[i] = __dsub_rn(b[i], __dmul_rn(f, b[k]));
        }
    }
#pragma unroll
    for (int i = Q - 1; i >= 0; --i) {
        double s = b[i];
#pragma unroll
        for (int j = i + 1; j < Q; ++j) s = __dsub_rn(s, __dmul_rn(A[i][j], x[j]));
        x[i] = __ddiv_rn(s, A[i][i]);
    }
}

template <int Q, typename WT>
__global__ void init_kernel(const void* __restrict__ W, int64_t n_groups, int n_in, int g, int G, int T, int clip,
                            float* __restrict__ DELTA, float* __restrict__ ZU, float* __restrict__ S,
                            float* __restrict__ SR, float* __restrict__ ALPHA, float* __restrict__ ZB,
                            uint8_t* __restrict__ CODES) {
    constexpr int L = 1 << Q;
    extern __shared__ __align__(16) unsigned char smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wpc = blockDim.x >> 5;
    __shared__ InitTab<Q> tabs[kInitMaxWarps];
    InitTab<Q>& tb = tabs[warp];
    float* xs = reinterpret_cast<float*>(smem) + (size_t)warp * g;
    uint8_t* cs = smem + (size_t)wpc * g * sizeof(float) + (size_t)warp * g;

    const int64_t grp = (int64_t)blockIdx.x * wpc + warp;
    if (grp >= n_groups) return;                       // whole warp; no block barrier follows
    const int Gr = n_in / g;
    const int64_t row = grp / Gr;
    const int64_t eoff = row * (int64_t)n_in + (grp % Gr) * (int64_t)g;
    auto wval = [&](int i) -> float {
        if constexpr (sizeof(typename WT::raw) == sizeof(float4))
            return __ldg(static_cast<const float*>(W) + eoff + i);
        else
            return __uint_as_float(uint32_t(__ldg(static_cast<const unsigned short*>(W) + eoff + i)) << 16);
    };

    float wmin = INFINITY, wmax = -INFINITY;
    for (int i = lane; i < g; i += 32) {
        const float w = wval(i);
        wmin = fminf(wmin, w);
        wmax = fmaxf(wmax, w);
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
        wmin = fminf(wmin, __shfl_xor_sync(kFull, wmin, off));
        wmax = fmaxf(wmax, __shfl_xor_sync(kFull, wmax, off));
    }
    const float top = (float)(L - 1);
    const float rng = fmaxf(__fsub_rn(wmax, wmin), 1e-12f);

    double e_best = INFINITY;
    float bd = 0.f, bz = 0.f, bzb = top * 0.5f, ba[Q];
#pragma unroll
    for (int j = 0; j < Q; ++j) ba[j] = 0.f;

    for (int gi = 1; gi <= G; ++gi) {
        const float gamma = __fdiv_rn((float)gi, (float)G);
        const float dc = __fdiv_rn(__fmul_rn(gamma, rng), top);
        float zc;
        if (clip == UQ_CLIP_FIXED_MIN) zc = __fdiv_rn(-wmin, dc);
        else if (clip == UQ_CLIP_FIXED_MAX) zc = __fsub_rn(top, __fdiv_rn(wmax, dc));
        else zc = __fdiv_rn(-__fmul_rn(gamma, wmin), dc);
        __syncwarp();
        for (int i = lane; i < g; i += 32) {
            float u;
            xs[i] = transform_x(wval(i), 1.f, dc, 1.f, zc, u);
            cs[i] = 0;
        }
        __syncwarp();

        // --- Algorithm 3: greedy start (one bit at a time) ---
        float a[Q], zb = bzb;
#pragma unroll
        for (int j = 0; j < Q; ++j) {
            double sabs = 0.0;
            for (int i = lane; i < g; i += 32) {
                float r = __fsub_rn(xs[i], zb);
                const int c = cs[i];
#pragma unroll
                for (int jj = 0; jj < j; ++jj) r = __fsub_rn(r, ((c >> jj) & 1) ? a[jj] : -a[jj]);
                sabs += (double)fabsf(r);
                if (r >= 0.f) cs[i] = (uint8_t)(c | (1 << j));
            }
            sabs = warp_sum_d(sabs);
            a[j] = (float)(sabs / (double)g);
        }
        __syncwarp();

        // --- T rounds of alpha, C (and z_B when G == 1) ---
        for (int it = 0; it < T; ++it) {
            long long ctc[Q][Q];
            double cty[Q];
#pragma unroll
            for (int j = 0; j < Q; ++j) {
                cty[j] = 0.0;
#pragma unroll
                for (int k = 0; k < Q; ++k) ctc[j][k] = 0;
            }
            const double zbd = (double)zb;
            for (int i = lane; i < g; i += 32) {
                const int c = cs[i];
                const double y = (double)xs[i] - zbd;
#pragma unroll
                for (int j = 0; j < Q; ++j) {
                    const int sj = ((c >> j) & 1) ? 1 : -1;
                    cty[j] += sj > 0 ? y : -y;
#pragma unroll
                    for (int k = j; k < Q; ++k) ctc[j][k] += (((c >> k) & 1) ? 1 : -1) * sj;
                }
            }
#pragma unroll
            for (int j = 0; j < Q; ++j) {
                cty[j] = warp_sum_d(cty[j]);
#pragma unroll
                for (int k = j; k < Q; ++k) {
                    long long v = ctc[j][k];
#pragma unroll
                    for (int off = 16; off >= 1; off >>= 1) v += __shfl_xor_sync(kFull, v, off);
                    ctc[j][k] = v;
                    ctc[k][j] = v;
                }
            }
            if (!int_singular<Q>(ctc)) {
                double sol[Q];
                solve_fp64<Q>(ctc, cty, sol);
#pragma unroll
                for (int j = 0; j < Q; ++j) a[j] = (float)sol[j];
            }
            float srt[L];
            sorted_levels<Q>(tb, lane, a, zb, srt);
            bool moved = false;
            for (int i = lane; i < g; i += 32) {
                float m;
                const int r = nearest_rank<L>(xs[i], srt, m);
                moved |= cs[i] != tb.cor[r];
                cs[i] = tb.cor[r];
            }
            moved = __any_sync(kFull, moved);
            __syncwarp();
            const float zb_prev = zb;
            if (G == 1) {
                double sres = 0.0;
                for (int i = lane; i < g; i += 32) {
                    const int c = cs[i];
                    double ca = 0.0;
#pragma unroll
                    for (int j = 0; j < Q; ++j) ca += ((c >> j) & 1) ? (double)a[j] : -(double)a[j];
                    sres += (double)xs[i] - ca;
                }
                sres = warp_sum_d(sres);
                zb = (float)(sres / (double)g);
            }
            // a fixed point (no code and not z_B moved): the remaining rounds
            // would repeat it bit for bit (warp-uniform: zb and moved are)
            if (!moved && __float_as_uint(zb) == __float_as_uint(zb_prev)) break;
        }

        // --- candidate error with the full mapping (Eq. 2), s = s_r = 1 ---
        float srt[L];
        sorted_levels<Q>(tb, lane, a, zb, srt);
        double e = 0.0;
        for (int i = lane; i < g; i += 32) {
            float m;
            nearest_rank<L>(xs[i], srt, m);
            const float what = __fmul_rn(dc, __fsub_rn(m, zc));
            const double df = (double)wval(i) - (double)what;
            e += df * df;
        }
        e = warp_sum_d(e);
        if (e < e_best) {
            e_best = e;
            bd = dc;
            bz = zc;
            bzb = zb;
#pragma unroll
            for (int j = 0; j < Q; ++j) ba[j] = a[j];
        }
    }

    if (lane == 0) {
        DELTA[grp] = bd;
        ZU[grp] = bz;
        ZB[grp] = bzb;
#pragma unroll
        for (int j = 0; j < Q; ++j) ALPHA[grp * Q + j] = ba[j];
        if (grp % Gr == 0) SR[row] = 1.f;
    }
    float srt[L];
    sorted_levels<Q>(tb, lane, ba, bzb, srt);
    for (int i = lane; i < g; i += 32) {
        float u, m;
        const float x = transform_x(wval(i), 1.f, bd, 1.f, bz, u);
        const int r = nearest_rank<L>(x, srt, m);
        CODES[eoff + i] = tb.cor[r];
        S[eoff + i] = 1.f;
    }
}

// ---------------------------------------------------------------------------
// One lane per group (g <= 128)
// ---------------------------------------------------------------------------
//
// The same computation as init_kernel, laid out for a GPU whose fp64 rate is
// a small fraction of its fp32 rate: lane l of a warp owns group 32 w + l
// whole, so every fp64 sum is lane-local (no fp64 shuffles) and each lane
// solves the normal equations of its own group once (init_kernel solves
// them on all 32 lanes of the group's warp).  During the T rounds x is
// fixed and only the code words move, so C^T (x - z_B) and C^T C are formed
// from per-code-word sums of x and counts (a round touches only the elements
// whose code moved).  Shared memory per warp, element-major so that the 32
// lanes touch consecutive words (init_lane_warp_bytes).  Every fp32
// operation and every decision is the one init_kernel takes; the fp64 sums
// run in another order (lane-sequential, grouped by code word), which gives
// the same values whenever they are exact.
constexpr int kLaneInitMaxG = 128;

// Shared memory of one warp: the per-code sums of x [L][32] fp64, x
// [g][32], the sorted levels [L][32], the code words [g][32] and the codes
// of the sorted levels [L][32]; rounded up to 16 bytes.
__host__ __device__ constexpr size_t init_lane_warp_bytes(int q, int g) {
    return (((size_t)(1 << q) * 32 * (8 + 4 + 1) + (size_t)g * 32 * (4 + 1)) + 15) & ~size_t(15);
}

// Counts of the L code words of one group (at most 255 each), 8 bits per
// code word packed in 64-bit registers; c is a compile-time index wherever
// get() is used, add() takes any c.
template <int L>
struct CodeHist {
    uint64_t lo = 0, hi = 0;                           // code words 0..7, 8..15
    __device__ __forceinline__ void add(int c, int d) {
        const uint64_t v = (uint64_t)(int64_t)d << (8 * (c & 7));
        if (L <= 8 || c < 8) lo += v;
        else hi += v;
    }
    __device__ __forceinline__ int get(int c) const {
        return (int)(((c < 8 ? lo : hi) >> (8 * (c & 7))) & 0xffu);
    }
};

template <int Q>
__device__ __forceinline__ void lane_sorted_levels(const float a[Q], float zb, float* srt_s, uint8_t* cor_s,
                                                   int lane, float srt[1 << Q], uint64_t& cor) {
    constexpr int L = 1 << Q;
    float lv[L];
#pragma unroll
    for (int c = 0; c < L; ++c) lv[c] = level_of<Q>(c, a, zb);
#pragma unroll
    for (int c = 0; c < L; ++c) {
        int r = 0;
#pragma unroll
        for (int c2 = 0; c2 < L; ++c2) r += (lv[c2] < lv[c]) || (lv[c2] == lv[c] && c2 < c);
        srt_s[r * 32 + lane] = lv[c];
        cor_s[r * 32 + lane] = static_cast<uint8_t>(c);
    }
    cor = 0;
#pragma unroll
    for (int r = 0; r < L; ++r) {
        srt[r] = srt_s[r * 32 + lane];
        cor |= uint64_t(cor_s[r * 32 + lane]) << (4 * r);
    }
}

template <int Q, typename WT, int G_>
__global__ void init_lane_kernel(const void* __restrict__ W, int64_t n_groups, int n_in, int G, int T, int clip,
                                 float* __restrict__ DELTA, float* __restrict__ ZU, float* __restrict__ S,
                                 float* __restrict__ SR, float* __restrict__ ALPHA, float* __restrict__ ZB,
                                 uint8_t* __restrict__ CODES) {
    constexpr int L = 1 << Q;
    constexpr size_t WARP_BYTES = init_lane_warp_bytes(Q, G_);
    extern __shared__ __align__(16) unsigned char smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    unsigned char* base = smem + (size_t)warp * WARP_BYTES;
    double* bx = reinterpret_cast<double*>(base);                       // [L][32]
    float* xs = reinterpret_cast<float*>(bx + L * 32);                  // [G_][32]
    float* srt_s = xs + G_ * 32;                                        // [L][32]
    uint8_t* cs = reinterpret_cast<uint8_t*>(srt_s + L * 32);           // [G_][32]
    uint8_t* cor_s = cs + G_ * 32;                                      // [L][32]

    const int64_t grp0 = ((int64_t)blockIdx.x * (blockDim.x >> 5) + warp) * 32;
    if (grp0 >= n_groups) return;                      // whole warp; no block barrier in this kernel
    const int64_t grp_raw = grp0 + lane;
    const bool live = grp_raw < n_groups;
    const int64_t grp = live ? grp_raw : n_groups - 1; // absent lanes repeat the last group, store nothing
    const int Gr = n_in / G_;
    const int64_t row = grp / Gr;
    const int64_t eoff = row * (int64_t)n_in + (grp % Gr) * (int64_t)G_;
    auto wval = [&](int i) -> float {
        if constexpr (sizeof(typename WT::raw) == sizeof(float4))
            return __ldg(static_cast<const float*>(W) + eoff + i);
        else
            return __uint_as_float(uint32_t(__ldg(static_cast<const unsigned short*>(W) + eoff + i)) << 16);
    };
    auto X = [&](int i) -> float& { return xs[i * 32 + lane]; };
    auto C = [&](int i) -> uint8_t& { return cs[i * 32 + lane]; };
    auto BX = [&](int c) -> double& { return bx[c * 32 + lane]; };

    float wmin = INFINITY, wmax = -INFINITY;
#pragma unroll 2
    for (int i = 0; i < G_; ++i) {
        const float w = wval(i);
        wmin = fminf(wmin, w);
        wmax = fmaxf(wmax, w);
    }
    const float top = (float)(L - 1);
    const float rng = fmaxf(__fsub_rn(wmax, wmin), 1e-12f);

    double e_best = INFINITY;
    float bd = 0.f, bz = 0.f, bzb = top * 0.5f, ba[Q];
#pragma unroll
    for (int j = 0; j < Q; ++j) ba[j] = 0.f;
    float srt[L];
    uint64_t cor;

    for (int gi = 1; gi <= G; ++gi) {
        const float gamma = __fdiv_rn((float)gi, (float)G);
        const float dc = __fdiv_rn(__fmul_rn(gamma, rng), top);
        float zc;
        if (clip == UQ_CLIP_FIXED_MIN) zc = __fdiv_rn(-wmin, dc);
        else if (clip == UQ_CLIP_FIXED_MAX) zc = __fsub_rn(top, __fdiv_rn(wmax, dc));
        else zc = __fdiv_rn(-__fmul_rn(gamma, wmin), dc);
#pragma unroll 2
        for (int i = 0; i < G_; ++i) {
            float u;
            X(i) = transform_x(wval(i), 1.f, dc, 1.f, zc, u);
            C(i) = 0;
        }

        // --- Algorithm 3: greedy start (one bit at a time) ---
        float a[Q], zb = bzb;
#pragma unroll
        for (int j = 0; j < Q; ++j) {
            double sabs = 0.0;
#pragma unroll 2
            for (int i = 0; i < G_; ++i) {
                float r = __fsub_rn(X(i), zb);
                const int c = C(i);
#pragma unroll
                for (int jj = 0; jj < j; ++jj) r = __fsub_rn(r, ((c >> jj) & 1) ? a[jj] : -a[jj]);
                sabs += (double)fabsf(r);
                if (r >= 0.f) C(i) = (uint8_t)(c | (1 << j));
            }
            a[j] = (float)(sabs / (double)G_);
        }
        // Per code word c: the fp64 sum of x over the group's elements with
        // code c (bx) and their count (hist).  Then C^T (x - z_B) =
        // sum_c s(c) (bx_c - n_c z_B) and C^T C = sum_c n_c s(c) s(c)^T, where
        // s(c) is the sign vector of c; a round only moves the elements whose
        // code changed from one sum to the other.
        CodeHist<L> hist;
#pragma unroll
        for (int c = 0; c < L; ++c) BX(c) = 0.0;
#pragma unroll 2
        for (int i = 0; i < G_; ++i) {
            const int c = C(i);
            BX(c) += (double)X(i);
            hist.add(c, 1);
        }

        // --- T rounds of alpha, C (and z_B when G == 1) ---
        for (int it = 0; it < T; ++it) {
            long long ctc[Q][Q];
            double cty[Q];
#pragma unroll
            for (int j = 0; j < Q; ++j) {
                cty[j] = 0.0;
#pragma unroll
                for (int k = 0; k < Q; ++k) ctc[j][k] = 0;
            }
            const double zbd = (double)zb;
#pragma unroll
            for (int c = 0; c < L; ++c) {
                const int n = hist.get(c);
                const double yc = BX(c) - (double)n * zbd;
#pragma unroll
                for (int j = 0; j < Q; ++j) {
                    const bool sj = (c >> j) & 1;
                    cty[j] += sj ? yc : -yc;
#pragma unroll
                    for (int k = j; k < Q; ++k) ctc[j][k] += (sj == (bool)((c >> k) & 1)) ? n : -n;
                }
            }
#pragma unroll
            for (int j = 0; j < Q; ++j)
#pragma unroll
                for (int k = 0; k < j; ++k) ctc[j][k] = ctc[k][j];
            if (!int_singular<Q>(ctc)) {
                double sol[Q];
                solve_fp64<Q>(ctc, cty, sol);
#pragma unroll
                for (int j = 0; j < Q; ++j) a[j] = (float)sol[j];
            }
            lane_sorted_levels<Q>(a, zb, srt_s, cor_s, lane, srt, cor);
            bool moved = false;
#pragma unroll 2
            for (int i = 0; i < G_; ++i) {
                float m;
                const float x = X(i);
                const int r = nearest_rank<L>(x, srt, m);
                const int c = (int)((cor >> (4 * r)) & 15u);
                const int old = C(i);
                if (c != old) {
                    moved = true;
                    const double xd = (double)x;
                    BX(old) -= xd;
                    BX(c) += xd;
                    hist.add(old, -1);
                    hist.add(c, 1);
                    C(i) = (uint8_t)c;
                }
            }
            const float zb_prev = zb;
            if (G == 1) {
                // z_B = mean of x - C alpha = sum_c (bx_c - n_c (s(c) . alpha)) / g
                double sres = 0.0;
#pragma unroll
                for (int c = 0; c < L; ++c) {
                    double ca = 0.0;
#pragma unroll
                    for (int j = 0; j < Q; ++j) ca += ((c >> j) & 1) ? (double)a[j] : -(double)a[j];
                    sres += BX(c) - (double)hist.get(c) * ca;
                }
                zb = (float)(sres / (double)G_);
            }
            // No code moved (and z_B did not either): the next round would
            // solve the same system, get the same alpha and the same codes, so
            // every remaining round repeats this state bit for bit.
            if (!moved && __float_as_uint(zb) == __float_as_uint(zb_prev)) break;
        }

        // --- candidate error with the full mapping (Eq. 2), s = s_r = 1 ---
        lane_sorted_levels<Q>(a, zb, srt_s, cor_s, lane, srt, cor);
        double e = 0.0;
#pragma unroll 2
        for (int i = 0; i < G_; ++i) {
            float m;
            nearest_rank<L>(X(i), srt, m);
            const float what = __fmul_rn(dc, __fsub_rn(m, zc));
            const double df = (double)wval(i) - (double)what;
            e += df * df;
        }
        if (e < e_best) {
            e_best = e;
            bd = dc;
            bz = zc;
            bzb = zb;
#pragma unroll
            for (int j = 0; j < Q; ++j) ba[j] = a[j];
        }
    }

    lane_sorted_levels<Q>(ba, bzb, srt_s, cor_s, lane, srt, cor);
    if (!live) return;                                 // no warp-wide operation follows
    DELTA[grp] = bd;
    ZU[grp] = bz;
    ZB[grp] = bzb;
#pragma unroll
    for (int j = 0; j < Q; ++j) ALPHA[grp * Q + j] = ba[j];
    if (grp % Gr == 0) SR[row] = 1.f;
#pragma unroll 2
    for (int i = 0; i < G_; ++i) {
        float u, m;
        const float x = transform_x(wval(i), 1.f, bd, 1.f, bz, u);
        const int r = nearest_rank<L>(x, srt, m);
        CODES[eoff + i] = (uint8_t)((cor >> (4 * r)) & 15u);
        S[eoff + i] = 1.f;
    }
}

template <int Q, typename WT, int G_>
static cudaError_t run_init_lane(const Shape& sh, const void* W, int G, int T, int clip, uq_params p,
                                 uint8_t* codes, cudaStream_t st) {
    constexpr int L = 1 << Q;
    constexpr size_t warp_bytes = init_lane_warp_bytes(Q, G_);
    // as many warps as fit in the 227 KB a block may opt in to, at most 16
    constexpr int wpb = (int)((227 * 1024) / warp_bytes) > 16 ? 16 : (int)((227 * 1024) / warp_bytes);
    static_assert(wpb >= 1, "one warp's tables must fit");
    const int64_t n_groups = sh.out * (int64_t)(sh.n_in / G_);
    const size_t dyn = warp_bytes * wpb;
    auto kern = init_lane_kernel<Q, WT, G_>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
    if (e != cudaSuccess) return e;
    const int64_t per_block = (int64_t)wpb * 32;
    const int64_t blocks = (n_groups + per_block - 1) / per_block;
    kern<<<dim3((unsigned)blocks), wpb * 32, dyn, st>>>(W, n_groups, sh.n_in, G, T, clip, p.delta, p.zu, p.s, p.sr,
                                                       p.alpha, p.zb, codes);
    return cudaGetLastError();
}

template <int Q, typename WT>
static cudaError_t run_init(const Shape& sh, const void* W, int G, int T, int clip, uq_params p, uint8_t* codes,
                            cudaStream_t st) {
    if (sh.g == 32) return run_init_lane<Q, WT, 32>(sh, W, G, T, clip, p, codes, st);
    if (sh.g == 64) return run_init_lane<Q, WT, 64>(sh, W, G, T, clip, p, codes, st);
    if (sh.g == kLaneInitMaxG) return run_init_lane<Q, WT, 128>(sh, W, G, T, clip, p, codes, st);
    const int64_t n_groups = sh.out * (int64_t)(sh.n_in / sh.g);
    const size_t per_warp = (size_t)sh.g * (sizeof(float) + 1);
    int wpc = (int)((96 * 1024) / per_warp);
    wpc = wpc < 1 ? 1 : (wpc > kInitMaxWarps ? kInitMaxWarps : wpc);
    const size_t dyn = per_warp * wpc;
    auto kern = init_kernel<Q, WT>;
    if (dyn > 32 * 1024) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e != cudaSuccess) return e;
    }
    const int64_t blocks = (n_groups + wpc - 1) / wpc;
    kern<<<dim3((unsigned)blocks), wpc * 32, dyn, st>>>(W, n_groups, sh.n_in, sh.g, G, T, clip, p.delta, p.zu,
                                                          p.s, p.sr, p.alpha, p.zb, codes);
    return cudaGetLastError();
}

template <int Q>
static cudaError_t init_w(const Shape& sh, const void* W, int G, int T, int clip, uq_params p, uint8_t* codes,
                          cudaStream_t st) {
    if (sh.wdtype == UQ_W_BF16) return run_init<Q, WBF16>(sh, W, G, T, clip, p, codes, st);
    return run_init<Q, WF32>(sh, W, G, T, clip, p, codes, st);
}

cudaError_t launch_init(const Shape& sh, const void* W, int G, int T, int clip, uq_params p, uint8_t* codes,
                        cudaStream_t st) {
    switch (sh.q) {
        case 1: return init_w<1>(sh, W, G, T, clip, p, codes, st);
        case 2: return init_w<2>(sh, W, G, T, clip, p, codes, st);
        case 3: return init_w<3>(sh, W, G, T, clip, p, codes, st);
        default: return init_w<4>(sh, W, G, T, clip, p, codes, st);
    }
}

}  // namespace uq
