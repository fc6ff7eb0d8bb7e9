// BCQ matrix-vector product from the exported format: y = W~ x with
// W~[r, i] = sum_j alpha*_{r,k,j} c_{j,r,i} + z*_{r,k} (k = i / g), the
// binary codes c = +-1 read from the bit-planes (Theorem 1 folds D_R into
// alpha*, z*, so this is the whole inference computation; App. F.1 format).
//
// Per row and group the product splits into one sum per bit-plane:
//   sum_i W~_ri x_i = sum_j alpha*_j (2 P_j - S) + z* S,
//   P_j = sum of x_i over the columns whose bit j is set,  S = sum of x_i.
// P_j is read from lookup tables: for every 8 consecutive columns, the 256
// possible sums of their x values, indexed by one byte of the plane.  The
// columns are cut into tiles of 512; a tile's tables (64 KB per token) sit in
// shared memory laid out [byte slot][entry][lane], so that every lane only
// ever touches its own bank: the lookups are free of bank conflicts.
//
// Split over the columns ("split-K"): thread block (t, b) owns column tile t
// and a range of rows, builds the tile's tables once per token and streams
// its rows' plane bytes and group parameters through a per-warp ring of
// shared-memory stages.  When every tile is whole (in a multiple of 512) and
// holds at least 4 groups (g <= 128), lane 0 fills a stage with three tensor
// copies (bcq_gemv_tma_kernel); otherwise every lane issues its share of
// 16- or 4-byte asynchronous copies (bcq_gemv_partial_kernel).  Lane l owns columns
// 16 l .. 16 l + 15 of the tile (one 16-bit half of a plane word).  A warp
// takes 8 rows at a time; a reduce-scatter over the warp (uq_common.cuh,
// SegReduce) leaves one row's tile partial on each of 8 lanes, which store it
// to the caller's workspace [tile][token][row].  A second kernel sums the
// partials of a row in tile order.  Deterministic; no atomics.
#include <cuda.h>   // CUtensorMap and its enums (the encoder is reached through the runtime)

#include <atomic>
#include <mutex>

#include "uq_common.cuh"
#include "uq_launch.h"
#include "uq_pipe.cuh"

namespace uq {

constexpr int kGemvThreads = 512;
constexpr int kGemvWarps = kGemvThreads / 32;
constexpr int kTileCols = 512;                  // columns per tile: 32 lanes x 16
constexpr int kTileWords = kTileCols / 32;      // plane words per tile and row
constexpr int kBatchRows = 8;                   // rows a warp takes at a time
constexpr int kMaxStagesGemv = 4;
constexpr int kLutFloats = 2 * 256 * 32;        // [byte slot][entry][lane]
constexpr int kNibFloats = 4 * 16 * 32;         // [nibble slot][entry][lane]
// x of the tile, lane-major with a padded stride of 17 floats per lane's 16
// columns, so that the table build's reads (one lane per 16 columns) fall
// in distinct banks
constexpr int kXsStride = 17;
constexpr int kXsFloats = 32 * kXsStride;
constexpr size_t kGemvFixedSmem = (size_t)(kLutFloats + kNibFloats + kXsFloats) * sizeof(float);
constexpr size_t kGemvSmemLimit = 227 * 1024;   // dynamic shared memory a block may opt in to

// Groups of one row inside one tile: 512 / g, or 1 when a group spans whole tiles.
__host__ __device__ constexpr int gemv_tile_groups(int g) { return g < kTileCols ? kTileCols / g : 1; }
// 32-bit words of one stage: 8 rows x (q planes x 16 words + the tile's alpha* and z*).
__host__ __device__ constexpr int gemv_stage_words(int q, int ng) { return kBatchRows * (q * kTileWords + ng * (q + 1)); }
// Stages per warp: as many (up to kMaxStagesGemv) as fit next to the tables.
__host__ __device__ constexpr int gemv_stages(int q, int ng) {
    return (int)((kGemvSmemLimit - kGemvFixedSmem) / (kGemvWarps * (size_t)gemv_stage_words(q, ng) * 4)) >
                   kMaxStagesGemv
               ? kMaxStagesGemv
               : (int)((kGemvSmemLimit - kGemvFixedSmem) / (kGemvWarps * (size_t)gemv_stage_words(q, ng) * 4));
}

struct XF32 {
    static __device__ __forceinline__ float get(const void* x, int64_t i) { return static_cast<const float*>(x)[i]; }
};
struct XBF16 {
    static __device__ __forceinline__ float get(const void* x, int64_t i) {
        return __uint_as_float(uint32_t(static_cast<const uint16_t*>(x)[i]) << 16);
    }
};

// Asynchronous global -> shared copies (completion per thread, by group).
__device__ __forceinline__ void cp4(void* dst, const void* src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
                 "l"(src)
                 : "memory");
}
__device__ __forceinline__ void cp16(void* dst, const void* src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
                 "l"(src)
                 : "memory");
}
__device__ __forceinline__ void cp_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

static_assert(kGemvThreads == 32 * 16, "the table build maps one thread to each (lane, low nibble)");

// NGT = groups of a row per tile (512 / g for g < 512, else 1).
template <int Q, typename XT, int NGT>
__global__ void __launch_bounds__(kGemvThreads, 1)
bcq_gemv_partial_kernel(const uint32_t* __restrict__ PLANES, const float* __restrict__ ASTAR,
                        const float* __restrict__ ZSTAR, const void* __restrict__ X, float* __restrict__ PART,
                        int64_t out, int n_in, int g, int batch, int n_tiles, int64_t rows_per_block, bool pwide) {
    constexpr int PR = NGT * (Q + 1);                 // parameter words per row and tile
    constexpr int PW = kBatchRows * Q * kTileWords;   // plane words per stage (the parameters follow)
    constexpr int SW = gemv_stage_words(Q, NGT);
    constexpr int NS = gemv_stages(Q, NGT);
    static_assert(NS >= 2, "two stages must fit");
    // 16-byte pieces of one row's alpha* and z* in a tile (pwide layout)
    constexpr int PA = NGT * Q / 4, PP = NGT * (Q + 1) / 4;
    constexpr int LPG = 32 / NGT;                     // lanes per group within a tile (NGT >= 2)
    extern __shared__ __align__(16) float gsm[];
    float* lut = gsm;                                 // [2][256][32]
    float* nib = lut + kLutFloats;                    // [4][16][32]
    float* xs = nib + kNibFloats;                     // [32][17]: lane l's columns at 17 l
    uint32_t* stages = reinterpret_cast<uint32_t*>(xs + kXsFloats);
    // the tile sum (a programmatic dependent) may be scheduled now; it waits for this grid's results
    asm volatile("griddepcontrol.launch_dependents;");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = (int)(blockIdx.x % n_tiles);
    const int64_t r0 = (int64_t)(blockIdx.x / n_tiles) * rows_per_block;
    const int nr = (int)(out - r0 < rows_per_block ? out - r0 : rows_per_block);
    if (nr <= 0) return;
    const int words = n_in / 32, Gr = n_in / g;
    const int c0 = t * kTileCols;
    const int tw = words - t * kTileWords < kTileWords ? words - t * kTileWords : kTileWords;
    const int g0 = c0 / g;                                        // first group of the tile
    const int ng = (Gr - g0) < NGT ? (Gr - g0) : NGT;            // groups present in the tile
    const bool wide = (words & 3) == 0 && tw == kTileWords;       // 16-byte aligned, whole tile
    const int nbat = (nr + kBatchRows - 1) / kBatchRows;
    const int my_nb = warp < nbat ? (nbat - warp + kGemvWarps - 1) / kGemvWarps : 0;
    uint32_t* wst = stages + (size_t)warp * NS * SW;
    const uint32_t* ptile = PLANES + r0 * words + t * kTileWords;   // row r0, plane 0, this tile
    const int64_t pstride = out * words;                               // plane to plane
    const float* atile = ASTAR + (r0 * Gr + g0) * Q;
    const float* ztile = ZSTAR + r0 * Gr + g0;
    const int gl = NGT > 1 ? lane / LPG : 0;                    // this lane's group within the tile
    const bool valid = c0 + 16 * lane < n_in;
    using SR = SegReduce<32>;

    // copies of this warp's k-th row batch into stage k % NS (NS a compile-time constant)
    auto issue = [&](int k) {
        uint32_t* st = wst + (size_t)(k % NS) * SW;
        const int rb = kBatchRows * (warp + kGemvWarps * k);
        const int rows = nr - rb < kBatchRows ? nr - rb : kBatchRows;
        const uint32_t* pb = ptile + (int64_t)rb * words;
        if (wide) {
#pragma unroll
            for (int i = 0; i < Q; ++i) {                           // 8 rows x Q planes x 4 pieces of 16 B
                const int p = lane + 32 * i, rj = p >> 2, pc = p & 3;
                const int rr = rj / Q, j = rj - rr * Q;
                if (rr < rows) cp16(st + rj * kTileWords + 4 * pc, pb + j * pstride + (int64_t)rr * words + 4 * pc);
            }
        } else if (lane < tw) {
#pragma unroll
            for (int rj = 0; rj < kBatchRows * Q; ++rj) {
                const int rr = rj / Q, j = rj - rr * Q;
                if (rr < rows) cp4(st + rj * kTileWords + lane, pb + j * pstride + (int64_t)rr * words + lane);
            }
        }
        const float* ab = atile + (int64_t)rb * Gr * Q;
        const float* zb = ztile + (int64_t)rb * Gr;
        if constexpr (NGT % 4 == 0) {
            if (pwide) {                                            // whole tile, 16-byte aligned rows
#pragma unroll
                for (int i = 0; i < (kBatchRows * PP + 31) / 32; ++i) {
                    const int e = lane + 32 * i;
                    const int rr = e / PP, f = e - rr * PP;
                    if (e < kBatchRows * PP && rr < rows) {
                        const bool isa = f < PA;
                        const float* src = isa ? ab + (int64_t)rr * Gr * Q + 4 * f : zb + (int64_t)rr * Gr + 4 * (f - PA);
                        cp16(st + PW + rr * PR + 4 * f, src);        // z* follows alpha* in the stage row
                    }
                }
                return;
            }
        }
#pragma unroll
        for (int i = 0; i < (kBatchRows * PR + 31) / 32; ++i) {
            const int e = lane + 32 * i;
            const int rr = e / PR, f = e - rr * PR;
            if (e < kBatchRows * PR && rr < rows) {
                if (f < NGT * Q) {
                    if (f < ng * Q) cp4(st + PW + e, ab + (int64_t)rr * Gr * Q + f);
                } else if (f - NGT * Q < ng) {
                    cp4(st + PW + e, zb + (int64_t)rr * Gr + (f - NGT * Q));
                }
            }
        }
    };

    for (int b = 0; b < batch; ++b) {                      // token b is row b of X
        __syncthreads();                                    // the previous token's readers are done
        // the first batches' copies fly while the tables are built
        for (int k = 0; k < NS - 1; ++k) {
            if (k < my_nb) issue(k);
            cp_commit();
        }
        for (int i = threadIdx.x; i < kTileCols; i += kGemvThreads)
            xs[kXsStride * (i >> 4) + (i & 15)] = c0 + i < n_in ? XT::get(X, (int64_t)b * n_in + c0 + i) : 0.f;
        __syncthreads();
        // nibble tables: slot s = 2 k + h covers columns 16 l + 8 k + 4 h + (0..3)
        for (int e = threadIdx.x; e < kNibFloats; e += kGemvThreads) {
            const int l = e & 31, v = (e >> 5) & 15, s = e >> 9;
            const float* xc = xs + kXsStride * l + 4 * s;
            float acc = 0.f;
#pragma unroll
            for (int bit = 0; bit < 4; ++bit)
                if ((v >> bit) & 1) acc = __fadd_rn(acc, xc[bit]);
            nib[e] = acc;
        }
        __syncthreads();
        // byte tables: entry v of slot k = low-nibble sum + high-nibble sum.  Thread
        // (lane l, low nibble n) writes the 16 entries v = 16 m + n of both slots.
        {
            const int l = threadIdx.x & 31, n = threadIdx.x >> 5;        // 512 threads = 32 x 16
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const float lo = nib[((2 * k) * 16 + n) * 32 + l];
                const float* hi = nib + (2 * k + 1) * 16 * 32 + l;
                float* dst = lut + (k * 256 + n) * 32 + l;
#pragma unroll
                for (int m = 0; m < 16; ++m) dst[m * 16 * 32] = __fadd_rn(lo, hi[m * 32]);
            }
        }
        __syncthreads();
        const float S = __fadd_rn(lut[(0 * 256 + 255) * 32 + lane], lut[(1 * 256 + 255) * 32 + lane]);
        const float* lut0 = lut + lane;
        const float* lut1 = lut + 256 * 32 + lane;
        float* prow = PART + ((int64_t)t * batch + b) * out + r0;
        for (int k = 0; k < my_nb; ++k) {
            if (k + NS - 1 < my_nb) issue(k + NS - 1);
            cp_commit();
            // this lane's copies of batch k have landed (NS - 1 newer groups may still fly)
            if (NS == 4) cp_wait<3>();
            else if (NS == 3) cp_wait<2>();
            else cp_wait<1>();
            __syncwarp();                                    // ... and every lane's
            const uint32_t* st = wst + (size_t)(k % NS) * SW;
            const uint16_t* ph = reinterpret_cast<const uint16_t*>(st) + lane;
            const float* pa = reinterpret_cast<const float*>(st + PW) + gl * Q;
            const float* pz = reinterpret_cast<const float*>(st + PW) + NGT * Q + gl;
            const int rb = kBatchRows * (warp + kGemvWarps * k);
            float v[kBatchRows];
#pragma unroll
            for (int rr = 0; rr < kBatchRows; ++rr) {
                float acc = __fmul_rn(pz[rr * PR], S);
#pragma unroll
                for (int j = 0; j < Q; ++j) {
                    const uint32_t h = ph[(rr * Q + j) * (2 * kTileWords)];
                    const float P = __fadd_rn(lut0[(h & 255u) * 32], lut1[(h >> 8) * 32]);
                    acc = fmaf(pa[rr * PR + j], fmaf(2.f, P, -S), acc);
                }
                v[rr] = (valid && rb + rr < nr) ? acc : 0.f;
            }
            const int slot0 = SR::run(v, lane);
            if (SR::writer(lane) && rb + slot0 < nr) prow[rb + slot0] = v[0];
            __syncwarp();                                    // stage k % NS is free for batch k + NS
        }
        cp_wait<0>();
    }
}

// ---------------------------------------------------------------------------
// TMA-staged variant (whole tiles: in a multiple of 512, g in {32, 64, 128})
// ---------------------------------------------------------------------------
//
// The same product, tiling, tables and reduction as bcq_gemv_partial_kernel;
// only the staging differs.  Lane 0 of a warp moves one 8-row batch with three
// tensor copies (cp.async.bulk.tensor) completing on the stage's mbarrier: the
// q bit-planes of the batch's rows in the tile as one box {16 words, 8 rows,
// q planes}, their alpha* as a box {NGT * q, 8 rows} and their z* as a box
// {NGT, 8 rows}.  The stage then holds planes [j][row][16 words], alpha*
// [row][NGT * q] and z* [row][NGT].  Rows past `out` read as zeros and are
// never stored.  Batches of the next token are staged while the current
// token's rows are processed (the stage contents do not depend on the token).
// Every wait on an mbarrier is bounded; one that runs out sets g_gemv_err
// (reported by uq_check_device), and the warp stops computing but still
// takes part in the block's barriers, then waits for its copies in flight.

__device__ unsigned int g_gemv_err = 0;

namespace tmap {
__device__ __forceinline__ void load_3d(uint32_t dst, const CUtensorMap* m, int x, int y, int z, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
        "[%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(z), "r"(bar)
        : "memory");
}
__device__ __forceinline__ void load_2d(uint32_t dst, const CUtensorMap* m, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::
            "r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}
}  // namespace tmap

// Bytes of one TMA stage: planes, alpha*, z* of 8 rows (each a multiple of 128).
__host__ __device__ constexpr int gemv_tma_planes_bytes(int q) { return q * kBatchRows * kTileWords * 4; }
__host__ __device__ constexpr int gemv_tma_alpha_bytes(int q, int ng) { return kBatchRows * ng * q * 4; }
__host__ __device__ constexpr int gemv_tma_stage_bytes(int q, int ng) {
    return gemv_tma_planes_bytes(q) + gemv_tma_alpha_bytes(q, ng) + kBatchRows * ng * 4;
}
static_assert(kGemvFixedSmem % 128 == 0, "TMA stages start on a 128-byte boundary");

template <int Q, typename XT, int NGT>
__global__ void __launch_bounds__(kGemvThreads, 1)
bcq_gemv_tma_kernel(const __grid_constant__ CUtensorMap tm_planes, const __grid_constant__ CUtensorMap tm_alpha,
                    const __grid_constant__ CUtensorMap tm_z, const void* __restrict__ X, float* __restrict__ PART,
                    int64_t out, int n_in, int batch, int n_tiles, int64_t rows_per_block) {
    constexpr int PLB = gemv_tma_planes_bytes(Q), ALB = gemv_tma_alpha_bytes(Q, NGT);
    constexpr int SB = gemv_tma_stage_bytes(Q, NGT);
    constexpr int NS = gemv_stages(Q, NGT);           // the same bytes per stage as the cp.async layout
    static_assert(SB == gemv_stage_words(Q, NGT) * 4 && SB % 128 == 0 && NS >= 2, "stage layout");
    static_assert(NGT >= 4, "alpha* and z* boxes must span at least 16 bytes");
    constexpr int LPG = 32 / NGT;
    extern __shared__ __align__(128) float gsm_tma[];
    float* lut = gsm_tma;                             // [2][256][32]
    float* nib = lut + kLutFloats;                    // [4][16][32]
    float* xs = nib + kNibFloats;                     // [32][17]
    unsigned char* stages = reinterpret_cast<unsigned char*>(xs + kXsFloats);
    unsigned long long* bars = reinterpret_cast<unsigned long long*>(stages + (size_t)kGemvWarps * NS * SB);
    // the tile sum (a programmatic dependent) may be scheduled now; it waits for this grid's results
    asm volatile("griddepcontrol.launch_dependents;");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = (int)(blockIdx.x % n_tiles);
    const int64_t r0 = (int64_t)(blockIdx.x / n_tiles) * rows_per_block;
    const int nr = (int)(out - r0 < rows_per_block ? out - r0 : rows_per_block);
    if (nr <= 0) return;                              // the whole block: before any barrier
    const int c0 = t * kTileCols;
    const int nbat = (nr + kBatchRows - 1) / kBatchRows;
    const int my_nb = warp < nbat ? (nbat - warp + kGemvWarps - 1) / kGemvWarps : 0;
    unsigned char* wst = stages + (size_t)warp * NS * SB;
    unsigned long long* wbar = bars + warp * NS;
    const int gl = lane / LPG;
    using SR = SegReduce<32>;

    if (lane == 0) {
        for (int s = 0; s < NS; ++s) tma::bar_init(tma::smem_addr(wbar + s), 1);
        tma::bar_init_fence();
    }
    __syncwarp();

    // items: token-major, this warp's batches k = 0 .. my_nb - 1 per token
    const long long total = (long long)batch * my_nb;
    long long issued = 0, waited = 0;
    int ik = 0;                                       // batch of the next item to issue
    auto issue_next = [&]() {                         // lane 0 only
        const int s = (int)(issued % NS);
        const uint32_t bar = tma::smem_addr(wbar + s);
        const uint32_t d = tma::smem_addr(wst + (size_t)s * SB);
        const int y = (int)(r0 + (int64_t)kBatchRows * (warp + kGemvWarps * ik));
        tma::fence_async_smem();                     // the warp's reads of this stage come first
        tma::bar_arrive_tx(bar, (uint32_t)SB);
        tmap::load_3d(d, &tm_planes, t * kTileWords, y, 0, bar);
        tmap::load_2d(d + PLB, &tm_alpha, t * NGT * Q, y, bar);
        tmap::load_2d(d + PLB + ALB, &tm_z, t * NGT, y, bar);
        ++issued;
        if (++ik == my_nb) ik = 0;
    };
    if (lane == 0)
        while (issued < total && issued < NS) issue_next();

    bool alive = true;
    for (int b = 0; b < batch; ++b) {                      // token b is row b of X
        __syncthreads();                                    // the previous token's readers are done
        for (int i = threadIdx.x; i < kTileCols; i += kGemvThreads)
            xs[kXsStride * (i >> 4) + (i & 15)] = XT::get(X, (int64_t)b * n_in + c0 + i);
        __syncthreads();
        for (int e = threadIdx.x; e < kNibFloats; e += kGemvThreads) {
            const int l = e & 31, v = (e >> 5) & 15, s = e >> 9;
            const float* xc = xs + kXsStride * l + 4 * s;
            float acc = 0.f;
#pragma unroll
            for (int bit = 0; bit < 4; ++bit)
                if ((v >> bit) & 1) acc = __fadd_rn(acc, xc[bit]);
            nib[e] = acc;
        }
        __syncthreads();
        {
            const int l = threadIdx.x & 31, n = threadIdx.x >> 5;
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                const float lo = nib[((2 * k) * 16 + n) * 32 + l];
                const float* hi = nib + (2 * k + 1) * 16 * 32 + l;
                float* dst = lut + (k * 256 + n) * 32 + l;
#pragma unroll
                for (int m = 0; m < 16; ++m) dst[m * 16 * 32] = __fadd_rn(lo, hi[m * 32]);
            }
        }
        __syncthreads();
        const float S = __fadd_rn(lut[(0 * 256 + 255) * 32 + lane], lut[(1 * 256 + 255) * 32 + lane]);
        const float* lut0 = lut + lane;
        const float* lut1 = lut + 256 * 32 + lane;
        float* prow = PART + ((int64_t)t * batch + b) * out + r0;
        for (int k = 0; k < my_nb; ++k) {
            const long long i = (long long)b * my_nb + k;
            const int s = (int)(i % NS);
            if (alive) {
                // one verdict for the whole warp (lanes poll the mbarrier separately)
                if (__all_sync(kFull, tma::bar_wait(tma::smem_addr(wbar + s), (uint32_t)((i / NS) & 1)))) {
                    ++waited;
                } else {
                    alive = false;
                    if (lane == 0) atomicOr(&g_gemv_err, 1u);
                }
            }
            if (alive) {
                const unsigned char* st = wst + (size_t)s * SB;
                const uint16_t* ph = reinterpret_cast<const uint16_t*>(st) + lane;
                const float* pa = reinterpret_cast<const float*>(st + PLB) + gl * Q;
                const float* pz = reinterpret_cast<const float*>(st + PLB + ALB) + gl;
                const int rb = kBatchRows * (warp + kGemvWarps * k);
                float v[kBatchRows];
#pragma unroll
                for (int rr = 0; rr < kBatchRows; ++rr) {
                    float acc = __fmul_rn(pz[rr * NGT], S);
#pragma unroll
                    for (int j = 0; j < Q; ++j) {
                        const uint32_t h = ph[(j * kBatchRows + rr) * (2 * kTileWords)];
                        const float P = __fadd_rn(lut0[(h & 255u) * 32], lut1[(h >> 8) * 32]);
                        acc = fmaf(pa[rr * NGT * Q + j], fmaf(2.f, P, -S), acc);
                    }
                    v[rr] = rb + rr < nr ? acc : 0.f;
                }
                const int slot0 = SR::run(v, lane);
                if (SR::writer(lane) && rb + slot0 < nr) prow[rb + slot0] = v[0];
            }
            __syncwarp();                                    // stage s is free for item i + NS
            if (alive && lane == 0 && issued < total) issue_next();
        }
    }
    if (!alive && lane == 0) {
        // copies issued but never waited for land before the block exits
        for (long long i = waited; i < issued; ++i)
            if (!tma::bar_wait(tma::smem_addr(wbar + (int)(i % NS)), (uint32_t)((i / NS) & 1))) {
                atomicOr(&g_gemv_err, kDrainTimeoutBit);   // copies may still be in flight
                break;
            }
    }
}

// ---------------------------------------------------------------------------
// Wide-lane variant (in a multiple of 1024, g in {32, 64, 128, 256})
// ---------------------------------------------------------------------------
//
// Tiles of 1024 columns; lane l owns columns 32 l .. 32 l + 31 of the tile,
// i.e. one whole plane word per (row, plane).  Its four bytes index four
// lookup tables (one per 8 columns), so a plane word costs one shared load,
// four table lookups and three adds, and the per-row work (parameters, the
// reduction over the warp) is spread over 32 q weights per lane instead of 16 q.
//
// The tables of a tile take 128 KB: [pair p][entry v][slot s][lane l] floats,
// byte slot k = 2 p + s, so that entry v sits at byte offset 256 v and lane l
// at 4 l.  The table is placed at a shared-memory address L that is a
// multiple of 65536: the byte address of entry v for lane l is then
// L + 256 v + 4 l + (65536 p + 128 s), and one byte permutation (PRMT) of
// the plane word with the per-lane constant L + 4 l puts the word's byte k
// into bits 8..15 of that address; the constant part is the load's
// immediate offset.  The rest of shared memory -- x of the tile (lane-major,
// stride 33 floats: conflict-free table build), the mbarriers and the
// stages -- fills the space below L first, then the space after the tables;
// the host requests enough bytes for any position of the dynamic base.
//
// Each warp runs its own ring of NS stages; lane 0 fills a stage with three
// tensor copies (planes {32 words, 8 rows, q}, alpha* {NGT q, 8 rows}, z*
// {NGT, 8 rows}) completing on the stage's mbarrier.  Rows past `out` read
// as zeros and give zero partials that are never stored, so no row needs a
// validity test.  Waits are bounded as in bcq_gemv_tma_kernel.

constexpr int kWideCols = 1024;                   // columns per tile: 32 lanes x 32
constexpr int kWideWords = kWideCols / 32;        // plane words per tile and row
constexpr uint32_t kWideLutBytes = 4u * 256u * 32u * 4u;
constexpr int kWideXsStride = 33;
constexpr int kWideXsBytes = 32 * kWideXsStride * 4;
constexpr int kWideMaxWarps = 16;
constexpr int kWideStages = 2;
constexpr int kWideHeadBytes = align_up(kWideXsBytes + kWideMaxWarps * kWideStages * 8, 128);   // x + mbarriers
constexpr int kSmemOptIn = 227 * 1024;
// A table build costs about as much as 64 rows.  Row blocks run over all the
// tiles side by side (block b takes tile b mod n_tiles), so the blocks in flight
// stream the same rows and DRAM pages: an equal split of (tile, row) pairs
// over every SM, tile-major, measured slower (33.1 vs 29.7 us on 8192 x 28672).
constexpr int kWideLutRows = 64;

// Groups of one row inside one wide tile.
__host__ __device__ constexpr int wide_tile_groups(int g) { return kWideCols / g; }
// Bytes of one stage: 8 rows x (q planes x 32 words + the tile's alpha* and z*).
__host__ __device__ constexpr int wide_stage_bytes(int q, int ngt) {
    return kBatchRows * (q * kWideWords + ngt * (q + 1)) * 4;
}
// Slack for the part of the space below the tables that cannot be used (at
// most one stage, or the head when the gap is smaller than the head).
__host__ __device__ constexpr int wide_slack(int q, int ngt) {
    return (wide_stage_bytes(q, ngt) > kWideHeadBytes ? wide_stage_bytes(q, ngt) : kWideHeadBytes) + 128;
}
// Warps per block: as many as fit two stages each next to the tables (at most 16).
__host__ __device__ constexpr int wide_warps(int q, int ngt) {
    return (int)((kSmemOptIn - (int)kWideLutBytes - kWideHeadBytes - wide_slack(q, ngt)) /
                 (kWideStages * wide_stage_bytes(q, ngt))) > kWideMaxWarps
               ? kWideMaxWarps
               : (int)((kSmemOptIn - (int)kWideLutBytes - kWideHeadBytes - wide_slack(q, ngt)) /
                       (kWideStages * wide_stage_bytes(q, ngt)));
}
// Dynamic shared memory to request.  The tables start at the first multiple
// of 65536 at or above the dynamic base D, so they end by D + 192 KB at the
// latest; when the head and the stages do not fit in the space below them,
// the rest follows the tables with at most wide_slack of that space unused.
__host__ __device__ constexpr int wide_smem_bytes(int q, int ngt) {
    return (int)kWideLutBytes + kWideHeadBytes + wide_slack(q, ngt) +
                       wide_warps(q, ngt) * kWideStages * wide_stage_bytes(q, ngt) >
                   (int)kWideLutBytes + 65536
               ? (int)kWideLutBytes + kWideHeadBytes + wide_slack(q, ngt) +
                     wide_warps(q, ngt) * kWideStages * wide_stage_bytes(q, ngt)
               : (int)kWideLutBytes + 65536;
}

// Index of the lowest set bit of n (1 <= n <= 15).
__host__ __device__ constexpr int low_bit(int n) { return (n & 1) ? 0 : (n & 2) ? 1 : (n & 4) ? 2 : 3; }

__device__ __forceinline__ uint32_t lds_u32(uint32_t a) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ float lds_f32(uint32_t a) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1];" : "=f"(v) : "r"(a));
    return v;
}

template <int Q, typename XT, int NGT>
__global__ void __launch_bounds__(kWideMaxWarps * 32, 1)
bcq_gemv_wide_kernel(const __grid_constant__ CUtensorMap tm_planes, const __grid_constant__ CUtensorMap tm_alpha,
                     const __grid_constant__ CUtensorMap tm_z, const void* __restrict__ X, float* __restrict__ PART,
                     int64_t out, int n_in, int batch, int n_tiles, int64_t rows_per_block) {
    constexpr int NW = wide_warps(Q, NGT);
    constexpr int NS = kWideStages;
    constexpr int SB = wide_stage_bytes(Q, NGT);
    constexpr int PLB = Q * kBatchRows * kWideWords * 4;       // planes of a stage
    constexpr int ALB = kBatchRows * NGT * Q * 4;              // alpha* of a stage
    constexpr int DYN = wide_smem_bytes(Q, NGT);
    constexpr int LPG = 32 / NGT;                              // lanes per group
    // every tensor-copy destination (stage, alpha*, z*) on a 128-byte boundary
    static_assert(NW >= 4 && SB % 128 == 0 && PLB % 128 == 0 && ALB % 128 == 0 && DYN <= kSmemOptIn,
                  "wide layout");
    static_assert(NGT >= 4 && (NGT * Q * 4) % 16 == 0, "alpha* and z* boxes must span a multiple of 16 bytes");
    extern __shared__ __align__(128) unsigned char wsm[];
    // the tile sum (a programmatic dependent) may be scheduled now; it waits for this grid's results
    asm volatile("griddepcontrol.launch_dependents;");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = (int)(blockIdx.x % n_tiles);
    const int64_t r0 = (int64_t)(blockIdx.x / n_tiles) * rows_per_block;
    const int nr = (int)(out - r0 < rows_per_block ? out - r0 : rows_per_block);
    if (nr <= 0) return;                                       // the whole block: before any barrier

    // shared-memory layout (uniform over the block)
    const uint32_t D = tma::smem_addr(wsm);
    const uint32_t L = (D + 0xFFFFu) & ~0xFFFFu;
    uint32_t lo = (D + 127u) & ~127u, hi = L + kWideLutBytes;
    uint32_t head;
    if (L >= lo + (uint32_t)kWideHeadBytes) { head = lo; lo += kWideHeadBytes; }
    else { head = hi; hi += kWideHeadBytes; }
    const uint32_t n_gap = L > lo ? (L - lo) / SB : 0u;
    if (hi + ((uint32_t)(NW * NS) > n_gap ? (uint32_t)(NW * NS) - n_gap : 0u) * SB > D + DYN) {
        if (threadIdx.x == 0) atomicOr(&g_gemv_err, 4u);       // cannot happen: the host sized DYN for any D
        return;
    }
    float* xs = reinterpret_cast<float*>(wsm + (head - D));
    float* lut = reinterpret_cast<float*>(wsm + (L - D));
    const uint32_t bar0 = head + (uint32_t)kWideXsBytes + (uint32_t)(warp * NS * 8);
    static_assert(NS == 2, "two stages per warp, held in two registers");
    const uint32_t i0 = (uint32_t)(warp * NS), i1 = i0 + 1u;
    const uint32_t st0 = i0 < n_gap ? lo + i0 * SB : hi + (i0 - n_gap) * SB;
    const uint32_t st1 = i1 < n_gap ? lo + i1 * SB : hi + (i1 - n_gap) * SB;

    const int c0 = t * kWideCols;
    const int nbat = (nr + kBatchRows - 1) / kBatchRows;
    const int my_nb = warp < nbat ? (nbat - warp + NW - 1) / NW : 0;
    const uint32_t lane_base = L + 4u * (uint32_t)lane;        // bits 8..15 are zero
    const int gl = lane / LPG;                                 // this lane's group within the tile
    using SR = SegReduce<32>;

    if (lane == 0) {
#pragma unroll
        for (int s = 0; s < NS; ++s) tma::bar_init(bar0 + 8u * s, 1);
        tma::bar_init_fence();
    }
    __syncwarp();
    // Launched as a programmatic dependent of the previous kernel on the stream
    // (the previous call's tile sum, which reads the partials this grid
    // overwrites, or whatever produced the inputs): nothing global is read or
    // written before that grid has completed.  Only the launch and the set-up
    // above overlap it.
    asm volatile("griddepcontrol.wait;" ::: "memory");

    const int total = batch * my_nb;                           // items: token-major, this warp's batches
    int issued = 0, waited = 0, ik = 0;
    auto issue_next = [&]() {                                  // lane 0 only
        const int s = issued & 1;
        const uint32_t bar = bar0 + 8u * s;
        const uint32_t d = s ? st1 : st0;
        const int y = (int)(r0 + (int64_t)kBatchRows * (warp + NW * ik));
        tma::fence_async_smem();                               // the warp's reads of this stage come first
        tma::bar_arrive_tx(bar, (uint32_t)SB);
        tmap::load_3d(d, &tm_planes, t * kWideWords, y, 0, bar);
        tmap::load_2d(d + PLB, &tm_alpha, t * NGT * Q, y, bar);
        tmap::load_2d(d + PLB + ALB, &tm_z, t * NGT, y, bar);
        ++issued;
        if (++ik == my_nb) ik = 0;
    };
    if (lane == 0)
        while (issued < total && issued < NS) issue_next();

    bool alive = true;
    for (int b = 0; b < batch; ++b) {                          // token b is row b of X
        __syncthreads();                                       // the previous token's readers are done
        for (int i = threadIdx.x; i < kWideCols; i += NW * 32)
            xs[kWideXsStride * (i >> 5) + (i & 31)] = XT::get(X, (int64_t)b * n_in + c0 + i);
        __syncthreads();
        // tables: item (lane l, slot k, high nibble m) writes entries 16 m + n, n = 0..15
        for (int it = threadIdx.x; it < 2048; it += NW * 32) {
            const int l = it & 31, k = (it >> 5) & 3, m = it >> 7;
            const float* xc = xs + kWideXsStride * l + 8 * k;
            float x[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) x[i] = xc[i];
            float lo4[16];
            lo4[0] = 0.f;
#pragma unroll
            for (int n = 1; n < 16; ++n) lo4[n] = __fadd_rn(lo4[n & (n - 1)], x[low_bit(n)]);
            float h = (m & 1) ? x[4] : 0.f;
            h = (m & 2) ? __fadd_rn(h, x[5]) : h;
            h = (m & 4) ? __fadd_rn(h, x[6]) : h;
            h = (m & 8) ? __fadd_rn(h, x[7]) : h;
            float* dst = lut + (k >> 1) * 16384 + (k & 1) * 32 + l + 16 * m * 64;
#pragma unroll
            for (int n = 0; n < 16; ++n) dst[n * 64] = __fadd_rn(lo4[n], h);
        }
        __syncthreads();
        // S = the sum of this lane's 32 x values (entry 255 of each slot)
        const float S = __fadd_rn(__fadd_rn(lds_f32(lane_base + 255u * 256u), lds_f32(lane_base + 255u * 256u + 128u)),
                                  __fadd_rn(lds_f32(lane_base + 65536u + 255u * 256u),
                                            lds_f32(lane_base + 65536u + 255u * 256u + 128u)));
        float* prow = PART + ((int64_t)t * batch + b) * out + r0;
        for (int k = 0; k < my_nb; ++k) {
            const int i = b * my_nb + k;
            const int s = i & 1;
            const uint32_t sa = s ? st1 : st0;
            if (alive) {
                // one verdict for the whole warp (lanes poll the mbarrier separately)
                if (__all_sync(kFull, tma::bar_wait(bar0 + 8u * s, (uint32_t)((i >> 1) & 1)))) {
                    ++waited;
                } else {
                    alive = false;
                    if (lane == 0) atomicOr(&g_gemv_err, 1u);
                }
            }
            if (alive) {
                const uint32_t pw = sa + 4u * (uint32_t)lane;                          // this lane's plane words
                const uint32_t pa = sa + PLB + 4u * (uint32_t)(gl * Q);               // its group's alpha*
                const uint32_t pz = sa + PLB + ALB + 4u * (uint32_t)gl;               // and z*
                float v[kBatchRows];
#pragma unroll
                for (int rr = 0; rr < kBatchRows; ++rr) {
                    float acc = __fmul_rn(lds_f32(pz + 4u * (uint32_t)(rr * NGT)), S);
#pragma unroll
                    for (int j = 0; j < Q; ++j) {
                        const uint32_t w = lds_u32(pw + 4u * (uint32_t)((j * kBatchRows + rr) * kWideWords));
                        const float t0 = lds_f32(__byte_perm(w, lane_base, 0x7604));
                        const float t1 = lds_f32(__byte_perm(w, lane_base, 0x7614) + 128u);
                        const float t2 = lds_f32(__byte_perm(w, lane_base, 0x7624) + 65536u);
                        const float t3 = lds_f32(__byte_perm(w, lane_base, 0x7634) + 65536u + 128u);
                        const float P = __fadd_rn(__fadd_rn(t0, t1), __fadd_rn(t2, t3));
                        acc = fmaf(lds_f32(pa + 4u * (uint32_t)(rr * NGT * Q + j)), fmaf(2.f, P, -S), acc);
                    }
                    v[rr] = acc;
                }
                const int rb = kBatchRows * (warp + NW * k);
                const int slot0 = SR::run(v, lane);
                if (SR::writer(lane) && rb + slot0 < nr) prow[rb + slot0] = v[0];
            }
            __syncwarp();                                      // stage s is free for item i + NS
            if (alive && lane == 0 && issued < total) issue_next();
        }
    }
    if (!alive && lane == 0) {
        // copies issued but never waited for land before the block exits
        for (int i = waited; i < issued; ++i)
            if (!tma::bar_wait(bar0 + 8u * (i & 1), (uint32_t)((i >> 1) & 1))) {
                atomicOr(&g_gemv_err, kDrainTimeoutBit);       // copies may still be in flight
                break;
            }
    }
}

// y[b, r] = sum over tiles of PART[t, b, r], in tile order.
__global__ void __launch_bounds__(256)
bcq_gemv_reduce_kernel(const float* __restrict__ PART, float* __restrict__ Y, int64_t n, int n_tiles) {
    // Launched as a programmatic dependent of the product kernel: it may start
    // while that kernel still runs, and waits here until the product grid has
    // completed and its partials are visible.  The next product kernel on the
    // stream may be scheduled once every block of this grid has started.
    asm volatile("griddepcontrol.launch_dependents;");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        float acc = 0.f;
        for (int t = 0; t < n_tiles; ++t) acc += __ldg(PART + (int64_t)t * n + i);
        Y[i] = acc;
    }
}

int64_t gemv_workspace_floats(int64_t out, int64_t n_in, int batch) {
    return ((n_in + kTileCols - 1) / kTileCols) * (int64_t)batch * out;
}

// Built-in scratch for uq_bcq_gemv_noalloc: the per-tile partials of one call,
// for callers that cannot allocate device memory themselves.  4 MiB, held by
// every GPU that loads the library until the process exits; shared by all
// calls (a call overwrites every word it later reads, so nothing has to be
// cleared between calls, but two calls in flight at once race on it).
constexpr int64_t kStaticWorkFloats = int64_t(1) << 20;
static __device__ __align__(256) float g_gemv_static_work[kStaticWorkFloats];

int64_t gemv_static_workspace_floats() { return kStaticWorkFloats; }

// Identifier of the calling thread's current CUDA context (unique for the
// life of the process, so a context created anew after cudaDeviceReset gets
// a new one), through the runtime's driver entry points.  False if no
// context is current yet or the driver lacks the calls.
static bool current_context_id(unsigned long long* id) {
    using GetCurrent = CUresult (*)(CUcontext*);
    using GetId = CUresult (*)(CUcontext, unsigned long long*);
    static std::atomic<void*> get_current{nullptr}, get_id{nullptr};
    void* fc = get_current.load(std::memory_order_acquire);
    void* fi = get_id.load(std::memory_order_acquire);
    if (fc == nullptr || fi == nullptr) {
        cudaDriverEntryPointQueryResult qr = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fc, 12000, cudaEnableDefault, &qr) != cudaSuccess ||
            qr != cudaDriverEntryPointSuccess || fc == nullptr)
            return false;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &fi, 12000, cudaEnableDefault, &qr) != cudaSuccess ||
            qr != cudaDriverEntryPointSuccess || fi == nullptr)
            return false;
        get_current.store(fc, std::memory_order_release);
        get_id.store(fi, std::memory_order_release);
    }
    CUcontext ctx = nullptr;
    if (reinterpret_cast<GetCurrent>(fc)(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
    return reinterpret_cast<GetId>(fi)(ctx, id) == CUDA_SUCCESS;
}

// Device address of g_gemv_static_work in the current device's context.  The
// name is only a host-side stand-in in host code, so the address is looked up
// with that device current (cudaGetSymbolAddress) and cached per device
// together with the context's identifier; a new context on the device (after
// cudaDeviceReset) is looked up again.
cudaError_t gemv_static_workspace(float** work) {
    struct Entry {
        unsigned long long ctx;
        float* ptr;
    };
    static Entry cache[kMaxDevices] = {};
    static std::mutex lock;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const bool cacheable = dev >= 0 && dev < kMaxDevices;
    unsigned long long id = 0;
    bool have_id = current_context_id(&id);
    if (cacheable && have_id) {
        std::lock_guard<std::mutex> g(lock);
        if (cache[dev].ptr != nullptr && cache[dev].ctx == id) {
            *work = cache[dev].ptr;
            return cudaSuccess;
        }
    }
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_gemv_static_work);   // makes the device's context current if it was not
    if (e != cudaSuccess) return e;
    if (!have_id) have_id = current_context_id(&id);
    if (cacheable && have_id) {
        std::lock_guard<std::mutex> g(lock);
        cache[dev] = Entry{id, static_cast<float*>(p)};
    }
    *work = static_cast<float*>(p);
    return cudaSuccess;
}

cudaError_t gemv_error(bool clear, unsigned int* flag) {
    unsigned int v = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, g_gemv_err, sizeof(v));
    if (e != cudaSuccess) return e;
    *flag = v;
    if (clear && v) {
        const unsigned int z = 0;
        e = cudaMemcpyToSymbol(g_gemv_err, &z, sizeof(z));
    }
    return e;
}

using TensorMapEncode = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                     const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                     CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

// The driver's tensor-map encoder, looked up once through the runtime (the
// library does not link against the driver library).  Null if unavailable.
static TensorMapEncode tensor_map_encoder() {
    static std::atomic<TensorMapEncode> cached{nullptr};
    static std::atomic<int> unavailable{0};
    TensorMapEncode f = cached.load(std::memory_order_acquire);
    if (f != nullptr || unavailable.load(std::memory_order_acquire)) return f;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult qr = cudaDriverEntryPointSymbolNotFound;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &qr) != cudaSuccess ||
        qr != cudaDriverEntryPointSuccess || p == nullptr) {
        unavailable.store(1, std::memory_order_release);
        return nullptr;
    }
    f = reinterpret_cast<TensorMapEncode>(p);
    cached.store(f, std::memory_order_release);
    return f;
}

// Tensor maps of the bit-planes [q][out][in/32] (u32), alpha* [out][Gr q] and
// z* [out][Gr] (fp32), Gr = in / g, with the boxes of one 8-row batch of one
// tile of `tile_cols` columns (512 or 1024).  Called only for in a multiple of
// tile_cols and at least 4 groups per tile, so every stride is a multiple of
// 16 bytes and every box starts on a 16-byte boundary.
// False if the encoder is unavailable or refuses a map.
static bool gemv_tensor_maps(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in,
                             int q, int g, int tile_cols, CUtensorMap* mp, CUtensorMap* ma, CUtensorMap* mz) {
    const TensorMapEncode enc = tensor_map_encoder();
    if (enc == nullptr) return false;
    const cuuint64_t words = (cuuint64_t)n_in / 32, gr = (cuuint64_t)(n_in / g), rows = (cuuint64_t)out;
    const cuuint32_t ngt = (cuuint32_t)(tile_cols / g), one[3] = {1, 1, 1};
    const cuuint64_t pdim[3] = {words, rows, (cuuint64_t)q};
    const cuuint64_t pstride[2] = {words * 4, words * 4 * rows};
    const cuuint32_t pbox[3] = {(cuuint32_t)(tile_cols / 32), (cuuint32_t)kBatchRows, (cuuint32_t)q};
    if (enc(mp, CU_TENSOR_MAP_DATA_TYPE_UINT32, 3, const_cast<uint32_t*>(planes), pdim, pstride, pbox, one,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return false;
    const cuuint64_t adim[2] = {gr * (cuuint64_t)q, rows};
    const cuuint64_t astride[1] = {gr * (cuuint64_t)q * 4};
    const cuuint32_t abox[2] = {ngt * (cuuint32_t)q, (cuuint32_t)kBatchRows};
    if (enc(ma, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(astar), adim, astride, abox, one,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
        return false;
    const cuuint64_t zdim[2] = {gr, rows};
    const cuuint64_t zstride[1] = {gr * 4};
    const cuuint32_t zbox[2] = {ngt, (cuuint32_t)kBatchRows};
    return enc(mz, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(zstar), zdim, zstride, zbox, one,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Opts a kernel into `smem` bytes of dynamic shared memory and returns its
// resident blocks per SM, once per device (Tag: one cache per kernel).
template <typename Tag, typename KERN>
static cudaError_t gemv_blocks_per_sm(KERN kern, size_t smem, int& per_sm, int threads = kGemvThreads) {
    static std::atomic<int> cache[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    per_sm = (dev >= 0 && dev < 64) ? cache[dev].load(std::memory_order_relaxed) : 0;
    if (per_sm != 0) return cudaSuccess;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, threads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
    if (dev >= 0 && dev < 64) cache[dev].store(per_sm, std::memory_order_relaxed);
    return cudaSuccess;
}

// Row blocks (of whole 8-row batches): the count that minimises
// waves x (one table build, worth about 32 rows, + rows per block), where
// a wave is one block per resident slot.
static void gemv_row_blocks(int64_t out, int n_tiles, int per_sm, int64_t& n_rb, int64_t& rpb,
                            double table_rows = 32.0) {
    const int64_t slots = (int64_t)sm_count() * per_sm;
    const int64_t max_rb = (out + kBatchRows - 1) / kBatchRows;
    n_rb = 1;
    rpb = max_rb * kBatchRows;
    double best = -1.0;
    const int64_t lim = max_rb < 8 * slots ? max_rb : 8 * slots;
    for (int64_t cand = 1; cand <= lim; ++cand) {
        int64_t r = (out + cand - 1) / cand;
        r = (r + kBatchRows - 1) / kBatchRows * kBatchRows;
        const int64_t nb = (out + r - 1) / r;
        const int64_t waves = (nb * n_tiles + slots - 1) / slots;
        const double cost = (double)waves * (table_rows + (double)r);
        if (best < 0.0 || cost < best) { best = cost; n_rb = nb; rpb = r; }
    }
}

// y = the per-tile partials summed in tile order.
// The tile sum is launched with programmatic stream serialization, so its
// launch overlaps the end of the product kernel (it waits for that grid's
// results with griddepcontrol.wait before reading them).
static cudaError_t gemv_reduce(const float* work, float* y, int64_t n, int n_tiles, cudaStream_t st) {
    int64_t blocks = (n + 255) / 256;
    const int64_t cap = (int64_t)sm_count() * 8;
    if (blocks > cap) blocks = cap;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, bcq_gemv_reduce_kernel, work, y, n, n_tiles);
}

template <int Q, typename XT, int NGT>
struct GemvCopyTag {};
template <int Q, typename XT, int NGT>
struct GemvTmaTag {};

template <int Q, typename XT, int NGT>
static cudaError_t run_gemv(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in,
                            int g, const void* x, int batch, float* y, float* work, cudaStream_t st) {
    constexpr size_t stage_bytes = (size_t)gemv_stage_words(Q, NGT) * 4;
    constexpr int NS = gemv_stages(Q, NGT);
    constexpr size_t smem = kGemvFixedSmem + kGemvWarps * (size_t)NS * stage_bytes;
    constexpr size_t smem_tma = smem + kGemvWarps * (size_t)NS * sizeof(unsigned long long);   // + mbarriers
    static_assert(NS >= 2 && smem_tma <= kGemvSmemLimit, "two stages must fit");
    // Whole tiles and at least 4 groups per tile: staged by tensor copies.
    // Otherwise by per-lane asynchronous copies; alpha* and z* rows of a tile
    // move in 16-byte pieces when every tile is whole (in a multiple of 512)
    // and holds a multiple of 4 groups (both arrays start on 16-byte
    // boundaries: the entry point checks that), else in 4-byte pieces.
    const bool whole = n_in % kTileCols == 0;
    const bool pwide = NGT % 4 == 0 && whole;
    const int n_tiles = (n_in + kTileCols - 1) / kTileCols;
    if constexpr (NGT >= 4) {
        const unsigned long long plane_bytes = (unsigned long long)(n_in / 32) * 4ull * (unsigned long long)out;
        CUtensorMap mp, ma, mz;
        if (whole && plane_bytes < (1ull << 40) && gemv_tensor_maps(planes, astar, zstar, out, n_in, Q, g, kTileCols, &mp, &ma, &mz)) {
            auto kern = bcq_gemv_tma_kernel<Q, XT, NGT>;
            int per_sm = 0;
            cudaError_t e = gemv_blocks_per_sm<GemvTmaTag<Q, XT, NGT>>(kern, smem_tma, per_sm);
            if (e != cudaSuccess) return e;
            int64_t n_rb = 0, rpb = 0;
            gemv_row_blocks(out, n_tiles, per_sm, n_rb, rpb);
            kern<<<(unsigned)(n_rb * n_tiles), kGemvThreads, smem_tma, st>>>(mp, ma, mz, x, work, out, n_in, batch,
                                                                           n_tiles, rpb);
            e = cudaGetLastError();
            if (e != cudaSuccess) return e;
            return gemv_reduce(work, y, (int64_t)batch * out, n_tiles, st);
        }
    }
    auto kern = bcq_gemv_partial_kernel<Q, XT, NGT>;
    int per_sm = 0;
    cudaError_t e = gemv_blocks_per_sm<GemvCopyTag<Q, XT, NGT>>(kern, smem, per_sm);
    if (e != cudaSuccess) return e;
    int64_t n_rb = 0, rpb = 0;
    gemv_row_blocks(out, n_tiles, per_sm, n_rb, rpb);
    kern<<<(unsigned)(n_rb * n_tiles), kGemvThreads, smem, st>>>(planes, astar, zstar, x, work, out, n_in, g, batch,
                                                                 n_tiles, rpb, pwide);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    return gemv_reduce(work, y, (int64_t)batch * out, n_tiles, st);
}

template <int Q, typename XT, int NGT>
struct GemvWideTag {};

// The wide-lane product (in a multiple of 1024, NGT = 1024 / g groups per
// tile).  Returns cudaErrorNotSupported, having launched nothing, when the
// shape or the driver does not allow it; the caller then takes the 512-column
// kernels.
template <int Q, typename XT, int NGT>
static cudaError_t run_gemv_wide(const uint32_t* planes, const float* astar, const float* zstar, int64_t out,
                                 int n_in, int g, const void* x, int batch, float* y, float* work, cudaStream_t st) {
    if constexpr (wide_warps(Q, NGT) >= 4) {
        constexpr int NW = wide_warps(Q, NGT);
        constexpr int DYN = wide_smem_bytes(Q, NGT);
        const unsigned long long plane_bytes = (unsigned long long)(n_in / 32) * 4ull * (unsigned long long)out;
        if (n_in % kWideCols != 0 || plane_bytes >= (1ull << 40)) return cudaErrorNotSupported;
        CUtensorMap mp, ma, mz;
        if (!gemv_tensor_maps(planes, astar, zstar, out, n_in, Q, g, kWideCols, &mp, &ma, &mz))
            return cudaErrorNotSupported;
        auto kern = bcq_gemv_wide_kernel<Q, XT, NGT>;
        int per_sm = 0;
        cudaError_t e = gemv_blocks_per_sm<GemvWideTag<Q, XT, NGT>>(kern, DYN, per_sm, NW * 32);
        if (e != cudaSuccess) return e;
        const int n_tiles = n_in / kWideCols;
        int64_t n_rb = 0, rpb = 0;
        gemv_row_blocks(out, n_tiles, per_sm, n_rb, rpb, (double)kWideLutRows);
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        cfg.gridDim = dim3((unsigned)(n_rb * n_tiles));
        cfg.blockDim = dim3(NW * 32);
        cfg.dynamicSmemBytes = DYN;
        cfg.stream = st;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, kern, mp, ma, mz, x, work, out, n_in, batch, n_tiles, rpb);
        if (e != cudaSuccess) return e;
        return gemv_reduce(work, y, (int64_t)batch * out, n_tiles, st);
    } else {
        return cudaErrorNotSupported;
    }
}

template <int Q, typename XT>
static cudaError_t gemv_g(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in, int g,
                          const void* x, int batch, float* y, float* work, cudaStream_t st) {
    if (n_in % kWideCols == 0 && g <= 256) {
        cudaError_t e = cudaErrorNotSupported;
        switch (wide_tile_groups(g)) {
            case 32: e = run_gemv_wide<Q, XT, 32>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st); break;
            case 16: e = run_gemv_wide<Q, XT, 16>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st); break;
            case 8: e = run_gemv_wide<Q, XT, 8>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st); break;
            default: e = run_gemv_wide<Q, XT, 4>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st); break;
        }
        if (e != cudaErrorNotSupported) return e;
    }
    switch (gemv_tile_groups(g)) {
        case 16: return run_gemv<Q, XT, 16>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st);
        case 8: return run_gemv<Q, XT, 8>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st);
        case 4: return run_gemv<Q, XT, 4>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st);
        case 2: return run_gemv<Q, XT, 2>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st);
        default: return run_gemv<Q, XT, 1>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st);
    }
}

template <int Q>
static cudaError_t gemv_x(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in, int g,
                          const void* x, int xdtype, int batch, float* y, float* work, cudaStream_t st) {
    if (xdtype == UQ_W_BF16) return gemv_g<Q, XBF16>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st);
    return gemv_g<Q, XF32>(planes, astar, zstar, out, n_in, g, x, batch, y, work, st);
}

cudaError_t launch_gemv(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in, int q,
                        int g, const void* x, int xdtype, int batch, float* y, float* work, cudaStream_t st) {
    switch (q) {
        case 1: return gemv_x<1>(planes, astar, zstar, out, n_in, g, x, xdtype, batch, y, work, st);
        case 2: return gemv_x<2>(planes, astar, zstar, out, n_in, g, x, xdtype, batch, y, work, st);
        case 3: return gemv_x<3>(planes, astar, zstar, out, n_in, g, x, xdtype, batch, y, work, st);
        default: return gemv_x<4>(planes, astar, zstar, out, n_in, g, x, xdtype, batch, y, work, st);
    }
}

}  // namespace uq
