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
// shared-memory stages filled by asynchronous copies.  Lane l owns columns
// 16 l .. 16 l + 15 of the tile (one 16-bit half of a plane word).  A warp
// takes 8 rows at a time; a reduce-scatter over the warp (uq_common.cuh,
// SegReduce) leaves one row's tile partial on each of 8 lanes, which store it
// to the caller's workspace [tile][token][row].  A second kernel sums the
// partials of a row in tile order.  Deterministic; no atomics.
#include <atomic>

#include "uq_common.cuh"
#include "uq_launch.h"

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

// y[b, r] = sum over tiles of PART[t, b, r], in tile order.
__global__ void __launch_bounds__(256)
bcq_gemv_reduce_kernel(const float* __restrict__ PART, float* __restrict__ Y, int64_t n, int n_tiles) {
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

// Device address of g_gemv_static_work on the current device.  The name is
// only a host-side stand-in in host code, so the address is looked up once
// per device with that device current, and cached.
cudaError_t gemv_static_workspace(float** work) {
    static std::atomic<float*> cached[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) {
        float* p = cached[dev].load(std::memory_order_acquire);
        if (p != nullptr) {
            *work = p;
            return cudaSuccess;
        }
    }
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_gemv_static_work);
    if (e != cudaSuccess) return e;
    if (dev >= 0 && dev < 64) cached[dev].store(static_cast<float*>(p), std::memory_order_release);
    *work = static_cast<float*>(p);
    return cudaSuccess;
}

template <int Q, typename XT, int NGT>
static cudaError_t run_gemv(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in,
                            int g, const void* x, int batch, float* y, float* work, cudaStream_t st) {
    auto kern = bcq_gemv_partial_kernel<Q, XT, NGT>;
    constexpr size_t stage_bytes = (size_t)gemv_stage_words(Q, NGT) * 4;
    constexpr size_t smem = kGemvFixedSmem + kGemvWarps * (size_t)gemv_stages(Q, NGT) * stage_bytes;
    static_assert(gemv_stages(Q, NGT) >= 2 && smem <= kGemvSmemLimit, "two stages must fit");
    // alpha* and z* rows of a tile move in 16-byte pieces when every tile is
    // whole (in a multiple of 512) and holds a multiple of 4 groups (both
    // arrays start on 16-byte boundaries: the entry point checks that);
    // otherwise in 4-byte pieces
    const bool pwide = NGT % 4 == 0 && n_in % kTileCols == 0;
    static int per_sm_cache[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int per_sm = (dev >= 0 && dev < 64) ? per_sm_cache[dev] : 0;
    if (per_sm == 0) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kGemvThreads, smem);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) per_sm = 1;
        if (dev >= 0 && dev < 64) per_sm_cache[dev] = per_sm;
    }
    // Row blocks (of whole 8-row batches): the count that minimises
    // waves x (one table build, worth about 32 rows, + rows per block), where
    // a wave is one block per resident slot.
    const int n_tiles = (n_in + kTileCols - 1) / kTileCols;
    const int64_t slots = (int64_t)sm_count() * per_sm;
    const int64_t max_rb = (out + kBatchRows - 1) / kBatchRows;
    int64_t n_rb = 1, rpb = max_rb * kBatchRows;
    double best = -1.0;
    const int64_t lim = max_rb < 8 * slots ? max_rb : 8 * slots;
    for (int64_t cand = 1; cand <= lim; ++cand) {
        int64_t r = (out + cand - 1) / cand;
        r = (r + kBatchRows - 1) / kBatchRows * kBatchRows;
        const int64_t nb = (out + r - 1) / r;
        const int64_t waves = (nb * n_tiles + slots - 1) / slots;
        const double cost = (double)waves * (32.0 + (double)r);
        if (best < 0.0 || cost < best) { best = cost; n_rb = nb; rpb = r; }
    }
    kern<<<(unsigned)(n_rb * n_tiles), kGemvThreads, smem, st>>>(planes, astar, zstar, x, work, out, n_in, g, batch,
                                                                 n_tiles, rpb, pwide);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const int64_t n = (int64_t)batch * out;
    int64_t blocks = (n + 255) / 256;
    const int64_t cap = (int64_t)sm_count() * 8;
    if (blocks > cap) blocks = cap;
    bcq_gemv_reduce_kernel<<<(unsigned)blocks, 256, 0, st>>>(work, y, n, n_tiles);
    return cudaGetLastError();
}

template <int Q, typename XT>
static cudaError_t gemv_g(const uint32_t* planes, const float* astar, const float* zstar, int64_t out, int n_in, int g,
                          const void* x, int batch, float* y, float* work, cudaStream_t st) {
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
