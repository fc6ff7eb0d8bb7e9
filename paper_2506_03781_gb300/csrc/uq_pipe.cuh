// Building blocks of the persistent TMA-pipelined kernels: bounded mbarrier
// waits, bulk global->shared copies, the shared-memory stage layout of one
// work unit, and the stage ring counter.
//
// A warp's pipeline: lane 0 arms an mbarrier with the byte count of a unit
// (expect_tx) and issues one cp.async.bulk per input stream into a stage;
// the warp waits on that mbarrier (bounded, see bar_wait) and computes from
// shared memory.  Every copy starts and ends on a 16-byte boundary.
#pragma once

#include <atomic>

#include "uq_common.cuh"
#include "uq_launch.h"

namespace uq {

#ifndef UQ_WAIT_HINT_NS
#define UQ_WAIT_HINT_NS 20000
#endif
constexpr uint32_t kWaitHintNs = UQ_WAIT_HINT_NS;   // suspend-time hint of one try_wait
// Bit of a kernel family's device flag set when, after a wait ran out, the
// bounded wait for the copies still in flight ran out too (bits 0-2 name the
// wait that ran out first).
constexpr unsigned int kDrainTimeoutBit = 8u;

namespace tma {

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void bar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void bar_init_fence() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void bar_arrive_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void bar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool bar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// try_wait with a suspend-time hint: the warp is parked by the hardware
// until the phase completes or about `ns` nanoseconds pass, instead of
// spinning through issue slots.
__device__ __forceinline__ bool bar_try_wait_sleep(uint32_t bar, uint32_t parity, uint32_t ns) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(ns)
        : "memory");
    return ok != 0;
}
// Bounded wait: gives up after `limit` GPU clock cycles (default 2^31, about one second).
__device__ __forceinline__ bool bar_wait(uint32_t bar, uint32_t parity, long long limit = 1ll << 31) {
    if (bar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    while (!bar_try_wait_sleep(bar, parity, kWaitHintNs)) {
        if (clock64() - t0 > limit) return false;
    }
    return true;
}
__device__ __forceinline__ void fence_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
// Global -> shared bulk copy; bytes a multiple of 16, both addresses 16-byte aligned.
__device__ __forceinline__ void copy_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

}  // namespace tma

constexpr int align_up(int x, int a) { return (x + a - 1) / a * a; }

constexpr int kMaxStages = 16;

// Shared-memory stage layout of one work unit.  HAS_X: weights and s are
// staged; HAS_G: dL/dW^ is staged; HAS_C: code words are staged.  The group
// parameters (Delta, z_U, z_B, alpha of the unit's NG groups) always are.
// HAS_S: s is staged with the weights (by default exactly when they are).
// GBYTES: bytes of one staged dL/dW^ element (4 for fp32, 2 for bf16).
template <int Q, typename WT, int G_, bool HAS_X, bool HAS_G, bool HAS_C, int BUDGET, bool HAS_S = HAS_X,
          int GBYTES = 4>
struct Stage {
    static constexpr int LPG = G_ <= 64 ? 4 : 8;
    static constexpr int NG = 32 / LPG;                  // groups per unit
    static constexpr int NV = G_ / (4 * LPG);            // vectors per lane
    static constexpr int UE = NG * G_;                   // elements per unit
    static constexpr int WBYTES = sizeof(typename WT::raw) / 4;
    static constexpr int SZ_W = HAS_X ? UE * WBYTES : 0;
    static constexpr int SZ_S = HAS_S ? UE * 4 : 0;
    static constexpr int GB = GBYTES;
    static constexpr int SZ_G = HAS_G ? UE * GBYTES : 0;
    static constexpr int SZ_C = HAS_C ? UE : 0;
    static constexpr int SZ_P = NG * 4, SZ_A = NG * Q * 4;
    static constexpr int OFF_W = 0;
    static constexpr int OFF_S = align_up(OFF_W + SZ_W, 16);
    static constexpr int OFF_G = OFF_S + SZ_S;
    static constexpr int OFF_C = OFF_G + SZ_G;
    static constexpr int OFF_D = align_up(OFF_C + SZ_C, 16);
    static constexpr int OFF_Z = OFF_D + SZ_P;
    static constexpr int OFF_B = OFF_Z + SZ_P;
    static constexpr int OFF_A = OFF_B + SZ_P;
    static constexpr int BYTES = align_up(OFF_A + SZ_A, 128);
    static constexpr uint32_t TX = SZ_W + SZ_S + SZ_G + SZ_C + 3 * SZ_P + SZ_A;   // bytes copied per unit
    // stages per warp within the per-warp shared-memory budget
    static constexpr int FIT = BUDGET / BYTES;
    static constexpr int NST = FIT < 2 ? 2 : (FIT > kMaxStages ? kMaxStages : FIT);
    static constexpr int WARP_BYTES = NST * BYTES;
    static_assert(SZ_P % 16 == 0 && SZ_A % 16 == 0 && SZ_C % 16 == 0, "bulk copy sizes must be multiples of 16");
};

// Stage ring position: stage index and the mbarrier phase parity of its next completion.
template <int NST>
struct Ring {
    int s = 0;
    uint32_t parity = 0;
    __device__ void next() {
        if (++s == NST) { s = 0; parity ^= 1u; }
    }
};

// Work items of one warp: for its row blocks k = 0, 1, ... (block rows
// (blockIdx.x + k * gridDim.x) * R + row_sub) the units wr, wr + WPR, ...
// (n_w per row block).  Positions advance with Cursor::next, without
// integer division.
struct Items {
    int R, WPR, row_sub, wr, n_w, n_blocks;
    long long total;
    __device__ Items(int U, int Rr, int n_rb, int warp) {
        R = Rr;
        WPR = kWarps / R;
        row_sub = warp / WPR;
        wr = warp % WPR;
        n_w = wr < U ? (U - wr + WPR - 1) / WPR : 0;
        n_blocks = (n_rb - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x;
        total = (long long)n_blocks * n_w;
    }
    __device__ int64_t row(int k) const { return ((int64_t)blockIdx.x + (int64_t)k * gridDim.x) * R + row_sub; }
    __device__ int unit(int j) const { return wr + WPR * j; }
};

struct Cursor {
    int k = 0, j = 0;                        // row block, unit slot
    __device__ void next(int n_w) {
        if (++j == n_w) { j = 0; ++k; }
    }
};


// After a wait ran out: waits (bounded again) for the copies of items
// [waited, issued) of a warp's stage ring, so that none lands in shared
// memory after the block has exited.  Lane 0 only.  False if one of these
// waits ran out as well: the block may then exit with copies still in
// flight into its shared memory, and the caller records kDrainTimeoutBit.
template <int NST>
__device__ bool drain(unsigned long long (&bars)[NST], long long waited, long long issued) {
    for (long long i = waited; i < issued; ++i)
        if (!tma::bar_wait(tma::smem_addr(&bars[i % NST]), (uint32_t)((i / NST) & 1))) return false;
    return true;
}

// The per-warp pipeline over a warp's work items, in Items/Cursor order:
// lane 0 keeps the copies of NST items in flight -- issue(cursor, stage)
// arms the stage's mbarrier and starts them -- and the warp waits (bounded)
// for each item in turn, runs body(cursor, stage) on it and refills the
// stage.  A wait that runs out sets `bit` in *flag, waits (bounded) for the
// copies still in flight and returns false; for use in kernels without
// block barriers.  Shared by the pipelined forwards and the OmniQuant and
// AWQ backwards, which differ only in what they stage and compute.
template <int NST, typename Issue, typename Body>
__device__ __forceinline__ bool pipe_run(const Items& it, unsigned long long (&bars)[NST], int lane,
                                         unsigned int* flag, unsigned int bit, Issue&& issue, Body&& body) {
    Cursor ic;                                   // next item to issue (lane 0)
    long long issued = 0;
    if (lane == 0) {
        for (int s = 0; s < NST && issued < it.total; ++s, ++issued) {
            issue(ic, s);
            ic.next(it.n_w);
        }
    }
    Ring<NST> ring;
    Cursor cc;                                   // item being computed
    for (long long i = 0; i < it.total; ++i) {
        const int s = ring.s;
        if (!__all_sync(kFull, tma::bar_wait(tma::smem_addr(&bars[s]), ring.parity))) {
            if (lane == 0) {
                atomicOr(flag, bit);
                if (!drain(bars, i, issued)) atomicOr(flag, kDrainTimeoutBit);
            }
            return false;
        }
        body(static_cast<const Cursor&>(cc), s);
        __syncwarp();                            // the stage is free again
        if (lane == 0 && issued < it.total) {
            issue(ic, s);
            ic.next(it.n_w);
            ++issued;
        }
        ring.next();
        cc.next(it.n_w);
    }
    return true;
}

constexpr int kMaxDevices = 64;

// Persistent grid: min(row blocks, SMs x resident blocks per SM).  The
// shared-memory attribute and the occupancy of a kernel instantiation are
// set and queried once per device (KERN is a distinct type per call site);
// the cache is atomic, so first calls from several host threads may race
// only to store the same value.
template <typename Tag, typename KERN>
static cudaError_t grid_for(KERN kern, size_t dyn, int n_rb, int& grid) {
    static std::atomic<int> per_sm_cache[kMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    int per_sm = (dev >= 0 && dev < kMaxDevices) ? per_sm_cache[dev].load(std::memory_order_relaxed) : 0;
    if (per_sm == 0) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn);
        if (e != cudaSuccess) return e;
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, dyn);
        if (e != cudaSuccess) return e;
        if (per_sm < 1) per_sm = 1;
        if (dev >= 0 && dev < kMaxDevices) per_sm_cache[dev].store(per_sm, std::memory_order_relaxed);
    }
    const long long cap = (long long)sm_count() * per_sm;
    grid = (int)(n_rb < cap ? n_rb : cap);
    return cudaSuccess;
}

}  // namespace uq
