// stream.cuh -- persistent row streaming through a shared-memory ring filled by
// 1-D bulk copies (cp.async.bulk, the TMA engine), sm_90+ / sm_103a.
//
// A launch streams R rows of V logits.  Rows are cut into tiles of kTileBytes
// (the last tile of a row may be short).  The R * tiles_per_row tiles are split
// into gridDim.x contiguous ranges, one per persistent CTA, so every CTA moves
// the same number of bytes; the part of a row that falls in one CTA's range is
// a "segment" of that row.  Thread 0 keeps kStages tiles in flight; every
// thread waits on the stage's mbarrier (bounded in time), processes the tile
// from shared memory, and the stage is refilled after a block barrier.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "rheo_device.cuh"

namespace rheo {

constexpr int kTileBytes = 16384;
constexpr int kStages = 4;     // ring depth of kernels with two CTAs per SM
constexpr int kMaxStages = 8;  // deepest ring (one CTA per SM)
constexpr unsigned long long kWaitLimitNs = 2000000000ull;  // 2 s: a copy that never lands is an error
constexpr uint32_t kStTimeout = 16u;

__device__ __forceinline__ uint32_t smem_u32(const void* p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void mbar_init(uint64_t* bar, unsigned count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, unsigned bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
                 : "memory");
}

// 1-D bulk copy global -> shared; completion counted on the mbarrier in bytes.
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_load(void* dst, const void* src, unsigned bytes, uint64_t* bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}

__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}

// Wait for phase `parity` of the mbarrier; gives up after kWaitLimitNs.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, unsigned parity) {
    const uint32_t a = smem_u32(bar);
    unsigned long long t0 = 0;
    for (unsigned it = 0;; ++it) {
        uint32_t ok;
        asm volatile(
            "{\n\t.reg .pred p;\n\t"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
            "selp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(a), "r"(parity)
            : "memory");
        if (ok) return true;
        if (it == 0) t0 = global_ns();
        else if ((it & 63) == 0 && global_ns() - t0 > kWaitLimitNs) return false;
    }
}

// Static split of the tile space over the persistent CTAs.
struct TileSplit {
    int64_t total;  // R * tpr
    int G;          // CTAs
    __device__ __forceinline__ int64_t begin(int i) const { return (int64_t)i * total / G; }
    // CTA whose range holds tile t
    __device__ __forceinline__ int owner(int64_t t) const { return (int)((t * G + G - 1) / total); }
};

}  // namespace rheo
