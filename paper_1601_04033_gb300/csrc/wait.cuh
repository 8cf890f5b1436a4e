// Shared-memory mbarrier wrappers (inline PTX) and the bounded waits of the
// dense pass's copy pipeline: a wait gives up after about a second of
// %globaltimer (or 2^26 polls), raises kErrWaitTimeout in the caller's error
// word and returns false, so a pipeline that can never complete ends the
// kernel with an error the host reads (fasgd_sync) instead of hanging it.
#pragma once

#include <stdint.h>

namespace fasgd {
namespace {

constexpr int kErrWaitTimeout = 8;
constexpr uint64_t kWaitLimitNs = 1000000000ull;

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t* bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// One thread waits for the phase with the given parity to complete.
__device__ bool wait_one(uint64_t* bar, uint32_t parity, int32_t* err) {
    if (mbar_test(bar, parity)) return true;
    const uint64_t t0 = global_ns();
    for (uint32_t i = 0; i < (1u << 26); ++i) {
        if (mbar_test(bar, parity)) return true;
        if ((i & 255u) == 255u && global_ns() - t0 > kWaitLimitNs) break;
    }
    atomicOr(err, kErrWaitTimeout);
    return false;
}
// A whole warp waits; every lane observes the barrier (acquire) and the warp
// leaves together.
__device__ bool wait_warp(uint64_t* bar, uint32_t parity, int32_t* err) {
    const uint64_t t0 = global_ns();
    for (uint32_t i = 0; i < (1u << 26); ++i) {
        if (__all_sync(0xffffffffu, mbar_test(bar, parity))) return true;
        const bool late = (i & 255u) == 255u && global_ns() - t0 > kWaitLimitNs;
        if (__any_sync(0xffffffffu, late)) break;
    }
    if ((threadIdx.x & 31) == 0) atomicOr(err, kErrWaitTimeout);
    return false;
}
}  // namespace
}  // namespace fasgd
