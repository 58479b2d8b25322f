// PTX helpers of the evaluation-pass kernels for sm_103a: mbarriers and 1-D bulk copies (the TMA
// engine's cp.async.bulk), with bounded waits.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "esp_common.h"

namespace esp {

namespace {

// ---------------------------------------------------------------------------------------------
// PTX helpers: mbarrier + 1-D bulk copy (TMA engine), sm_90+ forms that sm_103a accepts.

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// Hint: bring [src, src + bytes) into L2 (16-byte aligned address and size).
__device__ __forceinline__ void prefetch_l2(const void *src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

__device__ __forceinline__ void fence_proxy_async()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Plain arrival (one count) on a barrier.
__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// Waits on the phase of the given parity without a time hint: the thread may be suspended for a short,
// system-dependent time and resumes when the phase completes.
__device__ __forceinline__ bool mbar_try_wait_nohint(uint32_t bar, uint32_t parity)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(bar), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ uint64_t global_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait on a stage barrier: polls the phase (try_wait without a time hint resumes as soon as
// the phase completes) and gives up after `limit_ms` milliseconds of the GPU's global timer (4096 by
// default: seconds), flags a timeout and returns false so that the kernel can finish instead of
// hanging.
__device__ __forceinline__ bool wait_stage(uint32_t bar, uint32_t parity, unsigned int *err, uint32_t limit_ms)
{
    if (mbar_try_wait_nohint(bar, parity))
        return true;
    const uint64_t t0 = global_ns();
    const uint64_t limit = (uint64_t)limit_ms * 1000000ull;
    for (;;) {
        if (mbar_try_wait_nohint(bar, parity))
            return true;
        if (global_ns() - t0 > limit)
            break;
    }
    atomicOr(err, DEV_ERR_TIMEOUT);
    return false;
}

// Bounded wait until a shared word holds `want` (a stage's sequence word): polls it and gives up after
// `limit_ms` milliseconds of the global timer, flagging a timeout.
__device__ __forceinline__ bool wait_word(const volatile int *w, int want, unsigned int *err, uint32_t limit_ms)
{
    if (*w == want)
        return true;
    const uint64_t t0 = global_ns();
    const uint64_t limit = (uint64_t)limit_ms * 1000000ull;
    for (;;) {
        __nanosleep(32);
        if (*w == want)
            return true;
        if (global_ns() - t0 > limit)
            break;
    }
    atomicOr(err, DEV_ERR_TIMEOUT);
    return false;
}

}  // namespace

}  // namespace esp
