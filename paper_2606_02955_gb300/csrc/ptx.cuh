// ptx.cuh -- inline-PTX building blocks for sm_103a: mbarriers, 1-D bulk (TMA) copies,
// the MUFU base-2 exponential and bounded waits.
#pragma once

#include <cstdint>

namespace fdllm {

// A wait on an mbarrier gives up after this long and records kDevStatTimeout.
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s
// After a wait gave up, how long a CTA waits for its own asynchronous copies still in
// flight (they write its shared memory) before it exits.
constexpr uint64_t kDrainLimitNs = 100000000ull;  // 100 ms
// Bits of a workspace's sticky status word.  kDevStatTimeout: a kernel gave up a bounded
// wait (the step's rows report FDLLM_ROW_DEVICE_ERROR).  kDevStatNonfinite: a selection
// found a batch row with unusable logits (FDLLM_ROW_NONFINITE); the kernels themselves
// completed normally, so only the timeout bit makes later kernels treat the step as failed.
constexpr uint32_t kDevStatTimeout = 1u;
constexpr uint32_t kDevStatNonfinite = 2u;

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

// Makes barrier initialisation visible to the async (TMA) proxy and the rest of the CTA.
__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ uint64_t global_timer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Waits for the phase of `bar` with the given parity to complete.  Gives up after
// limit_ns, sets kDevStatTimeout in *status and returns false.
__device__ __forceinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, uint32_t *status,
                                          uint64_t limit_ns = kWaitLimitNs)
{
    if (mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 1;; ++it) {
        if (mbar_try_wait(bar, parity))
            return true;
        if ((it & 63u) == 0 && global_timer_ns() - t0 > limit_ns) {
            atomicOr(status, kDevStatTimeout);
            return false;
        }
    }
}

// One 1-D bulk copy global -> shared, completing `bytes` of transaction count on `bar`.
// dst and src 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void bulk_copy_g2s(void *dst, const void *src, uint32_t bytes,
                                              uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::
            "r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// Same copy with an L2 eviction-priority hint (a policy from make_evict_first_policy).
__device__ __forceinline__ void bulk_copy_g2s_hint(void *dst, const void *src, uint32_t bytes,
                                                   uint64_t *bar, uint64_t policy)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

// L2 policy marking every line a copy brings in as first to evict (data read once).
__device__ __forceinline__ uint64_t make_evict_first_policy()
{
    uint64_t policy;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(policy));
    return policy;
}

}  // namespace fdllm
