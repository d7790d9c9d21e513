// tma.cuh -- thin wrappers of the TMA bulk-copy and mbarrier instructions
// (PTX cp.async.bulk, mbarrier.*) used by the schedule kernel's staged
// block passes.
#pragma once

#include <cstdint>

namespace dpdr {
namespace tma {

__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count) : "memory");
}
// makes initialised mbarriers visible to the async proxy (the TMA unit)
__device__ __forceinline__ void fence_mbar_init()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)),
                 "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint64_t* b, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(smem_u32(b)), "r"(parity)
        : "memory");
    return ok != 0;
}
// global -> shared bulk copy of `bytes` (a multiple of 16, both addresses
// 16-byte aligned) whose completion counts against mbarrier bar's
// transaction bytes
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}
// orders this thread's view of global memory written through ordinary
// stores (by any thread it has synchronised with) before its later bulk
// copies, which run in the async proxy
__device__ __forceinline__ void fence_proxy_async_global()
{
    asm volatile("fence.proxy.async.global;" ::: "memory");
}
// brings [p, p + bytes) into L2 (a multiple of 16 bytes, 16-byte aligned)
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
// drops the 128-byte L2 line at p without writing it back; its contents
// become undefined
__device__ __forceinline__ void discard_l2_line(const void* p)
{
    asm volatile("discard.global.L2 [%0], 128;" ::"l"(p) : "memory");
}

}  // namespace tma
}  // namespace dpdr
