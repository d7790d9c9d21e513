// schedule_common.cuh -- device pieces shared by the two transports of the
// schedule-faithful kernel: counters and block reads (schedule.cu) and
// flagged words (schedule_ll.cu).
#pragma once

#include "dpdr_internal.h"
#include "ops.cuh"

namespace dpdr {
namespace sched {

constexpr int kMaxThreads = 256;
constexpr int kMaxGroups = 4;  // rank groups per CTA

// Rank groups of a CTA that owns R virtual ranks: min(R, warps, kMaxGroups)
// groups of whole warps, all of one size, each running its own ranks.
inline int group_count(int R, int threads)
{
    const int warps = threads / 32;
    return R < 1 ? 1 : (R < warps ? (R < kMaxGroups ? R : kMaxGroups)
                                  : (warps < kMaxGroups ? warps : kMaxGroups));
}
__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p)
{
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ void st_release(uint32_t* p, uint32_t v)
{
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ void st_relaxed(uint32_t* p, uint32_t v)
{
    asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ uint32_t ld_relaxed(const uint32_t* p)
{
    uint32_t v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ uint64_t now_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// First element of block j of Algorithm 1's partition of m elements into b
// blocks (q = floor(m/b), rem = m mod b: the first rem blocks are one longer).
__device__ __forceinline__ int64_t block_start(int64_t q, int64_t rem, int j)
{
    return int64_t(j) * q + lmin(j, rem);
}

// Start of column slice g (of n) of the element range [s, e): even shares,
// inner boundaries rounded down to a multiple of EPV elements.
template <int EPV>
__device__ __forceinline__ int64_t slice_bound(int64_t s, int64_t e, int g, int n)
{
    if (g <= 0) return s;
    if (g >= n) return e;
    const int64_t b = (s + (e - s) * g / n) / EPV * EPV;
    return b < s ? s : b;
}

__device__ __forceinline__ const char* rank_in(const char* const* t, int i)
{
    return reinterpret_cast<const char*>(__ldg(reinterpret_cast<const unsigned long long*>(t) + i));
}
__device__ __forceinline__ char* rank_out(char* const* t, int i)
{
    return reinterpret_cast<char*>(__ldg(reinterpret_cast<const unsigned long long*>(t) + i));
}

}  // namespace sched
}  // namespace dpdr
