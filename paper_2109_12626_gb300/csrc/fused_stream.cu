// fused_stream.cu -- column-streaming layout of the fused kernel: one
// thread owns one 16-byte column unit and walks the p ranks in post-order
// (the running fold of fused_common.cuh), eight ranks' loads ahead of the
// fold, then stores the result to all p outputs.  Suits m >> p.  With few
// columns, a pair of threads shares each column, one per tree.
#include "fused_common.cuh"

namespace dpdr {
namespace fused {
namespace {

// A pair of threads per column (one per tree) below kStreamPairUnitsPerSm
// columns per SM and from kStreamPairMinRanks ranks: p = 32, m = 2^16 int32
// in 6.6 us against 9.0, p = 64 in 12.0 against 17.5, p = 127, m = 2^17 in
// 29.0 against 34.8 (warm L2); at p = 2 to 7 the walks are short already
// and the pairing costs (p = 7, m = 1000: 3.2 against 2.8 us).
constexpr int64_t kStreamPairUnitsPerSm = 1024;
constexpr int kStreamPairMinRanks = 16;

template <class Op>
__global__ void __launch_bounds__(kStreamThreads, 4)
fused_stream_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int64_t u = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (u < a.nvec) {
        stream_column<VecUnit<Op>>(a, u, smem + threadIdx.x, blockDim.x);
    } else if (u < a.nvec + a.nscalar) {
        stream_column<OneUnit<Op>>(a, a.scalar_base + (u - a.nvec), one_slots<Op>(smem, threadIdx.x),
                                   one_slot_stride<Op>(blockDim.x));
    }
}


// The partner lane's value (lane ^ 16); only the two lanes take part.
__device__ __forceinline__ uint32_t swap_half(uint32_t v, unsigned pair)
{
    return __shfl_xor_sync(pair, v, 16);
}
__device__ __forceinline__ uint4 swap_half(const uint4& v, unsigned pair)
{
    return make_uint4(swap_half(v.x, pair), swap_half(v.y, pair), swap_half(v.z, pair),
                      swap_half(v.w, pair));
}
template <class Op>
__device__ __forceinline__ Elem<Op> swap_half(const Elem<Op>& v, unsigned pair)
{
    Elem<Op> o;
#pragma unroll
    for (int k = 0; k < Elem<Op>::kWords; k++) o.w[k] = swap_half(v.w[k], pair);
    return o;
}

// One tree's half of a column: the running fold over the tree's ranks
// [lo, hi) (tape bytes read 8 at a time from an 8-aligned start), the
// roots swapped with the partner lane, y = v(r0) (.) v(r1) formed in the
// same operand order by both, and y stored to the tree's own outputs.
template <class U>
__device__ __forceinline__ void stream_half(const FusedArgs& a, int64_t u, int h, unsigned pair,
                                            typename U::T* slot, int stride)
{
    using T = typename U::T;
    const int n0 = a.r0 + 1;
    const int lo = h ? n0 : 0, hi = h ? a.p : n0;
    T acc{};  // set by rank lo, a leaf
    for (int i0 = lo & ~(kStreamAhead - 1); i0 < hi; i0 += kStreamAhead) {
        T cur[kStreamAhead];
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k >= lo && i0 + k < hi) cur[k] = U::ld(rank_ptr(a.x, i0 + k), u);
        const unsigned long long tp =
            __ldg(reinterpret_cast<const unsigned long long*>(a.tape + i0));
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k >= lo && i0 + k < hi)
                fold_step<U>(unsigned(tp >> (8 * k)) & 0xffu, cur[k], acc, slot, stride);
    }
    const T other = swap_half(acc, pair);
    const T y = h ? U::op(other, acc) : U::op(acc, other);
#pragma unroll 4
    for (int i = lo; i < hi; i++) U::st(rank_ptr_w(a.y, i), u, y);
}

// Two threads per column, one per tree: Sec. 1.1's trees are disjoint
// rank intervals [0, n0) and [n0, p) that meet only in y = v(r0) (.) v(r1).
// Lanes 0-15 of a warp walk tree 0 for 16 columns, lanes 16-31 tree 1 for
// the same columns, so a plan with fewer columns than the GPU keeps in
// flight gets twice the threads and half the walk per thread.
template <class Op>
__global__ void __launch_bounds__(kStreamThreads, 4)
fused_stream_pair_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int lane = threadIdx.x & 31, h = lane >> 4;
    const int64_t c = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) / 32 * 16 + (lane & 15);
    const unsigned pair = (1u << lane) | (1u << (lane ^ 16));
    if (c < a.nvec) {
        stream_half<VecUnit<Op>>(a, c, h, pair, smem + threadIdx.x, blockDim.x);
    } else if (c < a.nvec + a.nscalar) {
        stream_half<OneUnit<Op>>(a, a.scalar_base + (c - a.nvec), h, pair,
                                 one_slots<Op>(smem, threadIdx.x), one_slot_stride<Op>(blockDim.x));
    }
}

template <class Op>
struct Stream {
    static int run(Plan* P, FusedArgs a, cudaStream_t s)
    {
        const int64_t units = a.nvec + a.nscalar;
        // a pair of threads per column while the columns alone leave the
        // GPU short of threads (dual trees only)
        const bool pairs = a.dual && a.p >= kStreamPairMinRanks &&
                           units < kStreamPairUnitsPerSm * int64_t(P->num_sms);
        const int64_t threads = pairs ? (units + 15) / 16 * 32 : units;
        const int64_t blocks = (threads + kStreamThreads - 1) / kStreamThreads;
        const size_t smem = size_t(P->max_depth + 1) * kStreamThreads * sizeof(uint4);
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        const void* kern = pairs ? reinterpret_cast<const void*>(&fused_stream_pair_kernel<Op>)
                                 : reinterpret_cast<const void*>(&fused_stream_kernel<Op>);
        if (int rc = grant_smem(kern, smem, &P->smem_attr[pairs ? 6 : 0], "fused stream attribute"))
            return rc;
        if (pairs)
            fused_stream_pair_kernel<Op><<<unsigned(blocks), kStreamThreads, smem, s>>>(a);
        else
            fused_stream_kernel<Op><<<unsigned(blocks), kStreamThreads, smem, s>>>(a);
        return launched();
    }
};

}  // namespace

int launch_stream(Plan* P, FusedArgs a, cudaStream_t s) { return dispatch<Stream>(P, a, s); }

}  // namespace fused
}  // namespace dpdr
