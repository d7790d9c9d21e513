// fused_split.cu -- subtree-split layout of the fused kernel (two kernels:
// a read phase that folds subtrees, a write phase that finishes the top of
// the tree and stores the result) and its plan-time preparation.
#include "fused_common.cuh"

namespace dpdr {
namespace fused {
namespace {

// -------------------------------------------------------------------- split
// For m too small to give every SM enough columns but p large: the rank axis
// is cut at a tree depth s.  Kernel 1 folds each depth-s subtree (a
// contiguous post-order interval) for its columns, in parallel over
// (subtree, column), and writes the subtree value to a scratch row; it also
// copies the inputs of the nodes above depth s into scratch rows.  Kernel 2
// folds the nodes above depth s from those rows, each subtree entering as
// one finished child, forms v(r0) (.) v(r1), and stores it to one group of
// ranks per CTA row.  The bracketing is unchanged: each subtree value is
// exactly its node value.
template <class U>
__device__ __forceinline__ void split_reduce_column(const FusedArgs& a, int g, int64_t u,
                                                    typename U::T* slot, int stride)
{
    using T = typename U::T;
    const int2 sg = __ldg(a.seg + g);
    const int lo = sg.x, hi = sg.y;  // inclusive; lo is a leaf unless lo == hi
    char* row = a.part + int64_t(g) * a.part_stride;
    if (lo == hi) {  // a one-leaf subtree, or a node above the cut: its input
        U::st_keep(row, u, U::ld(rank_ptr(a.x, lo), u));
        return;
    }
    T acc{};  // set by rank lo, a leaf
    for (int i0 = lo; i0 <= hi; i0 += kStreamAhead) {
        T cur[kStreamAhead];
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k <= hi) cur[k] = U::ld(rank_ptr(a.x, i0 + k), u);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k <= hi) fold_step<U>(__ldg(a.tape + i0 + k), cur[k], acc, slot, stride);
    }
    U::st_keep(row, u, acc);
}

template <class U>
__device__ __forceinline__ void split_finish_column(const FusedArgs& a, int r, int64_t u,
                                                    typename U::T* slot, int stride)
{
    using T = typename U::T;
    const int n = a.nitems;
    // every item is a scratch row: a subtree value or a copied input, so
    // this kernel never reads an input that another CTA may be overwriting
    // with the result (in-place use)
    auto load = [&](int k) -> T {
        return U::ld_keep(a.part + int64_t(__ldg(&a.items[k].x)) * a.part_stride, u);
    };
    T acc{};  // set by the first item, a subtree
    for (int k0 = 0; k0 < n; k0 += kStreamAhead) {
        T cur[kStreamAhead];
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (k0 + k < n) cur[k] = load(k0 + k);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (k0 + k < n)
                fold_step<U>(unsigned(__ldg(&a.items[k0 + k].y)) & 0xffu, cur[k], acc, slot, stride);
    }
    const T y = a.dual ? U::op(slot[0], acc) : acc;
    const int i1 = min(a.p, (r + 1) * a.group);
#pragma unroll 4
    for (int i = r * a.group; i < i1; i++) U::st(rank_ptr_w(a.y, i), u, y);
}

template <class Op>
__global__ void __launch_bounds__(kStreamThreads, 4)
fused_split_reduce_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int64_t u = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (u < a.nvec) {
        split_reduce_column<VecUnit<Op>>(a, blockIdx.y, u, smem + threadIdx.x, blockDim.x);
    } else if (u < a.nvec + a.nscalar) {
        split_reduce_column<OneUnit<Op>>(a, blockIdx.y, a.scalar_base + (u - a.nvec),
                                         one_slots<Op>(smem, threadIdx.x),
                                         one_slot_stride<Op>(blockDim.x));
    }
}

template <class Op>
__global__ void __launch_bounds__(kStreamThreads, 4)
fused_split_finish_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int64_t u = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (u < a.nvec) {
        split_finish_column<VecUnit<Op>>(a, blockIdx.y, u, smem + threadIdx.x, blockDim.x);
    } else if (u < a.nvec + a.nscalar) {
        split_finish_column<OneUnit<Op>>(a, blockIdx.y, a.scalar_base + (u - a.nvec),
                                         one_slots<Op>(smem, threadIdx.x),
                                         one_slot_stride<Op>(blockDim.x));
    }
}


template <class Op>
struct Split {
    static int run(Plan* P, FusedArgs a, cudaStream_t s)
    {
        const int64_t units = a.nvec + a.nscalar;
        const int64_t blocks = (units + kStreamThreads - 1) / kStreamThreads;
        const size_t smem = size_t(P->max_depth + 1) * kStreamThreads * sizeof(uint4);
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        if (int(smem) > P->smem_attr[2]) {
            int granted = P->smem_attr[2];
            if (int rc = grant_smem(reinterpret_cast<const void*>(&fused_split_reduce_kernel<Op>),
                                    smem, &granted, "fused split attribute"))
                return rc;
            if (int rc = grant_smem(reinterpret_cast<const void*>(&fused_split_finish_kernel<Op>),
                                    smem, &P->smem_attr[2], "fused split attribute"))
                return rc;
        }
        const int groups = (P->p + a.group - 1) / a.group;
        fused_split_reduce_kernel<Op>
            <<<dim3(unsigned(blocks), unsigned(P->split_nseg)), kStreamThreads, smem, s>>>(a);
        fused_split_finish_kernel<Op>
            <<<dim3(unsigned(blocks), unsigned(groups)), kStreamThreads, smem, s>>>(a);
        return launched();
    }
};

}  // namespace

int launch_split(Plan* P, FusedArgs a, cudaStream_t s) { return dispatch<Split>(P, a, s); }

}  // namespace fused
}  // namespace dpdr
