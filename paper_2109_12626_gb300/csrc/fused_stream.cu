// fused_stream.cu -- column-streaming layout of the fused kernel: one
// thread owns one 16-byte column unit and walks the p ranks in post-order
// (the running fold of fused_common.cuh), eight ranks' loads ahead of the
// fold, then stores the result to all p outputs.  Suits m >> p.
#include "fused_common.cuh"

namespace dpdr {
namespace fused {
namespace {

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


template <class Op>
struct Stream {
    static int run(Plan* P, FusedArgs a, cudaStream_t s)
    {
        const int64_t units = a.nvec + a.nscalar;
        const int64_t blocks = (units + kStreamThreads - 1) / kStreamThreads;
        const size_t smem = size_t(P->max_depth + 1) * kStreamThreads * sizeof(uint4);
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        if (int rc = grant_smem(reinterpret_cast<const void*>(&fused_stream_kernel<Op>), smem,
                                &P->smem_attr[0], "fused stream attribute"))
            return rc;
        fused_stream_kernel<Op><<<unsigned(blocks), kStreamThreads, smem, s>>>(a);
        return launched();
    }
};

}  // namespace

int launch_stream(Plan* P, FusedArgs a, cudaStream_t s) { return dispatch<Stream>(P, a, s); }

}  // namespace fused
}  // namespace dpdr
