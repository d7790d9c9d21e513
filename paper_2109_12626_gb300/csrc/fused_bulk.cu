// fused_bulk.cu -- bulk-copy pipeline layout of the fused kernel (TMA
// cp.async.bulk loads through an mbarrier ring, bulk stores of the result).
#include "fused_common.cuh"

namespace dpdr {
namespace fused {
namespace {

// --------------------------------------------------------------------- bulk
// Column streaming through a TMA bulk-copy pipeline.  A CTA owns column
// tiles of 4 KB (256 consumer threads x 16 bytes).  One producer thread
// walks the ranks of its tiles in post-order and issues one cp.async.bulk
// load of the tile's 4 KB row piece per rank into a ring of shared-memory
// stages, each stage guarded by a "full" mbarrier (transaction bytes) and an
// "empty" mbarrier (one arrival per consumer warp).  The consumers fold the
// ranks from shared memory with the running post-order fold, write the
// tile's result into one of two result buffers, and one consumer issues p
// bulk stores of that buffer, one per rank output.  The loads in flight per
// CTA are set by the ring depth, not by registers.  Columns past the last
// full tile are folded by the consumers with plain loads.
//
// Every wait is bounded in time; on expiry the CTA records the error in the
// plan's error word, stops issuing, waits (bounded) for its own copies in
// flight, and returns.

__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* b, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(b)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint64_t* b, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(b)),
                 "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* b)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(b)) : "memory");
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
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar))
        : "memory");
}
__device__ __forceinline__ void bulk_store(void* dst, const void* src, uint32_t bytes)
{
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(dst),
                 "r"(smem_u32(src)), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void fence_async_shared() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void consumers_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kBulkConsumers) : "memory"); }
__device__ __forceinline__ uint64_t gtime()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Wait for phase `parity` of barrier b, bounded by a.wait_ns; on expiry
// record the error (step 4: fused pipeline) and raise the CTA's abort flag.
__device__ __forceinline__ bool bulk_wait(const FusedArgs& a, uint64_t* b, uint32_t parity,
                                          volatile int* abort_flag)
{
    if (mbar_test(b, parity)) return true;
    const uint64_t t0 = gtime();
    for (uint32_t it = 1;; it++) {
        if (mbar_test(b, parity)) return true;
        if ((it & 63) == 0) {
            if (*abort_flag) return false;
            if (gtime() - t0 > uint64_t(a.wait_ns)) {
                if (atomicCAS(a.err, 0u, uint32_t(DPDR_ERR_TIMEOUT)) == 0u) {
                    a.err[1] = blockIdx.x;
                    a.err[2] = 0;
                    a.err[3] = 4;
                }
                *abort_flag = 1;
                return false;
            }
        }
    }
}

template <class Op>
__global__ void __launch_bounds__(kBulkThreads, 2)
fused_bulk_kernel(FusedArgs a)
{
    extern __shared__ __align__(128) uint4 smem[];
    char* base = reinterpret_cast<char*>(smem);
    char* ring = base;                                            // [S][tile]
    char* ybuf = ring + kBulkStages * kBulkTile;                  // [2][tile]
    uint4* slots = reinterpret_cast<uint4*>(ybuf + 2 * kBulkTile);  // [(D+1)][256]
    uint64_t* full = reinterpret_cast<uint64_t*>(base + a.bulk_bar_off);  // after the slots
    uint64_t* empty = full + kBulkStages;
    __shared__ volatile int abort_flag;
    const int tid = threadIdx.x;
    const int p = a.p;

    if (tid == 0) {
        for (int s = 0; s < kBulkStages; s++) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], kBulkConsumers / 32);
        }
        abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        fence_async_shared();
    }
    __syncthreads();

    if (tid >= kBulkConsumers) {
        // ---------------------------------------------------- producer
        if (tid == kBulkConsumers) {
            uint64_t k = 0;
            for (int64_t t = blockIdx.x; t < a.bulk_tiles && !abort_flag; t += gridDim.x) {
                for (int i = 0; i < p; i++, k++) {
                    const int s = int(k % kBulkStages);
                    const uint32_t ph = uint32_t(k / kBulkStages) & 1u;
                    if (!bulk_wait(a, &empty[s], ph ^ 1u, &abort_flag)) break;
                    mbar_expect_tx(&full[s], kBulkTile);
                    bulk_load(ring + s * kBulkTile, rank_ptr(a.x, i) + t * kBulkTile, kBulkTile, &full[s]);
                }
            }
            // every issued load must have landed before the CTA may exit
            const uint64_t issued = k;
            for (uint64_t q = issued > kBulkStages ? issued - kBulkStages : 0; q < issued; q++) {
                const int s = int(q % kBulkStages);
                const uint32_t ph = uint32_t(q / kBulkStages) & 1u;
                const uint64_t t0 = gtime();
                while (!mbar_test(&full[s], ph) && gtime() - t0 < uint64_t(a.wait_ns)) {
                }
            }
        }
        return;
    }

    // -------------------------------------------------------- consumers
    using U = VecUnit<Op>;
    uint4* slot = slots + tid;
    const int warp_lane = tid & 31;
    uint64_t k = 0;
    int buf = 0;
    for (int64_t t = blockIdx.x; t < a.bulk_tiles; t += gridDim.x) {
        uint4 acc = make_uint4(0, 0, 0, 0);
        bool ok = true;
        for (int i = 0; i < p; i++, k++) {
            const int s = int(k % kBulkStages);
            const uint32_t ph = uint32_t(k / kBulkStages) & 1u;
            if (!bulk_wait(a, &full[s], ph, &abort_flag)) { ok = false; break; }
            const uint4 v = reinterpret_cast<const uint4*>(ring + s * kBulkTile)[tid];
            __syncwarp();
            if (warp_lane == 0) mbar_arrive(&empty[s]);
            fold_step<U>(__ldg(a.tape + i), v, acc, slot, kBulkConsumers);
        }
        if (!ok) break;
        const uint4 y = a.dual ? U::op(slot[0], acc) : acc;
        // the stores that last read this result buffer (two tiles ago) must
        // have finished reading it
        if (tid == 0) bulk_wait_read1();
        consumers_sync();
        reinterpret_cast<uint4*>(ybuf + buf * kBulkTile)[tid] = y;
        fence_async_shared();
        consumers_sync();
        if (tid == 0) {
            for (int i = 0; i < p; i++)
                bulk_store(rank_ptr_w(a.y, i) + t * kBulkTile, ybuf + buf * kBulkTile, kBulkTile);
            bulk_commit();
        }
        buf ^= 1;
    }
    if (tid == 0) bulk_wait_all();
    if (abort_flag) return;
    // columns past the last full tile: plain loads, grid-stride
    const int64_t u_first = a.bulk_tiles * (kBulkTile / 16);
    const int64_t stride = int64_t(gridDim.x) * kBulkConsumers;
    for (int64_t u = u_first + int64_t(blockIdx.x) * kBulkConsumers + tid; u < a.nvec; u += stride)
        stream_column<VecUnit<Op>>(a, u, slot, kBulkConsumers);
    for (int64_t e = int64_t(blockIdx.x) * kBulkConsumers + tid; e < a.nscalar; e += stride)
        stream_column<OneUnit<Op>>(a, a.scalar_base + e, one_slots<Op>(slots, tid),
                                   one_slot_stride<Op>(kBulkConsumers));
}


template <class Op>
struct Bulk {
    static int run(Plan* P, FusedArgs a, cudaStream_t s)
    {
        const size_t slots = size_t(P->max_depth + 1) * kBulkConsumers * sizeof(uint4);
        const size_t bar_off = size_t(kBulkStages + 2) * kBulkTile + slots;
        const size_t smem = bar_off + 2 * kBulkStages * sizeof(uint64_t);
        a.bulk_bar_off = int(bar_off);
        if (int rc = grant_smem(reinterpret_cast<const void*>(&fused_bulk_kernel<Op>), smem,
                                &P->smem_attr[3], "fused bulk attribute"))
            return rc;
        int occ = 0;
        cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fused_bulk_kernel<Op>,
                                                                     kBulkThreads, smem);
        if (e != cudaSuccess) return cuda_fail(e, "fused bulk occupancy");
        const int64_t resident = int64_t(std::max(occ, 1)) * P->num_sms;
        const int64_t tail = (a.nvec - a.bulk_tiles * (kBulkTile / 16)) + a.nscalar;
        int64_t grid = std::min<int64_t>(a.bulk_tiles, resident);
        grid = std::max<int64_t>(grid, std::min<int64_t>(resident, (tail + kBulkConsumers - 1) / kBulkConsumers));
        fused_bulk_kernel<Op><<<unsigned(std::max<int64_t>(grid, 1)), kBulkThreads, smem, s>>>(a);
        return launched();
    }
};

}  // namespace

int launch_bulk(Plan* P, FusedArgs a, cudaStream_t s) { return dispatch<Bulk>(P, a, s); }

}  // namespace fused
}  // namespace dpdr
