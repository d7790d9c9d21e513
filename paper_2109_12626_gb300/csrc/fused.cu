// fused.cu -- the fused bandwidth kernel of dpdr_allreduce.
//
// One launch computes y = v(r0) (.) v(r1) with the post-order bracketing of
// Sec. 1.1 (v(i) = v(child_1) (.) (v(child_0) (.) x_i), child_0 = i-1) for
// every element column and stores it to all p outputs.  Every input element
// is read once and every output element written once: 2 p m element
// transfers, the floor for any reduction-to-all whose p inputs and p outputs
// live in device memory.  The tree's pipeline blocks (Algorithm 1) do not
// change the result, so this kernel tiles by columns only.
//
// Two layouts of the same computation:
//  * column streaming: one thread owns one 16-byte column unit and walks the
//    p ranks in post-order, folding them with a register accumulator and a
//    per-depth slot array in shared memory (the running post-order fold:
//    a node's child_0 is the rank just before it and arrives in the
//    accumulator; its child_1 value was parked in slot depth+1).  Eight
//    ranks are loaded ahead of the fold.  Suits m >> p.
//  * shared-memory tile: one CTA loads a tile of WU column units from all p
//    ranks into shared memory with cp.async, evaluates the tree level by
//    level (deepest first; all nodes of a level in parallel), then writes
//    the result row to all p outputs.  Suits small m with large p, where
//    column streaming would leave most SMs idle.
#include <algorithm>

#include "dpdr_internal.h"
#include "ops.cuh"

namespace dpdr {
namespace {

constexpr int kStreamThreads = 256;
constexpr int kStreamAhead = 8;  // ranks loaded ahead (tape read 8 at a time)
constexpr int kTileThreads = 256;
constexpr size_t kTileSmemTarget = 96 * 1024;

struct FusedArgs {
    const char* const* x;   // [p] rank inputs
    char* const* y;         // [p] rank outputs
    const uint8_t* tape;    // [p rounded up to 8]
    const LevelNode* levels;
    const int* level_off;
    int nlevels;
    int p;
    int r0, r1;
    int64_t nvec;           // 16-byte units
    int64_t nscalar;        // single elements after the vector units
    int64_t scalar_base;    // element index of the first single element
    int lg_wu;              // tile: log2 of vector units per row
    int64_t vec_tiles;      // tile: number of vector tiles
    // split layout
    const int2* seg;        // [nseg] (first rank, root rank) of each subtree
    const int2* items;      // [nitems] top fold: (source, tape byte | kind << 8)
    int nitems;
    char* part;             // [nseg] rows of subtree values
    int64_t part_stride;    // bytes per row
    int group;              // ranks stored by one CTA row of the finish kernel
    // bulk layout
    int64_t bulk_tiles;     // full tiles of kBulkTile bytes
    int bulk_bar_off;       // byte offset of the mbarriers in shared memory
    uint32_t* err;          // plan error record (an expired pipeline wait)
    int64_t wait_ns;
};

template <class Op>
struct VecUnit {
    using T = uint4;
    __device__ __forceinline__ static T ld(const char* row, int64_t u)
    {
        return ld_stream(row + u * 16);
    }
    __device__ __forceinline__ static void st(char* row, int64_t u, const T& v)
    {
        st_stream(row + u * 16, v);
    }
    __device__ __forceinline__ static T op(const T& a, const T& b) { return Op::vec(a, b); }
    // data read again soon (subtree values, top-of-tree inputs): keep in L2
    __device__ __forceinline__ static T ld_keep(const char* row, int64_t u)
    {
        return ld_l2(row + u * 16);
    }
    __device__ __forceinline__ static void st_keep(char* row, int64_t u, const T& v)
    {
        st_l2(row + u * 16, v);
    }
};

template <class Op>
struct OneUnit {
    using T = Elem<Op>;
    __device__ __forceinline__ static T ld(const char* row, int64_t e)
    {
        return ld_one_stream<Op>(row + e * Op::kEsize);
    }
    __device__ __forceinline__ static void st(char* row, int64_t e, const T& v)
    {
        st_one_stream<Op>(row + e * Op::kEsize, v);
    }
    __device__ __forceinline__ static T op(const T& a, const T& b) { return comb<Op>(a, b); }
    __device__ __forceinline__ static T ld_keep(const char* row, int64_t e)
    {
        return ld_one_l2<Op>(row + e * Op::kEsize);
    }
    __device__ __forceinline__ static void st_keep(char* row, int64_t e, const T& v)
    {
        st_one_l2<Op>(row + e * Op::kEsize, v);
    }
};

__device__ __forceinline__ const char* rank_ptr(const char* const* t, int i)
{
    return reinterpret_cast<const char*>(__ldg(reinterpret_cast<const unsigned long long*>(t) + i));
}
__device__ __forceinline__ char* rank_ptr_w(char* const* t, int i)
{
    return reinterpret_cast<char*>(__ldg(reinterpret_cast<const unsigned long long*>(t) + i));
}

// ---------------------------------------------------------------- streaming
// One step of the running post-order fold: v is rank i's own value x_i (or,
// in the split layout, a whole subtree's value with no children left); acc
// holds the value of rank i-1, which is child_0 whenever i has a child; a
// child_1 value waits in slot[depth+1]; a node that is a child_1 (or the
// lower root) parks its value in slot[depth].
template <class U>
__device__ __forceinline__ void fold_step(unsigned t, typename U::T v, typename U::T& acc,
                                          typename U::T* slot, int stride)
{
    const unsigned c = t & 3u, d = (t >> 3) & 31u;
    if (c >= 1) v = U::op(acc, v);                     // v(c0) (.) x_i
    if (c == 2) v = U::op(slot[(d + 1) * stride], v);  // v(c1) (.) (..)
    if (t & kTapeKeep) slot[d * stride] = v;
    acc = v;
}

template <class U>
__device__ __forceinline__ void stream_column(const FusedArgs& a, int64_t u,
                                              typename U::T* slot, int stride)
{
    using T = typename U::T;
    const int p = a.p;
    T cur[kStreamAhead], nxt[kStreamAhead];
#pragma unroll
    for (int k = 0; k < kStreamAhead; k++)
        if (k < p) cur[k] = U::ld(rank_ptr(a.x, k), u);
    T acc = cur[0];
    for (int i0 = 0; i0 < p; i0 += kStreamAhead) {
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + kStreamAhead + k < p)
                nxt[k] = U::ld(rank_ptr(a.x, i0 + kStreamAhead + k), u);
        const unsigned long long tp =
            __ldg(reinterpret_cast<const unsigned long long*>(a.tape + i0));
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k < p) fold_step<U>(unsigned(tp >> (8 * k)) & 0xffu, cur[k], acc, slot, stride);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++) cur[k] = nxt[k];
    }
    const T y = (p >= 2) ? U::op(slot[0], acc) : acc;  // v(r0) (.) v(r1)
#pragma unroll 4
    for (int i = 0; i < p; i++) U::st(rank_ptr_w(a.y, i), u, y);
}

template <class Op>
__global__ void __launch_bounds__(kStreamThreads, 3)
fused_stream_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int64_t u = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (u < a.nvec) {
        stream_column<VecUnit<Op>>(a, u, smem + threadIdx.x, blockDim.x);
    } else if (u < a.nvec + a.nscalar) {
        auto* slot = reinterpret_cast<Elem<Op>*>(smem) + threadIdx.x;
        stream_column<OneUnit<Op>>(a, a.scalar_base + (u - a.nvec), slot, blockDim.x);
    }
}

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
    T cur[kStreamAhead], nxt[kStreamAhead];
#pragma unroll
    for (int k = 0; k < kStreamAhead; k++)
        if (lo + k <= hi) cur[k] = U::ld(rank_ptr(a.x, lo + k), u);
    T acc = cur[0];
    for (int i0 = lo; i0 <= hi; i0 += kStreamAhead) {
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + kStreamAhead + k <= hi)
                nxt[k] = U::ld(rank_ptr(a.x, i0 + kStreamAhead + k), u);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k <= hi) fold_step<U>(__ldg(a.tape + i0 + k), cur[k], acc, slot, stride);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++) cur[k] = nxt[k];
    }
    U::st_keep(row, u, acc);
}

template <class U>
__device__ __forceinline__ void split_finish_column(const FusedArgs& a, int r, int64_t u,
                                                    typename U::T* slot, int stride)
{
    using T = typename U::T;
    const int n = a.nitems;
    T cur[kStreamAhead], nxt[kStreamAhead];
    // every item is a scratch row: a subtree value or a copied input, so
    // this kernel never reads an input that another CTA may be overwriting
    // with the result (in-place use)
    auto load = [&](int k) -> T {
        return U::ld_keep(a.part + int64_t(__ldg(&a.items[k].x)) * a.part_stride, u);
    };
#pragma unroll
    for (int k = 0; k < kStreamAhead; k++)
        if (k < n) cur[k] = load(k);
    T acc = cur[0];
    for (int k0 = 0; k0 < n; k0 += kStreamAhead) {
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (k0 + kStreamAhead + k < n) nxt[k] = load(k0 + kStreamAhead + k);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (k0 + k < n)
                fold_step<U>(unsigned(__ldg(&a.items[k0 + k].y)) & 0xffu, cur[k], acc, slot, stride);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++) cur[k] = nxt[k];
    }
    const T y = (a.p >= 2) ? U::op(slot[0], acc) : acc;
    const int i1 = min(a.p, (r + 1) * a.group);
#pragma unroll 4
    for (int i = r * a.group; i < i1; i++) U::st(rank_ptr_w(a.y, i), u, y);
}

template <class Op>
__global__ void __launch_bounds__(kStreamThreads, 3)
fused_split_reduce_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int64_t u = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (u < a.nvec) {
        split_reduce_column<VecUnit<Op>>(a, blockIdx.y, u, smem + threadIdx.x, blockDim.x);
    } else if (u < a.nvec + a.nscalar) {
        auto* slot = reinterpret_cast<Elem<Op>*>(smem) + threadIdx.x;
        split_reduce_column<OneUnit<Op>>(a, blockIdx.y, a.scalar_base + (u - a.nvec), slot,
                                         blockDim.x);
    }
}

template <class Op>
__global__ void __launch_bounds__(kStreamThreads, 3)
fused_split_finish_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int64_t u = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (u < a.nvec) {
        split_finish_column<VecUnit<Op>>(a, blockIdx.y, u, smem + threadIdx.x, blockDim.x);
    } else if (u < a.nvec + a.nscalar) {
        auto* slot = reinterpret_cast<Elem<Op>*>(smem) + threadIdx.x;
        split_finish_column<OneUnit<Op>>(a, blockIdx.y, a.scalar_base + (u - a.nvec), slot,
                                         blockDim.x);
    }
}

// --------------------------------------------------------------------- tile
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem)
{
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem)
{
    const unsigned s = static_cast<unsigned>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(s), "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async_wait_all()
{
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;\n" ::: "memory");
}

// rows of WU units: row i < p holds rank i's tile, row p the result.
// kVec: 16-byte units copied with 16-byte cp.async; otherwise single
// elements copied word by word with 4-byte cp.async.
template <class U, bool kVec, class Op>
__device__ __forceinline__ void tile_body(const FusedArgs& a, int64_t u0,
                                          int wu, int lg_wu, typename U::T* tile)
{
    using T = typename U::T;
    const int p = a.p, tid = threadIdx.x, bd = blockDim.x;
    const int WU = 1 << lg_wu;
    const int n = p << lg_wu;
    for (int idx = tid; idx < n; idx += bd) {
        const int i = idx >> lg_wu, c = idx & (WU - 1);
        if (c < wu) {
            if constexpr (kVec) {
                cp_async16(&tile[idx], rank_ptr(a.x, i) + (u0 + c) * 16);
            } else {
                const char* src = rank_ptr(a.x, i) + (u0 + c) * Op::kEsize;
                uint32_t* dst = reinterpret_cast<uint32_t*>(&tile[idx]);
#pragma unroll
                for (int w = 0; w < Op::kEsize / 4; w++) cp_async4(dst + w, src + 4 * w);
            }
        }
    }
    cp_async_wait_all();
    __syncthreads();
    for (int l = 0; l < a.nlevels; l++) {
        const int beg = __ldg(a.level_off + l), end = __ldg(a.level_off + l + 1);
        const int cnt = (end - beg) << lg_wu;
        for (int idx = tid; idx < cnt; idx += bd) {
            const int k = idx >> lg_wu, c = idx & (WU - 1);
            if (c >= wu) continue;
            const int node = __ldg(&a.levels[beg + k].node);
            const int c1 = __ldg(&a.levels[beg + k].child1);
            T v = U::op(tile[((node - 1) << lg_wu) + c], tile[(node << lg_wu) + c]);
            if (c1 >= 0) v = U::op(tile[(c1 << lg_wu) + c], v);
            tile[(node << lg_wu) + c] = v;
        }
        __syncthreads();
    }
    for (int c = tid; c < wu; c += bd) {
        const T v1 = tile[(a.r1 << lg_wu) + c];
        tile[(p << lg_wu) + c] = (p >= 2) ? U::op(tile[(a.r0 << lg_wu) + c], v1) : v1;
    }
    __syncthreads();
    for (int idx = tid; idx < n; idx += bd) {
        const int i = idx >> lg_wu, c = idx & (WU - 1);
        if (c < wu) U::st(rank_ptr_w(a.y, i), u0 + c, tile[(p << lg_wu) + c]);
    }
}

// smallest power-of-two exponent with 2^lg >= w
__device__ __forceinline__ int ceil_lg(int w)
{
    int lg = 0;
    while ((1 << lg) < w) lg++;
    return lg;
}

template <class Op>
__global__ void __launch_bounds__(kTileThreads)
fused_tile_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int64_t t = blockIdx.x;
    // a narrow last tile (small m) is packed with a row stride of its own
    // width, so no thread walks empty columns
    if (t < a.vec_tiles) {
        const int64_t u0 = t << a.lg_wu;
        const int wu = int(lmin(int64_t(1) << a.lg_wu, a.nvec - u0));
        tile_body<VecUnit<Op>, true, Op>(a, u0, wu, ceil_lg(wu), smem);
    } else {
        // single elements: a row of a tile holds as many bytes as in the
        // vector tiles, i.e. 16/esize times more units
        const int lg = a.lg_wu + (Op::kEsize == 4 ? 2 : 0);
        const int64_t e0 = (t - a.vec_tiles) << lg;
        const int wu = int(lmin(int64_t(1) << lg, a.nscalar - e0));
        tile_body<OneUnit<Op>, false, Op>(a, a.scalar_base + e0, wu, ceil_lg(wu),
                                          reinterpret_cast<Elem<Op>*>(smem));
    }
}

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
constexpr int kBulkConsumers = 256;                   // 8 warps
constexpr int kBulkThreads = kBulkConsumers + 32;     // + producer warp
constexpr int kBulkTile = kBulkConsumers * 16;        // bytes per rank row piece
constexpr int kBulkStages = 16;

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
        const uint4 y = (p >= 2) ? U::op(slot[0], acc) : acc;
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
        stream_column<OneUnit<Op>>(a, a.scalar_base + e, reinterpret_cast<Elem<Op>*>(slots) + tid,
                                   kBulkConsumers);
}

// --------------------------------------------------------------------- host
template <class Op>
int launch(Plan* P, FusedArgs a, int mode, cudaStream_t s)
{
    if (mode == 1) {
        const int64_t units = a.nvec + a.nscalar;
        const int64_t blocks = (units + kStreamThreads - 1) / kStreamThreads;
        const size_t smem = size_t(P->max_depth + 1) * kStreamThreads * sizeof(uint4);
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        if (int(smem) > P->smem_attr[0]) {
            cudaError_t e = cudaFuncSetAttribute(fused_stream_kernel<Op>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 int(smem));
            if (e != cudaSuccess) return cuda_fail(e, "fused stream attribute");
            P->smem_attr[0] = int(smem);
        }
        fused_stream_kernel<Op><<<unsigned(blocks), kStreamThreads, smem, s>>>(a);
    } else if (mode == 4) {
        const size_t slots = size_t(P->max_depth + 1) * kBulkConsumers * sizeof(uint4);
        const size_t bar_off = size_t(kBulkStages + 2) * kBulkTile + slots;
        const size_t smem = bar_off + 2 * kBulkStages * sizeof(uint64_t);
        a.bulk_bar_off = int(bar_off);
        if (int(smem) > P->smem_attr[3]) {
            cudaError_t e = cudaFuncSetAttribute(fused_bulk_kernel<Op>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 int(smem));
            if (e != cudaSuccess) return cuda_fail(e, "fused bulk attribute");
            P->smem_attr[3] = int(smem);
        }
        int occ = 0;
        cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, fused_bulk_kernel<Op>,
                                                                     kBulkThreads, smem);
        if (e != cudaSuccess) return cuda_fail(e, "fused bulk occupancy");
        const int64_t resident = int64_t(std::max(occ, 1)) * P->num_sms;
        const int64_t tail = (a.nvec - a.bulk_tiles * (kBulkTile / 16)) + a.nscalar;
        int64_t grid = std::min<int64_t>(a.bulk_tiles, resident);
        grid = std::max<int64_t>(grid, std::min<int64_t>(resident, (tail + kBulkConsumers - 1) / kBulkConsumers));
        fused_bulk_kernel<Op><<<unsigned(std::max<int64_t>(grid, 1)), kBulkThreads, smem, s>>>(a);
    } else if (mode == 3) {
        const int64_t units = a.nvec + a.nscalar;
        const int64_t blocks = (units + kStreamThreads - 1) / kStreamThreads;
        const size_t smem = size_t(P->max_depth + 1) * kStreamThreads * sizeof(uint4);
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        if (int(smem) > P->smem_attr[2]) {
            cudaError_t e = cudaFuncSetAttribute(fused_split_reduce_kernel<Op>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 int(smem));
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(fused_split_finish_kernel<Op>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
            if (e != cudaSuccess) return cuda_fail(e, "fused split attribute");
            P->smem_attr[2] = int(smem);
        }
        const int groups = (P->p + a.group - 1) / a.group;
        fused_split_reduce_kernel<Op>
            <<<dim3(unsigned(blocks), unsigned(P->split_nseg)), kStreamThreads, smem, s>>>(a);
        fused_split_finish_kernel<Op>
            <<<dim3(unsigned(blocks), unsigned(groups)), kStreamThreads, smem, s>>>(a);
    } else {
        const size_t smem = size_t(P->p + 1) * (size_t(16) << a.lg_wu);
        const int64_t lg_s = a.lg_wu + (Op::kEsize == 4 ? 2 : 0);
        const int64_t scal_tiles = (a.nscalar + (int64_t(1) << lg_s) - 1) >> lg_s;
        const int64_t blocks = a.vec_tiles + scal_tiles;
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        if (int(smem) > P->smem_attr[1]) {
            cudaError_t e = cudaFuncSetAttribute(fused_tile_kernel<Op>,
                                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 int(smem));
            if (e != cudaSuccess) return cuda_fail(e, "fused tile attribute");
            P->smem_attr[1] = int(smem);
        }
        fused_tile_kernel<Op><<<unsigned(blocks), kTileThreads, smem, s>>>(a);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "fused kernel launch");
    return DPDR_OK;
}

// largest power-of-two vector units per tile row that fits the smem target
int tile_lg_wu(const Plan* P)
{
    const size_t row = size_t(P->p + 1) * 16;
    if (row > 200 * 1024) return -1;  // not even one unit per row fits
    int lg = 0;
    while (lg < 6 && row * (size_t(2) << lg) <= kTileSmemTarget) lg++;
    return lg;
}

}  // namespace

// Threads the streaming layouts want in flight to cover HBM latency.
static int64_t stream_target(const Plan* P) { return int64_t(P->num_sms) * 1024; }

// Layout choice, from measurements on GB300:
//  * deep trees (p >= 128) with at least 8192 column units: the split layout,
//    whose read phase (first kernel) and write phase (second kernel) keep
//    HBM traffic one-directional; it beats column streaming from m = 2^15 up
//    to the largest sizes at p = 1152;
//  * otherwise column streaming once there are enough columns to fill the
//    GPU, and the shared-memory tile below that.
int fused_auto_mode(const Plan* P)
{
    const int64_t units = P->m * int64_t(P->esize) / 16;
    if (P->p >= 128 && units >= 8192 && P->split_ready) return 3;
    if (units >= stream_target(P)) return 1;
    if (tile_lg_wu(P) >= 0) return 2;
    return P->split_ready ? 3 : 1;
}

// Whether the automatic choice can be the split layout (then the plan
// prepares it up front).
static bool split_wanted(const Plan* P)
{
    const int64_t units = P->m * int64_t(P->esize) / 16;
    return P->p >= 128 && units >= 8192;
}

// Split layout: cut depth s, subtree table, top-of-tree item list, rank
// groups of the finish kernel, and the scratch rows of subtree values.
// depth < 0 picks the shallowest cut that gives the first kernel enough
// independent (subtree, column) work to fill the GPU.
int fused_split_prepare(Plan* P, bool force, int depth)
{
    const int p = P->p;
    if (p < 2) return DPDR_OK;  // one rank: nothing to split
    const int64_t units = std::max<int64_t>(1, P->m * int64_t(P->esize) / 16);
    const int64_t target = stream_target(P);
    // automatic cut: the shallowest depth whose subtrees give the first
    // kernel four times the columns the GPU needs in flight, but no deeper
    // than a third of the tree height (the second kernel's sequential walk
    // over the nodes above the cut grows as 2^(s+1))
    int s = depth;
    if (s < 0) {
        const int cap = std::max(1, P->max_depth / 3);
        for (s = 0; s < cap; s++) {
            int64_t n = 0;
            for (int i = 0; i < p; i++) n += P->depth[i] == s;
            if (n * units >= 4 * target) break;
        }
    }
    s = std::min(s, P->max_depth);
    if (P->split_ready && P->split_s == s) return DPDR_OK;
    if (!force && !split_wanted(P)) return DPDR_OK;
    // scratch rows: one per depth-s subtree (first rank, root), one per node
    // above the cut (its own input, first = root); items in post-order
    std::vector<int2> seg, items;
    for (int i = 0; i < p; i++) {
        if (P->depth[i] > s) continue;
        int lo = i;
        if (P->depth[i] == s)  // leftmost leaf of the subtree
            while (P->child0[lo] >= 0) lo = P->child1[lo] >= 0 ? P->child1[lo] : P->child0[lo];
        const unsigned t = P->depth[i] == s ? (P->tape[i] & ~3u) : P->tape[i];
        items.push_back(make_int2(int(seg.size()), int(t)));
        seg.push_back(make_int2(lo, i));
    }
    if (P->d_split) {
        cudaFree(P->d_split);
        P->d_split = nullptr;
        P->d_split_bytes = 0;
        P->split_ready = false;
    }
    int64_t groups = std::min<int64_t>(p, std::max<int64_t>(1, (target + units - 1) / units));
    P->split_group = int((p + groups - 1) / groups);
    P->split_s = s;
    P->split_nseg = int(seg.size());
    P->split_nitems = int(items.size());
    P->part_stride = int64_t((size_t(P->m) * P->esize + 255) / 256 * 256);
    const size_t o_items = (sizeof(int2) * seg.size() + 255) / 256 * 256;
    const size_t o_part = o_items + (sizeof(int2) * items.size() + 255) / 256 * 256;
    const size_t bytes = o_part + size_t(P->part_stride) * seg.size();
    cudaError_t e = cudaMalloc(&P->d_split, bytes);
    if (e != cudaSuccess) {
        P->d_split = nullptr;
        P->split_nseg = 0;
        return cuda_fail(e, "split layout: cudaMalloc");
    }
    P->d_split_bytes = bytes;
    P->d_seg = reinterpret_cast<int2*>(P->d_split);
    P->d_items = reinterpret_cast<int2*>(P->d_split + o_items);
    P->d_part = P->d_split + o_part;
    e = cudaMemcpy(P->d_seg, seg.data(), sizeof(int2) * seg.size(), cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
        e = cudaMemcpy(P->d_items, items.data(), sizeof(int2) * items.size(),
                       cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "split layout: upload");
    P->split_ready = true;
    return DPDR_OK;
}

int fused_launch(Plan* P, cudaStream_t s)
{
    return fused_launch_cols(P, P->d_x, P->d_y, P->m, P->last_vector_path != 0, s);
}

// The fused kernel on mc columns, with device tables of rank pointers that
// may point into the middle of the rank buffers (a column chunk).
int fused_launch_cols(Plan* P, const char* const* dx, char* const* dy, int64_t mc, bool vec,
                      cudaStream_t s)
{
    if (mc == 0) return DPDR_OK;
    int mode = P->fused_mode ? P->fused_mode : fused_auto_mode(P);
    const int lg = tile_lg_wu(P);
    if (mode == 2 && lg < 0) return fail(DPDR_ERR_INVALID, "tile mode: p too large");
    if (mode == 3 && !P->split_ready) return fail(DPDR_ERR_INVALID, "split mode: p < 2");
    if (mode < 1 || mode > 4) return fail(DPDR_ERR_INVALID, "unknown fused mode");

    FusedArgs a;
    a.x = dx;
    a.y = dy;
    a.tape = P->d_tape;
    a.levels = P->d_levels;
    a.level_off = P->d_level_off;
    a.nlevels = int(P->level_off.size()) - 1;
    a.p = P->p;
    a.r0 = P->r0;
    a.r1 = P->r1;
    const int epv = int(16 / P->esize);
    a.nvec = vec ? mc / epv : 0;
    a.scalar_base = a.nvec * epv;
    a.nscalar = mc - a.scalar_base;
    a.lg_wu = lg < 0 ? 0 : lg;
    a.vec_tiles = (a.nvec + (int64_t(1) << a.lg_wu) - 1) >> a.lg_wu;
    a.seg = P->d_seg;
    a.items = P->d_items;
    a.nitems = P->split_nitems;
    a.part = P->d_part;
    a.part_stride = P->part_stride;
    a.group = P->split_group;
    a.bulk_tiles = vec ? (a.nvec * 16) / kBulkTile : 0;
    a.bulk_bar_off = 0;
    a.err = P->d_err;
    a.wait_ns = P->wait_ns;
    if (mode == 4 && !vec) mode = 1;  // bulk copies need 16-byte aligned rows

    switch (P->dtype) {
    case DPDR_INT32: return launch<SumI32>(P, a, mode, s);
    case DPDR_FLOAT32: return launch<SumF32>(P, a, mode, s);
    default: return launch<MatU32>(P, a, mode, s);
    }
}

}  // namespace dpdr
