// fused_common.cuh -- shared pieces of the fused bandwidth kernel
// (dpdr_allreduce): its launch arguments, the 16-byte and single-element
// memory units, and the running post-order fold every layout uses.
//
// The fused kernel computes y = v(r0) (.) v(r1) with the post-order
// bracketing of Sec. 1.1 (v(i) = v(child_1) (.) (v(child_0) (.) x_i),
// child_0 = i-1) for every element column and stores it to all p outputs.
// Every input element is read once and every output element written once:
// 2 p m element transfers, the floor for any reduction-to-all whose p inputs
// and p outputs live in device memory.  The tree's pipeline blocks
// (Algorithm 1) do not change the result, so the kernel tiles by columns.
// Layouts (one file each): column streaming (fused_stream.cu),
// shared-memory tile (fused_tile.cu), subtree split (fused_split.cu),
// bulk-copy pipeline (fused_bulk.cu), hierarchical tile (fused_tree.cu);
// fused.cu chooses and launches.
#pragma once

#include <algorithm>

#include "dpdr_internal.h"
#include "ops.cuh"

namespace dpdr {
namespace fused {

constexpr int kStreamThreads = 256;
constexpr int kStreamAhead = 8;  // ranks loaded ahead (tape read 8 at a time)
constexpr int kTileThreads = 256;
constexpr size_t kTileSmemTarget = 96 * 1024;
constexpr int kBulkConsumers = 256;                   // 8 warps
constexpr int kBulkThreads = kBulkConsumers + 32;     // + producer warp
constexpr int kBulkTile = kBulkConsumers * 16;        // bytes per rank row piece
constexpr int kBulkStages = 16;
constexpr int kTreeThreads = 512;                     // hierarchical tile: threads per CTA,
constexpr int kTreeUnitsNarrow = 8;                   // 16-byte column units per CTA:
constexpr int kTreeUnitsWide = 16;                    // the two tile widths
constexpr int kTreeCtasPerSm = 2;                     // resident (registers, shared memory)

struct FusedArgs {
    const char* const* x;   // [p] rank inputs
    char* const* y;         // [p] rank outputs
    const uint8_t* tape;    // [p rounded up to 8]
    const LevelNode* levels;
    const int* level_off;
    int nlevels;
    int p;
    int r0, r1;
    int dual;               // 1: y = v(r0) (.) v(r1); 0: one tree, y = v(p-1)
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
    // hierarchical tile layout
    const int2* tree_seg;   // [tree_nseg] subtree intervals, then nodes above the cut
    const int4* tree_lev;   // levels above the cut: (node, child_0, child_1) entries
    const int* tree_levoff; // [tree_nlev + 1]
    int tree_nseg, tree_nlev, tree_r0, tree_r1, tree_s, tree_slots;
    int64_t tree_tiles;     // CTAs of tree_width vector units
    int tree_width;         // kTreeUnitsNarrow or kTreeUnitsWide
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
    T acc{};  // set by rank 0, a leaf
    // one batch of kStreamAhead loads in flight per thread; the other warps
    // of the four CTAs per SM cover the latency between batches
    for (int i0 = 0; i0 < p; i0 += kStreamAhead) {
        T cur[kStreamAhead];
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k < p) cur[k] = U::ld(rank_ptr(a.x, i0 + k), u);
        const unsigned long long tp =
            __ldg(reinterpret_cast<const unsigned long long*>(a.tape + i0));
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k < p) fold_step<U>(unsigned(tp >> (8 * k)) & 0xffu, cur[k], acc, slot, stride);
    }
    const T y = a.dual ? U::op(slot[0], acc) : acc;  // v(r0) (.) v(r1), or v(root)
#pragma unroll 4
    for (int i = 0; i < p; i++) U::st(rank_ptr_w(a.y, i), u, y);
}

// The depth slots of thread t sit in 16-byte cells t, t + n, t + 2n, ... of
// a [depth][n] array of uint4 (n threads).  A thread folding single elements
// keeps its slots in the same cells (an element is at most 16 bytes), so its
// slots never overlap another thread's, whatever unit each thread folds.
template <class Op>
__device__ __forceinline__ Elem<Op>* one_slots(uint4* cells, int t)
{
    return reinterpret_cast<Elem<Op>*>(cells + t);
}
template <class Op>
__device__ __forceinline__ int one_slot_stride(int n)
{
    return n * int(sizeof(uint4) / sizeof(Elem<Op>));
}

// launchers, one per layout (dispatch on the plan's element type)
// Raise kernel fn's dynamic shared memory limit on the current device to at
// least `bytes`, never lowering it: the attribute belongs to the function and
// is shared by every plan, so a plan that needs less must not take it away
// from one that needs more.  *granted is the plan's cache of what it already
// has (launches that fit skip the call).
int grant_smem(const void* fn, size_t bytes, int* granted, const char* what);

int launch_stream(Plan* P, FusedArgs a, cudaStream_t s);
int launch_tile(Plan* P, FusedArgs a, cudaStream_t s);
int launch_split(Plan* P, FusedArgs a, cudaStream_t s);
int launch_bulk(Plan* P, FusedArgs a, cudaStream_t s);
int launch_tree(Plan* P, FusedArgs a, cudaStream_t s);
int tile_lg_wu(const Plan* P);

template <template <class> class L>
int dispatch(Plan* P, FusedArgs a, cudaStream_t s)
{
    switch (P->dtype) {
    case DPDR_INT32: return L<SumI32>::run(P, a, s);
    case DPDR_FLOAT32: return L<SumF32>::run(P, a, s);
    case DPDR_MAT2X2_F32: return L<MatF32>::run(P, a, s);
    default: return L<MatU32>::run(P, a, s);
    }
}

inline int launched()
{
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "fused kernel launch");
    return DPDR_OK;
}

}  // namespace fused
}  // namespace dpdr
