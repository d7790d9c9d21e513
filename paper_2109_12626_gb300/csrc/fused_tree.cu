// fused_tree.cu -- hierarchical tile layout of the fused kernel: one CTA per
// tile of W column units (8 or 16) runs the whole fold of its columns.
//
//  1. The tree is cut at depth s (Sec. 1.1's trees are complete, so a
//     depth-s node roots a contiguous post-order interval of ranks).  Each
//     thread walks one depth-s subtree for one column with the running
//     post-order fold (loads kStreamAhead ranks ahead) and leaves the
//     subtree's value in shared memory; the inputs of the nodes above the
//     cut are loaded there too.
//  2. The nodes above the cut are evaluated level by level, deepest first,
//     v(i) = v(child_1) (.) (v(child_0) (.) x_i), all nodes of a level in
//     parallel; then y = v(r0) (.) v(r1) (or v(root) for one tree).
//  3. All threads store y to the p outputs.
//
// One kernel, no scratch rows in device memory, and every thread has a walk
// of about p / 2^(s+1) ranks: the layout for large p at mid m, where the
// column-streaming walk over all p ranks is too long and the subtree-split
// layout pays for a second kernel and a top fold per store group.  A CTA
// reads all p rows of its columns before it writes any (barrier between
// phases 1 and 3), and no other CTA touches those columns, so in-place use
// is safe.  Buffers that are not all 16-byte aligned go to the
// shared-memory tile (fused.cu); a ragged tail of single elements (fewer
// than 16 bytes per rank) gets one extra CTA that runs the same three
// phases on them.
#include <algorithm>
#include <vector>

#include "fused_common.cuh"

namespace dpdr {
namespace fused {
namespace {

// Walk of the subtree [lo, hi] (post-order interval, hi its root) at depth
// s for unit u: the running fold of fold_step with depths taken relative to
// s, so the slots hold depths s .. max depth.
template <class U>
__device__ __forceinline__ typename U::T walk_subtree(const FusedArgs& a, int lo, int hi,
                                                      int64_t u, typename U::T* slot,
                                                      int stride, int s)
{
    using T = typename U::T;
    const unsigned shift = unsigned(s) << 3;  // tape depth field starts at bit 3
    T acc{};  // set by rank lo, a leaf
    for (int i0 = lo; i0 <= hi; i0 += kStreamAhead) {
        T cur[kStreamAhead];
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k <= hi) cur[k] = U::ld(rank_ptr(a.x, i0 + k), u);
#pragma unroll
        for (int k = 0; k < kStreamAhead; k++)
            if (i0 + k <= hi)
                fold_step<U>(unsigned(__ldg(a.tape + i0 + k)) - shift, cur[k], acc, slot, stride);
    }
    return acc;
}

// The three phases for wu <= W units starting at u0 (16-byte units with
// VecUnit, single elements with OneUnit); slot/stride are this thread's
// walk slots.
template <class U, int W>
__device__ __forceinline__ void tree_body(const FusedArgs& a, int64_t u0, int wu, uint4* smem,
                                          typename U::T* slot, int stride)
{
    using T = typename U::T;
    const int tid = threadIdx.x;
    T* part = reinterpret_cast<T*>(smem + a.tree_slots * kTreeThreads);  // [nseg][W]
    T* yrow = part + a.tree_nseg * W;                                      // [W]

    // 1. subtree walks and the inputs above the cut
    const int npairs = a.tree_nseg * W;
    for (int idx = tid; idx < npairs; idx += kTreeThreads) {
        const int g = idx / W, c = idx % W;
        if (c >= wu) continue;
        const int2 sg = __ldg(a.tree_seg + g);
        const int64_t u = u0 + c;
        part[idx] = sg.x == sg.y ? U::ld(rank_ptr(a.x, sg.x), u)
                                 : walk_subtree<U>(a, sg.x, sg.y, u, slot, stride, a.tree_s);
    }
    __syncthreads();
    // 2. the nodes above the cut, deepest level first
    for (int l = 0; l < a.tree_nlev; l++) {
        const int beg = __ldg(a.tree_levoff + l), end = __ldg(a.tree_levoff + l + 1);
        const int cnt = (end - beg) * W;
        for (int idx = tid; idx < cnt; idx += kTreeThreads) {
            const int k = idx / W, c = idx % W;
            if (c >= wu) continue;
            const int4 e = __ldg(a.tree_lev + beg + k);  // node, child_0, child_1
            T v = part[e.x * W + c];
            if (e.y >= 0) v = U::op(part[e.y * W + c], v);
            if (e.z >= 0) v = U::op(part[e.z * W + c], v);
            part[e.x * W + c] = v;
        }
        __syncthreads();
    }
    if (tid < wu) {
        const T v1 = part[a.tree_r1 * W + tid];
        yrow[tid] = a.dual ? U::op(part[a.tree_r0 * W + tid], v1) : v1;
    }
    __syncthreads();
    // 3. the result to every output
    const int nst = a.p * W;
#pragma unroll 4
    for (int idx = tid; idx < nst; idx += kTreeThreads) {
        const int i = idx / W, c = idx % W;
        if (c < wu) U::st(rank_ptr_w(a.y, i), u0 + c, yrow[c]);
    }
}

// W column units per CTA: kTreeUnitsNarrow for few columns (more CTAs),
// kTreeUnitsWide for more (longer rows per rank, half the CTAs).
template <class Op, int W>
__global__ void __launch_bounds__(kTreeThreads, 2)
fused_tree_kernel(FusedArgs a)
{
    extern __shared__ uint4 smem[];
    const int tid = threadIdx.x;
    if (blockIdx.x < a.tree_tiles) {
        const int64_t u0 = int64_t(blockIdx.x) * W;
        tree_body<VecUnit<Op>, W>(a, u0, int(lmin(W, a.nvec - u0)), smem, smem + tid,
                                  kTreeThreads);
    } else {  // ragged tail: the single elements after the 16-byte units
        tree_body<OneUnit<Op>, W>(a, a.scalar_base, int(a.nscalar), smem,
                                  one_slots<Op>(smem, tid), one_slot_stride<Op>(kTreeThreads));
    }
}

size_t tree_smem(const FusedArgs& a)
{
    return (size_t(a.tree_slots) * kTreeThreads + size_t(a.tree_nseg) * a.tree_width +
            a.tree_width) * sizeof(uint4);
}

template <class Op>
struct Tree {
    static int run(Plan* P, FusedArgs a, cudaStream_t s)
    {
        const size_t smem = tree_smem(a);
        const int64_t blocks = a.tree_tiles + (a.nscalar ? 1 : 0);
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        const bool wide = a.tree_width == kTreeUnitsWide;
        const void* kern = wide ? reinterpret_cast<const void*>(&fused_tree_kernel<Op, kTreeUnitsWide>)
                                : reinterpret_cast<const void*>(&fused_tree_kernel<Op, kTreeUnitsNarrow>);
        if (int rc = grant_smem(kern, smem, &P->smem_attr[wide ? 5 : 4], "fused tree attribute"))
            return rc;
        if (wide)
            fused_tree_kernel<Op, kTreeUnitsWide><<<unsigned(blocks), kTreeThreads, smem, s>>>(a);
        else
            fused_tree_kernel<Op, kTreeUnitsNarrow><<<unsigned(blocks), kTreeThreads, smem, s>>>(a);
        return launched();
    }
};

}  // namespace

int launch_tree(Plan* P, FusedArgs a, cudaStream_t s) { return dispatch<Tree>(P, a, s); }

}  // namespace fused

// The tile width of the device path: kTreeUnitsNarrow column units per CTA
// while those CTAs fit in one wave of resident CTAs, else kTreeUnitsWide,
// whose CTAs cost about 1.6 times as much but are half as many (p = 1152,
// int32, cold L2: m = 2^13, one narrow wave: 22.2 against 24.6 us; m = 10240,
// two narrow waves against one wide: 38.8 against 28.9 us; m = 2^15, four
// against two: 81.5 against 63.6 us; from p = 256 to 2304 alike).  The
// host-buffer path always takes the narrow tile: over the host link, more
// CTAs drifting out of phase keep both directions busier (p = 1152,
// m = 2^20: 297 against 272 GB/s).
int fused_tree_index(const Plan* P)
{
    const int64_t units = P->m * int64_t(P->esize) / 16;
    const int64_t slots = int64_t(fused::kTreeCtasPerSm) * P->num_sms;
    return units > fused::kTreeUnitsNarrow * slots ? 1 : 0;
}

// Tables of the hierarchical tile layout for tile width W: the cut depth s
// (about kTreeThreads / W subtrees, one walk per thread), the entries --
// first the depth-s nodes with their subtree intervals, then the nodes above
// the cut (lo = hi = the node) -- and, per level above the cut, deepest
// first, (node, child_0, child_1) as entry indices.
static int tree_tables(Plan* P, int W, TreeTables* T)
{
    if (T->ready) return DPDR_OK;
    const int p = P->p;
    const int trees = P->r0 >= 0 ? 2 : 1;
    int s = 0;
    while (trees << s < fused::kTreeThreads / W) s++;
    s = std::min(s, P->max_depth);
    std::vector<int> idx(p, -1);
    std::vector<int2> seg;
    for (int i = 0; i < p; i++) {
        if (P->depth[i] != s) continue;
        int lo = i;  // leftmost leaf of the subtree
        while (P->child0[lo] >= 0) lo = P->child1[lo] >= 0 ? P->child1[lo] : P->child0[lo];
        idx[i] = int(seg.size());
        seg.push_back(make_int2(lo, i));
    }
    for (int i = 0; i < p; i++) {
        if (P->depth[i] >= s) continue;
        idx[i] = int(seg.size());
        seg.push_back(make_int2(i, i));
    }
    std::vector<int4> lev;
    std::vector<int> off(1, 0);
    for (int d = s - 1; d >= 0; d--) {
        for (int i = 0; i < p; i++) {
            if (P->depth[i] != d) continue;
            const int c0 = P->child0[i], c1 = P->child1[i];
            lev.push_back(make_int4(idx[i], c0 >= 0 ? idx[c0] : -1, c1 >= 0 ? idx[c1] : -1, 0));
        }
        off.push_back(int(lev.size()));
    }
    const size_t o_lev = (sizeof(int2) * seg.size() + 255) / 256 * 256;
    const size_t o_off = o_lev + (sizeof(int4) * std::max<size_t>(lev.size(), 1) + 255) / 256 * 256;
    const size_t bytes = o_off + sizeof(int) * off.size();
    char* d = nullptr;
    cudaError_t e = cudaMalloc(&d, bytes);
    if (e != cudaSuccess) return cuda_fail(e, "tree layout: cudaMalloc");
    e = cudaMemcpy(d, seg.data(), sizeof(int2) * seg.size(), cudaMemcpyHostToDevice);
    if (e == cudaSuccess && !lev.empty())
        e = cudaMemcpy(d + o_lev, lev.data(), sizeof(int4) * lev.size(), cudaMemcpyHostToDevice);
    if (e == cudaSuccess)
        e = cudaMemcpy(d + o_off, off.data(), sizeof(int) * off.size(), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        cudaFree(d);
        return cuda_fail(e, "tree layout: upload");
    }
    T->d = d;
    T->bytes = bytes;
    T->seg = reinterpret_cast<int2*>(d);
    T->lev = reinterpret_cast<int4*>(d + o_lev);
    T->levoff = reinterpret_cast<int*>(d + o_off);
    T->s = s;
    T->nseg = int(seg.size());
    T->nlev = int(off.size()) - 1;
    T->slots = P->max_depth - s + 1;
    T->r0 = P->r0 >= 0 ? idx[P->r0] : -1;
    T->r1 = idx[P->r1];
    T->width = W;
    T->ready = true;
    return DPDR_OK;
}

int fused_tree_prepare(Plan* P)
{
    int rc = tree_tables(P, fused::kTreeUnitsNarrow, &P->tree[0]);
    return rc ? rc : tree_tables(P, fused::kTreeUnitsWide, &P->tree[1]);
}

}  // namespace dpdr
