// fused_tile.cu -- shared-memory tile layout of the fused kernel: one CTA
// copies a tile of column units from all p ranks into shared memory with
// cp.async, evaluates the tree level by level (deepest first, all nodes of a
// level in parallel), then writes the result row to all p outputs.  Suits
// small m with large p, where column streaming would leave SMs idle.
#include "fused_common.cuh"

namespace dpdr {
namespace fused {
namespace {

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
        tile[(p << lg_wu) + c] = a.dual ? U::op(tile[(a.r0 << lg_wu) + c], v1) : v1;
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


template <class Op>
struct Tile {
    static int run(Plan* P, FusedArgs a, cudaStream_t s)
    {
        const size_t smem = size_t(P->p + 1) * (size_t(16) << a.lg_wu);
        const int64_t lg_s = a.lg_wu + (Op::kEsize == 4 ? 2 : 0);
        const int64_t scal_tiles = (a.nscalar + (int64_t(1) << lg_s) - 1) >> lg_s;
        const int64_t blocks = a.vec_tiles + scal_tiles;
        if (blocks > 0x7fffffff) return fail(DPDR_ERR_INVALID, "m too large");
        if (int rc = grant_smem(reinterpret_cast<const void*>(&fused_tile_kernel<Op>), smem,
                                &P->smem_attr[1], "fused tile attribute"))
            return rc;
        fused_tile_kernel<Op><<<unsigned(blocks), kTileThreads, smem, s>>>(a);
        return launched();
    }
};

}  // namespace

int launch_tile(Plan* P, FusedArgs a, cudaStream_t s) { return dispatch<Tile>(P, a, s); }

// largest power-of-two vector units per tile row that fits the smem target
int tile_lg_wu(const Plan* P)
{
    const size_t row = size_t(P->p + 1) * 16;
    if (row > 200 * 1024) return -1;  // not even one unit per row fits
    int lg = 0;
    while (lg < 6 && row * (size_t(2) << lg) <= kTileSmemTarget) lg++;
    return lg;
}

}  // namespace fused
}  // namespace dpdr
