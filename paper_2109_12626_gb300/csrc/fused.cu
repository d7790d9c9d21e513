// fused.cu -- layout choice and launch of the fused bandwidth kernel
// (dpdr_allreduce); the layouts themselves live in fused_stream.cu,
// fused_tile.cu, fused_split.cu, fused_bulk.cu and fused_tree.cu (see
// fused_common.cuh).
#include <algorithm>
#include <map>
#include <mutex>
#include <utility>

#include "fused_common.cuh"

namespace dpdr {

int fused::grant_smem(const void* fn, size_t bytes, int* granted, const char* what)
{
    if (int(bytes) <= *granted) return DPDR_OK;
    static std::mutex mu;
    static std::map<std::pair<int, const void*>, int> limit;  // (device, kernel) -> bytes
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, what);
    std::lock_guard<std::mutex> lock(mu);
    int& cur = limit[std::make_pair(dev, fn)];
    if (int(bytes) > cur) {
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, int(bytes));
        if (e != cudaSuccess) return cuda_fail(e, what);
        cur = int(bytes);
    }
    *granted = int(bytes);
    return DPDR_OK;
}

using fused::FusedArgs;
using fused::kBulkTile;
using fused::tile_lg_wu;

// Threads the streaming layouts want in flight to cover HBM latency.
static int64_t stream_target(const Plan* P) { return int64_t(P->num_sms) * 1024; }

// Layout choice, from layout sweeps measured on GB300 (int32, p = 128 ...
// 4096, m = 2^10 ... 2^20, warm and cold L2; where the two disagree, cold
// decides unless warm is far ahead):
//  * deep trees (p >= 128) with few columns -- at most 4096 16-byte column
//    units, 8192 from p = 256 -- but more than 20 MB of inputs once
//    p >= 1024: the hierarchical tile, one kernel with a walk of about
//    p / 64 (8 units per CTA) or p / 32 (16 units) ranks per thread
//    (p = 1152, m = 2^13, cold: 22.2 us against 36.2 us for the tile and
//    38.5 us for the split layout; m = 2^15: 63.6 against 67.1 us for the
//    split layout).  Both tiles take their time in waves of resident CTAs,
//    so where the shared-memory tile needs fewer waves than the
//    hierarchical one, the shared-memory tile takes over (p = 288,
//    m = 24576: one wave against two, 13.2 us warm and 18.3 cold against
//    19.3 and 21.7; with as many waves the hierarchical tile is ahead or
//    level: p = 256, m = 2^15, 17.5/20.8 against 19.8/26.3);
//  * deep trees whose p input rows total at most kTileMaxBytes: the
//    shared-memory tile, the layout with the lowest fixed cost, in tiles
//    narrowed until one wave of resident CTAs holds them when the columns
//    are few (p = 288, m = 256 int32: 5.6/8.1 us warm/cold against 9.3/16.2
//    at full width; p = 192,
//    m = 2^15 int32: 11.4 us against the split layout's 19.9 us and the
//    hierarchical tile's 17.7 us; at 75.5 MB the split layout wins at
//    p = 288, 576 and 1152);
//  * deep trees (p >= kSplitMinRanks) above that: the split layout, whose
//    read phase (first kernel) and write phase (second kernel) keep HBM
//    traffic one-directional; at p = 1152 it beats column streaming up to
//    the largest sizes;
//  * otherwise column streaming once there are a fifth of the columns it
//    needs to fill the GPU (p = 36, 2x2 matrices, m = 2^16: 13 us against the
//    tile's 15 us; 32768 int32 units: p = 64, 14.6 against 17.2 us, p = 127,
//    28.4 against 32.5), and the shared-memory tile below that (8192 units:
//    p = 64, 7.8 against 11.3 us; p = 127, 9.5 against 25.1) unless the
//    trees are shallow (p <= 16: column streaming at every size).
constexpr int64_t kTileMaxBytes = int64_t(40) << 20;
constexpr int kSplitMinRanks = 128;
constexpr int64_t kSplitWork = int64_t(1) << 17;
constexpr int64_t kTreeMinBytesLargeP = int64_t(20) << 20;
// Below p = 1024, up to this many column units the shared-memory tile, cut
// into as many narrow tiles as one wave holds, beats the hierarchical tile
// (p = 288, m = 1024 int32: 6.1/8.3 us warm/cold against 6.5/8.4; p = 576,
// m = 4096: 8.5/12.0 against 11.0/12.3; p = 128, m = 2048: 5.0/6.3
// against 6.2/8.2); above it the hierarchical tile leads cold (p = 576,
// m = 8192: 14.5 against 17.0 us).
constexpr int64_t kTileOverTreeUnits = 1024;
// Up to this many ranks column streaming takes even the fewest columns.
constexpr int kStreamMaxShallowRanks = 16;

// Resident CTAs of the shared-memory tile on the GPU: up to 4 per SM (256
// threads of 64 registers), fewer when its rows do not fit the 228 KB of
// shared memory per SM (1 KB of which is reserved per CTA).
static int64_t tile_slots(const Plan* P)
{
    const size_t smem = size_t(P->p + 1) * (size_t(16) << tile_lg_wu(P));
    return int64_t(P->num_sms) * std::min<int64_t>(4, int64_t((228 << 10) / (smem + 1024)));
}

static bool tree_preferred(const Plan* P)
{
    if (P->p < 128) return false;
    const int64_t units = P->m * int64_t(P->esize) / 16;
    const int64_t bytes = int64_t(P->p) * P->m * P->esize;
    if (units > (P->p >= 256 ? 8192 : 4096)) return false;
    if (P->p < 1024) return units > kTileOverTreeUnits;
    return bytes > kTreeMinBytesLargeP;
}

// Whether the shared-memory tile needs fewer waves of resident CTAs than
// the hierarchical tile for the plan's columns.
static bool tile_beats_tree(const Plan* P)
{
    const int lg = tile_lg_wu(P);
    if (lg < 0) return false;
    const int64_t units = P->m * int64_t(P->esize) / 16;
    const int64_t W = P->tree[fused_tree_index(P)].width;
    const int64_t tree_slots = int64_t(fused::kTreeCtasPerSm) * P->num_sms;
    const int64_t tiles = (units + (int64_t(1) << lg) - 1) >> lg;
    const int64_t tree_waves = ((units + W - 1) / W + tree_slots - 1) / tree_slots;
    const int64_t tile_waves = (tiles + tile_slots(P) - 1) / tile_slots(P);
    return tile_waves < tree_waves;
}

static bool tile_preferred(const Plan* P)
{
    return P->p >= 128 && tile_lg_wu(P) >= 0 &&
           int64_t(P->p) * P->m * P->esize <= kTileMaxBytes;
}

// Beyond p = 2048 a wide hierarchical tile is long (walks of p / 32 ranks),
// so a second wave of them that is less than 60 % full costs more than the
// split layout's two kernels (p = 4094, m = 24576 int32: 166 against 181 us;
// p = 8190, m = 20480: 282 against 322; p = 2304, m = 20480: 94 against
// 110); with a fuller second wave the tile leads again (p = 4094, m = 2^15:
// 186 against 194), and at p = 1152 it leads or ties throughout.
static bool split_over_tree(const Plan* P)
{
    if (P->p < 2048 || fused_tree_index(P) != 1) return false;
    const int64_t units = P->m * int64_t(P->esize) / 16;
    const int64_t slots = int64_t(fused::kTreeCtasPerSm) * P->num_sms;
    const int64_t ctas = (units + fused::kTreeUnitsWide - 1) / fused::kTreeUnitsWide;
    return ctas > slots && (ctas - slots) * 10 < slots * 6;
}

static bool split_beats_tree(const Plan* P) { return P->split_ready && split_over_tree(P); }

int fused_auto_mode(const Plan* P)
{
    const int64_t units = P->m * int64_t(P->esize) / 16;
    if (P->tree[fused_tree_index(P)].ready && tree_preferred(P))
        return tile_beats_tree(P) ? 2 : split_beats_tree(P) ? 3 : 5;
    if (tile_preferred(P)) return 2;
    if (P->p >= kSplitMinRanks && units >= 4096 && P->split_ready) return 3;
    if (units >= stream_target(P) / 5) return 1;
    // shallow trees: a column's walk is a batch or two of loads, and column
    // streaming beats staging rows through the tile (cold, p = 7, m = 1000
    // int32: 6.8 against 8.9 us; at p <= 16 it is never slower, from p = 32
    // the tile leads)
    if (P->p <= kStreamMaxShallowRanks) return 1;
    if (tile_lg_wu(P) >= 0) return 2;
    return P->split_ready ? 3 : 1;
}

// Whether the automatic choice can be the split layout (then the plan
// prepares it up front).
static bool split_wanted(const Plan* P)
{
    const int64_t units = P->m * int64_t(P->esize) / 16;
    return P->p >= kSplitMinRanks && units >= 4096 && !tile_preferred(P) &&
           (!tree_preferred(P) || split_over_tree(P));
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
    // automatic cut: the shallowest depth whose subtrees (2^s per tree) times
    // the column units give the first kernel kSplitWork independent walks;
    // a deeper cut only lengthens the second kernel's walk over the
    // 2^(s+2) - 2 rows.  Measured at p = 128 ... 1152, int32, m = 2^14 ...
    // 2^22: within 2 % of the best cut everywhere (at m = 2^17 the cut at
    // depth 1 takes 28.9 us at p = 128 where depth 3 took 39.5 us); never
    // deeper than 4 or than the tree allows
    int s = depth;
    if (s < 0) {
        const int64_t trees = P->r0 >= 0 ? 2 : 1;
        s = 0;
        while (s < 4 && (trees << s) * units < kSplitWork) s++;
        s = std::min(s, std::max(0, P->max_depth - 2));
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
    // store groups of the write phase: enough CTA rows of column threads to
    // fill the GPU once, and in the middle range more, shorter rows (each
    // refolds the top rows, which L2 holds): p = 1152 int32, m = 2^16 in 112.7
    // against 116.7 us with twice the rows, m = 2^17..2^20 2-5 % faster with
    // four times; at m = 2^15 and from 2^22 the extra rows cost more than
    // they give
    const int64_t target = stream_target(P);
    const int64_t more = units >= (int64_t(1) << 19) ? 1
                       : units >= (int64_t(1) << 15) ? 4
                       : units >= (int64_t(1) << 14) ? 2 : 1;
    int64_t groups = std::min<int64_t>(p, std::max<int64_t>(1, more * ((target + units - 1) / units)));
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
    return fused_launch_cols(P, P->d_x, P->d_y, P->m, P->last_vector_path != 0, s, 0);
}

// The fused kernel on mc columns, with device tables of rank pointers that
// may point into the middle of the rank buffers (a column chunk).
int fused_launch_cols(Plan* P, const char* const* dx, char* const* dy, int64_t mc, bool vec,
                      cudaStream_t s, int force_mode, int tree_index)
{
    if (mc == 0) return DPDR_OK;
    int mode = force_mode ? force_mode : P->fused_mode ? P->fused_mode : fused_auto_mode(P);
    const int lg = tile_lg_wu(P);
    if (mode == 2 && lg < 0) return fail(DPDR_ERR_INVALID, "tile mode: p too large");
    if (mode == 3 && !P->split_ready) return fail(DPDR_ERR_INVALID, "split mode: p < 2");
    const TreeTables& T = P->tree[tree_index < 0 ? fused_tree_index(P) : tree_index];
    if (mode == 5 && !T.ready) return fail(DPDR_ERR_INVALID, "tree mode not prepared");
    if (mode < 1 || mode > 5) return fail(DPDR_ERR_INVALID, "unknown fused mode");
    // the bulk and hierarchical layouts need 16-byte rows: without them the
    // bulk layout's work goes to column streaming, the hierarchical tile's to
    // the shared-memory tile (or, when a tile row does not fit, the split
    // layout), which keep its short walks (p = 288, m = 21250 int32 with
    // rows 8 bytes apart from 16: 22.8 against 57 us streamed)
    if (mode == 4 && !vec) mode = 1;
    if (mode == 5 && !vec) mode = lg >= 0 ? 2 : P->split_ready ? 3 : 1;

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
    a.dual = P->r0 >= 0 ? 1 : 0;
    const int epv = int(16 / P->esize);
    a.nvec = vec ? mc / epv : 0;
    a.scalar_base = a.nvec * epv;
    a.nscalar = mc - a.scalar_base;
    a.lg_wu = lg < 0 ? 0 : lg;
    if (mode == 2) {
        // few columns: narrower tiles, as many as one wave of resident CTAs
        // holds, so that each CTA copies fewer rank rows
        const int sc = P->esize == 4 ? 2 : 0;  // single elements per 16 bytes, log2
        auto tiles = [&](int l) {
            return ((a.nvec + (int64_t(1) << l) - 1) >> l) +
                   ((a.nscalar + (int64_t(1) << (l + sc)) - 1) >> (l + sc));
        };
        const int64_t slots = tile_slots(P);  // at the widest tile: a lower bound
        while (a.lg_wu > 0 && tiles(a.lg_wu - 1) <= slots) a.lg_wu--;
    }
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
    a.tree_seg = T.seg;
    a.tree_lev = T.lev;
    a.tree_levoff = T.levoff;
    a.tree_nseg = T.nseg;
    a.tree_nlev = T.nlev;
    a.tree_r0 = T.r0;
    a.tree_r1 = T.r1;
    a.tree_s = T.s;
    a.tree_slots = T.slots;
    a.tree_width = T.width;
    a.tree_tiles = T.width ? (a.nvec + T.width - 1) / T.width : 0;

    switch (mode) {
    case 1: return fused::launch_stream(P, a, s);
    case 2: return fused::launch_tile(P, a, s);
    case 3: return fused::launch_split(P, a, s);
    case 5: return fused::launch_tree(P, a, s);
    default: return fused::launch_bulk(P, a, s);
    }
}

}  // namespace dpdr
