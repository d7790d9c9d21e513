// dpdr_internal.h -- plan layout shared by the host code and the kernel
// launchers of the library (not part of the public ABI).
#pragma once

#include <cstddef>
#include <cstdint>
#include <string>
#include <vector>

#include <cuda_runtime.h>

#include "../../include/dpdr.h"

namespace dpdr {

// Tape byte of the column-streaming fold, one per rank in post-order:
//   bits 0-1  number of children c in {0,1,2}
//   bit  2    keep: the node value is parked in slot d (the node is the
//             child_1 of its parent, or the lower root r0)
//   bits 3-7  depth d
constexpr int kTapeKeep = 4;
constexpr int kMaxDepth = 31;
constexpr int kMaxSlices = 1024;   // column slices per rank of the schedule kernel

// Dual-root exchange slot of one column slice of the schedule kernel: the
// slice's share of the largest block, rounded up to 16 bytes, plus 48 bytes
// for the rounding of slice bounds to 16-byte units and for the offset that
// keeps every element congruent to the inputs modulo 16 bytes.  Each slice
// has a slot of its own: slices run independently, and a slice's range
// inside a block moves by a few elements from block to block, so slots
// shared across slices would let a slice that is two blocks ahead overwrite
// a neighbour's data before the dual root has read it.
inline size_t ring_sub_bytes(int64_t maxblk, size_t esize, int slices)
{
    const int64_t share = (maxblk + slices - 1) / slices;
    return (size_t(share) * esize + 15) / 16 * 16 + 48;
}

// Entries of the level table of the shared-memory tile fold: internal
// nodes, deepest level first, as (node, child_1 or -1); child_0 = node-1.
struct LevelNode {
    int node;
    int child1;
};

// Tables of the hierarchical tile layout for one tile width (fused_tree.cu):
// the entries (subtrees at depth s, then the nodes above the cut) and the
// level table above the cut.
struct TreeTables {
    bool ready = false;
    int width = 0;                   // 16-byte column units per CTA
    int s = 0, nseg = 0, nlev = 0, slots = 0, r0 = -1, r1 = 0;
    char* d = nullptr;               // own allocation
    size_t bytes = 0;
    int2* seg = nullptr;
    int4* lev = nullptr;
    int* levoff = nullptr;
};

struct Plan {
    int p = 0;
    int64_t m = 0;
    int dtype = 0;
    int op = 0;
    int topo = 0;              // DPDR_TOPO_DUAL or DPDR_TOPO_SINGLE
    int b = 1;
    size_t esize = 4;
    int device = 0;
    int num_sms = 0;
    int l2_bytes = 0;

    // trees (Sec. 1.1)
    std::vector<int> parent, child0, child1, dual, depth;
    int max_depth = 0;
    int r0 = -1, r1 = 0;       // roots (r0 = -1: one tree, no dual)
    std::vector<uint8_t> tape;                 // column-streaming fold
    std::vector<LevelNode> levels;             // tile fold
    std::vector<int> level_off;                // nlevels + 1

    // options
    int fused_mode = 0;        // 0 auto, 1 stream, 2 tile, 3 split, 4 bulk, 5 tree
    int64_t wait_ns = 4000000000LL;
    int skip_rank = -1;
    int sched_threads = 0;     // threads per schedule CTA, 0 = automatic
    int sched_rpc = 0;         // ranks per CTA, 0 = auto
    int sched_slices = 0;      // CTAs per rank (column slices), 0 = auto
    int split_depth = -1;      // cut depth of the split layout, -1 = auto
    int sched_transport = 0;   // schedule kernel: 0 auto, 1 counters, 2 flagged words
    int sched_layout = 0;      // counters kernels' CTA layout: 0 auto, 1 rank ranges, 2 by work
    int sched_copy = 0;        // counters kernels' block passes: 0 auto, 1 per-lane, 2 bulk
    int64_t host_chunk = int64_t(1) << 30;  // bytes of rank data per host-pipeline chunk
    int host_path = 0;         // dpdr_allreduce_host: 0 auto, 1 copy pipeline, 2 direct
    int last_host_path = 0;    // path the last dpdr_allreduce_host took (1 or 2)

    // device memory: one allocation carved into the tables below
    char* dmem = nullptr;
    size_t dmem_bytes = 0;
    const char** d_x = nullptr;      // [p] rank input pointers, then
    char** d_y = nullptr;            // [p] rank output pointers (d_x + p)
    uint8_t* d_tape = nullptr;       // [p rounded up to 8]
    LevelNode* d_levels = nullptr;
    int* d_level_off = nullptr;
    int* d_tables = nullptr;         // parent, child0, child1, depth: 4 x [p]
    uint32_t* d_ctrl = nullptr;      // up[G*p], down[G*p], abort word (in d_sched)
    uint32_t* d_err = nullptr;       // 4 words: status, rank, round, step
    char* d_ring = nullptr;          // dual-root exchange slots: [2][2][slot]
    size_t ring_slot_bytes = 0;
    int* d_cta_first = nullptr;      // flagged words: chunk -> first rank (+1 entry)
    int4* d_groups = nullptr;        // counters: [chunks][4] group descriptors
    int* d_rank_list = nullptr;      // counters: the groups' ranks
    char* d_sched = nullptr;         // own allocation: counters + CTA tables
    size_t d_sched_bytes = 0;
    // low-latency transport of the schedule kernel (schedule_ll.cu): control
    // words, then the up and down word arrays; own allocation
    char* d_ll = nullptr;
    size_t d_ll_bytes = 0;

    // rank-pointer staging (pinned host), copied to d_x / d_y when they change
    const void** h_ptrs = nullptr;   // [2p]
    std::vector<const void*> last_x, last_y;
    cudaEvent_t staged = nullptr;
    bool staged_pending = false;     // d_x / d_y hold last_x / last_y

    // dynamic shared memory already granted to the fused kernels of this
    // plan's element type (stream, tile, split, bulk, hierarchical tile of
    // either width, paired stream), so
    // launches skip the attribute call; the limits themselves only ever rise
    int smem_attr[7] = {48 * 1024, 48 * 1024, 48 * 1024, 48 * 1024, 48 * 1024, 48 * 1024,
                        48 * 1024};

    // split layout of the fused kernel (fused.cu): subtrees at depth split_s
    bool split_ready = false;
    int split_s = 0, split_nseg = 0, split_nitems = 0, split_group = 1;
    char* d_split = nullptr;         // own allocation: seg, items, subtree rows
    size_t d_split_bytes = 0;
    int2* d_seg = nullptr;
    int2* d_items = nullptr;
    char* d_part = nullptr;
    int64_t part_stride = 0;

    // hierarchical tile layout of the fused kernel (fused_tree.cu), one set
    // of tables per tile width: [0] 8 column units per CTA, [1] 16
    TreeTables tree[2];

    // host-buffer pipeline of dpdr_allreduce_host (api.cpp), made on first use:
    // column chunks copied in on one stream, reduced on the caller's stream,
    // copied out on another
    cudaStream_t pipe_in = nullptr, pipe_out = nullptr;
    std::vector<cudaEvent_t> pipe_ev;            // entry, done, then in/out per chunk
    char* d_pipe = nullptr;                      // per-chunk rank-pointer tables
    size_t d_pipe_bytes = 0;
    int64_t pipe_cols = 0;
    int pipe_chunks = 0;
    std::vector<const void*> pipe_xd, pipe_yd;
    // device addresses of host buffers the GPU reads and writes directly
    std::vector<const void*> direct_xh, direct_yh;   // host arrays they came from
    std::vector<const void*> direct_dx, direct_dy;
    bool direct_ok = false;

    // facts
    int last_vector_path = 0;
    int sched_ctas = 0, sched_ranks_per_cta = 0;
    int sched_rpc_ref = 1;         // ranks per CTA at 128 threads (transport choice)
    int sched_threads_used = 128;  // threads per CTA of the kernel that runs
    int sched_slices_used = 1, sched_chunks = 1;
    int sched_layout_used = 1;     // 1 rank ranges, 2 by work
    int sched_copy_used = 2;       // 1 per-lane copies, 2 bulk copies
    int sched_slot_bytes = 192;    // counters kernels: shared memory per thread
};

// host-side builders (plan.cpp)
void build_tree(int p, int topo, int* parent, int* child0, int* child1, int* dual,
                int* depth);
int block_count_rule(int p, int64_t m, double kappa);

// errors (plan.cpp)
int fail(int status, const std::string& msg);
int cuda_fail(cudaError_t e, const char* what);
// the same without building a std::string (no heap use)
int fail_c(int status, const char* msg);
int cuda_fail_c(cudaError_t e, const char* what);

// rank-pointer upload (api.cpp)
int stage_pointers(Plan* P, const void* const* x, const void* const* y,
                   cudaStream_t s);

// launchers
int fused_launch(Plan* P, cudaStream_t s);      // fused.cu
int fused_launch_cols(Plan* P, const char* const* dx, char* const* dy, int64_t mc, bool vec,
                      cudaStream_t s, int force_mode,  // fused.cu (0: plan's choice)
                      int tree_index = -1);  // hierarchical tile width: -1 plan's, 0 / 1
int fused_auto_mode(const Plan* P);             // fused.cu
int fused_split_prepare(Plan* P, bool force, int depth);  // fused.cu
int fused_tree_prepare(Plan* P);                // fused_tree.cu: both widths
int fused_tree_index(const Plan* P);            // fused_tree.cu: the device path's width
int schedule_launch(Plan* P, cudaStream_t s,   // schedule.cu: Algorithm 1 (algo 0)
                    int algo = 0);              // or reduce, then broadcast (1)
int schedule_configure(Plan* P);                // schedule.cu
int schedule_plan_rpc(Plan* P);                 // schedule.cu: ranks per CTA only
int schedule_transport(const Plan* P);          // schedule_ll.cu: 1 counters, 2 words
const void* schedule_ll_kernel_for(int dtype);  // schedule_ll.cu
size_t schedule_ll_bytes(const Plan* P);        // schedule_ll.cu
int64_t schedule_ll_slice_elems(const Plan* P); // schedule_ll.cu
int schedule_ll_prepare(Plan* P);               // schedule_ll.cu
int schedule_ll_launch(Plan* P, cudaStream_t s);  // schedule_ll.cu

}  // namespace dpdr
