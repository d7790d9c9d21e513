/*
 * dpdr.h -- C ABI of a one-GPU doubly pipelined, dual-root reduction-to-all
 * (J. L. Traff, "A Doubly-pipelined, Dual-root Reduction-to-all Algorithm
 * and Implementation", arXiv 2109.12626, 2021).
 *
 * The operation (Sec. 1, problem statement): each of p successively ranked
 * processors holds a vector x_i of m elements; the element-wise product
 * y = x_0 (.) x_1 (.) ... (.) x_{p-1} for an associative, not necessarily
 * commutative operator (.) is computed and delivered to all p processors.
 * Here the p processors are virtual ranks on one GPU: rank i is an input
 * buffer x[i] and an output buffer y[i], each m elements in device memory.
 *
 * The result is the bracketing of Sec. 1.1 and Algorithm 1: the ranks form
 * two post-order-numbered complete binary trees, tree 0 = ranks
 * [0, floor(p/2)) and tree 1 = [floor(p/2), p); the value of node i is
 * v(child_1) (.) ( v(child_0) (.) x_i ) with child_0 = i-1, and
 * y = v(r0) (.) v(r1) for the roots r0 = floor(p/2)-1 and r1 = p-1 (or, for
 * a plan made with DPDR_TOPO_SINGLE, y = v(p-1) of one tree).  Every entry
 * point below produces exactly this result, bit for bit, for every element
 * type (float32 included), in every y[i].
 *
 * Conventions for all functions:
 *   - Status codes (dpdr_status) are returned; nothing throws, the device
 *     never traps.  A failing call also sets a thread-local last error
 *     (dpdr_last_error, dpdr_last_error_message).
 *   - "host array of p device pointers": x and y are arrays in host memory
 *     holding p device addresses; the caller owns every buffer, each of
 *     m elements of the plan's element type, contiguous.  Every buffer must
 *     be aligned to its element size (4 bytes); 16-byte alignment of all
 *     2p buffers enables the vectorised path.
 *   - In-place use, y[i] == x[i] (Algorithm 1 initialises Y <- x_i and
 *     leaves y in Y), is allowed for every i.  Any other overlap between
 *     buffers is invalid.
 *   - Calls are asynchronous on the given stream; the inputs must stay
 *     valid and unmodified until the stream has passed the call.
 */
#ifndef DPDR_H
#define DPDR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Element types and operators (the operator functors of the library). */
typedef enum {
    DPDR_INT32 = 0,      /* int32, sum wraps mod 2^32                       */
    DPDR_FLOAT32 = 1,    /* IEEE float32, sum rounded to nearest even        */
    DPDR_MAT2X2_U32 = 2, /* 2x2 uint32 matrix, row-major a,b,c,d (16 bytes) */
    DPDR_MAT2X2_F32 = 3  /* 2x2 float32 matrix, row-major (16 bytes); each
                            product entry is two rounded products and one
                            rounded sum, never fused                        */
} dpdr_dtype;

typedef enum {
    DPDR_OP_SUM = 0,     /* with DPDR_INT32 or DPDR_FLOAT32                  */
    DPDR_OP_MATMUL = 1   /* with DPDR_MAT2X2_U32 (product mod 2^32) or
                            DPDR_MAT2X2_F32: the lower rank on the left
                            (non-commutative)                               */
} dpdr_op;

typedef enum {
    DPDR_OK = 0,
    DPDR_ERR_INVALID = 1,          /* bad argument, alignment or overlap     */
    DPDR_ERR_CUDA = 2,             /* a CUDA runtime call failed             */
    DPDR_ERR_TIMEOUT = 3,          /* a bounded wait of the schedule kernel
                                      expired (reported by dpdr_plan_sync)   */
    DPDR_ERR_NOT_COOPERATIVE = 4,  /* the schedule kernel's CTAs cannot all
                                      be resident at once                    */
    DPDR_ERR_OOM = 5               /* device or pinned host memory exhausted */
} dpdr_status;

/* How the ranks are arranged.  DPDR_TOPO_DUAL is the paper's method: two
 * post-order trees whose roots are duals (Sec. 1.1, Algorithm 1).
 * DPDR_TOPO_SINGLE is the one-tree variant Sec. 1.2 discusses: all p ranks
 * in one complete post-order tree, root p-1, no dual-root step (every
 * non-leaf applies (.) at most twice per round); y = v(p-1), a different
 * float32 bracketing from the dual trees'. */
typedef enum {
    DPDR_TOPO_DUAL = 0,
    DPDR_TOPO_SINGLE = 1
} dpdr_topology;

/* Opaque plan; owns the device-side tables and scratch of one (p, m, type). */
typedef struct dpdr_plan_s* dpdr_plan_t;

/* A CUDA stream (cudaStream_t / CUstream); NULL is the legacy default
 * stream. */
typedef struct CUstream_st* dpdr_stream_t;

/* ---------------------------------------------------------------- host only
 * These need no GPU. */

/* The dual post-order trees of Sec. 1.1 for p ranks.  Fills five
 * caller-owned int[p] arrays: parent (-1 at the roots), child0 (= i-1 when
 * i has a child, else -1), child1 (the root of the lower subtree interval,
 * -1 if none; a node with one child has only child0), dual (the other root
 * at r0 and r1, else -1) and depth (d_i, 0 at the roots; Algorithm 1 runs
 * rounds j = 0..b+d_i).  Any pointer may be NULL.  p >= 1. */
int dpdr_tree(int p, int* parent, int* child0, int* child1, int* dual,
              int* depth);

/* dpdr_tree for either topology (with DPDR_TOPO_SINGLE every dual is -1). */
int dpdr_tree_topo(int p, dpdr_topology topo, int* parent, int* child0,
                   int* child1, int* dual, int* depth);

/* Block partition of Algorithm 1 (Sec. 1.1: b successive blocks of roughly
 * m/b elements): writes b+1 caller-owned starts, block j = [starts[j],
 * starts[j+1]); the first m mod b blocks hold ceil(m/b) elements, the rest
 * floor(m/b).  Requires 1 <= b <= m. */
int dpdr_blocks(int64_t m, int b, int64_t* starts);

/* Block count from the pipelining-lemma optimum of Sec. 1.2,
 * b* = sqrt((4h-6) m beta / (3 alpha)) with h = ceil(log2(p+2)), written
 * with kappa = alpha/beta in elements: round(sqrt((4h-6) m / (3 kappa))),
 * clamped to [1, max(m,1)].  kappa <= 0 selects the default 1024. */
int dpdr_block_count_rule(int p, int64_t m, double kappa);

/* -------------------------------------------------------------------- plan */

/* Builds the trees, the block partition and the device tables for p ranks
 * of m elements of (dtype, op) on the current CUDA device, and allocates the
 * plan's device scratch (rank-pointer tables, handshake counters, the dual
 * roots' exchange slots, an error word, and the word arrays of the
 * schedule kernel's flagged-word transport when it is selected).  b is the
 * number of pipeline blocks (Algorithm 1), clamped to [1, max(m,1)].
 * b == 0 selects a block count measured for the schedule kernel on this
 * GPU: 1 when the flagged-word transport is selected (latency-bound);
 * otherwise dpdr_block_count_rule(p, m, kappa) with kappa = 46e6 / (p
 * esize) elements (alpha/beta of the counters transport; the ranks share
 * device memory, so beta grows with p), raised to at least
 * 2 p m esize / (L2 bytes) so that the blocks in flight stay in L2.
 * p >= 1, m >= 0.  Returns NULL on error (see dpdr_last_error).  Not
 * thread-safe with respect to one plan. */
dpdr_plan_t dpdr_plan(int p, int64_t m, dpdr_dtype dtype, dpdr_op op, int b);

/* dpdr_plan for either topology (dpdr_plan is DPDR_TOPO_DUAL).  Every entry
 * point then computes that topology's bracketing.  The allocation-free entry
 * point supports the dual topology only. */
dpdr_plan_t dpdr_plan_topo(int p, int64_t m, dpdr_dtype dtype, dpdr_op op,
                           int b, dpdr_topology topo);

/* Copies the plan's trees (caller-owned int[p] arrays, any may be NULL) and
 * the block count in use. */
int dpdr_plan_query(dpdr_plan_t plan, int* parent, int* child0, int* child1,
                    int* dual, int* depth, int* b_used);

/* Plan options (key, value):
 *   DPDR_OPT_FUSED_MODE       0 auto, 1 column-streaming, 2 shared-memory
 *                             tile, 3 subtree split, 4 bulk-copy pipeline,
 *                             5 hierarchical tile (the five layouts of
 *                             dpdr_allreduce; 3 needs p >= 2 and keeps
 *                             m * esize bytes of scratch per subtree; 4 and
 *                             5 need 16-byte aligned buffers: otherwise 4
 *                             runs as 1, and 5 as 2, or as 3 (else 1) when
 *                             a tile row of p elements does not fit)
 *   DPDR_OPT_WAIT_LIMIT_NS    bound of every wait of the schedule kernel,
 *                             nanoseconds: 1e3 .. 1e10 (default 4e9); values
 *                             outside that range are DPDR_ERR_INVALID, so a
 *                             wait can never become unbounded
 *   DPDR_OPT_SKIP_RANK        fault injection for tests: this rank of the
 *                             schedule kernel never publishes a block, so
 *                             its partners' waits expire (-1 = off)
 *   DPDR_OPT_SCHED_THREADS    threads per CTA of the schedule kernel
 *                             (64..256, multiple of 32); 0 (default) is
 *                             automatic: 128 with the counters transport
 *                             laid out by work and with flagged words, 64
 *                             with the counters transport on rank ranges
 *   DPDR_OPT_SCHED_RANKS_PER_CTA  virtual ranks per CTA (0 = fewest that
 *                             fit co-resident)
 *   DPDR_OPT_BLOCKS           change b (same rules as dpdr_plan's b)
 *   DPDR_OPT_SPLIT_DEPTH      tree depth at which the split layout cuts
 *                             the ranks into subtrees (-1 = automatic)
 *   DPDR_OPT_SCHED_SLICES     CTAs per virtual rank in the schedule kernel,
 *                             each owning one column slice of every block
 *                             (0 = as many as fit co-resident, slices of at
 *                             least 1024 elements, at most 64)
 *   DPDR_OPT_HOST_CHUNK_BYTES bytes of rank data per column chunk of
 *                             dpdr_allreduce_host's copy pipeline (default
 *                             2^30, minimum 4096)
 *   DPDR_OPT_HOST_PATH        dpdr_allreduce_host: 0 direct when possible,
 *                             else copy; 1 copy pipeline; 2 direct only
 *   DPDR_OPT_SCHED_TRANSPORT  how dpdr_allreduce_schedule moves a block
 *                             between virtual ranks (same rounds, steps and
 *                             result either way): 1 counters -- the block is
 *                             written, then a release/acquire counter
 *                             publishes it; 2 flagged words -- every 32-bit
 *                             word travels with the call's epoch in one
 *                             64-bit store and the receiver polls the words,
 *                             which halves the latency of short blocks but
 *                             keeps 4 p m esize bytes of word arrays on the
 *                             device; 0 (default) chooses 2 while the p
 *                             inputs total at most 12 MiB (24 MiB from
 *                             p = 1024) with one rank per schedule CTA,
 *                             8 MiB with two, never with more; else 1
 *   DPDR_OPT_SCHED_LAYOUT     how the counters transport of the schedule
 *                             kernels lays out virtual ranks on CTAs:
 *                             1 rank ranges -- each CTA owns a contiguous
 *                             range of ranks; 2 by work -- each rank has
 *                             warps of its own in proportion to its block
 *                             passes per round (a leaf one quarter of a
 *                             CTA, an inner node three quarters, a root a
 *                             whole CTA), DPDR_ERR_INVALID when one column
 *                             slice of it does not fit the GPU at once;
 *                             0 (default) takes 2 where it fits, else 1.
 *                             Set ranks per CTA always take rank ranges
 *   DPDR_OPT_SCHED_COPY       how the counters transport's block passes move
 *                             16-byte units (same result either way):
 *                             1 per-lane copies into private shared-memory
 *                             slots; 2 bulk (TMA) copies of chunks of a few KB
 *                             through a double-buffered region per rank;
 *                             0 (default) takes 1 while a column slice of a
 *                             block holds at most 1024 units, else 2 */
enum {
    DPDR_OPT_FUSED_MODE = 1,
    DPDR_OPT_WAIT_LIMIT_NS = 2,
    DPDR_OPT_SKIP_RANK = 3,
    DPDR_OPT_SCHED_THREADS = 4,
    DPDR_OPT_SCHED_RANKS_PER_CTA = 5,
    DPDR_OPT_BLOCKS = 6,
    DPDR_OPT_SPLIT_DEPTH = 7,
    DPDR_OPT_SCHED_SLICES = 8,
    DPDR_OPT_HOST_CHUNK_BYTES = 9,
    DPDR_OPT_HOST_PATH = 10,
    DPDR_OPT_SCHED_TRANSPORT = 11,
    DPDR_OPT_SCHED_LAYOUT = 12,
    DPDR_OPT_SCHED_COPY = 13
};
int dpdr_plan_set(dpdr_plan_t plan, int key, int64_t value);

/* Plan facts for tools and tests, int64 each, n of them:
 *   [0] p  [1] m  [2] b  [3] max depth  [4] fused mode that auto selects
 *   [5] schedule CTAs  [6] ranks per schedule CTA  [7] device scratch bytes
 *   [8] 1 if the last dpdr_allreduce ran the 16-byte vector path
 *   [9] split layout cut depth  [10] its scratch rows (subtrees plus nodes
 *   above the cut)  [11] ranks per store
 *   group of its second kernel (0 when the split layout is not prepared)
 *   [12] CTAs per rank (column slices) of the schedule kernel
 *   [13] topology (dpdr_topology)
 *   [14] path of the last dpdr_allreduce_host: 1 copy pipeline, 2 direct
 *   [15] transport of dpdr_allreduce_schedule: 1 counters, 2 flagged words
 *   [16] 16-byte column units per CTA of the hierarchical tile layout on
 *        device buffers (8 while those CTAs fit in one wave of resident
 *        CTAs, 2 per SM; else 16; host buffers always take 8)
 *   [17] CTA layout of the schedule kernels: 1 rank ranges, 2 by work
 *        (DPDR_OPT_SCHED_LAYOUT; flagged words always take rank ranges)
 *   [18] block passes of the counters transport: 1 per-lane copies, 2 bulk
 *        copies (DPDR_OPT_SCHED_COPY) */
int dpdr_plan_info(dpdr_plan_t plan, int64_t* info, int n);

/* Releases the plan's device and host memory.  The caller must first make
 * sure no call on the plan is still running on the GPU.  NULL is a no-op. */
void dpdr_plan_destroy(dpdr_plan_t plan);

/* --------------------------------------------------------------- run it */

/* Fused bandwidth kernel: y[i] = y for all i, one kernel launch.  Each
 * element column is read once from each of the p inputs and written once to
 * each of the p outputs (2 p m element transfers of device memory); the
 * (.)-combines follow the bracketing above exactly.  x, y: host arrays of p
 * device pointers.  Asynchronous on stream. */
int dpdr_allreduce(dpdr_plan_t plan, const void* const* x, void* const* y,
                   dpdr_stream_t stream);

/* Schedule-faithful kernel: runs Algorithm 1 for every virtual rank, rounds
 * j = 0..b+d_i, each round's exchanges with child_0, child_1 and the parent
 * or dual, as one cooperative persistent launch in which groups of warps
 * serve ranks (DPDR_OPT_SCHED_LAYOUT) and exchange pipeline blocks through
 * device memory, published either by release/acquire counters or as
 * epoch-flagged words (DPDR_OPT_SCHED_TRANSPORT); with counters, blocks
 * move between device memory and shared memory by bulk (TMA) or per-lane
 * copies (DPDR_OPT_SCHED_COPY).  Same result as dpdr_allreduce.  Two calls
 * on one plan that overlap on the GPU (two streams) race on its scratch.  Every wait is bounded
 * (DPDR_OPT_WAIT_LIMIT_NS); an expired wait ends the kernel early and is
 * reported as DPDR_ERR_TIMEOUT by dpdr_plan_sync.  Returns
 * DPDR_ERR_NOT_COOPERATIVE if the ranks cannot be co-resident.
 * Asynchronous on stream. */
int dpdr_allreduce_schedule(dpdr_plan_t plan, const void* const* x,
                            void* const* y, dpdr_stream_t stream);

/* The alternative that Sec. 1.2 analyses and Sec. 2 (item 3) measures
 * against Algorithm 1: a pipelined reduction of the plan's b blocks to the
 * root of one binary tree, followed by a pipelined broadcast of them from
 * the root, each phase moving blocks in one direction only.  Needs a plan
 * made with DPDR_TOPO_SINGLE (the complete post-order tree over all p ranks,
 * root p-1); any other plan is DPDR_ERR_INVALID.  Runs as one cooperative
 * persistent launch with the same CTA layout, handshakes, block passes and
 * bounded waits as dpdr_allreduce_schedule's counters transport: in the
 * reduction every rank forms Y[j] = v(child_1) (.) (v(child_0) (.) x_i) for
 * j = 0..b-1 and publishes it to its parent; once its reduction is done it
 * receives the final blocks from its parent in order and publishes each to
 * its children (the root publishes all b once its reduction is done).  The
 * result is the one tree's bracketing, bit for bit the same as
 * dpdr_allreduce and dpdr_allreduce_schedule on the same plan.  x, y: host
 * arrays of p device pointers, as for dpdr_allreduce; in place allowed.
 * Asynchronous on stream; an expired wait is reported by dpdr_plan_sync.
 * Two calls on one plan that overlap on the GPU race on its scratch. */
int dpdr_allreduce_reduce_bcast(dpdr_plan_t plan, const void* const* x,
                                void* const* y, dpdr_stream_t stream);

/* Host buffers end to end: y_host[i] = x_host[0] (.) ... (.) x_host[p-1]
 * for host memory x_host[i], y_host[i] (all four arguments are host arrays
 * of p pointers).  Two paths:
 *   direct  when the GPU can address every host buffer (pinned memory, or
 *           pageable memory on systems whose GPU uses the CPU page tables,
 *           such as Grace with NVLink-C2C): one launch of the fused kernel
 *           (the layout DPDR_OPT_FUSED_MODE names, else the hierarchical
 *           tile, or column streaming below 1 MiB of inputs and above 4 GiB
 *           at p < 64) loads the inputs from host memory and stores the result
 *           to host memory, both link directions at once; x_dev and y_dev
 *           are not used and may be NULL.
 *   copy    otherwise: the columns are cut into chunks (about 1 GB of rank
 *           data each) that flow through a pipeline -- copies into the
 *           device buffers x_dev[i] on one plan-owned stream, the kernel on
 *           `stream` into y_dev, copies out on another stream -- so the two
 *           copy directions and the kernel overlap.
 * DPDR_OPT_HOST_PATH picks (0 auto, 1 copy, 2 direct or fail).  The call is
 * ordered after earlier work on `stream`, and later work on `stream` sees
 * its results. */
int dpdr_allreduce_host(dpdr_plan_t plan, const void* const* x_host,
                        void* const* y_host, void* const* x_dev,
                        void* const* y_dev, dpdr_stream_t stream);

/* Waits for stream, then reports and clears any device-side error of the
 * plan's schedule kernel: DPDR_ERR_TIMEOUT with details in
 * dpdr_last_error_message ("rank r round j step s"). */
int dpdr_plan_sync(dpdr_plan_t plan, dpdr_stream_t stream);

/* ------------------------------------------------------ allocation-free
 * The paper has no counterpart to this entry point; it exists for callers
 * that cannot allocate device memory on the call path: code whose device
 * memory is owned by another allocator (a framework's caching pool, a fixed
 * application-wide budget), or that must not call cudaMalloc while running
 * because an allocation can fail mid-run or stall the whole device.  It
 * needs no plan (dpdr_plan allocates) and calls no cudaMalloc, cudaFree or
 * other allocating routine.
 *
 * It runs the same schedule kernel as dpdr_allreduce_schedule, with the same
 * result, using a scratch array of DPDR_NOALLOC_SCRATCH_BYTES in device
 * memory.  The array is created when the library's device code is loaded on
 * a GPU, and held until the process exits.  With CUDA's default lazy module
 * loading that happens at the first call into this library on that device,
 * so a caller that must not allocate during some section makes one call
 * first (any dpdr call on that device, this one included) or sets
 * CUDA_MODULE_LOADING=EAGER.  That array holds the rank-pointer and
 * tree tables, the handshake counters, the error word and the dual roots'
 * exchange slots (4 slots of one pipeline block each).  Limits: p <=
 * DPDR_NOALLOC_MAX_RANKS, and the tables plus 4 slots of ceil(m/b) elements
 * must fit the array; otherwise the call returns DPDR_ERR_INVALID saying
 * which limit was hit (raise b to shrink the blocks).
 *
 * x and y are host arrays of p device pointers, as for dpdr_allreduce; the
 * caller guarantees that no buffers overlap except y[i] == x[i] (this call
 * does not check overlap).  b: pipeline blocks, clamped to [1, m];
 * 0 selects dpdr_block_count_rule(p, m, 0).
 * The call is synchronous: it returns after stream has finished the
 * kernel, with DPDR_ERR_TIMEOUT if one of its bounded waits expired.  The
 * first call on each device looks up the array's device address (with that
 * device current) and keeps it; make that first call before any stream
 * capture.  The kept address does not survive cudaDeviceReset: after a
 * reset, do not call this entry point again in the process.  Every call shares the one array and
 * re-initialises what must start at zero; calls that overlap on the GPU
 * (from two host threads, or on two streams) race and must not be made. */
#define DPDR_NOALLOC_SCRATCH_BYTES (8u << 20)
#define DPDR_NOALLOC_MAX_RANKS 8192
int dpdr_allreduce_schedule_noalloc(int p, int64_t m, dpdr_dtype dtype,
                                    dpdr_op op, int b, const void* const* x,
                                    void* const* y, dpdr_stream_t stream);

/* ------------------------------------------------------------ errors */
int dpdr_last_error(void);
const char* dpdr_last_error_message(void);
const char* dpdr_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* DPDR_H */
