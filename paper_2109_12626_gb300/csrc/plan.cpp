// plan.cpp -- host side of the library: the dual post-order trees
// (Sec. 1.1), the block partition and block-count rule (Algorithm 1,
// Sec. 1.2), the device tables each kernel reads, and the plan object.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>

#include "dpdr_internal.h"

namespace dpdr {

// ------------------------------------------------------------------ errors
static thread_local int g_last = DPDR_OK;
static thread_local char g_msg[256] = "";

int fail(int status, const std::string& msg)
{
    g_last = status;
    std::snprintf(g_msg, sizeof g_msg, "%s", msg.c_str());
    return status;
}

int fail_c(int status, const char* msg)
{
    g_last = status;
    std::snprintf(g_msg, sizeof g_msg, "%s", msg);
    return status;
}

int cuda_fail_c(cudaError_t e, const char* what)
{
    g_last = e == cudaErrorMemoryAllocation ? DPDR_ERR_OOM : DPDR_ERR_CUDA;
    std::snprintf(g_msg, sizeof g_msg, "%s: %s", what, cudaGetErrorString(e));
    return g_last;
}

int cuda_fail(cudaError_t e, const char* what)
{
    std::string m = std::string(what) + ": " + cudaGetErrorString(e);
    return fail(e == cudaErrorMemoryAllocation ? DPDR_ERR_OOM : DPDR_ERR_CUDA, m);
}

// ------------------------------------------------------------------- trees
// A subtree of n ranks occupies the post-order interval [lo, lo+n-1] with
// its root at the top end.  "As balanced and complete as possible" is read
// as a complete binary tree: with H = floor(log2 n) the levels 0..H-1 are
// full and the n - (2^H - 1) nodes of level H fill from the left.  The left
// subtree, which post-order numbers first (the lower ranks [i', i'']), gets
// the 2^(H-1) - 1 nodes of its full levels plus up to 2^(H-1) of the last
// level; its root is child_1 = i''.  The right subtree [i''+1, i-1] has root
// child_0 = i-1.  A node with a single child calls it child_0.
static void subtree(int lo, int n, int up, int d, int* parent, int* c0,
                    int* c1, int* depth)
{
    while (n > 0) {
        const int root = lo + n - 1;
        parent[root] = up;
        depth[root] = d;
        if (n == 1) {
            c0[root] = c1[root] = -1;
            return;
        }
        int H = 0;
        while ((2 << H) <= n) H++;           // floor(log2 n)
        const int half = 1 << (H - 1);
        const int last_level = n - ((1 << H) - 1);
        const int L = (half - 1) + std::min(last_level, half);
        const int R = n - 1 - L;
        if (R > 0) {
            c0[root] = root - 1;
            c1[root] = lo + L - 1;
            subtree(lo, L, root, d + 1, parent, c0, c1, depth);
            lo = lo + L;                     // continue with the right subtree
            n = R;
        } else {
            c0[root] = root - 1;             // single (left) child
            c1[root] = -1;
            n = L;
        }
        up = root;
        d = d + 1;
    }
}

void build_tree(int p, int topo, int* parent, int* child0, int* child1, int* dual,
                int* depth)
{
    const int n0 = topo == DPDR_TOPO_SINGLE ? 0 : p / 2;
    subtree(0, n0, -1, 0, parent, child0, child1, depth);
    subtree(n0, p - n0, -1, 0, parent, child0, child1, depth);
    for (int i = 0; i < p; i++) dual[i] = -1;
    if (n0 > 0) {
        dual[n0 - 1] = p - 1;
        dual[p - 1] = n0 - 1;
    }
}

// Sec. 1.2: for p = 2^h - 2 the doubly pipelined time is
// (4h-3+3(b-1))(alpha + beta m/b); balancing the terms gives
// b* = sqrt((4h-6) beta m / (3 alpha)).  h is taken as ceil(log2(p+2)) for
// any p, and kappa = alpha/beta is expressed in elements.
int block_count_rule(int p, int64_t m, double kappa)
{
    if (kappa <= 0) kappa = 1024.0;
    int h = 0;
    while ((int64_t(1) << h) < int64_t(p) + 2) h++;
    const double v = std::sqrt(double(4 * h - 6) * double(m) / (3.0 * kappa));
    int64_t b = int64_t(std::llround(v));
    const int64_t hi = std::max<int64_t>(m, 1);
    b = std::max<int64_t>(1, std::min<int64_t>(b, hi));
    return int(std::min<int64_t>(b, int64_t(1) << 30));
}

}  // namespace dpdr

using namespace dpdr;

// ------------------------------------------------------------- host ABI
extern "C" int dpdr_tree_topo(int p, dpdr_topology topo, int* parent, int* child0,
                              int* child1, int* dual, int* depth)
{
    if (p < 1) return fail(DPDR_ERR_INVALID, "dpdr_tree: p < 1");
    if (topo != DPDR_TOPO_DUAL && topo != DPDR_TOPO_SINGLE)
        return fail(DPDR_ERR_INVALID, "dpdr_tree: unknown topology");
    std::vector<int> t(size_t(5) * size_t(p));
    int* T = t.data();
    build_tree(p, topo, T, T + p, T + 2 * p, T + 3 * p, T + 4 * p);
    int* outs[5] = {parent, child0, child1, dual, depth};
    for (int k = 0; k < 5; k++)
        if (outs[k]) std::memcpy(outs[k], T + size_t(k) * p, sizeof(int) * p);
    return DPDR_OK;
}

extern "C" int dpdr_tree(int p, int* parent, int* child0, int* child1,
                         int* dual, int* depth)
{
    return dpdr_tree_topo(p, DPDR_TOPO_DUAL, parent, child0, child1, dual, depth);
}

extern "C" int dpdr_blocks(int64_t m, int b, int64_t* starts)
{
    if (b < 1 || m < b || !starts)
        return fail(DPDR_ERR_INVALID, "dpdr_blocks: need 1 <= b <= m");
    const int64_t q = m / b, r = m % b;
    for (int j = 0; j <= b; j++) starts[j] = int64_t(j) * q + std::min<int64_t>(j, r);
    return DPDR_OK;
}

extern "C" int dpdr_block_count_rule(int p, int64_t m, double kappa)
{
    if (p < 1 || m < 0) return fail(DPDR_ERR_INVALID, "block rule: bad p or m");
    return block_count_rule(p, m, kappa);
}

extern "C" int dpdr_last_error(void) { return g_last; }
extern "C" const char* dpdr_last_error_message(void) { return g_msg; }

extern "C" const char* dpdr_status_string(int s)
{
    switch (s) {
    case DPDR_OK: return "ok";
    case DPDR_ERR_INVALID: return "invalid argument";
    case DPDR_ERR_CUDA: return "CUDA error";
    case DPDR_ERR_TIMEOUT: return "schedule kernel wait timed out";
    case DPDR_ERR_NOT_COOPERATIVE: return "ranks cannot be co-resident";
    case DPDR_ERR_OOM: return "out of memory";
    default: return "unknown status";
    }
}

// -------------------------------------------------------------------- plan
static size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

static int clamp_b(int64_t m, int64_t b)
{
    const int64_t hi = std::max<int64_t>(m, 1);
    return int(std::max<int64_t>(1, std::min<int64_t>(std::min<int64_t>(b, hi),
                                                      int64_t(1) << 30)));
}

// Block count for b == 0 (dpdr_plan, DPDR_OPT_BLOCKS 0): the Sec. 1.2
// optimum b* = sqrt((4h-6) m / (3 kappa)) with kappa = alpha/beta as
// measured for the schedule kernel on GB300, raised so that the blocks the
// p ranks hold at once fit in L2.
//  * counters transport: alpha is 2.2-2.7 us per round and beta grows with
//    p (the virtual ranks share HBM), so kappa ~ kKappaBytes / (p esize):
//    about 40 K elements at p = 288 and 10 K at p = 1152 for int32, the
//    best b of b sweeps at m = 2^14 .. 2^18.  From m ~ 2^20 the best b is
//    larger: the partial and final blocks stay in L2 when about four blocks
//    per rank (input, partial, final, the next block) fit, so
//    b >= 4 p m esize / L2 (p = 1152, m = 2^22: 14.7 ms at b = 512 against
//    17.9 ms at b = 128).
//  * flagged-word transport (m esize <= 32 KiB): latency-bound, b = 1.
constexpr double kKappaBytes = 46e6;
// Upper bound of DPDR_OPT_WAIT_LIMIT_NS: every wait of the schedule kernel
// stays bounded whatever the caller asks for.
constexpr int64_t kMaxWaitNs = 10000000000LL;

static int default_blocks(const Plan* P)
{
    if (schedule_transport(P) == 2) return 1;
    const double kappa = std::max(1.0, kKappaBytes / (double(P->p) * double(P->esize)));
    int64_t b = block_count_rule(P->p, P->m, kappa);
    if (P->l2_bytes > 0) {
        // two blocks per rank in L2 (the partial or final block in flight
        // and the next one): within 0-7 % of the best b from p = 32 to 1152
        const double need = 2.0 * double(P->p) * double(P->m) * double(P->esize) /
                            double(P->l2_bytes);
        b = std::max<int64_t>(b, int64_t(std::ceil(need)));
    }
    return clamp_b(P->m, b);
}

static void build_tables(Plan* P)
{
    const int p = P->p;
    P->parent.assign(p, -1);
    P->child0.assign(p, -1);
    P->child1.assign(p, -1);
    P->dual.assign(p, -1);
    P->depth.assign(p, 0);
    build_tree(p, P->topo, P->parent.data(), P->child0.data(), P->child1.data(),
               P->dual.data(), P->depth.data());
    P->max_depth = *std::max_element(P->depth.begin(), P->depth.end());
    P->r0 = P->topo == DPDR_TOPO_SINGLE ? -1 : p / 2 - 1;
    P->r1 = p - 1;

    // tape of the column-streaming fold
    P->tape.assign(align_up(size_t(p), 8), 0);
    for (int i = 0; i < p; i++) {
        const int c = (P->child0[i] >= 0) + (P->child1[i] >= 0);
        const int par = P->parent[i];
        const bool keep = (par >= 0 && P->child1[par] == i) || (i == P->r0);
        P->tape[i] = uint8_t(c | (keep ? kTapeKeep : 0) | (P->depth[i] << 3));
    }
    // level table of the tile fold: internal nodes, deepest level first
    P->levels.clear();
    P->level_off.assign(1, 0);
    for (int d = P->max_depth; d >= 0; d--) {
        for (int i = 0; i < p; i++)
            if (P->depth[i] == d && P->child0[i] >= 0)
                P->levels.push_back(LevelNode{i, P->child1[i]});
        P->level_off.push_back(int(P->levels.size()));
    }
}

static void free_plan(Plan* P)
{
    if (!P) return;
    if (P->staged) cudaEventDestroy(P->staged);
    for (cudaEvent_t e : P->pipe_ev) cudaEventDestroy(e);
    if (P->pipe_in) cudaStreamDestroy(P->pipe_in);
    if (P->pipe_out) cudaStreamDestroy(P->pipe_out);
    if (P->d_pipe) cudaFree(P->d_pipe);
    if (P->d_split) cudaFree(P->d_split);
    for (TreeTables& T : P->tree)
        if (T.d) cudaFree(T.d);
    if (P->d_sched) cudaFree(P->d_sched);
    if (P->d_ll) cudaFree(P->d_ll);
    if (P->h_ptrs) cudaFreeHost(P->h_ptrs);
    if (P->dmem) cudaFree(P->dmem);
    delete P;
}

// Bytes of one (root, parity) group of dual-root exchange slots: room for
// the per-slice slots of any slice count up to kMaxSlices (see
// ring_sub_bytes: slices x slot <= largest block + 79 bytes per slice).
static size_t ring_slot(const Plan* P)
{
    const int64_t maxblk = (P->m + P->b - 1) / std::max(P->b, 1);
    return align_up(size_t(maxblk) * P->esize + size_t(kMaxSlices) * 80, 256);
}

static int allocate(Plan* P)
{
    const int p = P->p;
    P->ring_slot_bytes = ring_slot(P);
    size_t off = 0;
    auto carve = [&](size_t bytes) {
        size_t o = off;
        off = align_up(off + bytes, 256);
        return o;
    };
    const size_t o_x = carve(sizeof(void*) * 2 * size_t(p));  // x then y
    const size_t o_tape = carve(P->tape.size());
    const size_t o_lv = carve(sizeof(LevelNode) * std::max<size_t>(P->levels.size(), 1));
    const size_t o_lo = carve(sizeof(int) * P->level_off.size());
    const size_t o_tab = carve(sizeof(int) * 4 * size_t(p));
    const size_t o_err = carve(sizeof(uint32_t) * 4);
    const size_t o_ring = carve(4 * P->ring_slot_bytes);
    P->dmem_bytes = off;
    cudaError_t e = cudaMalloc(&P->dmem, off);
    if (e != cudaSuccess) return cuda_fail(e, "dpdr_plan: cudaMalloc");
    char* base = P->dmem;
    P->d_x = reinterpret_cast<const char**>(base + o_x);
    P->d_y = reinterpret_cast<char**>(base + o_x + sizeof(void*) * size_t(p));
    P->d_tape = reinterpret_cast<uint8_t*>(base + o_tape);
    P->d_levels = reinterpret_cast<LevelNode*>(base + o_lv);
    P->d_level_off = reinterpret_cast<int*>(base + o_lo);
    P->d_tables = reinterpret_cast<int*>(base + o_tab);
    P->d_err = reinterpret_cast<uint32_t*>(base + o_err);
    P->d_ring = base + o_ring;

    std::vector<int> tab(size_t(4) * p);
    std::copy(P->parent.begin(), P->parent.end(), tab.begin());
    std::copy(P->child0.begin(), P->child0.end(), tab.begin() + p);
    std::copy(P->child1.begin(), P->child1.end(), tab.begin() + 2 * p);
    std::copy(P->depth.begin(), P->depth.end(), tab.begin() + 3 * p);
    struct Up { void* dst; const void* src; size_t n; } ups[] = {
        {P->d_tape, P->tape.data(), P->tape.size()},
        {P->d_levels, P->levels.data(), sizeof(LevelNode) * P->levels.size()},
        {P->d_level_off, P->level_off.data(), sizeof(int) * P->level_off.size()},
        {P->d_tables, tab.data(), sizeof(int) * tab.size()},
    };
    for (auto& u : ups) {
        if (!u.n) continue;
        e = cudaMemcpy(u.dst, u.src, u.n, cudaMemcpyHostToDevice);
        if (e != cudaSuccess) return cuda_fail(e, "dpdr_plan: upload");
    }
    e = cudaMemset(P->d_err, 0, sizeof(uint32_t) * 4);
    if (e != cudaSuccess) return cuda_fail(e, "dpdr_plan: memset");

    e = cudaHostAlloc(reinterpret_cast<void**>(&P->h_ptrs),
                      sizeof(void*) * 2 * size_t(p), cudaHostAllocDefault);
    if (e != cudaSuccess) return cuda_fail(e, "dpdr_plan: cudaHostAlloc");
    e = cudaEventCreateWithFlags(&P->staged, cudaEventDisableTiming);
    if (e != cudaSuccess) return cuda_fail(e, "dpdr_plan: event");
    return DPDR_OK;
}

extern "C" dpdr_plan_t dpdr_plan(int p, int64_t m, dpdr_dtype dtype,
                                 dpdr_op op, int b)
{
    return dpdr_plan_topo(p, m, dtype, op, b, DPDR_TOPO_DUAL);
}

extern "C" dpdr_plan_t dpdr_plan_topo(int p, int64_t m, dpdr_dtype dtype, dpdr_op op,
                                      int b, dpdr_topology topo)
{
    if (topo != DPDR_TOPO_DUAL && topo != DPDR_TOPO_SINGLE) {
        fail(DPDR_ERR_INVALID, "dpdr_plan: unknown topology");
        return nullptr;
    }
    if (p < 1 || m < 0) {
        fail(DPDR_ERR_INVALID, "dpdr_plan: need p >= 1 and m >= 0");
        return nullptr;
    }
    const bool sum_ok = (dtype == DPDR_INT32 || dtype == DPDR_FLOAT32) && op == DPDR_OP_SUM;
    const bool mat_ok = (dtype == DPDR_MAT2X2_U32 || dtype == DPDR_MAT2X2_F32) &&
                        op == DPDR_OP_MATMUL;
    if (!sum_ok && !mat_ok) {
        fail(DPDR_ERR_INVALID, "dpdr_plan: unsupported (dtype, op) pair");
        return nullptr;
    }
    if (b < 0) {
        fail(DPDR_ERR_INVALID, "dpdr_plan: b < 0");
        return nullptr;
    }
    Plan* P = new (std::nothrow) Plan;
    if (!P) {
        fail(DPDR_ERR_OOM, "dpdr_plan: host allocation");
        return nullptr;
    }
    P->p = p;
    P->m = m;
    P->topo = topo;
    P->dtype = dtype;
    P->op = op;
    P->esize = (dtype == DPDR_MAT2X2_U32 || dtype == DPDR_MAT2X2_F32) ? 16 : 4;
    build_tables(P);
    if (P->max_depth > kMaxDepth) {
        fail(DPDR_ERR_INVALID, "dpdr_plan: p too large");
        free_plan(P);
        return nullptr;
    }
    cudaError_t e = cudaGetDevice(&P->device);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&P->num_sms, cudaDevAttrMultiProcessorCount, P->device);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&P->l2_bytes, cudaDevAttrL2CacheSize, P->device);
    if (e != cudaSuccess) {
        cuda_fail(e, "dpdr_plan: device query");
        free_plan(P);
        return nullptr;
    }
    // ranks per schedule CTA first: the automatic transport, and with it the
    // default block count, depends on it
    if (schedule_plan_rpc(P) != DPDR_OK) {
        free_plan(P);
        return nullptr;
    }
    P->b = b == 0 ? default_blocks(P) : clamp_b(m, b);
    if (allocate(P) != DPDR_OK || schedule_configure(P) != DPDR_OK ||
        (schedule_transport(P) == 2 && schedule_ll_prepare(P) != DPDR_OK) ||
        fused_tree_prepare(P) != DPDR_OK ||  // small; the host path may use it
        fused_split_prepare(P, false, P->split_depth) != DPDR_OK) {
        free_plan(P);
        return nullptr;
    }
    P->last_x.assign(p, nullptr);
    P->last_y.assign(p, nullptr);
    return reinterpret_cast<dpdr_plan_t>(P);
}

extern "C" int dpdr_plan_query(dpdr_plan_t h, int* parent, int* child0,
                               int* child1, int* dual, int* depth, int* b_used)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_plan_query: NULL plan");
    const std::vector<int>* src[5] = {&P->parent, &P->child0, &P->child1,
                                      &P->dual, &P->depth};
    int* dst[5] = {parent, child0, child1, dual, depth};
    for (int k = 0; k < 5; k++)
        if (dst[k]) std::memcpy(dst[k], src[k]->data(), sizeof(int) * P->p);
    if (b_used) *b_used = P->b;
    return DPDR_OK;
}

extern "C" int dpdr_plan_set(dpdr_plan_t h, int key, int64_t v)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_plan_set: NULL plan");
    switch (key) {
    case DPDR_OPT_FUSED_MODE:
        if (v < 0 || v > 5) return fail(DPDR_ERR_INVALID, "fused mode: 0 to 5");
        if (v == 3) {
            int rc = fused_split_prepare(P, true, P->split_depth);
            if (rc) return rc;
            if (!P->split_ready) return fail(DPDR_ERR_INVALID, "split mode needs p >= 2");
        }
        if (v == 5) {
            int rc = fused_tree_prepare(P);
            if (rc) return rc;
        }
        P->fused_mode = int(v);
        return DPDR_OK;
    case DPDR_OPT_WAIT_LIMIT_NS:
        if (v < 1000) return fail(DPDR_ERR_INVALID, "wait limit below 1 us");
        if (v > kMaxWaitNs) return fail(DPDR_ERR_INVALID, "wait limit above 10 s");
        P->wait_ns = v;
        return DPDR_OK;
    case DPDR_OPT_SKIP_RANK:
        if (v < -1 || v >= P->p) return fail(DPDR_ERR_INVALID, "skip rank out of range");
        P->skip_rank = int(v);
        return DPDR_OK;
    case DPDR_OPT_SCHED_THREADS:
        if (v != 0 && (v < 64 || v > 256 || v % 32))
            return fail(DPDR_ERR_INVALID, "schedule threads: 0 or 64..256, multiple of 32");
        P->sched_threads = int(v);
        return schedule_configure(P);
    case DPDR_OPT_SCHED_RANKS_PER_CTA:
        if (v < 0 || v > P->p) return fail(DPDR_ERR_INVALID, "ranks per CTA out of range");
        P->sched_rpc = int(v);
        return schedule_configure(P);
    case DPDR_OPT_SCHED_LAYOUT: {
        if (v < 0 || v > 2) return fail(DPDR_ERR_INVALID, "schedule layout: 0, 1 or 2");
        const int was = P->sched_layout;
        P->sched_layout = int(v);
        const int rc = schedule_configure(P);
        if (rc) {
            P->sched_layout = was;
            schedule_configure(P);
        }
        return rc;
    }
    case DPDR_OPT_SCHED_COPY:
        if (v < 0 || v > 2) return fail(DPDR_ERR_INVALID, "schedule copy: 0, 1 or 2");
        P->sched_copy = int(v);
        return schedule_configure(P);
    case DPDR_OPT_SCHED_SLICES:
        if (v < 0 || v > kMaxSlices) return fail(DPDR_ERR_INVALID, "slices: 0..1024");
        P->sched_slices = int(v);
        return schedule_configure(P);
    case DPDR_OPT_SPLIT_DEPTH: {
        if (v < -1 || v > P->max_depth) return fail(DPDR_ERR_INVALID, "split depth out of range");
        P->split_depth = int(v);
        return fused_split_prepare(P, true, P->split_depth);
    }
    case DPDR_OPT_SCHED_TRANSPORT: {
        if (v < 0 || v > 2) return fail(DPDR_ERR_INVALID, "schedule transport: 0, 1 or 2");
        const int was = P->sched_transport;
        P->sched_transport = int(v);
        if (schedule_transport(P) == 2) {
            const int rc = schedule_ll_prepare(P);
            if (rc) {
                P->sched_transport = was;
                return rc;
            }
        }
        return schedule_configure(P);
    }
    case DPDR_OPT_HOST_PATH:
        if (v < 0 || v > 2) return fail(DPDR_ERR_INVALID, "host path: 0, 1 or 2");
        P->host_path = int(v);
        return DPDR_OK;
    case DPDR_OPT_HOST_CHUNK_BYTES:
        if (v < 4096) return fail(DPDR_ERR_INVALID, "host chunk below 4096 bytes");
        P->host_chunk = v;
        return DPDR_OK;
    case DPDR_OPT_BLOCKS: {
        if (v < 0) return fail(DPDR_ERR_INVALID, "b < 0");
        const int nb = v == 0 ? default_blocks(P) : clamp_b(P->m, v);
        Plan tmp;
        tmp.m = P->m;
        tmp.b = nb;
        tmp.esize = P->esize;
        if (ring_slot(&tmp) > P->ring_slot_bytes)
            return fail(DPDR_ERR_INVALID,
                        "fewer blocks than the plan was built for: make a new plan");
        P->b = nb;
        return schedule_configure(P);
    }
    default:
        return fail(DPDR_ERR_INVALID, "unknown option");
    }
}

extern "C" int dpdr_plan_info(dpdr_plan_t h, int64_t* info, int n)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P || !info) return fail(DPDR_ERR_INVALID, "dpdr_plan_info: NULL");
    const int64_t v[] = {P->p, P->m, P->b, P->max_depth, fused_auto_mode(P),
                         P->sched_ctas, P->sched_ranks_per_cta,
                         int64_t(P->dmem_bytes + P->d_split_bytes + P->d_sched_bytes +
                                 P->d_ll_bytes + P->tree[0].bytes + P->tree[1].bytes),
                         P->last_vector_path, P->split_s, P->split_nseg, P->split_group,
                         P->sched_slices_used, P->topo, P->last_host_path,
                         schedule_transport(P), P->tree[fused_tree_index(P)].width,
                         P->sched_layout_used, P->sched_copy_used};
    const int k = int(sizeof v / sizeof v[0]);
    for (int i = 0; i < n; i++) info[i] = i < k ? v[i] : 0;
    return DPDR_OK;
}

extern "C" void dpdr_plan_destroy(dpdr_plan_t h)
{
    free_plan(reinterpret_cast<Plan*>(h));
}
