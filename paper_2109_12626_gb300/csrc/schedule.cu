// schedule.cu -- the schedule-faithful persistent kernel of
// dpdr_allreduce_schedule: Algorithm 1 run by every virtual rank.
//
// Rank i runs rounds j = 0..b+d_i (d_i = depth).  Each round has the three
// bidirectional steps of Algorithm 1, in order:
//   child_0 : send final Y[j-(d_i+1)], receive the child's partial Y[j] into
//             t and form Y[j] = t (.) Y[j]
//   child_1 : the same with the second child
//   dual    : (roots) send the partial Y[j], receive the dual's partial t;
//             the lower root forms Y[j] (.) t, the higher t (.) Y[j]
//   parent  : (others) send the partial Y[j], receive final Y[j-d_i]
// Blocks outside [0,b) are empty; an exchange empty both ways is skipped.
//
// On one GPU an exchange is a pair of published blocks in device memory.
// Every rank owns two monotone counters: up[i] = number of partial blocks it
// has published, down[i] = number of final blocks it holds.  A send is a
// release store of the counter after the block is written; a receive is an
// acquire load of the partner's counter followed by reading the partner's
// block straight from the partner's buffer (bulk or per-lane copies into
// shared memory, served by L2), fused with the (.) -- the temporary t of
// Algorithm 1 never materialises in device memory.  Where a
// partial lives: a leaf's partial block j is x_i[j] itself, an inner node's
// is y_i[j], a root's is one of two exchange slots per root (the dual reads
// it while the root overwrites y_r[j] with the final block).  A child
// overwrites its partial y_c[k] with the final block only after its parent
// published final block k, which the parent does after it consumed partial
// k: the data dependencies of the algorithm order every reuse, so a sender
// never waits for its receiver.
//
// A virtual rank is served by nslices CTA groups, one per column slice of
// every pipeline block; slices are independent copies of the schedule (their
// own counters), since (.) acts column by column.  Within a slice, a CTA
// holds up to four rank groups: ranges of whole warps, each with its own
// list of ranks that it runs in increasing order inside each round (see
// Group below).  The host lays them out (schedule_configure): either by
// work, one rank per group with warps in proportion to the rank's block
// passes (a leaf only copies the final block down; an inner node also folds
// its children's partials with its input), or as contiguous rank ranges
// that never straddle the two trees when the ranks outnumber the CTAs.
// Every wait is on a lower rank of the same round, on an earlier round, or
// (roots only) on the dual's partial of the same round, which the dual
// publishes before it waits; the two roots are never in one group.  So with
// all CTAs resident (cooperative launch) the schedule cannot deadlock.
// With one tree (no dual) the root's partial block j is final and is
// published down at once.  Each wait is bounded in time; an expired wait
// records {rank, round, step} in the plan's error word, raises an abort flag
// that ends every other wait, and returns.
//
// Single-use data is marked for early eviction from L2 (an input block is
// read once, by its rank or by the parent of a leaf; a leaf's final block is
// not read again in the call), so that L2 keeps the inner nodes' partial and
// final blocks that their partners read next.
#include <algorithm>
#include <mutex>
#include <vector>

#include "schedule_common.cuh"

namespace dpdr {
namespace {

constexpr int kSchedMaxThreads = sched::kMaxThreads;
constexpr int kAlgoDoubly = 0;       // Algorithm 1 (dpdr_allreduce_schedule)
constexpr int kAlgoReduceBcast = 1;  // reduce, then broadcast (dpdr_allreduce_reduce_bcast)
// Words from one handshake counter to the next: each counter has a 128-byte
// L2 line of its own, so the release stores and polls of different ranks
// never queue on one line (with 4-byte counters side by side, the 32 ranks
// of a line serialised there: 20 % of the time at p = 32).
constexpr int kCtr = 32;
constexpr int kSchedMaxGroups = sched::kMaxGroups;

struct SchedArgs {
    const char* const* x;
    char* const* y;
    const int* parent;
    const int* child0;
    const int* child1;
    const int* depth;
    const int4* groups;    // [nchunks][kSchedMaxGroups] group descriptors
    const int* rank_list;  // the groups' ranks, each group's in increasing order
    uint32_t* up;
    uint32_t* down;
    uint32_t* abort_flag;
    uint32_t* err;
    char* ring;
    int64_t ring_slot;
    int p, b, r0, r1;
    int64_t m, q, rem;
    int64_t wait_ns;
    int skip_rank;
    int vec;
    int nslices;   // CTA groups per rank: each owns one column slice of every block
    int nchunks;   // CTAs per slice (CTA index = slice * nchunks + chunk)
    int slot_bytes;  // shared memory per thread for the block passes (multiple of 16)
};

using sched::ld_acquire;
using sched::ld_relaxed;
using sched::now_ns;
using sched::rank_in;
using sched::rank_out;
using sched::st_release;

__device__ __forceinline__ int64_t blk_start(const SchedArgs& a, int j)
{
    return sched::block_start(a.q, a.rem, j);
}

// Start of column slice g (of nslices) of the element range [s, e): even
// shares, inner boundaries rounded down to a 16-byte vector boundary.
template <int EPV>
__device__ __forceinline__ int64_t slice_at(const SchedArgs& a, int64_t s, int64_t e, int g)
{
    return sched::slice_bound<EPV>(s, e, g, a.nslices);
}

// One counter wait: *ctr >= target; step names the exchange for the error
// record (0 child_0, 1 child_1, 2 dual, 3 parent).
struct Wait {
    const uint32_t* ctr;
    uint32_t target;
    int step;
};

// The threads of a CTA that serve a list of virtual ranks.  A CTA holds up
// to kSchedMaxGroups groups; group k is the thread range [base, base +
// size) of whole warps named by the CTA's descriptor k and runs the rounds
// of its ranks on its own, so a rank that waits for another CTA holds up no
// rank of another group.  At most one group of a CTA has more than one warp
// (the host lays them out so): it synchronises on barrier 0 with its thread
// count, a one-warp group on the warp alone, so the kernel reserves a single
// hardware barrier (more would cap the CTAs per SM).
struct Group {
    int tid;   // thread index within the group
    int size;  // threads in the group
    int id;    // group index within the CTA
    int base;  // first thread of the group in the CTA
};

// This thread's group in CTA chunk `chunk`: descriptor {first, count,
// thread base, threads} (ranks rank_list[first .. first + count)).  False
// for threads outside every group.
__device__ __forceinline__ bool find_group(const SchedArgs& a, int chunk, Group* grp, int* first,
                                           int* count)
{
    const int t = int(threadIdx.x);
#pragma unroll
    for (int k = 0; k < kSchedMaxGroups; k++) {
        const int4 d = __ldg(a.groups + int64_t(chunk) * kSchedMaxGroups + k);
        if (d.y > 0 && t >= d.z && t < d.z + d.w) {
            *grp = Group{t - d.z, d.w, k, d.z};
            *first = d.x;
            *count = d.y;
            return true;
        }
    }
    return false;
}

__device__ __forceinline__ void group_sync(const Group& g)
{
    if (g.size == 32)
        __syncwarp();
    else
        asm volatile("bar.sync 0, %0;" ::"r"(g.size) : "memory");
}

// The group thread that polls counters, and the one that issues release
// stores: different warps when the group has two or more, so that the
// release that ends one step (its fence waits for the step's writes to
// reach L2) and the poll that begins the next run at the same time.
__device__ __forceinline__ int poller_tid(const Group& g) { return g.size >= 64 ? 32 : 0; }

// The poller thread waits until every one of the n counters (n <= 3, the
// same on all its threads) reaches its target, polling them together
// within the plan's time bound; the group learns the outcome through shared
// memory.  Returns false on timeout or abort (then the caller returns from
// the kernel).
__device__ __forceinline__ bool cta_wait(const SchedArgs& a, const Group& grp, const Wait* w,
                                         int n, int rank, int j)
{
    if (n == 0) return true;
    __shared__ int ok_slot[kSchedMaxGroups];
    int& ok = ok_slot[grp.id];
    if (grp.tid == poller_tid(grp)) {
        int r = 1;
        unsigned pending = 0;
        for (int k = 0; k < n; k++)
            if (ld_acquire(w[k].ctr) < w[k].target) pending |= 1u << k;
        if (pending) {
            // poll hot first (a partner is usually a few hundred ns away),
            // then back off gently; every poll checks the time bound
            const uint64_t t0 = now_ns();
            unsigned sleep = 0, polls = 0;
            while (true) {
                for (int k = 0; k < n; k++)
                    if (((pending >> k) & 1u) && ld_acquire(w[k].ctr) >= w[k].target)
                        pending &= ~(1u << k);
                if (!pending) break;
                if ((polls & 15) == 15 && ld_relaxed(a.abort_flag)) { r = 0; break; }
                if (now_ns() - t0 > uint64_t(a.wait_ns)) {
                    if (atomicCAS(a.err, 0u, uint32_t(DPDR_ERR_TIMEOUT)) == 0u) {
                        a.err[1] = uint32_t(rank);
                        a.err[2] = uint32_t(j);
                        a.err[3] = uint32_t(w[__ffs(pending) - 1].step);
                    }
                    __threadfence();
                    atomicExch(a.abort_flag, 1u);
                    r = 0;
                    break;
                }
                if (++polls > 32) {
                    sleep = sleep ? (sleep < 256 ? sleep * 2 : 256) : 32;
                    __nanosleep(sleep);
                }
            }
        }
        ok = r;
    }
    group_sync(grp);
    const int r = ok;
    group_sync(grp);
    return r != 0;
}

// Release the group's writes to the rank's partner(s): the barrier orders
// every thread's block writes before thread 0's gpu-scope release stores
// (release is cumulative over what thread 0 has observed), and the partner's
// acquire load orders its reads after them.  ctr1 may be null.
__device__ __forceinline__ void publish(const SchedArgs& a, const Group& grp, uint32_t* ctr0,
                                        uint32_t v0, uint32_t* ctr1, uint32_t v1, int rank)
{
    group_sync(grp);
    if (grp.tid == 0 && rank != a.skip_rank) {
        st_release(ctr0, v0);
        if (ctr1) st_release(ctr1, v1);
    }
}

// ------------------------------------------------------------ block passes
// A block pass combines up to three rows element by element over [s, e)
// and writes the result to dst:
//   NOPS 1  dst = src0                        (a final block copied down)
//   NOPS 2  dst = src0 (.) src1               (one child's partial with x_i,
//                                              or the dual roots' partials)
//   NOPS 3  dst = src1 (.) (src0 (.) src2)    (Y[j] = t1 (.) (t0 (.) x_i))
// Rows are virtual bases indexed by global element number.  dst may equal
// the last source (in place).  Every thread owns the same elements in every
// pass over the same range.
//
// On the vector path the group moves its 16-byte units through a
// double-buffered region of shared memory (slot_bytes per thread) with TMA
// bulk copies: one thread issues, for every operand, one cp.async.bulk
// of a contiguous chunk into a stage of the region, completing on the
// stage's mbarrier; the group combines the chunk from shared memory,
// stores the result and, once every thread is done with the stage, the
// chunk two ahead goes into it.  A chunk is a few KB, so one instruction
// fetches what 200 lanes would, and whole lines move (per-lane 16-byte
// copies that carry an L2 policy fetch a sector per lane).  Chunks of a few
// KB matter: with four stages per warp of half a KB each, the same passes
// took 1.5 times as long.  Elements outside the 16-byte units (an unaligned
// head and tail, or every element when some buffer is only 4-byte aligned)
// move singly with L2-coherent loads.
//
// Proxies: block data is written with generic stores and read by the TMA
// unit (the async proxy), by this group or by a partner after a counter
// handshake.  Every thread fences its own writes to the async proxy at the
// end of a pass (before the barrier that precedes the release), and the
// issuing thread fences again before its first copy of a pass (after the
// acquire that made a partner's writes visible).
//
// hints: bit o (o < 3) marks operand o as read once in the call, kHintDst
// marks dst as not read again in the call; those accesses take the L2
// evict-first policy.  kHintKeep marks dst as a partial block that a
// partner reads soon and that is then dropped from L2 unwritten: its stores
// take the evict-last policy, so that L2 keeps it until then.
constexpr int kSlotBytes = 192;  // shared memory per thread, at least (both stages)
constexpr unsigned kHintDst = 8;
constexpr unsigned kHintKeep = 16;
// Column slices of at most this many 16-byte units take the per-lane path
// in every pass of a launch (see block_pass).
constexpr int64_t kLaneSliceUnits = 1024;

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                     static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
                 "l"(gmem)
                 : "memory");
}
__device__ __forceinline__ void cp_async_wait_all()
{
    asm volatile("cp.async.commit_group;\ncp.async.wait_group 0;" ::: "memory");
}

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
                 "r"(bytes)
                 : "memory");
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
__device__ __forceinline__ void bulk_load_hint(void* dst, const void* src, uint32_t bytes,
                                               uint64_t* bar, uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
        "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(pol)
        : "memory");
}
__device__ __forceinline__ void fence_proxy_async_global()
{
    asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ uint64_t evict_first_policy()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ uint64_t evict_last_policy()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ void st_l2_hint(void* p, uint4 v, uint64_t pol)
{
    asm volatile("st.global.cg.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p),
                 "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "l"(pol)
                 : "memory");
}

// Wait for phase `parity` of a stage barrier.  A bulk copy of valid memory
// always completes, so this wait only guards against the impossible: past
// the plan's time bound it records a timeout (step 4, the CTA in the rank
// field) and raises the abort flag, then keeps waiting for the copy (its
// data lands in this CTA's shared memory) for at most as long again.
__device__ __forceinline__ void stage_wait(const SchedArgs& a, uint64_t* b, uint32_t parity)
{
    if (mbar_test(b, parity)) return;
    const uint64_t t0 = now_ns();
    bool late = false;
    for (uint32_t it = 1;; it++) {
        if (mbar_test(b, parity)) return;
        if ((it & 63) == 0) {
            const uint64_t dt = now_ns() - t0;
            if (!late && dt > uint64_t(a.wait_ns)) {
                late = true;
                if (atomicCAS(a.err, 0u, uint32_t(DPDR_ERR_TIMEOUT)) == 0u) {
                    a.err[1] = blockIdx.x;
                    a.err[2] = 0;
                    a.err[3] = 4;
                }
                __threadfence();
                atomicExch(a.abort_flag, 1u);
            }
            if (dt > 2 * uint64_t(a.wait_ns)) return;
        }
    }
}

// Per group: the two stage barriers (the parity each thread expects next
// lives in the caller's `sp`, bit k for stage k; every thread of a group
// runs the same passes, so the copies agree).
__shared__ uint64_t sched_stage_bar[sched::kMaxGroups][2];

template <int NOPS, class Op>
__device__ __forceinline__ uint4 combine_units(const uint4* v)
{
    if (NOPS == 1) return v[0];
    if (NOPS == 2) return Op::vec(v[0], v[1]);
    return Op::vec(v[1], Op::vec(v[0], v[2]));
}
template <int NOPS, class Op>
__device__ __forceinline__ Elem<Op> combine_elems(const char* s0, const char* s1, const char* s2,
                                                  int64_t off)
{
    if (NOPS == 1) return ld_one_l2<Op>(s0 + off);
    const Elem<Op> a0 = ld_one_l2<Op>(s0 + off), a1 = ld_one_l2<Op>(s1 + off);
    if (NOPS == 2) return comb<Op>(a0, a1);
    return comb<Op>(a1, comb<Op>(a0, ld_one_l2<Op>(s2 + off)));
}

// Short slices (the kLane kernels, which the host launches when a slice
// holds at most kLaneSliceUnits units): every lane copies its units [vs, ve) into
// private 16-byte slots of the group's region, without an L2 policy (with
// one, adjacent lanes' copies are not merged), waits for its own copies and
// combines; no barrier and no mbarrier round trip.  At 512 units per slice
// this is 8 % faster than the bulk copies, at 2048 units 10 % slower.  The
// two paths are separate kernels: compiled into one, the bulk path lost 2-4 %.
template <class Op, int NOPS>
__device__ __forceinline__ void units_lane(const SchedArgs& a, Group grp, unsigned hints, char* dst,
                                        const char* s0, const char* s1, const char* s2,
                                        int64_t vs, int64_t ve)
{
    extern __shared__ __align__(128) uint4 sched_slots[];
    const int tid = grp.tid, bd = grp.size;
    constexpr int LB = kSlotBytes / 16 / NOPS;  // units per operand per lane and batch
    const uint64_t pol = evict_first_policy();
    const uint64_t keep = evict_last_policy();
    uint4* const my = reinterpret_cast<uint4*>(reinterpret_cast<char*>(sched_slots) +
                                               int64_t(grp.base) * a.slot_bytes) + tid;
    const char* const src[3] = {s0, s1, s2};
    for (int64_t v0 = vs + tid; v0 < ve; v0 += int64_t(LB) * bd) {
#pragma unroll
        for (int t = 0; t < LB; t++) {
            const int64_t v = v0 + int64_t(t) * bd;
            if (v < ve) {
#pragma unroll
                for (int o = 0; o < NOPS; o++) cp_async16(my + (t * NOPS + o) * bd, src[o] + v * 16);
            }
        }
        cp_async_wait_all();
#pragma unroll
        for (int t = 0; t < LB; t++) {
            const int64_t v = v0 + int64_t(t) * bd;
            if (v < ve) {
                uint4 r[NOPS];
#pragma unroll
                for (int o = 0; o < NOPS; o++) r[o] = my[(t * NOPS + o) * bd];
                const uint4 out = combine_units<NOPS, Op>(r);
                if (hints & (kHintDst | kHintKeep))
                    st_l2_hint(dst + v * 16, out, (hints & kHintDst) ? pol : keep);
                else
                    st_l2(dst + v * 16, out);
            }
        }
    }
}

// Units [vs, ve) by bulk copies through the group's double-buffered region.
template <class Op, int NOPS>
__device__ __forceinline__ void units_bulk(const SchedArgs& a, Group grp, unsigned* sp, unsigned hints,
                                        char* dst, const char* s0, const char* s1, const char* s2,
                                        int64_t vs, int64_t ve)
{
    extern __shared__ __align__(128) uint4 sched_slots[];
    const int tid = grp.tid, bd = grp.size;
    const uint64_t pol = evict_first_policy();
    const uint64_t keep = evict_last_policy();
    char* const region = reinterpret_cast<char*>(sched_slots) + int64_t(grp.base) * a.slot_bytes;
    const uint32_t stage = uint32_t(bd) * uint32_t(a.slot_bytes / 2);  // bytes per stage
    const uint32_t C = stage / NOPS / 128 * 128;                       // bytes per operand chunk
    const int64_t uc = C / 16;                                          // units per chunk
    const int64_t nch = (ve - vs + uc - 1) / uc;
    uint64_t* const bars = sched_stage_bar[grp.id];
    const char* const src[3] = {s0, s1, s2};
    auto issue = [&](int64_t k) {
        const int st = int(k & 1);
        const int64_t u0 = vs + k * uc;
        const uint32_t bytes = uint32_t((ve - u0 < uc ? ve - u0 : uc) * 16);
        mbar_expect_tx(&bars[st], uint32_t(NOPS) * bytes);
#pragma unroll
        for (int o = 0; o < NOPS; o++) {
            char* d = region + st * stage + o * C;
            if ((hints >> o) & 1u)
                bulk_load_hint(d, src[o] + u0 * 16, bytes, &bars[st], pol);
            else
                bulk_load(d, src[o] + u0 * 16, bytes, &bars[st]);
        }
    };
    if (tid == 0) {
        fence_proxy_async_global();
        issue(0);
        if (nch > 1) issue(1);
    }
    for (int64_t k = 0; k < nch; k++) {
        const int st = int(k & 1);
        stage_wait(a, &bars[st], (*sp >> st) & 1u);
        *sp ^= 1u << st;
        const int64_t u0 = vs + k * uc;
        const int cnt = int(ve - u0 < uc ? ve - u0 : uc);
        const char* buf = region + st * stage;
        for (int u = tid; u < cnt; u += bd) {
            uint4 r[NOPS];
#pragma unroll
            for (int o = 0; o < NOPS; o++)
                r[o] = *reinterpret_cast<const uint4*>(buf + o * C + u * 16);
            const uint4 out = combine_units<NOPS, Op>(r);
            if (hints & (kHintDst | kHintKeep))
                st_l2_hint(dst + (u0 + u) * 16, out, (hints & kHintDst) ? pol : keep);
            else
                st_l2(dst + (u0 + u) * 16, out);
        }
        if (k + 2 < nch) {
            group_sync(grp);  // the stage is free again
            if (tid == 0) issue(k + 2);
        }
    }
}

template <class Op, int NOPS, bool kLane>
__device__ __noinline__ void block_pass(const SchedArgs& a, Group grp, unsigned* sp,
                                        unsigned hints, char* dst, const char* s0,
                                        const char* s1, const char* s2, int64_t s, int64_t e)
{
    constexpr int EPV = Op::kEpv;
    constexpr int ES = Op::kEsize;
    const int tid = grp.tid, bd = grp.size;
    int64_t vs = 0, ve = 0;
    if (a.vec) {
        vs = (s + EPV - 1) / EPV;
        ve = e / EPV;
        if (vs > ve) vs = ve = 0;
    }
    const int64_t head_end = vs < ve ? vs * EPV : e, tail_beg = vs < ve ? ve * EPV : e;
    for (int pass = 0; pass < 2; pass++) {
        const int64_t b0 = pass ? tail_beg : s, b1 = pass ? e : head_end;
        for (int64_t k = b0 + tid; k < b1; k += bd)
            st_one_l2<Op>(dst + k * ES, combine_elems<NOPS, Op>(s0, s1, s2, k * ES));
    }
    if (vs < ve) {
        if (kLane)
            units_lane<Op, NOPS>(a, grp, hints, dst, s0, s1, s2, vs, ve);
        else
            units_bulk<Op, NOPS>(a, grp, sp, hints, dst, s0, s1, s2, vs, ve);
    }
    fence_proxy_async_global();  // this pass's writes, before the release
    group_sync(grp);
}

// The group's stage barriers, made ready before its first pass; returns the
// parities the first waits expect.
__device__ __forceinline__ unsigned init_stages(const Group& grp)
{
    if (grp.tid == 0) {
        mbar_init(&sched_stage_bar[grp.id][0], 1);
        mbar_init(&sched_stage_bar[grp.id][1], 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    group_sync(grp);
    return 0u;
}

// dst = t1 (.) (t0 (.) x) over [s, e) for the children's partial blocks
// t0, t1 (null when the child does not exist; both null: a copy of x).
// leaf0 / leaf1: the child is a leaf, so its partial block is its input,
// read only here.  x itself is read only here.
// keep: dst is a partial block (kHintKeep).
template <class Op, bool kLane>
__device__ __forceinline__ void fold_children(const SchedArgs& a, const Group& grp, unsigned* sp,
                                              char* dst, const char* t0, const char* t1,
                                              const char* x, bool leaf0, bool leaf1, bool keep,
                                              int64_t s, int64_t e)
{
    const unsigned k = keep ? kHintKeep : 0u;
    if (!t0)
        block_pass<Op, 1, kLane>(a, grp, sp, 1u | k, dst, x, nullptr, nullptr, s, e);
    else if (!t1)
        block_pass<Op, 2, kLane>(a, grp, sp, unsigned(leaf0) | 2u | k, dst, t0, x, nullptr, s, e);
    else
        block_pass<Op, 3, kLane>(a, grp, sp, unsigned(leaf0) | (unsigned(leaf1) << 1) | 4u | k, dst, t0,
                          t1, x, s, e);
}

// An inner child's partial block is dead once its parent has combined it:
// the child overwrites it with the final block later.  Dropping its L2
// lines without write-back keeps the partial from ever reaching device
// memory, so y is written to DRAM once.  Only whole 128-byte lines inside
// [s, e) go: the lines at the ends may hold neighbouring slices' or blocks'
// live data.  Called after a barrier that follows every read of the range;
// the rank's next release orders the discards before the child's final
// write, which waits for a later release of this rank.
template <class Op>
__device__ __noinline__ void discard_consumed(Group grp, const char* row, int64_t s, int64_t e)
{
    const uintptr_t lo = (reinterpret_cast<uintptr_t>(row + s * Op::kEsize) + 127) & ~uintptr_t(127);
    const uintptr_t hi = reinterpret_cast<uintptr_t>(row + e * Op::kEsize) & ~uintptr_t(127);
    for (uintptr_t l = lo + uintptr_t(grp.tid) * 128; l < hi; l += uintptr_t(grp.size) * 128)
        asm volatile("discard.global.L2 [%0], 128;" ::"l"(l) : "memory");
}

__device__ __forceinline__ char* ring_base(const SchedArgs& a, int side, int j, int g,
                                           int64_t s, int epv, int es)
{
    // slot of (root side, block parity, slice g), ring_slot bytes each
    char* slot = a.ring + ((int64_t(side) * 2 + (j & 1)) * a.nslices + g) * a.ring_slot;
    return slot - (s - s % epv) * es;  // element k at slot + (k - s + s % epv) * es
}

// Round j of Algorithm 1 at rank i, column slice g.  The waits for the two
// children's partial blocks do not depend on each other, so they are polled
// together, and Y[j] = t1 (.) (t0 (.) x_i) (child_0's partial first, as the
// steps run) is formed in one pass.  The partial goes up before the wait for
// the parent's final block, so a parent's round j never waits for its own
// round j-1 to reach the child and come back; the release of the partial
// and the poll of the parent's counter run in different warps at once (as
// do the release of the final block and the next round's first poll).
template <class Op, bool kLane>
__device__ __forceinline__ bool run_round(const SchedArgs& a, const Group& grp, unsigned* sp,
                                          int i, int j, int g)
{
    constexpr int EPV = Op::kEpv;
    uint32_t* const up = a.up + int64_t(g) * a.p * kCtr;      // this slice's counters
    uint32_t* const down = a.down + int64_t(g) * a.p * kCtr;
    const int c0 = __ldg(a.child0 + i), c1 = __ldg(a.child1 + i);
    const int par = __ldg(a.parent + i);
    const char* xi = rank_in(a.x, i);
    char* yi = rank_out(a.y, i);
    const bool inb = j < a.b;
    const int64_t bs = inb ? blk_start(a, j) : 0, be = inb ? blk_start(a, j + 1) : 0;
    const int64_t s = slice_at<EPV>(a, bs, be, g), e = slice_at<EPV>(a, bs, be, g + 1);

    // steps 1 and 2: the children's partial blocks (a leaf's is x_c, an inner
    // node's y_c); the send half (final block j-(d+1)) is read by the child
    // itself from y_i once down[i] covers it.  inner0/inner1: the child has
    // children of its own, so its partial lives in y_c and dies here.
    const char* t0 = nullptr;
    const char* t1 = nullptr;
    bool inner0 = false, inner1 = false;
    if (inb && c0 >= 0) {
        inner0 = __ldg(a.child0 + c0) >= 0;
        t0 = inner0 ? rank_in(a.y, c0) : rank_in(a.x, c0);
        Wait w[2];
        w[0] = Wait{up + c0 * kCtr, uint32_t(j + 1), 0};
        if (c1 >= 0) {
            inner1 = __ldg(a.child0 + c1) >= 0;
            t1 = inner1 ? rank_in(a.y, c1) : rank_in(a.x, c1);
            w[1] = Wait{up + c1 * kCtr, uint32_t(j + 1), 1};
        }
        if (!cta_wait(a, grp, w, c1 >= 0 ? 2 : 1, i, j)) return false;
    }

    if (par < 0 && a.r0 >= 0) {  // step 3 at a root: exchange partials with the dual
        if (!inb) return true;
        const int side = (i == a.r0) ? 0 : 1;
        char* slot = ring_base(a, side, j, g, s, EPV, Op::kEsize);
        fold_children<Op, kLane>(a, grp, sp, slot, t0, t1, xi, !inner0, !inner1, true, s, e);
        publish(a, grp, up + i * kCtr, uint32_t(j + 1), nullptr, 0, i);
        if (inner0) discard_consumed<Op>(grp, t0, s, e);
        if (inner1) discard_consumed<Op>(grp, t1, s, e);
        const int du = (i == a.r0) ? a.r1 : a.r0;
        const Wait wd{up + du * kCtr, uint32_t(j + 1), 2};
        if (!cta_wait(a, grp, &wd, 1, i, j)) return false;
        const char* other = ring_base(a, 1 - side, j, g, s, EPV, Op::kEsize);
        // lower root: Y[j] (.) t; higher root: t (.) Y[j]; a root without
        // children (p == 2) is a leaf: its final block is not read again
        const unsigned h = c0 < 0 ? kHintDst : 0u;
        if (i == a.r0)
            block_pass<Op, 2, kLane>(a, grp, sp, h, yi, slot, other, nullptr, s, e);
        else
            block_pass<Op, 2, kLane>(a, grp, sp, h, yi, other, slot, nullptr, s, e);
        publish(a, grp, down + i * kCtr, uint32_t(j + 1), nullptr, 0, i);
        return true;
    }
    if (par < 0) {  // the root of a single tree (or p == 1): its block is final
        if (!inb) return true;
        if (t0 || xi != yi)
            fold_children<Op, kLane>(a, grp, sp, yi, t0, t1, xi, !inner0, !inner1, false, s, e);
        publish(a, grp, down + i * kCtr, uint32_t(j + 1), nullptr, 0, i);
        if (inner0) discard_consumed<Op>(grp, t0, s, e);
        if (inner1) discard_consumed<Op>(grp, t1, s, e);
        return true;
    }
    // step 3 elsewhere: partial Y[j] up (in y_i, or x_i itself for a leaf),
    // final Y[j-d] down from the parent.  A leaf's partial block is its
    // input, unchanged during the call, so its counter only tells the parent
    // that the step was taken: a relaxed store, no fence.  (In place, the
    // leaf overwrites x_i block k only after the parent has published final
    // block k, which follows the parent's read of x_i block k.)
    if (inb) {
        if (c0 < 0) {
            if (grp.tid == 0 && i != a.skip_rank) sched::st_relaxed(up + i * kCtr, uint32_t(j + 1));
        } else {
            fold_children<Op, kLane>(a, grp, sp, yi, t0, t1, xi, !inner0, !inner1, true, s, e);
            publish(a, grp, up + i * kCtr, uint32_t(j + 1), nullptr, 0, i);
            if (inner0) discard_consumed<Op>(grp, t0, s, e);
            if (inner1) discard_consumed<Op>(grp, t1, s, e);
        }
    }
    const int kf = j - __ldg(a.depth + i);
    if (kf >= 0 && kf < a.b) {
        const Wait wp{down + par * kCtr, uint32_t(kf + 1), 3};
        if (!cta_wait(a, grp, &wp, 1, i, j)) return false;
        const int64_t ks = blk_start(a, kf), ke = blk_start(a, kf + 1);
        // a leaf's final block is not read again in this call, and no rank
        // waits for a leaf's down counter
        block_pass<Op, 1, kLane>(a, grp, sp, c0 < 0 ? kHintDst : 0u, yi, rank_in(a.y, par), nullptr, nullptr,
                          slice_at<EPV>(a, ks, ke, g), slice_at<EPV>(a, ks, ke, g + 1));
        if (c0 >= 0) publish(a, grp, down + i * kCtr, uint32_t(kf + 1), nullptr, 0, i);
    }
    return true;
}

template <class Op, bool kLane>
__global__ void __launch_bounds__(kSchedMaxThreads, 4) schedule_kernel(SchedArgs a)
{
    const int g = blockIdx.x / a.nchunks, chunk = blockIdx.x % a.nchunks;
    Group grp;
    int first = 0, count = 0;
    if (!find_group(a, chunk, &grp, &first, &count)) return;  // warps outside every group
    unsigned sp = init_stages(grp);
    const int* ranks = a.rank_list + first;
    int rounds = 0;
    for (int k = 0; k < count; k++) rounds = max(rounds, a.b + __ldg(a.depth + __ldg(ranks + k)));
    for (int j = 0; j <= rounds; j++) {
        for (int k = 0; k < count; k++) {
            const int i = __ldg(ranks + k);
            if (j > a.b + __ldg(a.depth + i)) continue;
            if (!run_round<Op, kLane>(a, grp, &sp, i, j, g)) return;
        }
    }
}

// ------------------------------------------------- reduce, then broadcast
// The alternative the paper's analysis and experiment compare Algorithm 1
// with (Sec. 1.2, the reduction to the root followed by a broadcast, both
// pipelined on binary trees; Sec. 2, item 3): on the one-tree plan, every
// virtual rank first takes part in a pipelined reduction of the b blocks to
// the root p-1, then in a pipelined broadcast of them from it.  Each phase
// moves blocks in one direction only.  The same handshakes, block passes and
// column slices as Algorithm 1's kernel:
//   reduction, j = 0..b-1: wait for the children's partial blocks j (a
//     leaf's is its input x_c, published whole at once), form
//     Y[j] = t1 (.) (t0 (.) x_i) in y_i and publish it to the parent (at the
//     root Y[j] is final);
//   broadcast, j = 0..b-1: wait for the parent's final block j, copy it into
//     y_i and publish it to the children (the root publishes all b blocks
//     once its reduction is done).
// A rank group runs its ranks in increasing order in the reduction (every
// wait is on a child, a lower rank) and in decreasing order in the
// broadcast (every wait is on the parent, a higher rank); no reduction wait
// depends on a broadcast, so with all CTAs resident nothing deadlocks.  An
// inner child's partial block j is consumed once, by its parent, before the
// root's reduction ends, and overwritten by the final block only after it.
template <class Op, bool kLane>
__device__ __forceinline__ bool reduce_step(const SchedArgs& a, const Group& grp, unsigned* sp,
                                            int i, int j, int g)
{
    constexpr int EPV = Op::kEpv;
    uint32_t* const up = a.up + int64_t(g) * a.p * kCtr;
    const int c0 = __ldg(a.child0 + i), c1 = __ldg(a.child1 + i);
    const int par = __ldg(a.parent + i);
    const char* xi = rank_in(a.x, i);
    char* yi = rank_out(a.y, i);
    const int64_t bs = blk_start(a, j), be = blk_start(a, j + 1);
    const int64_t s = slice_at<EPV>(a, bs, be, g), e = slice_at<EPV>(a, bs, be, g + 1);
    if (c0 < 0) {
        if (par >= 0) {
            // a leaf: its partial blocks are its input, there from the start
            if (j == 0 && grp.tid == 0 && i != a.skip_rank)
                sched::st_relaxed(up + i * kCtr, uint32_t(a.b));
        } else if (xi != yi) {
            block_pass<Op, 1, kLane>(a, grp, sp, 1u | kHintDst, yi, xi, nullptr, nullptr, s, e);  // p == 1
        }
        return true;
    }
    const bool inner0 = __ldg(a.child0 + c0) >= 0;
    const char* t0 = inner0 ? rank_in(a.y, c0) : rank_in(a.x, c0);
    const char* t1 = nullptr;
    bool inner1 = false;
    Wait w[2];
    w[0] = Wait{up + c0 * kCtr, uint32_t(j + 1), 0};
    if (c1 >= 0) {
        inner1 = __ldg(a.child0 + c1) >= 0;
        t1 = inner1 ? rank_in(a.y, c1) : rank_in(a.x, c1);
        w[1] = Wait{up + c1 * kCtr, uint32_t(j + 1), 1};
    }
    if (!cta_wait(a, grp, w, c1 >= 0 ? 2 : 1, i, j)) return false;
    fold_children<Op, kLane>(a, grp, sp, yi, t0, t1, xi, !inner0, !inner1, par >= 0, s, e);
    if (par >= 0)
        publish(a, grp, up + i * kCtr, uint32_t(j + 1), nullptr, 0, i);
    else
        group_sync(grp);  // the discards below follow every read
    if (inner0) discard_consumed<Op>(grp, t0, s, e);
    if (inner1) discard_consumed<Op>(grp, t1, s, e);
    return true;
}

template <class Op, bool kLane>
__device__ __forceinline__ bool bcast_step(const SchedArgs& a, const Group& grp, unsigned* sp,
                                           int i, int j, int g)
{
    constexpr int EPV = Op::kEpv;
    uint32_t* const down = a.down + int64_t(g) * a.p * kCtr;
    const int par = __ldg(a.parent + i);
    if (par < 0) {  // the root holds every block: all of them go out at once
        if (j == 0) publish(a, grp, down + i * kCtr, uint32_t(a.b), nullptr, 0, i);
        return true;
    }
    const Wait wp{down + par * kCtr, uint32_t(j + 1), 3};
    if (!cta_wait(a, grp, &wp, 1, i, j)) return false;
    const int64_t bs = blk_start(a, j), be = blk_start(a, j + 1);
    const bool leaf = __ldg(a.child0 + i) < 0;
    block_pass<Op, 1, kLane>(a, grp, sp, leaf ? kHintDst : 0u, rank_out(a.y, i), rank_in(a.y, par),
                      nullptr, nullptr, slice_at<EPV>(a, bs, be, g), slice_at<EPV>(a, bs, be, g + 1));
    if (!leaf) publish(a, grp, down + i * kCtr, uint32_t(j + 1), nullptr, 0, i);  // no one waits on a leaf
    return true;
}

template <class Op, bool kLane>
__global__ void __launch_bounds__(kSchedMaxThreads, 4) reduce_bcast_kernel(SchedArgs a)
{
    const int g = blockIdx.x / a.nchunks, chunk = blockIdx.x % a.nchunks;
    Group grp;
    int first = 0, count = 0;
    if (!find_group(a, chunk, &grp, &first, &count)) return;  // warps outside every group
    unsigned sp = init_stages(grp);
    const int* ranks = a.rank_list + first;
    for (int j = 0; j < a.b; j++)
        for (int k = 0; k < count; k++)
            if (!reduce_step<Op, kLane>(a, grp, &sp, __ldg(ranks + k), j, g)) return;
    for (int j = 0; j < a.b; j++)
        for (int k = count - 1; k >= 0; k--)
            if (!bcast_step<Op, kLane>(a, grp, &sp, __ldg(ranks + k), j, g)) return;
}

template <class Op>
const void* kernel_ptr(int algo, bool lane)
{
    if (algo == kAlgoReduceBcast)
        return lane ? reinterpret_cast<const void*>(&reduce_bcast_kernel<Op, true>)
                    : reinterpret_cast<const void*>(&reduce_bcast_kernel<Op, false>);
    return lane ? reinterpret_cast<const void*>(&schedule_kernel<Op, true>)
                : reinterpret_cast<const void*>(&schedule_kernel<Op, false>);
}

// Algorithm 1's kernel (algo kAlgoDoubly) or the reduction then broadcast,
// with per-lane (lane) or bulk copies in its block passes.
const void* kernel_for(int dtype, int algo = kAlgoDoubly, bool lane = false)
{
    switch (dtype) {
    case DPDR_INT32: return kernel_ptr<SumI32>(algo, lane);
    case DPDR_FLOAT32: return kernel_ptr<SumF32>(algo, lane);
    case DPDR_MAT2X2_F32: return kernel_ptr<MatF32>(algo, lane);
    default: return kernel_ptr<MatU32>(algo, lane);
    }
}

// Shared memory per thread of the counters kernels' block passes at
// `threads` threads: what the SM has left once the CTAs that the 64-register
// budget allows are resident (each with its reserved and static shared
// memory), in 16-byte steps, at least kSlotBytes.
cudaError_t sched_slot_bytes(int dtype, int threads, int* slot)
{
    int dev = 0, per_sm = 0, reserved = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev);
    if (e == cudaSuccess)
        e = cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev);
    size_t stat = 0;
    for (int algo : {kAlgoDoubly, kAlgoReduceBcast})
        for (bool lane : {false, true}) {
            cudaFuncAttributes fa;
            if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, kernel_for(dtype, algo, lane));
            if (e == cudaSuccess) stat = std::max(stat, fa.sharedSizeBytes);
        }
    if (e != cudaSuccess) return e;
    const int ctas = std::max(1, 65536 / (64 * threads));
    const int64_t per = (int64_t(per_sm) / ctas - reserved - int64_t(stat)) / threads / 16 * 16;
    *slot = int(std::max<int64_t>(kSlotBytes, std::min<int64_t>(per, 512)));
    return cudaSuccess;
}

// The counters kernels' dynamic shared memory for CTAs of `threads`
// threads with `slot` bytes per thread.  Beyond 48 KB less the kernels'
// static shared memory the kernels must be granted the size first.
cudaError_t sched_smem(int dtype, int threads, int slot, size_t* bytes)
{
    *bytes = size_t(threads) * size_t(slot);
    if (*bytes + 1024 <= 48 * 1024) return cudaSuccess;
    cudaError_t e = cudaSuccess;
    for (int algo : {kAlgoDoubly, kAlgoReduceBcast})
        for (bool lane : {false, true})
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(kernel_for(dtype, algo, lane),
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(*bytes));
    return e;
}

// CTAs of `threads` threads that fit one SM for the counters kernels (with
// `slot` bytes of shared memory per thread) and the flagged-word kernel
// alike.
cudaError_t sched_occupancy(int dtype, int threads, int slot, int* occ)
{
    int o[5] = {0, 0, 0, 0, 0};
    size_t smem = 0;
    cudaError_t e = sched_smem(dtype, threads, slot, &smem);
    for (int algo : {kAlgoDoubly, kAlgoReduceBcast})
        for (int lane = 0; lane < 2; lane++)
            if (e == cudaSuccess)
                e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
                    &o[2 * algo + lane], kernel_for(dtype, algo, lane != 0), threads, smem);
    if (e == cudaSuccess)
        e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&o[4], schedule_ll_kernel_for(dtype),
                                                          threads, 0);
    *occ = *std::min_element(o, o + 5);
    return e;
}
cudaError_t sched_occupancy(int dtype, int threads, int* occ)
{
    int slot = kSlotBytes;
    cudaError_t e = sched_slot_bytes(dtype, threads, &slot);
    return e == cudaSuccess ? sched_occupancy(dtype, threads, slot, occ) : e;
}

// The CTAs of one column slice, as group descriptors {first, count, thread
// base, threads} (kSchedMaxGroups per CTA; count 0 = no group) over a list
// of ranks.
struct SchedLayout {
    std::vector<int4> groups;
    std::vector<int> ranks;
    int max_ranks = 0;  // most ranks in one CTA
    int ctas() const { return int(groups.size() / kSchedMaxGroups); }
    // one CTA of `threads` threads: its groups' rank lists and the warps of
    // each group (default: one warp for every group but the first, which
    // takes the rest -- at most one group of a CTA may span several warps)
    void add(const std::vector<std::vector<int>>& lists, int threads,
             const std::vector<int>& warps = {})
    {
        const int W = threads / 32, n = int(lists.size());
        int base = 0, total = 0;
        for (int k = 0; k < kSchedMaxGroups; k++) {
            if (k >= n) {
                groups.push_back(make_int4(0, 0, 0, 0));
                continue;
            }
            const int w = warps.empty() ? (k == 0 ? W - n + 1 : 1) : warps[k];
            groups.push_back(make_int4(int(ranks.size()), int(lists[k].size()), base, 32 * w));
            ranks.insert(ranks.end(), lists[k].begin(), lists[k].end());
            base += 32 * w;
            total += int(lists[k].size());
        }
        max_ranks = std::max(max_ranks, total);
    }
};

// Contiguous rank ranges of R ranks (never straddling the two trees), each
// CTA's warps split into min(R, warps, kSchedMaxGroups) groups that run
// contiguous shares of the range.
void layout_ranges(int p, int n0, int R, int threads, SchedLayout* L)
{
    const int ng = sched::group_count(R, threads);
    auto cta = [&](int lo, int hi) {
        const int n = hi - lo, k = std::min(n, ng);
        std::vector<std::vector<int>> lists(k);
        for (int g = 0; g < k; g++)
            for (int i = lo + n * g / k; i < lo + n * (g + 1) / k; i++) lists[g].push_back(i);
        L->add(lists, threads);
    };
    for (int lo = 0; lo < n0; lo += R) cta(lo, std::min(lo + R, n0));
    for (int lo = n0; lo < p; lo += R) cta(lo, std::min(lo + R, p));
}

// Work-balanced layout, one rank per group.  Per round a leaf copies its
// parent's final block (two block streams), an inner node also folds its
// children's partial blocks with its input (six streams), a dual root folds
// and combines with the dual (seven).  So a leaf gets one warp and an inner
// node the rest of the CTA (three warps of 128 threads), side by side, and
// each root a CTA of its own; leaves left over share CTAs, up to four to a
// CTA.  False when those CTAs, one per slice, do not fit `kmax`.
bool layout_balanced(const Plan* P, int threads, int64_t kmax, SchedLayout* L)
{
    const int W = threads / 32, wl = 1, wi = W - wl;
    if (wi < 1) return false;
    std::vector<int> leaves, inner, roots;
    for (int i = 0; i < P->p; i++) {
        if (P->parent[i] < 0)
            roots.push_back(i);
        else if (P->child0[i] < 0)
            leaves.push_back(i);
        else
            inner.push_back(i);
    }
    const size_t pairs = std::min(leaves.size(), inner.size());
    const size_t spare = leaves.size() - pairs;
    const int per = std::min(kSchedMaxGroups, W);
    const int64_t ctas = int64_t(roots.size() + inner.size()) + int64_t((spare + per - 1) / per);
    if (ctas > kmax) return false;
    for (int r : roots) L->add({{r}}, threads);
    for (size_t k = 0; k < pairs; k++) L->add({{leaves[k]}, {inner[k]}}, threads, {wl, wi});
    for (size_t k = pairs; k < inner.size(); k++) L->add({{inner[k]}}, threads);
    for (size_t k = pairs; k < leaves.size(); k += per) {
        std::vector<std::vector<int>> lists;
        for (size_t t = k; t < std::min(leaves.size(), k + per); t++) lists.push_back({leaves[t]});
        L->add(lists, threads);
    }
    return true;
}

}  // namespace

// Ranks per CTA and co-resident CTAs of the contiguous layout: the fewest
// ranks per CTA (none straddling the trees) with which every CTA -- times
// the slices a fixed DPDR_OPT_SCHED_SLICES asks for -- fits at once.
static int schedule_rpc(const Plan* P, int threads, int* R_out, int64_t* kmax_out)
{
    int occ = 0;
    cudaError_t e = sched_occupancy(P->dtype, threads, &occ);
    if (e != cudaSuccess) return cuda_fail(e, "schedule occupancy");
    const int64_t kmax = int64_t(occ) * P->num_sms;
    const int n0 = P->r0 >= 0 ? P->p / 2 : 0, n1 = P->p - n0;
    auto ctas = [&](int r) { return (n0 + r - 1) / r + (n1 + r - 1) / r; };
    const int64_t per_chunk = std::max(1, P->sched_slices);
    int R = P->sched_rpc;
    if (R == 0) {
        R = 1;
        while (R < P->p && ctas(R) * per_chunk > kmax) R++;
    }
    *R_out = R;
    if (kmax_out) *kmax_out = kmax;
    return DPDR_OK;
}

// Threads per CTA: the option's value, else 128 for the layout that decides
// the transport (the flagged-word kernel's choice was measured with it) and
// for that kernel.
static int reference_threads(const Plan* P) { return P->sched_threads ? P->sched_threads : 128; }

int schedule_plan_rpc(Plan* P)
{
    int rc = schedule_rpc(P, reference_threads(P), &P->sched_rpc_ref, nullptr);
    P->sched_ranks_per_cta = P->sched_rpc_ref;
    P->sched_threads_used = reference_threads(P);
    return rc;
}

// The CTA layout, chosen so that every CTA can be resident at once, and
// the device tables for it: ranks per CTA and, when the GPU has room for
// more CTAs than one slice needs, CTA groups per rank (column slices of at
// least 1024 elements with counters, one word batch per thread with
// flagged words).  The flagged-word kernel takes contiguous rank ranges
// (chunk -> first rank table); the counters kernels take group descriptors:
// the work-balanced layout (128 threads) where one slice of it fits,
// unless DPDR_OPT_SCHED_LAYOUT or DPDR_OPT_SCHED_RANKS_PER_CTA asks for
// rank ranges, else rank ranges (64 threads, the handshake-latency bound
// rounds then run twice the column slices).
int schedule_configure(Plan* P)
{
    int R = 1;
    int64_t kmax = 0;
    int threads = reference_threads(P);
    int rc = schedule_rpc(P, threads, &R, &kmax);
    if (rc) return rc;
    P->sched_rpc_ref = R;  // the transport choice depends on it
    const int n0 = P->r0 >= 0 ? P->p / 2 : 0;  // rank ranges never straddle the trees
    const bool words = schedule_transport(P) == 2;
    SchedLayout L;
    int layout = 1;
    if (!words) {
        const bool try_balanced = P->sched_layout != 1 && P->sched_rpc == 0 &&
                                  (P->sched_threads == 0 || P->sched_threads >= 64);
        if (try_balanced) {
            const int t = P->sched_threads ? P->sched_threads : 128;
            int occ = 0;
            cudaError_t e = sched_occupancy(P->dtype, t, &occ);
            if (e != cudaSuccess) return cuda_fail(e, "schedule occupancy");
            const int64_t k = int64_t(occ) * P->num_sms / std::max(1, P->sched_slices);
            if (layout_balanced(P, t, k, &L)) {
                layout = 2;
                threads = t;
                kmax = int64_t(occ) * P->num_sms;
            }
        }
        if (layout == 1 && try_balanced && P->sched_layout == 2)
            return fail(DPDR_ERR_INVALID, "schedule layout 2: one slice of it does not fit");
        if (layout == 1) {
            // counters kernel with rank ranges: 64 threads unless set
            if (P->sched_threads == 0) {
                threads = 64;
                rc = schedule_rpc(P, threads, &R, &kmax);
                if (rc) return rc;
            }
            layout_ranges(P->p, n0, R, threads, &L);
        }
    } else {
        // the reduce-then-broadcast kernel runs on counters whatever the
        // transport: descriptors of the flagged-word kernel's rank ranges
        layout_ranges(P->p, n0, R, threads, &L);
    }
    std::vector<int> first;
    for (int lo = 0; lo < n0; lo += R) first.push_back(lo);
    for (int lo = n0; lo < P->p; lo += R) first.push_back(lo);
    first.push_back(P->p);
    const int nchunks = words ? int(first.size()) - 1 : L.ctas();
    int G = P->sched_slices;
    if (G == 0) {
        // counters: slices of at least 1024 elements; flagged words: one
        // batch of words per thread
        const int64_t blk = (P->m + P->b - 1) / std::max(P->b, 1);
        const int64_t room = std::max<int64_t>(1, kmax / nchunks);
        const int64_t want = words
            ? (blk + schedule_ll_slice_elems(P) - 1) / schedule_ll_slice_elems(P)
            : blk / 1024;
        G = int(std::max<int64_t>(1, std::min<int64_t>({room, want, 64})));
    }
    const size_t words_n = (2 * size_t(P->p) * G + 1) * kCtr;
    const size_t off_first = (words_n * sizeof(uint32_t) + 255) / 256 * 256;
    const size_t off_groups = (off_first + sizeof(int) * first.size() + 255) / 256 * 256;
    const size_t off_ranks = off_groups + sizeof(int4) * L.groups.size();
    const size_t bytes = off_ranks + sizeof(int) * L.ranks.size() + 16;
    cudaError_t e;
    if (bytes > P->d_sched_bytes) {
        if (P->d_sched) cudaFree(P->d_sched);
        P->d_sched = nullptr;
        P->d_sched_bytes = 0;
        e = cudaMalloc(&P->d_sched, bytes);
        if (e != cudaSuccess) return cuda_fail(e, "schedule counters: cudaMalloc");
        P->d_sched_bytes = bytes;
    }
    P->d_ctrl = reinterpret_cast<uint32_t*>(P->d_sched);
    P->d_cta_first = reinterpret_cast<int*>(P->d_sched + off_first);
    P->d_groups = reinterpret_cast<int4*>(P->d_sched + off_groups);
    P->d_rank_list = reinterpret_cast<int*>(P->d_sched + off_ranks);
    P->sched_slices_used = G;
    P->sched_chunks = nchunks;
    P->sched_ctas = nchunks * G;
    {
        // block passes: per-lane copies while the largest slice of the largest
        // block holds at most kLaneSliceUnits 16-byte units, else bulk copies
        const int64_t maxblk = (P->m + P->b - 1) / std::max(P->b, 1);
        const int64_t units = (maxblk * int64_t(P->esize) + 15) / 16;
        P->sched_copy_used = P->sched_copy ? P->sched_copy
                                           : (units <= kLaneSliceUnits * G ? 1 : 2);
    }
    P->sched_layout_used = words ? 1 : layout;
    P->sched_threads_used = threads;
    {
        const cudaError_t es = sched_slot_bytes(P->dtype, threads, &P->sched_slot_bytes);
        if (es != cudaSuccess) return cuda_fail(es, "schedule shared memory");
    }
    P->sched_ranks_per_cta = words || layout == 1 ? R : L.max_ranks;
    e = cudaMemcpy(P->d_cta_first, first.data(), sizeof(int) * first.size(),
                   cudaMemcpyHostToDevice);
    if (e == cudaSuccess && !L.groups.empty())
        e = cudaMemcpy(P->d_groups, L.groups.data(), sizeof(int4) * L.groups.size(),
                       cudaMemcpyHostToDevice);
    if (e == cudaSuccess && !L.ranks.empty())
        e = cudaMemcpy(P->d_rank_list, L.ranks.data(), sizeof(int) * L.ranks.size(),
                       cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "schedule table upload");
    // the automatic transport may have changed with the layout
    return words ? schedule_ll_prepare(P) : DPDR_OK;
}

int schedule_launch(Plan* P, cudaStream_t s, int algo)
{
    if (P->m == 0) return DPDR_OK;
    SchedArgs a;
    a.x = P->d_x;
    a.y = P->d_y;
    a.parent = P->d_tables;
    a.child0 = P->d_tables + P->p;
    a.child1 = P->d_tables + 2 * P->p;
    a.depth = P->d_tables + 3 * P->p;
    a.groups = P->d_groups;
    a.rank_list = P->d_rank_list;
    const int64_t cw = int64_t(P->p) * P->sched_slices_used;
    a.up = P->d_ctrl;
    a.down = P->d_ctrl + cw * kCtr;
    a.abort_flag = P->d_ctrl + 2 * cw * kCtr;
    a.err = P->d_err;
    a.ring = P->d_ring;
    a.ring_slot = int64_t(ring_sub_bytes((P->m + P->b - 1) / P->b, P->esize, P->sched_slices_used));
    if (size_t(a.ring_slot) * P->sched_slices_used > P->ring_slot_bytes)
        return fail(DPDR_ERR_INVALID, "schedule: exchange slots too small for the slice count");
    a.p = P->p;
    a.b = P->b;
    a.r0 = P->r0;
    a.r1 = P->r1;
    a.m = P->m;
    a.q = P->m / P->b;
    a.rem = P->m % P->b;
    a.wait_ns = P->wait_ns;
    a.skip_rank = P->skip_rank;
    a.vec = P->last_vector_path;
    a.nslices = P->sched_slices_used;
    a.nchunks = P->sched_chunks;
    a.slot_bytes = P->sched_slot_bytes;

    cudaError_t e = cudaMemsetAsync(P->d_ctrl, 0, sizeof(uint32_t) * (2 * size_t(cw) + 1) * kCtr, s);
    if (e != cudaSuccess) return cuda_fail(e, "schedule counter reset");
    size_t smem = 0;
    e = sched_smem(P->dtype, P->sched_threads_used, P->sched_slot_bytes, &smem);
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel shared memory");
    void* args[] = {&a};
    e = cudaLaunchCooperativeKernel(kernel_for(P->dtype, algo, P->sched_copy_used == 1),
                                    dim3(P->sched_ctas),
                                    dim3(P->sched_threads_used), args, smem, s);
    if (e == cudaErrorCooperativeLaunchTooLarge) {
        cudaGetLastError();
        return fail(DPDR_ERR_NOT_COOPERATIVE, "schedule kernel: CTAs cannot be co-resident");
    }
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel launch");
    return DPDR_OK;
}


// ------------------------------------------------------------- no-alloc
// dpdr_allreduce_schedule_noalloc runs the schedule kernel above for
// callers that cannot allocate device memory.  Everything the kernel needs
// besides the caller's rank buffers -- the rank-pointer tables, the tree
// tables, the CTA group tables, the handshake counters, the error word and the
// dual roots' exchange slots -- lives in one file-scope device array that
// exists on every GPU that loads this library until the process exits.
// All calls share it, so two calls that overlap on the GPU race.
constexpr size_t kNoAllocBytes = size_t(DPDR_NOALLOC_SCRATCH_BYTES);
constexpr int kNoAllocMaxRanks = DPDR_NOALLOC_MAX_RANKS;
constexpr int kNoAllocThreads = 128;
constexpr int kNoAllocMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocBytes];

namespace {

// Offsets inside the scratch array (bytes), for p ranks.
struct NoAllocLayout {
    size_t x, y, tables, ctrl, err, groups, ranks, ring, slot, end;
};

__host__ __device__ inline size_t na_align(size_t v) { return (v + 255) / 256 * 256; }

inline NoAllocLayout noalloc_layout(int p, int64_t m, int b, size_t esize)
{
    NoAllocLayout L;
    L.x = 0;
    L.y = na_align(L.x + sizeof(void*) * size_t(p));
    L.tables = na_align(L.y + sizeof(void*) * size_t(p));
    L.ctrl = na_align(L.tables + sizeof(int) * 4 * size_t(p));
    L.err = na_align(L.ctrl + sizeof(uint32_t) * (2 * size_t(p) + 1) * kCtr);
    L.groups = na_align(L.err + sizeof(uint32_t) * 4);
    L.ranks = na_align(L.groups + sizeof(int4) * kSchedMaxGroups * size_t(p));
    L.ring = na_align(L.ranks + sizeof(int) * size_t(p));
    L.slot = na_align(ring_sub_bytes((m + b - 1) / b, esize, 1));
    L.end = L.ring + 4 * L.slot;
    return L;
}

// The complete-binary-tree split of a post-order interval of n ranks: the
// size of the left (lower-ranked) subtree.
__device__ __forceinline__ int left_size(int n)
{
    int H = 0;
    while ((2 << H) <= n) H++;
    const int half = 1 << (H - 1);
    const int last = n - ((1 << H) - 1);
    return (half - 1) + (last < half ? last : half);
}

// One thread per rank: parent, child0, child1 and depth by descending from
// the root of the rank's tree, and the identity rank list; the first nctas
// threads also write their CTA's group descriptors (R ranks per CTA, never
// straddling the trees, split into min(R, ng) groups that run contiguous
// shares of them: one warp each but the first, which takes the rest).
__global__ void noalloc_tables_kernel(int p, int R, int ng, int nctas, int* tables, int4* groups,
                                      int* rank_list)
{
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    const int n0 = p / 2;
    if (i < p) {
        int lo = i < n0 ? 0 : n0, n = i < n0 ? n0 : p - n0;
        int par = -1, d = 0;
        while (true) {
            const int root = lo + n - 1;
            if (i == root) break;
            const int L = left_size(n);
            par = root;
            d++;
            if (i < lo + L) {
                n = L;
            } else {
                lo += L;
                n = n - 1 - L;
            }
        }
        int c0 = -1, c1 = -1;
        if (n > 1) {
            const int L = left_size(n);
            c0 = i - 1;
            c1 = (n - 1 - L > 0) ? lo + L - 1 : -1;
        }
        tables[i] = par;
        tables[p + i] = c0;
        tables[2 * p + i] = c1;
        tables[3 * p + i] = d;
        rank_list[i] = i;
    }
    if (i < nctas) {
        const int k0 = (n0 + R - 1) / R;
        const int lo = i < k0 ? i * R : n0 + (i - k0) * R;
        const int hi = min(lo + R, i < k0 ? n0 : p);
        const int n = hi - lo, k = min(n, ng), W = kNoAllocThreads / 32;
        int base = 0;
        for (int g = 0; g < kSchedMaxGroups; g++) {
            if (g >= k) {
                groups[i * kSchedMaxGroups + g] = make_int4(0, 0, 0, 0);
                continue;
            }
            const int f = lo + n * g / k, l = lo + n * (g + 1) / k;
            const int w = g == 0 ? W - k + 1 : 1;  // one group of several warps at most
            groups[i * kSchedMaxGroups + g] = make_int4(f, l - f, base, 32 * w);
            base += 32 * w;
        }
    }
}

std::mutex g_noalloc_mu;
unsigned char* g_noalloc_ptr[kNoAllocMaxDevices];

// Device address of the scratch array on the current device, looked up
// once per device with that device current.
int noalloc_scratch(unsigned char** out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: cudaGetDevice");
    if (dev < 0 || dev >= kNoAllocMaxDevices) return fail_c(DPDR_ERR_INVALID, "no-alloc: device ordinal too large");
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* ptr = nullptr;
        e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
        if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: cudaGetSymbolAddress");
        g_noalloc_ptr[dev] = static_cast<unsigned char*>(ptr);
    }
    *out = g_noalloc_ptr[dev];
    return DPDR_OK;
}

}  // namespace

int schedule_noalloc(int p, int64_t m, int dtype, int op, int b, const void* const* x,
                     void* const* y, cudaStream_t s)
{
    if (p < 1 || m < 0) return fail_c(DPDR_ERR_INVALID, "no-alloc: need p >= 1 and m >= 0");
    if (p > kNoAllocMaxRanks)
        return fail_c(DPDR_ERR_INVALID, "no-alloc: p exceeds DPDR_NOALLOC_MAX_RANKS");
    const bool sum_ok = (dtype == DPDR_INT32 || dtype == DPDR_FLOAT32) && op == DPDR_OP_SUM;
    const bool mat_ok = (dtype == DPDR_MAT2X2_U32 || dtype == DPDR_MAT2X2_F32) &&
                        op == DPDR_OP_MATMUL;
    if (!sum_ok && !mat_ok) return fail_c(DPDR_ERR_INVALID, "no-alloc: unsupported (dtype, op)");
    if (b < 0) return fail_c(DPDR_ERR_INVALID, "no-alloc: b < 0");
    if (!x || !y) return fail_c(DPDR_ERR_INVALID, "no-alloc: x or y is NULL");
    const size_t esize = (dtype == DPDR_MAT2X2_U32 || dtype == DPDR_MAT2X2_F32) ? 16 : 4;
    int vec = 1;
    for (int i = 0; i < p; i++) {
        const uintptr_t a = reinterpret_cast<uintptr_t>(x[i]), c = reinterpret_cast<uintptr_t>(y[i]);
        if (!a || !c) return fail_c(DPDR_ERR_INVALID, "no-alloc: NULL rank buffer");
        if ((a | c) & 3u) return fail_c(DPDR_ERR_INVALID, "no-alloc: rank buffer not 4-byte aligned");
        if ((a | c) & 15u) vec = 0;
    }
    if (m == 0) return DPDR_OK;
    const int64_t hi = m < (int64_t(1) << 30) ? m : (int64_t(1) << 30);
    int bb = b == 0 ? block_count_rule(p, m, 0) : b;
    bb = int(bb < 1 ? 1 : (bb > hi ? hi : bb));
    const NoAllocLayout L = noalloc_layout(p, m, bb, esize);
    if (L.end > kNoAllocBytes)
        return fail_c(DPDR_ERR_INVALID,
                      "no-alloc: pipeline block too large for DPDR_NOALLOC_SCRATCH_BYTES; "
                      "use more blocks (larger b)");

    unsigned char* base = nullptr;
    int rc = noalloc_scratch(&base);
    if (rc) return rc;
    int dev = 0, sms = 0, occ = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess)
        e = sched_occupancy(dtype, kNoAllocThreads, &occ);
    if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: device query");
    const int64_t kmax = int64_t(occ) * sms;
    const int n0 = p / 2, n1 = p - n0;
    int R = 1;
    while (R < p && int64_t((n0 + R - 1) / R + (n1 + R - 1) / R) > kmax) R++;
    const int nctas = (n0 + R - 1) / R + (n1 + R - 1) / R;

    // rank pointers from the caller's host arrays, zeroed counters and
    // error word, tree and CTA tables
    e = cudaMemcpyAsync(base + L.x, x, sizeof(void*) * size_t(p), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess)
        e = cudaMemcpyAsync(base + L.y, y, sizeof(void*) * size_t(p), cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(base + L.ctrl, 0, L.groups - L.ctrl, s);
    if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: set-up copies");
    int* tables = reinterpret_cast<int*>(base + L.tables);
    int4* groups = reinterpret_cast<int4*>(base + L.groups);
    int* rank_list = reinterpret_cast<int*>(base + L.ranks);
    const int tb = 256, blocks = (p + tb - 1) / tb;
    noalloc_tables_kernel<<<blocks, tb, 0, s>>>(p, R, sched::group_count(R, kNoAllocThreads),
                                                nctas, tables, groups, rank_list);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: table kernel");

    SchedArgs a;
    a.x = reinterpret_cast<const char* const*>(base + L.x);
    a.y = reinterpret_cast<char* const*>(base + L.y);
    a.parent = tables;
    a.child0 = tables + p;
    a.child1 = tables + 2 * p;
    a.depth = tables + 3 * p;
    a.groups = groups;
    a.rank_list = rank_list;
    uint32_t* ctrl = reinterpret_cast<uint32_t*>(base + L.ctrl);
    a.up = ctrl;
    a.down = ctrl + int64_t(p) * kCtr;
    a.abort_flag = ctrl + 2 * int64_t(p) * kCtr;
    a.err = reinterpret_cast<uint32_t*>(base + L.err);
    a.ring = reinterpret_cast<char*>(base + L.ring);
    a.ring_slot = int64_t(L.slot);
    a.p = p;
    a.b = bb;
    a.r0 = p / 2 - 1;
    a.r1 = p - 1;
    a.m = m;
    a.q = m / bb;
    a.rem = m % bb;
    a.wait_ns = 4000000000LL;
    a.skip_rank = -1;
    a.vec = vec;
    a.nslices = 1;
    a.nchunks = nctas;
    a.slot_bytes = kSlotBytes;
    const bool lane = (((m + bb - 1) / bb) * int64_t(esize) + 15) / 16 <= kLaneSliceUnits;
    void* args[] = {&a};
    e = cudaLaunchCooperativeKernel(kernel_for(dtype, kAlgoDoubly, lane), dim3(nctas),
                                    dim3(kNoAllocThreads),
                                    args, size_t(kNoAllocThreads) * kSlotBytes, s);
    if (e == cudaErrorCooperativeLaunchTooLarge) {
        cudaGetLastError();
        return fail_c(DPDR_ERR_NOT_COOPERATIVE, "no-alloc: CTAs cannot be co-resident");
    }
    if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: schedule kernel launch");
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: stream synchronize");
    uint32_t err[4] = {0, 0, 0, 0};
    e = cudaMemcpy(err, base + L.err, sizeof err, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail_c(e, "no-alloc: error word read");
    if (err[0] != 0) return fail_c(int(err[0]), "no-alloc: schedule wait expired");
    return DPDR_OK;
}

}  // namespace dpdr

extern "C" int dpdr_allreduce_schedule_noalloc(int p, int64_t m, dpdr_dtype dtype, dpdr_op op,
                                               int b, const void* const* x, void* const* y,
                                               dpdr_stream_t stream)
{
    return dpdr::schedule_noalloc(p, m, int(dtype), int(op), b, x, y,
                                  reinterpret_cast<cudaStream_t>(stream));
}
