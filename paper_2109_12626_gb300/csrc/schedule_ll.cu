// schedule_ll.cu -- the low-latency transport of the schedule-faithful
// kernel (dpdr_allreduce_schedule on short pipeline blocks).
//
// Same virtual ranks, rounds, steps and bracketing as schedule.cu
// (Algorithm 1 for every rank i, rounds j = 0..b+d_i, the exchanges with
// child_0, child_1 and the parent or the dual root); only the way a block
// passes from one rank to the next differs.  schedule.cu publishes a block
// by writing it and then releasing a counter; its receiver acquires the
// counter and then reads the block: three dependent trips through L2 per
// exchange.  Here every 32-bit word of a sent block travels together with
// the call's epoch in one 64-bit store, which the GPU performs as a single
// access, and the receiver polls the words themselves: a word whose upper
// half equals the epoch holds the sent value.  An exchange then costs one
// trip through L2.  With b = 1 the path from the leaves to the roots and back
// is about 2 d_max + 1 exchanges long, so the trip is what a short block's
// latency is made of.
//
// Memory: two word arrays of p rows, "up" (partial blocks, toward the roots)
// and "down" (final blocks, toward the leaves).  Row i has a fixed place for
// each of the m elements (esize/4 words of 8 bytes each), so every block has
// its own words, nothing is reused within a call and a sender never waits for
// a receiver.  Calls differ by their epoch: the last CTA to finish advances
// it on the device, so the words need no clearing between calls and a
// captured CUDA graph replays correctly.  A leaf's partial block is its
// input x_i, present before the kernel starts, so its parent reads x_i
// directly: leaves send nothing up.
//
// Each thread serves the same columns of every rank its CTA owns and waits
// only for words of those columns, so a round needs no CTA-wide barrier.
// The CTA layout (rank ranges that never straddle the trees, column slices)
// and the deadlock argument are those of schedule.cu: every wait is on a
// lower rank in the same round, on an earlier round, or on the dual root.
// Every wait is bounded in time; an expired wait records {rank, round,
// step}, marks the call aborted (the abort word takes the epoch of the call)
// and every other wait of that call gives up at its next check.
#include <algorithm>

#include "schedule_common.cuh"

namespace dpdr {
namespace {

using sched::block_start;
using sched::ld_relaxed;
using sched::now_ns;
using sched::rank_in;
using sched::rank_out;

typedef unsigned long long u64;

struct LLArgs {
    const char* const* x;
    char* const* y;
    const int* parent;
    const int* child0;
    const int* child1;
    const int* depth;
    const int* cta_first;
    u64* up;            // [p][row] partial blocks
    u64* down;          // [p][row] final blocks
    int64_t row;        // words per rank row: m * esize / 4
    uint32_t* ctl;      // [0] epoch of this call, [1] CTAs finished, [2] aborted epoch
    uint32_t* err;
    int p, b, r0, r1;
    int64_t q, rem;
    int64_t wait_ns;
    int skip_rank;
    int nslices, nchunks;
};

// words handled together by one thread: 4 elements of 4 bytes, 1 of 16
// (twice that from the two children in flight at once; no register spills)
constexpr int kBatchWords = 4;

__device__ __forceinline__ void ll_st(u64* w, uint32_t v, uint32_t epoch)
{
    const u64 word = (u64(epoch) << 32) | v;
    asm volatile("st.relaxed.gpu.global.b64 [%0], %1;" ::"l"(w), "l"(word) : "memory");
}
__device__ __forceinline__ u64 ll_ld(const u64* w)
{
    u64 word;
    asm volatile("ld.relaxed.gpu.global.b64 %0, [%1];" : "=l"(word) : "l"(w) : "memory");
    return word;
}

// Records an expired wait (the first one of the call wins) and aborts the
// call: every other wait sees the abort word equal to its epoch.
__device__ __noinline__ void ll_expire(const LLArgs& a, uint32_t epoch, int rank, int j, int step)
{
    if (atomicCAS(a.err, 0u, uint32_t(DPDR_ERR_TIMEOUT)) == 0u) {
        a.err[1] = uint32_t(rank);
        a.err[2] = uint32_t(j);
        a.err[3] = uint32_t(step);
    }
    __threadfence();
    atomicExch(a.ctl + 2, epoch);
}

// Receives n <= U elements, k0, k0 + T, ..., k0 + (n-1) T, from one or
// two rows of words at once (a null row is skipped): polls every word until
// it carries this call's epoch.  Returns false when the wait expired or the
// call was aborted; an expired wait is recorded with step0 if row 0 was
// still incomplete, else step1.
template <class Op, int U>
__device__ __forceinline__ bool ll_recv(const LLArgs& a, const u64* row0, const u64* row1,
                                        int64_t k0, int n, int T, uint32_t epoch,
                                        Elem<Op>* out0, Elem<Op>* out1, int rank, int j,
                                        int step0, int step1)
{
    constexpr int W = Elem<Op>::kWords;
    static_assert(U * W <= 32, "one pending bit per word");
    uint32_t mask = 0;
#pragma unroll
    for (int u = 0; u < U; u++)
        if (u < n) mask |= ((1u << W) - 1u) << (u * W);
    uint32_t pend0 = row0 ? mask : 0u, pend1 = row1 ? mask : 0u;
    uint64_t t0 = 0;
    for (unsigned polls = 0;; polls++) {
#pragma unroll
        for (int u = 0; u < U; u++) {
#pragma unroll
            for (int w = 0; w < W; w++) {
                const int bit = u * W + w;
                const int64_t at = (k0 + int64_t(u) * T) * W + w;
                if ((pend0 >> bit) & 1u) {
                    const u64 word = ll_ld(row0 + at);
                    if (uint32_t(word >> 32) == epoch) {
                        out0[u].w[w] = uint32_t(word);
                        pend0 &= ~(1u << bit);
                    }
                }
                if ((pend1 >> bit) & 1u) {
                    const u64 word = ll_ld(row1 + at);
                    if (uint32_t(word >> 32) == epoch) {
                        out1[u].w[w] = uint32_t(word);
                        pend1 &= ~(1u << bit);
                    }
                }
            }
        }
        if (!(pend0 | pend1)) return true;
        if (polls == 0) {
            t0 = now_ns();
        } else if ((polls & 15) == 0) {
            if (ld_relaxed(a.ctl + 2) == epoch) return false;
            if (now_ns() - t0 > uint64_t(a.wait_ns)) {
                ll_expire(a, epoch, rank, j, pend0 ? step0 : step1);
                return false;
            }
            if (polls >= 64) __nanosleep(64);
        }
    }
}

template <class Op, int U>
__device__ __forceinline__ void ll_send(u64* row, int64_t k0, int n, int T, uint32_t epoch,
                                        const Elem<Op>* v)
{
    constexpr int W = Elem<Op>::kWords;
#pragma unroll
    for (int u = 0; u < U; u++)
        if (u < n) {
#pragma unroll
            for (int w = 0; w < W; w++) ll_st(row + (k0 + int64_t(u) * T) * W + w, v[u].w[w], epoch);
        }
}

// Round j of Algorithm 1 at rank i, column slice g, for this thread's
// columns.  Step numbers in error records: 0 child_0, 1 child_1, 2 dual,
// 3 parent.
template <class Op>
__device__ __forceinline__ bool ll_round(const LLArgs& a, int i, int j, int g, uint32_t epoch)
{
    using El = Elem<Op>;
    constexpr int W = El::kWords, U = kBatchWords / W, ES = Op::kEsize;
    const int T = blockDim.x;
    const int d = __ldg(a.depth + i);
    const int c0 = __ldg(a.child0 + i), c1 = __ldg(a.child1 + i);
    const int par = __ldg(a.parent + i);
    const bool root = par < 0, leaf = c0 < 0;
    const bool paired = root && a.r0 >= 0;
    const bool sends = i != a.skip_rank;
    u64* const up_i = a.up + int64_t(i) * a.row;
    u64* const down_i = a.down + int64_t(i) * a.row;

    // child_0, child_1, then the dual (roots): block j goes up
    if (j < a.b && (root || !leaf)) {
        const int64_t bs = block_start(a.q, a.rem, j), be = block_start(a.q, a.rem, j + 1);
        const int64_t s = sched::slice_bound<1>(bs, be, g, a.nslices);
        const int64_t e = sched::slice_bound<1>(bs, be, g + 1, a.nslices);
        const char* xi = rank_in(a.x, i);
        char* yi = rank_out(a.y, i);
        for (int64_t k0 = s + threadIdx.x; k0 < e; k0 += int64_t(U) * T) {
            const int n = int(lmin(U, (e - k0 + T - 1) / T));
            El v[U];
#pragma unroll
            for (int u = 0; u < U; u++)
                if (u < n) v[u] = ld_one_l2<Op>(xi + (k0 + int64_t(u) * T) * ES);
            // both children's partial blocks at once: a leaf child's is its
            // input; an inner child's arrives as words.  A leaf that never
            // sends (fault injection) fails the wait.
            El t0[U], t1[U];
            const u64* row[2] = {nullptr, nullptr};
#pragma unroll
            for (int h = 0; h < 2; h++) {
                const int c = h ? c1 : c0;
                if (c < 0) continue;
                if (__ldg(a.child0 + c) >= 0) {
                    row[h] = a.up + int64_t(c) * a.row;
                    continue;
                }
                if (c == a.skip_rank) {
                    ll_expire(a, epoch, i, j, h);
                    return false;
                }
                const char* xc = rank_in(a.x, c);
                El* t = h ? t1 : t0;
#pragma unroll
                for (int u = 0; u < U; u++)
                    if (u < n) t[u] = ld_one_l2<Op>(xc + (k0 + int64_t(u) * T) * ES);
            }
            if ((row[0] || row[1]) &&
                !ll_recv<Op, U>(a, row[0], row[1], k0, n, T, epoch, t0, t1, i, j, 0, 1))
                return false;
#pragma unroll
            for (int u = 0; u < U; u++)
                if (u < n) {
                    if (c0 >= 0) v[u] = comb<Op>(t0[u], v[u]);  // Y[j] = t (.) Y[j], child_0
                    if (c1 >= 0) v[u] = comb<Op>(t1[u], v[u]);  // then child_1
                }
            if (paired) {  // exchange partials with the dual root
                if (sends) ll_send<Op, U>(up_i, k0, n, T, epoch, v);
                const int du = i == a.r0 ? a.r1 : a.r0;
                El t[U];
                if (!ll_recv<Op, U>(a, a.up + int64_t(du) * a.row, nullptr, k0, n, T, epoch, t,
                                    t, i, j, 2, 2))
                    return false;
#pragma unroll
                for (int u = 0; u < U; u++)
                    if (u < n) v[u] = i == a.r0 ? comb<Op>(v[u], t[u]) : comb<Op>(t[u], v[u]);
            }
            if (root) {  // the block is final: keep it and send it down
#pragma unroll
                for (int u = 0; u < U; u++)
                    if (u < n) st_one_l2<Op>(yi + (k0 + int64_t(u) * T) * ES, v[u]);
                if (sends) ll_send<Op, U>(down_i, k0, n, T, epoch, v);
            } else if (sends) {
                ll_send<Op, U>(up_i, k0, n, T, epoch, v);
            }
        }
    }
    // parent: final block j - d comes down
    if (!root) {
        const int kf = j - d;
        if (kf >= 0 && kf < a.b) {
            const int64_t bs = block_start(a.q, a.rem, kf), be = block_start(a.q, a.rem, kf + 1);
            const int64_t s = sched::slice_bound<1>(bs, be, g, a.nslices);
            const int64_t e = sched::slice_bound<1>(bs, be, g + 1, a.nslices);
            char* yi = rank_out(a.y, i);
            const u64* down_p = a.down + int64_t(par) * a.row;
            for (int64_t k0 = s + threadIdx.x; k0 < e; k0 += int64_t(U) * T) {
                const int n = int(lmin(U, (e - k0 + T - 1) / T));
                El f[U];
                if (!ll_recv<Op, U>(a, down_p, nullptr, k0, n, T, epoch, f, f, i, j, 3, 3))
                    return false;
#pragma unroll
                for (int u = 0; u < U; u++)
                    if (u < n) st_one_l2<Op>(yi + (k0 + int64_t(u) * T) * ES, f[u]);
                if (!leaf && sends) ll_send<Op, U>(down_i, k0, n, T, epoch, f);
            }
        }
    }
    return true;
}

template <class Op>
__global__ void __launch_bounds__(sched::kMaxThreads, 4) schedule_ll_kernel(LLArgs a)
{
    const uint32_t epoch = *reinterpret_cast<volatile const uint32_t*>(a.ctl);
    const int g = blockIdx.x / a.nchunks, chunk = blockIdx.x % a.nchunks;
    const int first = __ldg(a.cta_first + chunk);
    const int last = __ldg(a.cta_first + chunk + 1);
    int rounds = 0;
    for (int i = first; i < last; i++) rounds = max(rounds, a.b + __ldg(a.depth + i));
    bool ok = true;
    for (int j = 0; j <= rounds && ok; j++)
        for (int i = first; i < last && ok; i++)
            if (j <= a.b + __ldg(a.depth + i)) ok = ll_round<Op>(a, i, j, g, epoch);
    // the last CTA to finish moves the plan to the next epoch (never 0, the
    // value of words no call has written)
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(a.ctl + 1, 1u) == gridDim.x - 1) {
            a.ctl[1] = 0;
            const uint32_t next = epoch + 1 == 0 ? 1 : epoch + 1;
            *reinterpret_cast<volatile uint32_t*>(a.ctl) = next;
        }
    }
}

template <class Op>
const void* ll_ptr()
{
    return reinterpret_cast<const void*>(&schedule_ll_kernel<Op>);
}

}  // namespace

const void* schedule_ll_kernel_for(int dtype)
{
    switch (dtype) {
    case DPDR_INT32: return ll_ptr<SumI32>();
    case DPDR_FLOAT32: return ll_ptr<SumF32>();
    case DPDR_MAT2X2_F32: return ll_ptr<MatF32>();
    default: return ll_ptr<MatU32>();
    }
}

// Transport of the schedule kernel: the plan's option, else flagged words
// while the p inputs total at most a cap that depends on the layout, else
// counters.  Flagged words cost one L2 trip per exchange against three, but
// move 8 bytes per 4-byte word and poll per thread, and a CTA that owns
// several ranks runs them one after another per thread (the counters kernel
// gives each its own warps).  Measured at b = 1..8, int32, best b each:
//  * one rank per CTA: up to 12 MB (p = 30, m = 2^16: 29 us either way;
//    p = 126, m = 2^15: counters 49 against 59 us), 24 MB from p = 1024
//    (p = 1152, m = 4096: 59 against 64 us; m = 16384: counters 125 against
//    183 us);
//  * two ranks per CTA: up to 8 MB (p = 2048, m = 1024: 48 against 64 us;
//    m = 4096: counters 97 against 104 us);
//  * more: counters (p = 4094, m = 1024: 85 against 98 us; p = 8190, m = 1:
//    367 against 479 us).
// The word arrays (4 p m esize bytes) never exceed 96 MB under these caps.
int schedule_transport(const Plan* P)
{
    if (P->sched_transport) return P->sched_transport;
    const int R = std::max(1, P->sched_rpc_ref);
    const int64_t bytes = int64_t(P->p) * P->m * int64_t(P->esize);
    const int64_t cap = R == 1 ? (P->p >= 1024 ? int64_t(24) << 20 : int64_t(12) << 20)
                      : R == 2 ? int64_t(8) << 20 : 0;
    return bytes <= cap ? 2 : 1;
}

// Elements one CTA of the flagged-word kernel takes per pass: a batch of
// kBatchWords words for each thread.  The plan sizes column slices by it.
int64_t schedule_ll_slice_elems(const Plan* P)
{
    return int64_t(P->sched_threads_used) * (kBatchWords / int64_t(P->esize / 4));
}

// Bytes of the word arrays (up and down, p rows of m elements, 8 bytes per
// 32-bit word) plus the control words.
size_t schedule_ll_bytes(const Plan* P)
{
    const size_t words = size_t(P->m) * (P->esize / 4);
    return 256 + 2 * size_t(P->p) * words * sizeof(u64);
}

// Allocates and clears the word arrays; epoch 1 first.
int schedule_ll_prepare(Plan* P)
{
    if (P->d_ll) return DPDR_OK;
    const size_t bytes = schedule_ll_bytes(P);
    cudaError_t e = cudaMalloc(&P->d_ll, bytes);
    if (e != cudaSuccess) {
        P->d_ll = nullptr;
        return cuda_fail(e, "schedule words: cudaMalloc");
    }
    e = cudaMemset(P->d_ll, 0, bytes);
    const uint32_t one = 1;
    if (e == cudaSuccess) e = cudaMemcpy(P->d_ll, &one, sizeof one, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        cudaFree(P->d_ll);
        P->d_ll = nullptr;
        return cuda_fail(e, "schedule words: clear");
    }
    P->d_ll_bytes = bytes;
    return DPDR_OK;
}

int schedule_ll_launch(Plan* P, cudaStream_t s)
{
    if (P->m == 0) return DPDR_OK;
    if (!P->d_ll) return fail(DPDR_ERR_INVALID, "schedule words not prepared");
    LLArgs a;
    a.x = P->d_x;
    a.y = P->d_y;
    a.parent = P->d_tables;
    a.child0 = P->d_tables + P->p;
    a.child1 = P->d_tables + 2 * P->p;
    a.depth = P->d_tables + 3 * P->p;
    a.cta_first = P->d_cta_first;
    a.ctl = reinterpret_cast<uint32_t*>(P->d_ll);
    const int64_t row = P->m * int64_t(P->esize / 4);
    a.up = reinterpret_cast<u64*>(P->d_ll + 256);
    a.down = a.up + int64_t(P->p) * row;
    a.row = row;
    a.err = P->d_err;
    a.p = P->p;
    a.b = P->b;
    a.r0 = P->r0;
    a.r1 = P->r1;
    a.q = P->m / P->b;
    a.rem = P->m % P->b;
    a.wait_ns = P->wait_ns;
    a.skip_rank = P->skip_rank;
    a.nslices = P->sched_slices_used;
    a.nchunks = P->sched_chunks;
    void* args[] = {&a};
    cudaError_t e = cudaLaunchCooperativeKernel(schedule_ll_kernel_for(P->dtype),
                                                dim3(P->sched_ctas), dim3(P->sched_threads_used),
                                                args, 0, s);
    if (e == cudaErrorCooperativeLaunchTooLarge) {
        cudaGetLastError();
        return fail(DPDR_ERR_NOT_COOPERATIVE, "schedule kernel: CTAs cannot be co-resident");
    }
    if (e != cudaSuccess) return cuda_fail(e, "schedule kernel launch");
    return DPDR_OK;
}

}  // namespace dpdr
