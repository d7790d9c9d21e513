// api.cpp -- argument checks, rank-pointer staging and the run entry points
// of the C ABI (dpdr_allreduce, dpdr_allreduce_schedule,
// dpdr_allreduce_reduce_bcast,
// dpdr_allreduce_host, dpdr_plan_sync).
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <utility>

#include "dpdr_internal.h"

namespace dpdr {

// Validates the 2p rank buffers: non-null, element-aligned, and no overlap
// except y[i] == x[i] (in place).  Inputs may overlap each other (they are
// only read).  Sets *vec when every buffer is 16-byte aligned.
static int check_buffers(const Plan* P, const void* const* x,
                         const void* const* y, int* vec)
{
    if (!x || !y) return fail(DPDR_ERR_INVALID, "x or y is NULL");
    const int p = P->p;
    const uintptr_t bytes = uintptr_t(P->m) * P->esize;
    bool all16 = true;
    std::vector<std::pair<uintptr_t, int>> ys;  // (start, rank)
    ys.reserve(p);
    for (int i = 0; i < p; i++) {
        const uintptr_t xs = reinterpret_cast<uintptr_t>(x[i]);
        const uintptr_t yv = reinterpret_cast<uintptr_t>(y[i]);
        if (!xs || !yv) return fail(DPDR_ERR_INVALID, "NULL rank buffer");
        if ((xs | yv) & 3u) return fail(DPDR_ERR_INVALID, "rank buffer not 4-byte aligned");
        if ((xs | yv) & 15u) all16 = false;
        ys.emplace_back(yv, i);
    }
    *vec = all16 ? 1 : 0;
    if (bytes == 0) return DPDR_OK;
    std::sort(ys.begin(), ys.end());
    for (int k = 1; k < p; k++)
        if (ys[k].first < ys[k - 1].first + bytes)
            return fail(DPDR_ERR_INVALID, "output buffers overlap");
    // every input against the outputs it could meet
    for (int i = 0; i < p; i++) {
        const uintptr_t xs = reinterpret_cast<uintptr_t>(x[i]);
        auto it = std::upper_bound(ys.begin(), ys.end(), std::make_pair(xs + bytes, -1));
        // candidates: outputs starting before xs + bytes; only the last two
        // can reach into [xs, xs+bytes) because outputs do not overlap
        for (int back = 0; back < 2 && it != ys.begin(); back++) {
            --it;
            const uintptr_t s0 = it->first;
            if (s0 + bytes <= xs) break;
            if (!(it->second == i && s0 == xs))
                return fail(DPDR_ERR_INVALID, "an output overlaps an input other than its own");
        }
    }
    return DPDR_OK;
}

int stage_pointers(Plan* P, const void* const* x, const void* const* y,
                   cudaStream_t s)
{
    const int p = P->p;
    bool same = true;
    for (int i = 0; i < p && same; i++)
        same = P->last_x[i] == x[i] && P->last_y[i] == y[i];
    if (same && P->staged_pending) return DPDR_OK;  // device table is current
    cudaError_t e;
    if (P->staged_pending) {  // the previous upload must have left the buffer
        e = cudaEventSynchronize(P->staged);
        if (e != cudaSuccess) return cuda_fail(e, "pointer staging wait");
    }
    for (int i = 0; i < p; i++) {
        P->h_ptrs[i] = x[i];
        P->h_ptrs[p + i] = y[i];
        P->last_x[i] = x[i];
        P->last_y[i] = y[i];
    }
    e = cudaMemcpyAsync(const_cast<const char**>(P->d_x), P->h_ptrs,
                        sizeof(void*) * 2 * size_t(p), cudaMemcpyHostToDevice, s);
    if (e != cudaSuccess) return cuda_fail(e, "pointer upload");
    e = cudaEventRecord(P->staged, s);
    if (e != cudaSuccess) return cuda_fail(e, "pointer staging event");
    P->staged_pending = true;
    return DPDR_OK;
}

static int prepare(Plan* P, const void* const* x, const void* const* y,
                   cudaStream_t s)
{
    if (!x || !y) return fail(DPDR_ERR_INVALID, "x or y is NULL");
    if (P->staged_pending) {  // same buffers as the last checked call: nothing to do
        bool same = true;
        for (int i = 0; i < P->p && same; i++)
            same = P->last_x[i] == x[i] && P->last_y[i] == y[i];
        if (same) return DPDR_OK;
    }
    int vec = 0;
    int rc = check_buffers(P, x, y, &vec);
    if (rc) return rc;
    P->last_vector_path = vec;
    return stage_pointers(P, x, y, s);
}

}  // namespace dpdr

using namespace dpdr;

extern "C" int dpdr_allreduce(dpdr_plan_t h, const void* const* x,
                              void* const* y, dpdr_stream_t stream)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_allreduce: NULL plan");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    int rc = prepare(P, x, reinterpret_cast<const void* const*>(y), s);
    if (rc) return rc;
    return fused_launch(P, s);
}

extern "C" int dpdr_allreduce_schedule(dpdr_plan_t h, const void* const* x,
                                       void* const* y, dpdr_stream_t stream)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_allreduce_schedule: NULL plan");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    int rc = prepare(P, x, reinterpret_cast<const void* const*>(y), s);
    if (rc) return rc;
    return schedule_transport(P) == 2 ? schedule_ll_launch(P, s) : schedule_launch(P, s);
}

extern "C" int dpdr_allreduce_reduce_bcast(dpdr_plan_t h, const void* const* x,
                                           void* const* y, dpdr_stream_t stream)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_allreduce_reduce_bcast: NULL plan");
    if (P->topo != DPDR_TOPO_SINGLE)
        return fail(DPDR_ERR_INVALID,
                    "dpdr_allreduce_reduce_bcast: needs a plan made with DPDR_TOPO_SINGLE");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    int rc = prepare(P, x, reinterpret_cast<const void* const*>(y), s);
    if (rc) return rc;
    return schedule_launch(P, s, 1);
}

// Column chunks of about host_chunk bytes of rank data (default 1 GB), each
// row piece at least min(2 MB, host_chunk) so copies stay large, at most 64
// chunks; chunk starts on 256-column boundaries (16-byte aligned).
static int pipe_prepare(Plan* P, void* const* x_dev, void* const* y_dev, bool vec)
{
    const int p = P->p;
    const int64_t es = int64_t(P->esize);
    const int64_t row_min = std::min<int64_t>(int64_t(2) << 20, P->host_chunk);
    int64_t cols = std::max<int64_t>(row_min / es, P->host_chunk / (p * es));
    cols = std::max<int64_t>(cols, (P->m + 63) / 64);
    cols = (cols + 255) / 256 * 256;
    const int chunks = int((P->m + cols - 1) / cols);
    cudaError_t e;
    if (!P->pipe_in) {
        e = cudaStreamCreateWithFlags(&P->pipe_in, cudaStreamNonBlocking);
        if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&P->pipe_out, cudaStreamNonBlocking);
        if (e != cudaSuccess) return cuda_fail(e, "host pipeline streams");
    }
    while (int(P->pipe_ev.size()) < 2 + 2 * chunks) {
        cudaEvent_t ev;
        e = cudaEventCreateWithFlags(&ev, cudaEventDisableTiming);
        if (e != cudaSuccess) return cuda_fail(e, "host pipeline events");
        P->pipe_ev.push_back(ev);
    }
    bool same = P->pipe_cols == cols && P->pipe_chunks == chunks &&
                int(P->pipe_xd.size()) == p && int(P->pipe_yd.size()) == p;
    for (int i = 0; i < p && same; i++) same = P->pipe_xd[i] == x_dev[i] && P->pipe_yd[i] == y_dev[i];
    if (same) return DPDR_OK;
    const size_t bytes = sizeof(void*) * 2 * size_t(p) * chunks;
    if (bytes > P->d_pipe_bytes) {
        if (P->d_pipe) cudaFree(P->d_pipe);
        P->d_pipe = nullptr;
        P->d_pipe_bytes = 0;
        e = cudaMalloc(&P->d_pipe, bytes);
        if (e != cudaSuccess) return cuda_fail(e, "host pipeline tables");
        P->d_pipe_bytes = bytes;
    }
    std::vector<const char*> t(2 * size_t(p) * chunks);
    for (int c = 0; c < chunks; c++)
        for (int i = 0; i < p; i++) {
            t[(size_t(c) * 2) * p + i] = static_cast<const char*>(x_dev[i]) + c * cols * es;
            t[(size_t(c) * 2 + 1) * p + i] = static_cast<const char*>(y_dev[i]) + c * cols * es;
        }
    e = cudaMemcpy(P->d_pipe, t.data(), bytes, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e, "host pipeline table upload");
    P->pipe_cols = cols;
    P->pipe_chunks = chunks;
    P->pipe_xd.assign(x_dev, x_dev + p);
    P->pipe_yd.assign(y_dev, y_dev + p);
    (void)vec;
    return DPDR_OK;
}

// Device addresses for host buffers the GPU can load and store directly:
// pinned (page-locked, mapped into the unified address space) memory, or
// pageable memory on systems whose GPU walks the CPU page tables (Grace
// with NVLink-C2C).  Resolved once per set of host arrays.
static bool resolve_direct(Plan* P, const void* const* xh, void* const* yh)
{
    const int p = P->p;
    bool same = P->direct_ok && int(P->direct_xh.size()) == p;
    for (int i = 0; i < p && same; i++) same = P->direct_xh[i] == xh[i] && P->direct_yh[i] == yh[i];
    if (same) return true;
    int pageable = 0;
    if (cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, P->device) != cudaSuccess)
        pageable = 0;
    std::vector<const void*> dx(p), dy(p);
    for (int k = 0; k < 2 * p; k++) {
        const void* hp = k < p ? xh[k] : yh[k - p];
        cudaPointerAttributes at;
        const void* dp = nullptr;
        if (cudaPointerGetAttributes(&at, hp) == cudaSuccess) {
            if (at.type == cudaMemoryTypeHost && at.devicePointer) dp = at.devicePointer;
            else if (at.type == cudaMemoryTypeUnregistered && pageable) dp = hp;
        } else {
            cudaGetLastError();
        }
        if (!dp) {
            P->direct_ok = false;
            return false;
        }
        (k < p ? dx[k] : dy[k - p]) = dp;
    }
    P->direct_xh.assign(xh, xh + p);
    P->direct_yh.assign(yh, yh + p);
    P->direct_dx = dx;
    P->direct_dy = dy;
    P->direct_ok = true;
    return true;
}

extern "C" int dpdr_allreduce_host(dpdr_plan_t h, const void* const* x_host,
                                   void* const* y_host, void* const* x_dev,
                                   void* const* y_dev, dpdr_stream_t stream)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_allreduce_host: NULL plan");
    if (!x_host || !y_host)
        return fail(DPDR_ERR_INVALID, "dpdr_allreduce_host: NULL pointer array");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    for (int i = 0; i < P->p; i++)
        if (!x_host[i] || !y_host[i]) return fail(DPDR_ERR_INVALID, "NULL host buffer");
    if (P->m == 0) return DPDR_OK;
    // direct: one launch loads the inputs from host memory and stores the
    // result to host memory, the link carrying both directions at once.  The
    // layout DPDR_OPT_FUSED_MODE names, else the hierarchical tile (8 column
    // units per CTA at every size, whose extra CTAs help here), whose
    // CTAs read all their columns, then write them, and drift out of phase
    // with each other (p = 1152, m = 2^20: 297 GB/s against 230 for column
    // streaming, whose threads read and write in long lockstep phases at
    // large p; p = 288, m = 2^22: 339 against 270; p = 36, 2x2 matrices,
    // m = 2^16: 315 against 213); column streaming below 1 MiB of inputs,
    // where one phase per thread has the least latency (p = 7, m = 1000:
    // 4.5 against 3.7 GB/s), and above 4 GiB at p < 64, where its 4 KB row
    // pieces per CTA suit the link better (p = 32, m = 2^27: 333 against
    // 318; m = 2^25: 320 against 343)
    if (P->host_path != 1 && resolve_direct(P, x_host, y_host)) {
        int rc = prepare(P, P->direct_dx.data(), P->direct_dy.data(), s);
        if (rc) return rc;
        const int64_t bytes = int64_t(P->p) * P->m * int64_t(P->esize);
        const bool stream = bytes < (int64_t(1) << 20) ||
                            (P->p < 64 && bytes > (int64_t(4) << 30));
        const int mode = P->fused_mode ? P->fused_mode : stream ? 1 : 5;
        if (mode == 5 && (rc = fused_tree_prepare(P)) != DPDR_OK) return rc;
        P->last_host_path = 2;
        return fused_launch_cols(P, P->d_x, P->d_y, P->m, P->last_vector_path != 0, s, mode, 0);
    }
    if (P->host_path == 2)
        return fail(DPDR_ERR_INVALID, "dpdr_allreduce_host: host buffers not addressable by the GPU");
    if (!x_dev || !y_dev)
        return fail(DPDR_ERR_INVALID, "dpdr_allreduce_host: device staging buffers needed");
    P->last_host_path = 1;
    int vec = 0;
    int rc = check_buffers(P, reinterpret_cast<const void* const*>(x_dev),
                           reinterpret_cast<const void* const*>(y_dev), &vec);
    if (rc) return rc;
    rc = pipe_prepare(P, x_dev, y_dev, vec != 0);
    if (rc) return rc;
    const int p = P->p, C = P->pipe_chunks;
    const int64_t es = int64_t(P->esize);
    cudaEvent_t entry = P->pipe_ev[0], done = P->pipe_ev[1];
    cudaError_t e = cudaEventRecord(entry, s);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(P->pipe_in, entry, 0);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(P->pipe_out, entry, 0);
    if (e != cudaSuccess) return cuda_fail(e, "host pipeline entry");
    char* const* tab = reinterpret_cast<char* const*>(P->d_pipe);
    for (int c = 0; c < C; c++) {
        const int64_t c0 = c * P->pipe_cols, mc = std::min<int64_t>(P->pipe_cols, P->m - c0);
        const size_t off = size_t(c0 * es), len = size_t(mc * es);
        cudaEvent_t in = P->pipe_ev[2 + 2 * c], out = P->pipe_ev[3 + 2 * c];
        for (int i = 0; i < p && e == cudaSuccess; i++)
            e = cudaMemcpyAsync(static_cast<char*>(x_dev[i]) + off,
                                static_cast<const char*>(x_host[i]) + off, len,
                                cudaMemcpyHostToDevice, P->pipe_in);
        if (e == cudaSuccess) e = cudaEventRecord(in, P->pipe_in);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(s, in, 0);
        if (e != cudaSuccess) return cuda_fail(e, "host to device copy");
        rc = fused_launch_cols(P, reinterpret_cast<const char* const*>(tab + size_t(c) * 2 * p),
                               tab + (size_t(c) * 2 + 1) * p, mc, vec != 0, s, 0);
        if (rc) return rc;
        e = cudaEventRecord(out, s);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(P->pipe_out, out, 0);
        for (int i = 0; i < p && e == cudaSuccess; i++)
            e = cudaMemcpyAsync(static_cast<char*>(y_host[i]) + off,
                                static_cast<const char*>(y_dev[i]) + off, len,
                                cudaMemcpyDeviceToHost, P->pipe_out);
        if (e != cudaSuccess) return cuda_fail(e, "device to host copy");
    }
    e = cudaEventRecord(done, P->pipe_out);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, done, 0);
    if (e != cudaSuccess) return cuda_fail(e, "host pipeline exit");
    return DPDR_OK;
}

extern "C" int dpdr_plan_sync(dpdr_plan_t h, dpdr_stream_t stream)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_plan_sync: NULL plan");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    uint32_t err[4] = {0, 0, 0, 0};
    e = cudaMemcpy(err, P->d_err, sizeof err, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "error word read");
    if (err[0] == 0) return DPDR_OK;
    e = cudaMemset(P->d_err, 0, sizeof err);
    if (e != cudaSuccess) return cuda_fail(e, "error word clear");
    char msg[160];
    static const char* steps[] = {"child_0", "child_1", "dual", "parent"};
    std::snprintf(msg, sizeof msg, "schedule wait expired: rank %u round %u step %s",
                  err[1], err[2], err[3] < 4 ? steps[err[3]] : "?");
    return fail(int(err[0]), msg);
}
