// api.cpp -- argument checks, rank-pointer staging and the run entry points
// of the C ABI (dpdr_allreduce, dpdr_allreduce_schedule,
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
    return schedule_launch(P, s);
}

extern "C" int dpdr_allreduce_host(dpdr_plan_t h, const void* const* x_host,
                                   void* const* y_host, void* const* x_dev,
                                   void* const* y_dev, dpdr_stream_t stream)
{
    Plan* P = reinterpret_cast<Plan*>(h);
    if (!P) return fail(DPDR_ERR_INVALID, "dpdr_allreduce_host: NULL plan");
    if (!x_host || !y_host || !x_dev || !y_dev)
        return fail(DPDR_ERR_INVALID, "dpdr_allreduce_host: NULL pointer array");
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    const size_t bytes = size_t(P->m) * P->esize;
    for (int i = 0; i < P->p; i++)
        if (!x_host[i] || !y_host[i]) return fail(DPDR_ERR_INVALID, "NULL host buffer");
    cudaError_t e;
    for (int i = 0; i < P->p && bytes; i++) {
        e = cudaMemcpyAsync(x_dev[i], x_host[i], bytes, cudaMemcpyHostToDevice, s);
        if (e != cudaSuccess) return cuda_fail(e, "host to device copy");
    }
    int rc = dpdr_allreduce(h, reinterpret_cast<const void* const*>(x_dev), y_dev, stream);
    if (rc) return rc;
    for (int i = 0; i < P->p && bytes; i++) {
        e = cudaMemcpyAsync(y_host[i], y_dev[i], bytes, cudaMemcpyDeviceToHost, s);
        if (e != cudaSuccess) return cuda_fail(e, "device to host copy");
    }
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
