/* c_abi_program.c -- the C ABI used from plain C99, without Python: a plan
 * for p ranks of int32 sums, the fused kernel, the schedule kernel with
 * each transport, the host-buffer entry point and the allocation-free entry
 * point, every result checked against an exact sum computed here
 * (int32 sums wrap modulo 2^32, so the order of the terms does not matter).
 *
 *   c_abi_program P M     -> prints "ok" and exits 0, else prints the
 *                            failing step and exits 1
 *
 * Test infrastructure: the tests compile it with gcc against
 * include/dpdr.h and libdpdr.so and run it on a GPU. */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "dpdr.h"

static int check(int rc, const char* what)
{
    if (rc != DPDR_OK) {
        printf("%s: %s (%s)\n", what, dpdr_status_string(rc), dpdr_last_error_message());
        return 1;
    }
    return 0;
}

static int compare(int p, int64_t m, int32_t* const* ys_host, const int32_t* want,
                   const char* what)
{
    for (int i = 0; i < p; i++)
        for (int64_t k = 0; k < m; k++)
            if (ys_host[i][k] != want[k]) {
                printf("%s: rank %d element %lld differs\n", what, i, (long long)k);
                return 1;
            }
    return 0;
}

int main(int argc, char** argv)
{
    const int p = argc > 1 ? atoi(argv[1]) : 7;
    const int64_t m = argc > 2 ? atoll(argv[2]) : 1000;
    const size_t bytes = (size_t)m * sizeof(int32_t);
    int32_t** xh = (int32_t**)calloc((size_t)p, sizeof(int32_t*));
    int32_t** yh = (int32_t**)calloc((size_t)p, sizeof(int32_t*));
    void** xd = (void**)calloc((size_t)p, sizeof(void*));
    void** yd = (void**)calloc((size_t)p, sizeof(void*));
    int32_t* want = (int32_t*)calloc((size_t)m, sizeof(int32_t));
    if (!xh || !yh || !xd || !yd || !want) return 1;

    /* inputs x_i[k] = (i * 2654435761 + k * 40503) mod 2^32, as int32 */
    for (int i = 0; i < p; i++) {
        xh[i] = (int32_t*)malloc(bytes);
        yh[i] = (int32_t*)malloc(bytes);
        if (!xh[i] || !yh[i]) return 1;
        for (int64_t k = 0; k < m; k++) {
            const uint32_t v = (uint32_t)i * 2654435761u + (uint32_t)k * 40503u;
            xh[i][k] = (int32_t)v;
            want[k] = (int32_t)((uint32_t)want[k] + v);
        }
        if (cudaMalloc(&xd[i], bytes) != cudaSuccess || cudaMalloc(&yd[i], bytes) != cudaSuccess ||
            cudaMemcpy(xd[i], xh[i], bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
            printf("cuda set-up failed\n");
            return 1;
        }
    }

    dpdr_plan_t plan = dpdr_plan(p, m, DPDR_INT32, DPDR_OP_SUM, 0);
    if (!plan) return check(dpdr_last_error(), "dpdr_plan");
    int b = 0;
    if (check(dpdr_plan_query(plan, NULL, NULL, NULL, NULL, NULL, &b), "dpdr_plan_query"))
        return 1;

    const char* names[3] = {"dpdr_allreduce", "dpdr_allreduce_schedule counters",
                            "dpdr_allreduce_schedule words"};
    for (int run = 0; run < 3; run++) {
        for (int i = 0; i < p; i++) cudaMemset(yd[i], 0xff, bytes);
        int rc;
        if (run == 0) {
            rc = dpdr_allreduce(plan, (const void* const*)xd, yd, NULL);
        } else {
            rc = dpdr_plan_set(plan, DPDR_OPT_SCHED_TRANSPORT, run);
            if (rc == DPDR_OK) rc = dpdr_allreduce_schedule(plan, (const void* const*)xd, yd, NULL);
        }
        if (check(rc, names[run]) || check(dpdr_plan_sync(plan, NULL), "dpdr_plan_sync")) return 1;
        for (int i = 0; i < p; i++)
            if (cudaMemcpy(yh[i], yd[i], bytes, cudaMemcpyDeviceToHost) != cudaSuccess) return 1;
        if (compare(p, m, yh, want, names[run])) return 1;
    }

    /* host buffers end to end (pageable memory: the direct path where the
       GPU reaches it, else the copy pipeline through xd / yd) */
    for (int i = 0; i < p; i++) memset(yh[i], 0, bytes);
    if (check(dpdr_allreduce_host(plan, (const void* const*)xh, (void* const*)yh, xd, yd, NULL),
              "dpdr_allreduce_host") ||
        check(dpdr_plan_sync(plan, NULL), "dpdr_plan_sync") ||
        compare(p, m, yh, want, "dpdr_allreduce_host"))
        return 1;
    /* reduce-then-broadcast needs a one-tree plan */
    if (dpdr_allreduce_reduce_bcast(plan, (const void* const*)xd, yd, NULL) != DPDR_ERR_INVALID) {
        printf("dpdr_allreduce_reduce_bcast accepted a dual-tree plan\n");
        return 1;
    }
    dpdr_plan_destroy(plan);

    /* pipelined reduce, then pipelined broadcast, on one tree */
    plan = dpdr_plan_topo(p, m, DPDR_INT32, DPDR_OP_SUM, 0, DPDR_TOPO_SINGLE);
    if (!plan) return check(dpdr_last_error(), "dpdr_plan_topo");
    for (int i = 0; i < p; i++) cudaMemset(yd[i], 0xff, bytes);
    if (check(dpdr_allreduce_reduce_bcast(plan, (const void* const*)xd, yd, NULL),
              "dpdr_allreduce_reduce_bcast") ||
        check(dpdr_plan_sync(plan, NULL), "dpdr_plan_sync"))
        return 1;
    for (int i = 0; i < p; i++)
        if (cudaMemcpy(yh[i], yd[i], bytes, cudaMemcpyDeviceToHost) != cudaSuccess) return 1;
    if (compare(p, m, yh, want, "dpdr_allreduce_reduce_bcast")) return 1;
    dpdr_plan_destroy(plan);

    /* the allocation-free entry point: no plan at all */
    for (int i = 0; i < p; i++) cudaMemset(yd[i], 0xff, bytes);
    if (check(dpdr_allreduce_schedule_noalloc(p, m, DPDR_INT32, DPDR_OP_SUM, b,
                                              (const void* const*)xd, yd, NULL),
              "dpdr_allreduce_schedule_noalloc"))
        return 1;
    for (int i = 0; i < p; i++)
        if (cudaMemcpy(yh[i], yd[i], bytes, cudaMemcpyDeviceToHost) != cudaSuccess) return 1;
    if (compare(p, m, yh, want, "dpdr_allreduce_schedule_noalloc")) return 1;

    for (int i = 0; i < p; i++) {
        cudaFree(xd[i]);
        cudaFree(yd[i]);
        free(xh[i]);
        free(yh[i]);
    }
    free(xh);
    free(yh);
    free(xd);
    free(yd);
    free(want);
    printf("ok\n");
    return 0;
}
