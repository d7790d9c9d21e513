"""The allocation-free entry point, dpdr_allreduce_schedule_noalloc.

It is for callers that cannot allocate device memory on the call path
(their memory belongs to another allocator, or an allocation could fail or
stall the device mid-run): it needs no plan and keeps its scratch in a
statically reserved device array.  These tests call it through the C ABI
and check, on two calls in a row with different inputs (the shared scratch
keeps the previous call's contents), that its outputs equal the CPU
oracle's tree fold bit for bit -- the same tolerance every parity test here
uses -- and those of the plan-based dpdr_allreduce_schedule; that sizes
beyond its stated limits are refused with an error instead of being run;
and that a large block the scratch admits gives the right result.  The
entry point builds the trees on the device itself, so the cases include
p = 1 (one rank, no tree) and p = 2^k - 1, 2^k, 2^k + 1 (the shapes where a
complete tree's last level is full, has one node, or has one missing)."""
import ctypes

import numpy as np
import pytest
import torch

from gpu_util import bits, empty_like_ranks, expect_bits, host_inputs, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def native():
    from paper_2109_12626_gb300 import build as B
    B.build()
    from paper_2109_12626_gb300 import _native as N
    N.lib()
    return N


def _call_noalloc(N, p, m, dt, op, b, xs, ys):
    L = N.lib()
    X = (ctypes.c_void_p * p)(*[x.data_ptr() for x in xs])
    Y = (ctypes.c_void_p * p)(*[y.data_ptr() for y in ys])
    stream = torch.cuda.current_stream().cuda_stream
    return L.dpdr_allreduce_schedule_noalloc(p, m, dt, op, b, X, Y, stream)


def _want(orc, x, kind):
    dt = {"int32": orc.I32, "float32": orc.F32, "mat2x2u32": orc.MAT}[kind]
    return expect_bits(orc.tree_fold(x, dt))


# p = 3000 puts several ranks on each CTA (rank groups)
CASES = [("int32", 7, 1000, 4), ("mat2x2u32", 36, 4099, 16),
         ("float32", 1152, 4099, 0), ("float32", 32, 65541, 64), ("int32", 2, 3, 3),
         ("int32", 3000, 257, 2), ("float32", 1, 100, 3), ("float32", 63, 999, 5),
         ("int32", 64, 1001, 7), ("float32", 65, 1003, 4), ("int32", 127, 500, 2),
         ("float32", 255, 257, 1), ("int32", 257, 300, 3)]


@pytest.mark.parametrize("kind,p,m,b", CASES)
def test_noalloc_matches_oracle_and_planned_schedule_twice(native, orc, kind, p, m, b):
    import paper_2109_12626_gb300 as pkg
    N = native
    dt = N.DTYPES[kind]
    op = N.DPDR_OP_MATMUL if kind == "mat2x2u32" else N.DPDR_OP_SUM
    dev = torch.device("cuda:0")
    for seed in (51, 52):                     # two calls in a row
        x = host_inputs(kind, seed, p, m)
        want = _want(orc, x, kind)
        xs, _ = to_device(x, kind, dev)
        ref, _ = empty_like_ranks(xs, fill=-1)
        with pkg.Plan(p, m, kind, b) as plan:
            plan.allreduce_schedule(xs, ref)
            plan.sync()
        got, _ = empty_like_ranks(xs, fill=-2)
        rc = _call_noalloc(N, p, m, dt, op, b, xs, got)
        assert rc == N.DPDR_OK, N.lib().dpdr_last_error_message()
        for i in range(p):
            assert np.array_equal(bits(got[i]), want), (seed, i)
            assert np.array_equal(bits(got[i]), bits(ref[i])), (seed, i)


def test_noalloc_refuses_sizes_beyond_its_limits(native, orc):
    N = native
    dev = torch.device("cuda:0")
    L = N.lib()
    # too many ranks
    p = 8193
    one = torch.zeros(4, dtype=torch.int32, device=dev)
    rc = _call_noalloc(N, p, 1, N.DPDR_INT32, N.DPDR_OP_SUM, 1, [one] * p, [one] * p)
    assert rc == N.DPDR_ERR_INVALID
    assert b"DPDR_NOALLOC_MAX_RANKS" in L.dpdr_last_error_message()
    # one pipeline block larger than the exchange slots allow
    p, m = 2, 1 << 22
    xs = [torch.zeros(m, dtype=torch.int32, device=dev) for _ in range(p)]
    ys = [torch.zeros(m, dtype=torch.int32, device=dev) for _ in range(p)]
    rc = _call_noalloc(N, p, m, N.DPDR_INT32, N.DPDR_OP_SUM, 1, xs, ys)
    assert rc == N.DPDR_ERR_INVALID
    assert b"larger b" in L.dpdr_last_error_message()
    # the same size with enough blocks runs, and is right
    x = host_inputs("int32", 53, p, m)
    want = _want(orc, x, "int32")
    xs, _ = to_device(x, "int32", dev)
    ys, _ = empty_like_ranks(xs, fill=-5)
    rc = _call_noalloc(N, p, m, N.DPDR_INT32, N.DPDR_OP_SUM, 64, xs, ys)
    assert rc == N.DPDR_OK, L.dpdr_last_error_message()
    for y in ys:
        assert np.array_equal(bits(y), want)
