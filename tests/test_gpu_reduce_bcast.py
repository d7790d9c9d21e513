"""GPU parity for the pipelined reduce, then pipelined broadcast, on one
tree (the alternative of Sec. 1.2 and Sec. 2, item 3), through the C ABI's
dpdr_allreduce_reduce_bcast: bit for bit against the oracle's one-tree fold
and its event-level simulation of the two phases, for every element type,
block counts from 1 to m, ragged blocks, column slices, several ranks per
CTA, in place and with 4-byte-aligned buffers."""
import numpy as np
import pytest
import torch

from gpu_util import bits, empty_like_ranks, expect_bits, host_inputs, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    from paper_2109_12626_gb300 import build as B
    B.build()
    import paper_2109_12626_gb300 as P
    return P


def _dt(orc, kind):
    return {"int32": orc.I32, "float32": orc.F32, "mat2x2u32": orc.MAT,
            "mat2x2f32": orc.MATF}[kind]


CASES = [("float32", 1, 33, 1), ("float32", 2, 1001, 3), ("int32", 3, 17, 17),
         ("mat2x2u32", 5, 300, 7), ("float32", 7, 4099, 4), ("float32", 15, 65541, 16),
         ("int32", 31, 2000, 1), ("mat2x2u32", 63, 129, 5), ("float32", 255, 3001, 9),
         ("float32", 1023, 1027, 2), ("int32", 1152, 4099, 8), ("mat2x2f32", 127, 700, 6),
         ("int32", 36, 100003, 64)]


@pytest.mark.parametrize("kind,p,m,b", CASES)
@pytest.mark.parametrize("layout", ["auto", "slices", "groups"])
@pytest.mark.parametrize("copy", [0, 2], ids=["copy_auto", "copy_bulk"])
def test_reduce_bcast_parity(pkg, orc, kind, p, m, b, layout, copy):
    x = host_inputs(kind, 91, p, m)
    want = expect_bits(orc.tree_fold(x, _dt(orc, kind), orc.SINGLE))
    dev = torch.device("cuda:0")
    xs, _ = to_device(x, kind, dev)
    ys, _ = empty_like_ranks(xs)
    with pkg.Plan(p, m, kind, b, topology="single") as plan:
        if layout == "slices":
            plan.set(pkg.OPT_SCHED_SLICES, 3)
        if layout == "groups":
            plan.set(pkg.OPT_SCHED_RANKS_PER_CTA, min(p, 3))
        plan.set(pkg.OPT_SCHED_COPY, copy)
        plan.allreduce_reduce_bcast(xs, ys)
        plan.sync()
    for i, y in enumerate(ys):
        assert np.array_equal(bits(y), want), (layout, i)
    for i, xr in enumerate(xs):  # inputs untouched
        assert np.array_equal(bits(xr), np.ascontiguousarray(x[i]).view(np.int32).reshape(-1))


@pytest.mark.parametrize("p,m,b", [(7, 40, 4), (31, 64, 8), (40, 33, 5)])
def test_matches_the_event_simulation(pkg, orc, p, m, b):
    """The same inputs through the oracle's simulation of the two phases."""
    x = host_inputs("float32", 92, p, m)
    ysim, _ = orc.simulate_rb(x, orc.F32, b)
    dev = torch.device("cuda:0")
    xs, _ = to_device(x, "float32", dev)
    ys, _ = empty_like_ranks(xs)
    with pkg.Plan(p, m, "float32", b, topology="single") as plan:
        plan.allreduce_reduce_bcast(xs, ys)
        plan.sync()
    for i, y in enumerate(ys):
        assert np.array_equal(bits(y), ysim[i].view(np.int32)), i


@pytest.mark.parametrize("kind,p,m,b", [("float32", 255, 3001, 9), ("mat2x2u32", 63, 129, 5),
                                        ("int32", 8, 1, 1)])
def test_in_place_and_unaligned(pkg, orc, kind, p, m, b):
    x = host_inputs(kind, 93, p, m)
    want = expect_bits(orc.tree_fold(x, _dt(orc, kind), orc.SINGLE))
    dev = torch.device("cuda:0")
    xs, _ = to_device(x, kind, dev)
    with pkg.Plan(p, m, kind, b, topology="single") as plan:
        plan.allreduce_reduce_bcast(xs, xs)          # y[i] == x[i]
        plan.sync()
        for y in xs:
            assert np.array_equal(bits(y), want)
        xs2, keep = to_device(x, kind, dev, pad_front=1)
        ys2, keep2 = empty_like_ranks(xs2, pad_front=1)
        plan.allreduce_reduce_bcast(xs2, ys2)         # 4-byte aligned only
        plan.sync()
        for y in ys2:
            assert np.array_equal(bits(y), want)


def test_same_bits_as_algorithm_1_on_the_same_tree(pkg, orc):
    """Both schedules compute the one tree's bracketing."""
    p, m = 100, 5000
    x = host_inputs("float32", 94, p, m)
    dev = torch.device("cuda:0")
    xs, _ = to_device(x, "float32", dev)
    a, _ = empty_like_ranks(xs)
    r, _ = empty_like_ranks(xs)
    with pkg.Plan(p, m, "float32", 7, topology="single") as plan:
        plan.allreduce_schedule(xs, a)
        plan.allreduce_reduce_bcast(xs, r)
        plan.sync()
    for u, v in zip(a, r):
        assert np.array_equal(bits(u), bits(v))


def test_needs_a_one_tree_plan(pkg):
    from paper_2109_12626_gb300 import DpdrError
    dev = torch.device("cuda:0")
    xs = [torch.zeros(16, dtype=torch.int32, device=dev) for _ in range(7)]
    with pkg.Plan(7, 16, "int32", 2) as plan:
        with pytest.raises(DpdrError) as e:
            plan.allreduce_reduce_bcast(xs, xs)
        assert e.value.status == pkg.DPDR_ERR_INVALID


@pytest.mark.parametrize("p,skip", [(7, 0), (31, 30), (255, 100)])
def test_silent_rank_times_out_and_recovers(pkg, orc, p, skip):
    from paper_2109_12626_gb300 import DpdrError
    kind, m = "int32", 1000
    x = host_inputs(kind, 95, p, m, lo=-1000, hi=1000)
    want = expect_bits(orc.tree_fold(x, orc.I32, orc.SINGLE))
    xs, _ = to_device(x, kind, torch.device("cuda:0"))
    with pkg.Plan(p, m, kind, 4, topology="single") as plan:
        plan.set(pkg.OPT_WAIT_LIMIT_NS, 20_000_000)
        plan.set(pkg.OPT_SKIP_RANK, skip)
        ys, _ = empty_like_ranks(xs)
        plan.allreduce_reduce_bcast(xs, ys)
        with pytest.raises(DpdrError) as e:
            plan.sync()
        assert e.value.status == pkg.DPDR_ERR_TIMEOUT
        plan.set(pkg.OPT_SKIP_RANK, -1)
        plan.allreduce_reduce_bcast(xs, ys)
        plan.sync()
        for y in ys:
            assert np.array_equal(bits(y), want)
