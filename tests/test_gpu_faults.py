"""Failure detection of the schedule kernel, without faulting the GPU.

Every wait of the kernel is bounded in time.  The test makes one virtual
rank never publish its blocks (a host-set plan option), so its partners'
waits run out after a short limit; the kernel then records where it gave up,
every CTA returns, and dpdr_plan_sync reports DPDR_ERR_TIMEOUT.  The CUDA
context stays usable: the next call on the same plan succeeds and is
correct."""
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


@pytest.mark.parametrize("p,skip", [(7, 0), (7, 6), (36, 17), (1152, 700), (4094, 3000)])
@pytest.mark.parametrize("transport", [1, 2], ids=["counters", "words"])
def test_silent_rank_times_out_and_recovers(pkg, orc, p, skip, transport):
    from paper_2109_12626_gb300 import DpdrError
    kind, m = "int32", 1000
    x = host_inputs(kind, 41, p, m, lo=-1000, hi=1000)
    want = expect_bits(orc.tree_fold(x, orc.I32))
    xs, _ = to_device(x, kind, torch.device("cuda:0"))
    with pkg.Plan(p, m, kind, 4) as plan:
        plan.set(pkg.OPT_WAIT_LIMIT_NS, 20_000_000)   # 20 ms
        plan.set(pkg.OPT_SKIP_RANK, skip)
        plan.set(pkg.OPT_SCHED_TRANSPORT, transport)
        ys, _ = empty_like_ranks(xs)
        plan.allreduce_schedule(xs, ys)
        with pytest.raises(DpdrError) as e:
            plan.sync()
        assert e.value.status == pkg.DPDR_ERR_TIMEOUT
        assert "rank" in str(e.value)
        # the error was consumed; the context and the plan still work
        plan.sync()
        plan.set(pkg.OPT_SKIP_RANK, -1)
        ys, _ = empty_like_ranks(xs)
        plan.allreduce_schedule(xs, ys)
        plan.sync()
        for y in ys:
            assert np.array_equal(bits(y), want)
        plan.allreduce(xs, ys)
        plan.sync()


def test_not_cooperative_is_an_error_not_a_hang(pkg):
    """Asking for more co-resident CTAs than fit is refused at launch."""
    from paper_2109_12626_gb300 import DpdrError
    p, m = 4097, 8
    dev = torch.device("cuda:0")
    xs = [torch.zeros(m, dtype=torch.int32, device=dev) for _ in range(p)]
    ys = [torch.zeros(m, dtype=torch.int32, device=dev) for _ in range(p)]
    with pkg.Plan(p, m, "int32", 1) as plan:
        plan.set(pkg.OPT_SCHED_THREADS, 256)
        plan.set(pkg.OPT_SCHED_RANKS_PER_CTA, 1)   # 4097 CTAs of 256 threads
        if plan.info()["sched_ctas"] <= 152 * 4:
            pytest.skip("this GPU fits them all")
        with pytest.raises(DpdrError) as e:
            plan.allreduce_schedule(xs, ys)
        assert e.value.status == pkg.DPDR_ERR_NOT_COOPERATIVE
        plan.set(pkg.OPT_SCHED_RANKS_PER_CTA, 0)   # fewest that fit: works
        plan.allreduce_schedule(xs, ys)
        plan.sync()


def test_wait_limit_is_bounded_above_and_below(pkg):
    """A wait limit outside [1 us, 10 s] is refused, so no caller can make
    the schedule kernel's waits unbounded."""
    from paper_2109_12626_gb300 import DpdrError
    with pkg.Plan(7, 64, "int32", 4) as plan:
        for bad in (999, 10_000_000_001, 1 << 62):
            with pytest.raises(DpdrError) as e:
                plan.set(pkg.OPT_WAIT_LIMIT_NS, bad)
            assert e.value.status == pkg.DPDR_ERR_INVALID
        for good in (1000, 10_000_000_000):
            plan.set(pkg.OPT_WAIT_LIMIT_NS, good)
