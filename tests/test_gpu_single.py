"""GPU parity for the one-tree topology (Sec. 1.2's single doubly pipelined
tree): every fused layout and the schedule kernel (both transports, column
slices, several ranks per CTA), bit for bit against the oracle's one-tree
fold, whose float32 bracketing differs from the dual trees'."""
import numpy as np
import pytest
import torch

from gpu_util import bits, empty_like_ranks, expect_bits, host_inputs, to_device

pytestmark = pytest.mark.gpu

CASES = [("float32", 1, 33), ("float32", 2, 1001), ("int32", 3, 17), ("mat2x2u32", 5, 300),
         ("float32", 7, 4099), ("float32", 15, 65541), ("int32", 31, 2000),
         ("mat2x2u32", 63, 129), ("float32", 255, 3001), ("float32", 1023, 1027),
         ("int32", 1152, 4099), ("mat2x2f32", 127, 700)]


@pytest.fixture(scope="module")
def pkg():
    from paper_2109_12626_gb300 import build as B
    B.build()
    import paper_2109_12626_gb300 as P
    return P


def _want(orc, x, kind):
    dt = {"int32": orc.I32, "float32": orc.F32, "mat2x2u32": orc.MAT,
          "mat2x2f32": orc.MATF}[kind]
    return expect_bits(orc.tree_fold(x, dt, orc.SINGLE))


@pytest.mark.parametrize("kind,p,m", CASES)
@pytest.mark.parametrize("run", ["stream", "tile", "split", "bulk", "tree", "schedule_counters",
                                 "schedule_words", "schedule_slices", "schedule_groups"])
def test_single_tree_parity(pkg, orc, kind, p, m, run):
    x = host_inputs(kind, 71, p, m)
    want = _want(orc, x, kind)
    dev = torch.device("cuda:0")
    xs, _ = to_device(x, kind, dev)
    ys, _ = empty_like_ranks(xs)
    with pkg.Plan(p, m, kind, 5, topology="single") as plan:
        assert plan.info()["topology"] == 1
        if run.startswith("schedule"):
            if run == "schedule_slices":
                plan.set(pkg.OPT_SCHED_SLICES, 3)
            if run == "schedule_groups":
                plan.set(pkg.OPT_SCHED_RANKS_PER_CTA, min(p, 3))
            if run in ("schedule_counters", "schedule_words"):
                plan.set(pkg.OPT_SCHED_TRANSPORT, 1 if run == "schedule_counters" else 2)
            plan.allreduce_schedule(xs, ys)
        else:
            mode = {"stream": 1, "tile": 2, "split": 3, "bulk": 4, "tree": 5}[run]
            if mode == 3 and p < 2:
                pytest.skip("split layout needs p >= 2")
            plan.set(pkg.OPT_FUSED_MODE, mode)
            plan.allreduce(xs, ys)
        plan.sync()
    for i, y in enumerate(ys):
        assert np.array_equal(bits(y), want), (run, i)


def test_single_and_dual_differ_in_float32(pkg, orc):
    """The golden case of the oracle pins, through the library: the two
    topologies bracket the same float32 inputs differently."""
    x = np.array([[1.0], [2.0**-24], [2.0**-24], [2.0**-24], [0.0]], np.float32)
    dev = torch.device("cuda:0")
    xs = [torch.from_numpy(r.copy()).to(dev) for r in x]
    got = {}
    for topo in ("dual", "single"):
        ys = [torch.zeros(1, device=dev) for _ in range(5)]
        with pkg.Plan(5, 1, "float32", 1, topology=topo) as plan:
            plan.allreduce(xs, ys)
            plan.sync()
        got[topo] = float(ys[0].item())
    assert got["dual"] == 1 + 2.0**-23 and got["single"] == 1 + 2.0**-22
