"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times (plans with automatic layout selection), on sampled
columns: all p ranks at >= 16384 random columns plus the first and last
element of every pipeline block and both vector ends.  The oracle computes
the sampled columns from inputs regenerated on the host (the generator is a
pure function of seed, rank and column), and every output row must also be
identical to every other (a property that holds at any size)."""
import math

import numpy as np
import pytest
import torch

from gpu_util import bits, expect_bits

from paper_2109_12626_gb300 import inputs as I

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    from paper_2109_12626_gb300 import build as B
    B.build()
    import paper_2109_12626_gb300 as P
    return P


def _device_inputs(w, m, dev):
    """One tensor per rank: [m] for scalars, [m, 4] for 2x2 matrices (so a
    column index picks a whole element)."""
    kw = I.workload_kwargs(w)
    return [I.rank_values(w["kind"], w["seed"], i, m, device=dev, **kw).contiguous()
            for i in range(w["p"])]


def _columns(m, b, k=16384, seed=0):
    rng = np.random.default_rng(seed)
    c = set(rng.integers(0, m, min(k, m)).tolist())
    q, r = divmod(m, b)
    for j in range(b):
        s0 = j * q + min(j, r)
        s1 = (j + 1) * q + min(j + 1, r)
        c.update((s0, s1 - 1))
    c.update(range(max(0, m - 5), m))
    c.update(range(min(5, m)))
    return np.array(sorted(c), dtype=np.int64)


def _sampled_check(orc, w, m, xs, ys, cols):
    p, kind = w["p"], w["kind"]
    kw = I.workload_kwargs(w)
    ct = torch.from_numpy(cols)
    host = torch.stack([I.rank_values(kind, w["seed"], i, ct, **kw) for i in range(p)])
    dt = {"int32": orc.I32, "float32": orc.F32, "mat2x2u32": orc.MAT,
          "mat2x2f32": orc.MATF}[kind]
    hx = host.numpy()
    if kind == "mat2x2u32":
        hx = hx.view(np.uint32).reshape(p, len(cols), 4)
    elif kind == "mat2x2f32":
        hx = np.ascontiguousarray(hx).reshape(p, len(cols), 4)
    want = expect_bits(orc.tree_fold(hx, dt))
    cd = ct.to(xs[0].device)
    # the device generated the same inputs
    for i in range(0, p, max(1, p // 16)):
        assert np.array_equal(bits(xs[i][cd]), expect_bits(hx[i]))
    for i in range(p):
        got = bits(ys[i][cd])
        bad = np.nonzero(got != want)[0]
        assert bad.size == 0, "rank %d: %d of %d sampled columns differ" % (i, bad.size, len(cols))
        if i:
            assert torch.equal(ys[i], ys[0]), "rank %d differs from rank 0" % i


@pytest.mark.parametrize("name,kernels", [
    # at the workload's b = 1024 the schedule kernel's column slices are short
    # (per-lane copies); at the plan's default b they are long (bulk copies)
    ("p32_m134217728_f32", ("fused", "schedule", "schedule_default_b")),
    ("p1152_m4194304_f32", ("fused", "schedule")),
    ("p36_m65536_mat2x2u32", ("fused", "schedule")),
    ("p36_m65536_mat2x2f32", ("fused", "schedule")),
    ("p7_m1000_int32", ("fused", "schedule")),
])
def test_full_size_workloads(pkg, orc, name, kernels):
    w = dict(I.WORKLOADS[name])
    m, p = w["m"], w["p"]
    dev = torch.device("cuda:0")
    xs = _device_inputs(w, m, dev)
    ys = [torch.empty_like(x) for x in xs]
    for k in kernels:
        with pkg.Plan(p, m, w["kind"], 0 if k == "schedule_default_b" else w.get("b") or 0) as plan:
            cols = _columns(m, plan.query()["b"])
            for y in ys:
                y.fill_(-1)
            (plan.allreduce if k == "fused" else plan.allreduce_schedule)(xs, ys)
            plan.sync()
            _sampled_check(orc, w, m, xs, ys, cols)
    del xs, ys
    torch.cuda.empty_cache()


SWEEP = [1 << k for k in range(0, 24)]


@pytest.mark.parametrize("m", SWEEP, ids=["m2^%d" % k for k in range(24)])
def test_p1152_int32_sweep(pkg, orc, m):
    """p = 1152 int32 sums over m = 2^0 .. 2^23 (the paper's Table 2 range),
    the fused kernel in its automatic layout and the schedule kernel at the
    block counts {1, 4, 16, 64, 256} within [1, m] and the block-count rule
    (the rule only, above m = 2^16, to bound the test's time)."""
    w = dict(I.WORKLOADS["p1152_int32_sweep"])
    p = w["p"]
    dev = torch.device("cuda:0")
    xs = _device_inputs(w, m, dev)
    ys = [torch.empty_like(x) for x in xs]
    rule = pkg.block_count_rule(p, m)
    bl = [b for b in (1, 4, 16, 64, 256) if b <= m] + [rule]
    if m > (1 << 16):
        bl = [rule]
    with pkg.Plan(p, m, "int32", rule) as plan:
        cols = _columns(m, rule) if m > 4096 else np.arange(m, dtype=np.int64)
        plan.allreduce(xs, ys)
        plan.sync()
        _sampled_check(orc, w, m, xs, ys, cols)
    for b in sorted(set(bl)):
        with pkg.Plan(p, m, "int32", b) as plan:
            for y in ys:
                y.fill_(-1)
            plan.allreduce_schedule(xs, ys)
            plan.sync()
            _sampled_check(orc, w, m, xs, ys, _columns(m, b) if m > 4096 else np.arange(m))
    del xs, ys
    torch.cuda.empty_cache()


def test_more_than_2_31_elements_per_rank(pkg, orc):
    """m = 2^31 + 19 int32 per rank (8.6 GB each, p = 3): element and byte
    offsets past 2^31 and 2^33, every fused layout that takes p = 3 and the
    schedule kernel with both transports' block sizes, checked on sampled
    columns around those boundaries and at random."""
    w = dict(I.WORKLOADS["p7_m1000_int32"])
    w["p"], m = 3, (1 << 31) + 19
    dev = torch.device("cuda:0")
    xs = _device_inputs(w, m, dev)
    ys = [torch.empty_like(x) for x in xs]
    with pkg.Plan(3, m, "int32", 0) as plan:
        b = plan.query()["b"]
        cols = _columns(m, b, k=4096)
        edges = [c for e in ((1 << 31) - 1, 1 << 31, (1 << 31) + 16) for c in range(e - 3, e + 4)
                 if c < m]
        cols = np.unique(np.concatenate([cols, np.array(edges, np.int64)]))
        for run, mode in (("fused", 0), ("fused", 2), ("fused", 4), ("fused", 5),
                          ("schedule", 0)):
            for y in ys:
                y.fill_(-1)
            if run == "fused":
                plan.set(pkg.OPT_FUSED_MODE, mode)
                plan.allreduce(xs, ys)
            else:
                plan.allreduce_schedule(xs, ys)
            plan.sync()
            _sampled_check(orc, w, m, xs, ys, cols)
    del xs, ys
    torch.cuda.empty_cache()
