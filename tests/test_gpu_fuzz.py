"""Seeded random configurations of both kernels against the oracle.

Each case draws, from its own seeded generator, the rank count p (1 to
3000), m, the block count b, the element type, the topology, the fused
layout, the schedule kernel's transport, CTA layout, column slices and ranks
per CTA, and the buffer layout (separate, in place, or only 4-byte aligned), then
checks every output of both kernels bit for bit against the oracle's fold.
The draws reach combinations no hand-written case names -- blocks of two
lengths cut into slices, ragged tails under every layout, deep trees with
few columns -- and a mismatch names its case number, which reproduces it.
DPDR_FUZZ_CASES and DPDR_FUZZ_LARGE_CASES set the number of cases (default
128 up to 16 MB of inputs and 32 up to 256 MB)."""
import os

import numpy as np
import pytest
import torch

from gpu_util import bits, expect_bits, host_inputs, to_device

pytestmark = pytest.mark.gpu

N_CASES = int(os.environ.get("DPDR_FUZZ_CASES", "128"))  # more for a longer hunt
KINDS = ("int32", "float32", "mat2x2u32", "mat2x2f32")
ESIZE = {"int32": 4, "float32": 4, "mat2x2u32": 16, "mat2x2f32": 16}


def draw(k: int) -> dict:
    rng = np.random.default_rng(7000 + k)
    kind = KINDS[int(rng.integers(4))]
    band = int(rng.integers(3))
    p = int(rng.integers(*((1, 9), (9, 300), (300, 3001))[band]))
    budget = (16 << 20) // ESIZE[kind] // p  # at most 16 MB of inputs
    m = int(max(1, min(rng.integers(1, 2 << int(rng.integers(0, 18))), budget)))
    slices = int(rng.integers(1, 9)) if rng.random() < 0.3 else 0
    rpc = int(rng.integers(1, 5)) if rng.random() < 0.2 else 0
    rpc = min(rpc, p)
    # a forced layout of the schedule kernel must still fit co-resident
    ctas = -(-p // max(rpc, 1)) * max(slices, 1) if rpc else 0
    if ctas > 1000:
        rpc = 0
    c = dict(kind=kind, p=p, m=m, b=int(rng.integers(1, min(m, 400) + 1)),
             topology="single" if rng.random() < 0.25 else "dual",
             mode=int(rng.integers(0, 6)), transport=int(rng.integers(0, 3)),
             slices=slices, rpc=rpc,
             layout=("aligned", "aligned", "in_place", "four_byte")[int(rng.integers(4))])
    # the schedule kernels' CTA layout: automatic (by work where it fits) or
    # rank ranges, drawn last so the draws above stay as they were
    c["sched_layout"] = 1 if rng.random() < 0.3 else 0
    c["sched_copy"] = int(rng.integers(0, 3))  # drawn after the layout, as above
    return c


@pytest.fixture(scope="module")
def pkg():
    from paper_2109_12626_gb300 import build as B
    B.build()
    import paper_2109_12626_gb300 as P
    return P


def _buffers(x, kind, layout, dev):
    pad = 1 if layout == "four_byte" else 0
    xs, keep = to_device(x, kind, dev, pad_front=pad)
    if layout == "in_place":
        return xs, xs, keep
    ys, keep2 = [], []
    for t in xs:
        if pad:
            base = torch.full((t.numel() + pad,), -3, dtype=t.dtype, device=dev)
            ys.append(base[pad:])
            keep2.append(base)
        else:
            ys.append(torch.full_like(t, -3))
    return xs, ys, keep + keep2


@pytest.mark.parametrize("k", range(N_CASES))
def test_random_configuration(pkg, orc, k):
    c = draw(k)
    kind, p, m = c["kind"], c["p"], c["m"]
    x = host_inputs(kind, 7000 + k, p, m)
    dt = {"int32": orc.I32, "float32": orc.F32, "mat2x2u32": orc.MAT,
          "mat2x2f32": orc.MATF}[kind]
    topo = orc.SINGLE if c["topology"] == "single" else orc.DUAL
    want = expect_bits(orc.tree_fold(x, dt, topo))
    dev = torch.device("cuda:0")
    with pkg.Plan(p, m, kind, c["b"], topology=c["topology"]) as plan:
        mode = c["mode"]
        if mode == 3 and plan.info()["max_depth"] < 3:
            mode = 0  # the split layout needs trees of depth >= 3
        for run in ("fused", "schedule"):
            xs, ys, _keep = _buffers(x, kind, c["layout"], dev)
            if run == "fused":
                plan.set(pkg.OPT_FUSED_MODE, mode)
                plan.allreduce(xs, ys)
            else:
                plan.set(pkg.OPT_SCHED_TRANSPORT, c["transport"])
                plan.set(pkg.OPT_SCHED_LAYOUT, c["sched_layout"])
                plan.set(pkg.OPT_SCHED_COPY, c["sched_copy"])
                if c["slices"]:
                    plan.set(pkg.OPT_SCHED_SLICES, c["slices"])
                if c["rpc"]:
                    plan.set(pkg.OPT_SCHED_RANKS_PER_CTA, c["rpc"])
                plan.allreduce_schedule(xs, ys)
            plan.sync()
            for i, y in enumerate(ys):
                got = bits(y)
                bad = np.nonzero(got != want)[0]
                assert bad.size == 0, "case %d %s %s: rank %d, %d words differ, first %d" % (
                    k, c, run, i, bad.size, bad[0])
            if c["layout"] != "in_place":
                for i in range(p):
                    assert np.array_equal(bits(xs[i]), expect_bits(x[i])), (k, run, i)


N_LARGE = int(os.environ.get("DPDR_FUZZ_LARGE_CASES", "32"))


def draw_large(k: int) -> dict:
    """Up to 256 MB of inputs: long pipelines of large blocks, where slices
    that run apart by several blocks meet reused buffers."""
    rng = np.random.default_rng(9000 + k)
    kind = KINDS[int(rng.integers(4))]
    p = int(rng.integers(2, 1500))
    budget = (256 << 20) // ESIZE[kind] // p
    m = int(rng.integers(max(1, budget // 8), budget + 1))
    # half the cases with blocks of at least 4096 elements (several column
    # slices per rank under the automatic layout)
    bmax = min(m, 2000) if rng.random() < 0.5 else max(1, m // 4096)
    c = dict(kind=kind, p=p, m=m, b=int(rng.integers(1, bmax + 1)),
             mode=int(rng.integers(0, 6)), transport=int(rng.choice([0, 1, 1, 2])),
             slices=int(rng.integers(1, 33)) if rng.random() < 0.5 else 0)
    c["sched_layout"] = 1 if rng.random() < 0.3 else 0  # drawn last, as above
    c["sched_copy"] = int(rng.integers(0, 3))
    return c


def _numpy_inputs(kind, rng, p, m):
    if kind == "int32":
        return rng.integers(-(1 << 20), 1 << 20, (p, m), dtype=np.int32)
    if kind == "float32":
        return rng.standard_normal((p, m)).astype(np.float32)
    if kind == "mat2x2u32":
        return rng.integers(0, 1 << 32, (p, m, 4), dtype=np.uint32)
    eye = np.array([1, 0, 0, 1], np.float32)  # near the identity: products stay finite
    return (eye + 0.01 * rng.standard_normal((p, m, 4))).astype(np.float32)


@pytest.mark.parametrize("k", range(N_LARGE))
def test_random_large_configuration(pkg, orc, k):
    c = draw_large(k)
    kind, p, m = c["kind"], c["p"], c["m"]
    x = _numpy_inputs(kind, np.random.default_rng(9500 + k), p, m)
    dt = {"int32": orc.I32, "float32": orc.F32, "mat2x2u32": orc.MAT,
          "mat2x2f32": orc.MATF}[kind]
    want = expect_bits(orc.tree_fold(x, dt)).reshape(1, -1)
    dev = torch.device("cuda:0")
    xt = torch.from_numpy(np.ascontiguousarray(x).view(np.int32).reshape(p, -1)).to(dev)
    xs = list(xt.unbind(0))
    with pkg.Plan(p, m, kind, c["b"]) as plan:
        mode = c["mode"]
        if mode == 3 and plan.info()["max_depth"] < 3:
            mode = 0
        for run in ("fused", "schedule"):
            yt = torch.full_like(xt, -3)
            if run == "fused":
                plan.set(pkg.OPT_FUSED_MODE, mode)
                plan.allreduce(xs, list(yt.unbind(0)))
            else:
                plan.set(pkg.OPT_SCHED_TRANSPORT, c["transport"])
                plan.set(pkg.OPT_SCHED_LAYOUT, c["sched_layout"])
                plan.set(pkg.OPT_SCHED_COPY, c["sched_copy"])
                if c["slices"]:
                    plan.set(pkg.OPT_SCHED_SLICES, c["slices"])
                plan.allreduce_schedule(xs, list(yt.unbind(0)))
            plan.sync()
            got = yt.cpu().numpy()
            bad = np.nonzero((got != want).any(axis=1))[0]
            assert bad.size == 0, "large case %d %s %s: %d ranks differ, first %d" % (
                k, c, run, bad.size, bad[0])
