"""GPU parity: both kernels of the C ABI against the CPU oracle, element by
element and bit for bit (float32 included: every kernel keeps the dual-tree
bracketing of Sec. 1.1 / Algorithm 1, so the bits must agree).

Sizes are ones the oracle finishes in seconds but that span several tiles
and a ragged tail; the edge cases are p = 1, 2, 3, m = 0 and 1, in-place
buffers, 4-byte-aligned (not 16-byte) buffers, and every block count from 1
to m."""
import numpy as np
import pytest
import torch

from gpu_util import bits, empty_like_ranks, expect_bits, host_inputs, to_device

pytestmark = pytest.mark.gpu

LOHI3 = dict(lo=-(1 << 20), hi=1 << 20)
CASES = [
    # id, kind, seed, p, m, kwargs, schedule block counts
    ("p7_m1000_int32", "int32", 1, 7, 1000, dict(lo=-1000, hi=1000), [4, 1, 3, 1000]),
    ("p36_m65536_mat", "mat2x2u32", 2, 36, 65536, {}, [16, 1, 5]),
    ("p1152_m1_int32", "int32", 3, 1152, 1, LOHI3, [1]),
    ("p1152_m3_int32", "int32", 3, 1152, 3, LOHI3, [1, 3]),
    ("p1152_m4099_int32", "int32", 3, 1152, 4099, LOHI3, [1, 4, 16, 64]),
    ("p1152_m4099_f32", "float32", 4, 1152, 4099, dict(sigma=1.0), [7, 0]),
    ("p32_m65541_f32", "float32", 5, 32, 65541, dict(sigma=1e-3), [64, 256]),
    ("p32_m300000_f32", "float32", 5, 32, 300000, dict(sigma=1e-3), [1024]),
    ("p1_m17_f32", "float32", 6, 1, 17, {}, [1, 5]),
    ("p2_m333_f32", "float32", 6, 2, 333, {}, [1, 2, 333]),
    ("p3_m10_mat", "mat2x2u32", 6, 3, 10, {}, [1, 10]),
    ("p5_m1_int32", "int32", 6, 5, 1, dict(lo=-5, hi=5), [1]),
    ("p100_m77_mat", "mat2x2u32", 7, 100, 77, {}, [1, 7, 77]),
    ("p255_m2050_f32", "float32", 8, 255, 2050, {}, [3, 16]),
    ("p36_m65536_matf", "mat2x2f32", 6, 36, 65536, {}, [16, 1, 7]),
    ("p1152_m1025_matf", "mat2x2f32", 6, 1152, 1025, {}, [1, 4]),
    ("p3_m9_matf", "mat2x2f32", 6, 3, 9, {}, [1, 9]),
    # ragged tails whose single-element thread sits in another warp than the
    # vector threads of its block (their shared-memory slots must not meet)
    ("p3_m801_f32", "float32", 9, 3, 801, {}, [2]),
    ("p32_m803_int32", "int32", 9, 32, 803, {}, [3]),
    ("p1152_m1021_f32", "float32", 9, 1152, 1021, {}, [2]),
    # near the largest p the allocation-free entry point takes (8192): deep
    # trees (depth 11), eight ranks per schedule CTA, a 131 KB tile row
    ("p8190_m33_int32", "int32", 10, 8190, 33, dict(lo=-1000, hi=1000), [1, 2]),
    ("p8190_m7_f32", "float32", 10, 8190, 7, dict(sigma=1.0), [1]),
    # 4097 16-byte units per rank plus a ragged tail: the hierarchical tile
    # takes its wide width (16 units per CTA) at a deep tree
    ("p1152_m16390_f32", "float32", 11, 1152, 16390, dict(sigma=1.0), [2]),
]


@pytest.fixture(scope="module")
def pkg():
    from paper_2109_12626_gb300 import build as B
    B.build()
    import paper_2109_12626_gb300 as P
    return P


def _want(orc, x, kind):
    dt = {"int32": orc.I32, "float32": orc.F32, "mat2x2u32": orc.MAT,
          "mat2x2f32": orc.MATF}[kind]
    return expect_bits(orc.tree_fold(x, dt))


def _check_all(ys, want, guards=None):
    for i, y in enumerate(ys):
        got = bits(y)
        assert got.shape == want.shape
        bad = np.nonzero(got != want)[0]
        assert bad.size == 0, "rank %d: %d mismatches, first at %d" % (i, bad.size, bad[0])


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("mode", [1, 2, 3, 4, 5], ids=["stream", "tile", "split", "bulk", "tree"])
def test_fused_matches_oracle(pkg, orc, case, mode):
    _, kind, seed, p, m, kw, _ = case
    dev = torch.device("cuda:0")
    x = host_inputs(kind, seed, p, m, **kw)
    want = _want(orc, x, kind)
    xs, _ = to_device(x, kind, dev)
    ys, _ = empty_like_ranks(xs)
    with pkg.Plan(p, m, kind, 4) as plan:
        if mode == 3 and plan.info()["max_depth"] < 3:
            pytest.skip("split layout needs trees of depth >= 3")
        plan.set(pkg.OPT_FUSED_MODE, mode)
        plan.allreduce(xs, ys)
        plan.sync()
        assert plan.info()["vector_path"] == 1
    _check_all(ys, want)
    for i in range(p):  # inputs untouched
        assert np.array_equal(bits(xs[i]), expect_bits(x[i]))


TRANSPORTS = {"counters": 1, "words": 2}
# (transport, CTA layout, block-pass copies): the counters transport laid out
# by work where it fits (the default) and on contiguous rank ranges, its block
# passes by per-lane copies (the automatic choice at these sizes) and by bulk
# copies, and flagged words
SCHED_VARIANTS = {"counters": (1, 0, 0), "counters_bulk": (1, 0, 2),
                  "counters_ranges_lane": (1, 1, 1), "counters_ranges_bulk": (1, 1, 2),
                  "words": (2, 0, 0)}


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
@pytest.mark.parametrize("variant", list(SCHED_VARIANTS))
def test_schedule_matches_oracle(pkg, orc, case, variant):
    _, kind, seed, p, m, kw, blist = case
    transport, layout, copy = SCHED_VARIANTS[variant]
    dev = torch.device("cuda:0")
    x = host_inputs(kind, seed, p, m, **kw)
    want = _want(orc, x, kind)
    xs, _ = to_device(x, kind, dev)
    for b in blist:
        ys, _ = empty_like_ranks(xs)
        with pkg.Plan(p, m, kind, b) as plan:
            plan.set(pkg.OPT_SCHED_TRANSPORT, transport)
            plan.set(pkg.OPT_SCHED_LAYOUT, layout)
            plan.set(pkg.OPT_SCHED_COPY, copy)
            assert plan.info()["sched_transport"] == transport
            if layout == 1:
                assert plan.info()["sched_layout"] == 1
            if copy:
                assert plan.info()["sched_copy"] == copy
            plan.allreduce_schedule(xs, ys)
            plan.sync()
        _check_all(ys, want)
    for i in range(p):
        assert np.array_equal(bits(xs[i]), expect_bits(x[i]))


FUSED_RUNS = {"fused_stream": 1, "fused_tile": 2, "fused_split": 3, "fused_bulk": 4,
              "fused_tree": 5}
SCHED_RUNS = {"schedule_counters": 1, "schedule_words": 2}
RUNS = list(FUSED_RUNS) + list(SCHED_RUNS)


def _run(pkg, plan, run, xs, ys):
    if run in SCHED_RUNS:
        plan.set(pkg.OPT_SCHED_TRANSPORT, SCHED_RUNS[run])
        plan.allreduce_schedule(xs, ys)
    else:
        if FUSED_RUNS[run] == 3 and plan.info()["max_depth"] < 3:
            pytest.skip("split layout needs trees of depth >= 3")
        plan.set(pkg.OPT_FUSED_MODE, FUSED_RUNS[run])
        plan.allreduce(xs, ys)


@pytest.mark.parametrize("kind,p,m", [("int32", 7, 1000), ("float32", 1152, 4099),
                                      ("mat2x2u32", 36, 999), ("float32", 2, 5),
                                      ("mat2x2f32", 100, 513)])
@pytest.mark.parametrize("run", RUNS)
def test_in_place(pkg, orc, kind, p, m, run):
    """y[i] == x[i]: Algorithm 1 works in place (Y <- x_i, y ends in Y)."""
    x = host_inputs(kind, 11, p, m)
    want = _want(orc, x, kind)
    xs, _ = to_device(x, kind, torch.device("cuda:0"))
    with pkg.Plan(p, m, kind, 3) as plan:
        _run(pkg, plan, run, xs, xs)
        plan.sync()
    _check_all(xs, want)


@pytest.mark.parametrize("kind,p,m", [("int32", 7, 1001), ("float32", 1152, 133),
                                      ("mat2x2u32", 36, 257), ("float32", 32, 9999),
                                      ("mat2x2f32", 36, 257)])
@pytest.mark.parametrize("run", RUNS)
def test_four_byte_aligned_buffers(pkg, orc, kind, p, m, run):
    """Buffers only 4-byte aligned take the single-element paths."""
    x = host_inputs(kind, 12, p, m)
    want = _want(orc, x, kind)
    dev = torch.device("cuda:0")
    xs, keep_x = to_device(x, kind, dev, pad_front=1)
    ys, keep_y = empty_like_ranks(xs, pad_front=3)
    with pkg.Plan(p, m, kind, 4) as plan:
        _run(pkg, plan, run, xs, ys)
        plan.sync()
        assert plan.info()["vector_path"] == 0
    _check_all(ys, want)


@pytest.mark.parametrize("run", RUNS)
def test_guard_words_untouched(pkg, orc, run):
    """No kernel writes past the m elements of an output."""
    kind, p, m = "float32", 36, 4097
    x = host_inputs(kind, 13, p, m)
    want = _want(orc, x, kind)
    dev = torch.device("cuda:0")
    xs, _ = to_device(x, kind, dev)
    bases = [torch.full((m + 64,), 7.25, device=dev) for _ in range(p)]
    ys = [bb[:m] for bb in bases]
    with pkg.Plan(p, m, kind, 5) as plan:
        _run(pkg, plan, run, xs, ys)
        plan.sync()
    _check_all(ys, want)
    for bb in bases:
        assert bool((bb[m:] == 7.25).all())


AUTO = [  # p, m, kind, layout the automatic choice takes on a 152-SM GPU
          # (1 stream, 2 tile, 3 split, 5 hierarchical tile)
    (32, 1 << 27, "float32", 1), (36, 65536, "mat2x2u32", 1),
    (1152, 4096, "int32", 2), (1152, 8192, "int32", 5), (1152, 32768, "int32", 5),
    (288, 4096, "int32", 2), (288, 4100, "int32", 5), (768, 4096, "int32", 2),
    (1152, 32772, "int32", 3), (128, 16384, "float32", 5), (192, 32768, "int32", 2),
    (288, 32768, "int32", 5), (288, 65536, "int32", 3), (4094, 2048, "int32", 5),
    (1152, 1 << 22, "float32", 3),
    # the shared-memory tile where it needs fewer waves of resident CTAs
    # than the hierarchical tile (p = 288: one against two)
    (288, 24576, "int32", 2), (288, 16384, "int32", 5), (576, 24576, "int32", 5),
    (576, 32768, "int32", 5), (768, 24576, "int32", 5), (256, 28672, "int32", 2),
    # below p = 128: column streaming from a fifth of the columns that fill
    # the GPU (31129 units on 152 SMs), the shared-memory tile below
    (64, 131072, "int32", 1), (64, 65536, "int32", 2),
    # shallow trees (p <= 16): column streaming at every size
    (7, 1000, "int32", 1), (16, 16, "int32", 1), (2, 3, "float32", 1), (32, 1000, "int32", 2),
    # from p = 2048 the split layout where the wide hierarchical tile's second
    # wave would be less than 60 % full
    (4094, 24576, "int32", 3), (4094, 32768, "int32", 5), (2304, 20480, "int32", 3),
    (1152, 24576, "int32", 5)]


@pytest.mark.parametrize("p,m,kind,mode", AUTO)
def test_auto_layout_choice(pkg, p, m, kind, mode):
    if torch.cuda.get_device_properties(0).multi_processor_count != 152:
        pytest.skip("the expected choices are for a 152-SM GPU")
    with pkg.Plan(p, m, kind, 1) as plan:
        assert plan.info()["auto_mode"] == mode


@pytest.mark.parametrize("p,m", [(1152, 9728), (1152, 9732), (1152, 16384), (32, 65541),
                                 (7, 70000), (4094, 100), (300, 40000)])
def test_tree_width(pkg, p, m):
    """On device buffers the hierarchical tile takes 8 column units per CTA
    while those CTAs fit in one wave of resident CTAs (2 per SM), else 16."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    units = m * 4 // 16
    with pkg.Plan(p, m, "float32", 1) as plan:
        plan.set(pkg.OPT_FUSED_MODE, 5)
        assert plan.info()["tree_width"] == (16 if units > 8 * 2 * sms else 8)


@pytest.mark.parametrize("mode", [2, 5], ids=["tile", "tree"])
def test_interleaved_plans_keep_their_shared_memory(pkg, orc, mode):
    """Plans of one element type whose fused kernels need different dynamic
    shared memory, called alternately (larger, smaller, larger): the kernel's
    limit belongs to the function, so the smaller plan must not take back
    what the larger one was granted.  Tile rows of 3001 and 2001 ranks need
    96 KB and 64 KB; the hierarchical tile at p = 4094 and 1152 needs 64 KB
    and 56 KB (all above the 48 KB default)."""
    kind, m = "int32", 1001
    dev = torch.device("cuda:0")
    sizes = (3000, 2000) if mode == 2 else (4094, 1152)
    data = {}
    plans = {}
    try:
        for p in sizes:
            x = host_inputs(kind, 30 + p % 7, p, m, lo=-1000, hi=1000)
            xs, _ = to_device(x, kind, dev)
            data[p] = (xs, _want(orc, x, kind))
            plans[p] = pkg.Plan(p, m, kind, 1)
            plans[p].set(pkg.OPT_FUSED_MODE, mode)
        for p in (sizes[0], sizes[1], sizes[0], sizes[1]):
            xs, want = data[p]
            ys, _ = empty_like_ranks(xs)
            plans[p].allreduce(xs, ys)
            plans[p].sync()
            _check_all(ys, want)
    finally:
        for plan in plans.values():
            plan.close()


def test_m_zero_is_a_no_op(pkg):
    dev = torch.device("cuda:0")
    xs = [torch.zeros(4, device=dev) for _ in range(5)]
    ys = [torch.full((4,), 3.0, device=dev) for _ in range(5)]
    with pkg.Plan(5, 0, "float32", 0) as plan:
        assert plan.query()["b"] == 1
        plan.allreduce(xs, ys)
        plan.allreduce_schedule(xs, ys)
        plan.sync()
    assert all(bool((y == 3.0).all()) for y in ys)


def test_repeated_calls_and_pointer_changes(pkg, orc):
    """The rank-pointer table is re-staged when the buffers change."""
    kind, p, m = "int32", 7, 1000
    dev = torch.device("cuda:0")
    with pkg.Plan(p, m, kind, 4) as plan:
        for seed in (21, 22, 23):
            x = host_inputs(kind, seed, p, m, lo=-1000, hi=1000)
            want = _want(orc, x, kind)
            xs, _ = to_device(x, kind, dev)
            for _ in range(2):
                ys, _ = empty_like_ranks(xs)
                plan.allreduce(xs, ys)
                _check_all(ys, want)
                ys2, _ = empty_like_ranks(xs)
                plan.allreduce_schedule(xs, ys2)
                plan.sync()
                _check_all(ys2, want)


@pytest.mark.parametrize("kind,p,m,chunk", [("float32", 32, 10007, 0), ("float32", 32, 10007, 4096),
                                            ("int32", 1152, 3001, 65536), ("mat2x2u32", 7, 2049, 4096),
                                            ("float32", 3, 257, 4096), ("mat2x2f32", 36, 1001, 0),
                                            # device buffers: 16 units per CTA; host: 8
                                            ("float32", 300, 16390, 0)])
@pytest.mark.parametrize("path", ["auto", "copy"])
@pytest.mark.parametrize("pinned", [True, False])
@pytest.mark.parametrize("in_place", [False, True])
def test_host_buffers_end_to_end(pkg, orc, kind, p, m, chunk, path, pinned, in_place):
    """dpdr_allreduce_host: host inputs and outputs.  "auto" runs the kernel
    directly on the host buffers when the GPU can address them (pinned, or
    pageable on a GPU that walks the CPU page tables), "copy" forces the
    pipeline of chunked copies through device buffers."""
    x = host_inputs(kind, 31, p, m)
    want = _want(orc, x, kind)
    dev = torch.device("cuda:0")
    xh = [torch.from_numpy(np.ascontiguousarray(x[i]).view(np.int32).reshape(-1).copy())
          for i in range(p)]
    yh = [torch.full_like(t, -9) for t in xh]
    if pinned:
        xh = [t.pin_memory() for t in xh]
        yh = [t.pin_memory() for t in yh]
    if in_place:
        yh = xh
    xd = [torch.empty_like(t, device=dev) for t in xh]
    yd = xd if in_place else [torch.empty_like(t, device=dev) for t in xh]
    with pkg.Plan(p, m, kind, 0) as plan:
        if chunk:
            plan.set(pkg.OPT_HOST_CHUNK_BYTES, chunk)
        if path == "copy":
            plan.set(pkg.OPT_HOST_PATH, 1)
        for _ in range(2):
            if in_place:  # the inputs are overwritten: restore them
                for i in range(p):
                    xh[i].copy_(torch.from_numpy(np.ascontiguousarray(x[i]).view(np.int32).reshape(-1)))
            plan.allreduce_host(xh, yh, xd, yd)
            plan.sync()
            _check_all(yh, want)
        took = plan.info()["host_path"]
        assert took == (1 if path == "copy" else took)
        if path == "auto" and pinned:
            assert took == 2  # pinned memory is always addressable


def test_host_buffers_direct_needs_no_device_buffers(pkg, orc):
    kind, p, m = "float32", 32, 4099
    x = host_inputs(kind, 33, p, m)
    want = _want(orc, x, kind)
    xh = [torch.from_numpy(x[i].copy()).pin_memory() for i in range(p)]
    yh = [torch.zeros(m).pin_memory() for _ in range(p)]
    with pkg.Plan(p, m, kind, 0) as plan:
        plan.allreduce_host(xh, yh)
        plan.sync()
        assert plan.info()["host_path"] == 2
    _check_all(yh, want)


def test_invalid_arguments(pkg):
    from paper_2109_12626_gb300 import DpdrError, _native as N
    dev = torch.device("cuda:0")
    L = N.lib()
    assert not L.dpdr_plan(0, 10, N.DPDR_INT32, N.DPDR_OP_SUM, 1)
    assert L.dpdr_last_error() == N.DPDR_ERR_INVALID
    assert not L.dpdr_plan(4, 10, N.DPDR_INT32, N.DPDR_OP_MATMUL, 1)
    assert not L.dpdr_plan(4, -1, N.DPDR_FLOAT32, N.DPDR_OP_SUM, 1)
    base = torch.zeros(4096, device=dev)
    with pkg.Plan(3, 100, "float32", 1) as plan:
        xs = [torch.zeros(100, device=dev) for _ in range(3)]
        # two outputs overlapping
        with pytest.raises(DpdrError) as e:
            plan.allreduce(xs, [base[0:100], base[50:150], base[200:300]])
        assert e.value.status == N.DPDR_ERR_INVALID
        # an output overlapping another rank's input
        with pytest.raises(DpdrError):
            plan.allreduce([base[0:100], xs[1], xs[2]], [xs[0], base[1000:1100], base[40:140]])
        # 2-byte misalignment
        raw = torch.zeros(1000, dtype=torch.int16, device=dev)
        with pytest.raises(DpdrError):
            plan.allreduce([raw.data_ptr() + 2] + xs[1:], [base[0:100], base[200:300], base[400:500]])
        # NULL buffer
        with pytest.raises(DpdrError):
            plan.allreduce([0] + xs[1:], [base[0:100], base[200:300], base[400:500]])
        # the plan still works afterwards
        ys = [base[0:100], base[200:300], base[400:500]]
        plan.allreduce(xs, ys)
        plan.sync()
        with pytest.raises(DpdrError):
            plan.set(N.OPT_FUSED_MODE, 6)
        with pytest.raises(DpdrError):
            plan.set(999, 1)


@pytest.mark.parametrize("kind,p,m,b,slices", [
    ("float32", 32, 65541, 4, 7), ("int32", 7, 1000, 4, 3), ("mat2x2u32", 36, 4099, 16, 5),
    ("float32", 1152, 4099, 3, 2), ("int32", 2, 333, 1, 64), ("float32", 1, 17, 2, 3)])
@pytest.mark.parametrize("layout", ["aligned", "in_place", "four_byte"])
@pytest.mark.parametrize("variant", list(SCHED_VARIANTS))
def test_schedule_column_slices(pkg, orc, kind, p, m, b, slices, layout, variant):
    """Several CTAs per virtual rank, each running the schedule on its own
    column slice of every block, give the same bits."""
    x = host_inputs(kind, 61, p, m)
    want = _want(orc, x, kind)
    dev = torch.device("cuda:0")
    pad = 1 if layout == "four_byte" else 0
    xs, keep = to_device(x, kind, dev, pad_front=pad)
    ys, keep_y = (xs, None) if layout == "in_place" else empty_like_ranks(xs, pad_front=pad)
    with pkg.Plan(p, m, kind, b) as plan:
        plan.set(pkg.OPT_SCHED_SLICES, slices)
        plan.set(pkg.OPT_SCHED_TRANSPORT, SCHED_VARIANTS[variant][0])
        plan.set(pkg.OPT_SCHED_LAYOUT, SCHED_VARIANTS[variant][1])
        plan.set(pkg.OPT_SCHED_COPY, SCHED_VARIANTS[variant][2])
        assert plan.info()["sched_slices"] == slices
        plan.allreduce_schedule(xs, ys)
        plan.sync()
    _check_all(ys, want)


def test_schedule_layout_choice(pkg, orc):
    """The counters kernels lay ranks out by work (one rank per group: a
    leaf on one warp beside an inner node on three, each root on a CTA of its
    own) while one column slice of that fits the GPU at once, and on rank
    ranges otherwise; forcing the work layout where it does not fit is
    refused and leaves the plan as it was."""
    from paper_2109_12626_gb300 import DpdrError
    for p, want in ((7, 2), (32, 2), (36, 2), (1152, 2), (2, 2), (1, 2), (8190, 1)):
        with pkg.Plan(p, 1 << 16, "int32", 64) as plan:
            plan.set(pkg.OPT_SCHED_TRANSPORT, 1)
            info = plan.info()
            assert info["sched_layout"] == want, p
            if want == 2:
                assert info["sched_ranks_per_cta"] <= 4
                assert info["sched_ctas"] % info["sched_slices"] == 0
    with pkg.Plan(32, 1 << 16, "int32", 64) as plan:
        plan.set(pkg.OPT_SCHED_TRANSPORT, 1)
        plan.set(pkg.OPT_SCHED_LAYOUT, 1)
        assert plan.info()["sched_layout"] == 1
        plan.set(pkg.OPT_SCHED_LAYOUT, 2)
        assert plan.info()["sched_layout"] == 2
        plan.set(pkg.OPT_SCHED_RANKS_PER_CTA, 2)  # ranks per CTA: rank ranges
        assert plan.info()["sched_layout"] == 1
    kind, p, m = "int32", 8190, 33
    x = host_inputs(kind, 73, p, m, lo=-1000, hi=1000)
    xs, _ = to_device(x, kind, torch.device("cuda:0"))
    ys, _ = empty_like_ranks(xs)
    with pkg.Plan(p, m, kind, 2) as plan:
        plan.set(pkg.OPT_SCHED_TRANSPORT, 1)
        before = plan.info()
        with pytest.raises(DpdrError):
            plan.set(pkg.OPT_SCHED_LAYOUT, 2)
        assert plan.info() == before
        plan.allreduce_schedule(xs, ys)
        plan.sync()
    _check_all(ys, _want(orc, x, kind))


@pytest.mark.parametrize("p", [2400, 2432, 2600])
def test_schedule_layout_at_its_limit(pkg, orc, p):
    """On both sides of the largest p whose work layout fits one slice of
    resident CTAs (128-thread CTAs, 8 per SM: a leaf and an inner node per
    CTA, a CTA per root, spare leaves four to a CTA), the automatic layout
    gives the same bits as the oracle; the work layout, where taken, has the
    CTAs per slice that its rule counts, and it is not taken where those
    cannot all reside."""
    kind, m = "int32", 37
    x = host_inputs(kind, 81, p, m, lo=-1000, hi=1000)
    xs, _ = to_device(x, kind, torch.device("cuda:0"))
    ys, _ = empty_like_ranks(xs)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    with pkg.Plan(p, m, kind, 3) as plan:
        plan.set(pkg.OPT_SCHED_TRANSPORT, 1)
        info = plan.info()
        par = plan.query()["parent"]
        c0 = plan.query()["child0"]
        leaves = sum(1 for i in range(p) if par[i] >= 0 and c0[i] < 0)
        inner = sum(1 for i in range(p) if par[i] >= 0 and c0[i] >= 0)
        ctas = 2 + inner + -(-(leaves - min(leaves, inner)) // 4)
        if ctas > 8 * sms:  # more than the 64-register budget lets reside
            assert info["sched_layout"] == 1, (p, ctas)
        if info["sched_layout"] == 2:
            assert info["sched_ctas"] == ctas * info["sched_slices"], (p, ctas)
        plan.allreduce_schedule(xs, ys)
        plan.sync()
    _check_all(ys, _want(orc, x, kind))


def test_schedule_copy_choice(pkg):
    """Block passes by per-lane copies while a column slice of a block holds
    at most 1024 16-byte units, by bulk copies beyond; the option forces
    either, and other values are refused."""
    from paper_2109_12626_gb300 import DpdrError
    for p, m, b, want in ((32, 1 << 23, 64, 1), (32, 1 << 23, 16, 2), (1152, 1 << 18, 18, 2),
                          (1152, 1 << 18, 72, 1), (32, 1 << 27, 1024, 1), (32, 1 << 27, 256, 2)):
        with pkg.Plan(p, m, "float32", b) as plan:
            plan.set(pkg.OPT_SCHED_TRANSPORT, 1)
            assert plan.info()["sched_copy"] == want, (p, m, b)
            plan.set(pkg.OPT_SCHED_COPY, 3 - want)
            assert plan.info()["sched_copy"] == 3 - want
            with pytest.raises(DpdrError):
                plan.set(pkg.OPT_SCHED_COPY, 3)


def test_schedule_transport_choice(pkg):
    """Flagged words while the p inputs total at most 12 MiB (24 MiB from
    p = 1024) with one rank per CTA, 8 MiB with two ranks per CTA, never with
    more; counters otherwise.  The option overrides either way."""
    MiB = 1 << 20
    cases = [(36, 12 * MiB // (36 * 4), "int32"), (1152, 24 * MiB // (1152 * 4), "int32"),
             (36, 12 * MiB // (36 * 16), "mat2x2u32")]
    for p, m_max, kind in cases:
        with pkg.Plan(p, m_max, kind, 0) as plan:
            assert plan.info()["sched_ranks_per_cta"] == 1
            assert plan.info()["sched_transport"] == 2, (p, m_max)
            plan.set(pkg.OPT_SCHED_TRANSPORT, 1)
            assert plan.info()["sched_transport"] == 1
        with pkg.Plan(p, m_max + 1, kind, 0) as plan:
            assert plan.info()["sched_transport"] == 1, (p, m_max + 1)
            plan.set(pkg.OPT_SCHED_TRANSPORT, 2)
            assert plan.info()["sched_transport"] == 2
    for p in (2048, 4094):
        with pkg.Plan(p, 1, "int32", 0) as plan:
            # the rule counts ranks per CTA of rank ranges at 128 threads
            plan.set(pkg.OPT_SCHED_THREADS, 128)
            plan.set(pkg.OPT_SCHED_LAYOUT, 1)
            rpc = plan.info()["sched_ranks_per_cta"]
            want = 2 if rpc <= 2 else 1
            assert plan.info()["sched_transport"] == want, (p, rpc)
    from paper_2109_12626_gb300 import DpdrError
    with pkg.Plan(3, 10, "int32", 0) as plan:
        with pytest.raises(DpdrError):
            plan.set(pkg.OPT_SCHED_TRANSPORT, 3)


@pytest.mark.parametrize("transport", list(TRANSPORTS))
def test_schedule_graph_replay(pkg, orc, transport):
    """A CUDA graph of two schedule calls (two plans, the second reducing the
    first's result) replayed with new input values in between: the
    flagged-word transport moves to a new epoch on the device at the end of
    every call, so a replay never accepts a previous call's words."""
    kind, p, m = "int32", 30, 777
    dev = torch.device("cuda:0")
    xs = [torch.empty(m, dtype=torch.int32, device=dev) for _ in range(p)]
    ys = [torch.empty(m, dtype=torch.int32, device=dev) for _ in range(p)]
    zs = [torch.empty(m, dtype=torch.int32, device=dev) for _ in range(p)]
    with pkg.Plan(p, m, kind, 3) as plan, pkg.Plan(p, m, kind, 2) as plan2:
        for pl in (plan, plan2):
            pl.set(pkg.OPT_SCHED_TRANSPORT, TRANSPORTS[transport])
        first, second = plan.bind(xs, ys), plan2.bind(ys, zs)
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):  # warm-up outside the capture
            first.allreduce_schedule()
            second.allreduce_schedule()
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            first.allreduce_schedule()
            second.allreduce_schedule()
        for seed in (31, 32, 33):
            x = host_inputs(kind, seed, p, m, lo=-1000, hi=1000)
            for i in range(p):
                xs[i].copy_(torch.from_numpy(x[i]))
            for t in ys + zs:
                t.fill_(-7)
            g.replay()
            torch.cuda.synchronize()
            want = _want(orc, x, kind)
            _check_all(ys, want)
            y = np.stack([want.view(np.int32)] * p)
            _check_all(zs, _want(orc, y, kind))
        plan.sync()
        plan2.sync()


def test_default_block_count(pkg):
    """b == 0: one block with flagged words; otherwise the Sec. 1.2 rule at
    kappa = 46e6 / (p esize), raised to 2 p m esize / L2 blocks."""
    import math
    l2 = torch.cuda.get_device_properties(0).L2_cache_size
    with pkg.Plan(288, 2500, "int32", 0) as plan:
        assert plan.info()["sched_transport"] == 2 and plan.query()["b"] == 1
    for p, m in ((288, 65536), (1152, 16384), (1152, 1 << 22), (36, 1 << 20)):
        with pkg.Plan(p, m, "int32", 0) as plan:
            assert plan.info()["sched_transport"] == 1
            rule = pkg.block_count_rule(p, m, 46e6 / (p * 4))
            want = max(rule, math.ceil(2 * p * m * 4 / l2))
            assert plan.query()["b"] == want, (p, m)
            plan.set(pkg.OPT_BLOCKS, 0)
            assert plan.query()["b"] == want


@pytest.mark.parametrize("kind,p,m,b", [("int32", 36, 1003, 3), ("float32", 255, 2050, 2),
                                        ("mat2x2u32", 100, 77, 7)])
@pytest.mark.parametrize("rpc", [2, 3, 4, 5])
@pytest.mark.parametrize("transport", list(TRANSPORTS))
def test_schedule_ranks_per_cta(pkg, orc, kind, p, m, b, rpc, transport):
    """CTAs that own several virtual ranks (the layout of p beyond the
    co-resident CTA count): the counters kernel splits them into rank groups
    of warps with their own barriers, up to one group per warp (rpc = 5 puts
    two ranks on one warp of a 128-thread CTA).  Same bits."""
    x = host_inputs(kind, 71, p, m)
    want = _want(orc, x, kind)
    dev = torch.device("cuda:0")
    xs, _ = to_device(x, kind, dev)
    for in_place in (False, True):
        xs_run = [t.clone() for t in xs] if in_place else xs
        ys = xs_run if in_place else empty_like_ranks(xs)[0]
        with pkg.Plan(p, m, kind, b) as plan:
            plan.set(pkg.OPT_SCHED_TRANSPORT, TRANSPORTS[transport])
            plan.set(pkg.OPT_SCHED_RANKS_PER_CTA, rpc)
            assert plan.info()["sched_ranks_per_cta"] == rpc
            plan.allreduce_schedule(xs_run, ys)
            plan.sync()
        _check_all(ys, want)


@pytest.mark.parametrize("run", RUNS)
def test_int32_sums_wrap(pkg, orc, run):
    """Full-range int32 inputs: the sums overflow and wrap modulo 2^32 (two's
    complement), the same on every path as in the oracle."""
    from paper_2109_12626_gb300 import inputs as I
    p, m = 1152, 1027
    x = np.stack([I.words_u32(12, i, m, 2)[:, 0].numpy() for i in range(p)])
    assert np.abs(x.astype(np.int64)).max() > (1 << 30)
    want = _want(orc, x, "int32")
    xs, _ = to_device(x, "int32", torch.device("cuda:0"))
    ys, _ = empty_like_ranks(xs)
    with pkg.Plan(p, m, "int32", 3) as plan:
        _run(pkg, plan, run, xs, ys)
        plan.sync()
    _check_all(ys, want)


@pytest.mark.parametrize("kind,p,m,b", [("int32", 288, 2500000, 86), ("float32", 32, 2500000, 86),
                                        ("mat2x2u32", 36, 300001, 7)])
def test_schedule_slices_with_shifting_block_bounds(pkg, orc, kind, p, m, b):
    """Blocks of two lengths (m mod b of them one element longer) cut into
    column slices, with the counters transport: a slice's range inside a
    block moves by a few elements from block to block and slices run
    independently, so each slice has its own dual-root exchange slots (with
    slots shared across slices, a slice two blocks ahead overwrote its
    neighbour's data before the other root had read it)."""
    rng = np.random.default_rng(90 + p)
    if kind == "int32":
        x = rng.integers(-1000, 1000, (p, m), dtype=np.int32)
    elif kind == "float32":
        x = rng.standard_normal((p, m)).astype(np.float32)
    else:
        x = rng.integers(0, 1 << 32, (p, m, 4), dtype=np.uint32)
    want = _want(orc, x, kind).reshape(1, -1)
    dev = torch.device("cuda:0")
    xt = torch.from_numpy(x.view(np.int32)).to(dev)
    xs = list(xt.unbind(0))
    with pkg.Plan(p, m, kind, b) as plan:
        plan.set(pkg.OPT_SCHED_TRANSPORT, 1)
        assert plan.info()["sched_slices"] > 1
        for _ in range(3):  # the overwrite was a race: several runs
            yt = torch.full_like(xt, -3)
            plan.allreduce_schedule(xs, list(yt.unbind(0)))
            plan.sync()
            got = yt.cpu().numpy().reshape(p, -1)
            bad = np.nonzero((got != want).any(axis=1))[0]
            assert bad.size == 0, "%d ranks differ, first %d" % (bad.size, bad[0])


@pytest.mark.parametrize("run", ["fused_auto", "fused_stream", "fused_tree", "fused_split",
                                 "schedule_auto"])
def test_very_many_ranks(pkg, orc, run):
    """p = 65535 ranks of 5 elements: trees of depth 15, about 54 ranks per
    schedule CTA (4 rank groups), the tile layout out of reach (a tile row
    would exceed shared memory).  Every path still gives the oracle's bits."""
    kind, p, m = "float32", 65535, 5
    # one seeded draw for all ranks (the per-rank generator takes ~30 s here);
    # both sides get the same array
    x = np.random.default_rng(81).standard_normal((p, m)).astype(np.float32)
    want = _want(orc, x, kind)
    dev = torch.device("cuda:0")
    xs = list(torch.from_numpy(x).to(dev).unbind(0))  # p views of one allocation
    ys = list(torch.full((p, m), -3.0, device=dev).unbind(0))
    with pkg.Plan(p, m, kind, 0) as plan:
        if run == "schedule_auto":
            assert plan.info()["sched_ranks_per_cta"] > 4
            plan.allreduce_schedule(xs, ys)
        else:
            mode = {"fused_auto": 0, "fused_stream": 1, "fused_tree": 5, "fused_split": 3}[run]
            if mode:
                plan.set(pkg.OPT_FUSED_MODE, mode)
            plan.allreduce(xs, ys)
        plan.sync()
    got = torch.stack(ys).cpu().numpy().view(np.int32)
    bad = np.nonzero((got != want.reshape(1, m)).any(axis=1))[0]
    assert bad.size == 0, "%d ranks differ, first %d" % (bad.size, bad[0] if bad.size else -1)
