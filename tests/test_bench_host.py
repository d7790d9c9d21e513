"""bench.py's host-side logic without a GPU: the max-over-ranks timing and
barrier with two gloo ranks on the CPU (the N > 1 replica path), the clock
sample parsing, the measured-traffic lookup, the reference arm (the CPU
oracle on a bounded sample) and the oracle-simulation timing leg."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    bench.barrier(world)
    t = bench.max_over_ranks(10.0 + 5.0 * rank, world)   # rank 1 is slower
    bench.barrier(world)
    q.put((rank, t))
    dist.destroy_process_group()


def test_max_over_ranks_gloo_two_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = dict(q.get(timeout=10) for _ in range(2))
    assert got == {0: 15.0, 1: 15.0}


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(3.5, 1) == 3.5
    bench.barrier(1)


def test_clock_summary():
    csv = "\n".join([
        "0, 2070, 2070, 900.5, 0x0, Not Active, Not Active, Not Active, Not Active",
        "0, 2055, 2070, 1100.0, 0x4, Not Active, Not Active, Not Active, Active",
        "0, 1980, 2070, 95.0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ])
    c = bench.summarize_clocks(csv)
    assert c["sm_max_mhz"] == 2070 and c["samples"] == 2   # idle sample dropped
    assert c["sm_mhz"] == pytest.approx((2070 + 2055) / 2)
    assert c["reasons"] == ["sw_power_cap"]
    assert bench.summarize_clocks("") is None


def test_profiled_traffic_tracks_the_kernel_source():
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))
    for kernel, table in rec.items():
        for wname, rs in table.items():
            rs = rs if isinstance(rs, list) else [rs]  # one record per block size
            blocks = [r.get("block_elems") for r in rs]
            for r in rs:
                blk = r.get("block_elems")
                got = bench.profiled_traffic(kernel, wname, 1000, blk)
                if r["source_hash"] == bench.kernel_source_hash(kernel):
                    assert got == pytest.approx(1000 * r["bytes_per_unit"])
                    if blk is not None:  # the schedule kernel's traffic depends on the block size
                        if all(b is None or abs(3 * blk - b) > 0.05 * b for b in blocks):
                            assert bench.profiled_traffic(kernel, wname, 1000, 3 * blk) is None
                        assert bench.profiled_traffic(kernel, wname, 1000, None) is None
                else:
                    assert got is None  # stale counters are not reported


def test_reference_arm_prints_one_json_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl",
                          "reference", "--workload", "p7_m1000_int32", "--steps", "2",
                          "--warmup", "3"], capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "GB/s" and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0


def test_oracle_simulation_timing_leg():
    """--oracle-sim times the oracle's event-level simulation of Algorithm 1
    on the small workloads and stops the sweep at its time bound."""
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--oracle-sim",
                          "--cpu-seconds", "0.05"], capture_output=True, text=True, timeout=300)
    assert out.returncode == 0, out.stderr
    rows = [json.loads(l) for l in out.stdout.splitlines() if l.strip()]
    assert [r["oracle_sim"] for r in rows[:2]] == ["p7_m1000_int32", "p36_m65536_mat2x2u32"]
    assert rows[0]["b"] == 4 and rows[0]["steps"] > 0 and rows[0]["cores"] == 1
    assert len(rows) < 14  # stopped before the largest sweep points


def test_cost_model_fit_recovers_known_constants():
    """The Sec. 1.2 model T(b) = T0 + (L + 3(b-1))(alpha + beta m / b) fitted
    to exact model points returns the constants it was made from, and the
    block-count rule with the fitted kappa = alpha/beta lands on the model's
    best b."""
    p, m = 1152, 1 << 22
    T0, alpha, beta = 8e-6, 2.5e-6, 0.4e-9
    L = bench.model_rounds(p)
    assert L == 4 * 11 - 7
    assert bench.model_rounds(1023, "single") == 4 * 10 - 4
    pts = [(b, T0 + (L + 3 * (b - 1)) * (alpha + beta * m / b)) for b in (1, 4, 16, 64, 256, 1024)]
    t0, a, bta = bench.fit_cost_model(p, m, pts)
    assert t0 == pytest.approx(T0, rel=1e-6) and a == pytest.approx(alpha, rel=1e-6)
    assert bta == pytest.approx(beta, rel=1e-6)
    import math
    T = lambda b: T0 + (L + 3 * (b - 1)) * (alpha + beta * m / b)
    best = min(range(1, 5000), key=T)
    kappa = a / bta
    h = 11
    rule = round(math.sqrt((4 * h - 6) * m / (3 * kappa)))
    assert T(rule) <= T(best) * 1.01
