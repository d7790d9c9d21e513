"""Benchmark of the one-GPU doubly pipelined, dual-root reduction-to-all.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
                    [--kernel fused|schedule] [--b B] [--impl reference]

A step is one reduction-to-all of p rank vectors of m elements: every rank's
y_i receives x_0 (.) ... (.) x_{p-1} (one launch of the fused kernel, or of
the schedule kernel with --kernel schedule).  Inputs are seeded synthetic
vectors generated on the device before timing (counter-based generator of
paper_2109_12626_gb300.inputs).  The metric is GB/s = 2 p m sizeof / t (p m
elements read plus p m written) over K timed steps after W warm-up steps.
Inputs larger than twice the L2 (the default workload's 17 GB) need no flush
between steps; smaller ones get a write of twice the L2 before every step,
and the time is then the sum of the steps' own CUDA-event intervals.

The JSON line also carries
  e2e           the same metric with pinned host buffers: per step the host
                to device copy of all p inputs, the kernel, and the device
                to host copy of all p outputs (dpdr_allreduce_host);
  roofline      achieved HBM bytes per launch / launch time (CUDA events on
                the launch stream) against the measured copy bandwidth;
  cpu_baseline  the CPU oracle (tree fold + copy to p rows, one thread) on a
                bounded column sample of the same workload;
  clocks        nvidia-smi samples taken during the timed region.

--impl reference times the CPU oracle itself on the host cores (the
reference arm; rank 0 only under torchrun).  Under torchrun with N > 1 every
rank runs an independent replica of the workload on its own GPU (the path
has no cross-GPU exchange); time is the max over ranks and value the total
over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "p32_m134217728_f32"
METRIC = "allreduce GB/s (p*m*sizeof read + p*m*sizeof written)"
ESIZE = {"int32": 4, "float32": 4, "mat2x2u32": 16, "mat2x2f32": 16}
DTYPE_TAG = {"int32": "int32", "float32": "f32", "mat2x2u32": "u32", "mat2x2f32": "f32"}
# source files whose change invalidates a layout's measured DRAM traffic
KERNEL_SOURCES = {"stream": ("fused_stream.cu", "fused_common.cuh"),
                  "tile": ("fused_tile.cu", "fused_common.cuh"),
                  "split": ("fused_split.cu", "fused_common.cuh"),
                  "bulk": ("fused_bulk.cu", "fused_common.cuh"),
                  "tree": ("fused_tree.cu", "fused_common.cuh"),
                  "schedule": ("schedule.cu", "schedule_common.cuh"),
                  "schedule_words": ("schedule_ll.cu", "schedule_common.cuh"),
                  "reduce_bcast": ("schedule.cu", "schedule_common.cuh")}
LAYOUTS = {1: "stream", 2: "tile", 3: "split", 4: "bulk", 5: "tree"}


# ------------------------------------------------------------ workload
def workload(name: str, m_override: int | None = None) -> dict:
    from paper_2109_12626_gb300.inputs import WORKLOADS
    w = dict(WORKLOADS[name])
    if m_override:
        w["m"] = int(m_override)
    if w["m"] is None:
        w["m"] = 1 << 23
    return w


def gen_device_inputs(w, dev):
    import torch
    from paper_2109_12626_gb300 import inputs as I
    kw = I.workload_kwargs(w)
    xs = []
    for i in range(w["p"]):
        v = I.rank_values(w["kind"], w["seed"], i, w["m"], device=dev, **kw)
        xs.append(v.reshape(-1).contiguous())
        del v
    torch.cuda.synchronize()
    return xs


# --------------------------------------------------------- distributed
def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Largest value over all ranks (the slowest rank's time)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int) -> None:
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# -------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, period_ms: int = 100):
        self.proc = None
        self.gpu = gpu_index
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(gpu_index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", str(period_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self) -> dict | None:
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=10)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        return summarize_clocks(out)


def summarize_clocks(csv_text: str) -> dict | None:
    rows = []
    for line in csv_text.strip().splitlines():
        f = [x.strip() for x in line.split(",")]
        if len(f) < 9:
            continue
        try:
            rows.append(dict(sm=float(f[1]), max=float(f[2]),
                             power=float(f[3]) if f[3] not in ("[N/A]", "N/A") else 0.0,
                             hw=f[5], hwt=f[6], swt=f[7], cap=f[8]))
        except ValueError:
            continue
    if not rows:
        return None
    load = [r for r in rows if r["power"] > 200.0] or rows
    reasons = set()
    for r in load:
        for k, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                        ("swt", "sw_thermal_slowdown"), ("cap", "sw_power_cap")):
            if r[k].lower() == "active":
                reasons.add(name)
    return {"sm_mhz": statistics.median(r["sm"] for r in load),
            "sm_max_mhz": max(r["max"] for r in load),
            "reasons": sorted(reasons), "samples": len(load)}


# ---------------------------------------------------------- host NUMA
def gpu_local_cpus(dev_index: int):
    """CPUs of the NUMA node the GPU is attached to (from sysfs), or None."""
    import torch
    try:
        bus = torch.cuda.get_device_properties(dev_index).pci_bus_id  # "0000:01:00.0" on new torch
    except Exception:
        bus = None
    if not bus:
        try:
            out = subprocess.run(["nvidia-smi", "-i", str(dev_index), "--query-gpu=pci.bus_id",
                                  "--format=csv,noheader"], capture_output=True, text=True,
                                 timeout=20).stdout.strip()
            bus = out.splitlines()[0] if out else None
        except (OSError, subprocess.SubprocessError):
            bus = None
    if not bus:
        return None, None
    bus = bus.lower()
    if bus.count(":") == 2 and len(bus.split(":")[0]) == 8:
        bus = bus[4:]  # nvidia-smi prints an 8-digit domain
    try:
        node = int(open("/sys/bus/pci/devices/%s/numa_node" % bus).read().strip())
        if node < 0:
            return None, None
        cpus = set()
        for part in open("/sys/devices/system/node/node%d/cpulist" % node).read().strip().split(","):
            a, _, b = part.partition("-")
            cpus.update(range(int(a), int(b or a) + 1))
        return node, cpus or None
    except (OSError, ValueError):
        return None, None


# ------------------------------------------------------------ roofline
def measured_peak_gbs() -> tuple[float, str]:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def _code_only(text: str) -> str:
    """C++ source without comments and blank space, so that editing a comment
    does not mark measured counters stale (string literals here hold no
    comment markers)."""
    import re
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_source_hash(kernel: str) -> str:
    """Hash of the code (comments and spacing aside) of a layout's sources."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel] + ("ops.cuh",):
        with open(os.path.join(ROOT, "paper_2109_12626_gb300", "csrc", f)) as fh:
            h.update(_code_only(fh.read()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, wname: str, units: int,
                     block: int | None = None) -> float | None:
    """DRAM bytes per launch from the committed ncu summary, scaled to the
    units of this launch; None if the kernel changed since the capture, or
    (schedule kernel) if the capture's pipeline block size was not within
    5 % of this run's, since the traffic depends on it."""
    path = os.path.join(ROOT, "profiles", "traffic.json")  # ncu figures, not code
    try:
        with open(path) as f:
            recs = json.load(f)[kernel][wname]
    except (OSError, KeyError, ValueError):
        return None
    # one record, or (schedule kernel) a list of records for several block sizes
    for rec in recs if isinstance(recs, list) else [recs]:
        if rec.get("source_hash") != kernel_source_hash(kernel):
            continue
        want = rec.get("block_elems")
        if want is not None and (block is None or abs(block - want) > 0.05 * want):
            continue
        return float(rec["bytes_per_unit"]) * units
    return None


# --------------------------------------------------------- CPU oracle
def cpu_sample(w: dict, target_s: float = 12.0, max_cols: int | None = None):
    """Time the oracle (tree fold + copy to all p rows) single-threaded on a
    column sample of the workload; returns (GB/s, description, reps)."""
    import numpy as np
    import torch
    from oracle import oracle as O
    from paper_2109_12626_gb300 import inputs as I
    p, kind = w["p"], w["kind"]
    es = ESIZE[kind]
    cols = max(1, min(w["m"], (1 << 24) // p if max_cols is None else max_cols))
    kw = I.workload_kwargs(w)
    x = torch.stack([I.rank_values(kind, w["seed"], i, cols, **kw) for i in range(p)])
    x = x.numpy()
    dt = {"int32": O.I32, "float32": O.F32, "mat2x2u32": O.MAT, "mat2x2f32": O.MATF}[kind]
    if kind == "mat2x2u32":
        x = x.view(np.uint32).reshape(p, cols, 4)
    y = np.empty_like(x)
    O.allreduce(x, dt, out=y)  # warm
    reps, t0 = 0, time.perf_counter()
    while True:
        O.allreduce(x, dt, out=y)
        reps += 1
        el = time.perf_counter() - t0
        if el >= target_s or reps >= 1000:
            break
    gbs = 2.0 * p * cols * es * reps / el / 1e9
    return gbs, "%d ranks x %d of %d columns, %d repetitions" % (p, cols, w["m"], reps), el / reps


def run_reference(args, w) -> dict:
    """The reference arm: the CPU oracle on the host cores, K timed steps of
    a bounded sample of the workload after W warm-up steps."""
    import numpy as np
    import torch
    from oracle import oracle as O
    from paper_2109_12626_gb300 import inputs as I
    p, kind = w["p"], w["kind"]
    es = ESIZE[kind]
    cols = max(1, min(w["m"], (1 << 22) // p))
    kw = I.workload_kwargs(w)
    x = torch.stack([I.rank_values(kind, w["seed"], i, cols, **kw) for i in range(p)]).numpy()
    dt = {"int32": O.I32, "float32": O.F32, "mat2x2u32": O.MAT, "mat2x2f32": O.MATF}[kind]
    if kind == "mat2x2u32":
        x = x.view(np.uint32).reshape(p, cols, 4)
    y = np.empty_like(x)
    for _ in range(args.warmup):
        O.allreduce(x, dt, out=y)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        O.allreduce(x, dt, out=y)
    el = time.perf_counter() - t0
    v = 2.0 * p * cols * es * args.steps / el / 1e9
    sample = "%d ranks x %d of %d columns per step" % (p, cols, w["m"])
    return {"impl": "reference", "metric": METRIC, "value": round(v, 4), "unit": "GB/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(el / args.steps * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": DTYPE_TAG[kind],
            "data": "synthetic (seeded counter-based generator)",
            "config": {"workload": args.workload, "p": p, "m": w["m"], "sample_columns": cols},
            "cpu_baseline": {"value": round(v, 4), "unit": "GB/s", "cores": 1,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(v, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def run_oracle_sim(args) -> int:
    """The oracle's event-level simulation of Algorithm 1 (every exchange of
    every rank and round, with its unit-step clock) timed on one host core:
    the two small workloads with their b, then the p = 1152 int32 sweep at
    b = min(m, 16) while the next point would take under --cpu-seconds.  One JSON line
    per point; CPU only, a reported baseline like cpu_baseline."""
    import numpy as np
    import torch
    from oracle import oracle as O
    from paper_2109_12626_gb300 import inputs as I
    points = [("p7_m1000_int32", None), ("p36_m65536_mat2x2u32", None)]
    points += [("p1152_int32_sweep", 1 << k) for k in range(0, 24, 2)]
    for name, m in points:
        w = workload(name, m)
        p, kind, m = w["p"], w["kind"], w["m"]
        kw = I.workload_kwargs(w)
        x = torch.stack([I.rank_values(kind, w["seed"], i, m, **kw) for i in range(p)]).numpy()
        dt = {"int32": O.I32, "float32": O.F32, "mat2x2u32": O.MAT, "mat2x2f32": O.MATF}[kind]
        if kind == "mat2x2u32":
            x = x.view(np.uint32).reshape(p, m, 4)
        b = int(w.get("b") or min(m, 16))
        t0 = time.perf_counter()
        _, st, _ = O.simulate(x, dt, b)
        el = time.perf_counter() - t0
        print(json.dumps({"oracle_sim": name, "p": p, "m": m, "b": b, "seconds": round(el, 4),
                          "ns_per_element": round(el * 1e9 / (p * m), 2), "cores": 1,
                          "steps": st["steps"], "exchanges": st["exchanges"]}), flush=True)
        if el * 4 > args.cpu_seconds:  # the next point is four times larger
            break
    return 0


# -------------------------------------------------------------- sweeps
def model_rounds(p: int, topology: str = "dual") -> int:
    """Unit steps before the first block reaches the last leaf in the
    schedule's rendezvous model: 4h-7 for dual trees with p = 2^h - 2
    (h >= 3), 4h-4 for one tree with p = 2^h - 1 (the oracle's simulation
    gives both)."""
    extra = 1 if topology == "single" else 2
    h = 0
    while (1 << h) < p + extra:
        h += 1
    return max(1, 4 * h - (4 if topology == "single" else 7))


TRANSPORTS = {"auto": 0, "counters": 1, "words": 2}


def fit_cost_model(p: int, m: int, points, topology: str = "dual"):
    """Least-squares fit of T(b) = T0 + (L + 3(b-1)) (alpha + beta m / b)
    (Sec. 1.2's cost model plus a launch constant T0) to (b, seconds)
    points; returns T0, alpha, beta (seconds, seconds/element)."""
    import numpy as np
    L = model_rounds(p, topology)
    A = np.array([[1.0, L + 3 * (b - 1), (L + 3 * (b - 1)) * m / b] for b, _ in points])
    y = np.array([t for _, t in points])
    try:  # the constants are times: fit them non-negative
        from scipy.optimize import nnls
        scale = A.max(axis=0)
        scale[scale == 0] = 1.0
        coef, _ = nnls(A / scale, y)
        coef = coef / scale
    except ImportError:
        coef, *_ = np.linalg.lstsq(A, y, rcond=None)
    return float(coef[0]), float(coef[1]), float(coef[2])


def set_schedule_options(pkg, plan, args) -> None:
    """The schedule kernels' transport, CTA layout, threads and slices."""
    plan.set(pkg.OPT_SCHED_TRANSPORT, TRANSPORTS[args.transport])
    if args.sched_threads:
        plan.set(pkg.OPT_SCHED_THREADS, args.sched_threads)
    plan.set(pkg.OPT_SCHED_LAYOUT, args.sched_layout)
    if args.sched_slices:
        plan.set(pkg.OPT_SCHED_SLICES, args.sched_slices)


def _timed(fn, reps, stream, graph=False):
    import torch
    for _ in range(2):
        fn()
    torch.cuda.synchronize()
    g = None
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for _ in range(reps):
                fn()
        g.replay()
        torch.cuda.synchronize()
    a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    if g is not None:
        g.replay()
    else:
        for _ in range(reps):
            fn()
    z.record()
    torch.cuda.synchronize()
    return a.elapsed_time(z) / reps * 1e-3


def _timed_reps(fn, reps):
    """Per-call times (seconds) of reps replays of a CUDA graph holding one
    call, each bracketed by its own events, after three untimed replays."""
    import torch
    for _ in range(2):
        fn()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(reps)]
    for a, z in ev:
        a.record()
        g.replay()
        z.record()
    torch.cuda.synchronize()
    return [a.elapsed_time(z) * 1e-3 for a, z in ev]


def _stats(ts):
    """mean, min (the paper's convention: the best of the measurement
    rounds) and median, in microseconds."""
    return {"us": round(statistics.fmean(ts) * 1e6, 2), "us_min": round(min(ts) * 1e6, 2),
            "us_median": round(statistics.median(ts) * 1e6, 2)}


def run_sweep(args, w) -> int:
    """--sweep m: every m = 2^0 .. 2^k of the workload, fused kernel (its
    automatic layout, or --mode) and schedule kernel (its automatic transport) at the
    block-count rule, both timed as CUDA-graph replays of one call each (host
    launch overhead excluded): mean, min and median over the replays.  --sweep b: the schedule
    kernel's time against b at one m, with the Sec. 1.2 cost model fitted.
    One JSON line per point, then a summary line."""
    import torch
    import paper_2109_12626_gb300 as pkg
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    p, kind, es = w["p"], w["kind"], ESIZE[w["kind"]]
    if args.sweep == "m":
        top = int(args.m or (1 << 23)).bit_length() - 1
        ms = ([int(v) for v in args.mlist.split(",")] if args.mlist
              else [1 << k for k in range(0, top + 1)])
        for m in ms:
            ww = dict(w, m=m)
            xs = gen_device_inputs(ww, dev)
            ys = [torch.empty_like(x) for x in xs]
            rec = {"sweep": "m", "workload": args.workload, "p": p, "m": m,
                   "topology": args.topology}
            b0 = -(-m // args.block_size) if args.block_size else 0
            with pkg.Plan(p, m, kind, b0, topology=args.topology) as plan:
                set_schedule_options(pkg, plan, args)
                if args.split_depth is not None:
                    plan.set(pkg.OPT_SPLIT_DEPTH, args.split_depth)
                if args.mode:
                    plan.set(pkg.OPT_FUSED_MODE, args.mode)
                bd = plan.bind(xs, ys)
                st = _stats(_timed_reps(lambda: bd.allreduce(), 20))
                info = plan.info()
                mode = args.mode or info["auto_mode"]
                rec["fused"] = dict(st, gbs=round(2 * p * m * es / (st["us"] * 1e-6) / 1e9, 2),
                                    layout=LAYOUTS[mode],
                                    split_depth=info["split_depth"] if mode == 3 else None)
                st = _stats(_timed_reps(lambda: bd.allreduce_schedule(),
                                        5 if m >= (1 << 20) else 20))
                plan.sync()
                rec["schedule"] = dict(st, b=info["b"],
                                       gbs=round(2 * p * m * es / (st["us"] * 1e-6) / 1e9, 2),
                                       slices=plan.info()["sched_slices"],
                                       sched_layout=plan.info()["sched_layout"],
                                       transport=("counters", "words")[
                                           info["sched_transport"] - 1])
            print(json.dumps(rec), flush=True)
            del xs, ys
            torch.cuda.empty_cache()
        return 0
    if args.sweep == "rb":
        return run_sweep_rb(args, w)
    # --sweep b
    m = w["m"]
    xs = gen_device_inputs(w, dev)
    ys = [torch.empty_like(x) for x in xs]
    bs = sorted(set(int(v) for v in args.blist.split(",") if int(v) <= max(m, 1)))
    points = []
    for b in bs:
        with pkg.Plan(p, m, kind, b, topology=args.topology) as plan:
            set_schedule_options(pkg, plan, args)
            bd = plan.bind(xs, ys)
            t = _timed(lambda: bd.allreduce_schedule(), 5 if m >= (1 << 20) else 10, None,
                       graph=True)
            plan.sync()
            points.append((b, t))
            print(json.dumps({"sweep": "b", "workload": args.workload, "topology": args.topology,
                              "transport": args.transport, "p": p, "m": m, "b": b,
                              "us": round(t * 1e6, 2), "slices": plan.info()["sched_slices"]}),
                  flush=True)
    t0, alpha, beta = fit_cost_model(p, m, points, args.topology)
    best = min(points, key=lambda x: x[1])
    kappa = alpha / beta if beta > 0 else float("inf")
    rule = pkg.block_count_rule(p, m, kappa) if beta > 0 and alpha > 0 else None
    print(json.dumps({"sweep": "b-fit", "workload": args.workload, "topology": args.topology,
                      "transport": args.transport, "p": p, "m": m,
                      "rounds_L": model_rounds(p, args.topology), "T0_us": round(t0 * 1e6, 3),
                      "alpha_us": round(alpha * 1e6, 4), "beta_ns_per_elem": round(beta * 1e9, 5),
                      "kappa_elems": round(kappa, 1) if beta > 0 else None,
                      "best_b": best[0], "best_us": round(best[1] * 1e6, 2),
                      "rule_b_with_fitted_kappa": rule,
                      "rule_b_default_kappa": pkg.block_count_rule(p, m)}), flush=True)
    return 0


def run_sweep_rb(args, w) -> int:
    """--sweep rb: the doubly pipelined dual-root schedule (Algorithm 1)
    against a pipelined reduce to the root of one tree followed by a
    pipelined broadcast (the comparison of Sec. 1.2 and Sec. 2, items 3
    and 4), both with the same pipeline blocks: b = ceil(m / --block-size),
    or the dual plan's default b.  Also Algorithm 1 on the one tree.  Each
    time is the min and mean of CUDA-graph replays of one call (launch
    included).  One JSON line per m."""
    import torch
    import paper_2109_12626_gb300 as pkg
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    p, kind, es = w["p"], w["kind"], ESIZE[w["kind"]]
    top = int(args.m or (1 << 23)).bit_length() - 1
    ms = ([int(v) for v in args.mlist.split(",")] if args.mlist
          else [1 << k for k in range(0, top + 1)])
    for m in ms:
        ww = dict(w, m=m)
        xs = gen_device_inputs(ww, dev)
        ys = [torch.empty_like(x) for x in xs]
        b = -(-m // args.block_size) if args.block_size else 0
        rec = {"sweep": "rb", "workload": args.workload, "p": p, "m": m}
        reps = 5 if p * m >= (1 << 26) else 20
        with pkg.Plan(p, m, kind, b) as dual:
            dual.set(pkg.OPT_SCHED_TRANSPORT, 1)
            dual.set(pkg.OPT_SCHED_LAYOUT, args.sched_layout)
            b = dual.query()["b"]
            bd = dual.bind(xs, ys)
            rec["dual_alg1"] = _stats(_timed_reps(lambda: bd.allreduce_schedule(), reps))
            dual.sync()
        with pkg.Plan(p, m, kind, b, topology="single") as one:
            one.set(pkg.OPT_SCHED_TRANSPORT, 1)
            one.set(pkg.OPT_SCHED_LAYOUT, args.sched_layout)
            bo = one.bind(xs, ys)
            rec["single_alg1"] = _stats(_timed_reps(lambda: bo.allreduce_schedule(), reps))
            rec["single_reduce_bcast"] = _stats(_timed_reps(lambda: bo.allreduce_reduce_bcast(),
                                                            reps))
            one.sync()
        rec["b"] = b
        rec["ratio_rb_over_dual"] = round(rec["single_reduce_bcast"]["us_min"]
                                          / rec["dual_alg1"]["us_min"], 3)
        rec["ratio_rb_over_single"] = round(rec["single_reduce_bcast"]["us_min"]
                                            / rec["single_alg1"]["us_min"], 3)
        rec["dual_gbs"] = round(2 * p * m * es / (rec["dual_alg1"]["us_min"] * 1e-6) / 1e9, 2)
        print(json.dumps(rec), flush=True)
        del xs, ys
        torch.cuda.empty_cache()
    return 0


# ---------------------------------------------------------------- main
def main(argv=None) -> int:
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--m", type=int, default=None, help="override m (sweeps)")
    ap.add_argument("--kernel", choices=("fused", "schedule", "reduce_bcast"), default="fused",
                    help="reduce_bcast: pipelined reduce then broadcast on one tree")
    ap.add_argument("--b", type=int, default=None, help="pipeline blocks (schedule)")
    ap.add_argument("--mode", type=int, default=0,
                    help="fused layout: 0 auto, 1 stream, 2 tile, 3 split, 4 bulk, 5 tree")
    ap.add_argument("--split-depth", type=int, default=None, help="split layout cut depth")
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--sweep", choices=("m", "b", "rb"), default=None,
                    help="m: all m = 2^k up to --m; b: schedule time against b")
    ap.add_argument("--blist", default="1,2,4,8,16,32,64,128,256,512,1024")
    ap.add_argument("--topology", choices=("dual", "single"), default="dual",
                    help="dual roots (the paper's method) or one tree (Sec. 1.2 variant)")
    ap.add_argument("--p", type=int, default=None, help="override p (sweeps)")
    ap.add_argument("--block-size", type=int, default=None,
                    help="schedule kernel blocks of this many elements: b = ceil(m / size)")
    ap.add_argument("--mlist", default=None, help="comma-separated m values for --sweep m")
    ap.add_argument("--host-path", type=int, default=0,
                    help="e2e leg: 0 direct when possible, 1 copy pipeline, 2 direct")
    ap.add_argument("--sched-layout", type=int, default=0, choices=(0, 1, 2),
                    help="schedule kernels' CTA layout: 0 auto, 1 rank ranges, 2 by work")
    ap.add_argument("--sched-threads", type=int, default=0,
                    help="threads per schedule CTA (0 = automatic)")
    ap.add_argument("--sched-slices", type=int, default=0,
                    help="column slices per rank of the schedule kernels (0 = automatic)")
    ap.add_argument("--transport", choices=tuple(TRANSPORTS), default="auto",
                    help="schedule kernel: how blocks pass between virtual ranks")
    ap.add_argument("--oracle-sim", action="store_true",
                    help="time the oracle's event-level simulation of Algorithm 1 (CPU)")
    args = ap.parse_args(argv)
    args.warmup = max(args.warmup, 3)
    if args.kernel == "reduce_bcast":
        args.topology = "single"   # the variant runs on the one-tree plan

    world, rank, local = dist_env()
    w = workload(args.workload, args.m)
    if args.p:
        w["p"] = int(args.p)

    if args.oracle_sim:
        return run_oracle_sim(args) if rank == 0 else 0
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args, w)), flush=True)
        return 0
    if args.sweep:
        return run_sweep(args, w)

    import torch
    import paper_2109_12626_gb300 as pkg
    from paper_2109_12626_gb300 import build as B

    assert torch.cuda.is_available(), "bench.py needs a GPU"
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if not os.path.exists(B.LIB):
        B.build()

    p, m, kind = w["p"], w["m"], w["kind"]
    es = ESIZE[kind]
    b = args.b if args.b is not None else (w.get("b") or 0)
    if args.block_size:
        b = -(-m // args.block_size)
    xs = gen_device_inputs(w, dev)
    ys = [torch.empty_like(x) for x in xs]
    plan = pkg.Plan(p, m, kind, b, topology=args.topology)
    set_schedule_options(pkg, plan, args)
    if args.split_depth is not None:
        plan.set(pkg.OPT_SPLIT_DEPTH, args.split_depth)
    if args.mode:
        plan.set(pkg.OPT_FUSED_MODE, args.mode)
    stream = torch.cuda.current_stream(dev)
    run = {"fused": plan.allreduce, "schedule": plan.allreduce_schedule,
           "reduce_bcast": plan.allreduce_reduce_bcast}[args.kernel]
    algo_bytes = 2 * p * m * es

    for _ in range(args.warmup):
        run(xs, ys, stream)
    plan.sync(stream)

    sampler = ClockSampler(local)
    time.sleep(0.3)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    bound = plan.bind(xs, ys)
    go = {"fused": bound.allreduce, "schedule": bound.allreduce_schedule,
          "reduce_bcast": bound.allreduce_reduce_bcast}[args.kernel]
    # inputs that L2 could hold: write a buffer of twice L2 before every step
    # and time the steps by their own events, so each step starts cold
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush = (torch.empty(2 * l2 // 4, dtype=torch.int32, device=dev)
             if p * m * es < 2 * l2 else None)
    barrier(world)
    torch.cuda.synchronize(dev)
    torch.cuda.nvtx.range_push("dpdr_timed")
    start.record(stream)
    for k in range(args.steps):
        if flush is not None:
            flush.fill_(k)
        ev[k][0].record(stream)
        go(stream)
        ev[k][1].record(stream)
    stop.record(stream)
    torch.cuda.synchronize(dev)
    torch.cuda.nvtx.range_pop()
    barrier(world)
    clocks = sampler.stop()
    plan.sync(stream)
    launch_ms = [a.elapsed_time(z) for a, z in ev]
    total_ms = start.elapsed_time(stop) if flush is None else sum(launch_ms)
    t_max = max_over_ranks(total_ms, world, dev)
    ms_per_step = t_max / args.steps
    value = world * algo_bytes / (ms_per_step * 1e-3) / 1e9
    avg_launch = sum(launch_ms) / len(launch_ms)
    achieved = algo_bytes / (avg_launch * 1e-3) / 1e9
    peak, peak_kind = measured_peak_gbs()
    units = p * m
    # small workloads start every step cold: a plain device copy of the same
    # bytes (p m esize read, as many written), timed the same way after the
    # same L2 flush, is the floor that method allows
    copy_ref = None
    if flush is not None and rank == 0:
        src_t = torch.empty(p * m * es // 4, dtype=torch.int32, device=dev)
        dst_t = torch.empty_like(src_t)
        for _ in range(3):
            dst_t.copy_(src_t)
        cts = []
        for k in range(args.steps):
            flush.fill_(k + 1)
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            dst_t.copy_(src_t)
            a1.record(stream)
            torch.cuda.synchronize(dev)
            cts.append(a0.elapsed_time(a1))
        copy_us = 1000 * sum(cts) / len(cts)
        copy_ref = {"us": round(copy_us, 2), "kernel_us": round(1000 * avg_launch, 2),
                    "kernel_over_copy": round(1000 * avg_launch / copy_us, 3),
                    "what": "torch device copy of p*m*esize bytes, L2 flushed before each, "
                            "mean of the same number of steps"}
        del src_t, dst_t

    # end to end with host buffers
    e2e = None
    if not args.no_e2e:
        # pinned host buffers on the CPU node next to the GPU (first touch)
        node, cpus = gpu_local_cpus(local)
        saved = os.sched_getaffinity(0)
        if cpus:
            try:
                os.sched_setaffinity(0, cpus)
            except OSError:
                node = None
        xh = [torch.empty(x.shape, dtype=x.dtype, pin_memory=True) for x in xs]
        yh = [torch.empty(x.shape, dtype=x.dtype, pin_memory=True) for x in xs]
        for h, x in zip(xh, xs):
            h.copy_(x)
        for h in yh:
            h.zero_()
        plan.set(pkg.OPT_HOST_PATH, args.host_path)
        for _ in range(2):
            plan.allreduce_host(xh, yh, xs, ys, stream)
        plan.sync(stream)
        k2 = max(3, min(args.steps, 10))
        barrier(world)
        torch.cuda.synchronize(dev)
        s2, e2 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        s2.record(stream)
        for _ in range(k2):
            plan.allreduce_host(xh, yh, xs, ys, stream)
        e2.record(stream)
        torch.cuda.synchronize(dev)
        t2 = max_over_ranks(s2.elapsed_time(e2), world, dev) / k2
        e2e = {"value": round(world * algo_bytes / (t2 * 1e-3) / 1e9, 3), "unit": "GB/s",
               "h2d_bytes_per_step": p * m * es, "d2h_bytes_per_step": p * m * es,
               "steps": k2, "ms_per_step": round(t2, 3), "host_numa_node": node,
               "path": {1: "copy pipeline", 2: "direct (kernel on host memory)"}.get(
                   plan.info()["host_path"], "?")}
        del xh, yh
        os.sched_setaffinity(0, saved)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:  # the CPU baseline: N = 1 only
        gbs, sample, _ = cpu_sample(w, args.cpu_seconds)
        cpu = {"value": round(gbs, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
               "sample": sample}

    info = plan.info()
    layout = (LAYOUTS[args.mode or info["auto_mode"]] if args.kernel == "fused"
              else "reduce_bcast" if args.kernel == "reduce_bcast"
              else ("schedule", "schedule_words")[info["sched_transport"] - 1])
    launches_per_step = 2 if layout == "split" else 1
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": DTYPE_TAG[kind],
        "data": "synthetic (seeded counter-based generator, generated on device)",
        "config": {"workload": args.workload, "p": p, "m": m, "kind": kind,
                   "topology": args.topology,
                   "kernel": args.kernel, "b": info["b"],
                   "sched_layout": (None if args.kernel == "fused" else
                                    {1: "rank ranges", 2: "by work"}[info["sched_layout"]]),
                   "fused_mode": args.mode or info["auto_mode"],
                   "split_depth": info["split_depth"] if (args.mode or info["auto_mode"]) == 3 else None,
                   "bytes_per_step": algo_bytes,
                   "l2": ("inputs larger than twice L2 (%.1f GB), no flush" % (algo_bytes / 2e9)
                          if flush is None else
                          "L2 flushed before every step (a 2 x L2 write); time = sum of the "
                          "steps' own CUDA-event intervals"),
                   "parallelism": "replicas" if world > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "kernel": layout, "achieved": round(achieved, 1), "peak": peak,
                     "unit": "GB/s", "frac": round(achieved / peak, 4),
                     "peak_kind": peak_kind + " copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
                     "traffic": profiled_traffic(layout, args.workload, units,
                                                 -(-m // max(1, info["b"]))),
                     "kernel_ms": round(avg_launch, 4)},
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": args.steps * launches_per_step,
        "clocks": clocks,
        "cold_copy_reference": copy_ref,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    plan.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
