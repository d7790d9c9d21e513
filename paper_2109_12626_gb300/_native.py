"""ctypes binding of libdpdr.so (the C ABI of include/dpdr.h).

The library is loaded on first use from this package's directory; it is
built by ``paper_2109_12626_gb300.build`` (or ``__graft_entry__.build()``).
There is no fallback: without the library every call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Sequence

import numpy as np

DPDR_INT32, DPDR_FLOAT32, DPDR_MAT2X2_U32, DPDR_MAT2X2_F32 = 0, 1, 2, 3
DPDR_OP_SUM, DPDR_OP_MATMUL = 0, 1
(DPDR_OK, DPDR_ERR_INVALID, DPDR_ERR_CUDA, DPDR_ERR_TIMEOUT,
 DPDR_ERR_NOT_COOPERATIVE, DPDR_ERR_OOM) = range(6)
(OPT_FUSED_MODE, OPT_WAIT_LIMIT_NS, OPT_SKIP_RANK, OPT_SCHED_THREADS,
 OPT_SCHED_RANKS_PER_CTA, OPT_BLOCKS, OPT_SPLIT_DEPTH, OPT_SCHED_SLICES,
 OPT_HOST_CHUNK_BYTES, OPT_HOST_PATH, OPT_SCHED_TRANSPORT,
 OPT_SCHED_LAYOUT, OPT_SCHED_COPY) = range(1, 14)

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libdpdr.so")

# every function the header declares, with its ctypes signature
_P = ctypes.c_void_p
_IP = ctypes.POINTER(ctypes.c_int)
_I64P = ctypes.POINTER(ctypes.c_int64)
SIGNATURES = {
    "dpdr_tree": (ctypes.c_int, [ctypes.c_int, _IP, _IP, _IP, _IP, _IP]),
    "dpdr_tree_topo": (ctypes.c_int, [ctypes.c_int, ctypes.c_int, _IP, _IP, _IP, _IP, _IP]),
    "dpdr_blocks": (ctypes.c_int, [ctypes.c_int64, ctypes.c_int, _I64P]),
    "dpdr_block_count_rule": (ctypes.c_int, [ctypes.c_int, ctypes.c_int64,
                                             ctypes.c_double]),
    "dpdr_plan": (_P, [ctypes.c_int, ctypes.c_int64, ctypes.c_int,
                       ctypes.c_int, ctypes.c_int]),
    "dpdr_plan_topo": (_P, [ctypes.c_int, ctypes.c_int64, ctypes.c_int,
                            ctypes.c_int, ctypes.c_int, ctypes.c_int]),
    "dpdr_plan_query": (ctypes.c_int, [_P, _IP, _IP, _IP, _IP, _IP, _IP]),
    "dpdr_plan_set": (ctypes.c_int, [_P, ctypes.c_int, ctypes.c_int64]),
    "dpdr_plan_info": (ctypes.c_int, [_P, _I64P, ctypes.c_int]),
    "dpdr_plan_destroy": (None, [_P]),
    "dpdr_allreduce": (ctypes.c_int, [_P, _P, _P, _P]),
    "dpdr_allreduce_schedule": (ctypes.c_int, [_P, _P, _P, _P]),
    "dpdr_allreduce_reduce_bcast": (ctypes.c_int, [_P, _P, _P, _P]),
    "dpdr_allreduce_host": (ctypes.c_int, [_P, _P, _P, _P, _P, _P]),
    "dpdr_plan_sync": (ctypes.c_int, [_P, _P]),
    "dpdr_allreduce_schedule_noalloc": (ctypes.c_int, [ctypes.c_int, ctypes.c_int64,
                                                       ctypes.c_int, ctypes.c_int,
                                                       ctypes.c_int, _P, _P, _P]),
    "dpdr_last_error": (ctypes.c_int, []),
    "dpdr_last_error_message": (ctypes.c_char_p, []),
    "dpdr_status_string": (ctypes.c_char_p, [ctypes.c_int]),
}

_lib = None


class DpdrError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = lib().dpdr_last_error_message().decode(errors="replace")
        name = lib().dpdr_status_string(status).decode()
        super().__init__("%s: %s (%d): %s" % (where, name, status, msg))


def lib():
    """The loaded library (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                "libdpdr.so is not built; run `python -m "
                "paper_2109_12626_gb300.build` (no CPU fallback exists)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(rc: int, where: str) -> None:
    if rc != DPDR_OK:
        raise DpdrError(rc, where)


TOPOLOGIES = {"dual": 0, "single": 1}


def tree(p: int, topology="dual") -> dict:
    """Post-order trees (host only): parent, child0, child1, dual, depth."""
    t = TOPOLOGIES[topology] if isinstance(topology, str) else int(topology)
    out = {k: np.zeros(p, np.int32) for k in ("parent", "child0", "child1",
                                               "dual", "depth")}
    _check(lib().dpdr_tree_topo(p, t, *[out[k].ctypes.data_as(_IP) for k in
                                         ("parent", "child0", "child1", "dual",
                                          "depth")]), "dpdr_tree")
    return out


def blocks(m: int, b: int) -> np.ndarray:
    s = np.zeros(b + 1, np.int64)
    _check(lib().dpdr_blocks(m, b, s.ctypes.data_as(_I64P)), "dpdr_blocks")
    return s


def block_count_rule(p: int, m: int, kappa: float = 0.0) -> int:
    b = lib().dpdr_block_count_rule(p, m, kappa)
    if b < 1:
        raise DpdrError(lib().dpdr_last_error(), "dpdr_block_count_rule")
    return b


def _addr(t) -> int:
    if isinstance(t, int):
        return t
    return int(t.data_ptr())


def _ptr_array(ts: Sequence) -> ctypes.Array:
    arr = (ctypes.c_void_p * len(ts))()
    for i, t in enumerate(ts):
        arr[i] = _addr(t)
    return arr


def _stream(stream) -> int:
    if stream is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


DTYPES = {"int32": DPDR_INT32, "float32": DPDR_FLOAT32,
          "mat2x2u32": DPDR_MAT2X2_U32, "mat2x2f32": DPDR_MAT2X2_F32}


# dpdr_plan_info's entries, in the header's order
INFO_KEYS = ("p", "m", "b", "max_depth", "auto_mode", "sched_ctas",
             "sched_ranks_per_cta", "scratch_bytes", "vector_path",
             "split_depth", "split_subtrees", "split_group", "sched_slices",
             "topology", "host_path", "sched_transport", "tree_width",
             "sched_layout", "sched_copy")


class Plan:
    """A plan for p virtual ranks of m elements (``dpdr_plan``)."""

    def __init__(self, p: int, m: int, dtype, b: int = 0, topology="dual"):
        dt = DTYPES[dtype] if isinstance(dtype, str) else int(dtype)
        op = DPDR_OP_MATMUL if dt in (DPDR_MAT2X2_U32, DPDR_MAT2X2_F32) else DPDR_OP_SUM
        topo = TOPOLOGIES[topology] if isinstance(topology, str) else int(topology)
        L = lib()
        h = L.dpdr_plan_topo(int(p), int(m), dt, op, int(b), topo)
        if not h:
            raise DpdrError(L.dpdr_last_error(), "dpdr_plan")
        self._h = h
        self.p, self.m, self.dtype = int(p), int(m), dt

    def close(self) -> None:
        if getattr(self, "_h", None):
            lib().dpdr_plan_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # ---------------------------------------------------------------- facts
    def query(self) -> dict:
        out = {k: np.zeros(self.p, np.int32) for k in ("parent", "child0",
                                                        "child1", "dual",
                                                        "depth")}
        b = ctypes.c_int(0)
        _check(lib().dpdr_plan_query(self._h, *[out[k].ctypes.data_as(_IP) for k in
                                                 ("parent", "child0", "child1",
                                                  "dual", "depth")],
                                     ctypes.byref(b)), "dpdr_plan_query")
        out["b"] = b.value
        return out

    def info(self) -> dict:
        n = len(INFO_KEYS)
        v = np.zeros(n, np.int64)
        _check(lib().dpdr_plan_info(self._h, v.ctypes.data_as(_I64P), n), "dpdr_plan_info")
        return {k: int(x) for k, x in zip(INFO_KEYS, v)}

    def set(self, key: int, value: int) -> None:
        _check(lib().dpdr_plan_set(self._h, int(key), int(value)), "dpdr_plan_set")

    # ------------------------------------------------------------------ run
    def allreduce(self, xs: Sequence, ys: Sequence, stream=None) -> None:
        """Fused kernel: every ys[i] <- x_0 (.) ... (.) x_{p-1}."""
        assert len(xs) == self.p and len(ys) == self.p
        _check(lib().dpdr_allreduce(self._h, _ptr_array(xs), _ptr_array(ys),
                                    _stream(stream)), "dpdr_allreduce")

    def allreduce_schedule(self, xs: Sequence, ys: Sequence, stream=None) -> None:
        """Schedule-faithful kernel (Algorithm 1 round by round)."""
        assert len(xs) == self.p and len(ys) == self.p
        _check(lib().dpdr_allreduce_schedule(self._h, _ptr_array(xs),
                                             _ptr_array(ys), _stream(stream)),
               "dpdr_allreduce_schedule")

    def allreduce_reduce_bcast(self, xs: Sequence, ys: Sequence, stream=None) -> None:
        """Pipelined reduce to the root, then pipelined broadcast, on a
        one-tree plan (Sec. 1.2; Sec. 2 item 3)."""
        assert len(xs) == self.p and len(ys) == self.p
        _check(lib().dpdr_allreduce_reduce_bcast(self._h, _ptr_array(xs),
                                                 _ptr_array(ys), _stream(stream)),
               "dpdr_allreduce_reduce_bcast")

    def allreduce_host(self, xh: Sequence, yh: Sequence, xd: Sequence | None = None,
                       yd: Sequence | None = None, stream=None) -> None:
        """Host buffers in and out (device buffers as staging when the GPU
        cannot address the host buffers directly)."""
        _check(lib().dpdr_allreduce_host(self._h, _ptr_array(xh), _ptr_array(yh),
                                         _ptr_array(xd) if xd is not None else None,
                                         _ptr_array(yd) if yd is not None else None,
                                         _stream(stream)), "dpdr_allreduce_host")

    def bind(self, xs: Sequence, ys: Sequence) -> "Bound":
        """Marshal the rank buffers once, for repeated calls on them."""
        return Bound(self, xs, ys)

    def sync(self, stream=None) -> None:
        """Wait for the stream; raise DpdrError on a schedule-kernel timeout."""
        _check(lib().dpdr_plan_sync(self._h, _stream(stream)), "dpdr_plan_sync")


class Bound:
    """A plan with its rank-pointer arrays marshalled once (repeated calls
    on the same buffers cost one C call each)."""

    def __init__(self, plan: Plan, xs: Sequence, ys: Sequence):
        assert len(xs) == plan.p and len(ys) == plan.p
        self.plan = plan
        self._keep = (list(xs), list(ys))
        self.X = _ptr_array(xs)
        self.Y = _ptr_array(ys)

    def allreduce(self, stream=None) -> None:
        _check(lib().dpdr_allreduce(self.plan._h, self.X, self.Y, _stream(stream)),
               "dpdr_allreduce")

    def allreduce_schedule(self, stream=None) -> None:
        _check(lib().dpdr_allreduce_schedule(self.plan._h, self.X, self.Y,
                                             _stream(stream)),
               "dpdr_allreduce_schedule")

    def allreduce_reduce_bcast(self, stream=None) -> None:
        _check(lib().dpdr_allreduce_reduce_bcast(self.plan._h, self.X, self.Y,
                                                 _stream(stream)),
               "dpdr_allreduce_reduce_bcast")
