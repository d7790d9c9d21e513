"""ctypes wrapper around the C oracle (``oracle.c``).

TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the benchmark's CPU
baseline use it; the product package never imports it.  Arrays are numpy,
row-major ``[p][m]`` (``[p][m][4]`` uint32 words for 2x2 matrices,
``[p][m][2]`` int32 for the interval witness, ``[p][m][4]`` float32 for
2x2 float32 matrices).

Functions and the passages they follow:
  trees(p, topo)           dual post-order trees, Sec. 1.1 (topo SINGLE: the
                           one-tree variant of Sec. 1.2)
  left_fold(x, dt)         y = x_0 (.) ... (.) x_{p-1}, Sec. 1 problem statement
  tree_fold(x, dt)         post-order bracketing, Sec. 1.1 + Algorithm 1 roots
  allreduce(x, dt)         tree fold copied to all p rows
  simulate(x, dt, b)       event-level simulation of Algorithm 1
  simulate_rb(x, dt, b)    event-level simulation of a pipelined reduce, then
                           a pipelined broadcast, on one tree (Sec. 1.2 cost
                           analysis; Sec. 2, item 3)
  left_fold_f64(x)         float32 inputs folded in double, with sum |x_i|
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

I32, F32, MAT, WIT, MATF = 0, 1, 2, 3, 4
_ESIZE = {I32: 4, F32: 4, MAT: 16, WIT: 8, MATF: 16}
_DTYPE = {I32: np.int32, F32: np.float32, MAT: np.uint32, WIT: np.int32, MATF: np.float32}

ERRORS = {0: "ok", 1: "invalid", 2: "no memory", 3: "mismatch", 4: "deadlock"}

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so with plain gcc (no fast-math, no
    floating-point contraction, no machine-specific flags)."""
    src = os.path.join(_HERE, "oracle.c")
    if force or not os.path.exists(LIB_PATH) or (
        os.path.getmtime(LIB_PATH) < os.path.getmtime(src)
    ):
        tmp = LIB_PATH + ".tmp%d" % os.getpid()
        subprocess.check_call(
            ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-ffp-contract=off",
             "-fno-fast-math", "-Wall", "-o", tmp, src]
        )
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(LIB_PATH)
        ip = ctypes.POINTER(ctypes.c_int)
        L.orc_trees.argtypes = [ctypes.c_int, ip, ip, ip, ip, ip]
        L.orc_trees_topo.argtypes = [ctypes.c_int, ctypes.c_int, ip, ip, ip, ip, ip]
        L.orc_tree_fold_topo.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int64,
                                         ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]
        L.orc_simulate_topo.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int64,
                                        ctypes.c_int, ctypes.c_int, ctypes.c_void_p,
                                        ctypes.c_void_p, ctypes.POINTER(ctypes.c_int64), ip]
        for f in (L.orc_left_fold, L.orc_tree_fold, L.orc_allreduce):
            f.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int,
                          ctypes.c_void_p, ctypes.c_void_p]
        L.orc_simulate.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int,
                                   ctypes.c_int, ctypes.c_void_p,
                                   ctypes.c_void_p,
                                   ctypes.POINTER(ctypes.c_int64), ip]
        L.orc_left_fold_f64.argtypes = [ctypes.c_int, ctypes.c_int64,
                                        ctypes.c_void_p, ctypes.c_void_p,
                                        ctypes.c_void_p]
        L.orc_simulate_rb.argtypes = [ctypes.c_int, ctypes.c_int64, ctypes.c_int,
                                      ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p,
                                      ctypes.POINTER(ctypes.c_int64)]
        L.orc_set_mutation.argtypes = [ctypes.c_int]
        for f in (L.orc_trees, L.orc_left_fold, L.orc_tree_fold,
                  L.orc_allreduce, L.orc_simulate, L.orc_left_fold_f64,
                  L.orc_trees_topo, L.orc_tree_fold_topo, L.orc_simulate_topo,
                  L.orc_simulate_rb):
            f.restype = ctypes.c_int
        _lib = L
    return _lib


class OracleError(RuntimeError):
    pass


def _check(rc: int) -> None:
    if rc != 0:
        raise OracleError(ERRORS.get(rc, str(rc)))


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _shape(x: np.ndarray, dt: int):
    x = np.ascontiguousarray(x)
    if dt == MAT:
        assert x.ndim == 3 and x.shape[2] == 4 and x.dtype == np.uint32
    elif dt == MATF:
        assert x.ndim == 3 and x.shape[2] == 4 and x.dtype == np.float32
    elif dt == WIT:
        assert x.ndim == 3 and x.shape[2] == 2 and x.dtype == np.int32
    else:
        assert x.ndim == 2 and x.dtype == _DTYPE[dt]
    return x, x.shape[0], x.shape[1]


def set_mutation(k: int) -> None:
    """Plant a known mistake in the oracle (tests of the pins only)."""
    lib().orc_set_mutation(int(k))


DUAL, SINGLE = 0, 1  # tree topologies: dual roots (Sec. 1.1), one tree (Sec. 1.2)


def trees(p: int, topo: int = DUAL) -> dict:
    arrs = {k: np.zeros(p, dtype=np.int32)
            for k in ("parent", "child0", "child1", "dual", "depth")}
    ip = ctypes.POINTER(ctypes.c_int)
    _check(lib().orc_trees_topo(p, topo, *[arrs[k].ctypes.data_as(ip) for k in
                                           ("parent", "child0", "child1", "dual",
                                            "depth")]))
    return arrs


def _fold(fn, x, dt):
    x, p, m = _shape(x, dt)
    y = np.empty(x.shape[1:], dtype=x.dtype)
    _check(fn(p, m, dt, _ptr(x), _ptr(y)))
    return y


def left_fold(x: np.ndarray, dt: int) -> np.ndarray:
    return _fold(lib().orc_left_fold, x, dt)


def tree_fold(x: np.ndarray, dt: int, topo: int = DUAL) -> np.ndarray:
    x, p, m = _shape(x, dt)
    y = np.empty(x.shape[1:], dtype=x.dtype)
    _check(lib().orc_tree_fold_topo(p, topo, m, dt, _ptr(x), _ptr(y)))
    return y


def allreduce(x: np.ndarray, dt: int, out: np.ndarray | None = None):
    x, p, m = _shape(x, dt)
    y = np.empty_like(x) if out is None else out
    _check(lib().orc_allreduce(p, m, dt, _ptr(x), _ptr(y)))
    return y


def simulate(x: np.ndarray, dt: int, b: int, topo: int = DUAL):
    """Run the event-level simulation; returns (Y [p][m...], stats, last_round)."""
    x, p, m = _shape(x, dt)
    y = np.empty_like(x)
    stats = (ctypes.c_int64 * 6)()
    last = np.zeros(p, dtype=np.int32)
    _check(lib().orc_simulate_topo(p, topo, m, b, dt, _ptr(x), _ptr(y), stats,
                                   last.ctypes.data_as(ctypes.POINTER(ctypes.c_int))))
    st = dict(zip(("steps", "first_block_last", "exchanges",
                   "max_ops_nonroot", "max_ops_root", "void_skipped"),
                  [int(v) for v in stats]))
    return y, st, last


def simulate_rb(x: np.ndarray, dt: int, b: int):
    """Event-level simulation of the pipelined reduce, then pipelined
    broadcast, on one tree (Sec. 1.2, Sec. 2 item 3); returns (Y [p][m...],
    stats)."""
    x, p, m = _shape(x, dt)
    y = np.empty_like(x)
    stats = (ctypes.c_int64 * 6)()
    _check(lib().orc_simulate_rb(p, m, b, dt, _ptr(x), _ptr(y), stats))
    st = dict(zip(("steps", "reduce_end_root", "transfers", "first_block_last",
                   "max_ops", "first_bcast_start"), [int(v) for v in stats]))
    return y, st


def left_fold_f64(x: np.ndarray):
    x, p, m = _shape(x, F32)
    y = np.empty(m, dtype=np.float64)
    a = np.empty(m, dtype=np.float64)
    _check(lib().orc_left_fold_f64(p, m, _ptr(x), _ptr(y), _ptr(a)))
    return y, a
