"""Pins for the oracle's left fold (O3) and tree fold (O2).

O3 is the plain definition of the result (Sec. 1); O2 is the bracketing of
Sec. 1.1 with the dual-root rule of Algorithm 1.  They are pinned by closed
forms, hand-derived golden values, brute force with Python integers on tiny
inputs, the interval witness, and the float32 error bound."""
import math
import os

import numpy as np
import pytest

GOLD = os.path.join(os.path.dirname(__file__), "golden")
M32 = (1 << 32) - 1


def witness(p, m):
    x = np.zeros((p, m, 2), np.int32)
    for i in range(p):
        x[i, :, :] = i
    return x


@pytest.mark.parametrize("p", list(range(1, 70)) + [255, 1152])
def test_witness_orders_every_operand(orc, p):
    x = witness(p, 3)
    for f in (orc.left_fold, orc.tree_fold):
        y = f(x, orc.WIT)
        assert (y[:, 0] == 0).all() and (y[:, 1] == p - 1).all()


def test_witness_is_not_commutative_and_absorbs(orc):
    x = np.array([[[1, 1]], [[0, 0]]], np.int32)  # [1,1] then [0,0]: misordered
    assert orc.left_fold(x, orc.WIT).tolist() == [[-1, -1]]
    x = np.array([[[0, 0]], [[0, 0]]], np.int32)  # repeated operand
    assert orc.left_fold(x, orc.WIT).tolist() == [[-1, -1]]


@pytest.mark.parametrize("p", [1, 2, 3, 7, 36, 100])
def test_int32_closed_form(orc, p):
    m = 17
    K = 1000003
    x = np.array([[(i * K + e) for e in range(m)] for i in range(p)],
                 dtype=np.int64).astype(np.int32)
    want = np.array([(K * p * (p - 1) // 2 + p * e) & M32 for e in range(m)],
                    dtype=np.uint64).astype(np.uint32).view(np.int32)
    for f in (orc.left_fold, orc.tree_fold):
        assert (f(x, orc.I32) == want).all()


def test_int32_wraps(orc):
    x = np.full((4, 3), 1 << 30, np.int32)  # 4 * 2^30 = 2^32 == 0 mod 2^32
    assert (orc.left_fold(x, orc.I32) == 0).all()
    assert (orc.tree_fold(x, orc.I32) == 0).all()
    x = np.full((3, 2), 2**31 - 1, np.int32)  # 3*(2^31-1) mod 2^32 = 2^31 - 3
    want = np.uint32((3 * (2**31 - 1)) & M32).view(np.int32)
    assert (orc.tree_fold(x, orc.I32) == want).all()


def _read_mats(line):
    return [[int(v) for v in t.split(",")] for t in line.split()]


def test_mat_golden(orc):
    n = 0
    for line in open(os.path.join(GOLD, "mat2x2_order.txt")):
        if not line.strip() or line.startswith("#"):
            continue
        p, xs, ys, _ = [f.strip() for f in line.split(";")]
        p = int(p)
        x = np.array(_read_mats(xs), dtype=np.uint32).reshape(p, 1, 4)
        want = np.array(_read_mats(ys)[0], dtype=np.uint32)
        for f in (orc.left_fold, orc.tree_fold):
            assert f(x, orc.MAT)[0].tolist() == want.tolist(), line
        n += 1
    assert n >= 6


def test_mat_affine_closed_form(orc):
    """[a_i b_i; 0 1] are affine maps; their product in rank order is
    [prod a_i, sum_i (prod_{k<i} a_k) b_i; 0 1] (mod 2^32)."""
    rng = np.random.default_rng(7)
    for p in (1, 2, 5, 36, 77):
        a = rng.integers(0, 2**32, p, dtype=np.uint64)
        b = rng.integers(0, 2**32, p, dtype=np.uint64)
        x = np.zeros((p, 1, 4), np.uint32)
        x[:, 0, 0] = a
        x[:, 0, 1] = b
        x[:, 0, 3] = 1
        A, B, pre = 1, 0, 1
        for i in range(p):
            B = (B + pre * int(b[i])) & M32
            pre = (pre * int(a[i])) & M32
        A = pre
        for f in (orc.left_fold, orc.tree_fold):
            assert f(x, orc.MAT)[0].tolist() == [A, B, 0, 1]


def test_mat_brute_force_python_ints(orc):
    rng = np.random.default_rng(11)
    for p in range(1, 11):
        for m in (1, 4):
            x = rng.integers(0, 2**32, (p, m, 4), dtype=np.uint64).astype(np.uint32)
            for e in range(m):
                P = [[1, 0], [0, 1]]
                for i in range(p):
                    Q = [[int(x[i, e, 0]), int(x[i, e, 1])],
                         [int(x[i, e, 2]), int(x[i, e, 3])]]
                    P = [[(P[r][0] * Q[0][c] + P[r][1] * Q[1][c]) & M32
                          for c in range(2)] for r in range(2)]
                want = [P[0][0], P[0][1], P[1][0], P[1][1]]
                assert orc.left_fold(x, orc.MAT)[e].tolist() == want
                assert orc.tree_fold(x, orc.MAT)[e].tolist() == want


@pytest.mark.parametrize("p", list(range(1, 41)) + [1152])
def test_tree_equals_left_for_exact_ops(orc, p):
    rng = np.random.default_rng(p)
    xi = rng.integers(-2**31, 2**31, (p, 9), dtype=np.int64).astype(np.int32)
    assert (orc.tree_fold(xi, orc.I32) == orc.left_fold(xi, orc.I32)).all()
    xm = rng.integers(0, 2**32, (p, 5, 4), dtype=np.uint64).astype(np.uint32)
    assert (orc.tree_fold(xm, orc.MAT) == orc.left_fold(xm, orc.MAT)).all()


def _golden_fp32(which="dual"):
    for line in open(os.path.join(GOLD, "fp32_bracketing.txt")):
        if not line.strip() or line.startswith("#"):
            continue
        p, xs, y, why = [f.strip() for f in line.split(";")]
        topo = "single" if p.startswith("single") else "dual"
        if topo != which:
            continue
        p = int(p.split()[-1])
        x = np.array([float.fromhex(v) if v != "0" else 0.0 for v in xs.split()],
                     dtype=np.float32).reshape(p, 1)
        yield p, x, np.float32(float.fromhex(y)), why


def test_fp32_golden_bracketing(orc):
    n = 0
    for which, topo in (("dual", orc.DUAL), ("single", orc.SINGLE)):
        for p, x, y, why in _golden_fp32(which):
            got = orc.tree_fold(x, orc.F32, topo)[0]
            assert got.tobytes() == y.tobytes(), (which, p, why, float(got).hex())
            n += 1
    assert n >= 9


def test_fp32_golden_differs_from_left_fold(orc):
    """The bracketing matters: at least one golden case differs from the
    left-to-right sum, so the golden values pin the tree, not the sum."""
    diffs = sum(orc.left_fold(x, orc.F32)[0] != y for _, x, y, _ in _golden_fp32())
    assert diffs >= 3


@pytest.mark.parametrize("p", [2, 3, 7, 32, 36, 200])
def test_fp32_error_bound(orc, p):
    """Any bracketing of a p-term float32 sum is within (p-1) u sum|x_i|
    (u = 2^-24) of the exact sum; a tree of height h within about h u sum|x|.
    The tree fold is checked against the float64 sum with the bound
    4 ceil(log2 p) 2^-24 sum|x_i| used for any re-bracketed float32 path."""
    rng = np.random.default_rng(p)
    x = rng.standard_normal((p, 4096)).astype(np.float32)
    y = orc.tree_fold(x, orc.F32).astype(np.float64)
    ref, absum = orc.left_fold_f64(x)
    bound = 4 * math.ceil(math.log2(p)) * 2.0**-24 * absum
    assert (np.abs(y - ref) <= bound).all()


def test_fp32_p1_and_p2(orc):
    x = np.array([[1.5, -2.25]], np.float32)
    assert orc.tree_fold(x, orc.F32).tolist() == [1.5, -2.25]
    x = np.array([[1.0], [2.0**-24]], np.float32)
    assert orc.tree_fold(x, orc.F32)[0] == np.float32(1.0)


def test_allreduce_copies_to_all_rows(orc):
    rng = np.random.default_rng(3)
    x = rng.integers(-1000, 1001, (7, 100), dtype=np.int64).astype(np.int32)
    y = orc.allreduce(x, orc.I32)
    assert (y == orc.tree_fold(x, orc.I32)[None, :]).all()


def _read_fmats(line):
    return [[float.fromhex(v) if v not in ("0", "-0") else 0.0 for v in t.split(",")]
            for t in line.split()]


def test_matf_golden(orc):
    n = 0
    for line in open(os.path.join(GOLD, "mat2x2_f32.txt")):
        if not line.strip() or line.startswith("#"):
            continue
        p, xs, ys, why = [f.strip() for f in line.split(";")]
        p = int(p)
        x = np.array(_read_fmats(xs), dtype=np.float32).reshape(p, 1, 4)
        want = np.array(_read_fmats(ys)[0], dtype=np.float32)
        got = orc.tree_fold(x, orc.MATF)[0]
        assert got.tobytes() == want.tobytes(), (why, got)
        n += 1
    assert n >= 2
    # the p = 3 case is one where the bracketing decides the bits
    x = np.array(_read_fmats("0x1.000002p+0,0,0,0x1p+0 0x1.fffffep-1,0,0,0x1p+0 "
                             "0x1.fffffep-1,0,0,0x1p+0"), np.float32).reshape(3, 1, 4)
    assert orc.left_fold(x, orc.MATF)[0, 0] == np.float32(1 - 2.0**-24)


@pytest.mark.parametrize("p", [1, 2, 3, 7, 12])
def test_matf_exact_on_small_integers(orc, p):
    """Small non-negative integer matrices: every product and sum is exact in
    float32, so the float32 product equals the uint32 product entry by entry
    (this pins the entry formulas and the operand order)."""
    rng = np.random.default_rng(100 + p)
    xi = rng.integers(0, 2, (p, 6, 4), dtype=np.int64)
    want = orc.left_fold(xi.astype(np.uint32), orc.MAT).astype(np.float64)
    assert want.max() < 2**24
    for f in (orc.left_fold, orc.tree_fold):
        assert np.array_equal(f(xi.astype(np.float32), orc.MATF).astype(np.float64), want)


@pytest.mark.parametrize("p", [2, 5, 16, 36])
def test_matf_close_to_exact_product(orc, p):
    """Near-identity float32 matrices: the tree-bracketed float32 product is
    within a few ulp (relative 1e-5) of the exact product computed with
    Python fractions."""
    from fractions import Fraction
    rng = np.random.default_rng(p)
    x = (np.eye(2).reshape(1, 1, 4) + rng.integers(-2**15, 2**15, (p, 3, 4)) * 2.0**-22)
    x = x.astype(np.float32)
    y = orc.tree_fold(x, orc.MATF)
    for e in range(3):
        P = [[Fraction(1), Fraction(0)], [Fraction(0), Fraction(1)]]
        for i in range(p):
            Q = [[Fraction(float(x[i, e, 0])), Fraction(float(x[i, e, 1]))],
                 [Fraction(float(x[i, e, 2])), Fraction(float(x[i, e, 3]))]]
            P = [[P[r][0] * Q[0][c] + P[r][1] * Q[1][c] for c in range(2)] for r in range(2)]
        ex = np.array([float(P[0][0]), float(P[0][1]), float(P[1][0]), float(P[1][1])])
        assert np.allclose(y[e].astype(np.float64), ex, rtol=0, atol=1e-5 * p)
