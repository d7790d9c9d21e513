"""Pins for the oracle's one-tree variant (Sec. 1.2: "only one, doubly
pipelined binary tree"): one complete post-order tree over all p ranks,
root p-1, no dual; Algorithm 1 then needs no dual-root step, every
non-leaf (the root included) applies (.) at most twice per round, and for
p + 1 = 2^h the first block of y reaches the last leaf within 4h steps."""
import math

import numpy as np
import pytest

from test_oracle_trees import _complete_by_bfs, subtree_interval


def witness(p, m):
    x = np.zeros((p, m, 2), np.int32)
    for i in range(p):
        x[i] = i
    return x


@pytest.mark.parametrize("p", list(range(1, 70)) + [255, 1023, 1152])
def test_single_tree_shape(orc, p):
    T = orc.trees(p, orc.SINGLE)
    roots = [i for i in range(p) if T["parent"][i] < 0]
    assert roots == [p - 1]
    assert (T["dual"] == -1).all()
    assert subtree_interval(T, p - 1) == 0
    assert _complete_by_bfs(T, p - 1)
    assert int(T["depth"].max()) == int(math.floor(math.log2(p)))
    for i in range(p):
        if T["child0"][i] >= 0:
            assert T["child0"][i] == i - 1


@pytest.mark.parametrize("p", list(range(1, 41)) + [255, 1152])
def test_single_tree_fold_orders_operands(orc, p):
    y = orc.tree_fold(witness(p, 2), orc.WIT, orc.SINGLE)
    assert (y[:, 0] == 0).all() and (y[:, 1] == p - 1).all()
    rng = np.random.default_rng(p)
    xm = rng.integers(0, 2**32, (p, 5, 4), dtype=np.uint64).astype(np.uint32)
    assert (orc.tree_fold(xm, orc.MAT, orc.SINGLE) == orc.left_fold(xm, orc.MAT)).all()


@pytest.mark.parametrize("p,b", [(p, b) for p in (1, 2, 3, 5, 7, 12, 31, 40) for b in (1, 2, 5)])
def test_single_simulation_equals_fold(orc, p, b):
    rng = np.random.default_rng(7 * p + b)
    m = 3 * b + 2
    xf = rng.standard_normal((p, m)).astype(np.float32)
    y, st, last = orc.simulate(xf, orc.F32, b, orc.SINGLE)
    want = orc.tree_fold(xf, orc.F32, orc.SINGLE)
    for i in range(p):
        assert y[i].tobytes() == want.tobytes()
    yw, _, _ = orc.simulate(witness(p, m), orc.WIT, b, orc.SINGLE)
    assert (yw[:, :, 0] == 0).all() and (yw[:, :, 1] == p - 1).all()
    T = orc.trees(p, orc.SINGLE)
    for i in range(p):
        d = int(T["depth"][i])
        if p == 1:
            assert last[i] == -1
        elif T["child0"][i] >= 0:
            assert last[i] == b + d
        else:
            assert last[i] == b + d - 1
    assert st["max_ops_nonroot"] <= 2 and st["max_ops_root"] == 0  # no dual step


@pytest.mark.parametrize("h", range(2, 9))
def test_single_tree_latency_bound(orc, h):
    """p + 1 = 2^h: the first block of y reaches the last leaf within 4h
    steps, and each block after the second costs three more (two for h = 2,
    where the only non-leaf is the root, which has no parent step)."""
    p = 2**h - 1
    steps = []
    for b in range(1, 6):
        _, st, _ = orc.simulate(witness(p, b), orc.WIT, b, orc.SINGLE)
        assert st["first_block_last"] <= 4 * h
        steps.append(st["steps"])
    assert np.diff(steps)[1:].tolist() == [3 if h >= 3 else 2] * 3
