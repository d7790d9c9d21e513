"""Pins for the oracle's simulation of the alternative the paper compares
against (Sec. 1.2, last paragraphs; Sec. 2, item 3, "User-Allreduce1"): a
pipelined reduction of b blocks to the root of one binary tree, followed by
a pipelined broadcast of the same b blocks from it.

What the paper fixes and these tests check:
  - the result is the one tree's post-order bracketing, so it equals the
    oracle's one-tree fold bit for bit (float32 included), orders every
    operand (interval witness), and equals the plain left fold for exact
    operators;
  - every transfer pairs (no mismatch, no deadlock), 2 (p-1) b transfers;
  - each phase takes two steps per block (a node receives from two children
    one after the other, and sends to two children one after the other), so
    the whole operation grows by four steps per block against Algorithm 1's
    three on the same tree -- the 4 beta m against 3 beta m of Sec. 1.2;
  - for p = 2^h - 1 the step counts have closed forms, within the paper's
    2 (2h + 2(b-1)): reduction ends at the root at 2(h-1) + 2(b-1), the
    whole operation at 4(h-1) + 4(b-1);
  - the broadcast starts only after the reduction has ended at the root; a
    planted mistake that broadcasts early is caught.
"""
import numpy as np
import pytest


def witness(p, m):
    x = np.zeros((p, m, 2), np.int32)
    for i in range(p):
        x[i] = i
    return x


@pytest.mark.parametrize("p", list(range(1, 41)) + [100, 255])
def test_result_is_the_one_tree_bracketing(orc, p):
    rng = np.random.default_rng(100 + p)
    m = 13
    for b in sorted({1, 2, 3, min(5, m), m}):
        x = rng.integers(-1000, 1000, (p, m), dtype=np.int32)
        y, st = orc.simulate_rb(x, orc.I32, b)
        assert (y == orc.left_fold(x, orc.I32)[None, :]).all()
        xf = rng.standard_normal((p, m)).astype(np.float32) * np.float32(1e3)
        yf, _ = orc.simulate_rb(xf, orc.F32, b)
        want = orc.tree_fold(xf, orc.F32, orc.SINGLE)
        assert (yf.view(np.uint32) == want.view(np.uint32)[None, :]).all()
        yw, _ = orc.simulate_rb(witness(p, m), orc.WIT, b)
        assert (yw[:, :, 0] == 0).all() and (yw[:, :, 1] == p - 1).all()
        xm = rng.integers(0, 2**32, (p, m, 4), dtype=np.uint64).astype(np.uint32)
        ym, _ = orc.simulate_rb(xm, orc.MAT, b)
        assert (ym == orc.left_fold(xm, orc.MAT)[None, :]).all()
        assert st["transfers"] == 2 * (p - 1) * b
        assert st["max_ops"] <= 2


@pytest.mark.parametrize("h", range(1, 8))
def test_closed_form_step_counts(orc, h):
    p = 2**h - 1
    x = np.zeros((p, 16), np.int32)
    for b in range(1, 10):
        _, st = orc.simulate_rb(x, orc.I32, b)
        if h == 1:
            assert st["steps"] == 0
            continue
        assert st["reduce_end_root"] == 2 * (h - 1) + 2 * (b - 1)
        assert st["first_bcast_start"] == st["reduce_end_root"]
        assert st["steps"] == 4 * (h - 1) + 4 * (b - 1)
        assert st["first_block_last"] == 4 * (h - 1) + 2 * (b - 1)
        assert st["steps"] <= 2 * (2 * h + 2 * (b - 1))   # the paper's count


@pytest.mark.parametrize("p", range(2, 70))
def test_four_steps_per_block(orc, p):
    """Two steps per block in each phase: four in all (two where the tree is a
    single edge, p = 2, whose nodes have one child)."""
    x = np.zeros((p, 16), np.int32)
    steps = [orc.simulate_rb(x, orc.I32, b)[1]["steps"] for b in range(1, 9)]
    slope = 2 if p == 2 else 4
    assert all(steps[k + 1] - steps[k] == slope for k in range(len(steps) - 1))
    for b in range(1, 9):
        _, st = orc.simulate_rb(x, orc.I32, b)
        assert st["first_bcast_start"] >= st["reduce_end_root"]


@pytest.mark.parametrize("h", range(3, 8))
def test_one_more_step_per_block_than_algorithm_1(orc, h):
    """On the same one tree, Algorithm 1 needs three steps per further block
    and the reduce-then-broadcast four: from the second block on, the gap
    grows by exactly one step per block."""
    p = 2**h - 1
    x = np.zeros((p, 16), np.int32)
    rb = [orc.simulate_rb(x, orc.I32, b)[1]["steps"] for b in range(1, 12)]
    a1 = [orc.simulate(x, orc.I32, b, orc.SINGLE)[1]["steps"] for b in range(1, 12)]
    for k in range(1, len(rb) - 1):
        assert rb[k + 1] - rb[k] == 4 and a1[k + 1] - a1[k] == 3


def test_empty_and_invalid(orc):
    x = np.zeros((3, 4), np.int32)
    with pytest.raises(orc.OracleError):
        orc.simulate_rb(x, orc.I32, 0)
    with pytest.raises(orc.OracleError):
        orc.simulate_rb(x, orc.I32, 5)    # b > m


@pytest.mark.parametrize("p", [3, 7, 10, 31, 40])
def test_planted_early_broadcast_is_caught(orc, p):
    """The root broadcasting a block as soon as child_0's part has arrived
    (before child_1's, before its reduction has ended) gives the children a
    block without child_1's subtree: the witness and the step pin see it."""
    try:
        orc.set_mutation(5)
        for b in (1, 2, 4):
            y, st = orc.simulate_rb(witness(p, 4), orc.WIT, b)
            wrong = not ((y[:, :, 0] == 0).all() and (y[:, :, 1] == p - 1).all())
            early = st["first_bcast_start"] < st["reduce_end_root"]
            assert wrong and early
    finally:
        orc.set_mutation(0)
