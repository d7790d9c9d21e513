"""Pins for the oracle's event-level simulation of Algorithm 1 (O4).

What the paper fixes and the simulation must show:
  - the correctness claim of Sec. 1.1: with d_i = depth every processor ends
    with y, by the same bracketing as the tree fold (bitwise, every op);
  - every bidirectional exchange finds its partner with matching blocks;
  - the loop bound b + d_i of Algorithm 1 / "b + d_i rounds" of Sec. 1.1;
  - at most two (.) per round for non-roots, three for roots (Sec. 1.2);
  - each further block costs three steps (Sec. 1.2), and the paper's
    latency count 4h-3 for p = 2^h - 2 bounds the first block's arrival.
Plus planted mistakes in the oracle, each caught by one of these pins."""
import numpy as np
import pytest


def witness(p, m):
    x = np.zeros((p, m, 2), np.int32)
    for i in range(p):
        x[i] = i
    return x


CASES = [(p, b) for p in range(1, 41) for b in (1, 2, 3, 5, 8)] + \
        [(62, 16), (126, 4), (255, 3), (1152, 2)]


@pytest.mark.parametrize("p,b", CASES)
def test_simulation_delivers_y_everywhere(orc, p, b):
    m = b + 3 if b < 8 else b
    y, st, last = orc.simulate(witness(p, m), orc.WIT, b)
    assert (y[:, :, 0] == 0).all() and (y[:, :, 1] == p - 1).all()


@pytest.mark.parametrize("p,b", [(p, b) for p in (1, 2, 3, 4, 7, 11, 32, 36)
                                 for b in (1, 2, 4, 7)])
def test_simulation_bitwise_equals_tree_fold(orc, p, b):
    rng = np.random.default_rng(1000 * p + b)
    m = 4 * b + 3
    xf = rng.standard_normal((p, m)).astype(np.float32)
    xi = rng.integers(-2**31, 2**31, (p, m), dtype=np.int64).astype(np.int32)
    xm = rng.integers(0, 2**32, (p, m, 4), dtype=np.uint64).astype(np.uint32)
    for x, dt in ((xf, orc.F32), (xi, orc.I32), (xm, orc.MAT)):
        y, _, _ = orc.simulate(x, dt, b)
        want = orc.tree_fold(x, dt)
        for i in range(p):
            assert y[i].tobytes() == want.tobytes(), (p, b, dt, i)


@pytest.mark.parametrize("p,b", [(p, b) for p in range(1, 70) for b in (1, 2, 5)])
def test_round_count(orc, p, b):
    """Last non-void exchange: round b+d_i for internal processors (the loop
    runs j = 0..b+d_i) and b+d_i-1 for leaves (b+d_i rounds)."""
    T = orc.trees(p)
    _, st, last = orc.simulate(witness(p, b), orc.WIT, b)
    for i in range(p):
        internal = T["child0"][i] >= 0
        d = int(T["depth"][i])
        if p == 1:
            assert last[i] == -1
        elif internal:
            assert last[i] == b + d
        else:
            assert last[i] == b + d - 1


@pytest.mark.parametrize("p", [3, 7, 36, 100])
def test_reduction_counts_per_round(orc, p):
    _, st, _ = orc.simulate(witness(p, 8), orc.WIT, 8)
    assert st["max_ops_nonroot"] <= 2
    assert st["max_ops_root"] <= 3
    if p >= 6:  # both roots have two children: the dual's (.) is the third
        assert st["max_ops_root"] == 3


@pytest.mark.parametrize("h", range(3, 9))
def test_latency_and_three_steps_per_block(orc, h):
    p = 2**h - 2
    steps = []
    for b in range(1, 7):
        _, st, _ = orc.simulate(witness(p, b), orc.WIT, b)
        assert st["first_block_last"] <= 4 * h - 3   # the paper's count bounds it
        assert st["steps"] <= 4 * h - 3 + 3 * (b - 1)
        steps.append(st["steps"])
    assert np.diff(steps).tolist() == [3] * 5       # three steps per block


def test_two_roots_only_exchange(orc):
    """p = 2: two single-node trees; each round is one exchange, b steps."""
    for b in (1, 2, 6):
        _, st, last = orc.simulate(witness(2, b), orc.WIT, b)
        assert st["steps"] == b and st["exchanges"] == b
        assert last.tolist() == [b - 1, b - 1]


# ------------------------------------------------------- planted mistakes

def _tree_pins_pass(orc):
    ok = True
    for p in (3, 7, 12):
        y = orc.tree_fold(witness(p, 2), orc.WIT)
        ok &= bool((y[:, 0] == 0).all() and (y[:, 1] == p - 1).all())
    return ok


def _sim_pins_pass(orc):
    from oracle.oracle import OracleError
    try:
        for p in (7, 12, 36):
            for b in (1, 3):
                y, _, last = orc.simulate(witness(p, b), orc.WIT, b)
                if not ((y[:, :, 0] == 0).all() and (y[:, :, 1] == p - 1).all()):
                    return False
        return True
    except OracleError:
        return False


@pytest.mark.parametrize("k,which", [(1, "tree"), (2, "tree"), (3, "sim"),
                                     (4, "sim")])
def test_planted_mistakes_are_caught(orc, k, which):
    assert _tree_pins_pass(orc) and _sim_pins_pass(orc)
    orc.set_mutation(k)
    try:
        if which == "tree":
            assert not _tree_pins_pass(orc)
        else:
            assert not _sim_pins_pass(orc)
    finally:
        orc.set_mutation(0)
    assert _tree_pins_pass(orc) and _sim_pins_pass(orc)
