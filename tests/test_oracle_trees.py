"""Pins for the oracle's tree builder (O1), against what Sec. 1.1 fixes:
two roughly equal trees, post-order numbering (every subtree a contiguous
rank interval ending at its root), child_0 = i-1, the second child i'' the
root of the lower interval [i', i''], roots that are duals, d_i = depth, and
trees "as balanced and complete as possible" (read: complete binary trees)."""
import itertools
import math

import numpy as np
import pytest

PS = list(range(1, 80)) + [127, 128, 254, 255, 256, 1152]


def subtree_interval(T, i):
    """Smallest rank in i's subtree, found by walking child links."""
    lo = i
    stack = [i]
    while stack:
        k = stack.pop()
        lo = min(lo, k)
        for c in (T["child0"][k], T["child1"][k]):
            if c >= 0:
                stack.append(int(c))
    return lo


@pytest.mark.parametrize("p", PS)
def test_sizes_roots_duals(orc, p):
    T = orc.trees(p)
    n0 = p // 2
    roots = [i for i in range(p) if T["parent"][i] < 0]
    if p == 1:
        assert roots == [0] and T["dual"][0] == -1
        return
    # two trees of floor(p/2) and ceil(p/2) ranks, roots r0 = n0-1, r1 = p-1
    assert roots == [n0 - 1, p - 1]
    assert T["dual"][n0 - 1] == p - 1 and T["dual"][p - 1] == n0 - 1
    assert all(T["dual"][i] == -1 for i in range(p) if i not in roots)
    assert subtree_interval(T, n0 - 1) == 0
    assert subtree_interval(T, p - 1) == n0


@pytest.mark.parametrize("p", PS)
def test_postorder_intervals(orc, p):
    T = orc.trees(p)
    c0, c1, par, dep = T["child0"], T["child1"], T["parent"], T["depth"]
    for i in range(p):
        if c0[i] < 0:
            assert c1[i] < 0, "a lone child must be child_0"
            continue
        assert c0[i] == i - 1, "child_0 = i-1"
        lo = subtree_interval(T, i)
        if c1[i] >= 0:
            # [i', i''] then [i''+1, i-1] then i
            assert lo == subtree_interval(T, int(c1[i]))
            assert subtree_interval(T, i - 1) == c1[i] + 1
            assert c1[i] < i - 1
        else:
            assert lo == subtree_interval(T, i - 1)
        for c in (c0[i], c1[i]):
            if c >= 0:
                assert par[c] == i
                assert dep[c] == dep[i] + 1
    for i in range(p):
        if par[i] < 0:
            assert dep[i] == 0


def _complete_by_bfs(T, root):
    """Textbook test of a complete binary tree: in breadth-first order with
    the lower-ranked (left) child first, no present node follows a missing
    child slot."""
    order = [root]
    seen_gap = False
    k = 0
    while k < len(order):
        i = order[k]
        k += 1
        c0, c1 = int(T["child0"][i]), int(T["child1"][i])
        # left child = lower interval: child_1 if two children, else child_0
        left, right = (c1, c0) if c1 >= 0 else (c0, -1)
        for c in (left, right):
            if c < 0:
                seen_gap = True
            else:
                if seen_gap:
                    return False
                order.append(c)
    return True


@pytest.mark.parametrize("p", PS)
def test_complete_and_balanced(orc, p):
    T = orc.trees(p)
    n0 = p // 2
    for root, n in ((n0 - 1, n0), (p - 1, p - n0)):
        if n == 0:
            continue
        assert _complete_by_bfs(T, root)
        members = [i for i in range(p) if subtree_interval(T, root) <= i <= root]
        height = max(int(T["depth"][i]) for i in members)
        assert height == int(math.floor(math.log2(n)))  # minimum possible


def _shapes(n):
    """All binary tree shapes with n nodes as nested (left, right) tuples."""
    if n == 0:
        yield None
        return
    for left in range(n):
        for L in _shapes(left):
            for R in _shapes(n - 1 - left):
                yield (L, R)


def _height(s):
    return -1 if s is None else 1 + max(_height(s[0]), _height(s[1]))


def _is_complete(s):
    q, gap = [s], False
    while q:
        t = q.pop(0)
        for c in (t[0], t[1]):
            if c is None:
                gap = True
            elif gap:
                return False
            else:
                q.append(c)
    return True


def _shape_of(T, i):
    c0, c1 = int(T["child0"][i]), int(T["child1"][i])
    if c0 < 0:
        return (None, None)
    if c1 < 0:
        return (_shape_of(T, c0), None)
    return (_shape_of(T, c1), _shape_of(T, c0))


@pytest.mark.parametrize("n", range(1, 10))
def test_shape_is_the_unique_complete_tree_brute_force(orc, n):
    """Enumerate every binary tree with n nodes: exactly one is complete,
    it has the minimum height, and it is the oracle's tree 1 for p = 2n-1
    (tree 1 has ceil(p/2) = n nodes)."""
    shapes = list(_shapes(n))
    assert len(shapes) == math.comb(2 * n, n) // (n + 1)  # Catalan number
    complete = [s for s in shapes if _is_complete(s)]
    assert len(complete) == 1
    hmin = min(_height(s) for s in shapes)
    assert _height(complete[0]) == hmin
    p = 2 * n - 1
    T = orc.trees(p)
    assert _shape_of(T, p - 1) == complete[0]


@pytest.mark.parametrize("p,roots,tree_sizes,max_depth", [
    (7, (2, 6), (3, 4), 2),        # the p=7 workload: trees of 3 and 4
    (32, (15, 31), (16, 16), 4),
    (36, (17, 35), (18, 18), 4),
    (1152, (575, 1151), (576, 576), 9),
])
def test_workload_trees(orc, p, roots, tree_sizes, max_depth):
    T = orc.trees(p)
    assert tuple(i for i in range(p) if T["parent"][i] < 0) == roots
    assert (p // 2, p - p // 2) == tree_sizes
    assert int(T["depth"].max()) == max_depth


def test_p7_tables_by_hand(orc):
    """p = 7 written out: tree 0 = {0,1,2}, tree 1 = {3,4,5,6}; the 4-node
    complete tree has a root with two children, the left one holding the
    fourth node."""
    T = orc.trees(7)
    assert T["parent"].tolist() == [2, 2, -1, 4, 6, 6, -1]
    assert T["child0"].tolist() == [-1, -1, 1, -1, 3, -1, 5]
    assert T["child1"].tolist() == [-1, -1, 0, -1, -1, -1, 4]
    assert T["depth"].tolist() == [1, 1, 0, 2, 1, 1, 0]
    assert T["dual"].tolist() == [-1, -1, 6, -1, -1, -1, 2]
