"""The C-ABI library without a GPU: it loads, exports every function that
include/dpdr.h declares, and its host-side plan logic (trees, block
partition, block-count rule) agrees with the independent oracle and with
what the paper fixes."""
import ctypes
import math
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def native():
    from paper_2109_12626_gb300 import build as B
    B.build()
    from paper_2109_12626_gb300 import _native as N
    N.lib()
    return N


def _declared():
    text = open(os.path.join(ROOT, "include", "dpdr.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(dpdr_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(native):
    names = _declared()
    assert len(names) >= 15
    L = ctypes.CDLL(native.LIB_PATH)
    for n in names:
        assert hasattr(L, n), n
    assert set(names) == set(native.SIGNATURES)


def test_no_cuda_runtime_dependency_at_load(native):
    # the runtime is linked statically: loading needs no GPU and no libcudart
    out = os.popen("ldd %s" % native.LIB_PATH).read()
    assert "libcudart" not in out


@pytest.mark.parametrize("p", list(range(1, 130)) + [255, 256, 1151, 1152, 4097])
def test_tree_matches_oracle(native, orc, p):
    a = native.tree(p)
    o = orc.trees(p)
    for k in ("parent", "child0", "child1", "dual", "depth"):
        assert np.array_equal(a[k], o[k]), k


@pytest.mark.parametrize("m,b", [(1, 1), (10, 3), (1000, 4), (65536, 16),
                                 (4194304, 228), (7, 7), (134217728, 1024)])
def test_block_partition(native, m, b):
    s = native.blocks(m, b)
    sizes = np.diff(s)
    assert s[0] == 0 and s[-1] == m
    assert sizes.max() - sizes.min() <= 1
    assert (sizes[: m % b] == -(-m // b)).all() and (sizes[m % b:] == m // b).all()


def test_block_partition_rejects(native):
    from paper_2109_12626_gb300 import DpdrError
    with pytest.raises(DpdrError):
        native.blocks(3, 4)
    with pytest.raises(DpdrError):
        native.blocks(3, 0)


@pytest.mark.parametrize("p,m", [(1152, 4194304), (1152, 1), (32, 134217728),
                                 (7, 1000), (2, 10**6), (1, 5)])
def test_block_count_rule(native, p, m):
    """Sec. 1.2 pipelining optimum b* = sqrt((4h-6) m beta / (3 alpha)),
    h = ceil(log2(p+2)), kappa = alpha/beta = 1024 elements by default."""
    h = math.ceil(math.log2(p + 2))
    want = min(max(round(math.sqrt((4 * h - 6) * m / (3 * 1024.0))), 1), max(m, 1))
    assert native.block_count_rule(p, m) == want
    if (p, m) == (1152, 4194304):
        assert want == 228  # h = 11: sqrt(38 * 4194304 / 3072)


def test_block_count_rule_minimises_model(native):
    """The rule's b minimises the Sec. 1.2 time (4h-3+3(b-1))(alpha+beta m/b)
    over integers, up to rounding, for p = 2^h - 2."""
    for h in (3, 5, 11):
        p = 2**h - 2
        for m in (10**4, 10**6, 4194304):
            for kappa in (64.0, 1024.0):
                T = lambda b: (4 * h - 3 + 3 * (b - 1)) * (kappa + m / b)
                b = native.block_count_rule(p, m, kappa)
                best = min(range(1, 20000), key=T)
                assert T(b) <= T(best) * 1.001


def test_status_strings(native):
    L = native.lib()
    for s in range(6):
        assert L.dpdr_status_string(s)
    assert b"unknown" in L.dpdr_status_string(99)


@pytest.mark.parametrize("p", list(range(1, 80)) + [1023, 1152, 4097])
def test_single_tree_matches_oracle(native, orc, p):
    a = native.tree(p, "single")
    o = orc.trees(p, orc.SINGLE)
    for k in ("parent", "child0", "child1", "dual", "depth"):
        assert np.array_equal(a[k], o[k]), k


def test_header_is_iso_c99_and_a_c_program_links(native, tmp_path):
    """The boundary stands without Python: include/dpdr.h compiles as strict
    C99, and a plain C program that calls every run entry point links
    against libdpdr.so and the CUDA runtime (it runs in the GPU tests)."""
    import c_build
    if c_build.cc() is None:
        pytest.skip("no C compiler")
    r = c_build.compile_header_as_c(str(tmp_path))
    assert r.returncode == 0, r.stderr
    if not os.path.exists(os.path.join(c_build.CUDA, "include", "cuda_runtime_api.h")):
        pytest.skip("no CUDA headers")
    r, exe = c_build.build_program(str(tmp_path))
    assert r.returncode == 0, r.stderr
    assert os.path.exists(exe)


def test_info_keys_follow_the_header():
    """The binding names one key per entry dpdr.h documents for
    dpdr_plan_info, no more and no fewer."""
    import re
    from paper_2109_12626_gb300 import _native as N
    h = open(os.path.join(ROOT, "include", "dpdr.h")).read()
    doc = h[h.index("Plan facts for tools and tests"):h.index("int dpdr_plan_info(")]
    idx = sorted({int(k) for k in re.findall(r"\[(\d+)\]", doc)})
    assert idx == list(range(len(N.INFO_KEYS)))

