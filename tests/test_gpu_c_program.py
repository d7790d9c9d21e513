"""The C ABI from a plain C99 program (tests/c_abi_program.c), with no
Python in the call path: plan, fused kernel, schedule kernel with both
transports, host buffers and the allocation-free entry point, each result
checked against an exact int32 sum inside the program."""
import subprocess

import pytest

import c_build

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def program(tmp_path_factory):
    from paper_2109_12626_gb300 import build as B
    B.build()
    if c_build.cc() is None:
        pytest.skip("no C compiler")
    r, exe = c_build.build_program(str(tmp_path_factory.mktemp("cprog")))
    assert r.returncode == 0, r.stderr
    return exe


@pytest.mark.parametrize("p,m", [(7, 1000), (1, 17), (2, 3), (1152, 4099), (3000, 33)])
def test_c_program(program, p, m):
    r = subprocess.run([program, str(p), str(m)], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr
