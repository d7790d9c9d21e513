"""Builds tests/c_abi_program.c, a plain C99 user of include/dpdr.h and
libdpdr.so (test infrastructure only)."""
import os
import shutil
import subprocess

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2109_12626_gb300")
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def cc():
    return shutil.which("gcc") or shutil.which("cc")


def compile_header_as_c(out_dir: str) -> subprocess.CompletedProcess:
    """dpdr.h alone, as strict ISO C99 with every warning an error."""
    src = os.path.join(out_dir, "header_only.c")
    with open(src, "w") as f:
        f.write('#include "dpdr.h"\nint main(void) { return dpdr_last_error(); }\n')
    return subprocess.run([cc(), "-std=c99", "-pedantic", "-Wall", "-Wextra", "-Werror", "-c",
                           "-I", os.path.join(ROOT, "include"), src, "-o",
                           os.path.join(out_dir, "header_only.o")],
                          capture_output=True, text=True)


def build_program(out_dir: str) -> tuple[subprocess.CompletedProcess, str]:
    """The example program linked against libdpdr.so and the CUDA runtime."""
    exe = os.path.join(out_dir, "c_abi_program")
    lib64 = os.path.join(CUDA, "lib64")
    r = subprocess.run([cc(), "-std=c99", "-Wall", "-Wextra", "-Werror", "-O1",
                        "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA, "include"),
                        os.path.join(ROOT, "tests", "c_abi_program.c"), "-o", exe,
                        "-L", PKG, "-ldpdr", "-L", lib64, "-lcudart",
                        "-Wl,-rpath," + PKG, "-Wl,-rpath," + lib64],
                       capture_output=True, text=True)
    return r, exe
