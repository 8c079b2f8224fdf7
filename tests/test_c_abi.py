"""The C ABI used from a plain C11 program (tests/c/rr_abi_check.c).

The header must compile as C11 (with -Wall -Wextra -Werror -pedantic), and the
library must link and answer from C exactly as the Python binding sees it.  The CPU
test runs the host-side calls on a host-only plan; the GPU test runs the same
program against the device: pack, verify, unpack, and damage detection,
compared with bytes worked out by hand in the program.
"""
import os
import subprocess

import pytest

from paper_2512_22492_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "tests", "c", "rr_abi_check.c")


def cudart_dir(cuda: str) -> str:
    """The directory holding libcudart.so (lib64, or the target tree on Arm)."""
    import glob
    for d in [os.path.join(cuda, "lib64"), os.path.join(cuda, "lib")] + \
            sorted(glob.glob(os.path.join(cuda, "targets", "*", "lib"))):
        if os.path.exists(os.path.join(d, "libcudart.so")):
            return d
    pytest.skip("libcudart.so not found under the CUDA toolkit")


def compile_check(tmp_path) -> str:
    cuda = B._cuda_home()
    rt = cudart_dir(cuda)
    exe = str(tmp_path / "rr_abi_check")
    lib_dir = os.path.dirname(B.LIB)
    subprocess.check_call(
        ["gcc", "-std=c11", "-O1", "-Wall", "-Wextra", "-Werror", "-pedantic",
         "-I", os.path.join(ROOT, "include"), "-I", os.path.join(cuda, "include"),
         SRC, "-o", exe, "-L", lib_dir, "-lrr", f"-Wl,-rpath,{lib_dir}",
         "-L", rt, "-lcudart", f"-Wl,-rpath,{rt}"])
    return exe


def test_c_program_host_side(tmp_path):
    exe = compile_check(tmp_path)
    out = subprocess.run([exe], capture_output=True, text=True, timeout=60)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip() == "host ok"


@pytest.mark.gpu
def test_c_program_on_the_gpu(tmp_path):
    exe = compile_check(tmp_path)
    out = subprocess.run([exe, "gpu"], capture_output=True, text=True, timeout=120)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip() == "gpu ok"
