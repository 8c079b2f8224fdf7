"""In-tree build of the weight-sync library (librr.so) for GB300 (sm_103a).

The host planner (C++) and the CUDA kernels compile in parallel and link into
one shared library next to this file.  No CMake, no torch extension machinery:
the library is a plain C ABI (include/rr.h) loaded with ctypes.
"""
from __future__ import annotations

import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "librr.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def _cuda_home() -> str:
    home = os.environ.get("CUDA_HOME") or os.environ.get("CUDA_PATH")
    if home:
        return home
    nvcc = shutil.which("nvcc")
    if nvcc:
        return os.path.dirname(os.path.dirname(os.path.realpath(nvcc)))
    return "/usr/local/cuda"


def _sources():
    return [os.path.join(CSRC, f) for f in ("rr_plan.cpp", "rr_device.cu", "rr_internal.h")] + \
        [os.path.join(INCLUDE, "rr.h")]


def stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(s) > t for s in _sources())


def build(force: bool = False, verbose: bool = False) -> str:
    if not force and not stale():
        return LIB
    os.makedirs(BUILD, exist_ok=True)
    cuda = _cuda_home()
    nvcc = os.path.join(cuda, "bin", "nvcc")
    if not os.path.exists(nvcc):
        nvcc = "nvcc"
    inc = ["-I", INCLUDE, "-I", CSRC, "-I", os.path.join(cuda, "include")]
    plan_o = os.path.join(BUILD, "rr_plan.o")
    dev_o = os.path.join(BUILD, "rr_device.o")
    jobs = [
        ["g++", "-O2", "-std=c++17", "-fPIC", "-Wall"] +
        os.environ.get("RR_EXTRA_CXX_FLAGS", "").split() +
        ["-c", os.path.join(CSRC, "rr_plan.cpp"), "-o", plan_o] + inc,
        [nvcc, "-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xptxas", "-v"] + ARCH +
        os.environ.get("RR_EXTRA_NVCC_FLAGS", "").split() +
        ["-c", os.path.join(CSRC, "rr_device.cu"), "-o", dev_o] + inc,
    ]
    procs = [subprocess.Popen(j, stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True)
             for j in jobs]
    logs = []
    for j, p in zip(jobs, procs):
        out, _ = p.communicate()
        logs.append(out)
        if p.returncode != 0:
            raise RuntimeError(f"build failed: {' '.join(j)}\n{out}")
    with open(os.path.join(BUILD, "ptxas.log"), "w") as f:
        f.write(logs[1])
    if verbose:
        print(logs[1])
    tmp = LIB + ".tmp"
    subprocess.check_call([nvcc, "-shared"] + ARCH + [plan_o, dev_o, "-o", tmp])
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    build(force=True, verbose=True)
