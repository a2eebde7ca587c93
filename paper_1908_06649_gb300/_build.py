"""In-tree build of libtcu_dft.so for sm_103a (nvcc, no cmake).

The library is four translation units compiled in parallel -- the host
plan/ABI and one kernel unit per radix -- then linked into one shared object.
"""
from __future__ import annotations

import os
import shutil
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
CSRC = os.path.join(HERE, "csrc")
UNITS = ["tcu_dft.cu", "host_tables.cu", "noalloc.cu", "grid_plan.cu",
         "kernels_r8.cu", "kernels_r16.cu", "kernels_r32.cu",
         "kernels_mixed_r8.cu", "kernels_mixed_r16.cu", "kernels_mixed_r32.cu",
         "kernels_bf16_r16.cu",
         "grid_kernels.cu"]
HEADERS = ["tcgen05.cuh", "group_kernel.cuh", "launch.h",
           "launch_impl.cuh", "host_plan.h"]
HDR = os.path.join(os.path.dirname(HERE), "include", "tcu_dft.h")
LIB_PATH = os.path.join(HERE, "libtcu_dft.so")
BUILD_DIR = os.path.join(HERE, "_build")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC"]


def nvcc() -> str:
    for c in (os.environ.get("NVCC"), shutil.which("nvcc"),
              "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def _sources():
    return ([os.path.join(CSRC, u) for u in UNITS]
            + [os.path.join(CSRC, h) for h in HEADERS] + [HDR])


def build(force: bool = False, verbose: bool = False) -> str:
    newest = max(os.path.getmtime(f) for f in _sources())
    if (not force and os.path.exists(LIB_PATH)
            and os.path.getmtime(LIB_PATH) >= newest):
        return LIB_PATH
    os.makedirs(BUILD_DIR, exist_ok=True)
    cc = nvcc()
    procs, objs = [], []
    for u in UNITS:
        obj = os.path.join(BUILD_DIR, u.replace(".cu", ".o"))
        cmd = [cc, *ARCH, *FLAGS, "-c", "-o", obj, os.path.join(CSRC, u)]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        procs.append((u, subprocess.Popen(cmd)))
        objs.append(obj)
    failed = [u for u, p in procs if p.wait() != 0]
    if failed:
        raise RuntimeError("nvcc failed on %s" % ", ".join(failed))
    tmp = LIB_PATH + ".tmp%d" % os.getpid()
    subprocess.run([cc, *ARCH, "-shared", "-o", tmp, *objs], check=True)
    os.replace(tmp, LIB_PATH)
    return LIB_PATH
