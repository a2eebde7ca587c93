"""In-tree build of libtcu_dft.so for sm_103a (nvcc, no cmake).

The library is a dozen translation units compiled in parallel -- the host
plan/ABI units and the kernel units (one per radix, mixed radix, BF16, the
element-wise grid kernels) -- linked into one shared object; the
bounds-checked variant is the same sources with -DTCU_DFT_CHECKED.
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
         "kernels_bf16_r8.cu", "kernels_bf16_r16.cu", "kernels_bf16_r32.cu",
         "grid_kernels.cu"]
HEADERS = ["tcgen05.cuh", "group_kernel.cuh", "launch.h",
           "launch_impl.cuh", "host_plan.h"]
HDR = os.path.join(os.path.dirname(HERE), "include", "tcu_dft.h")
LIB_PATH = os.path.join(HERE, "libtcu_dft.so")
BUILD_DIR = os.path.join(HERE, "_build")
# the bounds-checked variant: every shared-memory, tensor-memory and global
# index of the pass kernels checked; a violation skips the access and
# records TCU_DFT_ERR_BOUNDS
CHECKED_LIB_PATH = os.path.join(HERE, "libtcu_dft_checked.so")
CHECKED_BUILD_DIR = os.path.join(HERE, "_build_checked")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC"]
VARIANTS = {
    "release": ([], LIB_PATH, BUILD_DIR),
    "checked": (["-DTCU_DFT_CHECKED"], CHECKED_LIB_PATH, CHECKED_BUILD_DIR),
}


def nvcc() -> str:
    for c in (os.environ.get("NVCC"), shutil.which("nvcc"),
              "/usr/local/cuda/bin/nvcc"):
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found")


def _sources():
    return ([os.path.join(CSRC, u) for u in UNITS]
            + [os.path.join(CSRC, h) for h in HEADERS] + [HDR])


def build_variants(names=("release",), force: bool = False,
                   verbose: bool = False) -> list:
    """Compile the named variants (all translation units of all stale
    variants in parallel), link each; returns their library paths."""
    newest = max(os.path.getmtime(f) for f in _sources())
    cc = nvcc()
    jobs = []
    for name in names:
        defs, lib_path, build_dir = VARIANTS[name]
        if (not force and os.path.exists(lib_path)
                and os.path.getmtime(lib_path) >= newest):
            continue
        os.makedirs(build_dir, exist_ok=True)
        procs, objs = [], []
        for u in UNITS:
            obj = os.path.join(build_dir, u.replace(".cu", ".o"))
            cmd = [cc, *ARCH, *FLAGS, *defs, "-c", "-o", obj, os.path.join(CSRC, u)]
            if verbose:
                cmd.insert(1, "-Xptxas=-v")
            procs.append((u, subprocess.Popen(cmd)))
            objs.append(obj)
        jobs.append((name, lib_path, procs, objs))
    for name, lib_path, procs, objs in jobs:
        failed = [u for u, p in procs if p.wait() != 0]
        if failed:
            raise RuntimeError("nvcc failed on %s (%s)" % (", ".join(failed), name))
        tmp = lib_path + ".tmp%d" % os.getpid()
        subprocess.run([cc, *ARCH, "-shared", "-o", tmp, *objs], check=True)
        os.replace(tmp, lib_path)
    return [VARIANTS[n][1] for n in names]


def build(force: bool = False, verbose: bool = False, checked: bool = False) -> str:
    """Build libtcu_dft.so (or, with checked=True, libtcu_dft_checked.so)."""
    return build_variants(("checked",) if checked else ("release",), force, verbose)[0]


def build_all(force: bool = False) -> list:
    """Both variants, compiled together."""
    return build_variants(("release", "checked"), force)
