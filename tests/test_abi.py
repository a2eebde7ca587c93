"""The C ABI on the CPU: the library builds, loads, exports every symbol that
include/tcu_dft.h declares, and rejects bad arguments before touching CUDA."""
import ctypes
import os
import re
import subprocess

import pytest

from paper_1908_06649_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "tcu_dft.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tcu_[a-z0-9_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    _build.build()
    import paper_1908_06649_gb300 as pkg
    return pkg.lib()


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("tcu_dft_plan", "tcu_dft_exec", "tcu_dft_exec_dir",
                     "tcu_dft_destroy", "tcu_dft_last_error",
                     "tcu_dft_strerror"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", _build.LIB_PATH],
                         capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (\w+)", out))
    for name in declared_functions():
        assert name in exported, name
        assert getattr(lib, name) is not None


def test_checked_variant_exports_the_same_symbols():
    """The bounds-checked build (-DTCU_DFT_CHECKED) is the same boundary."""
    _build.build(checked=True)
    out = subprocess.run(["nm", "-D", "--defined-only", _build.CHECKED_LIB_PATH],
                         capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (\w+)", out))
    for name in declared_functions():
        assert name in exported, name


C_PROGRAM = r"""
#include <stdio.h>
#include <string.h>
#include "tcu_dft.h"
int main(void) {
  int32_t st[3] = {0, 0, 0};
  int64_t N = 0, B = 0;
  if (tcu_dft_plan_passes(65536, 16, st) != 2 || st[0] != 2 || st[1] != 2) return 1;
  if (tcu_dft_plan_passes(272, 16, st) != 0) return 2;             /* 17 * 16 */
  if (tcu_dft_plan_passes(48, 16, st) != 2 || st[0] != 1 || st[1] != 1) return 8;  /* 3 * 16 */
  if (tcu_stencil_tiles(4096, 16, 16, &N, &B) != 361 || N != 256 || B != 224) return 3;
  if (strcmp(tcu_dft_strerror(TCU_DFT_OK), "ok") != 0) return 4;
  if (tcu_dft_destroy(NULL) != TCU_DFT_OK) return 5;
  if (tcu_dft_plan(0, 1, 16, TCU_DFT_3XTF32) != NULL) return 6;
  if (tcu_dft_last_error() != TCU_DFT_ERR_INVALID) return 7;
  puts("c abi ok");
  return 0;
}
"""


def test_plain_c_program_uses_the_boundary(tmp_path):
    """The header is C99, and a plain C program links the library and calls
    its host-side entry points (no Python, no torch, no GPU)."""
    _build.build()
    src = tmp_path / "abi.c"
    src.write_text(C_PROGRAM)
    exe = tmp_path / "abi"
    libdir = os.path.dirname(_build.LIB_PATH)
    subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-pedantic",
                    "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe),
                    "-L", libdir, "-ltcu_dft", "-Wl,-rpath," + libdir],
                   check=True, capture_output=True, text=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True)
    assert out.returncode == 0 and "c abi ok" in out.stdout, (out.returncode, out.stderr)


def test_binding_lists_every_symbol():
    import paper_1908_06649_gb300 as pkg
    assert sorted(pkg.SYMBOLS) == declared_functions()


def test_strerror_and_null_handling(lib):
    import paper_1908_06649_gb300 as pkg
    assert lib.tcu_dft_strerror(0) == b"ok"
    assert lib.tcu_dft_strerror(pkg.ERR_TIMEOUT) == b"device wait timed out"
    assert b"out of range" in lib.tcu_dft_strerror(pkg.ERR_BOUNDS)
    assert lib.tcu_dft_destroy(None) == pkg.OK
    assert lib.tcu_dft_exec(None, None, None, None) == pkg.ERR_INVALID
    assert lib.tcu_dft_exec_dir(None, None, None, -1, None) == pkg.ERR_INVALID
    assert lib.tcu_dft_exec_host(None, None, None, None, -1, None) == pkg.ERR_INVALID
    assert lib.tcu_dft_check(None, None) == pkg.ERR_INVALID
    assert lib.tcu_dft_exec_stalled(None, None, None, None) == pkg.ERR_INVALID
    assert lib.tcu_dft_num_passes(None) == -1
    assert lib.tcu_dft_is_fused(None) == -1
    assert not lib.tcu_dft_plan_ex(256, 4, 16, 3, 8)   # unknown flag bit
    assert lib.tcu_dft_last_error() == pkg.ERR_INVALID
    assert not lib.tcu_dft_plan_ex(256, 4, 16, 3, 3)   # FUSE with NO_FUSE
    assert lib.tcu_dft_last_error() == pkg.ERR_INVALID
    assert not lib.tcu_dft_plan_ex(256, 4, 16, 3, 6)   # FUSE with ONE_PASS
    assert lib.tcu_dft_last_error() == pkg.ERR_INVALID
    assert not lib.tcu_dft_plan_ex(256, 4, 16, 3, 5)   # NO_FUSE with ONE_PASS
    assert lib.tcu_dft_last_error() == pkg.ERR_INVALID
    assert lib.tcu_dft_pass_stages(None, 0) == -1


@pytest.mark.parametrize("n,batch,r,prec,status", [
    (0, 1, 16, 3, 1),        # n < 1
    (16, 0, 16, 3, 1),       # batch < 1
    (16, 1, 16, 2, 1),       # precision not 1 or 3
    (16, 1, 16, 6, 1),       # precision not 1, 3, 4 or 5
    (128, 1, 8, 4, 2),       # BF16 modes: no mixed radix (2 x 8^2)
    (512, 1, 16, 5, 2),      # BF16 modes: no mixed radix
    (16, 1, 4, 3, 2),        # radix not in {8, 16, 32}
    (16, 1, 64, 3, 2),
    (17 * 16, 1, 16, 3, 2),  # a factor beyond 16
    (128, 1, 16, 3, 2),      # power of two but not of 16
    (2 * 16, 1, 16, 3, 2),   # mixed radix with one radix-16 stage (k < 2)
    (2 * 16 ** 5, 1, 16, 3, 2),  # mixed radix beyond k = 4
    (3 * 16 ** 3, 1, 16, 3, 2),  # an odd factor with more than one tensor pass
    (5 * 32 ** 3, 1, 32, 3, 2),
    (3 * 8 ** 4, 1, 8, 3, 2),
    (48, 1, 16, 4, 2),       # BF16 modes: no mixed radix (3 x 16)
    (16 ** 7, 1, 16, 3, 2),  # beyond three passes
    (32 ** 7, 1, 32, 3, 2),
    (8 ** 10, 1, 8, 3, 2),
])
def test_plan_rejects_before_cuda(lib, n, batch, r, prec, status):
    h = lib.tcu_dft_plan(n, batch, r, prec)
    assert not h
    assert lib.tcu_dft_last_error() == status


def test_plan_without_gpu_reports_cuda_error(lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    assert not lib.tcu_dft_plan(256, 4, 16, 3)
    assert lib.tcu_dft_last_error() == 3


@pytest.mark.parametrize("r,kmax", [(8, 3), (16, 2), (32, 2)])
def test_pass_grouping_odd_factors(lib, r, kmax):
    """n = q r^k with q = 2 .. 16 not a power of two: the q-point pass, then
    one tensor-core pass of k stages (k up to one warpgroup pass)."""
    import ctypes
    st = (ctypes.c_int32 * 3)()
    for q in (3, 5, 6, 7, 9, 10, 11, 12, 13, 14, 15):
        for k in range(1, kmax + 1):
            assert lib.tcu_dft_plan_passes(q * r ** k, r, st) == 2, (q, k)
            assert list(st)[:2] == [1, k]
        assert lib.tcu_dft_plan_passes(q * r ** (kmax + 1), r, st) == 0
    assert lib.tcu_dft_plan_passes(17 * r, r, st) == 0


def test_python_plan_raises(lib):
    import paper_1908_06649_gb300 as pkg
    with pytest.raises(pkg.TcuDftError) as e:
        pkg.Plan(17 * 16, 1, 16)
    assert e.value.status == pkg.ERR_UNSUPPORTED


@pytest.mark.parametrize("args,status", [
    ((0, 1, 16, 3, -1), 1),            # n < 1
    ((256, 0, 16, 3, -1), 1),          # batch < 1
    ((256, 1, 16, 2, -1), 1),          # precision
    ((256, 1, 16, 3, 0), 1),           # direction
    ((256, 1, 12, 3, -1), 2),          # radix
    ((48, 1, 16, 3, -1), 2),           # not a power of the radix
    ((16 ** 5, 1, 16, 3, -1), 6),      # three passes
    ((8 ** 7, 1, 8, 3, -1), 6),
    ((32 ** 4, 1, 32, 3, -1), 6),      # n beyond the fixed twiddle table
    ((65536, 65, 16, 3, -1), 6),       # batch*n beyond the fixed intermediate
    ((1, 1, 16, 3, -1), 2),            # n = 1 = r^0: k >= 1 is required
])
def test_noalloc_rejects_before_cuda(lib, args, status):
    import ctypes
    n, batch, r, prec, d = args
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: rejected first
    assert lib.tcu_dft_exec_noalloc(n, batch, r, prec, fake, fake, d, None) == status


@pytest.mark.parametrize("a,b", [
    ((1 << 20) + 8, 1 << 24),          # input not 16-byte aligned
    (1 << 20, (1 << 24) + 4),          # output not 16-byte aligned
    (1 << 20, (1 << 20) + 16),         # partial overlap of in and out
])
def test_noalloc_rejects_buffers_before_cuda(lib, a, b):
    import ctypes
    # never dereferenced: the pointers are rejected before any CUDA call
    assert lib.tcu_dft_exec_noalloc(256, 4, 16, 3, ctypes.c_void_p(a), ctypes.c_void_p(b),
                                    -1, None) == 1


def test_noalloc_null_buffers(lib):
    assert lib.tcu_dft_exec_noalloc(256, 1, 16, 3, None, None, -1, None) == 1
    assert b"fixed memory" in lib.tcu_dft_strerror(6)


@pytest.mark.parametrize("args,status", [
    ((0, 256, 1, 16, 3), 1),        # n1 < 1
    ((16, 256, 0, 16, 3), 1),       # batch < 1
    ((16, 256, 1, 16, 2), 1),       # precision
    ((16 ** 7, 16, 1, 16, 3), 2),   # an axis beyond the 1-D plans (three passes)
    ((48, 256, 1, 16, 3), 2),       # not a power of the radix
    ((16, 256, 1, 12, 3), 2),       # radix
])
def test_dft2_plan_rejects_before_cuda(lib, args, status):
    assert not lib.tcu_dft2_plan(*args)
    assert lib.tcu_dft_last_error() == status


@pytest.mark.parametrize("args,status", [
    ((0, 4, 8, 3), 1),              # side
    ((64, 0, 8, 3), 1),             # steps
    ((1024, 3000, 8, 3), 2),        # 3k beyond the largest tile (8192^2 points)
    ((64, 4, 12, 3), 2),            # radix
])
def test_stencil_plan_rejects_before_cuda(lib, args, status):
    assert not lib.tcu_stencil_plan(*args)
    assert lib.tcu_dft_last_error() == status


def test_stencil_tiling_choice(lib):
    """tcu_stencil_tiles: the smallest tile side N = r^s with N >= 3k and
    N^2 >= 128 r, at most 2^26 points a tile (one pass per axis where that
    holds them, the general 2-D path above), blocks of B = N - 2k, ceil(side /
    B)^2 tiles -- checked against the rule evaluated here."""
    import paper_1908_06649_gb300 as pkg
    for side, k, r in [(4096, 16, 8), (4096, 16, 16), (4096, 16, 32), (64, 4, 8),
                       (2000, 16, 8), (300, 16, 16), (120, 20, 8), (1, 1, 16),
                       (5000, 85, 16), (777, 3, 32), (100, 30, 8), (300, 128, 16),
                       (5000, 200, 8), (2000, 400, 32), (100, 3000, 16)]:
        Ns = [r ** s for s in range(1, 9)
              if r ** s >= 3 * k and r ** (2 * s) >= 128 * r and r ** (2 * s) <= 1 << 26]
        got = pkg.stencil_tiles(side, k, r)
        if not Ns:
            assert got == (0, 0, 0)
            continue
        N = Ns[0]
        B = N - 2 * k
        assert got == ((-(-side // B)) ** 2, N, B), (side, k, r, got)
    assert pkg.stencil_tiles(4096, 16, 8) == (16384, 64, 32)
    assert pkg.stencil_tiles(4096, 16, 16) == (361, 256, 224)
    assert pkg.stencil_tiles(64, 4, 12)[0] == 0
    assert lib.tcu_stencil_tiles(0, 4, 8, None, None) == 0


def test_grid_null_handling(lib):
    import paper_1908_06649_gb300 as pkg
    assert lib.tcu_dft2_destroy(None) == pkg.OK
    assert lib.tcu_stencil_destroy(None) == pkg.OK
    assert lib.tcu_dft2_exec(None, None, None, -1, None) == pkg.ERR_INVALID
    assert lib.tcu_conv2_exec(None, None, None, None, None) == pkg.ERR_INVALID
    assert lib.tcu_stencil_exec(None, None, None, None, None) == pkg.ERR_INVALID
    assert lib.tcu_dft2_check(None, None) == pkg.ERR_INVALID


@pytest.mark.parametrize("n,r,stages", [
    (16, 16, [1]), (256, 16, [2]), (4096, 16, [3]), (65536, 16, [2, 2]),
    (16 ** 5, 16, [1, 2, 2]), (16 ** 6, 16, [2, 2, 2]), (16 ** 7, 16, []),
    (8, 8, [1]), (512, 8, [3]), (8 ** 4, 8, [2, 2]), (8 ** 5, 8, [2, 3]), (8 ** 6, 8, [3, 3]),
    (8 ** 7, 8, [2, 2, 3]), (8 ** 8, 8, [2, 3, 3]), (8 ** 9, 8, [3, 3, 3]), (8 ** 10, 8, []),
    (32 ** 2, 32, [2]), (32 ** 3, 32, [1, 2]), (32 ** 4, 32, [2, 2]), (32 ** 5, 32, [1, 2, 2]),
    (32 ** 6, 32, [2, 2, 2]), (32 ** 7, 32, []),
    # mixed final radix n = q r^k: the q-point pass first
    (2 * 256, 16, [1, 2]), (8 * 4096, 16, [1, 1, 2]), (4 * 65536, 16, [1, 2, 2]),
    (2 * 64, 8, [1, 2]), (4 * 512, 8, [1, 3]), (2 * 4096, 8, [1, 2, 2]),
    (16 * 1024, 32, [1, 2]), (2 * 32 ** 3, 32, [1, 1, 2]),
    (2 * 16, 16, []), (3 * 256, 16, [1, 2]), (3 * 16 ** 3, 16, []), (2 * 16 ** 5, 16, []),
    (0, 16, [])])
def test_plan_grouping(n, r, stages):
    # the documented grouping, computed on the host without a GPU
    import paper_1908_06649_gb300 as pkg
    pkg.lib()
    assert pkg.plan_passes(n, r) == stages
