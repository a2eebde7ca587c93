"""fp64 CPU oracle for the batched complex DFT -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The GPU library never does, and this
package never imports the GPU library: the two share no code.

What it computes (arXiv 1908.06649, Sec. 4.5): y = x^T W with the symmetric
Fourier matrix W[r][c] = exp(-(2 pi i / n) r c), i.e. the unscaled forward DFT
y_k = sum_j x_j exp(-2 pi i j k / n).  The inverse (not defined in the paper)
is taken as the conjugate exponent with a 1/n factor, the numpy/torch
"backward" convention.

Two independent routes, both written in ``oracle.c``:
  * ``dft_direct``  -- the definition, O(n^2), angle index reduced mod n;
  * ``fft_radix2``  -- recursive radix-2 decimation in time, fp64 twiddles
    from cos/sin directly (no recurrence).
``dft`` picks the direct route for n <= 4096 and the FFT above that.

Parity pins for every function here live in ``tests/test_oracle.py``; no
function is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so with gcc (plain -O2, no -march)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC,
           "-lm", "-lpthread"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            dp = ctypes.POINTER(ctypes.c_double)
            for name in ("oracle_dft_direct", "oracle_fft_radix2"):
                f = getattr(lib, name)
                f.argtypes = [dp, dp, ctypes.c_int64, ctypes.c_int64,
                              ctypes.c_int, ctypes.c_double, ctypes.c_int]
                f.restype = ctypes.c_int
            lib.oracle_rel_l2.argtypes = [ctypes.POINTER(ctypes.c_float), dp,
                                          ctypes.c_int64, ctypes.c_int64, dp]
            lib.oracle_rel_l2.restype = None
            _lib = lib
    return _lib


def _as_c128(x, n):
    x = np.ascontiguousarray(np.asarray(x), dtype=np.complex128)
    if x.ndim == 1:
        x = x.reshape(1, -1)
    if x.shape[-1] != n:
        raise ValueError("last axis must have length n")
    return x.reshape(-1, n)


def _run(fname, x, sign, scale, threads):
    x = np.asarray(x)
    n = x.shape[-1]
    shape = x.shape
    xb = _as_c128(x, n)
    y = np.empty_like(xb)
    lib = _load()
    dp = ctypes.POINTER(ctypes.c_double)
    used = getattr(lib, fname)(xb.ctypes.data_as(dp), y.ctypes.data_as(dp),
                               n, xb.shape[0], sign, float(scale),
                               int(threads))
    if used < 0:
        raise ValueError("%s rejected n=%d batch=%d" % (fname, n, xb.shape[0]))
    return y.reshape(shape), used


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


def dft_direct(x, sign: int = -1, scale: float = 1.0, threads: int = 1):
    """Direct DFT along the last axis (Sec. 4.5 definition), fp64."""
    return _run("oracle_dft_direct", x, sign, scale, threads)[0]


def fft_radix2(x, sign: int = -1, scale: float = 1.0, threads: int = 1):
    """Recursive radix-2 FFT along the last axis (power-of-two n), fp64."""
    return _run("oracle_fft_radix2", x, sign, scale, threads)[0]


def fft_radix2_timed(x, sign: int = -1, scale: float = 1.0, threads: int = 1):
    """Same as fft_radix2, also returning the number of threads it used."""
    return _run("oracle_fft_radix2", x, sign, scale, threads)


def dft(x, inverse: bool = False, threads: int = 1):
    """Forward (sign -1, unscaled) or inverse (sign +1, 1/n) DFT, fp64."""
    n = np.asarray(x).shape[-1]
    sign, scale = (1, 1.0 / n) if inverse else (-1, 1.0)
    if n <= 4096 or (n & (n - 1)) != 0:
        return dft_direct(x, sign, scale, threads)
    return fft_radix2(x, sign, scale, threads)


def dft_entries(x, ks, inverse: bool = False):
    """Selected outputs y_k of the transforms in ``x`` (shape (B, n)), each
    straight from the definition: y_k = sum_j x_j w^{(j k) mod n}.  Used to
    check full-size GPU results at sampled positions."""
    x = np.asarray(x, dtype=np.complex128)
    n = x.shape[-1]
    ks = np.asarray(ks, dtype=np.int64)
    j = np.arange(n, dtype=np.int64)
    sign = 1.0 if inverse else -1.0
    out = np.empty(x.shape[:-1] + ks.shape, dtype=np.complex128)
    for idx, k in enumerate(ks.reshape(-1)):
        m = (j * k) % n
        w = np.exp(sign * 2j * np.pi * m / n)
        out[..., idx] = x @ w
    if inverse:
        out /= n
    return out


def rel_l2(y_gpu, y_ref):
    """Per-transform relative L2 error ||y_gpu - y_ref|| / ||y_ref|| (fp64)."""
    a = np.ascontiguousarray(np.asarray(y_gpu), dtype=np.complex64)
    b = np.ascontiguousarray(np.asarray(y_ref), dtype=np.complex128)
    n = a.shape[-1]
    a = a.reshape(-1, n)
    b = b.reshape(-1, n)
    if a.shape != b.shape:
        raise ValueError("shape mismatch")
    out = np.empty(a.shape[0], dtype=np.float64)
    lib = _load()
    lib.oracle_rel_l2(a.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                      b.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                      n, a.shape[0],
                      out.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    return out
