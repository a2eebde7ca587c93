"""The oracle, pinned against facts that do not come from the oracle itself.

CPU only.  Covers both oracle routes (direct definition and radix-2 FFT) and
shows that the pins catch planted mistakes: each mutant below is a textual
edit of oracle.c (a dropped term, a flipped sign, a wrong index, a swapped
operand), compiled on the CPU, which must fail at least one pin.
"""
import ctypes
import os
import subprocess

import numpy as np
import pytest

import oracle
import pins



def _fwd(route):
    f = oracle.dft_direct if route == "direct" else oracle.fft_radix2
    return lambda x: f(x, sign=-1)


def _inv(route):
    f = oracle.dft_direct if route == "direct" else oracle.fft_radix2
    return lambda x: f(x, sign=1, scale=1.0 / np.asarray(x).shape[-1])


@pytest.mark.parametrize("route", ["direct", "fft"])
def test_pins_hold(route):
    bad = pins.failures(_fwd(route), _inv(route),
                        pow2_only=(route == "fft"))
    assert bad == []


def test_direct_non_power_of_two():
    # the definition does not need n to be a power of two
    bad = pins.failures(_fwd("direct"), _inv("direct"), sizes=(3, 5, 6, 12))
    assert bad == []


@pytest.mark.parametrize("n", [1, 2, 8, 64, 1024, 4096])
def test_routes_agree(n):
    r = np.random.default_rng(100 + n)
    x = r.standard_normal((4, n)) + 1j * r.standard_normal((4, n))
    a = oracle.dft_direct(x)
    b = oracle.fft_radix2(x)
    den = np.linalg.norm(a, axis=1)
    assert np.max(np.linalg.norm(a - b, axis=1) / den) < 1e-12


@pytest.mark.parametrize("n", [16, 256, 4096, 65536])
def test_library_special_case(n):
    # numpy's pocketfft is an independent library implementation of the same
    # definition (special case that reduces to a library routine)
    r = np.random.default_rng(7 + n)
    x = r.standard_normal((2, n)) + 1j * r.standard_normal((2, n))
    y = oracle.dft(x)
    ref = np.fft.fft(x, axis=1)
    assert np.max(np.linalg.norm(y - ref, axis=1)
                  / np.linalg.norm(ref, axis=1)) < 1e-12
    xi = oracle.dft(y, inverse=True)
    assert np.max(np.abs(xi - x)) < 1e-10


def test_large_fft_tone_and_parseval():
    n = 1 << 20
    j = np.arange(n)
    f = 123457
    x = np.exp(2j * np.pi * ((f * j) % n) / n)[None]
    y = oracle.fft_radix2(x)[0]
    assert abs(y[f] - n) < 1e-6 * n
    y[f] = 0
    assert np.max(np.abs(y)) < 1e-6 * n
    r = np.random.default_rng(5)
    x = r.standard_normal((1, n)) + 1j * r.standard_normal((1, n))
    y = oracle.fft_radix2(x)
    assert abs(np.sum(np.abs(y) ** 2) / (n * np.sum(np.abs(x) ** 2)) - 1) < 1e-12


def test_dft_entries_matches_full():
    r = np.random.default_rng(11)
    n = 512
    x = r.standard_normal((3, n)) + 1j * r.standard_normal((3, n))
    ks = np.array([0, 1, 17, 255, 256, 511])
    full = oracle.dft(x)
    assert np.max(np.abs(oracle.dft_entries(x, ks) - full[:, ks])) < 1e-9
    fulli = oracle.dft(x, inverse=True)
    assert np.max(np.abs(oracle.dft_entries(x, ks, inverse=True)
                         - fulli[:, ks])) < 1e-12


def test_threads_do_not_change_results():
    r = np.random.default_rng(3)
    x = r.standard_normal((7, 1024)) + 1j * r.standard_normal((7, 1024))
    a = oracle.fft_radix2(x, threads=1)
    b, used = oracle.fft_radix2_timed(x, threads=4)
    assert used >= 1
    assert np.array_equal(a, b)


def test_rel_l2():
    b = np.array([[3 + 4j, 0]], dtype=np.complex128)
    a = np.array([[3 + 4j, 1]], dtype=np.complex64)
    assert abs(oracle.rel_l2(a, b)[0] - 0.2) < 1e-15


def test_bad_arguments():
    with pytest.raises(ValueError):
        oracle.fft_radix2(np.ones((1, 12), complex))  # not a power of two


# ---------------------------------------------------------------- mutants
SRC = os.path.join(os.path.dirname(oracle.__file__), "oracle.c")

MUTANTS = {
    # a term dropped from the complex product in the definition
    "direct_drops_im_term": ("acc_re += xr * c - xi * s;", "acc_re += xr * c;"),
    # the exponent sign flipped in the definition
    "direct_sign_flip": ("double ang = (double)sign * 2.0 * M_PI * (double)m",
                         "double ang = -(double)sign * 2.0 * M_PI * (double)m"),
    # the angle index not reduced correctly (j*k+1)
    "direct_wrong_index": ("int64_t m = (j * k) % n;",
                           "int64_t m = (j * k + 1) % n;"),
    # the radix-2 twiddle with a wrong index (k+1)
    "fft_twiddle_index": ("(double)k / (double)m;", "(double)(k + 1) / (double)m;"),
    # the radix-2 twiddle with the wrong sign
    "fft_twiddle_sign": ("double ang = (double)sign * 2.0 * M_PI * (double)k",
                         "double ang = -(double)sign * 2.0 * M_PI * (double)k"),
    # even and odd halves swapped (transposed operands of the butterfly)
    "fft_swapped_halves": ("fft_rec(x, 2 * stride, y, h, sign);",
                           "fft_rec(x + 2 * stride, 2 * stride, y, h, sign);"),
    # the butterfly's difference output dropped the twiddled term's sign
    "fft_butterfly_sign": ("y[2 * (k + h)] = er - tr;", "y[2 * (k + h)] = er + tr;"),
}


def _build_mutant(tmp_path, name, old, new):
    src = open(SRC).read()
    assert src.count(old) == 1, (name, old)
    path = tmp_path / ("%s.c" % name)
    path.write_text(src.replace(old, new))
    so = tmp_path / ("lib%s.so" % name)
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o",
                    str(so), str(path), "-lm", "-lpthread"], check=True)
    lib = ctypes.CDLL(str(so))
    dp = ctypes.POINTER(ctypes.c_double)
    fns = {}
    for fn in ("oracle_dft_direct", "oracle_fft_radix2"):
        f = getattr(lib, fn)
        f.argtypes = [dp, dp, ctypes.c_int64, ctypes.c_int64, ctypes.c_int,
                      ctypes.c_double, ctypes.c_int]
        f.restype = ctypes.c_int
        fns[fn] = f

    def call(fn, x, sign, scale):
        x = np.ascontiguousarray(np.asarray(x, dtype=np.complex128))
        y = np.empty_like(x)
        rc = fns[fn](x.ctypes.data_as(dp), y.ctypes.data_as(dp), x.shape[-1],
                     x.shape[0], sign, scale, 1)
        assert rc >= 0
        return y

    return call


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_pins_catch_planted_mistake(tmp_path, name):
    old, new = MUTANTS[name]
    call = _build_mutant(tmp_path, name, old, new)
    fn = "oracle_dft_direct" if name.startswith("direct") else "oracle_fft_radix2"
    fwd = lambda x: call(fn, x, -1, 1.0)
    inv = lambda x: call(fn, x, 1, 1.0 / np.asarray(x).shape[-1])
    bad = pins.failures(fwd, inv, pow2_only=(fn == "oracle_fft_radix2"))
    assert bad, "planted mistake %s passed every pin" % name
