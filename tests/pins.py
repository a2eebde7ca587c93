"""Pins for a DFT implementation that do not come from the implementation.

Each check states a fact fixed by the mathematics of the DFT as the paper
defines it (arXiv 1908.06649, Sec. 4.5: y = x^T W, W[r][c] =
exp(-(2 pi i/n) r c)), or by hand-derived values.  ``failures(fwd, inv)``
runs them all against a forward and an inverse transform (callables taking a
(B, n) complex array) and returns the names of the checks that failed, so the
same list can be run on the oracle (expect none) and on deliberately broken
copies of it (expect some).
"""
from __future__ import annotations

import json
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "dft_small.json")


def golden_cases():
    with open(GOLDEN) as f:
        d = json.load(f)
    out = []
    for c in d["cases"]:
        x = np.array([complex(*v) for v in c["x"]])
        y = np.array([complex(*v) for v in c["y"]])
        out.append((c["name"], c["n"], x, y))
    return out


def _rel(a, b):
    a = np.asarray(a, dtype=np.complex128)
    b = np.asarray(b, dtype=np.complex128)
    den = np.linalg.norm(b)
    return np.linalg.norm(a - b) / (den if den > 0 else 1.0)


def _rng(seed):
    return np.random.default_rng(seed)


def failures(fwd, inv, sizes=(2, 4, 8, 16, 32, 64), tol=1e-12,
             pow2_only=False):
    bad = []

    def check(name, ok):
        if not ok:
            bad.append(name)

    # 1. hand-derived golden vectors
    for name, n, x, y in golden_cases():
        if pow2_only and (n & (n - 1)):
            continue
        check("golden:" + name, _rel(fwd(x[None])[0], y) < tol)

    for n in sizes:
        j = np.arange(n)
        k = np.arange(n)
        w = np.exp(-2j * np.pi / n)
        # 2. DFT(delta_0) = all ones
        d0 = np.zeros((1, n), complex)
        d0[0, 0] = 1
        check("delta0:%d" % n, _rel(fwd(d0)[0], np.ones(n)) < tol)
        # 3. DFT(1) = n * delta_0
        one = np.ones((1, n), complex)
        e0 = np.zeros(n, complex)
        e0[0] = n
        check("const:%d" % n, _rel(fwd(one)[0], e0) < tol)
        # 4. a pure tone exp(+2 pi i f j / n) maps to n * delta_f (sign pin)
        for f in sorted({1, n // 3, n - 1}):
            x = np.exp(2j * np.pi * ((f * j) % n) / n)[None]
            ef = np.zeros(n, complex)
            ef[f] = n
            check("tone:%d:%d" % (n, f), _rel(fwd(x)[0], ef) < tol)
        # 5. delta_s -> w^{k s} (time-shift / index pin)
        for s in sorted({1, n // 2 + (n > 2), n - 1}):
            x = np.zeros((1, n), complex)
            x[0, s % n] = 1
            check("shift-delta:%d:%d" % (n, s),
                  _rel(fwd(x)[0], w ** ((k * (s % n)) % n)) < tol)
        # 6. ramp x_j = j: y_0 = n(n-1)/2, y_k = -n / (1 - w^k) for k != 0
        #    (arithmetic-geometric series with w^n = 1)
        ramp = j.astype(complex)[None]
        yk = np.empty(n, complex)
        yk[0] = n * (n - 1) / 2
        yk[1:] = -n / (1 - w ** k[1:])
        check("ramp:%d" % n, _rel(fwd(ramp)[0], yk) < tol)
        # random inputs for the invariants
        r = _rng(n)
        x = r.standard_normal((3, n)) + 1j * r.standard_normal((3, n))
        x2 = r.standard_normal((3, n)) + 1j * r.standard_normal((3, n))
        y = fwd(x)
        # 7. Parseval: sum |y|^2 = n sum |x|^2
        lhs = np.sum(np.abs(y) ** 2, axis=1)
        rhs = n * np.sum(np.abs(x) ** 2, axis=1)
        check("parseval:%d" % n, np.max(np.abs(lhs - rhs) / rhs) < tol * 10)
        # 8. linearity
        a, b = 0.7 - 0.2j, -1.3 + 0.5j
        check("linear:%d" % n,
              _rel(fwd(a * x + b * x2), a * y + b * fwd(x2)) < tol * 10)
        # 9. inverse round trip
        check("roundtrip:%d" % n, _rel(inv(y), x) < tol * 10)
        # 10. real input -> Hermitian output y_{n-k} = conj(y_k)
        xr = r.standard_normal((1, n)).astype(complex)
        yr = fwd(xr)[0]
        check("hermitian:%d" % n,
              _rel(yr[(-k) % n], np.conj(yr)) < tol * 10)
        # 11. circular shift by s multiplies y_k by w^{k s}
        s = max(1, n // 4 + 1) % n
        check("shift:%d" % n,
              _rel(fwd(np.roll(x, s, axis=1)), y * (w ** ((k * s) % n))[None])
              < tol * 10)
    return bad
