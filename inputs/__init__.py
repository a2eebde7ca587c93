"""Seeded synthetic inputs for the batched DFT (shared by tests, bench, oracle).

This module holds no DFT arithmetic: it only draws numbers.  Both the GPU
tests and the oracle consume its output, so neither side generates its own
inputs.

Generator: SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom
number generators", OOPSLA 2014), used as a counter-based stream: draw i of
stream ``seed`` is mix(seed + (i + 1) * 0x9E3779B97F4A7C15) with the
published finaliser mix(z) = z ^ (z >> 31) after the two multiply-xorshift
rounds (constants 0xBF58476D1CE4E5B9 and 0x94D049BB133111EB).

Draw -> number:
  * uniform [0, 1):  u = (draw >> 40) * 2^-24   (24 bits, exact in fp32)
  * uniform [-1, 1]: 2u - 1                     (exact in fp32)
  * N(0, 1) pair:    Box-Muller in fp64 on two successive uniforms,
                     u1 -> 1 - u1 in (0, 1];  (re, im) = r (cos t, sin t)
Order: transform-major, element-major, real part then imaginary part (draws
2*(b*n + j) and 2*(b*n + j) + 1 feed element j of transform b).
All values are rounded to fp32 (complex64); the oracle widens those same
fp32 values to fp64.

Workloads (seeded, synthetic; no dataset exists for this method):
  * ``uniform``   re, im i.i.d. U[-1, 1]
  * ``normal``    re, im i.i.d. N(0, 1)
  * ``tones``     per transform, 3 distinct integer frequencies f drawn
                  uniformly from [0, n) on stream seed ^ TONE_SALT (8 draws per
                  transform, first 3 distinct kept), x_j = sum_f
                  exp(+2 pi i f j / n), plus N(0, sigma^2) noise on re and im
                  (sigma = 0.01) from stream ``seed``.
"""
from __future__ import annotations

import numpy as np

GOLDEN = np.uint64(0x9E3779B97F4A7C15)
M1 = np.uint64(0xBF58476D1CE4E5B9)
M2 = np.uint64(0x94D049BB133111EB)
TONE_SALT = 0x70E5_5EED_0000_0005
CHUNK = 1 << 18  # points per generator chunk (chunks run on threads)


def splitmix64(seed: int, start: int, count: int) -> np.ndarray:
    """Draws start .. start+count-1 of the SplitMix64 stream ``seed``."""
    with np.errstate(over="ignore"):
        i = np.arange(start + 1, start + count + 1, dtype=np.uint64)
        z = np.uint64(seed & 0xFFFFFFFFFFFFFFFF) + i * GOLDEN
        z = (z ^ (z >> np.uint64(30))) * M1
        z = (z ^ (z >> np.uint64(27))) * M2
        z = z ^ (z >> np.uint64(31))
    return z


def uniform01(seed: int, start: int, count: int) -> np.ndarray:
    """u = (draw >> 40) * 2^-24 in [0, 1), as float64 (exact)."""
    d = splitmix64(seed, start, count) >> np.uint64(40)
    return d.astype(np.float64) * (1.0 / (1 << 24))


def _fill(out_flat: np.ndarray, seed: int, kind: str, first_point: int):
    """Fill complex64 points first_point .. first_point+len-1 of a stream."""
    npts = out_flat.shape[0]
    u = uniform01(seed, 2 * first_point, 2 * npts)
    u1, u2 = u[0::2], u[1::2]
    if kind == "uniform":
        out_flat.real = (2.0 * u1 - 1.0).astype(np.float32)
        out_flat.imag = (2.0 * u2 - 1.0).astype(np.float32)
    elif kind == "normal":
        r = np.sqrt(-2.0 * np.log(1.0 - u1))
        t = 2.0 * np.pi * u2
        out_flat.real = (r * np.cos(t)).astype(np.float32)
        out_flat.imag = (r * np.sin(t)).astype(np.float32)
    else:
        raise ValueError(kind)


def tone_frequencies(seed: int, n: int, batch: int, count: int = 3,
                     first: int = 0) -> np.ndarray:
    """The ``count`` distinct tone frequencies of transforms first..first+batch-1:
    8 draws per transform, the first ``count`` distinct values kept (in draw
    order); if 8 draws hold fewer, the last kept value is stepped by +1 mod n
    until enough are found (practically never happens)."""
    draws = 8
    d = splitmix64(seed ^ TONE_SALT, draws * first, draws * batch)
    cand = ((d >> np.uint64(32)) % np.uint64(n)).astype(np.int64)
    cand = cand.reshape(batch, draws)
    out = np.empty((batch, count), dtype=np.int64)
    # vectorised "first distinct" selection
    taken = np.zeros((batch, draws), dtype=bool)
    chosen = np.full((batch, count), -1, dtype=np.int64)
    rows = np.arange(batch)
    for c in range(count):
        fresh = np.ones((batch, draws), dtype=bool)
        for prev in range(c):
            fresh &= cand != chosen[:, prev:prev + 1]
        idx = np.argmax(fresh, axis=1)
        ok = fresh[rows, idx]
        chosen[:, c] = np.where(ok, cand[rows, idx], -1)
    out[:] = chosen
    bad = np.nonzero((chosen < 0).any(axis=1))[0]
    for b in bad:  # deterministic fill, as the scalar definition
        seen = []
        for c in cand[b]:
            if c not in seen:
                seen.append(int(c))
                if len(seen) == count:
                    break
        f = seen[-1]
        while len(seen) < count:
            f = (f + 1) % n
            if f not in seen:
                seen.append(f)
        out[b] = seen
    return out


def _threads() -> int:
    import os
    return max(1, min(16, os.cpu_count() or 1))


def _parallel(fn, starts):
    """fn(s) for every chunk start s; chunks are independent (disjoint output
    slices, counter-based draws), so they run on a thread pool (numpy
    releases the GIL in the array arithmetic).  Same values as in order."""
    starts = list(starts)
    if len(starts) <= 1 or _threads() == 1:
        for s in starts:
            fn(s)
        return
    from concurrent.futures import ThreadPoolExecutor
    with ThreadPoolExecutor(max_workers=_threads()) as ex:
        for _ in ex.map(fn, starts):
            pass


def make(kind: str, n: int, batch: int, seed: int, first: int = 0,
         count: int | None = None, sigma: float = 0.01) -> np.ndarray:
    """Transforms first .. first+count-1 of a workload, shape (count, n), c64."""
    if count is None:
        count = batch - first
    out = np.empty((count, n), dtype=np.complex64)
    flat = out.reshape(-1)
    base = first * n
    if kind in ("uniform", "normal"):
        def one(s):
            e = min(flat.shape[0], s + CHUNK)
            _fill(flat[s:e], seed, kind, base + s)
        _parallel(one, range(0, flat.shape[0], CHUNK))
        return out
    if kind == "tones":
        freqs = tone_frequencies(seed, n, count, first=first)
        j = np.arange(n, dtype=np.int64)
        # exp(2 pi i m / n) for every residue m, gathered below (the same
        # values as evaluating it per element)
        roots = np.exp(2j * np.pi * np.arange(n, dtype=np.int64) / n)
        step = max(1, CHUNK // n)

        def one(b0):
            b1 = min(count, b0 + step)
            nz = np.empty((b1 - b0) * n, dtype=np.complex64)
            _fill(nz, seed, "normal", base + b0 * n)
            sig = np.zeros((b1 - b0, n), dtype=np.complex128)
            for t in range(freqs.shape[1]):
                sig += roots[(freqs[b0:b1, t:t + 1] * j[None, :]) % n]
            sig += sigma * nz.reshape(b1 - b0, n).astype(np.complex128)
            out[b0:b1] = sig.astype(np.complex64)
        _parallel(one, range(0, count, step))
        return out
    raise ValueError(kind)


# The workloads of the method's evaluation: (name, n, sqrt_m, batch, kind,
# seed, directions).  All shapes are powers of sqrt_m.
WORKLOADS = {
    "n4096_b64": dict(n=4096, sqrt_m=16, batch=64, kind="uniform", seed=0,
                      dirs=("forward",)),
    "n65536_b1024": dict(n=65536, sqrt_m=16, batch=1024, kind="normal",
                         seed=1, dirs=("forward",)),
    "n32768_r8_b4096": dict(n=32768, sqrt_m=8, batch=4096, kind="normal",
                            seed=2, dirs=("forward", "inverse")),
    "n32768_r32_b4096": dict(n=32768, sqrt_m=32, batch=4096, kind="normal",
                             seed=2, dirs=("forward", "inverse")),
    "n16777216_b4": dict(n=1 << 24, sqrt_m=16, batch=4, kind="uniform",
                         seed=3, dirs=("forward",)),
    "n256_b1048576": dict(n=256, sqrt_m=16, batch=1 << 20, kind="tones",
                          seed=4, dirs=("forward",)),
}
