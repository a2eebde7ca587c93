"""fp64 CPU oracle for the 2-D transforms and the stencil computations of
arXiv 1908.06649, Sec. 4.6 -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module; the GPU library never does, and this
module never imports it.

Every function is the plain definition written out (numpy, float64), no
blocking or reordering beyond what the definition states:

  * ``dft2``            -- 2-D DFT: a 1-D DFT (the Sec. 4.5 oracle) of every
                           row, then of every column (Sec. 4.6 recalls that a
                           2-D DFT is exactly that);
  * ``conv2_circular``  -- circular 2-D convolution by its defining double
                           sum (the operation Lemma 1 reduces stencils to);
  * ``stencil_direct``  -- a linear (n, k)-stencil by k sweeps of
                           A_t[i,j] = sum_{a,b in {-1,0,1}} w[a,b] A_{t-1}[i+a,j+b];
  * ``stencil_weights`` -- the weight matrix W of Lemma 2: the coefficients
                           of P(x,y)^k, P(x,y) = sum w[a,b] x^a y^b, by k
                           direct polynomial products.

Boundary reading (the paper leaves cells outside the grid undefined, but
its unrolled form A_k = sum W[k+a, k+b] A[i+a, j+b] is exact only on the
free plane): the grid is zero outside at time 0 and the sweeps act on the
whole plane, so values may leave the grid and come back.  ``stencil_direct``
realises that by sweeping a grid padded by k zero cells on every side.

Parity pins for every function here live in ``tests/test_oracle_grid.py``.
"""
from __future__ import annotations

import numpy as np

from . import dft


def dft2(x, inverse: bool = False, threads: int = 1):
    """2-D DFT of the last two axes (..., n1, n2): rows (axis -1) then
    columns (axis -2), each by the fp64 1-D oracle (``threads`` splits the
    rows of each step between threads; the arithmetic is the same).  Forward
    unscaled; the inverse uses the conjugate exponent and 1/(n1 n2)."""
    x = np.asarray(x, dtype=np.complex128)
    n1, n2 = x.shape[-2], x.shape[-1]
    rows = dft(x.reshape(-1, n2), inverse=inverse, threads=threads).reshape(x.shape)
    cols = np.swapaxes(rows, -1, -2)
    out = dft(np.ascontiguousarray(cols).reshape(-1, n1), inverse=inverse,
              threads=threads)
    return np.swapaxes(out.reshape(cols.shape), -1, -2)


def conv2_circular(x, w):
    """(x (*) w)[i, j] = sum_{a, b} x[(i - a) mod n1, (j - b) mod n2] w[a, b]
    for every array of the batch x (..., n1, n2) with one w (n1, n2).  O(n^4):
    small sizes only."""
    x = np.asarray(x, dtype=np.complex128)
    w = np.asarray(w, dtype=np.complex128)
    n1, n2 = w.shape
    out = np.zeros(np.broadcast_shapes(x.shape, w.shape), dtype=np.complex128)
    for a in range(n1):
        for b in range(n2):
            if w[a, b] != 0:
                out += w[a, b] * np.roll(np.roll(x, a, axis=-2), b, axis=-1)
    return out


def stencil_sweep(A, w3):
    """One sweep A'[i,j] = sum_{a,b in {-1,0,1}} w3[a+1, b+1] A[i+a, j+b]
    over the array A, cells beyond its edge read as 0."""
    A = np.asarray(A, dtype=np.float64)
    w3 = np.asarray(w3, dtype=np.float64)
    P = np.pad(A, 1)
    out = np.zeros_like(A)
    for a in (-1, 0, 1):
        for b in (-1, 0, 1):
            out += w3[a + 1, b + 1] * P[1 + a:1 + a + A.shape[0], 1 + b:1 + b + A.shape[1]]
    return out


def stencil_direct(A, w3, k: int):
    """A_k of the linear (n, k)-stencil on the free plane: k sweeps of a
    grid padded by k zero cells on each side, cropped back."""
    A = np.asarray(A, dtype=np.float64)
    G = np.pad(A, k)
    for _ in range(k):
        G = stencil_sweep(G, w3)
    return G[k:k + A.shape[0], k:k + A.shape[1]]


def poly2_mul(p, q):
    """Product of two bivariate polynomials given as centred coefficient
    arrays (odd sides, entry [a + ha, b + hb] is the coefficient of
    x^a y^b): the full 2-D linear convolution by its double sum."""
    p = np.asarray(p, dtype=np.float64)
    q = np.asarray(q, dtype=np.float64)
    out = np.zeros((p.shape[0] + q.shape[0] - 1, p.shape[1] + q.shape[1] - 1))
    for a in range(p.shape[0]):
        for b in range(p.shape[1]):
            if p[a, b] != 0:
                out[a:a + q.shape[0], b:b + q.shape[1]] += p[a, b] * q
    return out


def stencil_weights(w3, k: int):
    """The (2k+1) x (2k+1) weight matrix of Lemma 2: W[k + a, k + b] is the
    coefficient of x^a y^b in P(x, y)^k, P(x, y) = sum w3[a+1, b+1] x^a y^b,
    computed as F_0 = 1, F_u = F_{u-1} P."""
    F = np.ones((1, 1))
    for _ in range(k):
        F = poly2_mul(F, w3)
    return F
