"""Pins of the 2-D / stencil oracle (oracle/grid.py) against facts that do
not come from it: brute-force double sums, closed forms, the convolution
theorem through numpy's independent FFT, and the stencil identities of
Sec. 4.6 (the unrolled sweep equals the weight matrix W of Lemma 2)."""
import numpy as np
import pytest

from oracle import grid


def _rng(s):
    return np.random.default_rng(s)


def _brute_dft2(x, sign=-1):
    n1, n2 = x.shape
    i = np.arange(n1)[:, None]
    j = np.arange(n2)[None, :]
    out = np.zeros((n1, n2), np.complex128)
    for k1 in range(n1):
        for k2 in range(n2):
            out[k1, k2] = np.sum(x * np.exp(sign * 2j * np.pi * (((i * k1) % n1) / n1 + ((j * k2) % n2) / n2)))
    return out


@pytest.mark.parametrize("n1,n2", [(2, 4), (4, 4), (8, 4), (3, 5)])
def test_dft2_brute_force(n1, n2):
    r = _rng(n1 * 10 + n2)
    x = r.standard_normal((n1, n2)) + 1j * r.standard_normal((n1, n2))
    y = grid.dft2(x)
    assert np.max(np.abs(y - _brute_dft2(x))) < 1e-11 * n1 * n2
    back = grid.dft2(y, inverse=True)
    assert np.max(np.abs(back - x)) < 1e-12


def test_dft2_closed_forms():
    n1, n2 = 16, 8
    d = np.zeros((n1, n2), complex)
    d[0, 0] = 1
    assert np.allclose(grid.dft2(d), 1)
    one = np.ones((n1, n2), complex)
    e = np.zeros((n1, n2), complex)
    e[0, 0] = n1 * n2
    assert np.allclose(grid.dft2(one), e)
    f1, f2 = 3, 5
    i = np.arange(n1)[:, None]
    j = np.arange(n2)[None, :]
    tone = np.exp(2j * np.pi * (f1 * i / n1 + f2 * j / n2))
    e = np.zeros((n1, n2), complex)
    e[f1, f2] = n1 * n2
    assert np.allclose(grid.dft2(tone), e, atol=1e-9)


def test_dft2_matches_numpy_fft2():
    # a library special case (pocketfft), not the oracle's own 1-D routine
    r = _rng(3)
    x = r.standard_normal((2, 32, 64)) + 1j * r.standard_normal((2, 32, 64))
    assert np.max(np.abs(grid.dft2(x) - np.fft.fft2(x))) < 1e-9
    assert np.max(np.abs(grid.dft2(x, inverse=True) - np.fft.ifft2(x))) < 1e-12


def test_conv2_identities():
    r = _rng(4)
    x = r.standard_normal((3, 8, 4)) + 1j * r.standard_normal((3, 8, 4))
    d = np.zeros((8, 4))
    d[0, 0] = 1
    assert np.allclose(grid.conv2_circular(x, d), x)          # delta: identity
    s = np.zeros((8, 4))
    s[2, 1] = 1
    assert np.allclose(grid.conv2_circular(x, s), np.roll(np.roll(x, 2, -2), 1, -1))
    w = r.standard_normal((8, 4))
    # convolution theorem through numpy's FFT
    ref = np.fft.ifft2(np.fft.fft2(x) * np.fft.fft2(w))
    assert np.max(np.abs(grid.conv2_circular(x, w) - ref)) < 1e-12
    # commutative in the two operands
    y = r.standard_normal((8, 4))
    assert np.allclose(grid.conv2_circular(y, w), grid.conv2_circular(w, y))


HEAT = np.array([[0.0, 0.1, 0.0], [0.15, 0.5, 0.15], [0.0, 0.1, 0.0]])


def test_stencil_one_sweep_by_hand():
    A = np.zeros((3, 3))
    A[1, 1] = 2.0
    A[0, 1] = 1.0
    out = grid.stencil_direct(A, HEAT, 1)
    # centre: 0.5*2 + 0.1*A[0,1] (a = -1 reads the row above) = 1.1
    assert abs(out[1, 1] - 1.1) < 1e-15
    # (0,1): 0.5*1 + w[+1][0]*A[1,1] = 0.5 + 0.1*2 = 0.7
    assert abs(out[0, 1] - 0.7) < 1e-15
    # (2,1): w[-1][0]*A[1,1] = 0.2
    assert abs(out[2, 1] - 0.2) < 1e-15


@pytest.mark.parametrize("k", [1, 2, 5])
def test_weights_are_the_impulse_response(k):
    # the unrolled stencil of a single 1 is W itself (an independent route:
    # sweeps vs polynomial products), read with the paper's indexing
    # A_k[i,j] = sum W[k+a, k+b] A[i+a, j+b]: a 1 at (c, c) lands on A_k[c-a, c-b]
    r = _rng(k)
    w3 = r.standard_normal((3, 3))
    W = grid.stencil_weights(w3, k)
    assert W.shape == (2 * k + 1, 2 * k + 1)
    n = 2 * k + 1
    A = np.zeros((n, n))
    A[k, k] = 1.0
    Ak = grid.stencil_direct(A, w3, k)
    assert np.max(np.abs(Ak - W[::-1, ::-1])) < 1e-12


def test_weights_closed_forms():
    # sum of coefficients = P(1, 1)^k; separable stencils give outer
    # products of binomial rows
    # only the a = 0 row: P = y^-1 + 2 + y = (y^-1/2 + y^1/2)^2
    w3 = np.array([[0.0, 0.0, 0.0], [1.0, 2.0, 1.0], [0.0, 0.0, 0.0]])
    k = 4
    W = grid.stencil_weights(w3, k)
    assert abs(W.sum() - 4.0 ** k) < 1e-9
    from math import comb
    row = np.array([comb(2 * k, i) for i in range(2 * k + 1)], float)
    assert np.allclose(W[k], row) and np.allclose(np.delete(W, k, axis=0), 0)
    r = _rng(9)
    w3 = r.standard_normal((3, 3))
    assert abs(grid.stencil_weights(w3, 3).sum() - w3.sum() ** 3) < 1e-9


def test_stencil_is_linear_and_matches_weights():
    # A_k[i,j] = sum W[k+a, k+b] A[i+a, j+b] on the free plane (Sec. 4.6)
    r = _rng(11)
    k = 3
    w3 = r.standard_normal((3, 3))
    A = r.standard_normal((10, 12))
    W = grid.stencil_weights(w3, k)
    Ak = grid.stencil_direct(A, w3, k)
    P = np.pad(A, k)
    ref = np.zeros_like(A)
    for a in range(-k, k + 1):
        for b in range(-k, k + 1):
            ref += W[k + a, k + b] * P[k + a:k + a + A.shape[0], k + b:k + b + A.shape[1]]
    assert np.max(np.abs(Ak - ref)) < 1e-12
    B = r.standard_normal((10, 12))
    assert np.allclose(grid.stencil_direct(2 * A - B, w3, k), 2 * Ak - grid.stencil_direct(B, w3, k))


def test_planted_mistakes_are_caught():
    # a wrong sweep (a dropped neighbour) or a wrong power (k-1 products)
    # must disagree with the closed forms / impulse response above
    w3 = HEAT
    k = 2
    W = grid.stencil_weights(w3, k)
    assert abs(W.sum() - w3.sum() ** k) < 1e-12
    bad = grid.stencil_weights(w3, k - 1)
    assert abs(bad.sum() - w3.sum() ** k) > 1e-3 or bad.shape != W.shape
    w_drop = w3.copy()
    w_drop[0, 1] = 0
    A = np.zeros((5, 5))
    A[2, 2] = 1
    assert np.max(np.abs(grid.stencil_direct(A, w_drop, k) - W[::-1, ::-1])) > 1e-3
