"""GPU parity of the 2-D rows (Sec. 4.6): 2-D DFT, batched circular 2-D
convolution, the stencil weight matrix by polynomial powering (Lemma 2) and
the stencil by batched tile convolutions (Lemma 1), through the C ABI,
against the fp64 oracle in oracle/grid.py on the same seeded inputs.

Bar: per-array relative L2 <= 1e-5 (3xTF32) / 3e-3 (TF32) for transforms
and convolutions; stencil outputs within 1e-5 of max |A_k| (3xTF32)."""
import numpy as np
import pytest

import inputs
from oracle import grid

pytestmark = pytest.mark.gpu

TOL = {3: 1e-5, 1: 3e-3}


@pytest.fixture(scope="module")
def pkg():
    import torch
    from paper_1908_06649_gb300 import _build
    _build.build()
    import paper_1908_06649_gb300 as p
    p.lib()
    assert torch.cuda.is_available()
    return p


def _rel(a, b):
    a = np.asarray(a, np.complex128).reshape(a.shape[0], -1)
    b = np.asarray(b, np.complex128).reshape(b.shape[0], -1)
    return np.linalg.norm(a - b, axis=1) / np.linalg.norm(b, axis=1)


@pytest.mark.parametrize("r,n1,n2,batch", [
    (16, 16, 256, 5), (16, 256, 16, 3), (16, 256, 256, 2),
    (8, 8, 512, 3), (8, 64, 64, 7), (8, 64, 512, 2), (8, 512, 8, 3), (8, 512, 512, 1),
    (32, 32, 1024, 2), (32, 1024, 32, 2), (32, 1024, 1024, 1)])
@pytest.mark.parametrize("prec", [3, 1])
def test_dft2(pkg, r, n1, n2, batch, prec):
    import torch
    x = inputs.make("normal", n1 * n2, batch, seed=n1 + n2).reshape(batch, n1, n2)
    plan = pkg.Plan2(n1, n2, batch, r, prec)
    xd = torch.from_numpy(x).cuda().reshape(-1)
    y = plan.forward(xd)
    back = plan.inverse(y)
    plan.check()
    yh = y.cpu().numpy().reshape(batch, n1, n2)
    ref = grid.dft2(x, threads=8)
    assert _rel(yh, ref).max() <= TOL[prec]
    bh = back.cpu().numpy().reshape(batch, n1, n2)
    assert _rel(bh, grid.dft2(yh, inverse=True, threads=8)).max() <= TOL[prec]
    plan.destroy()


# ---- the general 2-D path: axes beyond one warpgroup pass (1-D plans for
# the rows and, after a transpose, the columns), arrays below one column item,
# and the BF16 modes
@pytest.mark.parametrize("r,n1,n2,batch", [
    (16, 4096, 4096, 1), (16, 65536, 16, 2), (16, 16, 65536, 2), (16, 16, 16, 3),
    (8, 4096, 512, 1), (8, 8, 8, 5), (32, 32768, 32, 1), (32, 32, 32768, 1)])
def test_dft2_general(pkg, r, n1, n2, batch):
    import torch
    x = inputs.make("normal", n1 * n2, batch, seed=n1 + 3 * n2).reshape(batch, n1, n2)
    plan = pkg.Plan2(n1, n2, batch, r, 3)
    xd = torch.from_numpy(x).cuda().reshape(-1)
    y = plan.forward(xd)
    plan.check()
    yh = y.cpu().numpy().reshape(batch, n1, n2)
    assert _rel(yh, grid.dft2(x, threads=8)).max() <= TOL[3]
    back = plan.inverse(y)
    plan.check()
    bh = back.cpu().numpy().reshape(batch, n1, n2)
    assert _rel(bh, x).max() <= 2 * TOL[3]
    # in place
    plan.forward(xd, xd)
    plan.check()
    assert np.array_equal(xd.cpu().numpy().reshape(batch, n1, n2), yh)
    plan.destroy()


BF16_TOL = {4: 2e-2, 5: 1e-4}


@pytest.mark.parametrize("r,n1,n2", [(16, 256, 256), (8, 64, 512), (32, 1024, 32)])
@pytest.mark.parametrize("prec", [5, 4])
def test_dft2_bf16(pkg, r, n1, n2, prec):
    import torch
    batch = 2
    x = inputs.make("normal", n1 * n2, batch, seed=11).reshape(batch, n1, n2)
    plan = pkg.Plan2(n1, n2, batch, r, prec)
    y = plan.forward(torch.from_numpy(x).cuda().reshape(-1))
    plan.check()
    yh = y.cpu().numpy().reshape(batch, n1, n2)
    assert _rel(yh, grid.dft2(x, threads=8)).max() <= BF16_TOL[prec]
    plan.destroy()


@pytest.mark.parametrize("r,n1,n2,batch", [(16, 4096, 256, 2), (8, 512, 4096, 1),
                                           (16, 16, 16, 4)])
def test_conv2_general(pkg, r, n1, n2, batch):
    # against the convolution theorem on the oracle's 2-D DFT (pinned)
    import torch
    x = inputs.make("uniform", n1 * n2, batch, seed=8).reshape(batch, n1, n2)
    w = inputs.make("normal", n1 * n2, 1, seed=9).reshape(n1, n2)
    one = pkg.Plan2(n1, n2, 1, r, 3)
    spec = one.forward(torch.from_numpy(w).cuda().reshape(-1))
    plan = pkg.Plan2(n1, n2, batch, r, 3)
    xd = torch.from_numpy(x).cuda().reshape(-1)
    y = plan.conv(xd, spec)
    plan.check()
    one.check()
    yh = y.cpu().numpy().reshape(batch, n1, n2)
    ref = grid.dft2(grid.dft2(x, threads=8) * grid.dft2(w, threads=8)[None], inverse=True,
                    threads=8)
    assert _rel(yh, ref).max() <= 1e-5
    plan.destroy()
    one.destroy()


def test_dft2_in_place_and_closed_form(pkg):
    import torch
    n1, n2 = 64, 64
    x = np.zeros((2, n1, n2), np.complex64)
    x[0, 0, 0] = 1                   # delta -> all ones
    x[1] = 1                         # constant -> n1 n2 delta
    plan = pkg.Plan2(n1, n2, 2, 8, 3)
    xd = torch.from_numpy(x).cuda().reshape(-1)
    plan.forward(xd, xd)
    plan.check()
    y = xd.cpu().numpy().reshape(2, n1, n2)
    assert np.max(np.abs(y[0] - 1)) < 1e-5
    e = np.zeros((n1, n2))
    e[0, 0] = n1 * n2
    assert np.max(np.abs(y[1] - e)) < 1e-5 * n1 * n2
    plan.destroy()


@pytest.mark.parametrize("r,n1,n2,batch", [(16, 16, 256, 3), (8, 64, 64, 5), (32, 32, 1024, 2),
                                           (8, 512, 64, 2)])
def test_conv2_matches_the_definition(pkg, r, n1, n2, batch):
    import torch
    x = inputs.make("uniform", n1 * n2, batch, seed=7).reshape(batch, n1, n2)
    # a sparse kernel keeps the O(n^4) definition cheap
    rng = np.random.default_rng(3)
    w = np.zeros((n1, n2), np.complex64)
    for _ in range(9):
        w[rng.integers(n1), rng.integers(n2)] = complex(rng.standard_normal(), rng.standard_normal())
    one = pkg.Plan2(n1, n2, 1, r, 3)
    spec = one.forward(torch.from_numpy(w).cuda().reshape(-1))
    plan = pkg.Plan2(n1, n2, batch, r, 3)
    xd = torch.from_numpy(x).cuda().reshape(-1)
    y = plan.conv(xd, spec)
    plan.check()
    one.check()
    yh = y.cpu().numpy().reshape(batch, n1, n2)
    assert _rel(yh, grid.conv2_circular(x, w)).max() <= 1e-5
    # in place
    plan.conv(xd, spec, xd)
    plan.check()
    assert np.array_equal(xd.cpu().numpy().reshape(batch, n1, n2), yh)
    plan.destroy()
    one.destroy()


HEAT = [[0.0, 0.1, 0.0], [0.15, 0.5, 0.15], [0.0, 0.1, 0.0]]


@pytest.mark.parametrize("r,k", [(8, 1), (8, 5), (16, 20), (8, 40), (32, 100), (16, 128),
                                 (8, 200)])
def test_stencil_weights(pkg, r, k):
    # a positive stencil of unit sum (like the heat update): coefficients of
    # P^k stay within fp32 range for any k
    rng = np.random.default_rng(k)
    w3 = np.abs(np.array(HEAT) + 0.05 * rng.standard_normal((3, 3)))
    w3 = (w3 / w3.sum()).astype(np.float32)
    plan = pkg.StencilPlan(4 * k, k, r, 3)
    W = plan.weights(w3.tolist())
    plan.check()
    ref = grid.stencil_weights(w3.astype(np.float64), k)
    got = W.cpu().numpy()
    assert got.shape == ref.shape
    # Error bound, first order in the transforms' errors (P has unit sum and
    # non-negative entries, so |P^(w)| <= 1 at every frequency w):
    #  * forward 2-D DFT of P on the Nw x Nw grid: ||dP^||_2 <= 1e-5 ||P^||_2
    #    = 1e-5 Nw ||P||_2 (the per-transform relative L2 bar, Parseval);
    #  * k-th power: d(P^k) = k P^(k-1) dP^, and |P^|^(k-1) <= 1, so the
    #    spectrum error is at most k ||dP^||_2; the inverse (1/Nw^2 times a
    #    unitary-times-Nw map) turns it into k * 1e-5 ||P||_2 on W;
    #  * the inverse DFT's own error: 1e-5 ||W||_2 (same bar);
    #  * the pointwise power by repeated squaring in fp32: at most
    #    2 log2(k) roundings of 2^-24 per frequency, 2 log2(k) 2^-24 ||W||_2.
    pn, wn = np.linalg.norm(w3.astype(np.float64)), np.linalg.norm(ref)
    bound = 1e-5 * (k * pn + wn) + 2 * max(1.0, np.log2(k)) * 2.0 ** -24 * wn
    assert np.linalg.norm(got.astype(np.float64) - ref) <= bound
    plan.destroy()


# output blocks of N - 2k points: (8, 64, 4) one 56-block cut at 8, (8, 96, 8)
# blocks of 48, (16, 128, 16) and (8, 120, 20) blocks of 224 and 24, and
# sides that no block size divides: 100 with k = 6 (blocks of 52), 130 with
# k = 16 (blocks of 224: one cut block), 37 with k = 5 (blocks of 54)
# and more: (8, 2000, 16) 3969 tiles of 32^2 blocks, (16, 300, 16) four
# tiles of 224^2 blocks (256^2 tiles), (8, 100, 30) one 512^2 tile (3k > 64:
# three radix-8 stages per axis) whose 452^2 block is cut at 100
@pytest.mark.parametrize("r,side,k", [(8, 64, 4), (8, 96, 8), (16, 128, 16), (8, 120, 20),
                                      (8, 100, 6), (16, 130, 16), (8, 37, 5),
                                      (8, 2000, 16), (16, 300, 16), (8, 100, 30),
                                      (16, 300, 128), (8, 300, 200)])
def test_stencil_apply(pkg, r, side, k):
    import torch
    rng = np.random.default_rng(side + k)
    A = rng.standard_normal((side, side)).astype(np.float32)
    w3 = np.array(HEAT, np.float32)
    plan = pkg.StencilPlan(side, k, r, 3)
    Ad = torch.from_numpy(A).cuda().reshape(-1)
    Ak = plan.apply(Ad, w3x3=w3.tolist())
    plan.check()
    got = Ak.cpu().numpy().reshape(side, side)
    ref = grid.stencil_direct(A.astype(np.float64), w3.astype(np.float64), k)
    # Each 2-D transform of the convolution meets the 1e-5 relative bar with
    # respect to its own input, whose scale is the grid A's (the kernel's
    # spectrum is bounded by 1: a unit-sum, non-negative stencil); the k
    # steps of the stencil attenuate the output (the heat kernel spreads it),
    # so the bar is taken on max |A|, not on the smaller max |A_k|.
    assert np.max(np.abs(got - ref)) <= 1e-5 * np.max(np.abs(A))
    # in place
    plan.apply(Ad, Ad, w3x3=w3.tolist())
    plan.check()
    assert np.array_equal(Ad.cpu().numpy().reshape(side, side), got)
    plan.destroy()
