"""The allocation-free entry point, checked against the plan-based one.

tcu_dft_exec_noalloc serves callers that may not allocate device memory
(their memory belongs to a framework pool or an embedding application, or a
cudaMalloc would stall the device inside a latency budget): everything it
needs besides the caller's input and output lives in fixed arrays inside the
library.  This file is collected last so that a run stopping at the first
failure has already run every other test; it passes alone in a fresh process
as well as after the others (the first call on a device does the set-up).
"""
import ctypes

import numpy as np
import pytest

import inputs
import oracle

pytestmark = pytest.mark.gpu

TOL = 1e-5  # per-transform relative L2, the 3xTF32 bar of the parity tests


@pytest.fixture(scope="module")
def pkg():
    from paper_1908_06649_gb300 import _build
    _build.build()
    import paper_1908_06649_gb300 as p
    p.lib()
    return p


def _noalloc(pkg, x, n, batch, r, prec, direction):
    import torch
    out = torch.empty_like(x)
    stream = torch.cuda.current_stream()
    rc = pkg.lib().tcu_dft_exec_noalloc(
        n, batch, r, prec, ctypes.c_void_p(x.data_ptr()),
        ctypes.c_void_p(out.data_ptr()), direction,
        ctypes.c_void_p(stream.cuda_stream))
    assert rc == pkg.OK, pkg.strerror(rc)
    return out


def _with_plan(pkg, x, n, batch, r, prec, direction):
    plan = pkg.Plan(n, batch, r, prec)
    y = plan.exec(x, None, direction)
    plan.check()
    plan.destroy()
    return y


def _rel(a, b):
    a = a.cpu().numpy().astype(np.complex128)
    b = b.cpu().numpy().astype(np.complex128)
    return np.linalg.norm(a - b, axis=1) / np.linalg.norm(b, axis=1)


@pytest.mark.parametrize("n,batch,r,direction", [
    (65536, 16, 16, -1),   # two passes: the intermediate uses the fixed array
    (4096, 200, 8, 1),     # two passes, radix 8, inverse
    (32768, 24, 32, 1),    # two passes, radix 32: two-level inter-pass twiddles
])
def test_two_calls_in_a_row_match_the_plan_path(pkg, n, batch, r, direction):
    import torch
    xs = [torch.from_numpy(inputs.make("normal", n, batch, seed=40 + i)).cuda()
          .reshape(batch, n) for i in range(2)]
    ys = [_noalloc(pkg, x, n, batch, r, 3, direction) for x in xs]
    torch.cuda.synchronize()
    for x, y in zip(xs, ys):
        ref = _with_plan(pkg, x, n, batch, r, 3, direction)
        assert np.max(_rel(y, ref)) <= TOL
    # and against the fp64 oracle on a few transforms
    x0 = xs[1][:3].cpu().numpy()
    err = oracle.rel_l2(ys[1][:3].cpu().numpy(),
                        oracle.dft(x0, inverse=direction == 1, threads=8))
    assert err.max() <= TOL


def test_in_place_and_too_large(pkg):
    import torch
    n, batch, r = 4096, 8, 16
    x = torch.from_numpy(inputs.make("uniform", n, batch, seed=3)).cuda()
    ref = _with_plan(pkg, x, n, batch, r, 3, -1)
    y = x.clone()
    stream = torch.cuda.current_stream()
    rc = pkg.lib().tcu_dft_exec_noalloc(n, batch, r, 3, ctypes.c_void_p(y.data_ptr()),
                                        ctypes.c_void_p(y.data_ptr()), -1,
                                        ctypes.c_void_p(stream.cuda_stream))
    assert rc == pkg.OK
    torch.cuda.synchronize()
    assert np.max(_rel(y.reshape(batch, n), ref.reshape(batch, n))) <= TOL
    big = torch.zeros(65536 * 80, dtype=torch.complex64, device="cuda")
    rc = pkg.lib().tcu_dft_exec_noalloc(65536, 80, 16, 3, ctypes.c_void_p(big.data_ptr()),
                                        ctypes.c_void_p(big.data_ptr()), -1,
                                        ctypes.c_void_p(stream.cuda_stream))
    assert rc == pkg.ERR_TOO_LARGE
    torch.cuda.synchronize()
    assert torch.count_nonzero(big).item() == 0
