"""Failure detection on the GPU without a fault: a wait that runs out.

The fused schedule is started past work that never runs
(tcu_dft_exec_stalled), so its dependency waits cannot be satisfied; each
gives up after its bounded limit and the kernel reports TCU_DFT_ERR_TIMEOUT
through the plan's error word.  The test checks the status, then that the
same plan (and the context) still transforms correctly.  Collected after the
parity tests (file name) so that a slow stall does not delay them."""
import ctypes

import numpy as np
import pytest

import inputs
import oracle

pytestmark = pytest.mark.gpu


def test_wait_runs_out_and_context_recovers():
    import torch
    from paper_1908_06649_gb300 import _build
    _build.build()
    import paper_1908_06649_gb300 as pkg
    n, batch = 65536, 64
    plan = pkg.Plan(n, batch, 16, 3, pkg.PLAN_FUSE)
    assert plan.fused
    x = torch.from_numpy(inputs.make("normal", n, batch, seed=3)).cuda()
    y = torch.empty_like(x)
    L = pkg.lib()
    stream = torch.cuda.current_stream()
    rc = L.tcu_dft_exec_stalled(plan.handle, ctypes.c_void_p(x.data_ptr()),
                                ctypes.c_void_p(y.data_ptr()),
                                ctypes.c_void_p(stream.cuda_stream))
    assert rc == pkg.OK
    status = L.tcu_dft_check(plan.handle, ctypes.c_void_p(stream.cuda_stream))
    assert status == pkg.ERR_TIMEOUT
    # the word is cleared and the plan works again
    plan.forward(x, y)
    plan.check()
    got = y.cpu().numpy()[:2]
    err = oracle.rel_l2(got, oracle.dft(x.cpu().numpy()[:2], threads=8))
    assert err.max() <= 1e-5
    plan.destroy()


def test_stalled_needs_a_fused_plan():
    import torch
    import paper_1908_06649_gb300 as pkg
    plan = pkg.Plan(65536, 64, 16, 3)
    x = torch.zeros(65536 * 64, dtype=torch.complex64, device="cuda")
    assert pkg.lib().tcu_dft_exec_stalled(plan.handle, ctypes.c_void_p(x.data_ptr()),
                                          ctypes.c_void_p(x.data_ptr()), None) == pkg.ERR_INVALID
    plan.destroy()
