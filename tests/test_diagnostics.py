"""Diagnostics on the GPU: allocation failures injected on the host
(TCU_DFT_FAIL_ALLOC), the synchronising debug exec (TCU_DFT_DEBUG) and the
bounds-checked library (libtcu_dft_checked.so).  Nothing here faults or
hangs a GPU: a failed allocation is simply not made, and the checked
library skips an out-of-range access instead of making it."""
import os
import subprocess
import sys

import numpy as np
import pytest

import inputs
import oracle

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _plans(pkg):
    """One constructor per kind of plan (its device allocations differ)."""
    return {
        "one pass": lambda: pkg.Plan(4096, 4, 16, pkg.X3TF32),
        "two passes": lambda: pkg.Plan(65536, 8, 16, pkg.X3TF32),
        "three passes": lambda: pkg.Plan(1 << 20, 2, 16, pkg.X3TF32),
        "fused": lambda: pkg.Plan(65536, 64, 16, pkg.X3TF32, pkg.PLAN_FUSE),
        "mixed radix": lambda: pkg.Plan(2048, 4, 16, pkg.X3TF32),
        "2-D": lambda: pkg.Plan2(256, 256, 2, 16, pkg.X3TF32),
        "stencil": lambda: pkg.StencilPlan(256, 4, 16, pkg.X3TF32),
    }


@pytest.mark.parametrize("kind", ["one pass", "two passes", "three passes", "fused",
                                  "mixed radix", "2-D", "stencil"])
def test_every_failed_allocation_returns_oom_and_frees(kind, monkeypatch):
    import torch
    from paper_1908_06649_gb300 import _build
    _build.build()
    import paper_1908_06649_gb300 as pkg
    make = _plans(pkg)[kind]
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    failed = 0
    for k in range(1, 64):
        monkeypatch.setenv("TCU_DFT_FAIL_ALLOC", str(k))
        try:
            plan = make()
        except pkg.TcuDftError as e:
            assert e.status == pkg.ERR_OOM, (k, e.status)
            failed += 1
            continue
        # k is past the plan's last allocation: it was built normally
        plan.destroy()
        break
    else:
        raise AssertionError("the plan still failed at allocation 63")
    assert failed >= 2  # tables and error word at least
    monkeypatch.delenv("TCU_DFT_FAIL_ALLOC")
    # nothing of the failed plans stays allocated (2 MiB allocation granules)
    torch.cuda.synchronize()
    assert free0 - torch.cuda.mem_get_info()[0] <= 4 << 20
    # and a plan of the same kind still works
    make().destroy()


def test_debug_exec_synchronises_and_reports(monkeypatch):
    import torch
    import paper_1908_06649_gb300 as pkg
    n, batch = 65536, 4
    x = torch.from_numpy(inputs.make("normal", n, batch, seed=5)).cuda()
    plan = pkg.Plan(n, batch, 16, pkg.X3TF32)
    monkeypatch.setenv("TCU_DFT_DEBUG", "1")
    y = plan.forward(x)           # the exec returned the checked status (OK)
    assert torch.cuda.current_stream().query()  # and the stream has drained
    err = oracle.rel_l2(y.cpu().numpy(), oracle.dft(x.cpu().numpy(), threads=8))
    assert err.max() <= 1e-5
    plan.destroy()


CHECKED_SCRIPT = r'''
import sys
sys.path.insert(0, %(root)r)
sys.path.insert(0, %(tests)r)
import numpy as np, torch
import inputs, oracle
import paper_1908_06649_gb300 as pkg
assert pkg.lib_path().endswith("libtcu_dft_checked.so"), pkg.lib_path()
bad = []
def check(name, got, want, tol):
    err = float(oracle.rel_l2(got, want).max())
    if not err <= tol:
        bad.append((name, err))
# 1-D: one, two and three passes, every radix, mixed radix, both directions
for n, batch, r, prec, tol in [(4096, 3, 16, 3, 1e-5), (65536, 3, 16, 3, 1e-5),
                               (1 << 20, 1, 16, 3, 1e-5), (256, 5, 16, 1, 3e-3),
                               (32768, 2, 8, 3, 1e-5), (32768, 2, 32, 3, 1e-5),
                               (512, 7, 8, 3, 1e-5), (2048, 3, 16, 3, 1e-5),
                               (65536, 2, 16, 4, 1e-2)]:
    x = inputs.make("normal", n, batch, seed=7)
    plan = pkg.Plan(n, batch, r, prec)
    xd = torch.from_numpy(x).cuda()
    y = plan.forward(xd)
    plan.check()
    check("fwd %%d x %%d r %%d" %% (n, batch, r), y.cpu().numpy(), oracle.dft(x, threads=8), tol)
    z = plan.inverse(y)
    plan.check()
    check("round trip %%d r %%d" %% (n, r), z.cpu().numpy(), x, 2 * tol)
    plan.destroy()
# the fused schedule
n, batch = 65536, 64
x = inputs.make("normal", n, batch, seed=8)
plan = pkg.Plan(n, batch, 16, 3, pkg.PLAN_FUSE)
assert plan.fused
y = plan.forward(torch.from_numpy(x).cuda())
plan.check()
check("fused", y.cpu().numpy()[:4], oracle.dft(x[:4], threads=8), 1e-5)
plan.destroy()
# 2-D DFT, convolution (the spectrum-product row pass) and a stencil
from oracle import grid
p2 = pkg.Plan2(256, 256, 2, 16, 3)
x = inputs.make("normal", 256 * 256, 2, seed=9).reshape(2, 256, 256)
y = p2.forward(torch.from_numpy(x).cuda().reshape(-1))
p2.check()
check("dft2", y.cpu().numpy().reshape(2, -1), grid.dft2(x).reshape(2, -1), 1e-5)
w = np.zeros((256, 256), np.complex64)
w[0, 0], w[1, 2], w[255, 3] = 0.5, 0.25, -0.125
spec = p2.forward(torch.from_numpy(np.broadcast_to(w, (2, 256, 256)).copy()).cuda().reshape(-1))
c = p2.conv(torch.from_numpy(x).cuda().reshape(-1), spec[:256 * 256])
p2.check()
check("conv2", c.cpu().numpy().reshape(2, -1), grid.conv2_circular(x, w).reshape(2, -1), 1e-5)
p2.destroy()
st = pkg.StencilPlan(128, 16, 16, 3)
A = np.random.default_rng(1).standard_normal((128, 128)).astype(np.float32)
w3 = np.array([[0.05, 0.1, 0.05], [0.1, 0.4, 0.1], [0.05, 0.1, 0.05]], np.float32)
out = st.apply(torch.from_numpy(A).cuda().reshape(-1), w3x3=w3.tolist())
st.check()
ref = grid.stencil_direct(A.astype(np.float64), w3.astype(np.float64), 16)
e = float(np.max(np.abs(out.cpu().numpy().reshape(128, 128) - ref)) / np.max(np.abs(ref)))
if not e <= 1e-5:
    bad.append(("stencil", e))
st.destroy()
print("bad", bad)
sys.exit(1 if bad else 0)
'''


def test_checked_build_runs_clean():
    """Every path through the bounds-checked library: no index out of range
    (check() would raise ERR_BOUNDS) and the oracle's results."""
    from paper_1908_06649_gb300 import _build
    _build.build(checked=True)
    env = dict(os.environ, TCU_DFT_CHECKED="1")
    script = CHECKED_SCRIPT % {"root": ROOT, "tests": os.path.join(ROOT, "tests")}
    r = subprocess.run([sys.executable, "-c", script], env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
