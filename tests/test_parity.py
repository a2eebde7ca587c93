"""GPU parity: the tcgen05 DFT against the fp64 oracle on the same seeded
inputs, through the C ABI.

Bar (per-transform relative L2, max over the batch): <= 1e-5 in 3xTF32 mode,
<= 3e-3 in TF32 mode.
"""
import numpy as np
import pytest

import inputs
import oracle

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


def run(pkg, x, r, prec, inverse=False, inplace=False, flags=0):
    import torch
    batch, n = x.shape
    plan = pkg.Plan(n, batch, r, prec, flags)
    xd = torch.from_numpy(np.ascontiguousarray(x)).cuda()
    if inplace:
        y = plan.exec(xd, xd, pkg.INVERSE if inverse else pkg.FORWARD)
    else:
        y = plan.inverse(xd) if inverse else plan.forward(xd)
    plan.check()
    out = y.cpu().numpy()
    passes = plan.passes()
    plan.destroy()
    return out, passes


def check(y, x, prec, inverse=False):
    err = oracle.rel_l2(y, oracle.dft(x, inverse=inverse, threads=8))
    assert np.all(np.isfinite(err))
    assert err.max() <= TOL[prec], "max rel L2 %.3e" % err.max()
    return err


# ---- k = 1: one stage is a single tall-left product with F_r (the textbook
# matrix-vector DFT of the definition)
@pytest.mark.parametrize("r", [8, 16, 32])
def test_single_stage_deltas(pkg, r):
    n = r
    x = np.zeros((n, n), np.complex64)
    x[np.arange(n), np.arange(n)] = 1  # delta_j in row j -> row j of W
    y, _ = run(pkg, x, r, 3)
    j = np.arange(n)
    W = np.exp(-2j * np.pi * ((np.outer(j, j)) % n) / n)
    assert np.max(np.abs(y - W)) < 2e-6


@pytest.mark.parametrize("r,k", [(8, 1), (8, 2), (8, 3),
                                 (16, 1), (16, 2), (16, 3),
                                 (32, 1), (32, 2)])
@pytest.mark.parametrize("prec", [3, 1])
def test_single_pass(pkg, r, k, prec):
    n = r ** k
    batch = max(3, min(67, (1 << 16) // n))  # ragged: not a multiple of a tile
    x = inputs.make("normal", n, batch, seed=10 + k)
    y, passes = run(pkg, x, r, prec)
    assert sum(passes) == k
    check(y, x, prec)


# ---- several HBM passes (four-step split applied recursively): up to three
# passes of <= 2 stages (<= 3 for r = 8); the earlier passes take fewer
@pytest.mark.parametrize("r,k,batch,stages", [
    (16, 4, 5, [2, 2]), (16, 4, 40, [2, 2]), (8, 4, 6, [2, 2]),
    (32, 3, 3, [1, 2]), (32, 4, 1, [2, 2]),
    (16, 5, 2, [1, 2, 2]), (16, 6, 1, [2, 2, 2]), (8, 5, 3, [2, 3]),
    (8, 6, 2, [3, 3]), (8, 5, 41, [2, 3]), (8, 7, 1, [2, 2, 3]), (8, 8, 1, [2, 3, 3]),
    (32, 5, 1, [1, 2, 2])])
@pytest.mark.parametrize("prec", [3, 1])
def test_multi_pass(pkg, r, k, batch, stages, prec):
    n = r ** k
    x = inputs.make("uniform", n, batch, seed=20 + k)
    y, passes = run(pkg, x, r, prec)
    assert passes == stages
    check(y, x, prec)


@pytest.mark.parametrize("r,k,batch", [(16, 4, 5), (16, 4, 40), (8, 4, 6), (32, 4, 1)])
@pytest.mark.parametrize("prec", [3, 1])
def test_fused_two_pass(pkg, r, k, batch, prec):
    n = r ** k
    x = inputs.make("uniform", n, batch, seed=30 + k)
    y, passes = run(pkg, x, r, prec, flags=pkg.PLAN_FUSE)
    assert passes == [2, 2]
    check(y, x, prec)


@pytest.mark.parametrize("r,k", [(16, 4), (8, 4), (32, 4)])
def test_fused_schedule_is_used(pkg, r, k):
    n = r ** k
    plan = pkg.Plan(n, 2, r, 3, pkg.PLAN_FUSE)
    assert plan.fused
    plan.destroy()
    plan = pkg.Plan(n, 2, r, 3)
    assert not plan.fused
    plan.destroy()


# ---- one HBM pass on cluster pairs (TCU_DFT_PLAN_ONE_PASS, n = 16^4): both
# passes in one launch, each cluster's intermediates in two L2 slots.  Batches
# below, at and above the number of cluster pairs, odd batches (a last pair
# of one transform), forward and inverse, in place.
@pytest.mark.parametrize("batch", [1, 2, 3, 7, 40, 151, 152, 153, 305])
def test_one_pass_pairs(pkg, batch):
    n = 16 ** 4
    x = inputs.make("normal", n, batch, seed=300 + batch)
    y, passes = run(pkg, x, 16, 3, flags=pkg.PLAN_ONE_PASS)
    assert passes == [2, 2]
    check(y, x, 3)


@pytest.mark.parametrize("prec", [3, 1])
def test_one_pass_pairs_inverse_in_place(pkg, prec):
    import torch
    n, batch = 16 ** 4, 77
    x = inputs.make("uniform", n, batch, seed=31)
    plan = pkg.Plan(n, batch, 16, prec, pkg.PLAN_ONE_PASS)
    assert plan.fused
    xd = torch.from_numpy(x).cuda()
    y = plan.exec(xd, xd, pkg.INVERSE)  # in place
    plan.check()
    got = y.cpu().numpy()
    err = oracle.rel_l2(got, oracle.dft(x, inverse=True, threads=8))
    assert err.max() <= TOL[prec]
    # and forward again, out of place, from the inverse's output
    z = plan.forward(y)
    plan.check()
    back = z.cpu().numpy()
    rt = np.linalg.norm(back - x, axis=1) / np.linalg.norm(x, axis=1)
    assert rt.max() <= (1e-5 if prec == 3 else 3e-3)
    plan.destroy()


def test_one_pass_pairs_repeated_calls(pkg):
    # the slots and barriers start afresh at every launch: several launches
    # in a row on the same plan give the same bits
    import torch
    n, batch = 16 ** 4, 200
    x = torch.from_numpy(inputs.make("normal", n, batch, seed=32)).cuda()
    plan = pkg.Plan(n, batch, 16, 3, pkg.PLAN_ONE_PASS)
    outs = [plan.forward(x) for _ in range(3)]
    plan.check()
    for o in outs[1:]:
        assert torch.equal(o, outs[0])
    ref = pkg.Plan(n, batch, 16, 3)
    y2 = ref.forward(x)
    ref.check()
    err = oracle.rel_l2(outs[0][:4].cpu().numpy(), oracle.dft(x[:4].cpu().numpy(), threads=8))
    assert err.max() <= TOL[3]
    d = (outs[0] - y2).abs().max().item() / y2.abs().max().item()
    assert d < 1e-5
    plan.destroy()
    ref.destroy()


@pytest.mark.parametrize("r,k", [(16, 2), (16, 4), (8, 4)])
def test_inverse_fused(pkg, r, k):
    n = r ** k
    x = inputs.make("normal", n, 16, seed=9)
    y, _ = run(pkg, x, r, 3, inverse=True, flags=pkg.PLAN_FUSE)
    check(y, x, 3, inverse=True)


@pytest.mark.parametrize("r,k", [(16, 2), (16, 4), (8, 5), (32, 3), (16, 5)])
def test_inverse_and_round_trip(pkg, r, k):
    import torch
    n = r ** k
    batch = 3
    x = inputs.make("normal", n, batch, seed=2)
    y, _ = run(pkg, x, r, 3, inverse=True)
    check(y, x, 3, inverse=True)
    plan = pkg.Plan(n, batch, r, 3)
    xd = torch.from_numpy(x).cuda()
    back = plan.inverse(plan.forward(xd)).cpu().numpy()
    plan.check()
    plan.destroy()
    rt = np.linalg.norm(back - x, axis=1) / np.linalg.norm(x, axis=1)
    assert rt.max() <= 1e-5


@pytest.mark.parametrize("r,k", [(16, 2), (16, 3), (16, 4), (16, 5), (8, 6)])
def test_in_place(pkg, r, k):
    n = r ** k
    x = inputs.make("uniform", n, 4, seed=5)
    y, _ = run(pkg, x, r, 3, inplace=True)
    check(y, x, 3)


def test_closed_forms(pkg):
    # delta_0 -> ones, constant -> n delta_0, pure tone -> n delta_f
    n = 4096
    x = np.zeros((3, n), np.complex64)
    x[0, 0] = 1
    x[1, :] = 1
    f = 1234
    j = np.arange(n)
    x[2] = np.exp(2j * np.pi * ((f * j) % n) / n).astype(np.complex64)
    y, _ = run(pkg, x, 16, 3)
    assert np.max(np.abs(y[0] - 1)) < 1e-5
    e0 = np.zeros(n)
    e0[0] = n
    assert np.max(np.abs(y[1] - e0)) < 1e-5 * n
    ef = np.zeros(n)
    ef[f] = n
    assert np.max(np.abs(y[2] - ef)) < 1e-4 * n


def test_tones_workload_peaks(pkg):
    # the many-short-transforms workload: 3 tones + N(0, 0.01^2) noise,
    # n = 256; the spectrum peaks sit exactly at the seeded frequencies
    n, batch = 256, 4096
    x = inputs.make("tones", n, batch, seed=4)
    y, _ = run(pkg, x, 16, 3)
    f = inputs.tone_frequencies(4, n, batch)
    top = np.argsort(-np.abs(y), axis=1)[:, :3]
    assert np.array_equal(np.sort(top, axis=1), np.sort(f, axis=1))
    mags = np.take_along_axis(np.abs(y), f, axis=1)
    assert np.all(np.abs(mags / n - 1) < 0.05)
    check(y[:256], x[:256], 3)


def oracle_batch(x, inverse=False, chunk_points=1 << 23):
    """The oracle's transform of every row of x (power-of-two n), chunk by
    chunk through its recursive radix-2 FFT on every host core; yields
    (first row, fp64 outputs) per chunk."""
    batch, n = x.shape
    rows = max(1, chunk_points // n)
    sign, scale = (1, 1.0 / n) if inverse else (-1, 1.0)
    for a in range(0, batch, rows):
        yield a, oracle.fft_radix2(x[a:a + rows], sign, scale,
                                   threads=oracle.default_threads())


def check_whole_batch(yh, x, prec, inverse=False):
    """Per-transform relative L2 of EVERY transform of the batch against the
    oracle (max over the batch <= the bar); returns the errors."""
    err = np.empty(x.shape[0])
    for a, ref in oracle_batch(x, inverse):
        err[a:a + ref.shape[0]] = oracle.rel_l2(yh[a:a + ref.shape[0]], ref)
    assert np.all(np.isfinite(err))
    assert err.max() <= TOL[prec], "max rel L2 %.3e (transform %d)" % (err.max(),
                                                                       int(err.argmax()))
    return err


def check_entries(yh, x, inverse=False, nb=8, nk=32, seed=0):
    """Single entries of sampled transforms (the first and the last among
    them) by the direct definition, each within 1e-5 of the RMS magnitude
    of the sampled reference entries."""
    batch, n = x.shape
    rng = np.random.default_rng(seed)
    bs = np.unique(np.concatenate([[0, batch - 1], rng.integers(0, batch, nb)]))
    ks = np.unique(np.concatenate([[0, 1, n - 1], rng.integers(0, n, nk)]))
    ref = oracle.dft_entries(x[bs], ks, inverse=inverse)
    got = yh[bs][:, ks]
    mag = np.sqrt(np.mean(np.abs(ref) ** 2))
    assert np.max(np.abs(got - ref)) / mag <= 1e-5


def _device_transform(pkg, x, r, prec=3, inverse=False):
    import torch
    batch, n = x.shape
    plan = pkg.Plan(n, batch, r, prec)
    xd = torch.from_numpy(x).cuda()
    y = plan.inverse(xd) if inverse else plan.forward(xd)
    plan.check()
    passes = plan.passes()
    yh = y.cpu().numpy()
    del xd, y
    plan.destroy()
    return yh, passes


def test_full_size_small_transforms(pkg):
    # n = 4096 (16^3, one pass), batch 64, U[-1,1], seed 0: every transform
    x = inputs.make("uniform", 4096, 64, seed=0)
    yh, passes = _device_transform(pkg, x, 16)
    assert passes == [3]
    err = oracle.rel_l2(yh, oracle.dft(x, threads=oracle.default_threads()))
    assert err.max() <= TOL[3]


def test_full_size_headline(pkg):
    # n = 65536, batch = 1024, N(0,1), seed 1 -- in the launch configuration
    # the benchmark times: every transform whole against the oracle, and
    # single entries by the definition
    n, batch = 65536, 1024
    x = inputs.make("normal", n, batch, seed=1)
    yh, passes = _device_transform(pkg, x, 16)
    assert passes == [2, 2]
    check_whole_batch(yh, x, 3)
    check_entries(yh, x)


_CACHE = {}


def _sweep_input():
    if "sweep" not in _CACHE:
        _CACHE["sweep"] = inputs.make("normal", 32768, 4096, seed=2)
    return _CACHE["sweep"]


@pytest.mark.parametrize("r", [8, 32])
def test_full_size_radix_sweep(pkg, r):
    # n = 32768 (8^5 = 32^3), batch 4096, N(0,1), seed 2: forward and
    # inverse (of the forward outputs) of every transform, and the round trip
    x = _sweep_input()
    y, _ = _device_transform(pkg, x, r)
    check_whole_batch(y, x, 3)
    check_entries(y, x, seed=r)
    back, _ = _device_transform(pkg, y, r, inverse=True)
    check_whole_batch(back, y, 3, inverse=True)
    rt = np.linalg.norm(back - x, axis=1) / np.linalg.norm(x, axis=1)
    assert rt.max() <= 1e-5


def test_full_size_long_transforms(pkg):
    # n = 2^24 (16^6), batch 4, uniform, seed 3: three HBM passes, all four
    # transforms whole
    n, batch = 1 << 24, 4
    x = inputs.make("uniform", n, batch, seed=3)
    yh, passes = _device_transform(pkg, x, 16)
    assert passes == [2, 2, 2]
    check_whole_batch(yh, x, 3)
    check_entries(yh, x, nb=4, nk=16)


def test_full_size_many_short_transforms(pkg):
    # n = 256 (16^2), batch 2^20, three tones + N(0, 0.01^2) noise, seed 4:
    # every transform whole against the oracle, and on every transform the
    # three largest outputs sit exactly at its seeded frequencies
    n, batch = 256, 1 << 20
    x = inputs.make("tones", n, batch, seed=4)
    yh, passes = _device_transform(pkg, x, 16)
    assert passes == [2]
    check_whole_batch(yh, x, 3)
    f = np.sort(inputs.tone_frequencies(4, n, batch), axis=1)
    C = 1 << 16
    for a in range(0, batch, C):
        mag = np.abs(yh[a:a + C])
        top = np.sort(np.argpartition(-mag, 3, axis=1)[:, :3], axis=1)
        assert np.array_equal(top, f[a:a + C])
        peaks = np.take_along_axis(mag, f[a:a + C], axis=1)
        assert np.all(np.abs(peaks / n - 1) < 0.05)


def test_maximum_size_radix8(pkg):
    # n = 8^9 = 2^27, the longest radix-8 plan: three passes of three stages,
    # whole transform against the oracle, and back
    n = 8 ** 9
    x = inputs.make("normal", n, 1, seed=90)
    y, passes = run(pkg, x, 8, 3)
    assert passes == [3, 3, 3]
    check(y, x, 3)
    back, _ = run(pkg, y, 8, 3, inverse=True)
    assert np.linalg.norm(back - x) / np.linalg.norm(x) <= 1e-5


def _sumsq(v, chunk=1 << 24):
    """sum |v|^2 in fp64, chunk by chunk (v complex64, up to 2^30 entries)."""
    tot = 0.0
    for a in range(0, v.shape[0], chunk):
        seg = v[a:a + chunk].astype(np.complex128)
        tot += float(np.sum(seg.real ** 2 + seg.imag ** 2))
    return tot


def test_maximum_size_radix32_closed_forms(pkg):
    # n = 32^6 = 2^30, the longest radix-32 plan (three passes).  A whole
    # transform would cost the oracle 16 GB and minutes, so the check is by
    # closed forms at full size: DFT(delta_s)_k = w^{ks} on sampled k and
    # Parseval; DFT(e^{+2 pi i f j / n}) = n delta_f over the whole output.
    n = 32 ** 6
    s, f = 123456789, 987654321 % n
    x = np.zeros((2, n), np.complex64)
    x[0, s] = 1.0
    C = 1 << 24
    for a in range(0, n, C):
        j = np.arange(a, a + C, dtype=np.int64)
        x[1, a:a + C] = np.exp(2j * np.pi * ((j * f) % n) / n)
    y, passes = run(pkg, x, 32, 3)
    assert passes == [2, 2, 2]
    rng = np.random.default_rng(5)
    ks = np.concatenate([[0, 1, n - 1, f], rng.integers(0, n, 4096)])
    w = np.exp(-2j * np.pi * ((ks * s) % n) / n)
    assert np.max(np.abs(y[0, ks] - w)) <= 1e-5
    assert abs(_sumsq(y[0]) / n - 1.0) <= 1e-5
    peak = complex(y[1, f])
    assert abs(peak - n) / n <= 1e-5
    rest = _sumsq(y[1]) - abs(peak) ** 2        # everything off the peak
    assert np.sqrt(max(rest, 0.0)) / n <= 1e-5


def test_exec_host_path(pkg):
    import torch
    n, batch = 4096, 64
    x = inputs.make("uniform", n, batch, seed=0)
    plan = pkg.Plan(n, batch, 16, 3)
    h_in = torch.from_numpy(x).pin_memory()
    h_out = torch.empty_like(h_in).pin_memory()
    work = torch.empty(batch * n, dtype=torch.complex64, device="cuda")
    plan.exec_host(h_in, h_out, work)
    plan.check()
    plan.destroy()
    check(h_out.numpy(), x, 3)


def test_argument_errors_launch_nothing(pkg):
    import ctypes
    import torch
    n, batch = 256, 4
    plan = pkg.Plan(n, batch, 16, 3)
    L = pkg.lib()
    buf = torch.zeros(2 * batch * n + 8, dtype=torch.complex64, device="cuda")
    base = buf.data_ptr()
    h = plan.handle
    # misaligned
    assert L.tcu_dft_exec_dir(h, ctypes.c_void_p(base + 8), ctypes.c_void_p(base + 8 * (batch * n + 4)), -1, None) == pkg.ERR_INVALID
    # partial overlap
    assert L.tcu_dft_exec_dir(h, ctypes.c_void_p(base), ctypes.c_void_p(base + 16), -1, None) == pkg.ERR_INVALID
    # bad direction
    assert L.tcu_dft_exec_dir(h, ctypes.c_void_p(base), ctypes.c_void_p(base), 0, None) == pkg.ERR_INVALID
    torch.cuda.synchronize()
    assert torch.count_nonzero(buf).item() == 0
    plan.check()
    plan.destroy()


# ---- mixed final radix (the base case of size q < sqrt(m)): n = q r^k, a
# CUDA-core q-point first pass, then tensor-core passes of radix r
@pytest.mark.parametrize("r,q,k", [(16, 2, 2), (16, 4, 2), (16, 8, 2), (16, 2, 3), (16, 8, 3),
                                   (16, 2, 4), (16, 4, 4), (16, 8, 4),
                                   (8, 2, 2), (8, 4, 3), (8, 2, 4), (8, 4, 4),
                                   (32, 2, 2), (32, 16, 2), (32, 4, 3), (32, 16, 3)])
@pytest.mark.parametrize("prec", [3, 1])
def test_mixed_radix(pkg, r, q, k, prec):
    n = q * r ** k
    batch = max(2, min(37, (1 << 18) // n))
    x = inputs.make("normal", n, batch, seed=50 + q + k)
    y, passes = run(pkg, x, r, prec)
    assert passes[0] == 1 and sum(passes[1:]) == k
    check(y, x, prec)
    yi, _ = run(pkg, x, r, prec, inverse=True)
    check(yi, x, prec, inverse=True)


# ---- mixed radix with any factor q = 2 .. 16 (odd factors included): the
# q-point pass on CUDA cores, then one tensor-core pass whose output stride
# is q; forward and inverse (1/n with n not a power of two) against the
# oracle's direct definition
@pytest.mark.parametrize("r,q,k", [(8, 3, 3), (8, 5, 2), (8, 6, 3), (8, 12, 2), (8, 7, 1),
                                   (16, 3, 2), (16, 5, 2), (16, 6, 2), (16, 12, 2),
                                   (16, 15, 1), (16, 9, 2),
                                   (32, 3, 2), (32, 5, 1), (32, 6, 2), (32, 12, 2)])
@pytest.mark.parametrize("inverse", [False, True])
def test_mixed_radix_odd_factors(pkg, r, q, k, inverse):
    n = q * r ** k
    batch = 5  # ragged: not a multiple of an item's sub-transforms
    x = inputs.make("normal", n, batch, seed=1000 + n)
    y, passes = run(pkg, x, r, 3, inverse=inverse)
    assert passes == [1, k]
    check(y, x, 3, inverse=inverse)


@pytest.mark.parametrize("r,q,k", [(16, 3, 2), (8, 10, 3), (32, 7, 2)])
def test_mixed_radix_odd_factors_tf32_and_tones(pkg, r, q, k):
    n = q * r ** k
    x = inputs.make("uniform", n, 3, seed=77)
    y, _ = run(pkg, x, r, 1)
    check(y, x, 1)
    # a pure tone at frequency f -> n at f, zero elsewhere (3xTF32)
    f = (n // 3) + 1
    j = np.arange(n)
    tone = np.exp(2j * np.pi * ((f * j) % n) / n).astype(np.complex64)[None, :]
    yt, _ = run(pkg, np.repeat(tone, 2, axis=0), r, 3)
    ef = np.zeros(n)
    ef[f] = n
    assert np.max(np.abs(yt - ef)) < 1e-5 * n


def test_mixed_radix_odd_factor_in_place(pkg):
    n, batch = 5 * 16 ** 2, 9
    x = inputs.make("normal", n, batch, seed=5)
    y, _ = run(pkg, x, 16, 3, inplace=True)
    check(y, x, 3)


def test_mixed_radix_in_place(pkg):
    n = 8 * 16 ** 4
    x = inputs.make("uniform", n, 3, seed=8)
    y, _ = run(pkg, x, 16, 3, inplace=True)
    check(y, x, 3)


# ---- the low-precision variant: BF16 operands on kind::f16 (every radix).
# Tolerance from the arithmetic: bf16 keeps 8 significant bits (unit
# roundoff u = 2^-9 after rounding to nearest); one product per stage leaves
# ~sqrt(2) u per real operand pair, growing ~sqrt(k) over k stages, so the
# single product is held to 1e-2 and the hi/lo split (16 significant bits,
# u^2-level terms dropped) to 1e-4 for up to 7 stages.
BF16_TOL = {4: 1e-2, 5: 1e-4}


@pytest.mark.parametrize("r,k,batch", [
    (16, 1, 64), (16, 2, 37), (16, 3, 9), (16, 4, 3), (16, 5, 2), (16, 6, 1),
    (8, 1, 64), (8, 2, 37), (8, 3, 11), (8, 4, 5), (8, 5, 3), (8, 6, 2), (8, 7, 1),
    (32, 1, 64), (32, 2, 9), (32, 3, 3), (32, 4, 1)])
@pytest.mark.parametrize("prec", [5, 4])
def test_bf16_modes(pkg, r, k, batch, prec):
    n = r ** k
    x = inputs.make("normal", n, batch, seed=60 + k + r)
    y, passes = run(pkg, x, r, prec)
    assert sum(passes) == k
    err = oracle.rel_l2(y, oracle.dft(x, threads=8))
    assert np.all(np.isfinite(err)) and err.max() <= BF16_TOL[prec], err.max()
    yi, _ = run(pkg, x, r, prec, inverse=True)
    erri = oracle.rel_l2(yi, oracle.dft(x, inverse=True, threads=8))
    assert erri.max() <= BF16_TOL[prec], erri.max()


@pytest.mark.parametrize("n,batch,r", [(8 ** 4, 13, 8), (16 ** 5, 5, 16), (2 * 16 ** 4, 3, 16),
                                       (32 ** 3, 9, 32)])
def test_exec_host_pipelined(pkg, n, batch, r):
    # host buffers in chunks of transforms: copies on two internal streams
    # overlap the transforms of neighbouring chunks (ragged last chunk)
    import torch
    x = inputs.make("normal", n, batch, seed=70)
    plan = pkg.Plan(n, batch, r, 3)
    h_in = torch.from_numpy(x).pin_memory()
    h_out = torch.empty_like(h_in).pin_memory()
    work = torch.empty(batch * n, dtype=torch.complex64, device="cuda")
    for _ in range(2):  # twice in a row: the second reuses the streams
        plan.exec_host(h_in, h_out, work)
        plan.check()
        check(h_out.numpy().reshape(batch, n), x, 3)
    plan.exec_host(h_in, h_out, work, pkg.INVERSE)
    plan.check()
    check(h_out.numpy().reshape(batch, n), x, 3, inverse=True)
    plan.destroy()


@pytest.mark.parametrize("n,batch,r", [(4096, 64, 16), (8 ** 5, 6, 8), (16 ** 5, 2, 16)])
def test_exec_captures_into_a_cuda_graph(pkg, n, batch, r):
    # exec allocates nothing and synchronises nothing, so it can be captured
    # once into a CUDA graph and replayed
    import torch
    x = torch.from_numpy(inputs.make("uniform", n, batch, seed=80)).cuda()
    y = torch.empty_like(x)
    plan = pkg.Plan(n, batch, r, 3)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        plan.forward(x, y)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        plan.forward(x, y)
    y.zero_()
    torch.cuda.synchronize()
    for _ in range(2):
        g.replay()
    torch.cuda.synchronize()
    plan.check()
    check(y.cpu().numpy().reshape(batch, n), x.cpu().numpy().reshape(batch, n), 3)
    plan.destroy()
