"""bench.py's host logic on the CPU: the metric name, the L2-flush rule, the
traffic record's validity check and the accuracy figure of the CPU-baseline
leg (no GPU: the GPU's outputs are stood in for by exact and perturbed
spectra)."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
import inputs  # noqa: E402
import oracle  # noqa: E402


def test_metric_name_of_the_default_workload_is_the_headline():
    assert bench.metric_for(inputs.WORKLOADS["n65536_b1024"]) == bench.METRIC
    m = bench.metric_for(inputs.WORKLOADS["n4096_b64"])
    assert "n=2^12 ×64" in m and m != bench.METRIC


def test_l2_flush_rule():
    # buffers below twice the 129 MB L2 are flushed between steps
    assert bench.needs_flush(inputs.WORKLOADS["n4096_b64"])
    assert not bench.needs_flush(inputs.WORKLOADS["n65536_b1024"])
    assert not bench.needs_flush(inputs.WORKLOADS["n256_b1048576"])
    assert bench.needs_flush(dict(n=65536, batch=16))


def test_traffic_record_follows_the_kernel_sources(monkeypatch):
    rec = os.path.join(ROOT, "profiles", "traffic_dft_pass_kernel_n65536.txt")
    kv = {}
    for line in open(rec):
        if ":" in line and not line.startswith("#"):
            k, v = line.split(":", 1)
            kv[k.strip()] = v.strip()
    monkeypatch.setattr(bench, "kernel_sources_sha256", lambda: kv["sources_sha256"])
    per512 = float(kv["dram_bytes_per_launch_b512"])
    assert bench.profiled_traffic(1024, False) == per512 * 2
    assert bench.profiled_traffic(512, False) == per512
    assert bench.profiled_traffic(1024, True) is None        # fused: not this kernel
    monkeypatch.setattr(bench, "kernel_sources_sha256", lambda: "0" * 64)
    assert bench.profiled_traffic(1024, False) is None        # sources changed


def test_kernel_sources_hash_covers_the_csrc_files():
    h = bench.kernel_sources_sha256()
    assert len(h) == 64 and h == bench.kernel_sources_sha256()


def test_cpu_baseline_accuracy_figure():
    wl = dict(n=256, batch=8, kind="normal", seed=11, sqrt_m=16)
    x = inputs.make("normal", 256, 8, 11)
    exact = oracle.dft(x).astype(np.complex64)
    acc, cpu = bench.cpu_baseline(wl, seconds=0.2, sample=8, y_gpu=exact.reshape(-1),
                                  tol=1e-5)
    assert cpu["kind"] == "oracle" and cpu["cores"] >= 1 and cpu["value"] > 0
    assert acc["ok"] and acc["max_rel_l2"] < 1e-6 and acc["transforms"] == 8
    # a perturbed spectrum fails the tolerance
    bad = exact.copy()
    bad[3] *= 1.001
    acc, _ = bench.cpu_baseline(wl, seconds=0.2, sample=8, y_gpu=bad.reshape(-1),
                                tol=1e-5)
    assert not acc["ok"] and abs(acc["max_rel_l2"] - 1e-3) < 1e-4
    # the direct-definition timing appears for short transforms
    assert cpu["direct"] is not None
