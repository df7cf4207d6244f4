"""bench.py's host-side bookkeeping (no GPU): the measured-traffic record is
reported only for the workload it was taken on and only while the kernel
sources hash to the value stored with it."""
import importlib.util
import json
import os
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_csrc_digest_is_stable(bench):
    d = bench.csrc_digest()
    assert len(d) == 64 and d == bench.csrc_digest()


def test_traffic_reported_only_while_sources_match(bench, monkeypatch):
    with open(os.path.join(ROOT, "profiles", "conv_kernel_sweep_traffic.json")) as fh:
        rec = json.load(fh)
    sweep = types.SimpleNamespace(workload="sweep", layers="")
    monkeypatch.setattr(bench, "csrc_digest", lambda: rec["csrc_sha256"])
    value, note = bench.measured_traffic(sweep)
    assert value == rec["dram_bytes_per_launch"] and "launches" in note
    monkeypatch.setattr(bench, "csrc_digest", lambda: "0" * 64)
    value, note = bench.measured_traffic(sweep)
    assert value is None and "changed" in note
    for args in (types.SimpleNamespace(workload="vgg16", layers=""), types.SimpleNamespace(workload="sweep", layers="12")):
        assert bench.measured_traffic(args)[0] is None


def test_chained_step_bookkeeping(bench):
    """A chained network shares buffers between layers: each distinct tensor
    counts once toward the bytes that decide how many input sets rotate, and
    a layer whose pool is fused is one launch, a standalone pool a second."""
    import torch

    def t(n):
        return torch.empty(n, dtype=torch.int32)

    a0, o0, p0, o1, o2 = t(100), t(50), t(10), t(40), t(20)
    conv = lambda n: types.SimpleNamespace(prepared=t(n))
    built = [
        {"act": a0, "out": o0, "conv": conv(8), "pooled": p0, "fused_pool": False},  # conv, then a pool launch
        {"act": p0, "out": o1, "conv": conv(8), "pooled": None, "fused_pool": False},
        {"act": o1, "out": o2, "conv": conv(8), "pooled": t(5), "fused_pool": True},  # pool in the epilogue
    ]
    assert bench.launches_per_step(built) == 4
    want = 4 * (100 + 50 + 10 + 40 + 20 + 5 + 3 * 8)  # p0 and o1 counted once
    assert bench.unique_bytes(built) == want
