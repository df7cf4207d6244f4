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
