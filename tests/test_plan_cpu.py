"""The convolution planner on the host (no GPU): tests/plan_check.cu
compiles conv2d.cu's planning code with the kernel launchers stubbed and
checks every plan over a grid of shapes and formats against the
shared-memory, TMEM and layout limits."""
import os
import subprocess
import tempfile

import pytest

from paper_1809_10572_gb300 import build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_every_plan_fits_and_does_not_overlap():
    try:
        nvcc = build.nvcc()
    except RuntimeError:
        pytest.skip("nvcc not available")
    with tempfile.TemporaryDirectory(prefix="samd_plan_") as tmp:
        exe = os.path.join(tmp, "plan_check")
        cmd = [nvcc] + build.ARCH + ["-O2", "-std=c++17", "--expt-relaxed-constexpr", "-I", os.path.join(ROOT, "include"),
                                     os.path.join(ROOT, "tests", "plan_check.cu"), "-o", exe, "-lcuda"]
        r = subprocess.run(cmd, capture_output=True, text=True)
        assert r.returncode == 0, r.stderr[-2000:]
        r = subprocess.run([exe], capture_output=True, text=True, timeout=600)
        assert r.returncode == 0, r.stdout[-2000:]
        assert "bad 0" in r.stdout
        # the grid reaches every planning mode
        for mode in ("halo", "segmented", "e4m3", "resident", "two-half", "four-part", "window gather", "staging at the chosen depth",
                     "staged epilogue"):
            count = int(r.stdout.split(mode)[1].split()[0].strip("(),"))
            assert count > 0, (mode, r.stdout)
