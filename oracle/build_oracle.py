"""Compile oracle.c into liboracle.so with the host C compiler.

Test infrastructure: the product build calls this only to have the checker
ready on the machine that runs the tests. OpenMP is used when the compiler
supports it; otherwise the oracle runs single-threaded.
"""
from __future__ import annotations

import os
import subprocess
import tempfile

_HERE = os.path.dirname(os.path.abspath(__file__))


def oracle_lib_path() -> str:
    return os.path.join(_HERE, "liboracle.so")


def build_oracle(cc: str = "gcc") -> str:
    src = os.path.join(_HERE, "oracle.c")
    out = oracle_lib_path()
    base = [cc, "-O2", "-std=c11", "-fPIC", "-shared", "-Wall", "-Wextra"]
    # Build into a temporary file and rename, so a concurrent loader never
    # sees a half-written library.
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
    os.close(fd)
    try:
        for extra in (["-fopenmp"], []):
            r = subprocess.run(base + extra + [src, "-o", tmp], capture_output=True, text=True)
            if r.returncode == 0:
                os.replace(tmp, out)
                return out
        raise RuntimeError("oracle build failed:\n" + r.stderr)
    finally:
        if os.path.exists(tmp):
            os.remove(tmp)
