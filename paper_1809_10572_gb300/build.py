"""Build libsamd.so in-tree for sm_103a.

Each .cu translation unit under csrc/ is compiled in parallel with nvcc
(-gencode arch=compute_103a,code=sm_103a) -- conv_inst.cu once per kernel
instantiation group -- and the objects are linked into
paper_1809_10572_gb300/lib/libsamd.so. The measurement kernels under peaks/
(tensor-core rate microbenchmarks, not part of the hot path) go into
lib/libsamd_peaks.so. A rebuild happens only when a source or header is
newer than the library.
"""
from __future__ import annotations

import glob
import os
import shutil
import subprocess
import tempfile
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
LIBDIR = os.path.join(PKG, "lib")
LIB = os.path.join(LIBDIR, "libsamd.so")
PEAKS_DIR = os.path.join(PKG, "peaks")
PEAKS_LIB = os.path.join(LIBDIR, "libsamd_peaks.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "--expt-relaxed-constexpr",
              "-Xcompiler", "-fvisibility=hidden", "-I", os.path.join(ROOT, "include")]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found")


INST_SRC = os.path.join(CSRC, "conv_inst.cu")


def sources() -> list[str]:
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def units() -> list[tuple[str, list[str], str]]:
    """(source, extra nvcc flags, object name) of every translation unit:
    each .cu once, and conv_inst.cu once per (operand type, word width, lane
    width) -- e4m3 only for lanes of up to 5 bits."""
    out = [(src, [], os.path.basename(src) + ".o") for src in sources() if src != INST_SRC]
    for fp8, max_bits in ((0, 8), (1, 5)):
        for wb in (32, 64):
            for bits in range(1, max_bits + 1):
                defs = [f"-DSAMD_INST_FP8={fp8}", f"-DSAMD_INST_WB={wb}", f"-DSAMD_INST_BITS={bits}"]
                out.append((INST_SRC, defs, f"conv_inst_{'f8' if fp8 else 'f16'}_w{wb}_b{bits}.o"))
    return out


def _inputs() -> list[str]:
    return sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + [os.path.join(ROOT, "include", "samd.h")]


def up_to_date() -> bool:
    if not os.path.exists(LIB):
        return False
    t = os.path.getmtime(LIB)
    return all(os.path.getmtime(p) <= t for p in _inputs())


def peaks_up_to_date() -> bool:
    if not os.path.exists(PEAKS_LIB):
        return False
    t = os.path.getmtime(PEAKS_LIB)
    return all(os.path.getmtime(p) <= t for p in glob.glob(os.path.join(PEAKS_DIR, "*.cu")))


def build_peaks(force: bool = False) -> str:
    """lib/libsamd_peaks.so from peaks/*.cu (one nvcc call)."""
    if not force and peaks_up_to_date():
        return PEAKS_LIB
    os.makedirs(LIBDIR, exist_ok=True)
    srcs = sorted(glob.glob(os.path.join(PEAKS_DIR, "*.cu")))
    tmp = PEAKS_LIB + ".tmp"
    cmd = [nvcc()] + ARCH + NVCC_FLAGS + ["-shared", "-o", tmp] + srcs
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc failed on peaks/:\n{r.stderr}")
    os.replace(tmp, PEAKS_LIB)
    return PEAKS_LIB


def build(force: bool = False, verbose: bool = False, extra_flags: list[str] | None = None) -> str:
    build_peaks(force)
    if not force and up_to_date():
        return LIB
    os.makedirs(LIBDIR, exist_ok=True)
    cc = nvcc()
    flags = NVCC_FLAGS + list(extra_flags or [])
    with tempfile.TemporaryDirectory(prefix="samd_build_") as tmp:
        def compile_one(unit) -> str:
            src, defs, name = unit
            obj = os.path.join(tmp, name)
            cmd = [cc] + ARCH + flags + defs + ["-c", src, "-o", obj]
            r = subprocess.run(cmd, capture_output=True, text=True)
            if r.returncode != 0:
                raise RuntimeError(f"nvcc failed on {name}:\n{r.stderr}")
            if verbose and r.stderr:
                print(name, r.stderr)
            return obj

        # the slowest units (the kernel instantiations) first
        todo = sorted(units(), key=lambda u: u[0] != INST_SRC)
        with ThreadPoolExecutor(max_workers=max(1, min(len(todo), os.cpu_count() or 4))) as ex:
            objs = list(ex.map(compile_one, todo))
        out_tmp = os.path.join(tmp, "libsamd.so")
        cmd = [cc] + ARCH + ["-shared", "-o", out_tmp] + objs
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"link failed:\n{r.stderr}")
        shutil.move(out_tmp, LIB + ".tmp")
        os.replace(LIB + ".tmp", LIB)
    return LIB


if __name__ == "__main__":
    import sys

    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv,
                extra_flags=["-Xptxas", "-v"] if "--ptxas-v" in sys.argv else None))
