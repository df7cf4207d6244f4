"""CPU oracle for the bit-precise SAMD hot path (test infrastructure).

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. The product library (``libsamd``)
neither imports nor links it, and the two share no code.

Every function works on unpacked ``int64`` numpy arrays and forwards to the
plain C definitions in ``oracle.c``; the docstrings there cite the passage of
the paper each one follows. Functions without an independent pin are marked
"parity unpinned" in their docstring; all functions here are pinned by
``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from .build_oracle import build_oracle, oracle_lib_path

ADD, SUB, MUL, RELU, REQUANT = 0, 1, 2, 3, 4
OP_NAMES = {"add": ADD, "sub": SUB, "mul": MUL, "relu": RELU, "requant": REQUANT}

_lib = None

_i64p = ctypes.POINTER(ctypes.c_int64)
_u8p = ctypes.POINTER(ctypes.c_uint8)


class OracleError(RuntimeError):
    pass


class Int32BoundError(OracleError):
    """An accumulator left the int32 range (the bound every config must meet)."""


def _load():
    global _lib
    if _lib is not None:
        return _lib
    path = oracle_lib_path()
    src = os.path.join(os.path.dirname(__file__), "oracle.c")
    if not os.path.exists(path) or os.path.getmtime(path) < os.path.getmtime(src):
        build_oracle()
    lib = ctypes.CDLL(path)
    i, i64 = ctypes.c_int, ctypes.c_int64
    lib.oracle_lanes_per_word.argtypes = [i, i, i]
    lib.oracle_lanes_per_word.restype = i
    lib.oracle_packed_words.argtypes = [i, i, i, i64, i64]
    lib.oracle_packed_words.restype = i64
    lib.oracle_wrap.argtypes = [i64, i, i]
    lib.oracle_wrap.restype = i64
    lib.oracle_clamp.argtypes = [i64, i, i]
    lib.oracle_clamp.restype = i64
    lib.oracle_pack.argtypes = [i, i, i, i, _i64p, i64, i64, _u8p]
    lib.oracle_pack.restype = i
    lib.oracle_unpack.argtypes = [i, i, i, i, _u8p, i64, i64, _i64p]
    lib.oracle_unpack.restype = i
    lib.oracle_is_canonical.argtypes = [i, i, i, _u8p, i64, i64]
    lib.oracle_is_canonical.restype = i
    lib.oracle_elementwise.argtypes = [i, i, i, i, i, _i64p, _i64p, _i64p, i64, i, i]
    lib.oracle_elementwise.restype = i
    lib.oracle_conv2d.argtypes = [i, i, i, i, i, i, i, i, i, _i64p, _i64p, _i64p, i]
    lib.oracle_conv2d.restype = i
    lib.oracle_maxpool2x2.argtypes = [i, i, i, i, _i64p, _i64p]
    lib.oracle_maxpool2x2.restype = i
    lib.oracle_max_threads.argtypes = []
    lib.oracle_max_threads.restype = i
    _lib = lib
    return lib


def _p64(a: np.ndarray):
    assert a.dtype == np.int64 and a.flags.c_contiguous
    return a.ctypes.data_as(_i64p)


def _pu8(a: np.ndarray):
    assert a.flags.c_contiguous
    return a.ctypes.data_as(_u8p)


def _word_dtype(word_bits: int):
    return {32: np.uint32, 64: np.uint64}[word_bits]


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def lanes_per_word(bits: int, spacer: int = 0, word_bits: int = 32) -> int:
    """L = floor(word_bits / (bits + spacer)) lanes per word (section 2.1, Fig. 2)."""
    return int(_load().oracle_lanes_per_word(bits, spacer, word_bits))


def packed_words(bits: int, spacer: int, word_bits: int, rows: int, inner: int) -> int:
    return int(_load().oracle_packed_words(bits, spacer, word_bits, rows, inner))


def wrap(v: int, bits: int, signed: bool) -> int:
    return int(_load().oracle_wrap(v, bits, int(signed)))


def clamp(v: int, bits: int, signed: bool) -> int:
    return int(_load().oracle_clamp(v, bits, int(signed)))


def pack(vals, bits: int, signed: bool, spacer: int = 0, word_bits: int = 32) -> np.ndarray:
    """Pack a (rows, inner) integer array; returns the words as uint32/uint64."""
    v = np.ascontiguousarray(np.asarray(vals, dtype=np.int64))
    if v.ndim == 1:
        v = v.reshape(1, -1)
    rows, inner = v.shape
    nw = packed_words(bits, spacer, word_bits, rows, inner)
    if nw < 0:
        raise OracleError("bad format")
    out = np.zeros(nw, dtype=_word_dtype(word_bits))
    rc = _load().oracle_pack(bits, int(signed), spacer, word_bits, _p64(v), rows, inner, _pu8(out.view(np.uint8)))
    if rc:
        raise OracleError(f"oracle_pack failed ({rc})")
    return out


def unpack(words, bits: int, signed: bool, spacer: int, word_bits: int, rows: int, inner: int) -> np.ndarray:
    w = np.ascontiguousarray(np.asarray(words, dtype=_word_dtype(word_bits)))
    if w.size != packed_words(bits, spacer, word_bits, rows, inner):
        raise OracleError("word count does not match rows x inner")
    out = np.zeros((rows, inner), dtype=np.int64)
    rc = _load().oracle_unpack(bits, int(signed), spacer, word_bits, _pu8(w.view(np.uint8)), rows, inner, _p64(out))
    if rc:
        raise OracleError(f"oracle_unpack failed ({rc})")
    return out


def is_canonical(words, bits: int, spacer: int, word_bits: int, rows: int, inner: int) -> bool:
    w = np.ascontiguousarray(np.asarray(words, dtype=_word_dtype(word_bits)))
    return bool(_load().oracle_is_canonical(bits, spacer, word_bits, _pu8(w.view(np.uint8)), rows, inner))


def elementwise(op, x, y=None, *, bits: int, signed: bool, bits_o: int | None = None,
                signed_o: bool | None = None, shift: int = 0, saturate: bool = False) -> np.ndarray:
    """Lane-wise op on unpacked values (section 3 Figs. 5-6; ReLU/requantize per the header)."""
    if isinstance(op, str):
        op = OP_NAMES[op]
    xv = np.ascontiguousarray(np.asarray(x, dtype=np.int64)).ravel()
    yv = xv if y is None else np.ascontiguousarray(np.asarray(y, dtype=np.int64)).ravel()
    if yv.size != xv.size:
        raise OracleError("operand sizes differ")
    out = np.zeros_like(xv)
    bo = bits if bits_o is None else bits_o
    so = signed if signed_o is None else signed_o
    rc = _load().oracle_elementwise(op, bits, int(signed), bo, int(so), _p64(xv), _p64(yv), _p64(out), xv.size,
                                    shift, int(saturate))
    if rc:
        raise OracleError(f"oracle_elementwise failed ({rc})")
    return out


def requant(x, shift: int, bits_o: int, signed_o: bool) -> np.ndarray:
    """clamp_out(floor(x / 2^shift)) for int32 accumulators (the conv epilogue)."""
    return elementwise(REQUANT, x, bits=32, signed=True, bits_o=bits_o, signed_o=signed_o, shift=shift)


def conv2d(act_nchw, wt_mcrs, stride: int = 1, pad: int = 0, nthreads: int = 1, check_int32: bool = True):
    """Direct convolution (Fig. 12 loop nest) on unpacked CHW values; returns int64 NCHW."""
    a = np.ascontiguousarray(np.asarray(act_nchw, dtype=np.int64))
    w = np.ascontiguousarray(np.asarray(wt_mcrs, dtype=np.int64))
    N, C, H, W = a.shape
    M, C2, R, S = w.shape
    if C2 != C:
        raise OracleError("channel mismatch")
    Ho = (H + 2 * pad - R) // stride + 1
    Wo = (W + 2 * pad - S) // stride + 1
    out = np.zeros((N, M, Ho, Wo), dtype=np.int64)
    rc = _load().oracle_conv2d(N, C, H, W, M, R, S, stride, pad, _p64(a), _p64(w), _p64(out), nthreads)
    if rc == 7:
        if check_int32:
            raise Int32BoundError("an accumulator reached 2^31")
    elif rc:
        raise OracleError(f"oracle_conv2d failed ({rc})")
    return out


def maxpool2x2(x_nchw) -> np.ndarray:
    a = np.ascontiguousarray(np.asarray(x_nchw, dtype=np.int64))
    N, C, H, W = a.shape
    out = np.zeros((N, C, H // 2, W // 2), dtype=np.int64)
    rc = _load().oracle_maxpool2x2(N, C, H, W, _p64(a), _p64(out))
    if rc:
        raise OracleError(f"oracle_maxpool2x2 failed ({rc})")
    return out
