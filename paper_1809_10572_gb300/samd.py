"""Python binding of libsamd (argument marshalling only).

The functions named like the C ABI (samd_pack, samd_conv2d, ...) take torch
CUDA tensors, pass their device pointers and the current CUDA stream to the
library, and raise SamdError on a non-zero status. Every step of the
computation runs in libsamd's CUDA kernels; nothing here computes a result.
The helpers without the prefix (pack, conv2d, ...) only allocate the output
tensors with torch and call those bindings.

If libsamd.so is missing and cannot be built, load() raises: there is no
fallback.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

from . import build as _build

# ---- C types -----------------------------------------------------------------


class samd_fmt(ctypes.Structure):
    _fields_ = [("bits", ctypes.c_uint8), ("is_signed", ctypes.c_uint8), ("spacer", ctypes.c_uint8),
                ("word_bits", ctypes.c_uint8)]

    def __repr__(self):
        return f"samd_fmt(bits={self.bits}, is_signed={self.is_signed}, spacer={self.spacer}, word_bits={self.word_bits})"


class samd_conv_desc(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int), ("C", ctypes.c_int), ("H", ctypes.c_int), ("W", ctypes.c_int),
                ("K", ctypes.c_int), ("R", ctypes.c_int), ("S", ctypes.c_int), ("stride", ctypes.c_int),
                ("pad", ctypes.c_int), ("layout", ctypes.c_int)]


SAMD_OK, SAMD_EINVAL, SAMD_EALIGN, SAMD_ESHAPE, SAMD_EUNSUP, SAMD_ECUDA, SAMD_ETIMEOUT = range(7)
SAMD_ADD, SAMD_SUB, SAMD_MUL, SAMD_RELU, SAMD_REQUANT = range(5)
SAMD_NCHW, SAMD_NHWC = 0, 1
OPS = {"add": SAMD_ADD, "sub": SAMD_SUB, "mul": SAMD_MUL, "relu": SAMD_RELU, "requant": SAMD_REQUANT}

EXPORTED = ["samd_lanes_per_word", "samd_packed_words", "samd_pack", "samd_unpack", "samd_elementwise",
            "samd_conv2d", "samd_conv2d_workspace_size", "samd_conv2d_operand_bits", "samd_conv2d_set_min_tiles_per_cta", "samd_conv2d_prepare", "samd_conv2d_prepared",
            "samd_conv2d_noalloc", "samd_conv2d_prepared_pool2x2", "samd_conv2d_pool2x2_supported",
            "samd_maxpool2x2", "samd_device_status", "samd_selftest_wait_timeout", "samd_status_str", "samd_version"]
FMT_NONE = (0, 0, 0, 0)


class SamdError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {status_str(status)}")


_lib = None


def lib_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libsamd.so (building it in-tree first if it is missing or stale)."""
    global _lib
    if _lib is not None:
        return _lib
    if build_if_missing and not _build.up_to_date():
        _build.build()
    if not os.path.exists(_build.LIB):
        raise RuntimeError(f"libsamd.so not found at {_build.LIB}; the CUDA path has no fallback")
    lib = ctypes.CDLL(_build.LIB)
    c = ctypes
    vp, i64, i32, sz = c.c_void_p, c.c_int64, c.c_int, c.c_size_t
    lib.samd_lanes_per_word.argtypes, lib.samd_lanes_per_word.restype = [samd_fmt], sz
    lib.samd_packed_words.argtypes, lib.samd_packed_words.restype = [samd_fmt, i64, i64], i64
    lib.samd_pack.argtypes, lib.samd_pack.restype = [samd_fmt, vp, vp, i64, i64, vp], i32
    lib.samd_unpack.argtypes, lib.samd_unpack.restype = [samd_fmt, vp, vp, i64, i64, vp], i32
    lib.samd_elementwise.argtypes = [i32, samd_fmt, vp, vp, samd_fmt, vp, i64, i32, i32, vp]
    lib.samd_elementwise.restype = i32
    lib.samd_conv2d.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, vp, samd_fmt, vp, vp, samd_fmt, vp, i32, vp, sz,
                                vp]
    lib.samd_conv2d.restype = i32
    lib.samd_conv2d_noalloc.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, vp, samd_fmt, vp, vp, samd_fmt, vp, i32,
                                        vp]
    lib.samd_conv2d_noalloc.restype = i32
    lib.samd_conv2d_prepare.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, samd_fmt, vp, samd_fmt, vp, sz, vp]
    lib.samd_conv2d_prepare.restype = i32
    lib.samd_conv2d_prepared.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, vp, samd_fmt, vp, sz, vp, samd_fmt, vp,
                                         i32, vp]
    lib.samd_conv2d_prepared.restype = i32
    lib.samd_conv2d_prepared_pool2x2.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, vp, samd_fmt, vp, sz, samd_fmt,
                                                 vp, i32, vp]
    lib.samd_conv2d_prepared_pool2x2.restype = i32
    lib.samd_conv2d_pool2x2_supported.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, samd_fmt, samd_fmt]
    lib.samd_conv2d_pool2x2_supported.restype = i32
    lib.samd_conv2d_workspace_size.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, samd_fmt]
    lib.samd_conv2d_workspace_size.restype = sz
    lib.samd_conv2d_operand_bits.argtypes = [c.POINTER(samd_conv_desc), samd_fmt, samd_fmt]
    lib.samd_conv2d_operand_bits.restype = i32
    lib.samd_conv2d_set_min_tiles_per_cta.argtypes = [i32]
    lib.samd_conv2d_set_min_tiles_per_cta.restype = i32
    lib.samd_maxpool2x2.argtypes = [samd_fmt, vp, vp, i32, i32, i32, i32, i32, vp]
    lib.samd_maxpool2x2.restype = i32
    lib.samd_device_status.argtypes, lib.samd_device_status.restype = [c.POINTER(c.c_int), i32, vp], i32
    lib.samd_selftest_wait_timeout.argtypes, lib.samd_selftest_wait_timeout.restype = [c.c_uint64, vp], i32
    lib.samd_status_str.argtypes, lib.samd_status_str.restype = [i32], c.c_char_p
    lib.samd_version.argtypes, lib.samd_version.restype = [], c.c_char_p
    _lib = lib
    return lib


def status_str(status: int) -> str:
    return load().samd_status_str(status).decode()


def _check(status: int, what: str) -> None:
    if status != SAMD_OK:
        raise SamdError(status, what)


def _ptr(t):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        return t  # an integer address
    if not t.is_cuda:
        raise ValueError("libsamd takes device tensors")
    return t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


# ---- formats -------------------------------------------------------------------


def fmt(bits: int, signed: bool, spacer: int = 0, word_bits: int = 32) -> samd_fmt:
    return samd_fmt(bits, int(bool(signed)), spacer, word_bits)


def word_dtype(f: samd_fmt) -> torch.dtype:
    """torch dtype that stores one packed word (bit pattern)."""
    return torch.int32 if f.word_bits == 32 else torch.int64


def samd_lanes_per_word(f: samd_fmt) -> int:
    return int(load().samd_lanes_per_word(f))


def samd_packed_words(f: samd_fmt, rows: int, inner: int) -> int:
    return int(load().samd_packed_words(f, rows, inner))


# ---- the C ABI, one binding per entry point -------------------------------------


def samd_pack(f, src, dst, rows, inner, stream=None):
    _check(load().samd_pack(f, _ptr(src), _ptr(dst), rows, inner, _stream(stream)), "samd_pack")


def samd_unpack(f, src, dst, rows, inner, stream=None):
    _check(load().samd_unpack(f, _ptr(src), _ptr(dst), rows, inner, _stream(stream)), "samd_unpack")


def samd_elementwise(op, fa, a, b, fo, out, n, shift=0, saturate=0, stream=None):
    op = OPS[op] if isinstance(op, str) else op
    _check(load().samd_elementwise(op, fa, _ptr(a), _ptr(b), fo, _ptr(out), n, shift, int(saturate),
                                   _stream(stream)), "samd_elementwise")


def samd_conv2d_workspace_size(desc: samd_conv_desc, fa: samd_fmt, fw: samd_fmt) -> int:
    return int(load().samd_conv2d_workspace_size(ctypes.byref(desc), fa, fw))


def samd_conv2d_set_min_tiles_per_cta(tiles: int) -> None:
    """Minimum 128-pixel tiles per SM of a convolution launch (1: spread each layer
    over every SM; larger: leave SMs to layers running on other streams)."""
    _check(load().samd_conv2d_set_min_tiles_per_cta(int(tiles)), "samd_conv2d_set_min_tiles_per_cta")


def samd_conv2d_operand_bits(desc: samd_conv_desc, fa: samd_fmt, fw: samd_fmt) -> int:
    """8 (e4m3) or 16 (fp16): the tensor-core operand type of this convolution; 0 if rejected."""
    return int(load().samd_conv2d_operand_bits(ctypes.byref(desc), fa, fw))


def samd_conv2d(desc, fa, act, fw, wt, acc_out, fo, packed_out, shift, workspace, workspace_bytes=None,
                stream=None):
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size() if isinstance(workspace, torch.Tensor) else 0
    _check(load().samd_conv2d(ctypes.byref(desc), fa, _ptr(act), fw, _ptr(wt), _ptr(acc_out),
                              fo if fo is not None else samd_fmt(8, 1, 0, 32), _ptr(packed_out), shift,
                              _ptr(workspace), workspace_bytes, _stream(stream)), "samd_conv2d")


def samd_conv2d_noalloc(desc, fa, act, fw, wt, acc_out, fo, packed_out, shift, stream=None):
    """samd_conv2d without a workspace (the library's static scratch holds the widened weights)."""
    _check(load().samd_conv2d_noalloc(ctypes.byref(desc), fa, _ptr(act), fw, _ptr(wt), _ptr(acc_out),
                                      fo if fo is not None else samd_fmt(8, 1, 0, 32), _ptr(packed_out), shift,
                                      _stream(stream)), "samd_conv2d_noalloc")


def _nbytes(t):
    return t.numel() * t.element_size() if isinstance(t, torch.Tensor) else 0


def samd_conv2d_prepare(desc, fa, fw, wt, fo, prepared, prepared_bytes=None, stream=None):
    fo = fo if fo is not None else samd_fmt(*FMT_NONE)
    nb = _nbytes(prepared) if prepared_bytes is None else prepared_bytes
    _check(load().samd_conv2d_prepare(ctypes.byref(desc), fa, fw, _ptr(wt), fo, _ptr(prepared), nb, _stream(stream)),
           "samd_conv2d_prepare")


def samd_conv2d_prepared(desc, fa, act, fw, prepared, acc_out, fo, packed_out, shift, prepared_bytes=None,
                         stream=None):
    fo = fo if fo is not None else samd_fmt(*FMT_NONE)
    nb = _nbytes(prepared) if prepared_bytes is None else prepared_bytes
    _check(load().samd_conv2d_prepared(ctypes.byref(desc), fa, _ptr(act), fw, _ptr(prepared), nb, _ptr(acc_out), fo,
                                       _ptr(packed_out), shift, _stream(stream)), "samd_conv2d_prepared")


def samd_conv2d_prepared_pool2x2(desc, fa, act, fw, prepared, fo, pooled_out, shift, prepared_bytes=None,
                                 stream=None):
    nb = _nbytes(prepared) if prepared_bytes is None else prepared_bytes
    _check(load().samd_conv2d_prepared_pool2x2(ctypes.byref(desc), fa, _ptr(act), fw, _ptr(prepared), nb, fo,
                                               _ptr(pooled_out), shift, _stream(stream)),
           "samd_conv2d_prepared_pool2x2")


def samd_conv2d_pool2x2_supported(desc, fa, fw, fo) -> bool:
    return bool(load().samd_conv2d_pool2x2_supported(ctypes.byref(desc), fa, fw, fo))


def samd_maxpool2x2(f, inp, out, N, C, H, W, layout=SAMD_NHWC, stream=None):
    _check(load().samd_maxpool2x2(f, _ptr(inp), _ptr(out), N, C, H, W, layout, _stream(stream)),
           "samd_maxpool2x2")


def samd_device_status(reset: bool = False, stream=None) -> int:
    v = ctypes.c_int(0)
    _check(load().samd_device_status(ctypes.byref(v), int(reset), _stream(stream)), "samd_device_status")
    return v.value


def samd_selftest_wait_timeout(limit_ns: int, stream=None) -> None:
    _check(load().samd_selftest_wait_timeout(limit_ns, _stream(stream)), "samd_selftest_wait_timeout")


def samd_version() -> str:
    return load().samd_version().decode()


# ---- allocating helpers ---------------------------------------------------------


def empty_words(f: samd_fmt, rows: int, inner: int, device="cuda") -> torch.Tensor:
    n = samd_packed_words(f, rows, inner)
    if n < 0:
        raise ValueError(f"bad format {f}")
    return torch.empty(max(n, 1), dtype=word_dtype(f), device=device)[:n]


def pack(x: torch.Tensor, f: samd_fmt, rows: int | None = None, inner: int | None = None, stream=None):
    """int8 tensor (rows x inner, row-major) -> packed words."""
    x = x.contiguous()
    if rows is None:
        inner = x.shape[-1] if x.dim() else 1
        rows = x.numel() // max(inner, 1)
    out = empty_words(f, rows, inner, x.device)
    samd_pack(f, x, out, rows, inner, stream)
    return out


def unpack(words: torch.Tensor, f: samd_fmt, rows: int, inner: int, stream=None) -> torch.Tensor:
    out = torch.empty(rows * inner, dtype=torch.int8, device=words.device)
    samd_unpack(f, words, out, rows, inner, stream)
    return out.view(rows, inner)


def elementwise(op, a, b, fa: samd_fmt, n: int, fo: samd_fmt | None = None, shift: int = 0, saturate: bool = False,
                out=None, stream=None):
    fo = fa if fo is None else fo
    if out is None:
        out = empty_words(fo, 1, n, a.device)
    samd_elementwise(op, fa, a, b, fo, out, n, shift, saturate, stream)
    return out


@dataclass
class ConvShape:
    N: int
    C: int
    H: int
    W: int
    K: int
    R: int = 3
    S: int = 3
    stride: int = 1
    pad: int = 1

    @property
    def Ho(self):
        return (self.H + 2 * self.pad - self.R) // self.stride + 1

    @property
    def Wo(self):
        return (self.W + 2 * self.pad - self.S) // self.stride + 1

    @property
    def macs(self) -> int:
        return self.N * self.Ho * self.Wo * self.K * self.C * self.R * self.S

    def desc(self, layout=SAMD_NHWC) -> samd_conv_desc:
        return samd_conv_desc(self.N, self.C, self.H, self.W, self.K, self.R, self.S, self.stride, self.pad, layout)


def conv_workspace(shape: ConvShape, fa: samd_fmt, fw: samd_fmt, device="cuda") -> torch.Tensor:
    nbytes = samd_conv2d_workspace_size(shape.desc(), fa, fw)
    if nbytes == 0:
        raise ValueError("invalid convolution shape or format")
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def conv2d(act, wt, shape: ConvShape, fa: samd_fmt, fw: samd_fmt, fo: samd_fmt | None = None, shift: int = 0,
           want_acc: bool = True, workspace=None, stream=None):
    """NHWC packed conv; returns (int32 acc [N,Ho,Wo,K] or None, packed output words or None)."""
    dev = act.device
    acc = torch.empty((shape.N, shape.Ho, shape.Wo, shape.K), dtype=torch.int32, device=dev) if want_acc else None
    packed = empty_words(fo, shape.N * shape.Ho * shape.Wo, shape.K, dev) if fo is not None else None
    if workspace is None:
        workspace = conv_workspace(shape, fa, fw, dev)
    samd_conv2d(shape.desc(), fa, act, fw, wt, acc, fo, packed, shift, workspace, stream=stream)
    return acc, packed


def conv2d_nchw(act, wt, shape: ConvShape, fa: samd_fmt, fw: samd_fmt, fo: samd_fmt | None = None, shift: int = 0,
                want_acc: bool = True, workspace=None, stream=None):
    """NCHW packed along W (rows of W lanes; weights [K][C][R] rows of S lanes);
    returns (int32 acc [N,K,Ho,Wo] or None, packed output rows of Wo lanes or None)."""
    dev = act.device
    desc = shape.desc(SAMD_NCHW)
    acc = torch.empty((shape.N, shape.K, shape.Ho, shape.Wo), dtype=torch.int32, device=dev) if want_acc else None
    packed = empty_words(fo, shape.N * shape.K * shape.Ho, shape.Wo, dev) if fo is not None else None
    if workspace is None:
        nbytes = samd_conv2d_workspace_size(desc, fa, fw)
        if nbytes == 0:
            raise SamdError(SAMD_EUNSUP, "samd_conv2d_workspace_size")
        workspace = torch.empty(nbytes, dtype=torch.uint8, device=dev)
    samd_conv2d(desc, fa, act, fw, wt, acc, fo, packed, shift, workspace, stream=stream)
    return acc, packed


class PreparedConv:
    """A convolution layer whose weights were widened once (samd_conv2d_prepare)."""

    def __init__(self, wt_words, shape: ConvShape, fa: samd_fmt, fw: samd_fmt, fo: samd_fmt | None = None,
                 stream=None):
        self.shape, self.fa, self.fw, self.fo = shape, fa, fw, fo
        self.prepared = conv_workspace(shape, fa, fw, wt_words.device)
        samd_conv2d_prepare(shape.desc(), fa, fw, wt_words, fo, self.prepared, stream=stream)

    def __call__(self, act, acc_out=None, packed_out=None, shift: int = 0, stream=None):
        samd_conv2d_prepared(self.shape.desc(), self.fa, act, self.fw, self.prepared, acc_out, self.fo, packed_out,
                             shift, stream=stream)
        return acc_out, packed_out

    def pool2x2_supported(self) -> bool:
        return self.fo is not None and samd_conv2d_pool2x2_supported(self.shape.desc(), self.fa, self.fw, self.fo)

    def pool2x2(self, act, pooled_out, shift: int = 0, stream=None):
        """The convolution with the 2x2 max-pool of its packed output fused
        (samd_conv2d_prepared_pool2x2)."""
        samd_conv2d_prepared_pool2x2(self.shape.desc(), self.fa, act, self.fw, self.prepared, self.fo, pooled_out,
                                     shift, stream=stream)
        return pooled_out

    def outputs(self, want_acc=True, want_packed=True, device="cuda"):
        s = self.shape
        acc = torch.empty((s.N, s.Ho, s.Wo, s.K), dtype=torch.int32, device=device) if want_acc else None
        packed = empty_words(self.fo, s.N * s.Ho * s.Wo, s.K, device) if (want_packed and self.fo) else None
        return acc, packed


def maxpool2x2(words, f: samd_fmt, N: int, C: int, H: int, W: int, stream=None):
    out = empty_words(f, N * (H // 2) * (W // 2), C, words.device)
    samd_maxpool2x2(f, words, out, N, C, H, W, SAMD_NHWC, stream)
    return out
