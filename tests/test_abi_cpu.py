"""The C-ABI library loads and exports every entry point include/samd.h
declares; host-only queries and argument checks answer without a GPU (no
compute call is made here)."""
import ctypes
import os
import re

import pytest

from paper_1809_10572_gb300 import build, samd

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "samd.h")


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"SAMD_API[^;(]*?\b(samd_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    return samd.load()


def test_header_declares_the_boundary():
    names = declared_symbols()
    for required in ("samd_pack", "samd_unpack", "samd_elementwise", "samd_conv2d", "samd_maxpool2x2"):
        assert required in names
    assert sorted(samd.EXPORTED) == names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


def test_library_is_built_in_tree_for_sm103a():
    assert os.path.dirname(build.LIB).startswith(os.path.dirname(os.path.abspath(build.__file__)))
    assert "arch=compute_103a,code=sm_103a" in build.ARCH


def test_format_queries(lib):
    for bits in range(1, 9):
        for wb in (32, 64):
            assert samd.samd_lanes_per_word(samd.fmt(bits, True, 0, wb)) == wb // bits
            assert samd.samd_lanes_per_word(samd.fmt(bits, False, 1, wb)) == wb // (bits + 1)
    f = samd.fmt(3, False)
    assert samd.samd_packed_words(f, 7, 64) == 7 * 7
    assert samd.samd_packed_words(f, 0, 64) == 0
    assert samd.samd_packed_words(samd.fmt(9, False), 1, 1) == -1
    assert samd.samd_packed_words(samd.fmt(4, False, 0, 16), 1, 1) == -1
    assert samd.samd_lanes_per_word(samd.fmt(0, False)) == 0


def test_invalid_arguments_are_rejected_before_any_launch(lib):
    bad = samd.fmt(9, False)
    assert lib.samd_pack(bad, None, None, 1, 1, None) == samd.SAMD_EINVAL
    assert lib.samd_unpack(samd.fmt(4, False), None, None, -1, 4, None) == samd.SAMD_ESHAPE
    assert lib.samd_pack(samd.fmt(4, False), None, None, 0, 5, None) == samd.SAMD_OK  # empty: nothing to do
    assert lib.samd_pack(samd.fmt(4, False), None, None, 1, 5, None) == samd.SAMD_EINVAL
    assert lib.samd_pack(samd.fmt(4, False), 16, 17, 1, 5, None) == samd.SAMD_EALIGN
    f4 = samd.fmt(4, True)
    assert lib.samd_elementwise(7, f4, None, None, f4, None, 1, 0, 0, None) == samd.SAMD_EINVAL
    assert lib.samd_elementwise(samd.SAMD_ADD, f4, None, None, samd.fmt(3, True), None, 1, 0, 0, None) == samd.SAMD_EINVAL
    assert lib.samd_elementwise(samd.SAMD_REQUANT, f4, None, None, f4, None, 1, 32, 0, None) == samd.SAMD_EINVAL
    assert lib.samd_elementwise(samd.SAMD_ADD, f4, 16, None, f4, 16, 8, 0, 0, None) == samd.SAMD_EINVAL
    assert lib.samd_elementwise(samd.SAMD_ADD, f4, 16, 32, f4, 8, 8, 0, 0, None) == samd.SAMD_EALIGN
    assert lib.samd_maxpool2x2(f4, None, None, 1, 4, 3, 4, samd.SAMD_NHWC, None) == samd.SAMD_ESHAPE
    assert lib.samd_maxpool2x2(f4, 16, 16, 1, 4, 4, 4, samd.SAMD_NCHW, None) == samd.SAMD_EUNSUP
    assert lib.samd_status_str(samd.SAMD_EUNSUP).startswith(b"SAMD_EUNSUP")


def test_conv_argument_checks(lib):
    fa, fw = samd.fmt(4, False), samd.fmt(4, True)
    d = samd.ConvShape(1, 16, 8, 8, 16).desc()
    assert lib.samd_conv2d(None, fa, 16, fw, 16, 16, fa, None, 0, 16, 1 << 20, None) == samd.SAMD_EINVAL
    assert lib.samd_conv2d(ctypes.byref(d), fa, 16, fw, 16, None, fa, None, 0, 16, 1 << 20, None) == samd.SAMD_EINVAL
    # NCHW (the wide-multiply engine): stride 1 only; pointers checked before any launch
    nchw = samd.ConvShape(1, 16, 8, 8, 16).desc(samd.SAMD_NCHW)
    assert lib.samd_conv2d(ctypes.byref(nchw), fa, 16, fw, 24, 16, fa, None, 0, 16, 1 << 20, None) == samd.SAMD_EALIGN
    nchw2 = samd.ConvShape(1, 16, 8, 8, 16, stride=2).desc(samd.SAMD_NCHW)
    assert lib.samd_conv2d(ctypes.byref(nchw2), fa, 16, fw, 16, 16, fa, None, 0, 16, 1 << 20, None) == samd.SAMD_EUNSUP
    assert lib.samd_conv2d_prepare(ctypes.byref(nchw), fa, fw, 16, fa, 16, 1 << 20, None) == samd.SAMD_EUNSUP
    bad = samd.ConvShape(1, 16, 2, 2, 16, R=5, S=5, pad=1).desc()
    assert lib.samd_conv2d(ctypes.byref(bad), fa, 16, fw, 16, 16, fa, None, 0, 16, 1 << 20, None) == samd.SAMD_ESHAPE
    # u8 x s8 over 3x3x512 taps: even split weight digits exceed 2^24 (4608 * 255 * 16)
    big = samd.ConvShape(1, 512, 8, 8, 16).desc()
    u8, s8, u4 = samd.fmt(8, False), samd.fmt(8, True), samd.fmt(4, False)
    assert lib.samd_conv2d(ctypes.byref(big), u8, 16, s8, 16, 16, u8, None, 0, 16, 1 << 20, None) == samd.SAMD_EUNSUP
    # 4-bit weights are not split: 4608 * 255 * 15 >= 2^24
    assert lib.samd_conv2d(ctypes.byref(big), u8, 16, u4, 16, 16, u8, None, 0, 16, 1 << 20, None) == samd.SAMD_EUNSUP
    assert lib.samd_conv2d_prepare(ctypes.byref(big), u8, s8, 16, u8, 16, 1 << 20, None) == samd.SAMD_EUNSUP
    # the 3x3 x 64-channel u8 x u8 layer fits with split digits: rejected here only for the misaligned pointer
    mid = samd.ConvShape(1, 64, 8, 8, 16).desc()
    assert lib.samd_conv2d(ctypes.byref(mid), u8, 16, u8, 24, 16, u8, None, 0, 16, 1 << 20, None) == samd.SAMD_EALIGN
    assert lib.samd_conv2d(ctypes.byref(d), fa, 16, fw, 24, 16, fa, None, 0, 16, 1 << 20, None) == samd.SAMD_EALIGN
    assert lib.samd_conv2d_prepared(ctypes.byref(d), fa, 16, fw, 16, 1 << 20, None, fa, None, 0, None) == samd.SAMD_EINVAL
    assert lib.samd_conv2d_prepared(ctypes.byref(d), fa, 16, fw, 16, 1 << 20, None, samd.samd_fmt(0, 0, 0, 0), 16, 0,
                                    None) == samd.SAMD_EINVAL
    assert samd.samd_conv2d_workspace_size(d, fa, fw) > 0
    assert samd.samd_conv2d_workspace_size(samd.ConvShape(1, 0, 8, 8, 16).desc(), fa, fw) == 0


def test_conv_operand_type_query(lib):
    """e4m3 holds every integer of [-16, 16] exactly (sign, 4 exponent bits,
    3 mantissa bits: 16 = 1.000b x 2^4, 15 = 1.111b x 2^3), so lanes with
    max|a|, max|w| <= 16 are contracted on e4m3 operands; every other format
    (and every split-digit layer) on fp16."""
    d = samd.ConvShape(2, 64, 16, 16, 64).desc()
    bits = lambda ba, sa, bw, sw, desc=d: samd.samd_conv2d_operand_bits(desc, samd.fmt(ba, sa), samd.fmt(bw, sw))
    for b in (1, 2, 3, 4):
        for sa in (False, True):
            for sw in (False, True):
                assert bits(b, sa, b, sw) == 8
    assert bits(5, True, 5, True) == 8      # [-16, 15]
    assert bits(5, False, 4, True) == 16    # 31 > 16
    assert bits(4, False, 5, False) == 16
    assert bits(6, False, 2, True) == 16
    assert bits(8, False, 8, True) == 16    # split digits
    assert bits(8, False, 8, True, samd.ConvShape(1, 512, 8, 8, 16).desc()) == 0  # SAMD_EUNSUP
    assert samd.samd_conv2d_operand_bits(d, samd.fmt(4, False, spacer=1), samd.fmt(4, True)) == 0
    assert samd.samd_conv2d_operand_bits(samd.ConvShape(1, 0, 8, 8, 16).desc(), samd.fmt(4, False),
                                         samd.fmt(4, True)) == 0


def test_nchw_wide_multiply_plan():
    """Section 5.1 engine: fields of F = bits(R*S*C*max|a|*max|w|) + 1 bits,
    nx = floor(64 / F) inputs per word, the kernel row in one word (S*F <= 64).
    u4 x s4 over 3x3x16: bound 17280 (15 bits) -> F = 16, nx = 4; an 8-wide
    output row needs the 10 coefficients of the full 1D convolution, G = 3
    words per input row. Workspace: 8 bytes x (N*C*H*G + K*C*R)."""
    fa, fw = samd.fmt(4, False), samd.fmt(4, True)
    d = samd.ConvShape(1, 16, 8, 8, 16).desc(samd.SAMD_NCHW)
    assert samd.samd_conv2d_workspace_size(d, fa, fw) == 8 * (1 * 16 * 8 * 3 + 16 * 16 * 3)
    assert samd.samd_conv2d_operand_bits(d, fa, fw) == 64
    # u8 x s8 over 3x3x64: bound 576 * 255 * 128 = 18.8 M (25 bits) -> F = 26, 3 x 26 > 64
    big = samd.ConvShape(1, 64, 8, 8, 16).desc(samd.SAMD_NCHW)
    assert samd.samd_conv2d_operand_bits(big, samd.fmt(8, False), samd.fmt(8, True)) == 0
    assert samd.samd_conv2d_workspace_size(big, samd.fmt(8, False), samd.fmt(8, True)) == 0
    # the same sums over 1x2 kernels fit (2 x 26 <= 64)
    ok = samd.ConvShape(1, 64, 8, 8, 16, R=1, S=2, pad=0).desc(samd.SAMD_NCHW)
    assert samd.samd_conv2d_operand_bits(ok, samd.fmt(8, False), samd.fmt(8, True)) == 64


def test_min_tiles_per_cta_setting(lib):
    assert lib.samd_conv2d_set_min_tiles_per_cta(0) == samd.SAMD_EINVAL
    assert lib.samd_conv2d_set_min_tiles_per_cta(1025) == samd.SAMD_EINVAL
    assert lib.samd_conv2d_set_min_tiles_per_cta(8) == samd.SAMD_OK
    assert lib.samd_conv2d_set_min_tiles_per_cta(4) == samd.SAMD_OK  # the default again


def test_fused_pool_support_query(lib):
    # host-only: which layers samd_conv2d_prepared_pool2x2 runs (halo tiles
    # holding whole pairs of padded rows, even outputs, 1/2/4/8-bit outputs
    # in 32-bit words without spacers)
    from paper_1809_10572_gb300 import workloads

    fa, fw, u4 = samd.fmt(4, False), samd.fmt(4, True), samd.fmt(4, False)
    got = {l.name: samd.samd_conv2d_pool2x2_supported(l.shape.desc(), fa, fw, u4)
           for l in workloads.vgg16() if l.pool_after}
    assert got == {"conv2": False, "conv4": True, "conv7": True, "conv10": True}  # conv2: 2 (224 + 2) > 256
    s = samd.ConvShape(2, 64, 56, 56, 64)
    assert samd.samd_conv2d_pool2x2_supported(s.desc(), fa, fw, u4)
    for fo in (samd.fmt(1, False), samd.fmt(2, True), samd.fmt(8, True)):
        assert samd.samd_conv2d_pool2x2_supported(s.desc(), fa, fw, fo)
    for fo in (samd.fmt(3, False), samd.fmt(4, False, spacer=1), samd.fmt(4, False, word_bits=64),
               samd.fmt(*samd.FMT_NONE)):
        assert not samd.samd_conv2d_pool2x2_supported(s.desc(), fa, fw, fo)
    for bad in (samd.ConvShape(2, 64, 56, 57, 64), samd.ConvShape(2, 64, 56, 56, 64, stride=2),
                samd.ConvShape(2, 64, 8, 8, 64)):
        assert not samd.samd_conv2d_pool2x2_supported(bad.desc(), fa, fw, u4)
    assert not samd.samd_conv2d_pool2x2_supported(s.desc(samd.SAMD_NCHW), fa, fw, u4)
