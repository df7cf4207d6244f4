"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle, bit
for bit, on seeded inputs that span several tiles and a ragged tail."""
import itertools

import numpy as np
import pytest
import torch

import oracle
from gpu_util import (assert_status_clean, conv_case, conv_supported, gpu_pack, harness_shift, np_words,
                      oracle_conv_nhwc, oracle_requant_pack, values_and_bytes)
from paper_1809_10572_gb300 import samd, synth

pytestmark = pytest.mark.gpu

BITS = range(1, 9)
SIGNS = (False, True)


# ---- pack / unpack ---------------------------------------------------------------

def pack_shapes(L):
    return [(1, 3 * L * 256 + 7), (1, L - 1), (1, 1), (37, 64), (5, 2 * L + 3), (9, L), (4, 1)]


@pytest.mark.parametrize("word_bits", (32, 64))
@pytest.mark.parametrize("spacer", (0, 1, 3))
@pytest.mark.parametrize("signed", SIGNS)
@pytest.mark.parametrize("bits", BITS)
def test_pack_unpack(samd_lib, bits, signed, spacer, word_bits):
    f = samd.fmt(bits, signed, spacer, word_bits)
    L = samd.samd_lanes_per_word(f)
    for rows, inner in pack_shapes(L):
        v, b = values_and_bytes(synth.seed_for("pk", bits, signed, spacer, word_bits, rows, inner), (rows, inner),
                                bits, signed)
        got = gpu_pack(b, f, rows, inner)
        want = oracle.pack(v, bits, signed, spacer, word_bits)
        assert np.array_equal(np_words(got, word_bits), want), (rows, inner)
        # unpack the oracle's words
        words = torch.from_numpy(want.view(np.int32 if word_bits == 32 else np.int64)).cuda()
        back = samd.unpack(words, f, rows, inner).cpu().numpy().astype(np.int64)
        expect = ((v & 0xFF) ^ 0x80) - 0x80  # the value as a byte (uint8 pattern for unsigned 8-bit)
        assert np.array_equal(back, expect)
    assert_status_clean()


def test_pack_keeps_low_bits(samd_lib):
    f = samd.fmt(4, False)
    b = torch.tensor([[16, -1, 17, 0x7F]], dtype=torch.int8).cuda()
    got = np_words(gpu_pack(b, f, 1, 4), 32)
    assert np.array_equal(got, oracle.pack(np.array([[16, -1, 17, 0x7F]]), 4, False))


# ---- elementwise ------------------------------------------------------------------

N_EW = [70001, 1, 13]


@pytest.mark.parametrize("word_bits", (32, 64))
@pytest.mark.parametrize("signed", SIGNS)
@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("op", ("add", "sub", "mul"))
def test_binary_ops(samd_lib, op, bits, signed, word_bits):
    f = samd.fmt(bits, signed, 0, word_bits)
    for n, sat in itertools.product(N_EW, (False, True)):
        xv, xb = values_and_bytes(synth.seed_for("x", op, bits, signed, n), (n,), bits, signed)
        yv, yb = values_and_bytes(synth.seed_for("y", op, bits, signed, n), (n,), bits, signed)
        xw, yw = gpu_pack(xb, f, 1, n), gpu_pack(yb, f, 1, n)
        got = samd.elementwise(op, xw, yw, f, n, saturate=sat)
        want_v = oracle.elementwise(op, xv, yv, bits=bits, signed=signed, saturate=sat)
        want = oracle.pack(want_v, bits, signed, 0, word_bits)
        assert np.array_equal(np_words(got, word_bits), want), (n, sat)
    assert_status_clean()


@pytest.mark.parametrize("word_bits", (32, 64))
@pytest.mark.parametrize("signed", SIGNS)
@pytest.mark.parametrize("bits", BITS)
def test_relu_and_requant_same_format(samd_lib, bits, signed, word_bits):
    f = samd.fmt(bits, signed, 0, word_bits)
    for n in N_EW:
        xv, xb = values_and_bytes(synth.seed_for("r", bits, signed, n), (n,), bits, signed)
        xw = gpu_pack(xb, f, 1, n)
        got = samd.elementwise("relu", xw, None, f, n)
        want = oracle.pack(oracle.elementwise("relu", xv, bits=bits, signed=signed), bits, signed, 0, word_bits)
        assert np.array_equal(np_words(got, word_bits), want)
        for shift in range(0, bits + 2):
            got = samd.elementwise("requant", xw, None, f, n, shift=shift)
            want_v = oracle.elementwise("requant", xv, bits=bits, signed=signed, bits_o=bits, signed_o=signed,
                                        shift=shift)
            assert np.array_equal(np_words(got, word_bits), oracle.pack(want_v, bits, signed, 0, word_bits)), shift
    assert_status_clean()


@pytest.mark.parametrize("fa_t,fo_t", [
    ((8, True, 0, 32), (4, True, 0, 32)), ((8, True, 0, 32), (4, False, 0, 32)), ((3, False, 0, 32), (6, True, 0, 64)),
    ((6, True, 0, 64), (2, True, 0, 32)), ((5, True, 1, 32), (5, True, 0, 32)), ((4, False, 2, 64), (1, False, 1, 32)),
])
def test_requant_format_change(samd_lib, fa_t, fo_t):
    fa, fo = samd.fmt(*fa_t), samd.fmt(*fo_t)
    for n in (50003, 7):
        xv, xb = values_and_bytes(synth.seed_for("rq", fa_t, fo_t, n), (n,), fa.bits, bool(fa.is_signed))
        xw = gpu_pack(xb, fa, 1, n)
        for shift in (0, 1, 3, 9):
            got = samd.elementwise("requant", xw, None, fa, n, fo=fo, shift=shift)
            want_v = oracle.elementwise("requant", xv, bits=fa.bits, signed=bool(fa.is_signed), bits_o=fo.bits,
                                        signed_o=bool(fo.is_signed), shift=shift)
            want = oracle.pack(want_v, fo.bits, bool(fo.is_signed), fo.spacer, fo.word_bits)
            assert np.array_equal(np_words(got, fo.word_bits), want)
    assert_status_clean()


@pytest.mark.parametrize("spacer", (1, 2, 4))
@pytest.mark.parametrize("op", ("add", "sub", "mul", "relu"))
def test_ops_with_spacer_bits(samd_lib, op, spacer):
    for bits, signed, word_bits in [(3, True, 32), (4, False, 64), (7, True, 32), (1, False, 32), (2, True, 32),
                                    (2, False, 64), (1, True, 32), (8, False, 64), (5, True, 64), (4, True, 32),
                                    (5, False, 32), (6, True, 32)]:
        f = samd.fmt(bits, signed, spacer, word_bits)
        n = 30011
        xv, xb = values_and_bytes(synth.seed_for("sx", op, bits, spacer), (n,), bits, signed)
        yv, yb = values_and_bytes(synth.seed_for("sy", op, bits, spacer), (n,), bits, signed)
        xw, yw = gpu_pack(xb, f, 1, n), gpu_pack(yb, f, 1, n)
        for sat in (False, True):
            got = samd.elementwise(op, xw, yw if op != "relu" else None, f, n, saturate=sat and op != "relu")
            want_v = oracle.elementwise(op, xv, yv, bits=bits, signed=signed, saturate=sat and op != "relu")
            assert np.array_equal(np_words(got, word_bits), oracle.pack(want_v, bits, signed, spacer, word_bits))
    assert_status_clean()


@pytest.mark.parametrize("spacer", (1, 2, 5))
@pytest.mark.parametrize("bits,signed,word_bits", [(1, False, 32), (3, True, 32), (4, False, 64), (7, True, 32),
                                                   (8, True, 64), (2, True, 32)])
def test_requant_same_format_with_spacer_bits(samd_lib, bits, signed, word_bits, spacer):
    f = samd.fmt(bits, signed, spacer, word_bits)
    n = 20011
    xv, xb = values_and_bytes(synth.seed_for("rqs", bits, signed, spacer, word_bits), (n,), bits, signed)
    xw = gpu_pack(xb, f, 1, n)
    for shift in range(0, bits + 2):
        got = samd.elementwise("requant", xw, None, f, n, shift=shift)
        want_v = oracle.elementwise("requant", xv, bits=bits, signed=signed, bits_o=bits, signed_o=signed, shift=shift)
        assert np.array_equal(np_words(got, word_bits), oracle.pack(want_v, bits, signed, spacer, word_bits)), shift
    got = samd.elementwise("relu", xw, None, f, n)
    want = oracle.pack(oracle.elementwise("relu", xv, bits=bits, signed=signed), bits, signed, spacer, word_bits)
    assert np.array_equal(np_words(got, word_bits), want)
    assert_status_clean()


def test_elementwise_in_place(samd_lib):
    f = samd.fmt(4, True)
    n = 4099
    xv, xb = values_and_bytes(11, (n,), 4, True)
    yv, yb = values_and_bytes(12, (n,), 4, True)
    xw, yw = gpu_pack(xb, f, 1, n), gpu_pack(yb, f, 1, n)
    samd.samd_elementwise("add", f, xw, yw, f, xw, n)
    want = oracle.pack(oracle.elementwise("add", xv, yv, bits=4, signed=True), 4, True)
    assert np.array_equal(np_words(xw, 32), want)


# ---- max-pool -----------------------------------------------------------------------

@pytest.mark.parametrize("spacer", (0, 1))
@pytest.mark.parametrize("word_bits", (32, 64))
@pytest.mark.parametrize("signed", SIGNS)
@pytest.mark.parametrize("bits", BITS)
def test_maxpool(samd_lib, bits, signed, word_bits, spacer):
    f = samd.fmt(bits, signed, spacer, word_bits)
    for N, C, H, W in [(2, 13, 6, 10), (1, 64, 8, 8), (3, 1, 2, 2)]:
        v, b = values_and_bytes(synth.seed_for("mp", bits, signed, C), (N, H, W, C), bits, signed)
        w = gpu_pack(b, f, N * H * W, C)
        got = samd.maxpool2x2(w, f, N, C, H, W)
        want_v = oracle.maxpool2x2(v.transpose(0, 3, 1, 2)).transpose(0, 2, 3, 1)
        want = oracle.pack(want_v.reshape(-1, C), bits, signed, spacer, word_bits)
        assert np.array_equal(np_words(got, word_bits), want)
    assert_status_clean()


# ---- convolution ---------------------------------------------------------------------

def run_conv_check(shape, ba, sa, bw, sw, word_bits=32, fo_t=None, shift=None, seed=0, act_gen=None, wt_gen=None):
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, ba, sa, bw, sw, seed, word_bits, act_gen, wt_gen)
    fo = samd.fmt(*fo_t) if fo_t else None
    if shift is None:
        shift = harness_shift(ba, bw, fo.bits if fo else 8, shape.C * shape.R * shape.S)
    acc, packed = samd.conv2d(a_w, w_w, shape, fa, fw, fo, shift=shift)
    torch.cuda.synchronize()
    want = oracle_conv_nhwc(a_v, w_v, shape)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
    if fo is not None:
        assert np.array_equal(np_words(packed, fo.word_bits), oracle_requant_pack(want, shift, fo))
    assert_status_clean()


def test_conv_single_layer_c16_u4_s4_64bit_words(samd_lib):
    # N1 C16 -> 16, 32x32, 3x3 s1 p1; u4 activations, s4 weights, 16 lanes per 64-bit word; seed 0
    run_conv_check(samd.ConvShape(1, 16, 32, 32, 16), 4, False, 4, True, word_bits=64, seed=0)


CONV_SHAPES = [
    samd.ConvShape(2, 64, 9, 11, 64),             # M = 198: one full tile and a ragged one
    samd.ConvShape(1, 3, 17, 13, 64),             # three input channels (first VGG layer shape)
    samd.ConvShape(2, 67, 7, 6, 40),              # C and K off every multiple
    samd.ConvShape(1, 32, 15, 15, 48, stride=2),  # stride 2
    samd.ConvShape(3, 96, 5, 7, 24, R=1, S=1, pad=0),  # 1x1
    samd.ConvShape(1, 16, 12, 12, 32, R=5, S=5, pad=2),
    samd.ConvShape(1, 128, 6, 6, 300, R=1, S=1, pad=0),  # more than 256 output channels: two channel blocks
]


@pytest.mark.parametrize("shape", CONV_SHAPES, ids=lambda s: f"{s.N}x{s.C}x{s.H}x{s.W}-K{s.K}-{s.R}x{s.S}s{s.stride}")
@pytest.mark.parametrize("ba,sa,bw,sw", [(4, False, 4, True), (2, True, 6, False), (3, True, 3, True),
                                         (1, False, 1, True), (7, False, 5, True), (8, True, 8, True)])
def test_conv_shapes(samd_lib, shape, ba, sa, bw, sw):
    assert conv_supported(shape, ba, sa, bw, sw)
    run_conv_check(shape, ba, sa, bw, sw, fo_t=(ba, sa, 0, 32), seed=synth.seed_for(shape, ba, sa, bw, sw))


@pytest.mark.parametrize("word_bits", (32, 64))
@pytest.mark.parametrize("sw", SIGNS)
@pytest.mark.parametrize("sa", SIGNS)
@pytest.mark.parametrize("bits", BITS)
def test_conv_every_width_and_sign(samd_lib, bits, sa, sw, word_bits):
    shape = samd.ConvShape(2, 24, 10, 9, 32)
    assert conv_supported(shape, bits, sa, bits, sw)
    run_conv_check(shape, bits, sa, bits, sw, word_bits=word_bits, fo_t=(bits, sa, 0, word_bits),
                   seed=synth.seed_for("w", bits, sa, sw, word_bits))


def test_conv_output_formats(samd_lib):
    shape = samd.ConvShape(2, 40, 8, 8, 290, R=1, S=1, pad=0)
    for fo_t in [(3, True, 0, 32), (6, False, 0, 64), (5, True, 1, 32), (1, False, 0, 32), (2, True, 0, 64)]:
        run_conv_check(shape, 4, False, 4, True, fo_t=fo_t, shift=3, seed=5)


def test_conv_extreme_values_at_the_exactness_bound(samd_lib):
    # u8 x s8, 3x3 over 57 channels: 513 taps * 255 * 128 = 16,744,320 < 2^24
    shape = samd.ConvShape(1, 57, 6, 6, 32)
    for a_val, w_val in [(255, -128), (255, 127), (1, -128), (255, -1)]:
        run_conv_check(shape, 8, False, 8, True, act_gen=lambda s, a=a_val: np.full(s, a, np.int64),
                       wt_gen=lambda s, w=w_val: np.full(s, w, np.int64), shift=0)
    # alternating signs through the reduction
    run_conv_check(shape, 8, False, 8, True,
                   act_gen=lambda s: np.full(s, 255, np.int64),
                   wt_gen=lambda s: np.where(np.arange(np.prod(s)).reshape(s) % 3 == 0, -128, 127).astype(np.int64))


def test_conv_empty_batch(samd_lib):
    shape = samd.ConvShape(0, 16, 8, 8, 16)
    fa, fw = samd.fmt(4, False), samd.fmt(4, True)
    ws = samd.conv_workspace(samd.ConvShape(1, 16, 8, 8, 16), fa, fw)
    dummy = torch.empty(16, dtype=torch.int32, device="cuda")
    samd.samd_conv2d(shape.desc(), fa, dummy, fw, dummy, dummy, None, None, 0, ws)


def test_conv_misaligned_pointer_rejected(samd_lib):
    shape = samd.ConvShape(1, 16, 8, 8, 16)
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, 4, False, 4, True, 3)
    ws = samd.conv_workspace(shape, fa, fw)
    acc = torch.empty(shape.N * shape.Ho * shape.Wo * shape.K + 1, dtype=torch.int32, device="cuda")
    with pytest.raises(samd.SamdError) as e:
        samd.samd_conv2d(shape.desc(), fa, a_w, fw, w_w, acc[1:], None, None, 0, ws)
    assert e.value.status == samd.SAMD_EALIGN


def test_bounded_wait_timeout_is_recorded_and_the_context_survives(samd_lib):
    # a wait on an mbarrier phase that nothing completes runs out after 2 ms
    # and records SAMD_ETIMEOUT; no trap, the context stays usable
    assert samd.samd_device_status(reset=True) in (samd.SAMD_OK, samd.SAMD_ETIMEOUT)
    assert samd.samd_device_status() == samd.SAMD_OK
    samd.samd_selftest_wait_timeout(2_000_000)
    torch.cuda.synchronize()
    assert samd.samd_device_status(reset=True) == samd.SAMD_ETIMEOUT
    assert samd.samd_device_status() == samd.SAMD_OK
    # a convolution after the reset is bit-exact and leaves the status clean
    shape = samd.ConvShape(2, 24, 10, 9, 32)
    run_conv_check(shape, 4, False, 4, True, fo_t=(4, False, 0, 32), seed=11)
    with pytest.raises(samd.SamdError) as e:
        samd.samd_selftest_wait_timeout(10)
    assert e.value.status == samd.SAMD_EINVAL


# 1x1 layers whose packed pixel rows are not 16-byte multiples take the
# gather through 16-byte windows: rows at every 4-byte offset, the last chunk
# of a pixel running past its words, stride 2, 64-bit words, and the last
# pixel's window reaching past the end of the activation tensor.
WINDOW_CASES = [
    (samd.ConvShape(2, 64, 7, 9, 48, R=1, S=1, pad=0), 6, False, 2, True, 32),    # 52-byte rows (full chunk)
    (samd.ConvShape(2, 128, 5, 7, 40, R=1, S=1, pad=0), 6, False, 2, True, 32),   # 104-byte rows
    (samd.ConvShape(1, 192, 9, 5, 24, R=1, S=1, pad=0), 6, True, 5, True, 32),    # 156-byte rows
    (samd.ConvShape(1, 512, 4, 5, 72, R=1, S=1, pad=0), 6, False, 2, True, 32),   # 412-byte rows, 9 chunks
    (samd.ConvShape(3, 40, 6, 6, 16, R=1, S=1, pad=0), 4, False, 4, True, 32),    # 20-byte rows, e4m3
    (samd.ConvShape(2, 30, 5, 5, 20, R=1, S=1, pad=0), 6, False, 3, True, 64),    # 24-byte rows, 64-bit words
    (samd.ConvShape(2, 128, 9, 9, 40, R=1, S=1, pad=0, stride=2), 6, False, 2, True, 32),  # projection
]


@pytest.mark.parametrize("shape,ba,sa,bw,sw,word_bits", WINDOW_CASES,
                         ids=lambda v: f"{v.N}x{v.C}x{v.H}x{v.W}-K{v.K}s{v.stride}" if isinstance(v, samd.ConvShape) else None)
def test_conv_1x1_window_gather(samd_lib, shape, ba, sa, bw, sw, word_bits):
    assert conv_supported(shape, ba, sa, bw, sw)
    run_conv_check(shape, ba, sa, bw, sw, word_bits=word_bits, fo_t=(ba, sa, 0, word_bits),
                   seed=synth.seed_for("win", shape, ba, sa, bw, sw, word_bits))


# Packed-only outputs (no int32 accumulator requested) take the fast
# requantize-and-pack epilogues. Channel counts that are not multiples of 32
# leave the last 32-column group partly past the last channel: the words the
# row holds must be exact and nothing past them written (guard words after
# the output and the neighbouring rows' words stay as they were).
PACKED_ONLY_K = (40, 70, 290)


@pytest.mark.parametrize("fo_signed", SIGNS)
@pytest.mark.parametrize("fo_bits", BITS)
def test_conv_packed_only_outputs_partial_groups(samd_lib, fo_bits, fo_signed):
    for K, (R, word_bits, spacer) in itertools.product(PACKED_ONLY_K, [(3, 32, 0), (1, 32, 0), (3, 64, 0), (1, 32, 1)]):
        shape = samd.ConvShape(2, 24, 6, 5, K, R=R, S=R, pad=R // 2)
        a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, 4, False, 3, True,
                                               synth.seed_for("po", K, R, fo_bits, fo_signed, word_bits))
        fo = samd.fmt(fo_bits, fo_signed, spacer, word_bits)
        shift = harness_shift(4, 3, fo_bits, shape.C * shape.R * shape.S)
        n = samd.samd_packed_words(fo, shape.N * shape.Ho * shape.Wo, K)
        guard = 64
        buf = torch.full((n + guard,), 0x5A5A5A5A, dtype=samd.word_dtype(fo), device="cuda")
        ws = samd.conv_workspace(shape, fa, fw)
        samd.samd_conv2d(shape.desc(), fa, a_w, fw, w_w, None, fo, buf, shift, ws)
        torch.cuda.synchronize()
        got = np_words(buf, word_bits)
        want = oracle_requant_pack(oracle_conv_nhwc(a_v, w_v, shape), shift, fo)
        assert np.array_equal(got[:n], want), (K, R, word_bits, spacer)
        assert np.array_equal(got[n:], np_words(torch.full((guard,), 0x5A5A5A5A, dtype=samd.word_dtype(fo)), word_bits))
    assert_status_clean()
