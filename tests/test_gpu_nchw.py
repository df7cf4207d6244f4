"""GPU parity of the NCHW convolution: tensors packed along the image width
(rows of W lanes, the layout of the paper's Fig. 12 x-loop), computed by the
paper's wide-multiply engine (section 5.1 with the Fig. 10 sign extension
and Fig. 11 repair) on the CUDA cores. Compared with the CPU oracle's direct
convolution element by element; the requantized output packed along W
against the oracle's requantize + pack."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_status_clean, np_words, values_and_bytes
from paper_1809_10572_gb300 import samd, synth

pytestmark = pytest.mark.gpu


def nchw_case(shape, ba, sa, bw, sw, seed, word_bits=32, act_gen=None, wt_gen=None):
    fa, fw = samd.fmt(ba, sa, 0, word_bits), samd.fmt(bw, sw, 0, word_bits)
    if act_gen is None:
        a_v, a_b = values_and_bytes(seed, (shape.N, shape.C, shape.H, shape.W), ba, sa)
    else:
        a_v = act_gen((shape.N, shape.C, shape.H, shape.W))
        a_b = synth.to_bytes_t(torch.from_numpy(a_v)).cuda()
    if wt_gen is None:
        w_v, w_b = values_and_bytes(seed + 1, (shape.K, shape.C, shape.R, shape.S), bw, sw)
    else:
        w_v = wt_gen((shape.K, shape.C, shape.R, shape.S))
        w_b = synth.to_bytes_t(torch.from_numpy(w_v)).cuda()
    a_w = samd.pack(a_b, fa, shape.N * shape.C * shape.H, shape.W)
    w_w = samd.pack(w_b, fw, shape.K * shape.C * shape.R, shape.S)
    return a_v, w_v, a_w, w_w, fa, fw


def check(shape, ba, sa, bw, sw, seed, fo=None, shift=0, word_bits=32, act_gen=None, wt_gen=None):
    a_v, w_v, a_w, w_w, fa, fw = nchw_case(shape, ba, sa, bw, sw, seed, word_bits, act_gen, wt_gen)
    assert samd.samd_conv2d_operand_bits(shape.desc(samd.SAMD_NCHW), fa, fw) == 64
    acc, packed = samd.conv2d_nchw(a_w, w_w, shape, fa, fw, fo, shift=shift)
    torch.cuda.synchronize()
    want = oracle.conv2d(a_v, w_v, stride=1, pad=shape.pad, nthreads=oracle.max_threads())
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
    if fo is not None:
        q = oracle.requant(want.ravel(), shift, fo.bits, bool(fo.is_signed)).reshape(-1, shape.Wo)
        assert np.array_equal(np_words(packed, fo.word_bits), oracle.pack(q, fo.bits, bool(fo.is_signed), fo.spacer,
                                                                          fo.word_bits))
    assert_status_clean()


ONE_ROW = [  # 1D convolutions: one input row, one kernel row (section 5: the polynomial product)
    samd.ConvShape(1, 1, 1, 37, 1, R=1, S=3, pad=0),
    samd.ConvShape(2, 3, 1, 100, 4, R=1, S=3, pad=1),
    samd.ConvShape(1, 2, 1, 301, 3, R=1, S=5, pad=2),    # several 31-segment chunks per row
    samd.ConvShape(1, 4, 1, 9, 2, R=1, S=1, pad=0),
]
TWO_D = [
    samd.ConvShape(2, 5, 7, 33, 6),
    samd.ConvShape(1, 16, 12, 12, 8, R=5, S=5, pad=2),
    samd.ConvShape(1, 3, 9, 70, 5, R=2, S=2, pad=0),
    samd.ConvShape(3, 64, 6, 56, 4),
]
FORMATS = [(4, False, 4, True), (2, True, 2, True), (1, False, 1, True), (3, True, 5, False), (5, True, 5, True),
           (8, False, 3, True), (1, True, 1, True)]


@pytest.mark.parametrize("shape", ONE_ROW + TWO_D, ids=lambda s: f"{s.N}x{s.C}x{s.H}x{s.W}-K{s.K}-{s.R}x{s.S}p{s.pad}")
@pytest.mark.parametrize("ba,sa,bw,sw", FORMATS)
def test_nchw_widemul_conv(samd_lib, shape, ba, sa, bw, sw):
    fa, fw = samd.fmt(ba, sa), samd.fmt(bw, sw)
    if samd.samd_conv2d_operand_bits(shape.desc(samd.SAMD_NCHW), fa, fw) == 0:
        pytest.skip("outside the wide-multiply engine's limits (S x F > 64)")
    check(shape, ba, sa, bw, sw, synth.seed_for("nchw", shape, ba, sa, bw, sw), fo=samd.fmt(ba, sa), shift=3)


@pytest.mark.parametrize("word_bits", (32, 64))
def test_nchw_output_formats_and_word_widths(samd_lib, word_bits):
    shape = samd.ConvShape(2, 8, 5, 45, 3)
    for fo in (samd.fmt(3, True, 0, word_bits), samd.fmt(6, False, 0, word_bits), samd.fmt(4, False, 1, word_bits)):
        check(shape, 4, False, 3, True, 77, fo=fo, shift=2, word_bits=word_bits)


def test_nchw_extreme_values(samd_lib):
    # every lane at its most negative value: the largest sums, every borrow repaired
    shape = samd.ConvShape(1, 40, 4, 50, 3)
    for ba, sa, bw, sw in [(4, True, 4, True), (2, True, 2, True), (5, False, 3, True)]:
        amin = -(1 << (ba - 1)) if sa else (1 << ba) - 1
        wmin = -(1 << (bw - 1))
        check(shape, ba, sa, bw, sw, 0, act_gen=lambda s, v=amin: np.full(s, v, np.int64),
              wt_gen=lambda s, v=wmin: np.full(s, v, np.int64))
        # the extreme value next to zero and next to the other extreme along the row:
        # coefficients of zero beside negative ones (the double increment of section 6)
        amax = (1 << (ba - 1)) - 1 if sa else 0
        for other in (0, amax):
            check(shape, ba, sa, bw, sw, 0,
                  act_gen=lambda s, v=amin, o=other: np.where(np.arange(np.prod(s)).reshape(s) % 2 == 0, v, o),
                  wt_gen=lambda s, v=wmin: np.full(s, v, np.int64))


def test_nchw_sweep_layer_shape(samd_lib):
    # the 3x3 C64 -> 64 56x56 layer of the bit-width sweep, batch 2, at the
    # widths the engine holds
    shape = samd.ConvShape(2, 64, 56, 56, 64)
    for b, sa, sw in [(1, False, False), (2, True, True), (4, False, True)]:
        check(shape, b, sa, b, sw, synth.seed_for("nchw-sweep", b, sa, sw), fo=samd.fmt(b, sa), shift=b)


def test_nchw_limits(samd_lib):
    fa, fw = samd.fmt(4, False), samd.fmt(4, True)
    # stride 2 and kernel rows that do not fit one word are outside the engine
    assert samd.samd_conv2d_operand_bits(samd.ConvShape(1, 8, 8, 8, 4, stride=2).desc(samd.SAMD_NCHW), fa, fw) == 0
    assert samd.samd_conv2d_operand_bits(samd.ConvShape(1, 8, 8, 16, 4, R=7, S=7, pad=3).desc(samd.SAMD_NCHW),
                                         samd.fmt(8, False), samd.fmt(8, True)) == 0
    shape = samd.ConvShape(1, 8, 8, 8, 4, stride=2)
    dummy = torch.zeros(4096, dtype=torch.int32, device="cuda")
    with pytest.raises(samd.SamdError) as e:
        samd.samd_conv2d(shape.desc(samd.SAMD_NCHW), fa, dummy, fw, dummy, dummy, None, None, 0, dummy)
    assert e.value.status == samd.SAMD_EUNSUP
    # weights are not prepared ahead for this layout
    with pytest.raises(samd.SamdError) as e:
        samd.samd_conv2d_prepare(samd.ConvShape(1, 8, 8, 8, 4).desc(samd.SAMD_NCHW), fa, fw, dummy, None, dummy)
    assert e.value.status == samd.SAMD_EUNSUP
    assert not dummy.any()
