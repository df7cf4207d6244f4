"""GPU parity at the sizes the kernels are timed at, and at the edges of the
exactness argument.

- Elementwise, pack and unpack on arrays of 2^26 + 77 lanes: every thread of
  the capped grid runs its grid-stride loop several times and the ragged tail
  takes the word kernel, the regime the 2^28-lane benchmark times. Compared
  word for word with the oracle.
- The 2x2 max-pool at the size of the first VGG-16 pool (batch 16, 224 x 224,
  64 channels), the whole output against the oracle.
- The convolution on e4m3 operands (tcgen05 kind::f8f6f4) with accumulators
  between 2^23 and 2^24, where a float32 sum of integers has no spare bit:
  the largest products (-16 x -16) mixed with odd small ones, checked
  element by element against the oracle. The library admits a layer to e4m3
  operands when R*S*C*max|a|*max|w| < 2^24; these layers sit just under
  that bound.
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_status_clean, conv_case, np_words, oracle_conv_nhwc
from paper_1809_10572_gb300 import samd, synth

pytestmark = pytest.mark.gpu

N_BIG = (1 << 26) + 77


def big_lanes(tag, bits, signed, n=N_BIG):
    """Seeded lane values generated on the GPU; (int64 numpy, int8 bytes on the GPU)."""
    v = synth.lanes_t(synth.seed_for(tag, bits, signed, n), (n,), bits, signed, device="cuda")
    return v.cpu().numpy(), synth.to_bytes_t(v)


def words_to_gpu(words: np.ndarray, word_bits: int) -> torch.Tensor:
    return torch.from_numpy(words.view(np.int32 if word_bits == 32 else np.int64)).cuda()


@pytest.mark.parametrize("signed", (False, True))
@pytest.mark.parametrize("bits", (1, 3, 8))
def test_elementwise_full_grid(samd_lib, bits, signed):
    f = samd.fmt(bits, signed)
    xv, _ = big_lanes("fx", bits, signed)
    yv, _ = big_lanes("fy", bits, signed)
    # inputs packed by the oracle, so every op below is checked on its own
    xw = words_to_gpu(oracle.pack(xv, bits, signed), 32)
    yw = words_to_gpu(oracle.pack(yv, bits, signed), 32)
    for op in ("add", "sub", "mul"):
        for sat in (False, True):
            got = samd.elementwise(op, xw, yw, f, N_BIG, saturate=sat)
            want = oracle.pack(oracle.elementwise(op, xv, yv, bits=bits, signed=signed, saturate=sat), bits, signed)
            assert np.array_equal(np_words(got, 32), want), (op, sat)
    got = samd.elementwise("relu", xw, None, f, N_BIG)
    want = oracle.pack(oracle.elementwise("relu", xv, bits=bits, signed=signed), bits, signed)
    assert np.array_equal(np_words(got, 32), want)
    for shift in (1, bits):
        got = samd.elementwise("requant", xw, None, f, N_BIG, shift=shift)
        want_v = oracle.elementwise("requant", xv, bits=bits, signed=signed, bits_o=bits, signed_o=signed,
                                    shift=shift)
        assert np.array_equal(np_words(got, 32), oracle.pack(want_v, bits, signed)), shift
    assert_status_clean()


@pytest.mark.parametrize("signed", (False, True))
@pytest.mark.parametrize("bits", (1, 3, 5, 7))
def test_elementwise_full_grid_one_spacer_bit(samd_lib, bits, signed):
    # the permanent-spacer word forms (one zero bit above each lane, Fig. 2)
    f = samd.fmt(bits, signed, 1)
    xv, _ = big_lanes("fsx", bits, signed)
    yv, _ = big_lanes("fsy", bits, signed)
    xw = words_to_gpu(oracle.pack(xv, bits, signed, 1), 32)
    yw = words_to_gpu(oracle.pack(yv, bits, signed, 1), 32)
    for op in ("add", "sub", "mul"):
        for sat in (False, True):
            got = samd.elementwise(op, xw, yw, f, N_BIG, saturate=sat)
            want = oracle.pack(oracle.elementwise(op, xv, yv, bits=bits, signed=signed, saturate=sat), bits, signed, 1)
            assert np.array_equal(np_words(got, 32), want), (op, sat)
    got = samd.elementwise("relu", xw, None, f, N_BIG)
    want = oracle.pack(oracle.elementwise("relu", xv, bits=bits, signed=signed), bits, signed, 1)
    assert np.array_equal(np_words(got, 32), want)
    got = samd.elementwise("requant", xw, None, f, N_BIG, shift=1)
    want_v = oracle.elementwise("requant", xv, bits=bits, signed=signed, bits_o=bits, signed_o=signed, shift=1)
    assert np.array_equal(np_words(got, 32), oracle.pack(want_v, bits, signed, 1))
    assert_status_clean()


@pytest.mark.parametrize("signed", (False, True))
@pytest.mark.parametrize("bits", range(1, 9))
def test_pack_unpack_full_grid(samd_lib, bits, signed):
    f = samd.fmt(bits, signed)
    v, b = big_lanes("fp", bits, signed)
    got = samd.pack(b, f, 1, N_BIG)
    want = oracle.pack(v, bits, signed)
    assert np.array_equal(np_words(got, 32), want)
    back = samd.unpack(words_to_gpu(want, 32), f, 1, N_BIG).cpu().numpy().astype(np.int64).ravel()
    assert np.array_equal(back, ((v & 0xFF) ^ 0x80) - 0x80)
    assert_status_clean()


@pytest.mark.parametrize("bits,signed,N", [(4, False, 16), (4, True, 4), (1, False, 4), (8, True, 2)])
def test_maxpool_vgg_block1_size(samd_lib, bits, signed, N):
    C, H, W = 64, 224, 224
    f = samd.fmt(bits, signed)
    v = synth.lanes_t(synth.seed_for("mpv", bits, signed, N), (N, H, W, C), bits, signed, device="cuda")
    words = samd.pack(synth.to_bytes_t(v), f, N * H * W, C)
    got = samd.maxpool2x2(words, f, N, C, H, W)
    want_v = oracle.maxpool2x2(v.cpu().numpy().transpose(0, 3, 1, 2)).transpose(0, 2, 3, 1)
    want = oracle.pack(np.ascontiguousarray(want_v).reshape(-1, C), bits, signed)
    assert np.array_equal(np_words(got, 32), want)
    assert_status_clean()


def mostly(value, odd_every, odd_value, odd2_every, odd2_value):
    """Arrays of `value` with odd_value at every odd_every-th flat position and
    odd2_value at every odd2_every-th (small odd terms among the largest ones)."""
    def gen(shape):
        idx = np.arange(int(np.prod(shape))).reshape(shape)
        out = np.full(shape, value, np.int64)
        out[idx % odd_every == 3] = odd_value
        out[idx % odd2_every == 5] = odd2_value
        return out
    return gen


E4M3_BOUND_CASES = [
    # 3x3 over 7281 channels of signed 5-bit lanes: 9 * 7281 * 16 * 16 = 16,775,424 < 2^24
    (samd.ConvShape(1, 7281, 5, 4, 16), 5, True, 5, True),
    # 1x1 over 65535 channels: 65535 * 16 * 16 = 16,776,960 < 2^24
    (samd.ConvShape(1, 65535, 3, 5, 16, R=1, S=1, pad=0), 5, True, 5, True),
    # unsigned 4-bit activations x signed 5-bit weights: 9 * 7767 * 15 * 16 = 16,776,720 < 2^24
    (samd.ConvShape(1, 7767, 4, 3, 24), 4, False, 5, True),
]


@pytest.mark.parametrize("shape,ba,sa,bw,sw", E4M3_BOUND_CASES,
                         ids=lambda v: f"C{v.C}-{v.R}x{v.S}" if isinstance(v, samd.ConvShape) else None)
def test_conv_e4m3_accumulators_between_2p23_and_2p24(samd_lib, shape, ba, sa, bw, sw):
    fa, fw = samd.fmt(ba, sa), samd.fmt(bw, sw)
    assert samd.samd_conv2d_operand_bits(shape.desc(), fa, fw) == 8  # the e4m3 path
    amax = -16 if sa else 15
    cases = [
        (mostly(amax, 7, -15 if sa else 13, 11, 1), mostly(-16, 5, -13, 13, 3)),
        (mostly(amax, 3, -1 if sa else 1, 17, -3 if sa else 3), mostly(-16, 9, 1, 23, -7)),
    ]
    for act_gen, wt_gen in cases:
        a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, ba, sa, bw, sw, 0, act_gen=act_gen, wt_gen=wt_gen)
        acc, _ = samd.conv2d(a_w, w_w, shape, fa, fw, None)
        torch.cuda.synchronize()
        want = oracle_conv_nhwc(a_v, w_v, shape)
        assert np.abs(want).max() > (1 << 23)  # the range under test is reached
        assert np.abs(want).max() < (1 << 24)
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
    assert_status_clean()
