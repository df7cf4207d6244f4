"""The convolution with the 2x2 max-pool fused into its epilogue
(samd_conv2d_prepared_pool2x2) against the oracle: oracle.conv2d, then
oracle.requant, then oracle.maxpool2x2 on the requantized lanes, packed,
compared word for word. Shapes cover one and several row pairs per tile,
channel counts that leave partial words and channel blocks, one- and
two-half tiles, every supported output width and sign, e4m3 and fp16
operands, batch tails, and the VGG-16 layers whose pool the step fuses
(conv4, conv7, conv10) at batch 16 (whole first and last images)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import assert_status_clean, conv_case, harness_shift, np_words, oracle_conv_nhwc, oracle_conv_rows
from paper_1809_10572_gb300 import samd, synth, workloads

pytestmark = pytest.mark.gpu


def oracle_pooled_words(acc_nhwk, shift, fo):
    """requantize every output, pool 2x2 lane-wise, pack rows of K lanes"""
    N, Ho, Wo, K = acc_nhwk.shape
    q = oracle.requant(acc_nhwk.reshape(-1), shift, fo.bits, bool(fo.is_signed)).reshape(N, Ho, Wo, K)
    pooled = oracle.maxpool2x2(q.transpose(0, 3, 1, 2)).transpose(0, 2, 3, 1)
    return oracle.pack(pooled.reshape(-1, K), fo.bits, bool(fo.is_signed), 0, 32)


def run_pool_case(shape, ba, sa, bw, sw, fo, seed, shift=None):
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, ba, sa, bw, sw, seed)
    if shift is None:
        shift = harness_shift(ba, bw, fo.bits, shape.C * shape.R * shape.S)
    conv = samd.PreparedConv(w_w, shape, fa, fw, fo)
    assert conv.pool2x2_supported(), (shape, fo)
    # the pooled rows, then 64 guard words that must stay untouched
    nwords = samd.samd_packed_words(fo, shape.N * (shape.Ho // 2) * (shape.Wo // 2), shape.K)
    buf = torch.full((nwords + 64,), 0x5A5A5A5A, dtype=torch.int32, device="cuda")
    pooled = buf[:nwords]
    conv.pool2x2(a_w, pooled, shift)
    # the unfused pair of calls on the same prepared weights
    _, packed = conv.outputs(want_acc=False)
    conv(a_w, None, packed, shift)
    two_step = samd.maxpool2x2(packed, fo, shape.N, shape.K, shape.Ho, shape.Wo)
    torch.cuda.synchronize()
    want = oracle_pooled_words(oracle_conv_nhwc(a_v, w_v, shape), shift, fo)
    assert np.array_equal(np_words(pooled, 32), want)
    assert bool((buf[nwords:] == 0x5A5A5A5A).all())
    assert np.array_equal(np_words(two_step, 32), want)
    assert_status_clean()


CASES = [
    # N, C, H, W, K; activation, weight formats; output format. Every shape
    # takes halo tiles (little padding per image), the fused pool's domain.
    (samd.ConvShape(2, 16, 28, 28, 16), 4, False, 4, True, (4, False)),     # 4 row pairs per tile, last tile partial
    (samd.ConvShape(3, 64, 28, 28, 64), 4, False, 4, True, (4, False)),     # batch tail
    (samd.ConvShape(1, 40, 30, 32, 70), 4, True, 4, True, (4, True)),       # partial last word, signed
    (samd.ConvShape(2, 24, 28, 28, 40), 6, False, 2, True, (8, False)),     # fp16 operands, 8-bit out
    (samd.ConvShape(1, 128, 56, 56, 96), 4, False, 4, True, (2, True)),     # two row pairs per tile
    (samd.ConvShape(1, 64, 112, 112, 32), 3, False, 3, True, (1, False)),   # one row pair per tile
    (samd.ConvShape(2, 96, 28, 28, 300), 4, False, 4, True, (4, False)),    # one-half tiles, two channel blocks
    (samd.ConvShape(1, 32, 30, 60, 48), 5, True, 5, True, (8, True)),       # Ho / 2 not a multiple of q
    (samd.ConvShape(2, 256, 28, 28, 256), 4, False, 4, True, (4, False)),   # one-half tiles, 256 channels
]


@pytest.mark.parametrize("case", range(len(CASES)))
def test_fused_pool_matches_oracle(samd_lib, case):
    shape, ba, sa, bw, sw, fo_t = CASES[case]
    run_pool_case(shape, ba, sa, bw, sw, samd.fmt(fo_t[0], fo_t[1]), seed=700 + case)


def test_fused_pool_unsupported_shapes_are_rejected(samd_lib):
    fa, fw = samd.fmt(4, False), samd.fmt(4, True)
    rejected = [
        (samd.ConvShape(1, 64, 224, 224, 64), samd.fmt(4, False)),  # 2 (W + 2) > 256
        (samd.ConvShape(1, 64, 28, 29, 64), samd.fmt(4, False)),    # odd width
        (samd.ConvShape(1, 64, 28, 28, 64), samd.fmt(3, False)),    # 3-bit lanes
        (samd.ConvShape(1, 64, 56, 56, 64, stride=2), samd.fmt(4, False)),
        (samd.ConvShape(1, 64, 8, 8, 64), samd.fmt(4, False)),      # small images: no halo tiles
    ]
    for shape, fo in rejected:
        assert not samd.samd_conv2d_pool2x2_supported(shape.desc(), fa, fw, fo)
        with pytest.raises(samd.SamdError) as e:
            samd.samd_conv2d_prepared_pool2x2(shape.desc(), fa, torch.zeros(4, dtype=torch.int32, device="cuda"), fw,
                                             torch.zeros(4, dtype=torch.uint8, device="cuda"), fo,
                                             torch.zeros(4, dtype=torch.int32, device="cuda"), 0)
        assert e.value.status == samd.SAMD_EUNSUP


VGG_POOLED = [l for l in workloads.vgg16() if l.pool_after and samd.samd_conv2d_pool2x2_supported(
    l.shape.desc(), samd.fmt(l.ba, l.sa), samd.fmt(l.bw, l.sw), samd.fmt(l.bo, l.so))]


@pytest.mark.parametrize("name", [l.name for l in VGG_POOLED])
def test_fused_pool_vgg16_layers_full_batch(samd_lib, name):
    """The VGG-16 layers the step fuses, at batch 16: the whole pooled output
    of the first and the last image against the oracle (each image
    regenerated alone from the counter-based generator)."""
    layer = next(l for l in VGG_POOLED if l.name == name)
    s = layer.shape
    fa, fw, fo = samd.fmt(layer.ba, layer.sa), samd.fmt(layer.bw, layer.sw), samd.fmt(layer.bo, layer.so)
    seed = synth.seed_for("poolvgg", s.C, s.K)
    a = synth.lanes_t(seed, (s.N * s.H * s.W, s.C), layer.ba, layer.sa, device="cuda")
    a_w = samd.pack(synth.to_bytes_t(a), fa)
    del a
    w_v = synth.lanes_t(seed + 1, (s.K, s.R, s.S, s.C), layer.bw, layer.sw)
    w_w = samd.pack(synth.to_bytes_t(w_v).cuda(), fw)
    conv = samd.PreparedConv(w_w, s, fa, fw, fo)
    shift = workloads.harness_shift(layer.ba, layer.bw, layer.bo, s.C * s.R * s.S)
    pooled = samd.empty_words(fo, s.N * (s.Ho // 2) * (s.Wo // 2), s.K)
    conv.pool2x2(a_w, pooled, shift)
    torch.cuda.synchronize()
    got = np_words(pooled, 32)
    rows_img = (s.Ho // 2) * (s.Wo // 2)
    wpr = samd.samd_packed_words(fo, 1, s.K)
    for n in (0, s.N - 1):
        # image n alone: the rows of the flat (N*H*W, C) input starting at n*H*W
        img = synth.lanes_t(seed, (s.H, s.W, s.C), layer.ba, layer.sa, offset=n * s.H * s.W * s.C).numpy()
        acc = oracle_conv_rows(img, w_v.numpy(), s, 0, s.Ho)
        want = oracle_pooled_words(acc[None], shift, fo)
        assert np.array_equal(got[n * rows_img * wpr:(n + 1) * rows_img * wpr], want), (name, n)
    assert_status_clean()
