"""GPU parity at the workload sizes: the bit-width sweep, every VGG-16 and
ResNet-50 layer at full batch (checked on sampled output rows the oracle
computes one by one), a chained small VGG-16, the prepared-weight entry
points and the split weight digits."""
import numpy as np
import pytest
import torch

import oracle
from gpu_util import (assert_status_clean, conv_case, gpu_pack, np_words, oracle_conv_nhwc, oracle_conv_rows,
                      oracle_requant_pack, values_and_bytes)
from paper_1809_10572_gb300 import samd, synth, workloads

pytestmark = pytest.mark.gpu


def test_generator_same_on_cpu_and_gpu(samd_lib):
    a = synth.lanes_t(123, (1000, 37), 5, True, device="cuda").cpu()
    b = synth.lanes_t(123, (1000, 37), 5, True)
    assert torch.equal(a, b)
    c = synth.lanes_t(123, (10, 37), 5, True, offset=500 * 37)
    assert torch.equal(b[500:510], c)


def full_layer_check(layer, seed, rows_per_image=2, images=(0,)):
    """Run one layer at full size on the GPU (inputs generated on the device),
    then check int32 and packed outputs on sampled rows of sampled images
    against the oracle, fed from the same generator on the CPU."""
    s = layer.shape
    fa = samd.fmt(layer.ba, layer.sa, 0, layer.word_bits)
    fw = samd.fmt(layer.bw, layer.sw, 0, layer.word_bits)
    fo = samd.fmt(layer.bo, layer.so, 0, layer.word_bits)
    shift = workloads.harness_shift(layer.ba, layer.bw, layer.bo, s.C * s.R * s.S)
    a_dev = synth.lanes_t(seed, (s.N, s.H, s.W, s.C), layer.ba, layer.sa, device="cuda")
    a_w = gpu_pack(synth.to_bytes_t(a_dev), fa, s.N * s.H * s.W, s.C)
    del a_dev
    w_v = synth.lanes_t(seed + 1, (s.K, s.R, s.S, s.C), layer.bw, layer.sw)
    w_w = gpu_pack(synth.to_bytes_t(w_v).cuda(), fw, s.K * s.R * s.S, s.C)
    conv = samd.PreparedConv(w_w, s, fa, fw, fo)
    acc, packed = conv.outputs()
    conv(a_w, acc, packed, shift)
    torch.cuda.synchronize()
    assert_status_clean()
    wpr_o = samd.samd_packed_words(fo, 1, s.K)
    w_np = w_v.numpy()
    for n in images:
        img = synth.lanes_t(seed, (s.H, s.W, s.C), layer.ba, layer.sa, offset=n * s.H * s.W * s.C).numpy()
        for h0 in sorted({0, s.Ho // 2, s.Ho - rows_per_image}):
            h1 = min(s.Ho, h0 + rows_per_image)
            want = oracle_conv_rows(img, w_np, s, h0, h1)
            got = acc[n, h0:h1].cpu().numpy().astype(np.int64)
            assert np.array_equal(got, want), (layer.name, n, h0)
            p0 = (n * s.Ho + h0) * s.Wo
            got_p = np_words(packed[p0 * wpr_o:(p0 + (h1 - h0) * s.Wo) * wpr_o], fo.word_bits)
            assert np.array_equal(got_p, oracle_requant_pack(want, shift, fo)), (layer.name, n, h0)
    return acc, packed


@pytest.mark.parametrize("layer", workloads.sweep(), ids=lambda l: l.name)
def test_sweep_full_size(samd_lib, layer):
    """N8 C64 -> 64 on 56x56 at every width and sign combination: whole
    output of two of the eight images (int32 and requantized packed)."""
    full_layer_check(layer, synth.seed_for("sweep", layer.name), rows_per_image=56, images=(0, 7))


@pytest.mark.parametrize("layer", workloads.vgg16(), ids=lambda l: l.name)
def test_vgg16_layer_full_batch(samd_lib, layer):
    full_layer_check(layer, synth.seed_for("vgg", layer.name), images=(0, 15))


@pytest.mark.parametrize("layer", workloads.resnet50(), ids=lambda l: l.name)
def test_resnet50_layer_full_batch(samd_lib, layer):
    full_layer_check(layer, synth.seed_for("r50", layer.name), images=(0, 63))


def test_vgg16_chain_small(samd_lib):
    """All 13 VGG-16 convolutions and the four pools chained on 32x32 inputs
    (batch 2): requantized u4 outputs feed the next layer on both sides; each
    layer's output is compared. The s4 weights are drawn from [-7, 7] so their
    mean is zero, and each layer's shift is calibrated on the oracle's sums
    (their positive 99th percentile maps near the top of u4); a fixed shift
    lets the ReLU'd signal decay to zero within a few layers."""
    layers = workloads.vgg16(N=2, H=32)
    s0 = layers[0].shape
    x = synth.lanes(synth.seed_for("chain"), (s0.N, s0.H, s0.W, s0.C), 4, False)  # NHWC values, oracle side
    f4u, f4s = samd.fmt(4, False), samd.fmt(4, True)
    xw = gpu_pack(synth.to_bytes_t(torch.from_numpy(x)).cuda(), f4u, s0.N * s0.H * s0.W, s0.C)
    for i, layer in enumerate(layers):
        s = layer.shape
        w_v = synth.uniform_ints(synth.seed_for("chainw", i), (s.K, s.R, s.S, s.C), -7, 7)
        w_w = gpu_pack(synth.to_bytes_t(torch.from_numpy(w_v)).cuda(), f4s, s.K * s.R * s.S, s.C)
        acc = oracle_conv_nhwc(x, w_v, s)
        pos = acc[acc > 0]
        p99 = int(np.percentile(pos, 99)) if pos.size else 0
        shift = max(0, p99.bit_length() - 4)
        _, yw = samd.conv2d(xw, w_w, s, f4u, f4s, f4u, shift=shift, want_acc=False)
        y = oracle.requant(acc.ravel(), shift, 4, False).reshape(acc.shape)
        assert np.array_equal(np_words(yw, 32), oracle.pack(y.reshape(-1, s.K), 4, False)), layer.name
        assert 0 < np.count_nonzero(y) < y.size  # the chain neither saturates nor vanishes
        if layer.pool_after:
            yw = samd.maxpool2x2(yw, f4u, s.N, s.K, s.Ho, s.Wo)
            y = oracle.maxpool2x2(y.transpose(0, 3, 1, 2)).transpose(0, 2, 3, 1)
            assert np.array_equal(np_words(yw, 32), oracle.pack(y.reshape(-1, s.K), 4, False)), layer.name + " pool"
        x, xw = y, yw
    assert_status_clean()


def test_prepared_weights_reused(samd_lib):
    shape = samd.ConvShape(2, 64, 12, 12, 96)
    fo = samd.fmt(5, True)
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, 5, True, 6, True, 41)
    conv = samd.PreparedConv(w_w, shape, fa, fw, fo)
    for seed in (41, 42):
        if seed == 42:
            a_v, a_b = values_and_bytes(seed, (shape.N, shape.H, shape.W, shape.C), 5, True)
            a_w = gpu_pack(a_b, fa, shape.N * shape.H * shape.W, shape.C)
        acc, packed = conv.outputs()
        conv(a_w, acc, packed, 6)
        want = oracle_conv_nhwc(a_v, w_v, shape)
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
        assert np.array_equal(np_words(packed, 32), oracle_requant_pack(want, 6, fo))
        # the one-shot entry point gives the same words
        _, p2 = samd.conv2d(a_w, w_w, shape, fa, fw, fo, shift=6, want_acc=False)
        assert torch.equal(p2, packed)
    assert_status_clean()


def test_prepared_conv_in_cuda_graph(samd_lib):
    shape = samd.ConvShape(1, 64, 20, 20, 64)
    fo = samd.fmt(4, False)
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, 4, False, 4, True, 77)
    conv = samd.PreparedConv(w_w, shape, fa, fw, fo)
    acc, packed = conv.outputs()
    conv(a_w, acc, packed, 5)  # first call outside capture sets kernel attributes
    torch.cuda.synchronize()
    acc.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        conv(a_w, acc, packed, 5)
    g.replay()
    torch.cuda.synchronize()
    want = oracle_conv_nhwc(a_v, w_v, shape)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)


@pytest.mark.parametrize("ba,sa,bw,sw", [(8, False, 8, False), (8, False, 8, True), (8, True, 8, False),
                                         (7, False, 8, True), (8, False, 6, False)])
def test_split_weight_digits_extremes(samd_lib, ba, sa, bw, sw):
    """Sums far above 2^24 (up to 576 * 255 * 255 = 37,454,400) stay exact
    through the two-digit weight split."""
    shape = samd.ConvShape(1, 64, 6, 6, 72)
    lo_a, hi_a = synth.lane_range(ba, sa)
    lo_w, hi_w = synth.lane_range(bw, sw)
    cases = [(hi_a, hi_w), (hi_a, lo_w), (lo_a, lo_w), (hi_a, hi_w - 1)]
    for av, wv in cases:
        a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, ba, sa, bw, sw, 0,
                                               act_gen=lambda s, v=av: np.full(s, v, np.int64),
                                               wt_gen=lambda s, v=wv: np.full(s, v, np.int64))
        acc, _ = samd.conv2d(a_w, w_w, shape, fa, fw)
        want = oracle_conv_nhwc(a_v, w_v, shape)
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), want), (av, wv)
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, ba, sa, bw, sw, synth.seed_for("split", ba, sa, bw, sw))
    fo = samd.fmt(ba, sa)
    acc, packed = samd.conv2d(a_w, w_w, shape, fa, fw, fo, shift=9)
    want = oracle_conv_nhwc(a_v, w_v, shape)
    assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
    assert np.array_equal(np_words(packed, 32), oracle_requant_pack(want, 9, fo))
    assert_status_clean()


def test_split_with_channel_blocks(samd_lib):
    """Split digits with more output channels than one block holds (K > 128)."""
    shape = samd.ConvShape(1, 48, 7, 9, 300)
    for fo_t in [(3, False, 0, 32), (8, True, 0, 32)]:
        a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, 8, False, 8, True, 5)
        fo = samd.fmt(*fo_t)
        acc, packed = samd.conv2d(a_w, w_w, shape, fa, fw, fo, shift=10)
        want = oracle_conv_nhwc(a_v, w_v, shape)
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
        assert np.array_equal(np_words(packed, 32), oracle_requant_pack(want, 10, fo))
