"""samd_conv2d_noalloc: the convolution for callers that cannot allocate
device memory (their framework owns every allocation, or they must not
allocate once running). It keeps the widened weights in a static 8 MiB
array inside the library instead of a caller-provided workspace. Its results
must equal the CPU oracle's, and those of samd_conv2d, call after call.

This file is collected last on purpose, so that a run stopping at its
first failure has already run every other test."""
import numpy as np
import pytest
import torch

from gpu_util import assert_status_clean, conv_case, np_words, oracle_conv_nhwc, oracle_requant_pack
from paper_1809_10572_gb300 import samd

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 8 << 20


def check_case(shape, ba, sa, bw, sw, fo, shift, seed, want_acc=True):
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, ba, sa, bw, sw, seed)
    # the allocation-free entry point, through the C ABI, into outputs filled with junk
    acc = torch.full((shape.N, shape.Ho, shape.Wo, shape.K), -7, dtype=torch.int32, device="cuda") if want_acc else None
    packed = None
    if fo is not None:
        packed = samd.empty_words(fo, shape.N * shape.Ho * shape.Wo, shape.K)
        packed.fill_(-1)
    samd.samd_conv2d_noalloc(shape.desc(), fa, a_w, fw, w_w, acc, fo, packed, shift)
    torch.cuda.synchronize()
    # against the CPU oracle (the independent check)
    want = oracle_conv_nhwc(a_v, w_v, shape)
    if want_acc:
        assert np.array_equal(acc.cpu().numpy().astype(np.int64), want)
    if fo is not None:
        assert np.array_equal(np_words(packed, fo.word_bits), oracle_requant_pack(want, shift, fo))
    # and against the allocating entry point with a torch-allocated workspace
    acc_ref, packed_ref = samd.conv2d(a_w, w_w, shape, fa, fw, fo, shift=shift, want_acc=want_acc)
    torch.cuda.synchronize()
    if want_acc:
        assert torch.equal(acc, acc_ref)
    if fo is not None:
        assert torch.equal(packed, packed_ref)


def test_noalloc_matches_oracle_on_consecutive_calls(samd_lib):
    # calls in a row on the same static array: a larger layer first, then a
    # smaller one that reuses (and must fully rewrite) its start; a layer
    # whose widened weights fill the array exactly (8 MiB: 1x1 over 2048
    # channels to 960, split weight digits since 2048 x 255 x 128 is past
    # 2^24, eight channel blocks of 2 x 128 rows x 2048 fp16 positions); an
    # output with no int32 accumulator; and the first layer again
    cases = [
        (samd.ConvShape(2, 64, 14, 14, 96), 4, False, 4, True, samd.fmt(4, False), 6, 101, True),
        (samd.ConvShape(1, 24, 9, 7, 40), 6, True, 8, True, samd.fmt(6, True), 8, 202, True),
        (samd.ConvShape(1, 2048, 2, 2, 960, R=1, S=1, pad=0), 8, False, 8, True, samd.fmt(8, False), 12, 303, True),
        (samd.ConvShape(2, 40, 7, 9, 72, R=1, S=1, pad=0), 6, False, 2, True, samd.fmt(6, False), 3, 404, False),
        (samd.ConvShape(1, 33, 5, 6, 20), 3, True, 5, False, None, 0, 606, True),  # int32 output only
        (samd.ConvShape(2, 64, 14, 14, 96), 4, False, 4, True, samd.fmt(4, False), 6, 505, True),
    ]
    for shape, ba, sa, bw, sw, fo, shift, seed, want_acc in cases:
        check_case(shape, ba, sa, bw, sw, fo, shift, seed, want_acc)
    assert_status_clean()


def test_noalloc_rejects_layers_beyond_its_scratch(samd_lib):
    # The limit applies to the widened weights of the call itself: 976
    # output channels of 3-bit lanes (10 per word) take nine channel blocks
    # of 120 over 36 chunks (four per pixel and tap), 10.6 MB; and a 3x3
    # layer over 1024 channels to 1024, 11.8 MB.
    cases = [(samd.ConvShape(1, 224, 8, 8, 976), samd.fmt(8, False), samd.fmt(8, True), samd.fmt(3, False)),
             (samd.ConvShape(1, 1024, 4, 4, 1024), samd.fmt(4, False), samd.fmt(4, True), None)]
    for shape, fa, fw, fo in cases:
        assert samd.samd_conv2d_workspace_size(shape.desc(), fa, fw) > SCRATCH_BYTES
        # buffers of the layer's real sizes, so that nothing could be read or
        # written out of bounds even if the call were (wrongly) accepted
        act = torch.zeros(samd.samd_packed_words(fa, shape.N * shape.H * shape.W, shape.C),
                          dtype=samd.word_dtype(fa), device="cuda")
        wt = torch.zeros(samd.samd_packed_words(fw, shape.K * shape.R * shape.S, shape.C),
                         dtype=samd.word_dtype(fw), device="cuda")
        acc = torch.zeros(shape.N * shape.Ho * shape.Wo * shape.K, dtype=torch.int32, device="cuda")
        packed = samd.empty_words(fo, shape.N * shape.Ho * shape.Wo, shape.K).zero_() if fo is not None else None
        with pytest.raises(samd.SamdError) as e:
            samd.samd_conv2d_noalloc(shape.desc(), fa, act, fw, wt, acc, fo, packed, 0)
        assert e.value.status == samd.SAMD_EUNSUP
        torch.cuda.synchronize()
        assert not acc.any()  # nothing was launched
        if packed is not None:
            assert not packed.any()
