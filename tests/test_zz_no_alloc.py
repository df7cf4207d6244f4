"""samd_conv2d_noalloc: the convolution for callers that cannot allocate
device memory (their framework owns every allocation, or they must not
allocate once running). It keeps the widened weights in a static 8 MiB
array inside the library instead of a caller-provided workspace; its
results must equal those of samd_conv2d, call after call.

This file is collected last on purpose, so that a run stopping at its
first failure has already run every other test."""
import numpy as np
import pytest
import torch

from gpu_util import assert_status_clean, conv_case
from paper_1809_10572_gb300 import samd

pytestmark = pytest.mark.gpu


def run_both(shape, ba, sa, bw, sw, fo, shift, seed):
    a_v, w_v, a_w, w_w, fa, fw = conv_case(shape, ba, sa, bw, sw, seed)
    # reference: the allocating entry point with a torch-allocated workspace
    acc_ref, packed_ref = samd.conv2d(a_w, w_w, shape, fa, fw, fo, shift=shift)
    # the allocation-free entry point, through the C ABI, into fresh outputs
    acc = torch.full_like(acc_ref, -7)
    packed = torch.full_like(packed_ref, -1)
    samd.samd_conv2d_noalloc(shape.desc(), fa, a_w, fw, w_w, acc, fo, packed, shift)
    torch.cuda.synchronize()
    return acc_ref, packed_ref, acc, packed


def test_noalloc_matches_conv2d_on_consecutive_calls(samd_lib):
    # two calls in a row: a larger layer first, then a smaller one that reuses
    # (and must fully rewrite) the start of the same static array
    cases = [
        (samd.ConvShape(2, 64, 14, 14, 96), 4, False, 4, True, samd.fmt(4, False), 6, 101),
        (samd.ConvShape(1, 24, 9, 7, 40), 6, True, 8, True, samd.fmt(6, True), 8, 202),
    ]
    for shape, ba, sa, bw, sw, fo, shift, seed in cases:
        acc_ref, packed_ref, acc, packed = run_both(shape, ba, sa, bw, sw, fo, shift, seed)
        assert torch.equal(acc, acc_ref)        # integers: bit-exact is the tolerance
        assert torch.equal(packed, packed_ref)
    assert_status_clean()


def test_noalloc_rejects_layers_beyond_its_scratch(samd_lib):
    # 3x3 over 1024 -> 1024 channels at 4 bits needs more than 8 MiB of widened weights
    shape = samd.ConvShape(1, 1024, 4, 4, 1024)
    fa, fw = samd.fmt(4, False), samd.fmt(4, True)
    assert samd.samd_conv2d_workspace_size(shape.desc(), fa, fw) > (8 << 20)
    dummy = torch.zeros(1 << 16, dtype=torch.int32, device="cuda")
    with pytest.raises(samd.SamdError) as e:
        samd.samd_conv2d_noalloc(shape.desc(), fa, dummy, fw, dummy, dummy, None, None, 0)
    assert e.value.status == samd.SAMD_EUNSUP
    assert np.all(dummy.cpu().numpy() == 0)  # nothing was launched
