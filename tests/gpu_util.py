"""Helpers shared by the GPU parity tests: seeded inputs on both sides,
CUDA results copied back as numpy words."""
import numpy as np
import torch

import oracle
from paper_1809_10572_gb300 import samd, synth


def np_words(t: torch.Tensor, word_bits: int) -> np.ndarray:
    a = t.detach().cpu().numpy()
    return a.view(np.uint32 if word_bits == 32 else np.uint64)


def values_and_bytes(seed, shape, bits, signed):
    """The same seeded lane values as int64 numpy (oracle side) and as int8
    bytes on the GPU (CUDA side)."""
    v = synth.lanes_t(seed, shape, bits, signed)
    return v.numpy(), synth.to_bytes_t(v).cuda()


def gpu_pack(bytes_t, f, rows, inner):
    out = samd.empty_words(f, rows, inner)
    samd.samd_pack(f, bytes_t, out, rows, inner)
    return out


def assert_status_clean():
    assert samd.samd_device_status(reset=False) == samd.SAMD_OK


def conv_case(shape: samd.ConvShape, ba, sa, bw, sw, seed, word_bits=32, act_gen=None, wt_gen=None):
    """Seeded NHWC activations and KRSC weights, packed on the GPU; returns
    (act values NHWC, wt values KRSC, act words, wt words, fa, fw)."""
    fa, fw = samd.fmt(ba, sa, 0, word_bits), samd.fmt(bw, sw, 0, word_bits)
    if act_gen is None:
        a_v, a_b = values_and_bytes(seed, (shape.N, shape.H, shape.W, shape.C), ba, sa)
    else:
        a_v = act_gen((shape.N, shape.H, shape.W, shape.C))
        a_b = synth.to_bytes_t(torch.from_numpy(a_v)).cuda()
    if wt_gen is None:
        w_v, w_b = values_and_bytes(seed + 1, (shape.K, shape.R, shape.S, shape.C), bw, sw)
    else:
        w_v = wt_gen((shape.K, shape.R, shape.S, shape.C))
        w_b = synth.to_bytes_t(torch.from_numpy(w_v)).cuda()
    a_w = gpu_pack(a_b, fa, shape.N * shape.H * shape.W, shape.C)
    w_w = gpu_pack(w_b, fw, shape.K * shape.R * shape.S, shape.C)
    return a_v, w_v, a_w, w_w, fa, fw


def oracle_conv_nhwc(a_v, w_v, shape: samd.ConvShape, nthreads=None):
    """Oracle convolution from NHWC values and KRSC weights -> int64 NHWK."""
    nt = nthreads or oracle.max_threads()
    out = oracle.conv2d(a_v.transpose(0, 3, 1, 2), w_v.transpose(0, 3, 1, 2), stride=shape.stride, pad=shape.pad,
                        nthreads=nt)
    return out.transpose(0, 2, 3, 1)


def oracle_requant_pack(acc_nhwk, shift, fo):
    flat = acc_nhwk.reshape(-1, acc_nhwk.shape[-1])
    q = oracle.requant(flat.ravel(), shift, fo.bits, bool(fo.is_signed)).reshape(flat.shape)
    return oracle.pack(q, fo.bits, bool(fo.is_signed), fo.spacer, fo.word_bits)


def harness_shift(ba, bw, bo, k_taps):
    from paper_1809_10572_gb300.workloads import harness_shift as hs

    return hs(ba, bw, bo, k_taps)


def max_abs(bits, signed):
    return (1 << (bits - 1)) if signed else (1 << bits) - 1


def conv_supported(shape, ba, sa, bw, sw):
    """The exactness limits include/samd.h states for samd_conv2d."""
    taps = shape.C * shape.R * shape.S
    if taps * max_abs(ba, sa) * max_abs(bw, sw) < (1 << 24):
        return True
    return bw > 4 and taps * max_abs(ba, sa) * 16 < (1 << 24)


def oracle_conv_rows(a_img_nhwc, w_v, shape, h0, h1):
    """Oracle output rows [h0, h1) of one image (input given as [H][W][C]):
    the zero padding is materialised, the needed input rows are cut out and
    the oracle convolves them without further padding. Returns [h1-h0][Wo][K]."""
    p, st = shape.pad, shape.stride
    img = np.pad(a_img_nhwc, ((p, p), (p, p), (0, 0)))
    crop = img[h0 * st:(h1 - 1) * st + shape.R]
    out = oracle.conv2d(crop.transpose(2, 0, 1)[None], w_v.transpose(0, 3, 1, 2), stride=st, pad=0,
                        nthreads=oracle.max_threads())
    return out[0].transpose(1, 2, 0)
