"""Layer shapes of the synthetic workloads (shapes and formats only).

- conv1x: one 3x3 convolution, N1 C16 -> 16 on 32x32, u4 x s4 in 64-bit words.
- sweep:  3x3 convolution N8 C64 -> 64 on 56x56, pad 1, for every lane width
          b = 1..8 of activations and weights and all four sign combinations,
          requantized to a packed b-bit output (32-bit words).
- vgg16:  the 13 3x3 convolutions of VGG-16 (Simonyan and Zisserman), 224x224
          input, batch 16, u4 activations x s4 weights requantized to u4, a
          2x2 max-pool after blocks 1-4.
- resnet50: the 1x1 and 3x3 convolutions of the four bottleneck stages of
          ResNet-50 v1.5 (stride 2 on the 3x3 and on the projection of the
          first block of stages 2-4), 56x56 stage input, batch 64, s2 weights x
          u6 activations requantized to u6; every layer gets its own input.
- elementwise: 2^28-lane arrays in 32-bit words for every lane width 1..8.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

from .samd import ConvShape


@dataclass(frozen=True)
class ConvLayer:
    name: str
    shape: ConvShape
    ba: int
    sa: bool
    bw: int
    sw: bool
    bo: int
    so: bool
    word_bits: int = 32
    pool_after: bool = False

    @property
    def macs(self) -> int:
        return self.shape.macs


def harness_shift(ba: int, bw: int, bo: int, taps: int) -> int:
    """Requantize shift of the synthetic workloads: scales a sum of `taps`
    uniform products back into a bo-bit lane without saturating or zeroing
    most of it (a harness choice; the paper fixes no shift)."""
    return max(0, ba + bw - bo + math.ceil(math.log2(taps) / 2) - 2)


def conv1x() -> list[ConvLayer]:
    return [ConvLayer("conv3x3_c16", ConvShape(1, 16, 32, 32, 16), 4, False, 4, True, 4, False, word_bits=64)]


SIGN_COMBOS = [(False, False), (False, True), (True, False), (True, True)]  # (activation, weight) signed


def sweep(N: int = 8) -> list[ConvLayer]:
    out = []
    for b in range(1, 9):
        for sa, sw in SIGN_COMBOS:
            out.append(ConvLayer(f"b{b}_{'s' if sa else 'u'}{'s' if sw else 'u'}", ConvShape(N, 64, 56, 56, 64),
                                 b, sa, b, sw, b, sa))
    return out


def vgg16(N: int = 16, H: int = 224) -> list[ConvLayer]:
    cfg = [(3, 64), (64, 64), "P", (64, 128), (128, 128), "P", (128, 256), (256, 256), (256, 256), "P",
           (256, 512), (512, 512), (512, 512), "P", (512, 512), (512, 512), (512, 512)]
    layers, h, i = [], H, 0
    for j, c in enumerate(cfg):
        if c == "P":
            continue
        cin, cout = c
        i += 1
        pool = j + 1 < len(cfg) and cfg[j + 1] == "P"
        layers.append(ConvLayer(f"conv{i}", ConvShape(N, cin, h, h, cout), 4, False, 4, True, 4, False,
                                pool_after=pool))
        if pool:
            h //= 2
    return layers


def resnet50(N: int = 64, H: int = 56) -> list[ConvLayer]:
    layers = []
    cin, h = 64, H
    for stage, (blocks, mid, out) in enumerate([(3, 64, 256), (4, 128, 512), (6, 256, 1024), (3, 512, 2048)]):
        for blk in range(blocks):
            stride = 2 if (blk == 0 and stage > 0) else 1
            ho = (h - 1) // stride + 1
            pre = f"s{stage + 1}b{blk + 1}"
            layers.append(ConvLayer(f"{pre}_1x1a", ConvShape(N, cin, h, h, mid, 1, 1, 1, 0), 6, False, 2, True, 6, False))
            layers.append(ConvLayer(f"{pre}_3x3", ConvShape(N, mid, h, h, mid, 3, 3, stride, 1), 6, False, 2, True, 6,
                                    False))
            layers.append(ConvLayer(f"{pre}_1x1b", ConvShape(N, mid, ho, ho, out, 1, 1, 1, 0), 6, False, 2, True, 6,
                                    False))
            if blk == 0:
                layers.append(ConvLayer(f"{pre}_proj", ConvShape(N, cin, h, h, out, 1, 1, stride, 0), 6, False, 2, True,
                                        6, False))
            cin, h = out, ho
    return layers


WORKLOADS = {"conv1x": conv1x, "sweep": sweep, "vgg16": vgg16, "resnet50": resnet50}

ELEMENTWISE_N = 1 << 28
ELEMENTWISE_OPS = ("add", "sub", "mul", "relu", "requant")


def total_macs(layers) -> int:
    return sum(layer.macs for layer in layers)
