"""Seeded synthetic inputs for tests and benchmarks.

Values are drawn from splitmix64 (Steele, Lea, Flood, "Fast splittable
pseudorandom number generators", OOPSLA 2014): output i (1-based) of seed s
is mix(s + i * 0x9E3779B97F4A7C15). Because it is counter-based, any slice
of a large input can be regenerated on its own, which the sampled parity
checks rely on.

This module holds no arithmetic of the method itself: it only produces
integer arrays, which both the CUDA path and the CPU oracle consume. It
imports neither. The generator runs on torch int64 tensors (wrapping
multiply, logical shifts emulated with masks) so the same definition serves
the CPU (tests) and the GPU (benchmark inputs).
"""
from __future__ import annotations

import numpy as np
import torch

_U64 = (1 << 64) - 1


def _s64(u: int) -> int:
    """The int64 with the same bit pattern as the uint64 u."""
    u &= _U64
    return u - (1 << 64) if u >> 63 else u


_GOLDEN = _s64(0x9E3779B97F4A7C15)
_M1 = _s64(0xBF58476D1CE4E5B9)
_M2 = _s64(0x94D049BB133111EB)


def _lsr(z: torch.Tensor, k: int) -> torch.Tensor:
    """Logical right shift of int64 bit patterns."""
    return (z >> k) & ((1 << (64 - k)) - 1)


def splitmix64(seed: int, n: int, offset: int = 0, device="cpu") -> torch.Tensor:
    """Outputs offset+1 .. offset+n of splitmix64(seed), as int64 bit patterns."""
    i = torch.arange(offset + 1, offset + n + 1, dtype=torch.int64, device=device)
    z = i * _GOLDEN + _s64(seed)
    z = (z ^ _lsr(z, 30)) * _M1
    z = (z ^ _lsr(z, 27)) * _M2
    return z ^ _lsr(z, 31)


def splitmix64_reference(seed: int, n: int, offset: int = 0) -> list[int]:
    """Python big-int splitmix64, the definition the tensor version must match."""
    out = []
    for i in range(offset + 1, offset + n + 1):
        z = (seed + i * 0x9E3779B97F4A7C15) & _U64
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _U64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _U64
        out.append(z ^ (z >> 31))
    return out


def lane_range(bits: int, signed: bool) -> tuple[int, int]:
    """Inclusive [lo, hi] of a b-bit lane: two's complement when signed."""
    if signed:
        return -(1 << (bits - 1)), (1 << (bits - 1)) - 1
    return 0, (1 << bits) - 1


def uniform_ints_t(seed: int, shape, lo: int, hi: int, device="cpu", offset: int = 0) -> torch.Tensor:
    """int64 tensor uniform on [lo, hi] (inclusive), reproducible from seed.

    A power-of-two span takes the top bits of each draw; other spans take
    the draw's top 53 bits modulo the span (bias below 2^-40 for the spans
    used here).
    """
    shape = tuple(shape) if isinstance(shape, (tuple, list)) else (int(shape),)
    n = 1
    for s in shape:
        n *= int(s)
    span = hi - lo + 1
    z = splitmix64(seed, n, offset, device)
    if span & (span - 1) == 0:
        k = span.bit_length() - 1
        v = _lsr(z, 64 - k) if k else torch.zeros_like(z)
    else:
        v = _lsr(z, 11) % span
    return (v + lo).reshape(shape)


def lanes_t(seed: int, shape, bits: int, signed: bool, device="cpu", offset: int = 0) -> torch.Tensor:
    """Lane values for draws offset+1 .. offset+prod(shape); a slice of a large
    input can be regenerated alone by passing its flat offset."""
    lo, hi = lane_range(bits, signed)
    return uniform_ints_t(seed, shape, lo, hi, device, offset)


def lanes(seed: int, shape, bits: int, signed: bool) -> np.ndarray:
    """Values uniform over the full range of a b-bit (un)signed lane (int64 numpy)."""
    return lanes_t(seed, shape, bits, signed).numpy()


def uniform_ints(seed: int, shape, lo: int, hi: int) -> np.ndarray:
    return uniform_ints_t(seed, shape, lo, hi).numpy()


def to_bytes_t(v: torch.Tensor) -> torch.Tensor:
    """One value per byte (the int8 bit pattern; unsigned 200 -> 0xC8 -> -56)."""
    return (v & 0xFF).to(torch.uint8).view(torch.int8)


def lanes_as_bytes(seed: int, shape, bits: int, signed: bool) -> np.ndarray:
    return to_bytes_t(lanes_t(seed, shape, bits, signed)).numpy()


def seed_for(*parts) -> int:
    """A stable 63-bit seed from a tuple of small ints/strings (FNV-1a)."""
    h = 0xCBF29CE484222325
    for p in parts:
        for ch in str(p).encode() + b"\x1f":
            h ^= ch
            h = (h * 0x100000001B3) & _U64
    return h >> 1
