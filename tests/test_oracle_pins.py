"""Pins for the CPU oracle: each check ties an oracle function to something
other than itself -- the paper's word-level routines (a different algorithm),
the paper's worked example, library special cases, closed forms and
invariants. CPU only."""
import itertools
import os

import numpy as np
import pytest
import torch

import oracle
import paper_swar as P
from paper_1809_10572_gb300 import synth

BITS = range(1, 9)
SIGNS = (False, True)
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def all_pairs(bits, signed):
    lo, hi = synth.lane_range(bits, signed)
    vals = np.arange(lo, hi + 1, dtype=np.int64)
    x, y = np.meshgrid(vals, vals, indexing="ij")
    return x.ravel(), y.ravel()


def swar_apply(fn, x, y, bits, signed, word=64):
    """Run a word-level routine over lane vectors packed `word // bits` per word."""
    L = word // bits
    out = []
    for s in range(0, len(x), L):
        xs, ys = x[s:s + L].tolist(), y[s:s + L].tolist()
        r = fn(P.to_word(xs, bits), P.to_word(ys, bits), bits, word)
        r &= P.live_mask(bits, len(xs))
        out.extend(P.from_word(r, bits, len(xs), signed))
    return np.array(out, dtype=np.int64)


# ---- format ---------------------------------------------------------------

# Hand-derived words for the format (lane i at bit offset i*(bits+spacer),
# least-significant lane first, two's complement in `bits` bits, zero
# padding; section 2.1 and Fig. 2 for the spacer, section 6 for lane order).
PACK_CASES = [
    # bits, signed, spacer, word_bits, rows x inner values, words
    (4, False, 0, 32, [[1, 2, 3, 4, 5, 6, 7, 8]], [0x87654321]),
    (3, True, 0, 32, [[-1, 1, -4, 3]], [0x0000070F]),
    (1, False, 0, 32, [[1] * 33], [0xFFFFFFFF, 0x00000001]),
    (8, True, 0, 32, [[-1, 127, -128, 0, 5]], [0x00807FFF, 0x00000005]),
    (5, False, 0, 32, [[31, 0, 1, 2, 3, 4, 5]], [0x0831041F, 0x00000005]),
    (3, False, 1, 32, [[7, 1, 2, 3]], [0x00003217]),
    (4, True, 0, 64, [list(range(-8, 8))], [0x76543210FEDCBA98]),
    (4, False, 0, 32, [[1, 2, 3], [4, 5, 6]], [0x00000321, 0x00000654]),
    (7, True, 0, 32, [[-64, 63, -1, 1, 2]], [0x003FDFC0, 0x00000002]),
    (2, True, 0, 64, [[-2, -1, 0, 1] * 8 + [1]], [0x4E4E4E4E4E4E4E4E, 0x1]),
]


@pytest.mark.parametrize("bits,signed,spacer,word_bits,vals,words", PACK_CASES)
def test_pack_hand_derived_words(bits, signed, spacer, word_bits, vals, words):
    v = np.array(vals, dtype=np.int64)
    got = oracle.pack(v, bits, signed, spacer, word_bits)
    assert [int(w) for w in got] == words
    back = oracle.unpack(got, bits, signed, spacer, word_bits, *v.shape)
    assert np.array_equal(back, v)


@pytest.mark.parametrize("word_bits", (32, 64))
@pytest.mark.parametrize("spacer", (0, 1))
def test_pack_roundtrip_every_value_and_tail(word_bits, spacer):
    for bits, signed in itertools.product(BITS, SIGNS):
        L = oracle.lanes_per_word(bits, spacer, word_bits)
        assert L == word_bits // (bits + spacer)
        lo, hi = synth.lane_range(bits, signed)
        for inner in range(0, 2 * L + 2):
            rows = 3
            v = synth.uniform_ints(synth.seed_for("rt", bits, signed, inner), (rows, inner), lo, hi)
            if inner:
                v.ravel()[: hi - lo + 1] = np.arange(lo, hi + 1)[: v.size]
            w = oracle.pack(v, bits, signed, spacer, word_bits)
            assert w.size == rows * -(-inner // L)
            assert oracle.is_canonical(w, bits, spacer, word_bits, rows, inner)
            assert np.array_equal(oracle.unpack(w, bits, signed, spacer, word_bits, rows, inner), v)


def test_canonical_detects_stray_bits():
    w = oracle.pack([[1, 2, 3]], 3, False, 0, 32)  # lanes 0..2 live, lanes 3..9 and bits 30-31 dead
    assert oracle.is_canonical(w, 3, 0, 32, 1, 3)
    for bit in (9, 29, 30, 31):
        bad = w.copy()
        bad[0] |= np.uint32(1 << bit)
        assert not oracle.is_canonical(bad, 3, 0, 32, 1, 3)
    ws = oracle.pack([[1, 2]], 3, False, 1, 32)  # spacer bit of lane 0 is bit 3
    bad = ws.copy()
    bad[0] |= np.uint32(1 << 3)
    assert not oracle.is_canonical(bad, 3, 1, 32, 1, 2)


def test_pack_keeps_low_bits_of_out_of_range_values():
    v = np.array([[16, -1, 17]], dtype=np.int64)  # 4-bit: 16 -> 0, -1 -> 15, 17 -> 1
    w = oracle.pack(v, 4, False, 0, 32)
    assert int(w[0]) == 0x1F0


# ---- elementwise against the paper's word-level routines --------------------

@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("signed", SIGNS)
def test_add_sub_match_fig5(bits, signed):
    x, y = all_pairs(bits, signed)
    assert np.array_equal(oracle.elementwise("add", x, y, bits=bits, signed=signed),
                          swar_apply(P.samd_add, x, y, bits, signed))
    assert np.array_equal(oracle.elementwise("sub", x, y, bits=bits, signed=signed),
                          swar_apply(P.samd_sub, x, y, bits, signed))


@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("signed", SIGNS)
def test_mul_matches_fig6(bits, signed):
    x, y = all_pairs(bits, signed)
    assert np.array_equal(oracle.elementwise("mul", x, y, bits=bits, signed=signed),
                          swar_apply(P.samd_mul, x, y, bits, signed))


@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("signed", SIGNS)
def test_mul_matches_vector_scale_fig8(bits, signed):
    lo, hi = synth.lane_range(bits, signed)
    vals = np.arange(lo, hi + 1, dtype=np.int64)
    for s in range(lo, hi + 1):
        ys = np.full_like(vals, s)
        want = oracle.elementwise("mul", vals, ys, bits=bits, signed=signed)

        def scale(a, b, bits_, word, s=s):
            return P.vector_scale_wrap(a, s & ((1 << bits_) - 1), bits_, word)

        assert np.array_equal(swar_apply(scale, vals, ys, bits, signed), want)


@pytest.mark.parametrize("bits", range(1, 8))
def test_unsigned_add_with_spacer_fig2(bits):
    x, y = all_pairs(bits, False)
    L = 64 // (bits + 1)
    wrap = oracle.elementwise("add", x, y, bits=bits, signed=False)
    sat = oracle.elementwise("add", x, y, bits=bits, signed=False, saturate=True)
    for s in range(0, len(x), L):
        xs, ys = x[s:s + L].tolist(), y[s:s + L].tolist()
        r = P.unsigned_add_spacer(P.to_word(xs, bits, bits + 1), P.to_word(ys, bits, bits + 1), bits)
        full = P.from_word(r, bits + 1, len(xs), False, bits + 1)  # value bits plus the carry in the spacer
        low = P.from_word(r, bits, len(xs), False, bits + 1)
        assert low == wrap[s:s + L].tolist()
        # the spacer holds the carry: the full field is the exact sum, whose
        # clamp is the saturating add
        assert [min(f, (1 << bits) - 1) for f in full] == sat[s:s + L].tolist()


@pytest.mark.parametrize("bits", range(1, 9))
def test_scale_with_b_spacers_fig7(bits):
    lo, hi = synth.lane_range(bits, False)
    vals = np.arange(lo, hi + 1, dtype=np.int64)
    L = 64 // (2 * bits)
    for s in range(lo, hi + 1):
        want = oracle.elementwise("mul", vals, np.full_like(vals, s), bits=bits, signed=False)
        for a in range(0, len(vals), L):
            vs = vals[a:a + L].tolist()
            r = P.unsigned_scale_b_spacers(P.to_word(vs, bits, 2 * bits), s, bits)
            prods = P.from_word(r, 2 * bits, len(vs), False, 2 * bits)
            assert prods == [v * s for v in vs]  # the 2b-bit field holds the exact product
            assert [p & ((1 << bits) - 1) for p in prods] == want[a:a + L].tolist()


@pytest.mark.parametrize("bits", BITS)
def test_low_product_bits_sign_agnostic(bits):
    # sections 4.1 and 6: the low b bits of a b x b product do not depend on
    # whether the operands are read as signed or unsigned.
    xs, ys = all_pairs(bits, True)
    mask = (1 << bits) - 1
    signed_out = oracle.elementwise("mul", xs, ys, bits=bits, signed=True)
    unsigned_out = oracle.elementwise("mul", xs & mask, ys & mask, bits=bits, signed=False)
    assert np.array_equal(signed_out & mask, unsigned_out)


@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("signed", SIGNS)
@pytest.mark.parametrize("op", ("add", "sub", "mul"))
def test_saturating_ops_clamp_the_exact_result(bits, signed, op):
    x, y = all_pairs(bits, signed)
    lo, hi = synth.lane_range(bits, signed)
    exact = {"add": torch.add, "sub": torch.sub, "mul": torch.mul}[op](torch.from_numpy(x), torch.from_numpy(y))
    want = torch.clamp(exact, lo, hi).numpy()
    got = oracle.elementwise(op, x, y, bits=bits, signed=signed, saturate=True)
    assert np.array_equal(got, want)
    wrapped = oracle.elementwise(op, x, y, bits=bits, signed=signed)
    inside = (exact.numpy() >= lo) & (exact.numpy() <= hi)
    assert np.array_equal(wrapped[inside], got[inside])
    # outside the range the wrapped result differs from the exact one by a multiple of 2^b
    assert np.all((exact.numpy() - wrapped) % (1 << bits) == 0)


@pytest.mark.parametrize("bits", BITS)
@pytest.mark.parametrize("signed", SIGNS)
def test_relu_matches_torch(bits, signed):
    lo, hi = synth.lane_range(bits, signed)
    v = np.arange(lo, hi + 1, dtype=np.int64)
    got = oracle.elementwise("relu", v, bits=bits, signed=signed)
    assert np.array_equal(got, torch.relu(torch.from_numpy(v)).numpy())


@pytest.mark.parametrize("bits_in", BITS)
@pytest.mark.parametrize("signed_in", SIGNS)
@pytest.mark.parametrize("bits_o,signed_o", [(b, s) for b in (1, 2, 4, 6, 8) for s in SIGNS])
def test_requant_matches_floor_division(bits_in, signed_in, bits_o, signed_o):
    lo, hi = synth.lane_range(bits_in, signed_in)
    v = torch.arange(lo, hi + 1, dtype=torch.int64)
    olo, ohi = synth.lane_range(bits_o, signed_o)
    for shift in range(0, 10):
        want = torch.clamp(torch.div(v, 2 ** shift, rounding_mode="floor"), olo, ohi)
        got = oracle.elementwise("requant", v.numpy(), bits=bits_in, signed=signed_in, bits_o=bits_o,
                                 signed_o=signed_o, shift=shift)
        assert np.array_equal(got, want.numpy())


def test_requant_int32_boundaries():
    edges = [-(1 << 31), -(1 << 31) + 1, -65536, -129, -128, -1, 0, 1, 127, 128, 255, 256, 65535, (1 << 31) - 1]
    v = torch.tensor(edges, dtype=torch.int64)
    for shift, (bo, so) in itertools.product(range(0, 31, 3), [(4, True), (4, False), (8, True), (8, False), (1, True)]):
        want = torch.clamp(torch.div(v, 2 ** shift, rounding_mode="floor"), *synth.lane_range(bo, so))
        assert np.array_equal(oracle.requant(v.numpy(), shift, bo, so), want.numpy())
    # monotone and idempotent on in-range values with shift 0
    x = np.arange(-300, 300)
    r = oracle.requant(x, 2, 4, True)
    assert np.all(np.diff(r) >= 0)
    assert np.array_equal(oracle.requant(r, 0, 4, True), r)


# ---- convolution ------------------------------------------------------------

def read_poly_golden():
    with open(os.path.join(GOLDEN, "poly_conv_sec5.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                a, b, c = ([int(t) for t in part.split()] for part in line.split(";"))
                return a, b, c
    raise AssertionError("no golden line")


def full_conv1d_by_oracle(x, k):
    """Full 1D convolution through the oracle's 2D cross-correlation: one row,
    the kernel reversed, padding len(k)-1 on both sides."""
    a = np.array(x, dtype=np.int64).reshape(1, 1, 1, -1)
    w = np.array(k[::-1], dtype=np.int64).reshape(1, 1, 1, -1)
    # pad only along W: place the row in a 1-high image and pad W by hand
    pw = len(k) - 1
    a_p = np.pad(a, ((0, 0), (0, 0), (0, 0), (pw, pw)))
    out = oracle.conv2d(a_p, w, stride=1, pad=0)
    return out.ravel().tolist()


def test_paper_polynomial_example():
    a, b, c = read_poly_golden()
    assert full_conv1d_by_oracle(a, b) == c
    assert P.conv1d_by_wide_multiply(a, b, bits=4, lane=12) == c


@pytest.mark.parametrize("bits", range(2, 9))
@pytest.mark.parametrize("signed_x,signed_k", [(True, True), (False, True), (True, False), (False, False)])
def test_wide_multiply_conv1d_equals_oracle(bits, signed_x, signed_k):
    # sections 5.1 and 6 (Figs. 9-11): one 128-bit product of sign-extended
    # words yields a short 1D convolution; lanes are wide enough for the sums.
    rng_seed = synth.seed_for("wm", bits, signed_x, signed_k)
    for trial in range(60):
        nx, nk = 4 + trial % 3, 3
        lane = 2 * bits + 3
        while (nx + nk - 1) * lane > 128:
            nx -= 1
        x = synth.lanes(rng_seed + trial, (nx,), bits, signed_x).tolist()
        k = synth.lanes(rng_seed + 1000 + trial, (nk,), bits, signed_k).tolist()
        want = full_conv1d_by_oracle(x, k)
        assert P.conv1d_by_wide_multiply(x, k, bits, lane, 128, signed_x, signed_k) == want


def test_naive_underflow_fix_double_counts_but_fig11_does_not():
    # section 6: a lane whose true value is 0 sits above a negative lane. The
    # shift-and-add repair increments the lane above twice; Fig. 11's repair
    # does not. x * k = [-1, 0, ...] style pattern: conv([-1, 1], [1, 1]) = [-1, 0, 1].
    x, k = [-1, 1], [1, 1]
    want = full_conv1d_by_oracle(x, k)
    assert want == [-1, 0, 1]
    assert P.conv1d_by_wide_multiply(x, k, bits=2, lane=6) == want
    assert P.conv1d_by_wide_multiply(x, k, bits=2, lane=6, fix=P.naive_product_fix) != want


def conv_cases():
    cases = []
    for i, (C, H, W, M, R, S, stride, pad) in enumerate([
        (1, 5, 5, 1, 3, 3, 1, 1), (3, 7, 6, 4, 3, 3, 1, 1), (5, 8, 8, 3, 1, 1, 1, 0), (4, 9, 7, 2, 3, 3, 2, 1),
        (2, 6, 6, 5, 1, 1, 2, 0), (6, 5, 9, 3, 3, 1, 1, 0), (3, 4, 4, 2, 3, 3, 1, 2), (7, 10, 10, 4, 5, 5, 2, 2),
    ]):
        for ba, sa, bw, sw in [(4, False, 4, True), (8, True, 8, True), (2, True, 6, False), (1, False, 1, True)]:
            cases.append((i, 2, C, H, W, M, R, S, stride, pad, ba, sa, bw, sw))
    return cases


@pytest.mark.parametrize("case", conv_cases())
def test_conv2d_matches_torch_float64(case):
    i, N, C, H, W, M, R, S, stride, pad, ba, sa, bw, sw = case
    a = synth.lanes(synth.seed_for("ca", *case), (N, C, H, W), ba, sa)
    w = synth.lanes(synth.seed_for("cw", *case), (M, C, R, S), bw, sw)
    got = oracle.conv2d(a, w, stride=stride, pad=pad)
    want = torch.nn.functional.conv2d(torch.from_numpy(a).double(), torch.from_numpy(w).double(), stride=stride,
                                      padding=pad)
    assert np.array_equal(got, want.numpy().astype(np.int64))


@pytest.mark.parametrize("H,W,R,S,stride,pad", [(6, 6, 3, 3, 1, 1), (7, 5, 3, 3, 2, 1), (8, 8, 1, 1, 1, 0),
                                                 (5, 5, 5, 5, 1, 2)])
def test_conv2d_all_ones_counts_in_bounds_taps(H, W, R, S, stride, pad):
    C, M = 3, 2
    out = oracle.conv2d(np.ones((1, C, H, W)), np.ones((M, C, R, S)), stride=stride, pad=pad)
    Ho, Wo = out.shape[2:]
    for h in range(Ho):
        for wv in range(Wo):
            rows = sum(0 <= h * stride - pad + y < H for y in range(R))
            cols = sum(0 <= wv * stride - pad + x < W for x in range(S))
            assert out[0, 0, h, wv] == C * rows * cols


def test_conv2d_multithreaded_equals_single():
    a = synth.lanes(3, (2, 4, 6, 6), 4, False)
    w = synth.lanes(4, (6, 4, 3, 3), 4, True)
    assert np.array_equal(oracle.conv2d(a, w, pad=1, nthreads=1), oracle.conv2d(a, w, pad=1, nthreads=4))


def test_conv2d_int32_bound():
    # 3x3 taps over 4096 channels of u8 x u8 maximum values: 36864 * 255 * 255 > 2^31
    C = 4096
    a = np.full((1, C, 3, 3), 255, dtype=np.int64)
    w = np.full((1, C, 3, 3), 255, dtype=np.int64)
    with pytest.raises(oracle.Int32BoundError):
        oracle.conv2d(a, w)
    w[:, :, 0, 0] = 0  # 8 taps: 32768 * 65025 = 2130739200 < 2^31
    assert oracle.conv2d(a, w)[0, 0, 0, 0] == 8 * C * 255 * 255


def test_config_accumulators_fit_int32():
    # |acc| <= C_in * k^2 * max|a| * max|w| for every workload shape used here
    worst = [
        (16 * 9, 15, 8),            # 3x3, C16, u4 x s4
        (64 * 9, 255, 255),         # 3x3, C64, up to u8 x u8
        (512 * 9, 15, 8),           # VGG-16 deepest 3x3, u4 x s4
        (512 * 9, 63, 2),           # ResNet-50 3x3 at 512 channels, u6 x s2
        (2048, 63, 2),              # ResNet-50 1x1 at 2048 channels
    ]
    for k, ma, mw in worst:
        assert k * ma * mw < 2 ** 31


# ---- max-pool -----------------------------------------------------------------

@pytest.mark.parametrize("bits,signed", [(4, False), (4, True), (1, True), (8, False), (3, True)])
def test_maxpool_matches_torch(bits, signed):
    x = synth.lanes(synth.seed_for("mp", bits, signed), (2, 5, 6, 8), bits, signed)
    got = oracle.maxpool2x2(x)
    want = torch.nn.functional.max_pool2d(torch.from_numpy(x).double(), 2, 2).numpy().astype(np.int64)
    assert np.array_equal(got, want)


# ---- generator ----------------------------------------------------------------

def test_generator_matches_splitmix64_definition():
    got = synth.splitmix64(0x1234, 257, 1000).tolist()
    want = synth.splitmix64_reference(0x1234, 257, 1000)
    assert [g & ((1 << 64) - 1) for g in got] == want
    for bits, signed in itertools.product(BITS, SIGNS):
        v = synth.lanes(7, (4096,), bits, signed)
        lo, hi = synth.lane_range(bits, signed)
        assert v.min() == lo and v.max() == hi
