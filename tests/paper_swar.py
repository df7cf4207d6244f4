"""The paper's word-level SAMD routines, restated on Python integers.

These are a second, independent route to the lane-wise results the oracle
defines: they operate on whole packed words with masks, carries and wide
multiplies, while the oracle works lane by lane on unpacked values. The
pin tests require the two to agree lane for lane. Nothing here is used by
the product path or by the oracle.

Word width is a parameter (64 for the paper's scalar words, 128 for the
double-width products of section 5). Masks follow the build_mask idea of
Fig. 3 with full-width shifts (the listing's `1 << len` is an int shift;
it is read as a word-wide shift here).
"""
from __future__ import annotations


def full(word: int) -> int:
    return (1 << word) - 1


def build_mask(start: int, length: int, stride: int, word: int = 64) -> int:
    """Fig. 3: `length` ones laid down every `stride` bits from bit `start`."""
    unit = (1 << length) - 1
    m = 0
    pos = start
    while pos < word:
        m |= unit << pos
        pos += stride
    return m & full(word)


def msb_lane_mask(w: int, word: int = 64) -> int:
    return build_mask(w - 1, 1, w, word)


def lsb_lane_mask(w: int, word: int = 64) -> int:
    return build_mask(0, 1, w, word)


def odd_lane_mask(w: int, word: int = 64) -> int:
    return build_mask(w, w, 2 * w, word)


def even_lane_mask(w: int, word: int = 64) -> int:
    return build_mask(0, w, 2 * w, word)


def live_mask(bits: int, lanes: int) -> int:
    """Ones over the value bits of the first `lanes` lanes of width `bits`."""
    return (1 << (bits * lanes)) - 1


# ---- packing on Python ints (spacer-free lanes, least-significant first) ----

def to_word(values, bits: int, width: int | None = None) -> int:
    """Place each value's low `bits` bits at lane i of width `width` (default bits)."""
    w = bits if width is None else width
    word = 0
    for i, v in enumerate(values):
        word |= (v & ((1 << bits) - 1)) << (i * w)
    return word


def from_word(word: int, bits: int, count: int, signed: bool, width: int | None = None):
    w = bits if width is None else width
    out = []
    for i in range(count):
        p = (word >> (i * w)) & ((1 << bits) - 1)
        if signed and p >> (bits - 1):
            p -= 1 << bits
        out.append(p)
    return out


# ---- section 3, Fig. 5: add and subtract with temporary spacer bits ----------

def samd_add(a: int, b: int, bits: int, word: int = 64) -> int:
    """Lane-wise add: the lane MSBs act as temporary spacers that catch the
    carries of the low bits; the true MSB is the xor of both MSBs and the
    caught carry."""
    top = msb_lane_mask(bits, word)
    low_sum = (a & ~top) + (b & ~top)
    return ((a ^ b) & top) ^ (low_sum & full(word))


def samd_sub(a: int, b: int, bits: int, word: int = 64) -> int:
    """Lane-wise subtract: set each lane MSB of the minuend and clear it in the
    subtrahend, so no lane borrows from its neighbour; then repair the MSB."""
    top = msb_lane_mask(bits, word)
    diff = ((a | top) - (b & ~top)) & full(word)
    return ((a ^ b) & top) ^ diff ^ top


# ---- section 3, Fig. 6: lane-wise multiply in O(b) steps ---------------------

def samd_mul(a: int, b: int, bits: int, word: int = 64) -> int:
    """Shift-and-add multiply of every lane pair. In step j (j = 0..bits-1) the
    j-th bit of each lane of b selects a (shifted left by j) into a write
    mask that runs from that bit to the top of the lane, built in one step
    as (bit << (bits - j)) - bit; the selected partial products are summed
    with the lane-wise add."""
    read = lsb_lane_mask(bits, word)
    acc = 0
    shifted = a
    for j in range(bits):
        bit = b & read
        write = ((bit << (bits - j)) - bit) & full(word)
        acc = samd_add(acc, shifted & write, bits, word)
        shifted = (shifted << 1) & full(word)
        read = (read << 1) & full(word)
    return acc


# ---- section 2.1, Fig. 2: unsigned add with one permanent spacer bit ---------

def unsigned_add_spacer(a: int, b: int, bits: int, word: int = 64) -> int:
    """Lanes of `bits` value bits plus one spacer above; clearing the spacers
    and adding leaves each lane's carry in its spacer bit."""
    keep = ~msb_lane_mask(bits + 1, word) & full(word)
    return ((a & keep) + (b & keep)) & full(word)


# ---- section 4, Figs. 7 and 8: vector scale ----------------------------------

def unsigned_scale_b_spacers(vec: int, scalar: int, bits: int, word: int = 64) -> int:
    """Unsigned lanes separated by `bits` zero spacer bits times one scalar:
    each lane's 2b-bit product fills the lane and the spacer above it. The
    data sit in the even b-wide fields; the odd fields are cleared first."""
    data = even_lane_mask(bits, word)
    return ((vec & data) * scalar) & full(word)


def vector_scale_wrap(vec: int, scalar: int, bits: int, word: int = 64) -> int:
    """Scale packed b-bit lanes by one b-bit scalar, keeping the low b bits of
    each product: split the even and odd lanes so b zero bits separate the
    lanes of each half, multiply each half, keep the low halves, merge."""
    ev, od = even_lane_mask(bits, word), odd_lane_mask(bits, word)
    lo = ((vec & ev) * scalar) & ev
    hi = ((vec & od) * scalar) & od
    return (lo | hi) & full(word)


# ---- section 6, Figs. 10 and 11: signed lanes in wide multiplies -------------

def sign_extend4mul(vec: int, bits: int, lane: int, word: int) -> int:
    """Lanes hold a `bits`-bit two's-complement pattern in the low bits of a
    `lane`-bit field (zeros above). Subtracting each sign bit from the spacer
    bit just above it sign-extends the lane through the spacers; the borrow
    runs on into the next lane, so the word now equals sum_i v_i * 2^(i*lane)
    modulo 2^word."""
    sign = vec & build_mask(bits - 1, 1, lane, word)
    return (vec - (sign << 1)) & full(word)


def signed_product_fix(product: int, lane: int, word: int) -> int:
    """Fig. 11's repair of a product of sign-extended words: a negative lane
    has borrowed one from the lane above. Adding each lane's sign bit to
    itself carries +1 into the lane above; xoring the sign bits back
    restores each lane's own top bit. Lanes then read as `lane`-bit two's
    complement coefficients."""
    s = product & build_mask(lane - 1, 1, lane, word)
    return ((product + s) & full(word)) ^ s


def naive_product_fix(product: int, lane: int, word: int) -> int:
    """The 'obvious' repair that section 6 warns about: shift each sign bit one
    place left onto the next lane's LSB and add. It double-counts when a
    lane that should read 0 sits above a negative lane."""
    s = product & build_mask(lane - 1, 1, lane, word)
    return (product + (s << 1)) & full(word)


def conv1d_by_wide_multiply(x, k, bits: int, lane: int, word: int = 128, signed_x: bool = True,
                            signed_k: bool = True, fix=signed_product_fix):
    """Full 1D convolution (polynomial product) of two short vectors by one
    wide multiply (section 5.1, Fig. 9): place each value in a `lane`-bit
    field, sign-extend the signed word(s) (Fig. 10), multiply, repair the
    borrows (Fig. 11) and read len(x)+len(k)-1 coefficients. Unsigned
    vectors need no extension: their lanes already hold their values."""
    vx = to_word(x, bits, lane)
    vk = to_word(k, bits, lane)
    if signed_x:
        vx = sign_extend4mul(vx, bits, lane, word)
    if signed_k:
        vk = sign_extend4mul(vk, bits, lane, word)
    prod = fix((vx * vk) & full(word), lane, word)
    n = len(x) + len(k) - 1
    return from_word(prod, lane, n, True, lane)
