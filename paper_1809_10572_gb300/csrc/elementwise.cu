// elementwise.cu -- lane-wise ops on packed words.
//
// Spacer-free formats with the same input and output format take the
// word-level (SAMD) forms: every lane of a word is updated by a handful of
// whole-word integer instructions, the way section 3 of the paper adds and
// subtracts with temporary spacer bits (Fig. 5) and multiplies by masked
// shift-and-add (Fig. 6) at 1-2-bit lanes (from 3 bits, lane by lane on the
// integer multiplier, lane_mul). On GB300 this keeps the per-word ALU cost below
// what HBM bandwidth leaves per word even at 1-2 bit lanes, where a
// lane-by-lane loop would run 16-32 iterations per word. Words move with
// 128-bit loads and stores.
//
// Formats with permanent spacer bits (section 2.1, Fig. 2) and the same
// input and output format take word-level forms too: the zero spacer bits
// above each lane catch the carry of an add and the borrow of a subtract, so
// a wrapping add is one add and one mask, and the saturating forms read each
// lane's carry or borrow from its first spacer bit; the other ops use the
// temporary-spacer forms with masks over the spacer-separated fields.
//
// Requantize into another format takes the per-lane path: one thread per
// output word, bit-field extract, integer op, clamp, insert.
#include "samd_internal.cuh"

namespace samd {
namespace {

constexpr int kThreads = 256;

// ---- compile-time lane masks for spacer-free lanes -------------------------

template <typename W, int BITS>
struct Masks {
  static constexpr int L = WordTraits<W>::kBits / BITS;
  static constexpr W lsb() {
    W m = 0;
    for (int i = 0; i < L; ++i) m |= W(1) << (i * BITS);
    return m;
  }
  static constexpr W kLsb = lsb();                     // bit 0 of every lane
  static constexpr W kMsb = kLsb << (BITS - 1);        // top bit of every lane
  static constexpr W kLane = (W(1) << BITS) - 1;       // one lane's bits
  static constexpr W kLive = kLsb * kLane;             // every lane bit
};

// Spread a mask holding only lane MSBs over the whole of those lanes.
template <typename W, int BITS>
__device__ __forceinline__ W expand_msb(W m) {
  return (m - (m >> (BITS - 1))) | m;
}

// Section 3, Fig. 5: add with the lane MSBs as temporary spacers.
template <typename W, int BITS>
__device__ __forceinline__ W swar_add(W a, W b) {
  constexpr W M = Masks<W, BITS>::kMsb;
  return ((a ^ b) & M) ^ ((a & ~M) + (b & ~M));
}

// Section 3, Fig. 5: subtract; the minuend's MSBs are set and the
// subtrahend's cleared so no lane borrows from the next.
template <typename W, int BITS>
__device__ __forceinline__ W swar_sub(W a, W b) {
  constexpr W M = Masks<W, BITS>::kMsb;
  return ((a ^ b) & M) ^ ((a | M) - (b & ~M)) ^ M;
}

// Saturating add/sub: detect each lane's overflow from the MSBs of the
// operands and the wrapped result, then replace those lanes by the bound.
template <typename W, int BITS>
__device__ __forceinline__ W swar_add_sat(W a, W b, bool is_signed) {
  constexpr W M = Masks<W, BITS>::kMsb;
  constexpr W LIVE = Masks<W, BITS>::kLive;
  W s = swar_add<W, BITS>(a, b);
  if (!is_signed) {
    W carry = ((a & b) | ((a | b) & ~s)) & M;  // carry out of each lane
    return s | expand_msb<W, BITS>(carry);
  }
  W ovf = ~(a ^ b) & (a ^ s) & M;  // same-sign operands, other-sign result
  W E = expand_msb<W, BITS>(ovf);
  W na = a & M;
  W sat = (E & ~expand_msb<W, BITS>(na) & ~M & LIVE) | (E & na);  // 011..1 or 100..0
  return (s & ~E) | sat;
}

template <typename W, int BITS>
__device__ __forceinline__ W swar_sub_sat(W a, W b, bool is_signed) {
  constexpr W M = Masks<W, BITS>::kMsb;
  constexpr W LIVE = Masks<W, BITS>::kLive;
  W d = swar_sub<W, BITS>(a, b);
  if (!is_signed) {
    W borrow = ((~a & b) | ((~a | b) & d)) & M;  // borrow out of each lane
    return d & ~expand_msb<W, BITS>(borrow);
  }
  W ovf = (a ^ b) & (a ^ d) & M;  // other-sign operands, result sign differs from a
  W E = expand_msb<W, BITS>(ovf);
  W na = a & M;
  W sat = (E & ~expand_msb<W, BITS>(na) & ~M & LIVE) | (E & na);
  return (d & ~E) | sat;
}

// Section 3, Fig. 6: lane-wise multiply, low bits, by masked shift-and-add;
// in step j the j-th bit of each lane of b selects a << j, cut at the top of
// the lane by a mask built in one subtraction.
template <typename W, int BITS>
__device__ __forceinline__ W swar_mul(W a, W b) {
  constexpr W LSB = Masks<W, BITS>::kLsb;
  W acc = 0;
#pragma unroll
  for (int j = 0; j < BITS; ++j) {
    W bit = b & (LSB << j);
    W write = (bit << (BITS - j)) - bit;
    acc = swar_add<W, BITS>(acc, (a << j) & write);
  }
  return acc;
}

// Wrapping lane product on the integer multiplier without taking a's lane
// out: with s the lane's offset and M = (2^bits - 1) << s its data bits,
// b & M is b_i * 2^s, so (a >> s) * (b & M) = ((a >> s) * b_i) << s, whose
// bits [s, s + bits) are a_i * b_i mod 2^bits (the bits of a above lane i
// reach only higher product bits). One shift, one multiply and two logic
// operations per lane; the low bits are the same for signed and unsigned
// lanes (section 4.1). 32-bit words only (s + bits <= 32).
__device__ __forceinline__ uint32_t lane_mul_at(uint32_t r, uint32_t a, uint32_t b, int s, uint32_t M) {
  return r | (((a >> s) * (b & M)) & M);
}

// Lane-by-lane multiply (cheaper than shift-and-add from 3-bit lanes up).
template <typename W, int BITS>
__device__ __forceinline__ W lane_mul(W a, W b, bool is_signed, bool sat) {
  constexpr int L = Masks<W, BITS>::L;
  constexpr uint32_t LM = (1u << BITS) - 1;
  if constexpr (sizeof(W) == 4) {
    if (!sat) {
      uint32_t r = 0;
#pragma unroll
      for (int i = 0; i < L; ++i) r = lane_mul_at(r, a, b, i * BITS, LM << (i * BITS));
      return r;
    }
  }
  const int lo = lane_lo(BITS, is_signed), hi = lane_hi(BITS, is_signed);
  W r = 0;
#pragma unroll
  for (int i = 0; i < L; ++i) {
    uint32_t pa = static_cast<uint32_t>(a >> (i * BITS)) & LM;
    uint32_t pb = static_cast<uint32_t>(b >> (i * BITS)) & LM;
    uint32_t p;
    if (sat) {
      int v = lane_value(pa, BITS, is_signed) * lane_value(pb, BITS, is_signed);
      p = static_cast<uint32_t>(clamp_int(v, lo, hi)) & LM;
    } else {
      p = (pa * pb) & LM;  // low bits are the same for signed and unsigned (section 4.1)
    }
    r |= W(p) << (i * BITS);
  }
  return r;
}

template <typename W, int BITS>
__device__ __forceinline__ W swar_relu(W a, bool is_signed) {
  if (!is_signed) return a;
  constexpr W M = Masks<W, BITS>::kMsb;
  return a & ~expand_msb<W, BITS>(a & M);
}

// Requantize within the format: floor(x / 2^shift) per lane. A right shift
// never leaves the lane range, so no clamp is needed. `keep` holds the low
// (BITS - shift) bits of every lane.
template <typename W, int BITS>
__device__ __forceinline__ W swar_shift(W a, int shift, W keep, bool is_signed) {
  if (shift == 0) return a;
  W r = (a >> shift) & keep;
  if (is_signed) {
    constexpr W M = Masks<W, BITS>::kMsb;
    W sg = a & M;
    W t = sg >> (shift - 1);
    r |= (sg - t) | sg;  // sign fill of the top `shift` bits of negative lanes
  }
  return r;
}

template <typename W, int BITS, int OP>
__device__ __forceinline__ W apply_op(W a, W b, bool is_signed, bool sat, int shift, W keep) {
  if constexpr (OP == SAMD_ADD) {
    return sat ? swar_add_sat<W, BITS>(a, b, is_signed) : swar_add<W, BITS>(a, b);
  } else if constexpr (OP == SAMD_SUB) {
    return sat ? swar_sub_sat<W, BITS>(a, b, is_signed) : swar_sub<W, BITS>(a, b);
  } else if constexpr (OP == SAMD_MUL) {
    if constexpr (BITS == 1) {
      if (!sat || !is_signed) return a & b;  // 1-bit: product = AND (u1 never overflows)
      return lane_mul<W, BITS>(a, b, is_signed, sat);
    } else if constexpr (BITS == 2) {
      if (!sat) return swar_mul<W, BITS>(a, b);
      return lane_mul<W, BITS>(a, b, is_signed, sat);
    } else {
      return lane_mul<W, BITS>(a, b, is_signed, sat);
    }
  } else if constexpr (OP == SAMD_RELU) {
    return swar_relu<W, BITS>(a, is_signed);
  } else {
    return swar_shift<W, BITS>(a, shift, keep, is_signed);
  }
}

template <typename W>
struct Vec4 {
  static constexpr int kWords = 16 / sizeof(W);
};

template <typename W, int BITS, int OP>
__global__ void __launch_bounds__(kThreads)
    ew_swar_kernel(const W *__restrict__ a, const W *__restrict__ b, W *__restrict__ out, int64_t nwords,
                   int is_signed, int sat, int shift) {
  constexpr int V = Vec4<W>::kWords;
  constexpr bool kBinary = (OP == SAMD_ADD || OP == SAMD_SUB || OP == SAMD_MUL);
  W keep = 0;
  if (OP == SAMD_REQUANT) {
    int s = shift < BITS ? shift : BITS;
    keep = Masks<W, BITS>::kLsb * ((W(1) << (BITS - s)) - 1);
    shift = s;
  }
  const int64_t nvec = nwords / V;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < nvec; v += stride) {
    uint4 ra = __ldcs(reinterpret_cast<const uint4 *>(a) + v);
    uint4 rb = ra;
    if (kBinary) rb = __ldcs(reinterpret_cast<const uint4 *>(b) + v);
    W wa[V], wb[V], wo[V];
    memcpy(wa, &ra, 16);
    memcpy(wb, &rb, 16);
#pragma unroll
    for (int k = 0; k < V; ++k) wo[k] = apply_op<W, BITS, OP>(wa[k], wb[k], is_signed, sat, shift, keep);
    uint4 ro;
    memcpy(&ro, wo, 16);
    __stcs(reinterpret_cast<uint4 *>(out) + v, ro);
  }
  // tail words that do not fill a 128-bit vector
  for (int64_t w = nvec * V + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < nwords; w += stride) {
    W x = a[w];
    W y = kBinary ? b[w] : x;
    out[w] = apply_op<W, BITS, OP>(x, y, is_signed, sat, shift, keep);
  }
}

// Per-lane path: any spacer, any output format. One thread per output word.
struct LaneFmt {
  int bits, is_signed, lane_w, L;
};

template <typename WI, typename WO>
__global__ void __launch_bounds__(kThreads)
    ew_lane_kernel(int op, LaneFmt fa, const WI *__restrict__ a, const WI *__restrict__ b, LaneFmt fo,
                   WO *__restrict__ out, int64_t n, int64_t nwords_out, int shift, int sat) {
  const uint32_t ma = (1u << fa.bits) - 1, mo = (1u << fo.bits) - 1;
  const int lo = lane_lo(fo.bits, fo.is_signed), hi = lane_hi(fo.bits, fo.is_signed);
  for (int64_t w = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < nwords_out;
       w += (int64_t)gridDim.x * blockDim.x) {
    WO word = 0;
    for (int l = 0; l < fo.L; ++l) {
      int64_t e = w * fo.L + l;
      if (e >= n) break;
      int64_t wi = e / fa.L;
      int li = static_cast<int>(e - wi * fa.L);
      int x = lane_value(static_cast<uint32_t>(a[wi] >> (li * fa.lane_w)) & ma, fa.bits, fa.is_signed);
      int y = 0;
      if (op == SAMD_ADD || op == SAMD_SUB || op == SAMD_MUL)
        y = lane_value(static_cast<uint32_t>(b[wi] >> (li * fa.lane_w)) & ma, fa.bits, fa.is_signed);
      int v;
      switch (op) {
        case SAMD_ADD: v = x + y; break;
        case SAMD_SUB: v = x - y; break;
        case SAMD_MUL: v = x * y; break;
        case SAMD_RELU: v = x < 0 ? 0 : x; break;
        default: v = x >> shift; break;  // arithmetic shift: floor(x / 2^shift)
      }
      if (op == SAMD_REQUANT || sat) v = clamp_int(v, lo, hi);
      word |= WO(static_cast<uint32_t>(v) & mo) << (l * fo.lane_w);
    }
    out[w] = word;
  }
}

// ---- formats with permanent spacer bits ------------------------------------
//
// A lane field is bits data bits plus spacer zero bits above them, L fields
// per word (FieldMasks, samd_internal.cuh).

template <typename W>
__device__ __forceinline__ W field_relu(W a, const FieldMasks<W> &f, bool is_signed) {
  if (!is_signed) return a;
  return a & ~spread_down<W>(a & f.msb, f.bits - 1);
}

template <typename W>
__device__ __forceinline__ W field_shift(W a, int shift, W keep, const FieldMasks<W> &f, bool is_signed) {
  if (shift == 0) return a;
  W r = (a >> shift) & keep;
  if (is_signed) {
    W sg = a & f.msb;
    W t = sg >> (shift - 1);
    r |= (sg - t) | sg;  // sign fill of the top `shift` data bits of negative lanes
  }
  return r;
}

// Fig. 2: with the spacers zero (canonical inputs) the word add leaves each
// lane's carry in its first spacer bit. Wrapping: drop it. Saturating,
// unsigned: a set carry bit turns the lane's data bits all ones. Signed:
// overflow where same-sign operands give a result of the other sign.
template <typename W>
__device__ __forceinline__ W field_add(W a, W b, const FieldMasks<W> &f, bool is_signed, bool sat) {
  const W s = a + b;
  if (!sat) return s & f.live;
  if (!is_signed) {
    const W c = s & f.carry;
    return (s | (c - (c >> f.bits))) & f.live;
  }
  const W w = s & f.live;
  const W E = spread_down<W>(~(a ^ b) & (a ^ w) & f.msb, f.bits - 1);  // overflowed lanes
  const W na = a & f.msb;                                                 // their operands' sign
  const W sat_v = (E & ~spread_down<W>(na, f.bits - 1) & ~f.msb & f.live) | (E & na);  // 011..1 or 100..0
  return (w & ~E) | sat_v;
}

// (a | carry) - b: each field computes 2^bits + a - b > 0, so no borrow
// leaves a field, and the carry bit stays set exactly where a >= b
// (unsigned).
template <typename W>
__device__ __forceinline__ W field_sub(W a, W b, const FieldMasks<W> &f, bool is_signed, bool sat) {
  const W d = (a | f.carry) - b;
  if (!sat) return d & f.live;
  if (!is_signed) {
    const W ge = d & f.carry;
    return d & (ge - (ge >> f.bits)) & f.live;  // lanes with a < b clamp to 0
  }
  const W w = d & f.live;
  const W E = spread_down<W>((a ^ b) & (a ^ w) & f.msb, f.bits - 1);
  const W na = a & f.msb;
  const W sat_v = (E & ~spread_down<W>(na, f.bits - 1) & ~f.msb & f.live) | (E & na);
  return (w & ~E) | sat_v;
}

template <typename W>
__device__ __forceinline__ W field_mul(W a, W b, const FieldMasks<W> &f, bool is_signed, bool sat) {
  if (!sat && f.bits <= f.L) {
    // Fig. 6 shift-and-add over the fields: step j adds a << j where bit j
    // of the lane of b is set, cut at the top of the lane's data bits; bits
    // steps of a few word operations each, against L lanes of extract,
    // multiply and insert (measured: shift-and-add wins while bits <= L,
    // e.g. 0.51 -> 0.90 of HBM at 3-bit lanes with one spacer bit in 32-bit
    // words, and loses at 6 and 7 bits, four lanes per word). 32-bit words
    // reach this only where field_mul_by_lanes declines the multiplier form.
    W acc = 0;
    for (int j = 0; j < f.bits; ++j) {
      const W bit = b & (f.lsb << j);
      const W write = (bit << (f.bits - j)) - bit;
      acc = (acc + ((a << j) & write)) & f.live;  // the spacer catches the carry
    }
    return acc;
  }
  const uint32_t lm = (1u << f.bits) - 1;
  const int lo = lane_lo(f.bits, is_signed), hi = lane_hi(f.bits, is_signed);
  W r = 0;
  for (int i = 0; i < f.L; ++i) {
    const uint32_t pa = static_cast<uint32_t>(a >> (i * f.fw)) & lm;
    const uint32_t pb = static_cast<uint32_t>(b >> (i * f.fw)) & lm;
    uint32_t p;
    if (sat)
      p = static_cast<uint32_t>(clamp_int(lane_value(pa, f.bits, is_signed) * lane_value(pb, f.bits, is_signed), lo,
                                          hi)) & lm;
    else
      p = (pa * pb) & lm;
    r |= W(p) << (i * f.fw);
  }
  return r;
}

// The wrapping multiply of V words of 32-bit spacer-separated fields, lane
// outermost so the runtime lane loop's bookkeeping is shared by the words
// (lane_mul_at per field).
template <int V>
__device__ __forceinline__ void field_mul_lanes(const uint32_t *a, const uint32_t *b, uint32_t *o,
                                                const FieldMasks<uint32_t> &f) {
#pragma unroll
  for (int k = 0; k < V; ++k) o[k] = 0;
  uint32_t M = (1u << f.bits) - 1;
  for (int s = 0, i = 0; i < f.L; ++i, s += f.fw, M <<= f.fw) {
#pragma unroll
    for (int k = 0; k < V; ++k) o[k] = lane_mul_at(o[k], a[k], b[k], s, M);
  }
}

// Per word, shift-and-add costs about nine operations a step (bits steps)
// and field_mul_lanes about five a lane (L lanes): take the lanes form where
// it is cheaper (from 4-bit lanes with one spacer bit in 32-bit words).
__device__ __forceinline__ bool field_mul_by_lanes(const FieldMasks<uint32_t> &f) {
  return 5 * f.L < 9 * f.bits;
}

template <typename W, int OP>
__device__ __forceinline__ W field_op(W a, W b, const FieldMasks<W> &f, bool is_signed, bool sat, int shift,
                                      W keep) {
  if constexpr (OP == SAMD_ADD) return field_add<W>(a, b, f, is_signed, sat);
  else if constexpr (OP == SAMD_SUB) return field_sub<W>(a, b, f, is_signed, sat);
  else if constexpr (OP == SAMD_MUL) return field_mul<W>(a, b, f, is_signed, sat);
  else if constexpr (OP == SAMD_RELU) return field_relu<W>(a, f, is_signed);
  else return field_shift<W>(a, shift, keep, f, is_signed);
}

// Held to 8 CTAs of 256 threads per SM (32 registers): the multiply's two
// forms in one kernel would otherwise take 40 and fit 6.
template <typename W, int OP>
__global__ void __launch_bounds__(kThreads, 8)
    ew_field_kernel(const W *__restrict__ a, const W *__restrict__ b, W *__restrict__ out, int64_t nwords,
                    const FieldMasks<W> f, int is_signed, int sat, int shift) {
  constexpr int V = 16 / sizeof(W);
  constexpr bool kBinary = (OP == SAMD_ADD || OP == SAMD_SUB || OP == SAMD_MUL);
  W keep = 0;
  if (OP == SAMD_REQUANT) {
    const int s = shift < f.bits ? shift : f.bits;
    keep = f.lsb * ((W(1) << (f.bits - s)) - 1);
    shift = s;
  }
  const int64_t nvec = nwords / V;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < nvec; v += stride) {
    const uint4 ra = __ldcs(reinterpret_cast<const uint4 *>(a) + v);
    uint4 rb = ra;
    if (kBinary) rb = __ldcs(reinterpret_cast<const uint4 *>(b) + v);
    W wa[V], wb[V], wo[V];
    memcpy(wa, &ra, 16);
    memcpy(wb, &rb, 16);
    if constexpr (OP == SAMD_MUL && sizeof(W) == 4) {
      if (!sat && field_mul_by_lanes(f)) {
        field_mul_lanes<V>(wa, wb, wo, f);
      } else {
#pragma unroll
        for (int k = 0; k < V; ++k) wo[k] = field_op<W, OP>(wa[k], wb[k], f, is_signed, sat, shift, keep);
      }
    } else {
#pragma unroll
      for (int k = 0; k < V; ++k) wo[k] = field_op<W, OP>(wa[k], wb[k], f, is_signed, sat, shift, keep);
    }
    uint4 ro;
    memcpy(&ro, wo, 16);
    __stcs(reinterpret_cast<uint4 *>(out) + v, ro);
  }
  for (int64_t w = nvec * V + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < nwords; w += stride) {
    const W x = a[w];
    const W y = kBinary ? b[w] : x;
    if constexpr (OP == SAMD_MUL && sizeof(W) == 4) {
      if (!sat && field_mul_by_lanes(f)) {
        uint32_t r;
        field_mul_lanes<1>(&x, &y, &r, f);
        out[w] = r;
        continue;
      }
    }
    out[w] = field_op<W, OP>(x, y, f, is_signed, sat, shift, keep);
  }
}

template <typename W>
cudaError_t field_dispatch(samd_op op, samd_fmt f, const void *a, const void *b, void *out, int64_t n, int shift,
                           int sat, cudaStream_t s) {
  const int64_t nwords = words_per_row(f, n);
  const int64_t work = nwords / (16 / sizeof(W)) + 1;
  const FieldMasks<W> m = field_masks<W>(f);
  const W *pa = static_cast<const W *>(a);
  const W *pb = static_cast<const W *>(b);
  W *po = static_cast<W *>(out);
  switch (op) {
#define SAMD_FIELD_CASE(OPC)                                                                     \
  case OPC:                                                                                      \
    ew_field_kernel<W, OPC><<<resident_grid<ew_field_kernel<W, OPC>>(work, kThreads), kThreads, 0, s>>>( \
        pa, pb, po, nwords, m, f.is_signed, sat, shift);                                         \
    break;
    SAMD_FIELD_CASE(SAMD_ADD) SAMD_FIELD_CASE(SAMD_SUB) SAMD_FIELD_CASE(SAMD_MUL) SAMD_FIELD_CASE(SAMD_RELU)
#undef SAMD_FIELD_CASE
    default:
      ew_field_kernel<W, SAMD_REQUANT><<<resident_grid<ew_field_kernel<W, SAMD_REQUANT>>(work, kThreads), kThreads,
                                          0, s>>>(pa, pb, po, nwords, m, f.is_signed, sat, shift);
      break;
  }
  return cudaGetLastError();
}

template <typename W, int OP>
cudaError_t swar_dispatch_bits(int bits, const void *a, const void *b, void *out, int64_t nwords, int is_signed,
                               int sat, int shift, cudaStream_t s) {
  int64_t work = nwords / Vec4<W>::kWords + 1;
  const W *pa = static_cast<const W *>(a);
  const W *pb = static_cast<const W *>(b);
  W *po = static_cast<W *>(out);
  switch (bits) {
#define SAMD_EW_CASE(B) \
  case B:               \
    ew_swar_kernel<W, B, OP><<<resident_grid<ew_swar_kernel<W, B, OP>>(work, kThreads), kThreads, 0, s>>>( \
        pa, pb, po, nwords, is_signed, sat, shift);                                                    \
    break;
    SAMD_EW_CASE(1) SAMD_EW_CASE(2) SAMD_EW_CASE(3) SAMD_EW_CASE(4)
    SAMD_EW_CASE(5) SAMD_EW_CASE(6) SAMD_EW_CASE(7) SAMD_EW_CASE(8)
#undef SAMD_EW_CASE
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

template <typename W>
cudaError_t swar_dispatch(samd_op op, int bits, const void *a, const void *b, void *out, int64_t nwords,
                          int is_signed, int sat, int shift, cudaStream_t s) {
  switch (op) {
    case SAMD_ADD: return swar_dispatch_bits<W, SAMD_ADD>(bits, a, b, out, nwords, is_signed, sat, shift, s);
    case SAMD_SUB: return swar_dispatch_bits<W, SAMD_SUB>(bits, a, b, out, nwords, is_signed, sat, shift, s);
    case SAMD_MUL: return swar_dispatch_bits<W, SAMD_MUL>(bits, a, b, out, nwords, is_signed, sat, shift, s);
    case SAMD_RELU: return swar_dispatch_bits<W, SAMD_RELU>(bits, a, b, out, nwords, is_signed, sat, shift, s);
    default: return swar_dispatch_bits<W, SAMD_REQUANT>(bits, a, b, out, nwords, is_signed, sat, shift, s);
  }
}

LaneFmt lane_fmt(samd_fmt f) {
  return LaneFmt{f.bits, f.is_signed, f.bits + f.spacer, lanes_per_word(f)};
}

template <typename WI, typename WO>
cudaError_t lane_dispatch(samd_op op, samd_fmt fa, const void *a, const void *b, samd_fmt fo, void *out, int64_t n,
                          int shift, int sat, cudaStream_t s) {
  int64_t nwo = words_per_row(fo, n);
  int grid = grid_for(nwo, kThreads, sm_count() * 16);
  ew_lane_kernel<WI, WO><<<grid, kThreads, 0, s>>>(static_cast<int>(op), lane_fmt(fa), static_cast<const WI *>(a),
                                                   static_cast<const WI *>(b), lane_fmt(fo), static_cast<WO *>(out),
                                                   n, nwo, shift, sat);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_elementwise(samd_op op, samd_fmt fa, const void *a, const void *b, samd_fmt fo, void *out,
                               int64_t n, int shift, int saturate, cudaStream_t s) {
  if (same_fmt(fa, fo) && fa.spacer != 0) {  // permanent spacer bits: the field forms above
    if (fa.word_bits == 32) return field_dispatch<uint32_t>(op, fa, a, b, out, n, shift, saturate, s);
    return field_dispatch<uint64_t>(op, fa, a, b, out, n, shift, saturate, s);
  }
  bool swar = same_fmt(fa, fo) && fa.spacer == 0;
  if (swar) {
    int64_t nwords = words_per_row(fa, n);
    if (fa.word_bits == 32)
      return swar_dispatch<uint32_t>(op, fa.bits, a, b, out, nwords, fa.is_signed, saturate, shift, s);
    return swar_dispatch<uint64_t>(op, fa.bits, a, b, out, nwords, fa.is_signed, saturate, shift, s);
  }
  if (fa.word_bits == 32 && fo.word_bits == 32)
    return lane_dispatch<uint32_t, uint32_t>(op, fa, a, b, fo, out, n, shift, saturate, s);
  if (fa.word_bits == 32)
    return lane_dispatch<uint32_t, uint64_t>(op, fa, a, b, fo, out, n, shift, saturate, s);
  if (fo.word_bits == 32)
    return lane_dispatch<uint64_t, uint32_t>(op, fa, a, b, fo, out, n, shift, saturate, s);
  return lane_dispatch<uint64_t, uint64_t>(op, fa, a, b, fo, out, n, shift, saturate, s);
}

}  // namespace samd
