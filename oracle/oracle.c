/*
 * oracle.c -- plain, slow CPU definition of the bit-precise SAMD hot path.
 *
 * TEST INFRASTRUCTURE. Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg load this library. The product library
 * (libsamd) never calls it; the two share no source, header, table or
 * helper. Every value here is an unpacked int64; no word-level tricks are
 * used to compute a reference result.
 *
 * Paper: Anderson, Doyle, Gregg, "Scalar Arithmetic Multiple Data:
 * Customizable Precision for Deep Neural Networks" (arXiv 1809.10572).
 *
 * Packed format (the SAMD vector of section 2, "Emulating Vector
 * Architectures", with the permanent spacer bits of Fig. 2 as an option):
 *   lane width w = bits + spacer; L = floor(word_bits / w) lanes per word.
 *   Element i of a row sits in word floor(i / L) at bit offset (i mod L) * w,
 *   least-significant lane first (section 6: the "rightmost" lane is the
 *   lowest one). The lane's value occupies its low `bits` bits, two's
 *   complement when signed (section 6); the spacer bits above it, the bits
 *   above the last whole lane and the lanes past the end of a row are zero.
 *   Every row starts on a word boundary. Words are stored little-endian.
 *
 * Parity pins for each function live in tests/test_oracle_*.py.
 */
#include <stdint.h>
#include <stddef.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_EINVAL 1
#define OR_ERANGE 7 /* an int32 accumulator bound was exceeded */

enum { OR_ADD = 0, OR_SUB = 1, OR_MUL = 2, OR_RELU = 3, OR_REQUANT = 4 };

static int valid_fmt(int bits, int spacer, int word_bits) {
  if (bits < 1 || bits > 8) return 0;
  if (spacer < 0 || spacer > 8) return 0;
  if (word_bits != 32 && word_bits != 64) return 0;
  return bits + spacer <= word_bits;
}

int oracle_lanes_per_word(int bits, int spacer, int word_bits) {
  if (!valid_fmt(bits, spacer, word_bits)) return 0;
  return word_bits / (bits + spacer);
}

int64_t oracle_packed_words(int bits, int spacer, int word_bits, int64_t rows, int64_t inner) {
  int L = oracle_lanes_per_word(bits, spacer, word_bits);
  if (L == 0 || rows < 0 || inner < 0) return -1;
  return rows * ((inner + L - 1) / L);
}

/* The range of a b-bit lane: [-2^(b-1), 2^(b-1)-1] signed, [0, 2^b-1] unsigned
 * (two's complement, section 6). */
static int64_t lane_min(int bits, int is_signed) { return is_signed ? -((int64_t)1 << (bits - 1)) : 0; }
static int64_t lane_max(int bits, int is_signed) {
  return is_signed ? (((int64_t)1 << (bits - 1)) - 1) : (((int64_t)1 << bits) - 1);
}

/* Reduce v modulo 2^bits into the lane's range: the wrap-around that a
 * b-bit scalar has (section 5.1: the same overflow behaviour as a b-bit
 * scalar; section 3: add and subtract are correct for signed and unsigned). */
int64_t oracle_wrap(int64_t v, int bits, int is_signed) {
  int64_t m = (int64_t)1 << bits;
  int64_t r = v % m;
  if (r < 0) r += m;
  if (is_signed && r > lane_max(bits, 1)) r -= m;
  return r;
}

int64_t oracle_clamp(int64_t v, int bits, int is_signed) {
  int64_t lo = lane_min(bits, is_signed), hi = lane_max(bits, is_signed);
  return v < lo ? lo : (v > hi ? hi : v);
}

/* floor(v / 2^shift): the arithmetic right shift of a two's-complement value. */
static int64_t floor_shift(int64_t v, int shift) {
  int64_t d = (int64_t)1 << shift;
  int64_t q = v / d;
  if ((v % d) != 0 && v < 0) q -= 1;
  return q;
}

/* ---- pack / unpack ----------------------------------------------------- */

static void put_bit(uint8_t *words, int64_t bitpos, int bit) {
  if (bit) words[bitpos >> 3] |= (uint8_t)(1u << (bitpos & 7));
}
static int get_bit(const uint8_t *words, int64_t bitpos) {
  return (words[bitpos >> 3] >> (bitpos & 7)) & 1;
}

/* Pack rows x inner values into the packed format. Each value contributes
 * its low `bits` bits (v mod 2^bits). `out` holds
 * oracle_packed_words(...) * word_bits / 8 bytes and is fully written. */
int oracle_pack(int bits, int is_signed, int spacer, int word_bits, const int64_t *vals, int64_t rows,
                int64_t inner, uint8_t *out) {
  (void)is_signed;
  int L = oracle_lanes_per_word(bits, spacer, word_bits);
  if (L == 0 || rows < 0 || inner < 0) return OR_EINVAL;
  int64_t wpr = (inner + L - 1) / L;
  int64_t nbytes = rows * wpr * (word_bits / 8);
  memset(out, 0, (size_t)nbytes);
  for (int64_t r = 0; r < rows; r++) {
    for (int64_t i = 0; i < inner; i++) {
      int64_t word = r * wpr + i / L;
      int64_t off = (i % L) * (bits + spacer);
      int64_t pattern = oracle_wrap(vals[r * inner + i], bits, 0);
      for (int k = 0; k < bits; k++) put_bit(out, word * word_bits + off + k, (int)((pattern >> k) & 1));
    }
  }
  return OR_OK;
}

/* Unpack: each lane's bit pattern is read back as a two's-complement
 * (signed) or plain binary (unsigned) number. */
int oracle_unpack(int bits, int is_signed, int spacer, int word_bits, const uint8_t *in, int64_t rows,
                  int64_t inner, int64_t *vals) {
  int L = oracle_lanes_per_word(bits, spacer, word_bits);
  if (L == 0 || rows < 0 || inner < 0) return OR_EINVAL;
  int64_t wpr = (inner + L - 1) / L;
  for (int64_t r = 0; r < rows; r++) {
    for (int64_t i = 0; i < inner; i++) {
      int64_t word = r * wpr + i / L;
      int64_t off = (i % L) * (bits + spacer);
      int64_t pattern = 0;
      for (int k = 0; k < bits; k++) pattern |= (int64_t)get_bit(in, word * word_bits + off + k) << k;
      if (is_signed && pattern > lane_max(bits, 1)) pattern -= (int64_t)1 << bits;
      vals[r * inner + i] = pattern;
    }
  }
  return OR_OK;
}

/* 1 if every spacer bit, every bit above the last whole lane and every lane
 * past the end of a row is zero (the canonical form of the format). */
int oracle_is_canonical(int bits, int spacer, int word_bits, const uint8_t *in, int64_t rows, int64_t inner) {
  int L = oracle_lanes_per_word(bits, spacer, word_bits);
  if (L == 0) return 0;
  int64_t wpr = (inner + L - 1) / L;
  for (int64_t r = 0; r < rows; r++)
    for (int64_t w = 0; w < wpr; w++)
      for (int k = 0; k < word_bits; k++) {
        int lane = k / (bits + spacer);
        int in_lane = k % (bits + spacer);
        int64_t elem = w * L + lane;
        int live = lane < L && in_lane < bits && elem < inner;
        if (!live && get_bit(in, (r * wpr + w) * word_bits + k)) return 0;
      }
  return 1;
}

/* ---- elementwise -------------------------------------------------------- */

/* Lane-wise operations on unpacked values.
 *   ADD/SUB (section 3, Fig. 5): (x +/- y) wrapped to the lane width, or
 *     clamped to the lane range when `saturate` is set.
 *   MUL (section 3, Fig. 6; section 4.1): the low `bits` bits of x*y, the
 *     same for signed and unsigned lanes; clamped when `saturate` is set.
 *   RELU: max(x, 0) for signed lanes, the identity for unsigned lanes.
 *   REQUANT: clamp_out(floor(x / 2^shift)) into the output lane format
 *     (bits_o, signed_o); an unsigned output clamps negatives to 0.
 * ADD/SUB/MUL/RELU keep the input format (bits_o/signed_o are ignored). */
int oracle_elementwise(int op, int bits_a, int signed_a, int bits_o, int signed_o, const int64_t *x,
                       const int64_t *y, int64_t *out, int64_t n, int shift, int saturate) {
  if (bits_a < 1 || bits_a > 32 || n < 0) return OR_EINVAL;
  for (int64_t i = 0; i < n; i++) {
    int64_t v;
    switch (op) {
      case OR_ADD:
        v = x[i] + y[i];
        out[i] = saturate ? oracle_clamp(v, bits_a, signed_a) : oracle_wrap(v, bits_a, signed_a);
        break;
      case OR_SUB:
        v = x[i] - y[i];
        out[i] = saturate ? oracle_clamp(v, bits_a, signed_a) : oracle_wrap(v, bits_a, signed_a);
        break;
      case OR_MUL:
        v = x[i] * y[i];
        out[i] = saturate ? oracle_clamp(v, bits_a, signed_a) : oracle_wrap(v, bits_a, signed_a);
        break;
      case OR_RELU:
        out[i] = (signed_a && x[i] < 0) ? 0 : x[i];
        break;
      case OR_REQUANT:
        if (shift < 0 || shift > 31 || bits_o < 1 || bits_o > 8) return OR_EINVAL;
        out[i] = oracle_clamp(floor_shift(x[i], shift), bits_o, signed_o);
        break;
      default:
        return OR_EINVAL;
    }
  }
  return OR_OK;
}

/* ---- convolution -------------------------------------------------------- */

/* DNN convolution, the direct-sum2d loop nest of Fig. 12 (section 7),
 * generalised to a batch dimension, a stride, zero padding and M output
 * channels. Layout is the paper's CHW per image:
 *   act[n][c][h][w], wt[m][c][y][x], out[n][m][ho][wo],
 *   out[n][m][ho][wo] = sum_{c,y,x} act[n][c][ho*stride-pad+y][wo*stride-pad+x] * wt[m][c][y][x]
 * (cross-correlation, no kernel flip; taps outside the image read zero).
 * Outputs start at zero. Sums are exact int64; the function returns
 * OR_ERANGE if any |sum| reaches 2^31 (the int32 accumulator bound).
 * `nthreads` > 1 splits the outermost (n, m) loop over OpenMP threads. */
int oracle_conv2d(int N, int C, int H, int W, int M, int R, int S, int stride, int pad, const int64_t *act,
                  const int64_t *wt, int64_t *out, int nthreads) {
  if (N < 0 || C < 1 || H < 1 || W < 1 || M < 1 || R < 1 || S < 1 || stride < 1 || pad < 0) return OR_EINVAL;
  int Ho = (H + 2 * pad - R) / stride + 1;
  int Wo = (W + 2 * pad - S) / stride + 1;
  if (H + 2 * pad < R || W + 2 * pad < S) return OR_EINVAL;
  int overflow = 0;
  int64_t limit = (int64_t)1 << 31;
  int64_t nm_total = (int64_t)N * M;
  (void)nthreads;
#ifdef _OPENMP
  if (nthreads < 1) nthreads = 1;
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 1) reduction(| : overflow)
#endif
  for (int64_t nm = 0; nm < nm_total; nm++) {
    int64_t n = nm / M, m = nm % M;
    for (int h = 0; h < Ho; h++)
      for (int w = 0; w < Wo; w++) {
        int64_t result = 0;
        for (int d = 0; d < C; d++)
          for (int y = 0; y < R; y++)
            for (int x = 0; x < S; x++) {
              int ih = h * stride - pad + y;
              int iw = w * stride - pad + x;
              if (ih < 0 || ih >= H || iw < 0 || iw >= W) continue;
              result += act[((n * C + d) * H + ih) * W + iw] * wt[((m * C + d) * R + y) * S + x];
            }
        if (result >= limit || result < -limit) overflow = 1;
        out[((n * M + m) * Ho + h) * Wo + w] = result;
      }
  }
  return overflow ? OR_ERANGE : OR_OK;
}

/* Lane-wise 2x2 max-pool with stride 2 on CHW images:
 * out[n][c][i][j] = max over act[n][c][2i+u][2j+v], u, v in {0, 1}.
 * H and W must be even. */
int oracle_maxpool2x2(int N, int C, int H, int W, const int64_t *in, int64_t *out) {
  if (N < 0 || C < 1 || H < 2 || W < 2 || (H & 1) || (W & 1)) return OR_EINVAL;
  int Ho = H / 2, Wo = W / 2;
  for (int64_t n = 0; n < N; n++)
    for (int c = 0; c < C; c++)
      for (int i = 0; i < Ho; i++)
        for (int j = 0; j < Wo; j++) {
          int64_t best = in[((n * C + c) * H + 2 * i) * W + 2 * j];
          for (int u = 0; u < 2; u++)
            for (int v = 0; v < 2; v++) {
              int64_t t = in[((n * C + c) * H + 2 * i + u) * W + 2 * j + v];
              if (t > best) best = t;
            }
          out[((n * C + c) * Ho + i) * Wo + j] = best;
        }
  return OR_OK;
}

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}
