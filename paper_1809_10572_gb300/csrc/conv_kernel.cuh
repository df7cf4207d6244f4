// conv_kernel.cuh -- the persistent tcgen05 convolution kernel (device code
// shared by the translation units that instantiate it).
//
// The paper's DNN convolution (section 7, Fig. 12, direct-sum2d) is
//   acc[n][k][ho][wo] = sum_{c,r,s} act[n][c][ho*st-p+r][wo*st-p+s] * wt[k][c][r][s].
// Here it is the GEMM D[M x K] = A[M x Kg] * B[K x Kg]^T with M = N*Ho*Wo
// output pixels and a reduction index Kg running over (tap, packed word,
// lane). Activations and weights stay packed in HBM and L2 and are widened
// only in shared memory, right before the MMA (the "unpack to the native
// type" baseline of section 7, moved on-chip).
//
// Exactness. sm_103a has no integer MMA, so lanes are widened to a float
// type whose every value in play is an exact integer, and the fp32
// accumulators hold exact integers while every partial sum stays below 2^24:
//   e4m3 (kind::f8f6f4, K = 32 per MMA) when |a| <= 16 and |w| <= 16 (lane
//        widths up to 4 bits, and signed 5-bit lanes); half the shared-memory
//        bytes of fp16 per product, twice the tensor rate;
//   fp16 (kind::f16, K = 16 per MMA) otherwise: every integer of [-128, 255].
// When R*S*C*max|a|*max|w| reaches 2^24 (wide weights over many taps), the
// fp16 weights are split into two 4-bit digits w = 16*hi + lo stacked along
// the MMA's N; the epilogue forms 16*hi + lo in int32.
//
// Both operand types use rows of 64 reduction positions: 128-byte rows with
// the 128-byte swizzle (fp16) or 64-byte rows with the 64-byte swizzle
// (e4m3). An MMA consumes 32 bytes of a row either way, so the descriptors
// advance by the same 32 bytes per MMA.
#pragma once

#include <cuda.h>
#include <cuda_fp16.h>

#include <cstring>
#include <type_traits>
#include <utility>

#include "samd_internal.cuh"
#include "tc_ptx.cuh"

namespace samd {
namespace conv {

constexpr int BM = 128;  // output pixels per tile = MMA M = TMEM lanes
constexpr int BK = 64;   // reduction positions per chunk = one operand row
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s
constexpr int kGatherDepth = 4;                    // packed chunks in flight per producer thread
constexpr int kProdWarps = 8;                      // operand producers
constexpr int kEpiWarps = 8;                       // epilogue
constexpr int kProdThreads = 32 * kProdWarps;
constexpr int kThreads = 32 * (2 + kProdWarps + kEpiWarps);
constexpr int kFirstEpiWarp = 2 + kProdWarps;
// Optional epilogue staging (ConvArgs::e_stage): per epilogue warp 32 rows of
// one packing period (at most 32 words), rows kEpiPitch words apart (odd, so
// that 32 lanes writing one word of their own rows hit 32 banks).
constexpr int kEpiPitch = 33;
constexpr uint32_t kEpiStageBytes = kEpiWarps * 32 * kEpiPitch * 4;

template <bool FP8>
struct OpTraits {
  static constexpr int kRowBytes = FP8 ? 64 : 128;  // one row of BK positions
  static constexpr int kKPerMma = FP8 ? 32 : 16;
  static constexpr uint32_t kTileBytes = BM * kRowBytes;
  // 16-byte chunk c of row r (rows kRowBytes apart from a 1024-byte-aligned base)
  __device__ static __forceinline__ int swz(int r, int c) { return FP8 ? (c ^ ((r >> 1) & 3)) : (c ^ (r & 7)); }
  __device__ static __forceinline__ uint64_t desc(uint32_t saddr) {
    return FP8 ? ptx::sw64_kmajor_desc(saddr) : ptx::sw128_kmajor_desc(saddr);
  }
};

__host__ __device__ constexpr bool pair16(int bits) { return bits == 1 || bits == 2 || bits == 4 || bits == 8; }

// The lane of a packed word held by reduction position `pos` (0 <= pos < L)
// of that word. For lane widths dividing 16, positions 2p and 2p+1 hold
// lanes p and p + 16/bits of the same 32-bit half, which sit exactly 16 bits
// apart, so one masked shift widens both at once. Other widths keep lane
// order. A and B use the same map, so the dot products are unchanged.
__host__ __device__ constexpr int kpos_lane(int bits, int pos) {
  if (pair16(bits)) {
    int g = 32 / bits, half = pos / g, jj = pos % g;
    return half * g + jj / 2 + (jj & 1) * (g / 2);
  }
  return pos;
}

// e4m3 widening by byte permutes (1- and 2-bit lanes, unsigned 4-bit lanes):
// each lane of a 32-bit half-word becomes a selector nibble of prmt over a
// table of e4m3 codes. The reduction positions of such a half-word are
// ordered by how the nibbles are formed (identity for 4 bits; even then odd
// lanes for 2 bits; lanes k, k+4, ... for 1 bit); A and B use the same order.
__host__ __device__ constexpr bool prmt8(int bits, bool is_signed) {
  return bits == 1 || bits == 2 || (bits == 4 && !is_signed);
}
__host__ __device__ constexpr int kpos_lane_prmt32(int bits, int p) {
  return bits == 4 ? p : (bits == 2 ? 2 * (p % 4 + 4 * ((p / 4) % 2)) + p / 8 : 4 * (p % 8) + p / 8);
}
// The lane of an activation word held by reduction position `pos` for the
// operand type in use.
__host__ __device__ constexpr int kpos_lane_op(int bits, bool is_signed, bool fp8, int pos) {
  return (fp8 && prmt8(bits, is_signed)) ? (pos / (32 / bits)) * (32 / bits) + kpos_lane_prmt32(bits, pos % (32 / bits))
                                         : kpos_lane(bits, pos);
}

// e4m3 code of a small integer (|v| <= 16): sign, exponent biased by 7, three
// mantissa bits.
__host__ __device__ constexpr uint32_t e4m3_code(int v) {
  if (v == 0) return 0u;
  const uint32_t sign = v < 0 ? 0x80u : 0u;
  const int a = v < 0 ? -v : v;
  int e = 0;
  while ((a >> (e + 1)) != 0) ++e;
  return sign | static_cast<uint32_t>((e + 7) << 3) | static_cast<uint32_t>(((a << 3) >> e) - 8);
}
__host__ __device__ constexpr uint32_t e4m3_table4(int v0, int v1, int v2, int v3) {
  return e4m3_code(v0) | (e4m3_code(v1) << 8) | (e4m3_code(v2) << 16) | (e4m3_code(v3) << 24);
}

// prmt.b32 in its default mode: byte i of the result is byte (c_i & 7) of
// {b, a}, or, when bit 3 of selector nibble c_i is set, that byte's sign bit
// repeated eight times.
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}

// n / d for 0 <= n < 2^31 by one multiply-high, an add and a shift:
// l = ceil(log2 d), m = floor(2^32 (2^l - d) / d) + 1, q = (umulhi(m, n) + n) >> l.
struct FastDiv {
  uint32_t m;
  int l;
  uint32_t d;
};

inline FastDiv make_fastdiv(uint32_t d) {
  int l = 0;
  while ((uint64_t(1) << l) < d) ++l;
  const uint64_t m = ((uint64_t(1) << 32) * ((uint64_t(1) << l) - d)) / d + 1;
  return FastDiv{static_cast<uint32_t>(m), l, d};
}

__device__ __forceinline__ uint32_t fdiv(uint32_t n, const FastDiv &f) { return (__umulhi(f.m, n) + n) >> f.l; }

struct ConvArgs {
  const void *act;
  int32_t *acc_out;
  void *packed_out;
  int *status;  // sticky SAMD_ETIMEOUT record of this device
  int N, C, H, W, K, R, S, stride, pad, Ho, Wo;
  long long M;
  int wpr;          // activation words per pixel
  int words_total;  // R * S * wpr: reduction length in packed words (GATHER)
  int nchunks;      // weight tiles per output tile
  int NBc;          // output channels per channel block
  int n_mma;        // NBc rounded up to 16
  int mma_n;        // MMA N: n_mma, or 2 * n_mma with split weight digits
  int split;        // 1: accumulator columns [0, n_mma) hold hi digits, [n_mma, 2 n_mma) lo digits
  int stages;       // weight tiles in flight (or resident)
  int stages_a;     // GATHER: A tiles in flight
  int b_resident;   // 1: all weight tiles of the layer stay in shared memory
  long long grid_m; // 128-position tiles along the output
  int nblocks;      // channel blocks
  int gather_vec;   // AGather::vec
  int gather_win;   // AGather::issue_win (chunks that are not aligned 16-byte vectors); chunk = (channel chunk, tap)
  int g_row;        // GATHER staging row pitch in bytes
  int gdepth;       // HALO: packed staging slots; gathers run gdepth - 1 items ahead
  int hbufs;        // HALO: widened halo buffers (2 or 3); item k goes to buffer k mod hbufs
  long long act_bytes;  // bytes of the activation tensor (the windows stop at its end)
  uint32_t tmem_cols;
  int out_bits, out_signed, out_lane_w, out_L, out_word64, out_wpr;
  int out_fast;     // output lanes per word when they divide 32 (whole words per 32 channels), else 0
  int shift;
  float out_scale;  // 2^-shift
  int fast_req;     // |acc| / 2^shift < 2^22: requantize through floor_scaled_biased
  int fast_acc;     // |acc| < 2^22: int32 outputs through floor_scaled_biased
  // HALO (stride 1): virtual output grid of N x Hv x Wp positions. A tile of
  // 128 consecutive positions v0.. reads nseg segments of the input grid:
  // segment g holds seg_used rows starting at virtual row v0 + g * Wp and
  // occupies seg_rows rows of the halo buffer; tap (r, s) reads the 128 rows
  // starting at halo row r * row_step + s.
  int Hv, Wp;
  int nseg, seg_rows, seg_used, row_step;
  int nck;   // channel chunks per pixel (ceil(wpr / WC))
  int full;  // AUnpack FULL: one chunk holds all the pixel's words
  int hv;    // tile of hv parts of 128 output positions (1, 2, or 4 for e4m3 halo layers)
  int taps;  // R * S
  FastDiv fd_plane, fd_wp;  // / (Hv * Wp), / Wp
  FastDiv fd_seg;           // / seg_rows
  FastDiv fd_wo, fd_ho;     // output pixel index -> (n, oh, ow)
  FastDiv fd_gm;            // tile -> (channel block, position tile)
  // shared memory carve-up (bytes from the 1024-byte-aligned base)
  uint32_t op_stride;  // one halo buffer or one A tile
  uint32_t off_b, b_bytes, off_g, g_stride, off_e, off_bar;
  int e_stage;  // 1: kEpiStageBytes at off_e stage the 3/5/6-bit packed rows (epilogue_row_period_staged)
  // Fused 2x2 max-pool (pool = 1; halo layers): tile mt is pool_rows output
  // rows (pool_rows / 2 row pairs) of one image from an even row on, at
  // virtual position img * Hv * Wp + g * pool_rows * Wp (img = mt / tiles
  // per image, g its remainder). The epilogue warps that drain a tile pack
  // its rows into the pool_pitch-word rows of their buffer at off_e (pool_nw
  // words of the channel block per row) and write only the lane-wise maxima
  // of the 2x2 windows, rows of (N, Ho / 2, Wo / 2) pixels, to packed_out.
  int pool, pool_rows, pool_nw, pool_pitch;
  FastDiv fd_tpi;  // tiles per image
};

// First position, in the padded virtual grid N x Hv x Wp, of tile mt of a
// halo layer (tiles of bmt consecutive positions, or pooled tiles of whole
// row pairs).
__device__ __forceinline__ uint32_t tile_first_pos(const ConvArgs &args, uint32_t mt, int bmt) {
  if (!args.pool) return mt * static_cast<uint32_t>(bmt);
  const uint32_t img = fdiv(mt, args.fd_tpi);
  const uint32_t g = mt - img * args.fd_tpi.d;
  return img * args.fd_plane.d + g * static_cast<uint32_t>(args.pool_rows * args.Wp);
}

__device__ __forceinline__ uint32_t hsub2_bits(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// two fp16 integers (|v| <= 16, exact in e4m3) -> two e4m3 bytes, low half first
__device__ __forceinline__ uint32_t f16x2_to_e4m3x2(uint32_t h) {
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f16x2 %0, %1;" : "=h"(r) : "r"(h));
  return r;
}

// Widening of one 64-position row of the A operand (one pixel, one chunk).
// A chunk is WC whole words. FULL (lanes per word not dividing 64, at most
// 64 channels in ceil(64 / L) words): one chunk holds all the pixel's words
// and its 64 positions are channels 0..63 -- the last word's lanes past 64
// are padding; otherwise WC = floor(64 / L) and positions past WC * L are
// zero.
template <typename W, int BITS, bool SIGNED, bool FP8, bool FULL = false>
struct AUnpack {
  static constexpr int WB = WordTraits<W>::kBits;
  static constexpr int L = WB / BITS;
  static constexpr int WC = FULL ? (BK + L - 1) / L : BK / L;  // packed words per chunk
  static constexpr int KUSED = FULL ? BK : WC * L;             // positions holding lanes; the rest are zero
  static constexpr uint32_t LM = (1u << BITS) - 1;
  static constexpr uint32_t OFF = SIGNED ? (1u << (BITS - 1)) : 0u;  // offset-binary zero
  static constexpr uint32_t BIAS = 0x6400u + OFF;                   // fp16 bits of 1024 + OFF
  static constexpr uint32_t BIAS2 = BIAS | (BIAS << 16);

  static constexpr W sign_mask() {
    W m = 0;
    for (int i = 0; i < L; ++i) m |= W(1) << (i * BITS + BITS - 1);
    return m;
  }

  template <int POS>
  __device__ static __forceinline__ uint32_t field(W w) {
    return static_cast<uint32_t>(w >> (kpos_lane(BITS, POS) * BITS)) & LM;
  }

  // A lane pattern v (offset binary when signed) becomes fp16 1024 + v by
  // or-ing it into the mantissa of 1024.0; subtracting 1024 + OFF leaves the
  // lane's value exactly. A zero word (padding) therefore widens to zeros.
  template <int P>
  __device__ static __forceinline__ uint32_t pair(const W (&w)[WC]) {
    constexpr int j0 = 2 * P, j1 = 2 * P + 1;
    if constexpr (j0 >= KUSED) {
      return 0u;
    } else if constexpr (pair16(BITS)) {
      constexpr int q = j0 / L, pos = j0 % L, g = 32 / BITS, half = pos / g;
      constexpr int lane0 = kpos_lane(BITS, pos) - half * g;
      const uint32_t x = static_cast<uint32_t>(w[q] >> (half * 32));
      const uint32_t t = ((x >> (lane0 * BITS)) & (LM | (LM << 16))) | 0x64006400u;
      return hsub2_bits(t, BIAS2);
    } else {
      const uint32_t v0 = field<j0 % L>(w[j0 / L]);
      uint32_t v1 = OFF;
      if constexpr (j1 < KUSED) v1 = field<j1 % L>(w[j1 / L]);
      return hsub2_bits(v0 | (v1 << 16) | 0x64006400u, BIAS2);
    }
  }

  template <int... P>
  __device__ static __forceinline__ void pairs(const W (&w)[WC], uint32_t (&h)[32],
                                               std::integer_sequence<int, P...>) {
    ((h[P] = pair<P>(w)), ...);
  }

  static constexpr bool kPrmt = FP8 && prmt8(BITS, SIGNED);

  // The e4m3 bytes of the lanes of one 32-bit half-word, in reduction order
  // (32 / BITS bytes into out[0 .. 8 / BITS)).
  __device__ static __forceinline__ void prmt_half(uint32_t x, uint32_t *out) {
    if constexpr (BITS == 4) {
      // nibbles 0-7 select e(0..7); nibbles 8-15 select the sign (0) of that
      // table and, with bit 3 flipped, e(8..15) from the other one
      constexpr uint32_t t0 = e4m3_table4(0, 1, 2, 3), t1 = e4m3_table4(4, 5, 6, 7);
      constexpr uint32_t t2 = e4m3_table4(8, 9, 10, 11), t3 = e4m3_table4(12, 13, 14, 15);
      const uint32_t xx = x ^ 0x88888888u;
      out[0] = prmt(t0, t1, x) | prmt(t2, t3, xx);
      out[1] = prmt(t0, t1, x >> 16) | prmt(t2, t3, xx >> 16);
    } else if constexpr (BITS == 2) {
      constexpr uint32_t t = SIGNED ? e4m3_table4(0, 1, -2, -1) : e4m3_table4(0, 1, 2, 3);
      const uint32_t se = x & 0x33333333u, so = (x >> 2) & 0x33333333u;
      out[0] = prmt(t, 0u, se);
      out[1] = prmt(t, 0u, se >> 16);
      out[2] = prmt(t, 0u, so);
      out[3] = prmt(t, 0u, so >> 16);
    } else {
      constexpr uint32_t t = SIGNED ? e4m3_table4(0, -1, 0, 0) : e4m3_table4(0, 1, 0, 0);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint32_t sk = (x >> k) & 0x11111111u;
        out[2 * k] = prmt(t, 0u, sk);
        out[2 * k + 1] = prmt(t, 0u, sk >> 16);
      }
    }
  }

  // Widen one pixel's chunk and store it as row `row` of a swizzled K-major
  // operand whose rows are OpTraits::kRowBytes apart.
  __device__ static __forceinline__ void unpack_row(W (&w)[WC], uint8_t *tile, int row) {
    using T = OpTraits<FP8>;
    if constexpr (kPrmt) {
      constexpr int kHalves = WB / 32, kPer = 8 / BITS;  // 32-bit words of e4m3 bytes per half-word
      uint32_t b[16];
#pragma unroll
      for (int q = 0; q < WC; ++q)
#pragma unroll
        for (int hh = 0; hh < kHalves; ++hh)
          prmt_half(static_cast<uint32_t>(w[q] >> (32 * hh)), b + (q * kHalves + hh) * kPer);
      uint8_t *rp = tile + row * T::kRowBytes;
#pragma unroll
      for (int c = 0; c < 4; ++c)
        *reinterpret_cast<uint4 *>(rp + (T::swz(row, c) << 4)) = make_uint4(b[4 * c], b[4 * c + 1], b[4 * c + 2], b[4 * c + 3]);
      return;
    }
    if constexpr (SIGNED) {
#pragma unroll
      for (int q = 0; q < WC; ++q) w[q] ^= sign_mask();
    }
    uint32_t h[32];
    pairs(w, h, std::make_integer_sequence<int, 32>{});
    uint8_t *rp = tile + row * T::kRowBytes;
    if constexpr (FP8) {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t b[4];
#pragma unroll
        for (int k = 0; k < 4; ++k)
          b[k] = f16x2_to_e4m3x2(h[8 * c + 2 * k]) | (f16x2_to_e4m3x2(h[8 * c + 2 * k + 1]) << 16);
        *reinterpret_cast<uint4 *>(rp + (T::swz(row, c) << 4)) = make_uint4(b[0], b[1], b[2], b[3]);
      }
    } else {
#pragma unroll
      for (int c = 0; c < 8; ++c)
        *reinterpret_cast<uint4 *>(rp + (T::swz(row, c) << 4)) =
            make_uint4(h[4 * c], h[4 * c + 1], h[4 * c + 2], h[4 * c + 3]);
    }
  }
};

// Bytes of one pixel-chunk row in the packed staging buffers (a multiple of 16).
template <typename W, int WC>
struct Staging {
  static constexpr int kBytes = WC * static_cast<int>(sizeof(W));
  static constexpr int kRowBytes = (kBytes + 15) / 16 * 16;
  // widest cp.async that divides a whole chunk held by one pixel
  static constexpr int kVec = kBytes % 16 == 0 ? 16 : (kBytes % 8 == 0 ? 8 : static_cast<int>(sizeof(W)));
};

// Copies a pixel-chunk of kBytes from `src` (vector-aligned) to staging with
// cp.async; nbytes = 0 zero-fills it.
template <typename W, int WC>
__device__ __forceinline__ void stage_chunk(uint32_t dst, const char *src, uint32_t valid) {
  using St = Staging<W, WC>;
#pragma unroll
  for (int v = 0; v < St::kBytes / St::kVec; ++v) {
    if constexpr (St::kVec == 16)
      ptx::cp_async_16(dst + 16 * v, src + 16 * v, valid ? 16u : 0u);
    else if constexpr (St::kVec == 8)
      ptx::cp_async_8(dst + 8 * v, src + 8 * v, valid ? 8u : 0u);
    else
      ptx::cp_async_4(dst + 4 * v, src + 4 * v, valid ? 4u : 0u);
  }
}

// Reads a staged pixel-chunk back into words.
template <typename W, int WC>
__device__ __forceinline__ void load_staged(const uint8_t *src, W (&cur)[WC]) {
  using St = Staging<W, WC>;
#pragma unroll
  for (int v = 0; v < St::kRowBytes / 16; ++v) {
    const uint4 q4 = *reinterpret_cast<const uint4 *>(src + 16 * v);
    const uint32_t tw[4] = {q4.x, q4.y, q4.z, q4.w};
#pragma unroll
    for (int kq = 0; kq < 4; ++kq) {
      const int byte = 16 * v + 4 * kq;
      if (byte < St::kBytes) {
        if constexpr (sizeof(W) == 4) {
          cur[byte / 4] = tw[kq];
        } else if ((kq & 1) == 0) {
          cur[byte / 8] = static_cast<W>(tw[kq]) | (static_cast<W>(tw[kq + 1]) << 32);
        }
      }
    }
  }
}

// 16-byte pieces that cover one chunk from the 16-byte boundary at or below
// its first byte (the chunk then starts o bytes into the staged row, o < 16).
template <typename W, int WC>
constexpr int kWinPieces = (WC * static_cast<int>(sizeof(W)) + 15) / 16 + 1;

// Reads a chunk staged through its 16-byte window (AGather::issue_win): the
// chunk starts o4 32-bit units into the row; words from nw on are zero.
template <typename W, int WC>
__device__ __forceinline__ void load_window(const uint8_t *row, int o4, int nw, W (&cur)[WC]) {
  constexpr int kU = WC * static_cast<int>(sizeof(W)) / 4;  // 32-bit units of a chunk
  constexpr int kV = (kU + 3 + 3) / 4;                       // 16-byte reads covering kU + 3 units
  static_assert(kV <= kWinPieces<W, WC>, "the window holds every unit read");
  uint32_t u[4 * kV];
#pragma unroll
  for (int v = 0; v < kV; ++v) {
    const uint4 q = *reinterpret_cast<const uint4 *>(row + 16 * v);
    u[4 * v] = q.x, u[4 * v + 1] = q.y, u[4 * v + 2] = q.z, u[4 * v + 3] = q.w;
  }
  // shift down by o4 units: by one unit, then by two
  uint32_t s1[kU + 2];
#pragma unroll
  for (int i = 0; i < kU + 2; ++i) s1[i] = (o4 & 1) ? u[i + 1] : u[i];
  const int nu = nw * static_cast<int>(sizeof(W)) / 4;
#pragma unroll
  for (int i = 0; i < kU; ++i) {
    uint32_t x = (o4 & 2) ? s1[i + 2] : s1[i];
    if (i >= nu) x = 0u;
    if constexpr (sizeof(W) == 4)
      cur[i] = x;
    else if (i & 1)
      cur[i / 2] |= static_cast<W>(x) << 32;
    else
      cur[i / 2] = x;
  }
}

// Gathers the packed words of one pixel's chunk into shared memory with
// cp.async: word kw of the reduction is word (kw mod wpr) of the input pixel
// at tap kw / wpr; taps outside the image and words past the end are
// zero-filled (source size 0).
template <typename W, int WC>
struct AGather {
  const W *act;
  int H, W_, wpr, S, stride, pad, words_total, taps;
  int n, oh, ow;
  bool row_valid;
  bool vec;  // every chunk lies inside one pixel at a kVec-aligned offset

  __device__ __forceinline__ const W *pixel(int tap, bool &valid) const {
    int r = tap / S, s = tap - (tap / S) * S;
    int ih = oh * stride - pad + r, iw = ow * stride - pad + s;
    valid = row_valid && ih >= 0 && ih < H && iw >= 0 && iw < W_;
    return act + ((static_cast<long long>(n) * H + ih) * W_ + iw) * wpr;
  }

  __device__ __forceinline__ void issue(int chunk, uint32_t dst) const {
    const int kw0 = chunk * WC;
    int tap = kw0 / wpr, wi = kw0 - tap * wpr;
    bool valid;
    const W *px = pixel(tap, valid);
    if (vec) {
      stage_chunk<W, WC>(dst, reinterpret_cast<const char *>(valid ? px + wi : act), valid ? 1u : 0u);
      return;
    }
#pragma unroll
    for (int q = 0; q < WC; ++q) {
      const bool in = valid && kw0 + q < words_total;
      const W *src = in ? px + wi : act;
      if constexpr (sizeof(W) == 8)
        ptx::cp_async_8(dst + 8 * q, src, in ? 8u : 0u);
      else
        ptx::cp_async_4(dst + 4 * q, src, in ? 4u : 0u);
      if (++wi == wpr) {
        wi = 0;
        ++tap;
        px = pixel(tap, valid);
      }
    }
  }

  // Chunks that are not whole 16-byte vectors (issue_win): chunk c is
  // channel chunk j = c / taps of the pixel at tap c % taps, the words
  // [j WC, min((j + 1) WC, wpr)) of that pixel, copied as the 16-byte pieces
  // of the aligned window around them, so that every copy is 16 bytes wide
  // whatever the pixel's alignment. Pieces past the chunk are zero-filled;
  // a piece that reaches past the end of the activation tensor (act_end)
  // copies only the bytes before it. Returns the chunk's offset into the
  // staged row in 32-bit units (load_window). act is 16-byte aligned.
  __device__ __forceinline__ int issue_win(int chunk, uint32_t dst, uintptr_t act_end) const {
    const int j = chunk / taps;
    const int wi = j * WC;
    const int nw = wpr - wi < WC ? wpr - wi : WC;
    bool valid;
    const W *px = pixel(chunk - j * taps, valid);
    const uintptr_t a = valid ? reinterpret_cast<uintptr_t>(px + wi) : reinterpret_cast<uintptr_t>(act);
    const uintptr_t a0 = a & ~static_cast<uintptr_t>(15);
    const uintptr_t end = a + static_cast<uintptr_t>(nw) * sizeof(W);
#pragma unroll
    for (int v = 0; v < kWinPieces<W, WC>; ++v) {
      const uintptr_t pa = a0 + 16u * v;
      uint32_t n = 0;
      if (valid && pa < end) n = act_end - pa < 16 ? static_cast<uint32_t>(act_end - pa) : 16u;
      ptx::cp_async_16(dst + 16 * v, n ? reinterpret_cast<const void *>(pa) : static_cast<const void *>(act), n);
    }
    return static_cast<int>((a - a0) >> 2);
  }
};

// Packs 32 requantized lane patterns (zero past `cnt`) into 32 / LO words of
// LO lanes each and stores them; LO divides 32, so every word of the
// 32-channel group is whole.
template <int LO, typename WO>
__device__ __forceinline__ void pack_regs(const uint32_t (&y)[32], int lane_w, int cnt, WO *dst) {
  constexpr int NW = 32 / LO;  // words of this 32-channel group
  WO w[NW];
#pragma unroll
  for (int k = 0; k < NW; ++k) {
    w[k] = 0;
#pragma unroll
    for (int l = 0; l < LO; ++l) w[k] |= static_cast<WO>(y[k * LO + l]) << (l * lane_w);
  }
  constexpr int kWordBytes = static_cast<int>(sizeof(WO));
  if (cnt == 32 && (NW * kWordBytes) % 16 == 0 && (reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
    for (int v = 0; v < NW * kWordBytes / 16; ++v) {
      uint4 q;
      memcpy(&q, reinterpret_cast<const uint8_t *>(w) + 16 * v, 16);
      reinterpret_cast<uint4 *>(dst)[v] = q;
    }
  } else {
#pragma unroll
    for (int k = 0; k < NW; ++k)
      if (k * LO < cnt) dst[k] = w[k];
  }
}

constexpr int32_t kMagicBits = 0x4B400000;  // encoding of 1.5 * 2^23

// floor(acc * scale) + 1.5 * 2^23 as the encoding of a float: with rounding
// toward minus infinity the fma result, which lies in [2^23, 2^24) where the
// unit in the last place is 1, is exactly floor(acc * scale) + 1.5 * 2^23
// while |acc * scale| < 2^22 (scale = 2^-shift makes acc * scale exact).
// The encoding is then kMagicBits + floor(acc * scale), monotonic in it.
__device__ __forceinline__ int32_t floor_scaled_biased(float acc, float scale) {
  float r;
  asm("fma.rm.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(acc), "f"(scale), "f"(12582912.0f));
  return __float_as_int(r);
}

// Packs lane patterns into words of L lanes one channel at a time (any L):
// the running word `cur` receives lane nl at bit sh and is stored when full.
template <typename WO>
struct RowPacker {
  WO *dst;
  WO cur = 0;
  int nl = 0, sh = 0;
  __device__ __forceinline__ void put(uint32_t y, int L, int lw) {
    cur |= static_cast<WO>(y) << sh;
    sh += lw;
    if (++nl == L) {
      *dst++ = cur;
      cur = 0;
      sh = 0;
      nl = 0;
    }
  }
  __device__ __forceinline__ void flush() {
    if (nl) *dst = cur;
  }
};

// Epilogue of one accumulator row (one output pixel m) of channel block nb:
// fp32 accumulators -> exact integers -> optional int32 store, optional
// requantize-and-pack. Called by whole warps (tcgen05.ld is collective; rows
// outside the output only skip the stores).
//
// The common case (packed output only, no split digits, |acc| / 2^shift <
// 2^22) requantizes each accumulator with one fma in place.
template <typename WO>
__device__ __forceinline__ void epilogue_row_fast(const ConvArgs &args, uint32_t taddr, bool row_valid, long long m,
                                                  int nb) {
  const int ch0 = nb * args.NBc;
  const int nvalid = args.K - ch0 < args.NBc ? args.K - ch0 : args.NBc;
  const int lo = lane_lo(args.out_bits, args.out_signed), hi = lane_hi(args.out_bits, args.out_signed);
  const int32_t blo = kMagicBits + lo, bhi = kMagicBits + hi;
  const uint32_t omask = (1u << args.out_bits) - 1;
  const float scale = args.out_scale;
  const int L = args.out_L, lw = args.out_lane_w;
  RowPacker<WO> pk;
  pk.dst = static_cast<WO *>(args.packed_out) + (m * args.out_wpr + ch0 / L);
  for (int col = 0; col < nvalid; col += 32) {
    uint32_t y[32];
    ptx::tmem_ld_32x32b_x32(taddr + col, y);
    ptx::tmem_wait_ld();
    const int cnt = nvalid - col < 32 ? nvalid - col : 32;
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      int32_t t = floor_scaled_biased(__uint_as_float(y[k]), scale);
      t = t < blo ? blo : (t > bhi ? bhi : t);
      y[k] = k < cnt ? static_cast<uint32_t>(t) & omask : 0u;
    }
    if (!row_valid) continue;
    if (args.out_fast) {  // L divides 32: whole words per 32-channel group
      WO *dst = static_cast<WO *>(args.packed_out) + (m * args.out_wpr + (ch0 + col) / L);
      switch (args.out_fast) {
        case 4:
          if constexpr (sizeof(WO) == 4) pack_regs<4>(y, lw, cnt, dst);
          break;
        case 8: pack_regs<8>(y, lw, cnt, dst); break;
        case 16: pack_regs<16>(y, lw, cnt, dst); break;
        default: pack_regs<32>(y, lw, cnt, dst); break;
      }
    } else {
#pragma unroll
      for (int k = 0; k < 32; ++k)
        if (k < cnt) pk.put(y[k], L, lw);
    }
  }
  if (!args.out_fast && row_valid) pk.flush();
}

// The fast epilogue for output lanes of OB = 1, 2, 4, 7 or 8 bits without
// spacers (7 only in 32-bit words): the words of a 32-channel group are built
// 32 bits at a time (for OB dividing 32 a 64-bit word is its two 32-bit
// halves, low half first, so the bytes are the same) with compile-time
// shifts. Unsigned lanes are summed in the
// biased domain and the bias sum is removed once per word; signed lanes are
// masked to their two's complement bits first.
template <int OB, bool OS>
__device__ __forceinline__ void epilogue_row_spec(const ConvArgs &args, uint32_t taddr, bool row_valid, long long m,
                                                  int nb) {
  constexpr int LH = 32 / OB;  // lanes per 32-bit half-word (a divisor of 32: OB = 1, 2, 4, 7, 8)
  constexpr int NH = 32 / LH;  // half-words per 32-channel group
  static_assert(32 % LH == 0, "whole half-words per 32-channel group");
  constexpr int32_t lo = OS ? -(1 << (OB - 1)) : 0, hi = OS ? (1 << (OB - 1)) - 1 : (1 << OB) - 1;
  constexpr int32_t blo = kMagicBits + lo, bhi = kMagicBits + hi;
  constexpr uint32_t omask = (1u << OB) - 1;
  constexpr uint32_t bias_sum = [] {
    uint32_t b = 0;
    for (int l = 0; l < LH; ++l) b += static_cast<uint32_t>(kMagicBits) << (l * OB);
    return b;
  }();
  const int ch0 = nb * args.NBc;
  const int nvalid = args.K - ch0 < args.NBc ? args.K - ch0 : args.NBc;
  const float scale = args.out_scale;
  // 32-bit half-words of this row: output channel c sits in half-word c / LH
  uint32_t *row32 = reinterpret_cast<uint32_t *>(static_cast<uint8_t *>(args.packed_out) +
                                                 static_cast<size_t>(m) * args.out_wpr * (args.out_word64 ? 8 : 4)) +
                    ch0 / LH;
  // 4-bit lanes: two 32-channel groups make one 32-byte store (a warp's
  // 32-byte rows then cover whole 128-byte lines, in the L1 data path the
  // MMAs' operand reads share)
  const bool pair32 = NH == 4 && nvalid % 64 == 0 && (reinterpret_cast<uintptr_t>(row32) & 31) == 0;
  uint32_t p0 = 0, p1 = 0, p2 = 0, p3 = 0;
  for (int col = 0; col < nvalid; col += 32) {
    uint32_t r[32];
    ptx::tmem_ld_32x32b_x32(taddr + col, r);
    ptx::tmem_wait_ld();
    const int cnt = nvalid - col < 32 ? nvalid - col : 32;
    uint32_t h[NH];
#pragma unroll
    for (int j = 0; j < NH; ++j) {
      uint32_t w = 0;
#pragma unroll
      for (int l = 0; l < LH; ++l) {
        int32_t t = floor_scaled_biased(__uint_as_float(r[j * LH + l]), scale);
        t = t < blo ? blo : (t > bhi ? bhi : t);
        if constexpr (OS)
          w |= (static_cast<uint32_t>(t) & omask) << (l * OB);
        else
          w += static_cast<uint32_t>(t) << (l * OB);
      }
      h[j] = OS ? w : w - bias_sum;
    }
    if constexpr (NH == 4) {
      if (pair32) {
        if ((col & 32) == 0) {
          p0 = h[0], p1 = h[1], p2 = h[2], p3 = h[3];
        } else if (row_valid) {
          ptx::st_global_v8(row32 + (col - 32) / LH, p0, p1, p2, p3, h[0], h[1], h[2], h[3]);
        }
        continue;
      }
    }
    if (!row_valid) continue;
    uint32_t *dst = row32 + col / LH;
    if (cnt < 32) {  // the last group of a channel count that is not a multiple of 32
#pragma unroll
      for (int j = 0; j < NH; ++j) {
        const int c0 = j * LH;  // first channel of half-word j
        if (c0 < cnt) {
          const int nl = cnt - c0 < LH ? cnt - c0 : LH;
          dst[j] = nl == LH ? h[j] : (h[j] & ((1u << (nl * OB)) - 1));
        }
      }
    } else if constexpr (NH == 8) {
      if ((reinterpret_cast<uintptr_t>(dst) & 31) == 0) {
        // one 32-byte store per row: with 32-byte rows a warp writes whole lines
        ptx::st_global_v8(dst, h[0], h[1], h[2], h[3], h[4], h[5], h[6], h[7]);
      } else if ((reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
        reinterpret_cast<uint4 *>(dst)[0] = make_uint4(h[0], h[1], h[2], h[3]);
        reinterpret_cast<uint4 *>(dst)[1] = make_uint4(h[4], h[5], h[6], h[7]);
      } else {
#pragma unroll
        for (int j = 0; j < NH; ++j) dst[j] = h[j];
      }
    } else if constexpr (NH % 4 == 0) {
      if ((reinterpret_cast<uintptr_t>(dst) & 15) == 0) {
#pragma unroll
        for (int v = 0; v < NH / 4; ++v)
          reinterpret_cast<uint4 *>(dst)[v] = make_uint4(h[4 * v], h[4 * v + 1], h[4 * v + 2], h[4 * v + 3]);
      } else {
#pragma unroll
        for (int j = 0; j < NH; ++j) dst[j] = h[j];
      }
    } else if constexpr (NH == 2) {
      if ((reinterpret_cast<uintptr_t>(dst) & 7) == 0)
        *reinterpret_cast<uint2 *>(dst) = make_uint2(h[0], h[1]);
      else
        dst[0] = h[0], dst[1] = h[1];
    } else {
      dst[0] = h[0];
    }
  }
}

__host__ __device__ constexpr int gcd_c(int a, int b) { return b == 0 ? a : gcd_c(b, a % b); }

// The fast epilogue for 32-bit output words whose L = 32 / OB lanes do not
// divide 32 (OB = 3, 5, 6: L = 10, 6, 5). Word boundaries repeat every
// lcm(32, L) channels, so one such period (G groups of 32 columns) is
// unrolled and every lane's word and shift are compile-time. Lanes past the
// last channel read the biased zero, so a final partial word is zero-filled.
template <int OB, bool OS>
__device__ __forceinline__ void epilogue_row_period(const ConvArgs &args, uint32_t taddr, bool row_valid,
                                                    long long m, int nb) {
  constexpr int L = 32 / OB;
  constexpr int G = L / gcd_c(32, L);  // lcm(32, L) / 32
  constexpr int32_t lo = OS ? -(1 << (OB - 1)) : 0, hi = OS ? (1 << (OB - 1)) - 1 : (1 << OB) - 1;
  constexpr int32_t blo = kMagicBits + lo, bhi = kMagicBits + hi;
  constexpr uint32_t omask = (1u << OB) - 1;  // the low bits of kMagicBits + y are those of y
  const int ch0 = nb * args.NBc;
  const int nvalid = args.K - ch0 < args.NBc ? args.K - ch0 : args.NBc;
  const float scale = args.out_scale;
  uint32_t *dst = static_cast<uint32_t *>(args.packed_out) + (m * args.out_wpr + ch0 / L);
  // The last 32-column group may run past the block's channels: its lanes
  // read the biased zero, and words that lie wholly past the last channel
  // belong to the next row, so only the block's words are stored.
  int wleft = (nvalid + L - 1) / L;
  for (int c0 = 0; c0 < nvalid; c0 += 32 * G) {
    uint32_t cur = 0;
    bool open = false;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const int col = c0 + 32 * g;
      if (col >= nvalid) break;
      uint32_t r[32];
      ptx::tmem_ld_32x32b_x32(taddr + col, r);
      ptx::tmem_wait_ld();
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const int q = 32 * g + k;  // channel within the period (compile-time after unrolling)
        const int l = q % L;
        int32_t t = floor_scaled_biased(__uint_as_float(r[k]), scale);
        t = t < blo ? blo : (t > bhi ? bhi : t);
        if (col + k >= nvalid) t = kMagicBits;
        cur |= (static_cast<uint32_t>(t) & omask) << (l * OB);
        open = true;
        if (l == L - 1) {
          if (row_valid && wleft > 0) *dst = cur;
          ++dst;
          --wleft;
          cur = 0;
          open = false;
        }
      }
    }
    if (open && row_valid && wleft > 0) *dst = cur;  // the row's last, partial word
  }
}

// epilogue_row_period with the stores staged: a warp's 32 rows of one
// period (PW = lcm(32, L) / L words per row, 16 or 32) go to the warp's
// shared-memory area first, and the warp then writes them out row by row,
// PW consecutive words of 32 / PW rows per store instruction, instead of
// every thread storing its own row one word at a time (32 rows, 32 sectors,
// per instruction). Every word of a period is computed (channels past the
// block's last read as the biased zero; 32-column groups wholly past it are
// skipped), and only the block's words are stored.
template <int OB, bool OS>
__device__ __forceinline__ void epilogue_row_period_staged(const ConvArgs &args, uint32_t taddr, bool row_valid,
                                                           long long m, int nb, uint32_t *stg) {
  constexpr int L = 32 / OB;
  constexpr int G = L / gcd_c(32, L);  // lcm(32, L) / 32
  constexpr int PW = 32 * G / L;       // words per row and period
  constexpr int RPI = 32 / PW;         // rows per store instruction
  static_assert(PW * RPI == 32, "a period is 16 or 32 words");
  constexpr int32_t lo = OS ? -(1 << (OB - 1)) : 0, hi = OS ? (1 << (OB - 1)) - 1 : (1 << OB) - 1;
  constexpr int32_t blo = kMagicBits + lo, bhi = kMagicBits + hi;
  constexpr uint32_t omask = (1u << OB) - 1;
  const int lane = threadIdx.x & 31;
  const int ch0 = nb * args.NBc;
  const int nvalid = args.K - ch0 < args.NBc ? args.K - ch0 : args.NBc;
  const int nwords = (nvalid + L - 1) / L;  // the block's words in a row
  const float scale = args.out_scale;
  const unsigned vmask = __ballot_sync(0xffffffffu, row_valid);
  uint32_t *const out = static_cast<uint32_t *>(args.packed_out) + ch0 / L;
  uint32_t *const mine = stg + lane * kEpiPitch;
  for (int c0 = 0, wbase = 0; c0 < nvalid; c0 += 32 * G, wbase += PW) {
    uint32_t cur = 0;
    bool open = false;
    int wcur = 0;  // words of this period staged so far
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const int col = c0 + 32 * g;
      if (col >= nvalid) break;
      uint32_t r[32];
      ptx::tmem_ld_32x32b_x32(taddr + col, r);
      ptx::tmem_wait_ld();
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const int q = 32 * g + k;  // channel within the period (compile-time after unrolling)
        const int l = q % L;
        int32_t t = floor_scaled_biased(__uint_as_float(r[k]), scale);
        t = t < blo ? blo : (t > bhi ? bhi : t);
        if (col + k >= nvalid) t = kMagicBits;
        cur |= (static_cast<uint32_t>(t) & omask) << (l * OB);
        open = true;
        if (l == L - 1) {
          mine[wcur++] = cur;
          cur = 0;
          open = false;
        }
      }
    }
    if (open) mine[wcur] = cur;  // the row's last, partial word
    __syncwarp();
    const int nw = nwords - wbase < PW ? nwords - wbase : PW;  // this period's words inside the block
    const int wi = lane % PW;
#pragma unroll 4
    for (int r0 = 0; r0 < 32; r0 += RPI) {
      const int rr = r0 + lane / PW;
      const long long mr = __shfl_sync(0xffffffffu, m, rr);
      if (((vmask >> rr) & 1u) && wi < nw) out[mr * args.out_wpr + wbase + wi] = stg[rr * kEpiPitch + wi];
    }
    __syncwarp();
  }
}

// Every other case, 16 columns at a time: split digits (acc = 16 hi + lo),
// int32 outputs, accumulators too large for the fma path.
template <typename WO>
__device__ __forceinline__ void epilogue_row_general(const ConvArgs &args, uint32_t taddr, bool row_valid,
                                                     long long m, int nb) {
  const int ch0 = nb * args.NBc;
  const int nvalid = args.K - ch0 < args.NBc ? args.K - ch0 : args.NBc;
  const bool vec_ok = (args.K % 4 == 0) && (ch0 % 4 == 0);
  const int lo = lane_lo(args.out_bits, args.out_signed), hi = lane_hi(args.out_bits, args.out_signed);
  const uint32_t omask = (1u << args.out_bits) - 1;
  const int L = args.out_L, lw = args.out_lane_w;
  RowPacker<WO> pk;
  pk.dst = static_cast<WO *>(args.packed_out) + (m * args.out_wpr + ch0 / (L > 0 ? L : 1));
  for (int col = 0; col < nvalid; col += 16) {
    uint32_t r[16];
    int v[16];
    ptx::tmem_ld_32x32b_x16(taddr + col, r);
    if (args.split) {  // acc = 16 * hi + lo
      uint32_t r2[16];
      ptx::tmem_ld_32x32b_x16(taddr + args.n_mma + col, r2);
      ptx::tmem_wait_ld();
#pragma unroll
      for (int k = 0; k < 16; ++k)
        v[k] = 16 * __float2int_rn(__uint_as_float(r[k])) + __float2int_rn(__uint_as_float(r2[k]));
    } else {
      ptx::tmem_wait_ld();
      if (args.fast_acc) {  // |acc| < 2^22: the exact integer from the float's encoding
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = floor_scaled_biased(__uint_as_float(r[k]), 1.0f) - kMagicBits;
      } else {
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = __float2int_rn(__uint_as_float(r[k]));
      }
    }
    if (!row_valid) continue;
    const int cnt = nvalid - col < 16 ? nvalid - col : 16;
    if (args.acc_out) {
      int32_t *dst = args.acc_out + m * args.K + ch0 + col;
      if (cnt == 16 && vec_ok) {
#pragma unroll
        for (int k = 0; k < 4; ++k)
          reinterpret_cast<int4 *>(dst)[k] = make_int4(v[4 * k], v[4 * k + 1], v[4 * k + 2], v[4 * k + 3]);
      } else {
#pragma unroll
        for (int k = 0; k < 16; ++k)
          if (k < cnt) dst[k] = v[k];
      }
    }
    if (args.packed_out) {
#pragma unroll
      for (int k = 0; k < 16; ++k)
        if (k < cnt) pk.put(static_cast<uint32_t>(clamp_int(v[k] >> args.shift, lo, hi)) & omask, L, lw);
    }
  }
  if (args.packed_out && row_valid) pk.flush();
}

__device__ __forceinline__ void epilogue_row(const ConvArgs &args, uint32_t taddr, bool row_valid, long long m,
                                             int nb, uint32_t *estage) {
  const bool fast = args.packed_out && !args.acc_out && !args.split && args.fast_req;
  if (fast && args.out_lane_w == args.out_bits && (!args.out_word64 || (args.out_bits & (args.out_bits - 1)) == 0)) {
    switch (args.out_bits * 2 + (args.out_signed ? 1 : 0)) {
      case 2: epilogue_row_spec<1, false>(args, taddr, row_valid, m, nb); return;
      case 3: epilogue_row_spec<1, true>(args, taddr, row_valid, m, nb); return;
      case 4: epilogue_row_spec<2, false>(args, taddr, row_valid, m, nb); return;
      case 5: epilogue_row_spec<2, true>(args, taddr, row_valid, m, nb); return;
      case 6:
        if (estage)
          epilogue_row_period_staged<3, false>(args, taddr, row_valid, m, nb, estage);
        else
          epilogue_row_period<3, false>(args, taddr, row_valid, m, nb);
        return;
      case 7:
        if (estage)
          epilogue_row_period_staged<3, true>(args, taddr, row_valid, m, nb, estage);
        else
          epilogue_row_period<3, true>(args, taddr, row_valid, m, nb);
        return;
      case 8: epilogue_row_spec<4, false>(args, taddr, row_valid, m, nb); return;
      case 9: epilogue_row_spec<4, true>(args, taddr, row_valid, m, nb); return;
      case 10:
        if (estage)
          epilogue_row_period_staged<5, false>(args, taddr, row_valid, m, nb, estage);
        else
          epilogue_row_period<5, false>(args, taddr, row_valid, m, nb);
        return;
      case 11:
        if (estage)
          epilogue_row_period_staged<5, true>(args, taddr, row_valid, m, nb, estage);
        else
          epilogue_row_period<5, true>(args, taddr, row_valid, m, nb);
        return;
      case 12:
        if (estage)
          epilogue_row_period_staged<6, false>(args, taddr, row_valid, m, nb, estage);
        else
          epilogue_row_period<6, false>(args, taddr, row_valid, m, nb);
        return;
      case 13:
        if (estage)
          epilogue_row_period_staged<6, true>(args, taddr, row_valid, m, nb, estage);
        else
          epilogue_row_period<6, true>(args, taddr, row_valid, m, nb);
        return;
      case 14: epilogue_row_spec<7, false>(args, taddr, row_valid, m, nb); return;
      case 15: epilogue_row_spec<7, true>(args, taddr, row_valid, m, nb); return;
      case 16: epilogue_row_spec<8, false>(args, taddr, row_valid, m, nb); return;
      case 17: epilogue_row_spec<8, true>(args, taddr, row_valid, m, nb); return;
      default: break;
    }
  }
  if (args.out_word64) {
    if (fast)
      epilogue_row_fast<uint64_t>(args, taddr, row_valid, m, nb);
    else
      epilogue_row_general<uint64_t>(args, taddr, row_valid, m, nb);
  } else {
    if (fast)
      epilogue_row_fast<uint32_t>(args, taddr, row_valid, m, nb);
    else
      epilogue_row_general<uint32_t>(args, taddr, row_valid, m, nb);
  }
}

// The epilogue warps' meeting point of a pooled tile: every warp of the
// tile's group arrives on `bar` once its part of the step is done, then
// waits, bounded, for the phase; false if the wait gave up.
__device__ __forceinline__ bool epi_group_sync(uint32_t bar, uint32_t &phase, volatile int *status) {
  __syncwarp();
  bool ok = true;
  if ((threadIdx.x & 31) == 0) {
    ptx::mbar_arrive(bar);
    ok = ptx::mbar_wait_bounded(bar, phase & 1u, status, kWaitLimitNs);
  }
  ++phase;
  ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
  __syncwarp();
  return ok;
}

// Epilogue of one pooled tile for output lanes of OB = 1, 2, 4 or 8 bits
// (32-bit words, no spacers), called by each warp of the tile's group of
// gw warps (gi = this warp's index in it) for its 32 rows:
// requantize and pack the row (tile row trow) into the pool buffer, free the
// accumulator, meet the other epilogue warps, then write the lane-wise max of
// every 2x2 window of the tile's row pairs (the maximum commutes with the
// monotone requantize, so this is the pool of the requantized output), and
// meet again before the buffer is reused. False if a wait gave up.
template <int OB, bool OS>
__device__ __noinline__ bool epilogue_pool_tile(const ConvArgs &args, uint32_t taddr, int trow, uint32_t mt, int nb,
                                                uint32_t *pbuf, uint32_t acc_empty, uint32_t group_bar,
                                                uint32_t &phase, volatile int *status, int gw, int gi) {
  constexpr int LH = 32 / OB;  // lanes per word
  constexpr int NH = 32 / LH;  // words per 32 channels
  constexpr int32_t lo = OS ? -(1 << (OB - 1)) : 0, hi = OS ? (1 << (OB - 1)) - 1 : (1 << OB) - 1;
  constexpr int32_t blo = kMagicBits + lo, bhi = kMagicBits + hi;
  constexpr uint32_t omask = (1u << OB) - 1;
  constexpr uint32_t bias_sum = [] {
    uint32_t b = 0;
    for (int l = 0; l < LH; ++l) b += static_cast<uint32_t>(kMagicBits) << (l * OB);
    return b;
  }();
  const int ch0 = nb * args.NBc;
  const int nvalid = args.K - ch0 < args.NBc ? args.K - ch0 : args.NBc;
  const int nw = (nvalid + LH - 1) / LH;  // this block's words of a row (<= pool_nw; fewer in a last, partial block)
  const int pitch = args.pool_pitch;
  const float scale = args.out_scale;
  uint32_t *prow = pbuf + trow * pitch;
  for (int col = 0; col < nvalid; col += 32) {
    uint32_t r[32];
    ptx::tmem_ld_32x32b_x32(taddr + col, r);
    ptx::tmem_wait_ld();
    const int cnt = nvalid - col < 32 ? nvalid - col : 32;
#pragma unroll
    for (int j = 0; j < NH; ++j) {
      uint32_t w = 0;
#pragma unroll
      for (int l = 0; l < LH; ++l) {
        int32_t t = floor_scaled_biased(__uint_as_float(r[j * LH + l]), scale);
        t = t < blo ? blo : (t > bhi ? bhi : t);
        if (j * LH + l >= cnt) t = kMagicBits;  // lanes past the block's channels stay zero
        if constexpr (OS)
          w |= (static_cast<uint32_t>(t) & omask) << (l * OB);
        else
          w += static_cast<uint32_t>(t) << (l * OB);
      }
      const int wi = col / LH + j;
      if (wi < nw) prow[wi] = OS ? w : w - bias_sum;
    }
  }
  ptx::tc_fence_before();
  __syncwarp();
  if ((threadIdx.x & 31) == 0) ptx::mbar_arrive(acc_empty);
  if (!epi_group_sync(group_bar, phase, status)) return false;
  // the 2x2 windows of this tile's row pairs
  const uint32_t img = fdiv(mt, args.fd_tpi);
  const int g = static_cast<int>(mt - img * args.fd_tpi.d);
  const int Ho2 = args.Ho / 2, Wo2 = args.Wo / 2, q = args.pool_rows / 2;
  const int q_here = Ho2 - g * q < q ? Ho2 - g * q : q;
  const int total = q_here * Wo2 * nw;
  const uint32_t flip = OS ? LaneMsb<uint32_t, OB>::kValue : 0u;
  uint32_t *out = static_cast<uint32_t *>(args.packed_out) + ch0 / LH;
  const int Wp = args.Wp;
  for (int idx = 32 * gi + static_cast<int>(threadIdx.x & 31); idx < total; idx += 32 * gw) {
    const int pix = idx / nw, w = idx - (idx / nw) * nw;
    const int i = pix / Wo2, j = pix - (pix / Wo2) * Wo2;
    const uint32_t *b0 = pbuf + (2 * i * Wp + 2 * j) * pitch + w;
    const uint32_t top = swar_lane_max<uint32_t, OB>(b0[0], b0[pitch], flip);
    const uint32_t bot = swar_lane_max<uint32_t, OB>(b0[Wp * pitch], b0[(Wp + 1) * pitch], flip);
    const long long orow = (static_cast<long long>(img) * Ho2 + g * q + i) * Wo2 + j;
    out[orow * args.out_wpr + w] = swar_lane_max<uint32_t, OB>(top, bot, flip);
  }
  return epi_group_sync(group_bar, phase, status);
}

__device__ __forceinline__ bool epilogue_pool_dispatch(const ConvArgs &args, uint32_t taddr, int trow, uint32_t mt,
                                                       int nb, uint32_t *pbuf, uint32_t acc_empty, uint32_t group_bar,
                                                       uint32_t &phase, volatile int *status, int gw, int gi) {
#define SAMD_POOL_TILE(OB, OS) \
  epilogue_pool_tile<OB, OS>(args, taddr, trow, mt, nb, pbuf, acc_empty, group_bar, phase, status, gw, gi)
  switch (args.out_bits * 2 + (args.out_signed ? 1 : 0)) {
    case 2: return SAMD_POOL_TILE(1, false);
    case 3: return SAMD_POOL_TILE(1, true);
    case 4: return SAMD_POOL_TILE(2, false);
    case 5: return SAMD_POOL_TILE(2, true);
    case 8: return SAMD_POOL_TILE(4, false);
    case 9: return SAMD_POOL_TILE(4, true);
    case 16: return SAMD_POOL_TILE(8, false);
    default: return SAMD_POOL_TILE(8, true);
  }
#undef SAMD_POOL_TILE
}

// One MMA.
template <bool FP8>
__device__ __forceinline__ void mma_op(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
  if constexpr (FP8)
    ptx::mma_f8(d, a, b, idesc, acc);
  else
    ptx::mma_f16(d, a, b, idesc, acc);
}

// For a tile of HV parts of 128 rows (HV = 1, 2, 4), each k-step issues one
// MMA per part: part h accumulates into d + h * dn from A rows 128 h on
// (a + h * ah).
template <bool FP8, int HV>
__device__ __forceinline__ void mma_kstep(uint32_t d, uint32_t dn, uint64_t a, uint64_t ah, uint64_t b, uint32_t idesc,
                                          uint32_t acc) {
  mma_op<FP8>(d, a, b, idesc, acc);
  if constexpr (HV >= 2) mma_op<FP8>(d + dn, a + ah, b, idesc, acc);
  if constexpr (HV == 4) {
    mma_op<FP8>(d + 2 * dn, a + 2 * ah, b, idesc, acc);
    mma_op<FP8>(d + 3 * dn, a + 3 * ah, b, idesc, acc);
  }
}

// Issues `ksteps` (1..4) k-steps of one operand row as straight-line code.
template <bool FP8, int HV>
__device__ __forceinline__ void mma_ksteps(int ksteps, uint32_t d, uint32_t dn, uint64_t a, uint64_t ah, uint64_t b,
                                           uint32_t idesc, uint32_t acc) {
  switch (ksteps) {
    case 4:
      mma_kstep<FP8, HV>(d, dn, a, ah, b, idesc, acc);
      mma_kstep<FP8, HV>(d, dn, a + 2, ah, b + 2, idesc, 1u);
      mma_kstep<FP8, HV>(d, dn, a + 4, ah, b + 4, idesc, 1u);
      mma_kstep<FP8, HV>(d, dn, a + 6, ah, b + 6, idesc, 1u);
      break;
    case 3:
      mma_kstep<FP8, HV>(d, dn, a, ah, b, idesc, acc);
      mma_kstep<FP8, HV>(d, dn, a + 2, ah, b + 2, idesc, 1u);
      mma_kstep<FP8, HV>(d, dn, a + 4, ah, b + 4, idesc, 1u);
      break;
    case 2:
      mma_kstep<FP8, HV>(d, dn, a, ah, b, idesc, acc);
      mma_kstep<FP8, HV>(d, dn, a + 2, ah, b + 2, idesc, 1u);
      break;
    default:
      mma_kstep<FP8, HV>(d, dn, a, ah, b, idesc, acc);
      break;
  }
}

// Issues the MMAs of all `taps` taps of one operand stage with resident
// weights: tap t reads weight tile t (b advances by b_step16) and the A
// operand one row further on, skipping a_skip16 at the end of each filter
// row (HALO); straight-line issue keeps the tensor core fed. Descriptors
// advance in 16-byte units of their start-address field.
template <bool FP8, int HV>
__device__ __forceinline__ void issue_taps(uint32_t d, uint32_t dn, uint64_t a, uint64_t ah, uint64_t b, uint32_t idesc,
                                           int ksteps, int taps, int S, uint32_t a_row16, uint32_t a_skip16,
                                           uint32_t b_step16, uint32_t acc) {
  int s = 0;
  for (int t = 0; t < taps; ++t) {
    mma_ksteps<FP8, HV>(ksteps, d, dn, a, ah, b, idesc, acc);
    acc = 1;
    b += b_step16;
    a += a_row16;
    if (++s == S) {
      s = 0;
      a += a_skip16;
    }
  }
}

// ---- the persistent convolution kernel ----------------------------------------
//
// One CTA per SM loops over output tiles (tile = blockIdx.x + i * gridDim.x;
// tile = nb * grid_m + mt: channel block nb, position tile mt of 128 * HV
// positions; with HV = 2 or 4 each k-step issues one MMA per 128-row part,
// so the parts share every synchronization). Eighteen warps with fixed
// roles, connected by mbarrier rings:
//   warp 0      TMEM allocation; lane 0 streams weight tiles with TMA. When
//               the layer has one channel block and all its weight tiles fit,
//               they are loaded once and stay resident.
//   warp 1      issues tcgen05.mma (one elected lane) into one of two TMEM
//               accumulators, so tile i+1 accumulates while the epilogue
//               drains tile i.
//   warps 2-9   operand producers.
//               HALO: for each (tile, channel chunk) the halo rows the tile
//               needs are gathered with cp.async and widened once into one of
//               two or three halo buffers; every tap reads the halo through a
//               descriptor shifted by r * row_step + s rows.
//               GATHER: each thread gathers its pixel's packed words (implicit
//               im2col, zero padding) through a cp.async ring and widens them
//               into a ring of A tiles; with HV = 1 two groups of four warps
//               take alternate (tile, chunk) items, with HV = 2 the two groups
//               fill the two halves of every item. Chunks that are not whole
//               16-byte vectors are copied as 16-byte windows.
//   warps 10-17 epilogue: tcgen05.ld, exact integers, optional int32 store,
//               optional requantize-and-pack. HV = 1: warps 10-13 drain
//               accumulator 0 (the CTA's even tiles), warps 14-17
//               accumulator 1; HV = 2: warps 10-13 drain the first half and
//               14-17 the second half of every tile; HV = 4 (halo layers on
//               e4m3 operands): warps 10-13 drain parts 0 and 1, 14-17 parts
//               2 and 3. Warp w reads the TMEM lanes of quadrant w % 4. A
//               first, store-free pass over the first tile fetches the
//               epilogue's code early. Pooled tiles (ConvArgs::pool) are
//               drained, requantized and pooled by the warps of a group.
// Every wait is bounded; a role that gives up records SAMD_ETIMEOUT and stops.
template <typename W, int BITS, bool SIGNED, bool HALO, bool FP8, bool FULL, int HV>
__global__ void __launch_bounds__(kThreads, 1) conv_kernel(const __grid_constant__ CUtensorMap tmap_b,
                                                           const ConvArgs args) {
  using U = AUnpack<W, BITS, SIGNED, FP8, FULL>;
  constexpr int BMT = BM * HV;  // output positions per tile
  using T = OpTraits<FP8>;
  constexpr int WC = U::WC;
  using St = Staging<W, WC>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int STB = args.stages;  // weight tiles in flight (or resident)
  const bool resident = args.b_resident != 0;
  const uint32_t b_bytes = args.b_bytes;
  uint8_t *sOp = smem;  // HALO: hbufs halo buffers; GATHER: stages_a A tiles
  uint8_t *sB = smem + args.off_b;
  uint8_t *sG = smem + args.off_g;  // packed staging
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + args.off_bar);
  // barriers: full_b[STB] empty_b[STB] opfull[NO] opempty[NO] accfull[2] accempty[2] drain group[2]
  const int NO = HALO ? args.hbufs : args.stages_a;
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + 2 * STB + 2 * NO + 7);
  auto full_b = [&](int s) { return ptx::smem_addr(bars + s); };
  auto empty_b = [&](int s) { return ptx::smem_addr(bars + STB + s); };
  auto opfull = [&](int s) { return ptx::smem_addr(bars + 2 * STB + s); };
  auto opempty = [&](int s) { return ptx::smem_addr(bars + 2 * STB + NO + s); };
  auto accfull = [&](int a) { return ptx::smem_addr(bars + 2 * STB + 2 * NO + a); };
  auto accempty = [&](int a) { return ptx::smem_addr(bars + 2 * STB + 2 * NO + 2 + a); };
  const uint32_t drain_bar = ptx::smem_addr(bars + 2 * STB + 2 * NO + 4);
  // the epilogue warps of a pooled tile: all eight (two-half tiles), or the
  // four of epilogue set g (one-half tiles, group_bar(g))
  auto group_bar = [&](int g) { return ptx::smem_addr(bars + 2 * STB + 2 * NO + 5 + g); };

  volatile int *status = args.status;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // No global read precedes the setup barrier: a failure recorded by an
  // earlier launch is seen by the first wait that has to wait.
  if (warp == 0) {
    ptx::tmem_alloc(ptx::smem_addr(tmem_holder), args.tmem_cols);
    ptx::tmem_relinquish();
  }
  if (threadIdx.x == 32) {
    for (int s = 0; s < STB; ++s) {
      ptx::mbar_init(full_b(s), 1);
      ptx::mbar_init(empty_b(s), 1);
    }
    for (int s = 0; s < NO; ++s) {
      ptx::mbar_init(opfull(s), (HALO || HV == 2) ? kProdWarps : kProdWarps / 2);
      ptx::mbar_init(opempty(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(accfull(a), 1);
      ptx::mbar_init(accempty(a), HV >= 2 ? kEpiWarps : kEpiWarps / 2);  // the warps that drain accumulator a
    }
    ptx::mbar_init(drain_bar, 1);
    for (int g = 0; g < 2; ++g) ptx::mbar_init(group_bar(g), HV >= 2 ? kEpiWarps : kEpiWarps / 2);
    ptx::fence_barrier_init();
  }
  __syncwarp();  // every warp reaches the barrier converged (bar.sync counts whole warps)
  ptx::tc_fence_before();
  __syncthreads();
  ptx::tc_fence_after();
  const uint32_t tmem_base = *tmem_holder;

  const long long total_tiles = static_cast<long long>(args.grid_m) * args.nblocks;
  const long long first_tile = blockIdx.x, tile_step = gridDim.x;
  const int nchunks = args.nchunks;  // weight tiles per output tile
  bool ok = true;

  if (warp == 0) {
    if (lane == 0) {
      // ---- weight tiles ----
      ptx::prefetch_tmap(&tmap_b);
      int quiet = 0;  // the waits below end only when the copies land (or time out)
      if (resident) {
        for (int c = 0; c < nchunks; ++c) {
          ptx::mbar_arrive_expect_tx(full_b(c), b_bytes);
          ptx::tma_load_2d(ptx::smem_addr(sB + c * b_bytes), &tmap_b, c * BK, 0, full_b(c));
        }
        // the CTA does not exit with a copy in flight, whatever the other roles do
        for (int c = 0; c < nchunks; ++c) ptx::mbar_wait_bounded(full_b(c), 0, &quiet, kWaitLimitNs);
      } else {
        long long cb = 0;
        for (long long tile = first_tile; tile < total_tiles && ok; tile += tile_step) {
          const int nb = static_cast<int>(tile / args.grid_m);
          for (int c = 0; c < nchunks; ++c, ++cb) {
            const int s = static_cast<int>(cb % STB);
            const long long round = cb / STB;
            if (round > 0 &&
                !ptx::mbar_wait_bounded(empty_b(s), static_cast<uint32_t>((round - 1) & 1), status, kWaitLimitNs)) {
              ok = false;
              break;
            }
            ptx::mbar_arrive_expect_tx(full_b(s), b_bytes);
            ptx::tma_load_2d(ptx::smem_addr(sB + s * b_bytes), &tmap_b, c * BK, nb * args.mma_n, full_b(s));
          }
        }
        if (!ok) {  // leave no copy in flight: wait (bounded) for the last ring's worth
          for (long long k = (cb > STB ? cb - STB : 0); k < cb; ++k)
            ptx::mbar_wait_bounded(full_b(static_cast<int>(k % STB)), static_cast<uint32_t>((k / STB) & 1), &quiet,
                                   kWaitLimitNs / 10);
        }
      }
    }
  } else if (warp == 1) {
    // ---- MMA issue ----
    // The whole warp runs this loop on warp-uniform values and one elected
    // lane (always the same one: all lanes are converged) issues each
    // tcgen05.mma and tcgen05.commit. Running the loop in one thread alone
    // turns every descriptor into a per-thread value that has to be moved to
    // the uniform datapath before each MMA, which costs more than the MMA.
    const uint32_t idesc = ptx::idesc_f16_f32(BM, args.mma_n);
    auto wait = [&](uint32_t bar, uint32_t parity) {
      bool w_ok = true;
      if (lane == 0) w_ok = ptx::mbar_wait_bounded(bar, parity, status, kWaitLimitNs);
      return __shfl_sync(0xffffffffu, w_ok ? 1 : 0, 0) != 0;
    };
    // Ring positions advance by increments (no division in this loop).
    int sb = 0, so = 0;
    uint32_t bpar = 0, opar = 0;
    const uint32_t sB_addr = ptx::smem_addr(sB), sOp_addr = ptx::smem_addr(sOp);
    const int nops = HALO ? args.nck : nchunks;  // operand stages per tile
    const int taps_here = HALO ? args.taps : 1;
    constexpr uint32_t a_row16 = T::kRowBytes / 16;  // one operand row in descriptor units
    constexpr uint64_t a_half16 = static_cast<uint64_t>(BM) * a_row16;  // from one 128-row part's A rows to the next
    const uint32_t dn = static_cast<uint32_t>(args.mma_n);          // the second half's accumulator columns
    const uint32_t a_skip16 = HALO ? static_cast<uint32_t>(args.row_step - args.S) * a_row16 : 0u;
    if (resident)  // resident weights: wait for all of them once
      for (int c = 0; c < nchunks && ok; ++c)
        if (!wait(full_b(c), 0)) ok = false;
    long long i = 0;
    for (long long tile = first_tile; tile < total_tiles && ok; tile += tile_step, ++i) {
      const int a = static_cast<int>(i & 1);
      if (i >= 2 && !wait(accempty(a), static_cast<uint32_t>(((i >> 1) - 1) & 1))) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();  // the epilogue's reads of this accumulator are complete
      const uint32_t tmem_d = tmem_base + static_cast<uint32_t>(a * HV * args.mma_n);
      uint32_t acc = 0;
      for (int j = 0; j < nops && ok; ++j) {
        if (!wait(opfull(so), opar)) {
          ok = false;
          break;
        }
        // words of the packed chunk: channel chunk j (halo) or j / taps
        // (window gather) of a pixel, else words j WC.. of the whole reduction
        int words = HALO ? args.wpr - j * WC
                         : (args.gather_win ? args.wpr - (j / args.taps) * WC : args.words_total - j * WC);
        if (words > WC) words = WC;
        int npos = words * U::L;
        if (npos > BK) npos = BK;  // FULL: the last word's lanes past 64 are padding
        const int ksteps = (npos + T::kKPerMma - 1) / T::kKPerMma;
        // No tcgen05 fence here: the operands arrived through the async proxy
        // (TMA, or stores fenced with fence.proxy.async before the producers'
        // arrive), which the mbarrier wait already orders.
        const uint64_t a0 = T::desc(sOp_addr + so * args.op_stride);
        if (resident) {
          const uint64_t b0 = T::desc(sB_addr + (HALO ? j * taps_here : j) * b_bytes);
          if (ptx::elect_one())
            issue_taps<FP8, HV>(tmem_d, dn, a0, a_half16, b0, idesc, ksteps, taps_here, args.S, a_row16, a_skip16,
                                b_bytes >> 4, acc);
          __syncwarp();
          acc = 1;
        } else {
          uint64_t adesc = a0;
          int ts = 0;
          for (int t = 0; t < taps_here; ++t) {
            if (!wait(full_b(sb), bpar)) {
              ok = false;
              break;
            }
            const uint64_t bdesc = T::desc(sB_addr + sb * b_bytes);
            if (ptx::elect_one()) {
              mma_ksteps<FP8, HV>(ksteps, tmem_d, dn, adesc, a_half16, bdesc, idesc, acc);
              ptx::mma_commit(empty_b(sb));
            }
            __syncwarp();
            acc = 1;
            if (++sb == STB) {
              sb = 0;
              bpar ^= 1;
            }
            if (HALO) {
              adesc += a_row16;  // next halo row
              if (++ts == args.S) {
                ts = 0;
                adesc += a_skip16;
              }
            }
          }
        }
        if (ptx::elect_one()) ptx::mma_commit(opempty(so));  // the stage is free once these MMAs complete
        __syncwarp();
        if (++so == NO) {
          so = 0;
          opar ^= 1;
        }
      }
      if (ok) {
        if (ptx::elect_one()) ptx::mma_commit(accfull(a));
        __syncwarp();
      }
    }
    if (ptx::elect_one()) ptx::mma_commit(drain_bar);
    __syncwarp();
    if (lane == 0) {
      int quiet = 0;
      ptx::mbar_wait_bounded(drain_bar, 0, &quiet, kWaitLimitNs);
    }
    __syncwarp();
  } else if (warp < kFirstEpiWarp) {
    // ---- operand producers ----
    const int t = threadIdx.x - 64;  // 0 .. kProdThreads - 1
    const W *act = static_cast<const W *>(args.act);
    auto wait_lane0 = [&](uint32_t bar, uint32_t parity) {
      bool w_ok = true;
      if (lane == 0) w_ok = ptx::mbar_wait_bounded(bar, parity, status, kWaitLimitNs);
      return __shfl_sync(0xffffffffu, w_ok ? 1 : 0, 0) != 0;
    };
    if constexpr (HALO) {
      const int halo_rows = args.nseg * args.seg_rows;
      // halo row hr -> virtual offset from the tile's first position, or -1
      auto voff = [&](int hr) -> int {
        const int g = static_cast<int>(fdiv(static_cast<uint32_t>(hr), args.fd_seg));
        const int q = hr - g * args.seg_rows;
        return q < args.seg_used ? g * args.Wp + q : -1;
      };
      // items k = (tile i, channel chunk j), in the MMA's order
      auto gather = [&](long long tile, int j, int slot) {
        const uint32_t mt = static_cast<uint32_t>(tile) - fdiv(static_cast<uint32_t>(tile), args.fd_gm) * args.fd_gm.d;
        const uint32_t v0 = tile_first_pos(args, mt, BMT);
        const uint32_t dst0 = ptx::smem_addr(sG + slot * args.g_stride);
        for (int hr = t; hr < halo_rows; hr += kProdThreads) {
          const int off = voff(hr);
          if (off < 0) continue;
          const uint32_t u = v0 + static_cast<uint32_t>(off);
          const uint32_t img = fdiv(u, args.fd_plane);
          const uint32_t rem = u - img * args.fd_plane.d;
          const uint32_t ihp = fdiv(rem, args.fd_wp);
          const int ih = static_cast<int>(ihp) - args.pad;
          const int iw = static_cast<int>(rem - ihp * args.fd_wp.d) - args.pad;
          const bool valid = static_cast<int>(img) < args.N && ih >= 0 && ih < args.H && iw >= 0 && iw < args.W;
          const W *px = act + ((static_cast<long long>(img) * args.H + ih) * args.W + iw) * args.wpr + j * WC;
          const uint32_t dst = dst0 + hr * St::kRowBytes;
          if (args.gather_vec) {
            stage_chunk<W, WC>(dst, reinterpret_cast<const char *>(valid ? px : act), valid ? 1u : 0u);
          } else {
#pragma unroll
            for (int q = 0; q < WC; ++q) {
              const bool in = valid && j * WC + q < args.wpr;
              const W *src = in ? px + q : act;
              if constexpr (sizeof(W) == 8)
                ptx::cp_async_8(dst + 8 * q, src, in ? 8u : 0u);
              else
                ptx::cp_async_4(dst + 4 * q, src, in ? 4u : 0u);
            }
          }
        }
      };
      auto advance = [&](long long &tile, int &j) {
        if (++j == args.nck) {
          j = 0;
          tile += tile_step;
        }
      };
      // Packed staging is a ring of D = gdepth slots: item k is gathered
      // into slot k mod D, D - 1 items before it is widened. Each iteration
      // commits exactly one cp.async group (empty past the last item), so
      // waiting until at most D - 1 groups are pending means item k landed.
      // A thread reads back only the rows it gathered itself, so refilling
      // the slot it finished with one item earlier needs no barrier.
      const int D = args.gdepth;
      long long gtile = first_tile;  // issue side
      int gj = 0, gslot = 0;
      auto issue = [&]() {
        if (gtile < total_tiles) gather(gtile, gj, gslot);
        ptx::cp_async_commit();
        advance(gtile, gj);
        if (++gslot == D) gslot = 0;
      };
      for (int d = 0; d + 1 < D; ++d) issue();
      long long ctile = first_tile;  // widening side
      int cj = 0, cslot = 0;
      for (long long k = 0; ctile < total_tiles; ++k) {
        issue();
        if (D == 4)
          ptx::cp_async_wait<3>();
        else if (D == 3)
          ptx::cp_async_wait<2>();
        else
          ptx::cp_async_wait<1>();  // item k of this thread's rows has landed
        const int hb = static_cast<int>(k % NO);
        if (k >= NO && !wait_lane0(opempty(hb), static_cast<uint32_t>(((k / NO) - 1) & 1))) {
          ok = false;
          break;
        }
        const uint8_t *stg = sG + cslot * args.g_stride;
        for (int hr = t; hr < halo_rows; hr += kProdThreads) {
          if (voff(hr) < 0) continue;  // a row no tap reads
          W cur[WC];
          load_staged<W, WC>(stg + hr * St::kRowBytes, cur);
          U::unpack_row(cur, sOp + hb * args.op_stride, hr);
        }
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(opfull(hb));
        advance(ctile, cj);
        if (++cslot == D) cslot = 0;
      }
      ptx::cp_async_wait<0>();
    } else {
      // GATHER: with one-half tiles group grp (four warps) takes items grp,
      // grp + 2, ...; with two-half tiles both groups take every item, group
      // grp filling rows 128 grp .. 128 grp + 127. A thread owns one row.
      const int grp = t / BM;
      const int row = (HV == 2 ? grp * BM : 0) + t % BM;  // row of the A tile
      constexpr int kItemStep = HV == 2 ? 1 : 2;
      AGather<W, WC> g;
      g.act = act;
      g.H = args.H;
      g.W_ = args.W;
      g.wpr = args.wpr;
      g.S = args.S;
      g.stride = args.stride;
      g.pad = args.pad;
      g.words_total = args.words_total;
      g.taps = args.taps;
      g.vec = args.gather_vec != 0;
      auto set_tile = [&](long long tile) {
        const uint32_t tl = static_cast<uint32_t>(tile);
        const uint32_t mt = tl - fdiv(tl, args.fd_gm) * args.fd_gm.d;
        const uint32_t m = mt * BMT + row;
        g.row_valid = m < static_cast<uint64_t>(args.M);
        const uint32_t mm = g.row_valid ? m : 0u;
        const uint32_t tq = fdiv(mm, args.fd_wo);
        g.ow = static_cast<int>(mm - tq * args.fd_wo.d);
        const uint32_t nq = fdiv(tq, args.fd_ho);
        g.oh = static_cast<int>(tq - nq * args.fd_ho.d);
        g.n = static_cast<int>(nq);
      };
      const uint32_t g_row = static_cast<uint32_t>(args.g_row);  // staging row pitch
      const uint32_t kSlotBytes = BM * g_row;
      const uint32_t slot0 = ptx::smem_addr(sG) + grp * (kGatherDepth * kSlotBytes) + (t % BM) * g_row;
      const bool win = args.gather_win != 0;
      const uintptr_t act_end = reinterpret_cast<uintptr_t>(args.act) + static_cast<uintptr_t>(args.act_bytes);
      uint32_t o4s = 0;  // window offsets of the kGatherDepth slots, 2 bits each
      // issue side: this group's item (itile, ic), kGatherDepth ahead of the consume side
      long long itile = first_tile;
      int ic = 0;
      auto step = [&]() {
        if (++ic == nchunks) {
          ic = 0;
          itile += tile_step;
        }
      };
      if (HV == 1 && grp == 1) step();
      if (itile < total_tiles) set_tile(itile);
      auto issue_next = [&](int slot) {
        if (itile < total_tiles) {
          if (win) {
            const int o4 = g.issue_win(ic, slot0 + slot * kSlotBytes, act_end);
            o4s = (o4s & ~(3u << (2 * slot))) | (static_cast<uint32_t>(o4) << (2 * slot));
          } else {
            g.issue(ic, slot0 + slot * kSlotBytes);
          }
          const long long prev = itile;
          step();
          if (kItemStep == 2) step();
          if (itile != prev && itile < total_tiles) set_tile(itile);
        }
        ptx::cp_async_commit();
      };
#pragma unroll 1
      for (int d = 0; d < kGatherDepth; ++d) issue_next(d);
      const long long items = ((total_tiles - first_tile + tile_step - 1) / tile_step) * nchunks;
      int slot = 0;
      for (long long k = HV == 2 ? 0 : grp; k < items; k += kItemStep) {
        ptx::cp_async_wait<kGatherDepth - 1>();
        W cur[WC];
        const uint8_t *srow = sG + grp * (kGatherDepth * kSlotBytes) + slot * kSlotBytes + (t % BM) * g_row;
        if (win) {
          const int chunk = static_cast<int>(k % nchunks);
          const int wi = (chunk / args.taps) * WC;
          const int nw = args.wpr - wi < WC ? args.wpr - wi : WC;
          load_window<W, WC>(srow, static_cast<int>((o4s >> (2 * slot)) & 3u), nw, cur);
        } else {
          load_staged<W, WC>(srow, cur);
        }
        const int sa = static_cast<int>(k % NO);
        const long long round = k / NO;
        if (round > 0 && !wait_lane0(opempty(sa), static_cast<uint32_t>((round - 1) & 1))) {
          ok = false;
          break;
        }
        U::unpack_row(cur, sOp + sa * args.op_stride, row);
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(opfull(sa));
        issue_next(slot);  // refill the slot just read
        if (++slot == kGatherDepth) slot = 0;
      }
      ptx::cp_async_wait<0>();
    }
  } else {
    // ---- epilogue ----
    // One-half tiles: warp set `set` drains accumulator `set`, i.e. the CTA's
    // tiles i with i % 2 == set. Two-half tiles: both sets drain every tile,
    // set `set` its half `set`. Warp w reads the TMEM lanes of quadrant w % 4.
    const int quad = warp & 3;
    const int set = (warp - kFirstEpiWarp) / 4;
    uint32_t *const estage =
        args.e_stage ? reinterpret_cast<uint32_t *>(smem + args.off_e) + (warp - kFirstEpiWarp) * 32 * kEpiPitch
                     : nullptr;
    const int row = quad * 32 + lane;
    constexpr int kTileStep = HV >= 2 ? 1 : 2;
    // parts of 128 rows of a tile this warp drains: set `set` takes parts
    // set * kParts .. set * kParts + kParts - 1 (HV = 2: its half; HV = 4:
    // two of the four parts); with HV = 1 the sets take alternate tiles
    constexpr int kParts = HV == 4 ? 2 : 1;
    long long i = HV >= 2 ? 0 : set;
    // The first pass over the first tile runs with its stores off and without
    // waiting for the accumulator (whatever it reads is discarded): the row
    // epilogue is the largest code of the kernel, and this way its
    // instructions are fetched while the first tile is being computed rather
    // than after it.
    bool warm = true;
    bool pooled = false;
    if constexpr (HALO && HV <= 2) {
      if (args.pool) {
        // pooled tiles (no warm-up pass): two-half tiles are drained and
        // pooled by all eight epilogue warps, one-half tiles by the four of
        // the set that drains them (alternate tiles, own buffer and barrier)
        pooled = true;
        constexpr int gw = HV == 2 ? kEpiWarps : kEpiWarps / 2;
        const int gi = HV == 2 ? warp - kFirstEpiWarp : warp - kFirstEpiWarp - 4 * set;
        uint32_t *const pbuf = reinterpret_cast<uint32_t *>(smem + args.off_e) + (HV == 2 ? 0 : set * BM * args.pool_pitch);
        const uint32_t gbar = group_bar(HV == 2 ? 0 : set);
        constexpr int kStep = HV == 2 ? 1 : 2;
        uint32_t gphase = 0;
        long long ip = HV == 2 ? 0 : set;
        for (long long tile = first_tile + (HV == 2 ? 0 : set) * tile_step; tile < total_tiles;
             tile += kStep * tile_step, ip += kStep) {
          const int acc_i = HV == 2 ? static_cast<int>(ip & 1) : set;
          bool w_ok = true;
          if (lane == 0)
            w_ok = ptx::mbar_wait_bounded(accfull(acc_i), static_cast<uint32_t>((ip >> 1) & 1), status, kWaitLimitNs);
          if (!__shfl_sync(0xffffffffu, w_ok ? 1 : 0, 0)) {
            ok = false;
            break;
          }
          ptx::tc_fence_after();
          const uint32_t tl = static_cast<uint32_t>(tile);
          const uint32_t nbu = fdiv(tl, args.fd_gm);
          const uint32_t mt = tl - nbu * args.fd_gm.d;
          const uint32_t taddr = tmem_base + static_cast<uint32_t>((acc_i * HV + (HV == 2 ? set : 0)) * args.mma_n) +
                                 (static_cast<uint32_t>(quad * 32) << 16);
          if (!epilogue_pool_dispatch(args, taddr, (HV == 2 ? set * BM : 0) + row, mt, static_cast<int>(nbu), pbuf,
                                      accempty(acc_i), gbar, gphase, status, gw, gi)) {
            ok = false;
            break;
          }
        }
      }
    }
    for (long long tile = first_tile + (HV >= 2 ? 0 : set) * tile_step; !pooled && tile < total_tiles;) {
      const int acc_i = HV >= 2 ? static_cast<int>(i & 1) : set;  // accumulator of this tile
      if (!warm) {
        bool w_ok = true;
        if (lane == 0)
          w_ok = ptx::mbar_wait_bounded(accfull(acc_i), static_cast<uint32_t>((i >> 1) & 1), status, kWaitLimitNs);
        if (!__shfl_sync(0xffffffffu, w_ok ? 1 : 0, 0)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();
      }
      const uint32_t tl = static_cast<uint32_t>(tile);
      const uint32_t nbu = fdiv(tl, args.fd_gm);
      const int nb = static_cast<int>(nbu);
      const uint32_t mt = tl - nbu * args.fd_gm.d;
#pragma unroll 1
      for (int hh = 0; hh < kParts; ++hh) {
        const int part = HV >= 2 ? set * kParts + hh : 0;
        bool valid;
        long long m;
        const int trow = part * BM + row;  // row of the tile
        if (HALO) {
          const uint32_t v = tile_first_pos(args, mt, BMT) + trow;
          const uint32_t img = fdiv(v, args.fd_plane);
          const uint32_t rem = v - img * args.fd_plane.d;
          const uint32_t oh = fdiv(rem, args.fd_wp);
          const uint32_t ow = rem - oh * args.fd_wp.d;
          valid = static_cast<int>(img) < args.N && static_cast<int>(oh) < args.Ho && static_cast<int>(ow) < args.Wo;
          m = (static_cast<long long>(img) * args.Ho + oh) * args.Wo + ow;
        } else {
          m = static_cast<long long>(mt) * BMT + trow;
          valid = m < args.M;
        }
        const uint32_t taddr = tmem_base + static_cast<uint32_t>((acc_i * HV + part) * args.mma_n) +
                               (static_cast<uint32_t>(quad * 32) << 16);
        epilogue_row(args, taddr, valid && !warm, m, nb, estage);
      }
      if (warm) {
        warm = false;
        continue;
      }
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(accempty(acc_i));
      tile += kTileStep * tile_step;
      i += kTileStep;
    }
  }

  __syncwarp();
  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem_base, args.tmem_cols);
  }
  if (!ok) atomicOr(const_cast<int *>(status), static_cast<int>(SAMD_ETIMEOUT));
}

// cudaFuncSetAttribute once per (kernel, device); defined in conv2d.cu.
cudaError_t ensure_smem_attr(const void *kern, size_t smem);

// FULL variants exist only for lane counts that do not divide 64.
__host__ __device__ constexpr bool needs_full(int word_bits, int bits) { return 64 % (word_bits / bits) != 0; }

template <typename W, int BITS, bool SIGNED, bool FP8>
cudaError_t launch_conv(const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid, size_t smem,
                        cudaStream_t s) {
  constexpr bool kHasFull = needs_full(WordTraits<W>::kBits, BITS);
  using K = void (*)(const CUtensorMap, const ConvArgs);
  K kern;
  if (args.hv == 2)
    kern = halo ? conv_kernel<W, BITS, SIGNED, true, FP8, false, 2> : conv_kernel<W, BITS, SIGNED, false, FP8, false, 2>;
  else
    kern = halo ? conv_kernel<W, BITS, SIGNED, true, FP8, false, 1> : conv_kernel<W, BITS, SIGNED, false, FP8, false, 1>;
  if constexpr (kHasFull) {
    if (args.full && args.hv == 2)
      kern = halo ? conv_kernel<W, BITS, SIGNED, true, FP8, true, 2> : conv_kernel<W, BITS, SIGNED, false, FP8, true, 2>;
    else if (args.full)
      kern = halo ? conv_kernel<W, BITS, SIGNED, true, FP8, true, 1> : conv_kernel<W, BITS, SIGNED, false, FP8, true, 1>;
  }
  // four-part tiles: halo layers on e4m3 operands only (planned so)
  if constexpr (FP8) {
    if (args.hv == 4) {
      if (!halo) return cudaErrorInvalidValue;
      kern = conv_kernel<W, BITS, SIGNED, true, FP8, false, 4>;
      if constexpr (kHasFull)
        if (args.full) kern = conv_kernel<W, BITS, SIGNED, true, FP8, true, 4>;
    }
  } else {
    if (args.hv == 4) return cudaErrorInvalidValue;
  }
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void *>(kern), smem);
  if (e != cudaSuccess) return e;
  kern<<<grid, kThreads, smem, s>>>(tmap, args);
  return cudaGetLastError();
}

// Launchers, one per (operand type, activation word width, lane width), each
// compiled from conv_inst.cu in its own unit.
using LaunchFn = cudaError_t (*)(bool is_signed, const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid,
                                 size_t smem, cudaStream_t s);
#define SAMD_CONV_LAUNCHER(name) \
  cudaError_t name(bool is_signed, const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid, size_t smem, \
                   cudaStream_t s);
#define SAMD_CONV_LAUNCHERS(t, wb)                                                                          \
  SAMD_CONV_LAUNCHER(launch_conv_##t##_w##wb##_b1) SAMD_CONV_LAUNCHER(launch_conv_##t##_w##wb##_b2)        \
  SAMD_CONV_LAUNCHER(launch_conv_##t##_w##wb##_b3) SAMD_CONV_LAUNCHER(launch_conv_##t##_w##wb##_b4)        \
  SAMD_CONV_LAUNCHER(launch_conv_##t##_w##wb##_b5)
SAMD_CONV_LAUNCHERS(f16, 32)
SAMD_CONV_LAUNCHERS(f16, 64)
SAMD_CONV_LAUNCHERS(f8, 32)
SAMD_CONV_LAUNCHERS(f8, 64)
SAMD_CONV_LAUNCHER(launch_conv_f16_w32_b6)
SAMD_CONV_LAUNCHER(launch_conv_f16_w32_b7)
SAMD_CONV_LAUNCHER(launch_conv_f16_w32_b8)
SAMD_CONV_LAUNCHER(launch_conv_f16_w64_b6)
SAMD_CONV_LAUNCHER(launch_conv_f16_w64_b7)
SAMD_CONV_LAUNCHER(launch_conv_f16_w64_b8)
#undef SAMD_CONV_LAUNCHERS
#undef SAMD_CONV_LAUNCHER

}  // namespace conv
}  // namespace samd
