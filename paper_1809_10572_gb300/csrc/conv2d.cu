// conv2d.cu -- bit-precise convolution as an implicit GEMM on the tcgen05
// tensor cores.
//
// The paper's DNN convolution (section 7, Fig. 12, direct-sum2d) is
//   acc[n][k][ho][wo] = sum_{c,r,s} act[n][c][ho*st-p+r][wo*st-p+s] * wt[k][c][r][s].
// Here it is the GEMM D[M x K] = A[M x Kg] * B[K x Kg]^T with M = N*Ho*Wo
// output pixels and a reduction index Kg running over (tap, packed word,
// lane). The paper's own engine -- 1D convolution by one wide scalar
// multiply per packed word (section 5) -- is a CPU technique; on GB300 the
// dense contraction belongs on the tensor cores, and the packing still pays
// where the data moves: activations and weights stay packed in HBM and in
// L2, and are widened only in shared memory, right before the MMA (the
// "unpack to the native type" baseline of section 7, moved on-chip).
//
// Exactness. tcgen05 has no integer MMA on sm_103a, so lanes are widened to
// fp16, which holds every integer of [-128, 255] exactly; products are exact
// and the fp32 accumulators hold exact integers while every partial sum
// stays below 2^24. When R*S*C*max|a|*max|w| reaches 2^24 (wide weights over
// many taps), the weights are split into two 4-bit digits w = 16*hi + lo,
// stacked along the MMA's N: one MMA fills two accumulator halves, each far
// below 2^24, and the epilogue forms 16*hi + lo in int32.
//
// CTA = 6 warps, one 128-pixel tile x one block of output channels:
//   warp 0      TMEM allocation; lane 0 streams weight tiles with TMA
//   warp 1      lane 0 issues tcgen05.mma (128 x N x 16 per instruction)
//   warps 2-5   load packed activation words (implicit im2col, zero pad),
//               widen them to fp16 in the 128-byte-swizzled K-major layout,
//               then run the epilogue: tcgen05.ld of the fp32 accumulators,
//               int32 store and/or requantize-and-pack to fo.
// Weights are widened into a [K][Kg] fp16 matrix in the same Kg order by
// wprep_kernel: once per call (samd_conv2d), or once for many calls
// (samd_conv2d_prepare + samd_conv2d_prepared).
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <cstring>
#include <mutex>

#include "samd_internal.cuh"
#include "tc_ptx.cuh"

namespace samd {

// Sticky record of a bounded wait that ran out (SAMD_ETIMEOUT), per device.
__device__ int g_conv_status;

// Scratch of samd_conv2d_noalloc: the widened weights of one layer. Every GPU
// that loads the library holds these bytes until the process exits.
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

namespace {

constexpr int BM = 128;             // output pixels per tile = MMA M = TMEM lanes
constexpr int BK = 64;              // fp16 reduction elements per chunk = one 128-byte row
constexpr int kUnpackThreads = 128;
constexpr uint32_t kATileBytes = BM * BK * 2;
constexpr uint64_t kWaitLimitNs = 1000000000ull;  // 1 s
constexpr int kGatherDepth = 4;                    // packed chunks in flight per thread
constexpr int kUnpackWarps = 4;

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
  int N, C, H, W, K, R, S, stride, pad, Ho, Wo;
  long long M;
  int wpr;          // activation words per pixel
  int words_total;  // R * S * wpr: reduction length in packed words
  int nchunks;      // ceil(words_total / words per chunk)
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
  uint32_t tmem_cols;
  int out_bits, out_signed, out_lane_w, out_L, out_word64, out_wpr;
  int out_fast;     // output lanes per word when they divide 32 (packing in registers), else 0
  int shift;
  // halo mode (stride 1): virtual output grid of N x Hv x Wp positions
  int Hv, Wp, HR;   // HR halo rows per tile
  int nck;          // channel chunks per pixel (ceil(wpr / WC))
  int taps;         // R * S
  FastDiv fd_plane, fd_wp;  // halo: / (Hv * Wp), / Wp
  FastDiv fd_wo, fd_ho;     // output pixel index -> (n, oh, ow)
  FastDiv fd_gm;            // tile -> (channel block, position tile)
};

__device__ __forceinline__ uint32_t hsub2_bits(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Widening of one 64-position row of the A tile (one pixel, one chunk).
template <typename W, int BITS, bool SIGNED>
struct AUnpack {
  static constexpr int WB = WordTraits<W>::kBits;
  static constexpr int L = WB / BITS;
  static constexpr int WC = BK / L;        // packed words per chunk
  static constexpr int KUSED = WC * L;     // positions holding lanes; the rest are zero
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

  // Widen one pixel's chunk and store it as row `row` of a 128-byte
  // swizzled K-major tile: 16-byte block c goes to block c ^ (row % 8).
  __device__ static __forceinline__ void unpack_row(W (&w)[WC], uint8_t *tile, int row) {
    if constexpr (SIGNED) {
#pragma unroll
      for (int q = 0; q < WC; ++q) w[q] ^= sign_mask();
    }
    uint32_t h[32];
    pairs(w, h, std::make_integer_sequence<int, 32>{});
    uint8_t *rp = tile + row * 128;
    const int swz = row & 7;
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      *reinterpret_cast<uint4 *>(rp + ((c ^ swz) << 4)) = make_uint4(h[4 * c], h[4 * c + 1], h[4 * c + 2], h[4 * c + 3]);
    }
  }
};

// Bytes of one pixel-chunk row in the packed staging ring (a multiple of 16).
template <typename W, int WC>
struct Staging {
  static constexpr int kBytes = WC * static_cast<int>(sizeof(W));
  static constexpr int kRowBytes = (kBytes + 15) / 16 * 16;
  // widest cp.async that divides a whole chunk held by one pixel
  static constexpr int kVec = kBytes % 16 == 0 ? 16 : (kBytes % 8 == 0 ? 8 : static_cast<int>(sizeof(W)));
};

// Gathers the packed words of one pixel's chunk into shared memory with
// cp.async: word kw of the reduction is word (kw mod wpr) of the input pixel
// at tap kw / wpr; taps outside the image and words past the end are
// zero-filled (source size 0).
template <typename W, int WC>
struct AGather {
  const W *act;
  int H, W_, wpr, S, stride, pad, words_total;
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
    using St = Staging<W, WC>;
    const int kw0 = chunk * WC;
    int tap = kw0 / wpr, wi = kw0 - tap * wpr;
    bool valid;
    const W *px = pixel(tap, valid);
    if (vec) {
      const char *src = reinterpret_cast<const char *>(valid ? px + wi : act);
      const uint32_t nb = valid ? St::kVec : 0u;
#pragma unroll
      for (int v = 0; v < St::kBytes / St::kVec; ++v) {
        if constexpr (St::kVec == 16)
          ptx::cp_async_16(dst + 16 * v, src + 16 * v, nb);
        else if constexpr (St::kVec == 8)
          ptx::cp_async_8(dst + 8 * v, src + 8 * v, nb);
        else
          ptx::cp_async_4(dst + 4 * v, src + 4 * v, nb);
      }
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

// Epilogue of one accumulator row (one output pixel m) of channel block nb:
// fp32 accumulators -> exact int32 -> optional int32 store, optional
// requantize-and-pack. Called by whole warps (tcgen05.ld is collective);
// `ebuf` is idle operand memory of at least 128 x 260 bytes.
__device__ __forceinline__ void epilogue_row(const ConvArgs &args, uint32_t taddr, bool row_valid, long long m, int nb,
                                             uint8_t *ebuf, int row) {
      const int ch0 = nb * args.NBc;
      const int nvalid = args.K - ch0 < args.NBc ? args.K - ch0 : args.NBc;
      const bool vec_ok = (args.K % 4 == 0) && (ch0 % 4 == 0);
      const int lo = lane_lo(args.out_bits, args.out_signed), hi = lane_hi(args.out_bits, args.out_signed);
      const uint32_t omask = (1u << args.out_bits) - 1;
      // The requantized lane patterns of this row, one byte per channel, go to
      // shared memory first (the operand ring is idle once the accumulators
      // are complete). A row holds whole 32-channel groups plus 4 bytes: an
      // odd number of 32-bit words, so the warp's 4-byte stores fall in
      // distinct banks. 128 rows x (256 + 4) bytes fit in the ring.
      const int ebytes = (args.n_mma + 31) / 32 * 32 + 4;
      uint8_t *erow = ebuf + row * ebytes;
      for (int col = 0; col < nvalid; col += 32) {
        uint32_t r[32];
        int v[32];
        ptx::tmem_ld_32x32b_x32(taddr + col, r);
        ptx::tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = __float2int_rn(__uint_as_float(r[i]));
        if (args.split) {  // acc = 16 * hi + lo
          ptx::tmem_ld_32x32b_x32(taddr + args.n_mma + col, r);
          ptx::tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 16 * v[i] + __float2int_rn(__uint_as_float(r[i]));
        }
        if (!row_valid) continue;
        const int cnt = nvalid - col < 32 ? nvalid - col : 32;
        if (args.acc_out) {
          int32_t *dst = args.acc_out + m * args.K + ch0 + col;
          if (cnt == 32 && vec_ok) {
#pragma unroll
            for (int i = 0; i < 8; ++i)
              reinterpret_cast<int4 *>(dst)[i] = make_int4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (i < cnt) dst[i] = v[i];
          }
        }
        if (args.packed_out) {
          uint32_t y[32];
#pragma unroll
          for (int i = 0; i < 32; ++i)
            y[i] = i < cnt ? static_cast<uint32_t>(clamp_int(v[i] >> args.shift, lo, hi)) & omask : 0u;
          if (args.out_fast) {
            const long long w0 = m * args.out_wpr + (ch0 + col) / args.out_L;
            const int lw = args.out_lane_w;
            if (args.out_word64) {
              uint64_t *dst = static_cast<uint64_t *>(args.packed_out) + w0;
              switch (args.out_fast) {
                case 8: pack_regs<8>(y, lw, cnt, dst); break;
                case 16: pack_regs<16>(y, lw, cnt, dst); break;
                default: pack_regs<32>(y, lw, cnt, dst); break;
              }
            } else {
              uint32_t *dst = static_cast<uint32_t *>(args.packed_out) + w0;
              switch (args.out_fast) {
                case 4: pack_regs<4>(y, lw, cnt, dst); break;
                case 8: pack_regs<8>(y, lw, cnt, dst); break;
                case 16: pack_regs<16>(y, lw, cnt, dst); break;
                default: pack_regs<32>(y, lw, cnt, dst); break;
              }
            }
          } else {
#pragma unroll
            for (int i4 = 0; i4 < 8; ++i4)
              *reinterpret_cast<uint32_t *>(erow + col + 4 * i4) =
                  y[4 * i4] | (y[4 * i4 + 1] << 8) | (y[4 * i4 + 2] << 16) | (y[4 * i4 + 3] << 24);
          }
        }
      }
      // each output word packs L consecutive channels of this row
      if (row_valid && args.packed_out && !args.out_fast) {
        const int Lo = args.out_L, lw = args.out_lane_w;
        const int nwords = (nvalid + Lo - 1) / Lo;
        const long long w0 = m * args.out_wpr + ch0 / Lo;
        if (args.out_word64) {
          uint64_t *dst = static_cast<uint64_t *>(args.packed_out) + w0;
          for (int j = 0; j < nwords; ++j) {
            const int c0 = j * Lo, cn = nvalid - c0 < Lo ? nvalid - c0 : Lo;
            uint64_t wv = 0;
            for (int l = 0; l < cn; ++l) wv |= static_cast<uint64_t>(erow[c0 + l]) << (l * lw);
            dst[j] = wv;
          }
        } else {
          uint32_t *dst = static_cast<uint32_t *>(args.packed_out) + w0;
          for (int j = 0; j < nwords; ++j) {
            const int c0 = j * Lo, cn = nvalid - c0 < Lo ? nvalid - c0 : Lo;
            uint32_t wv = 0;
            for (int l = 0; l < cn; ++l) wv |= static_cast<uint32_t>(erow[c0 + l]) << (l * lw);
            dst[j] = wv;
          }
        }
      }
}

// ---- halo mode: each input pixel widened once per tile ----------------------
//
// Stride-1 convolutions. Output positions are numbered on a virtual grid of
// N x Hv x Wp (Hv = H + 2 pad rows and Wp = W + 2 pad columns per image);
// rows oh < Ho and columns ow < Wo of it are real outputs, the rest are
// computed and dropped. Position u of the same grid, read as an input, is
// pixel (u / Wp mod Hv - pad, u mod Wp - pad) of image u / (Hv Wp), zero
// outside the image. Output v at tap (r, s) reads input v + r Wp + s, a fixed
// shift, so a tile of 128 consecutive v needs the HR = 128 + (R-1) Wp + S - 1
// consecutive input rows from its first v. They are widened once into a
// 128-byte-swizzled fp16 halo; the MMAs of tap (r, s) read halo rows
// r Wp + s .. r Wp + s + 127 through a descriptor whose start address moves
// by (r Wp + s) x 128 bytes. The swizzle acts on absolute address bits, so
// any row may start a 128-row operand (base offset field 0).
// Reduction order: channel chunk j (WC packed words of a pixel), then tap,
// then the chunk's lane positions.
// Issues `ksteps` (1..4) MMAs of K = 16 as straight-line code: an issuing
// loop between them measurably slows the tensor core's intake.
__device__ __forceinline__ void mma_ksteps(int ksteps, uint32_t d, uint64_t a, uint64_t b, uint32_t idesc,
                                           uint32_t acc) {
  switch (ksteps) {
    case 4:
      ptx::mma_f16(d, a, b, idesc, acc);
      ptx::mma_f16(d, a + 2, b + 2, idesc, 1u);
      ptx::mma_f16(d, a + 4, b + 4, idesc, 1u);
      ptx::mma_f16(d, a + 6, b + 6, idesc, 1u);
      break;
    case 3:
      ptx::mma_f16(d, a, b, idesc, acc);
      ptx::mma_f16(d, a + 2, b + 2, idesc, 1u);
      ptx::mma_f16(d, a + 4, b + 4, idesc, 1u);
      break;
    case 2:
      ptx::mma_f16(d, a, b, idesc, acc);
      ptx::mma_f16(d, a + 2, b + 2, idesc, 1u);
      break;
    default:
      ptx::mma_f16(d, a, b, idesc, acc);
      break;
  }
}

// ---- the persistent convolution kernel ----------------------------------------
//
// One CTA per SM loops over output tiles (tile = blockIdx.x + i * gridDim.x;
// tile = nb * grid_m + mt: channel block nb, 128-position tile mt). Ten warps
// with fixed roles, connected by mbarrier rings:
//   warp 0      TMEM allocation; lane 0 streams weight tiles with TMA. When
//               the layer has one channel block and all its weight tiles fit,
//               they are loaded once and stay resident.
//   warp 1      lane 0 issues tcgen05.mma into one of two TMEM accumulators,
//               so tile i+1 accumulates while the epilogue drains tile i.
//   warps 2-5   operand producers.
//               HALO: for each (tile, channel chunk) the HR input rows the tile
//               needs are gathered with cp.async and widened once into one of
//               two fp16 halo buffers; every tap reads the halo through a
//               descriptor shifted by r*Wp + s rows (see the halo notes above).
//               GATHER: for each (tile, chunk) each thread gathers its pixel's
//               packed words (implicit im2col, zero padding) through a
//               cp.async ring and widens them into a ring of A tiles.
//   warps 6-9   epilogue: tcgen05.ld, exact int32, optional int32 store,
//               optional requantize-and-pack (warp w reads TMEM lanes of
//               quadrant w % 4).
// Every wait is bounded; a role that gives up records SAMD_ETIMEOUT and stops.
constexpr int kPThreads = 320;

template <typename W, int BITS, bool SIGNED, bool HALO>
__global__ void __launch_bounds__(kPThreads, 1) conv_persistent_kernel(const __grid_constant__ CUtensorMap tmap_b,
                                                                       const ConvArgs args) {
  using U = AUnpack<W, BITS, SIGNED>;
  constexpr int WC = U::WC;
  using St = Staging<W, WC>;
  extern __shared__ uint8_t smem_raw[];
  __shared__ int s_skip;
  __shared__ uint32_t s_aoff[256];  // HALO: byte offset of tap t's first halo row
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int STA = args.stages_a;  // GATHER: A tiles in flight
  const int STB = args.stages;    // weight tiles in flight (or resident)
  const bool resident = args.b_resident != 0;
  const uint32_t b_bytes = static_cast<uint32_t>(args.mma_n) * 128u;
  const uint32_t halo_bytes = static_cast<uint32_t>((args.HR + 7) / 8 * 8) * 128u;
  const uint32_t stage_g = static_cast<uint32_t>((args.HR * St::kRowBytes + 15) / 16 * 16);
  constexpr uint32_t kSlotBytes = BM * St::kRowBytes;  // GATHER staging slot

  // shared memory carve-up (the host sizes the same regions)
  uint8_t *sOp = smem;  // HALO: 2 halo buffers; GATHER: STA A tiles
  const uint32_t op_bytes = HALO ? 2 * halo_bytes : STA * kATileBytes;
  uint8_t *sB = sOp + op_bytes;
  uint8_t *sG = sB + STB * b_bytes;  // packed staging
  const uint32_t g_bytes = HALO ? 2 * stage_g : kGatherDepth * kSlotBytes;
  uint8_t *sE = sG + g_bytes;  // epilogue byte rows (only for output words the registers cannot pack)
  const uint32_t e_bytes = args.out_fast || !args.packed_out ? 0u
                                                             : static_cast<uint32_t>(BM * ((args.n_mma + 31) / 32 * 32 + 4));
  uint64_t *bars = reinterpret_cast<uint64_t *>(sE + (e_bytes + 15) / 16 * 16);
  // barriers: full_b[STB] empty_b[STB] opfull[NO] opempty[NO] accfull[2] accempty[2] drain
  const int NO = HALO ? 2 : STA;
  uint32_t *tmem_holder = reinterpret_cast<uint32_t *>(bars + 2 * STB + 2 * NO + 5);
  auto full_b = [&](int s) { return ptx::smem_addr(bars + s); };
  auto empty_b = [&](int s) { return ptx::smem_addr(bars + STB + s); };
  auto opfull = [&](int s) { return ptx::smem_addr(bars + 2 * STB + s); };
  auto opempty = [&](int s) { return ptx::smem_addr(bars + 2 * STB + NO + s); };
  auto accfull = [&](int a) { return ptx::smem_addr(bars + 2 * STB + 2 * NO + a); };
  auto accempty = [&](int a) { return ptx::smem_addr(bars + 2 * STB + 2 * NO + 2 + a); };
  const uint32_t drain_bar = ptx::smem_addr(bars + 2 * STB + 2 * NO + 4);

  volatile int *status = &g_conv_status;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) s_skip = *status;
  __syncthreads();
  if (s_skip) return;
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
      ptx::mbar_init(opfull(s), kUnpackWarps);
      ptx::mbar_init(opempty(s), 1);
    }
    for (int a = 0; a < 2; ++a) {
      ptx::mbar_init(accfull(a), 1);
      ptx::mbar_init(accempty(a), kUnpackWarps);  // the four epilogue warps
    }
    ptx::mbar_init(drain_bar, 1);
    ptx::fence_barrier_init();
    if (HALO)
      for (int t = 0; t < args.taps && t < 256; ++t)
        s_aoff[t] = static_cast<uint32_t>((t / args.S) * args.Wp + t % args.S) * 128u;
  }
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
      if (resident) {
        for (int c = 0; c < nchunks; ++c) {
          ptx::mbar_arrive_expect_tx(full_b(c), b_bytes);
          ptx::tma_load_2d(ptx::smem_addr(sB + c * b_bytes), &tmap_b, c * BK, 0, full_b(c));
        }
      } else {
        long long cb = 0, issued_from = 0;
        for (long long tile = first_tile; tile < total_tiles && ok; tile += tile_step) {
          const int nb = static_cast<int>(tile / args.grid_m);
          for (int c = 0; c < nchunks; ++c, ++cb) {
            const int s = static_cast<int>(cb % STB);
            const long long round = cb / STB;
            if (round > 0 && !ptx::mbar_wait_bounded(empty_b(s), static_cast<uint32_t>((round - 1) & 1), status,
                                                      kWaitLimitNs)) {
              ok = false;
              break;
            }
            ptx::mbar_arrive_expect_tx(full_b(s), b_bytes);
            ptx::tma_load_2d(ptx::smem_addr(sB + s * b_bytes), &tmap_b, c * BK, nb * args.mma_n, full_b(s));
          }
        }
        if (!ok) {  // leave no copy in flight: wait (bounded) for the last ring's worth
          for (long long k = (cb - STB > issued_from ? cb - STB : issued_from); k < cb; ++k)
            ptx::mbar_wait_bounded(full_b(static_cast<int>(k % STB)), static_cast<uint32_t>((k / STB) & 1), status,
                                   kWaitLimitNs / 10);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- MMA issue ----
      const uint32_t idesc = ptx::idesc_f16_f32(BM, args.mma_n);
      // Ring positions advance by increments (no division in this loop: the
      // issuing thread must keep ahead of the tensor core).
      int sb = 0, so = 0;
      uint32_t bpar = 0, opar = 0;
      bool b_ready = false;  // resident weights already observed
      const uint32_t sB_addr = ptx::smem_addr(sB), sOp_addr = ptx::smem_addr(sOp);
      const uint32_t op_stride = HALO ? halo_bytes : kATileBytes;
      const int nops = HALO ? args.nck : nchunks;  // operand stages per tile
      const int taps_here = HALO ? args.taps : 1;
      long long i = 0;
      for (long long tile = first_tile; tile < total_tiles && ok; tile += tile_step, ++i) {
        const int a = static_cast<int>(i & 1);
        if (i >= 2 && !ptx::mbar_wait_bounded(accempty(a), static_cast<uint32_t>(((i >> 1) - 1) & 1), status,
                                               kWaitLimitNs)) {
          ok = false;
          break;
        }
        ptx::tc_fence_after();  // the epilogue's reads of this accumulator are complete
        const uint32_t tmem_d = tmem_base + static_cast<uint32_t>(a * args.mma_n);
        uint32_t acc = 0;
        for (int j = 0; j < nops && ok; ++j) {
          if (!ptx::mbar_wait_bounded(opfull(so), opar, status, kWaitLimitNs)) {
            ok = false;
            break;
          }
          int words = (HALO ? args.wpr : args.words_total) - j * WC;
          if (words > WC) words = WC;
          const int ksteps = (words * U::L + 15) / 16;
          const uint32_t opbase = sOp_addr + so * op_stride;
          for (int t = 0; t < taps_here; ++t) {
            uint32_t baddr;
            if (resident) {
              const int c = HALO ? j * args.taps + t : j;
              if (!b_ready && !ptx::mbar_wait_bounded(full_b(c), 0, status, kWaitLimitNs)) {
                ok = false;
                break;
              }
              baddr = sB_addr + c * b_bytes;
            } else {
              if (!ptx::mbar_wait_bounded(full_b(sb), bpar, status, kWaitLimitNs)) {
                ok = false;
                break;
              }
              baddr = sB_addr + sb * b_bytes;
            }
            // No tcgen05 fence here: the operands arrived through the async
            // proxy (TMA, or stores fenced with fence.proxy.async before the
            // producers' arrive), which the mbarrier wait already orders.
            const uint64_t adesc = ptx::sw128_kmajor_desc(opbase + (HALO ? s_aoff[t] : 0u));
            const uint64_t bdesc = ptx::sw128_kmajor_desc(baddr);
            mma_ksteps(ksteps, tmem_d, adesc, bdesc, idesc, acc);
            acc = 1;
            if (!resident) {
              ptx::mma_commit(empty_b(sb));
              if (++sb == STB) {
                sb = 0;
                bpar ^= 1;
              }
            }
          }
          ptx::mma_commit(opempty(so));  // the operand stage is free once these MMAs complete
          if (++so == NO) {
            so = 0;
            opar ^= 1;
          }
        }
        if (ok) ptx::mma_commit(accfull(a));
        b_ready = true;
      }
      ptx::mma_commit(drain_bar);
      int quiet = 0;
      ptx::mbar_wait_bounded(drain_bar, 0, &quiet, kWaitLimitNs);
    }
  } else if (warp < 6) {
    // ---- operand producers ----
    const int t = threadIdx.x - 64;  // 0..127
    const W *act = static_cast<const W *>(args.act);
    if constexpr (HALO) {
      // items k = (tile i, channel chunk j), in the MMA's order
      auto gather = [&](long long tile, int j, int slot) {
        const uint32_t mt = static_cast<uint32_t>(tile) - fdiv(static_cast<uint32_t>(tile), args.fd_gm) * args.fd_gm.d;
        const uint32_t v0 = mt * BM;
        const uint32_t dst0 = ptx::smem_addr(sG + slot * stage_g);
        for (int hr = t; hr < args.HR; hr += kUnpackThreads) {
          const uint32_t u = v0 + hr;
          const uint32_t img = fdiv(u, args.fd_plane);
          const uint32_t rem = u - img * args.fd_plane.d;
          const uint32_t ihp = fdiv(rem, args.fd_wp);
          const int ih = static_cast<int>(ihp) - args.pad;
          const int iw = static_cast<int>(rem - ihp * args.fd_wp.d) - args.pad;
          const bool valid = static_cast<int>(img) < args.N && ih >= 0 && ih < args.H && iw >= 0 && iw < args.W;
          const W *px = act + ((static_cast<long long>(img) * args.H + ih) * args.W + iw) * args.wpr + j * WC;
          const uint32_t dst = dst0 + hr * St::kRowBytes;
          if (args.gather_vec) {
            const char *src = reinterpret_cast<const char *>(valid ? px : act);
            const uint32_t nbytes = valid ? St::kVec : 0u;
#pragma unroll
            for (int v = 0; v < St::kBytes / St::kVec; ++v) {
              if constexpr (St::kVec == 16)
                ptx::cp_async_16(dst + 16 * v, src + 16 * v, nbytes);
              else if constexpr (St::kVec == 8)
                ptx::cp_async_8(dst + 8 * v, src + 8 * v, nbytes);
              else
                ptx::cp_async_4(dst + 4 * v, src + 4 * v, nbytes);
            }
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
      // the sequence of items as (tile, j) pairs
      long long ntile = first_tile;
      int nj = 0;
      auto advance = [&](long long &tile, int &j) {
        if (++j == args.nck) {
          j = 0;
          tile += tile_step;
        }
      };
      if (ntile < total_tiles) gather(ntile, nj, 0);
      ptx::cp_async_commit();
      long long ctile = ntile;
      int cj = nj;
      advance(ntile, nj);
      for (long long k = 0; ctile < total_tiles; ++k) {
        if (ntile < total_tiles) gather(ntile, nj, static_cast<int>((k + 1) & 1));
        ptx::cp_async_commit();
        ptx::cp_async_wait<1>();  // item k of this thread's rows has landed
        const int hb = static_cast<int>(k & 1);
        if (k >= 2) {
          bool w_ok = true;
          if (lane == 0)
            w_ok = ptx::mbar_wait_bounded(opempty(hb), static_cast<uint32_t>(((k >> 1) - 1) & 1), status, kWaitLimitNs);
          if (!__shfl_sync(0xffffffffu, w_ok ? 1 : 0, 0)) {
            ok = false;
            break;
          }
        }
        const uint8_t *stg = sG + (k & 1) * stage_g;
        for (int hr = t; hr < args.HR; hr += kUnpackThreads) {
          W cur[WC];
          const uint8_t *src = stg + hr * St::kRowBytes;
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
          U::unpack_row(cur, sOp + hb * halo_bytes, hr);
        }
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(opfull(hb));
        (void)cj;
        ctile = ntile;
        cj = nj;
        advance(ntile, nj);
      }
      ptx::cp_async_wait<0>();
    } else {
      // GATHER: thread t owns row t of every A tile
      const int row = t;
      AGather<W, WC> g;
      g.act = act;
      g.H = args.H;
      g.W_ = args.W;
      g.wpr = args.wpr;
      g.S = args.S;
      g.stride = args.stride;
      g.pad = args.pad;
      g.words_total = args.words_total;
      g.vec = args.gather_vec != 0;
      auto set_tile = [&](long long tile) {
        const uint32_t tl = static_cast<uint32_t>(tile);
        const uint32_t mt = tl - fdiv(tl, args.fd_gm) * args.fd_gm.d;
        const uint32_t m = mt * BM + row;
        g.row_valid = m < static_cast<uint64_t>(args.M);
        const uint32_t mm = g.row_valid ? m : 0u;
        const uint32_t tq = fdiv(mm, args.fd_wo);
        g.ow = static_cast<int>(mm - tq * args.fd_wo.d);
        const uint32_t nq = fdiv(tq, args.fd_ho);
        g.oh = static_cast<int>(tq - nq * args.fd_ho.d);
        g.n = static_cast<int>(nq);
      };
      const uint32_t slot0 = ptx::smem_addr(sG) + row * St::kRowBytes;
      // issue side: item (itile, ic) kGatherDepth ahead of the consume side
      long long itile = first_tile;
      int ic = 0;
      if (itile < total_tiles) set_tile(itile);
      auto issue_next = [&](int slot) {
        if (itile < total_tiles) {
          g.issue(ic, slot0 + slot * kSlotBytes);
          if (++ic == nchunks) {
            ic = 0;
            itile += tile_step;
            if (itile < total_tiles) set_tile(itile);
          }
        }
        ptx::cp_async_commit();
      };
#pragma unroll 1
      for (int d = 0; d < kGatherDepth; ++d) issue_next(d);
      const long long items = ((total_tiles - first_tile + tile_step - 1) / tile_step) * nchunks;
      for (long long k = 0; k < items; ++k) {
        const int slot = static_cast<int>(k % kGatherDepth);
        ptx::cp_async_wait<kGatherDepth - 1>();
        W cur[WC];
        const uint8_t *src = sG + slot * kSlotBytes + row * St::kRowBytes;
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
        const int sa = static_cast<int>(k % NO);
        const long long round = k / NO;
        if (round > 0) {
          bool w_ok = true;
          if (lane == 0)
            w_ok = ptx::mbar_wait_bounded(opempty(sa), static_cast<uint32_t>((round - 1) & 1), status, kWaitLimitNs);
          if (!__shfl_sync(0xffffffffu, w_ok ? 1 : 0, 0)) {
            ok = false;
            break;
          }
        }
        U::unpack_row(cur, sOp + sa * kATileBytes, row);
        ptx::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(opfull(sa));
        issue_next(slot);  // refill the slot just read
      }
      ptx::cp_async_wait<0>();
    }
  } else {
    // ---- epilogue ----
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    long long i = 0;
    for (long long tile = first_tile; tile < total_tiles; tile += tile_step, ++i) {
      const int a = static_cast<int>(i & 1);
      bool w_ok = true;
      if (lane == 0) w_ok = ptx::mbar_wait_bounded(accfull(a), static_cast<uint32_t>((i >> 1) & 1), status, kWaitLimitNs);
      if (!__shfl_sync(0xffffffffu, w_ok ? 1 : 0, 0)) {
        ok = false;
        break;
      }
      ptx::tc_fence_after();
      const uint32_t tl = static_cast<uint32_t>(tile);
      const uint32_t nbu = fdiv(tl, args.fd_gm);
      const int nb = static_cast<int>(nbu);
      const uint32_t mt = tl - nbu * args.fd_gm.d;
      bool valid;
      long long m;
      if (HALO) {
        const uint32_t v = mt * BM + row;
        const uint32_t img = fdiv(v, args.fd_plane);
        const uint32_t rem = v - img * args.fd_plane.d;
        const uint32_t oh = fdiv(rem, args.fd_wp);
        const uint32_t ow = rem - oh * args.fd_wp.d;
        valid = static_cast<int>(img) < args.N && static_cast<int>(oh) < args.Ho && static_cast<int>(ow) < args.Wo;
        m = (static_cast<long long>(img) * args.Ho + oh) * args.Wo + ow;
      } else {
        m = static_cast<long long>(mt) * BM + row;
        valid = m < args.M;
      }
      const uint32_t taddr = tmem_base + static_cast<uint32_t>(a * args.mma_n) + (static_cast<uint32_t>(quad * 32) << 16);
      epilogue_row(args, taddr, valid, m, nb, sE, row);
      ptx::tc_fence_before();
      __syncwarp();
      if (lane == 0) ptx::mbar_arrive(accempty(a));
    }
  }

  ptx::tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    ptx::tc_fence_after();
    ptx::tmem_dealloc(tmem_base, args.tmem_cols);
  }
  if (!ok) atomicOr(const_cast<int *>(status), static_cast<int>(SAMD_ETIMEOUT));
}

// ---- weight widening into the workspace ----------------------------------

struct WPrepArgs {
  int K, C, RS;
  int bits_w, signed_w, lane_w_w, Lw, wpr_w;  // weight format
  int bits_a, La, WC, wpr_a, words_total;      // reduction order set by the activation format
  int Kpad, n_mma, mma_n, NBc, split;
  int halo, taps;  // halo: reduction order (chunk, tap, position); else (tap-major words, position)
  long long rows_total;
};

template <typename WW>
__global__ void __launch_bounds__(256) wprep_kernel(const WW *__restrict__ wt, __half *__restrict__ B,
                                                    const WPrepArgs a) {
  const long long total = a.rows_total * a.Kpad;
  const uint32_t mask = (1u << a.bits_w) - 1;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const long long rowi = idx / a.Kpad;
    const int kpos = static_cast<int>(idx - rowi * a.Kpad);
    const int nb = static_cast<int>(rowi / a.mma_n), rb = static_cast<int>(rowi % a.mma_n);
    const int plane = a.split ? rb / a.n_mma : -1;  // 0: high digit, 1: low digit
    const int r = a.split ? rb % a.n_mma : rb;
    const int k = nb * a.NBc + r;
    const int chunk = kpos / BK, j = kpos % BK;
    const int q = j / a.La, pos = j % a.La;
    int v = 0;
    if (r < a.NBc && k < a.K && q < a.WC) {
      int tap, wi, kw;
      if (a.halo) {  // chunk = (channel chunk, tap)
        tap = chunk % a.taps;
        wi = (chunk / a.taps) * a.WC + q;
        kw = wi < a.wpr_a ? 0 : a.words_total;  // past the pixel's last word: zero
      } else {
        kw = chunk * a.WC + q;
        tap = kw / a.wpr_a;
        wi = kw % a.wpr_a;
      }
      if (kw < a.words_total) {
        const int ch = wi * a.La + kpos_lane(a.bits_a, pos);
        if (ch < a.C) {
          const long long wrow = static_cast<long long>(k) * a.RS + tap;
          const WW word = wt[wrow * a.wpr_w + ch / a.Lw];
          const uint32_t p = static_cast<uint32_t>(word >> ((ch % a.Lw) * a.lane_w_w)) & mask;
          v = lane_value(p, a.bits_w, a.signed_w);
          if (plane == 0) v >>= 4;       // floor(v / 16)
          else if (plane == 1) v &= 15;  // v - 16 * floor(v / 16)
        }
      }
    }
    B[idx] = __int2half_rn(v);
  }
}

// ---- host side -------------------------------------------------------------

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

struct Plan {
  int wpr, words_total, La, WC, nchunks, Kpad, NBc, n_mma, mma_n, split, nblocks, stages, Ho, Wo, gather_vec;
  int halo, Hv, Wp, HR, nck, taps;  // halo mode (see conv_persistent_kernel)
  long long grid_m;                 // 128-position tiles along the output
  int stages_a, b_resident, ctas;
  long long M;
  uint32_t tmem_cols;
  size_t smem_bytes;
  size_t ws_bytes;
};

long long max_abs(samd_fmt f) { return f.is_signed ? (1LL << (f.bits - 1)) : ((1LL << f.bits) - 1); }

// Tiling, reduction order and exactness mode for one convolution. fo.bits == 0
// means no packed output. Returns SAMD_EUNSUP when no mode keeps every
// accumulator below 2^24.
samd_status make_plan(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo, Plan &p) {
  p.La = lanes_per_word(fa);
  if (p.La == 0) return SAMD_EINVAL;
  const long long taps = static_cast<long long>(d->R) * d->S * d->C;
  const long long bound = taps * max_abs(fa) * max_abs(fw);
  p.split = 0;
  if (bound >= (1LL << 24)) {
    // two 4-bit weight digits: each accumulator sums at most taps * max|a| * 16
    if (fw.bits <= 4 || taps * max_abs(fa) * 16 >= (1LL << 24)) return SAMD_EUNSUP;
    p.split = 1;
  }
  p.WC = BK / p.La;
  p.wpr = static_cast<int>((d->C + p.La - 1) / p.La);
  p.words_total = d->R * d->S * p.wpr;
  p.nchunks = (p.words_total + p.WC - 1) / p.WC;
  p.Kpad = p.nchunks * BK;
  p.Ho = (d->H + 2 * d->pad - d->R) / d->stride + 1;
  p.Wo = (d->W + 2 * d->pad - d->S) / d->stride + 1;
  p.M = static_cast<long long>(d->N) * p.Ho * p.Wo;
  // A channel block must cover whole output words so that no packed word is
  // shared by two CTAs.
  const int limit = p.split ? 128 : 256;
  if (d->K <= limit) {
    p.NBc = d->K;
  } else {
    const int Lo = fo.bits ? lanes_per_word(fo) : 1;
    p.NBc = (limit / Lo) * Lo;
  }
  p.n_mma = (p.NBc + 15) / 16 * 16;
  p.mma_n = p.split ? 2 * p.n_mma : p.n_mma;
  p.nblocks = (d->K + p.NBc - 1) / p.NBc;
  // ---- shared memory of the persistent kernel (same carve-up as the kernel)
  const int wb = fa.word_bits / 8;
  const int chunk_bytes = p.WC * wb;
  const int row_bytes = (chunk_bytes + 15) / 16 * 16;  // Staging::kRowBytes
  const int vec = chunk_bytes % 16 == 0 ? 16 : (chunk_bytes % 8 == 0 ? 8 : wb);
  p.gather_vec = (p.wpr % p.WC == 0) && ((static_cast<long long>(p.wpr) * wb) % vec == 0) ? 1 : 0;
  const size_t bst = static_cast<size_t>(p.mma_n) * 128;
  const bool fast_out = fo.bits != 0 && (fo.word_bits == 32 ? (32 % lanes_per_word(fo) == 0 && lanes_per_word(fo) >= 4)
                                                            : (32 % lanes_per_word(fo) == 0 && lanes_per_word(fo) >= 8));
  const size_t e_bytes = (fo.bits == 0 || fast_out) ? 0 : ((BM * ((p.n_mma + 31) / 32 * 32 + 4) + 15) / 16 * 16);
  const size_t kBudget = 224 * 1024;  // below the 227 KB opt-in limit minus static shared memory
  const size_t extra = 1024 + e_bytes + 512;  // alignment slack, epilogue rows, barriers
  p.grid_m = (p.M + BM - 1) / BM;
  p.taps = d->R * d->S;
  p.nck = (p.wpr + p.WC - 1) / p.WC;
  p.Hv = d->H + 2 * d->pad;
  p.Wp = d->W + 2 * d->pad;
  p.HR = BM + (d->R - 1) * p.Wp + (d->S - 1);
  p.halo = 0;
  p.b_resident = 0;
  p.stages_a = 0;
  // Halo mode: stride 1, several taps, little padded-grid waste, halo fits.
  if (d->stride == 1 && p.taps >= 2 && p.M > 0 && p.HR <= 640) {
    const double waste = static_cast<double>(d->N) * p.Hv * p.Wp / static_cast<double>(p.M);
    const size_t halo_bytes = static_cast<size_t>((p.HR + 7) / 8 * 8) * 128;
    const size_t stage_g = static_cast<size_t>((p.HR * row_bytes + 15) / 16 * 16);
    const size_t fixed = extra + 2 * halo_bytes + 2 * stage_g;
    const int ntiles_b = p.nck * p.taps;
    if (waste <= 1.16 && fixed + 2 * bst <= kBudget) {
      p.halo = 1;
      p.nchunks = ntiles_b;
      p.Kpad = ntiles_b * BK;
      p.grid_m = (static_cast<long long>(d->N) * p.Hv * p.Wp + BM - 1) / BM;
      if (p.nblocks == 1 && fixed + ntiles_b * bst <= kBudget) {
        p.b_resident = 1;
        p.stages = ntiles_b;
      } else {
        long long st = static_cast<long long>((kBudget - fixed) / bst);
        p.stages = static_cast<int>(st > 8 ? 8 : st);
      }
      p.smem_bytes = fixed + p.stages * bst;
    }
  }
  if (!p.halo) {
    const size_t staging = static_cast<size_t>(kGatherDepth) * BM * row_bytes;
    for (int sta = 4; sta >= 2; --sta) {
      const size_t fixed = extra + sta * static_cast<size_t>(kATileBytes) + staging;
      if (fixed + 2 * bst > kBudget) continue;
      p.stages_a = sta;
      if (p.nblocks == 1 && fixed + p.nchunks * bst <= kBudget) {
        p.b_resident = 1;
        p.stages = p.nchunks;
      } else {
        long long st = static_cast<long long>((kBudget - fixed) / bst);
        p.stages = static_cast<int>(st > 8 ? 8 : st);
      }
      p.smem_bytes = fixed + p.stages * bst;
      break;
    }
    if (p.stages_a == 0) return SAMD_EUNSUP;  // operand tiles do not fit (not reached for N <= 256)
  }
  uint32_t cols = 32;
  while (cols < static_cast<uint32_t>(2 * p.mma_n)) cols <<= 1;  // two accumulators
  p.tmem_cols = cols;
  p.ws_bytes = static_cast<size_t>(p.nblocks) * p.mma_n * p.Kpad * sizeof(__half);
  return SAMD_OK;
}

// cudaFuncSetAttribute once per (kernel, device), so that launches made
// while a stream is being captured into a graph issue no other CUDA call.
// The dynamic limit is the per-block maximum minus the kernel's static
// shared memory. Returns cudaErrorInvalidValue if `smem` does not fit.
cudaError_t ensure_smem_attr(const void *kern, size_t smem) {
  static std::mutex mu;
  static const void *done_fn[256];
  static int done_dev[256];
  static size_t done_smem[256];
  static int n_done = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < n_done; ++i)
    if (done_fn[i] == kern && done_dev[i] == dev) return smem <= done_smem[i] ? cudaSuccess : cudaErrorInvalidValue;
  int optin = 0;
  e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  cudaFuncAttributes fa;
  e = cudaFuncGetAttributes(&fa, kern);
  if (e != cudaSuccess) return e;
  const size_t limit = static_cast<size_t>(optin) - fa.sharedSizeBytes;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(limit));
  if (e != cudaSuccess) return e;
  if (n_done < 256) {
    done_fn[n_done] = kern;
    done_dev[n_done] = dev;
    done_smem[n_done] = limit;
    ++n_done;
  }
  return smem <= limit ? cudaSuccess : cudaErrorInvalidValue;
}

template <typename W, int BITS, bool SIGNED>
cudaError_t launch_conv_variant(const CUtensorMap &tmap, const ConvArgs &args, dim3 grid, size_t smem,
                                cudaStream_t s) {
  auto kern = args.HR > 0 ? conv_persistent_kernel<W, BITS, SIGNED, true> : conv_persistent_kernel<W, BITS, SIGNED, false>;
  cudaError_t e = ensure_smem_attr(reinterpret_cast<const void *>(kern), smem);
  if (e != cudaSuccess) return e;
  kern<<<grid, kPThreads, smem, s>>>(tmap, args);
  return cudaGetLastError();
}

template <typename W>
cudaError_t launch_conv_word(samd_fmt fa, const CUtensorMap &tmap, const ConvArgs &args, dim3 grid, size_t smem,
                             cudaStream_t s) {
  switch (fa.bits * 2 + (fa.is_signed ? 1 : 0)) {
#define SAMD_CONV_CASE(B)                                                              \
  case 2 * B:                                                                          \
    return launch_conv_variant<W, B, false>(tmap, args, grid, smem, s);                \
  case 2 * B + 1:                                                                      \
    return launch_conv_variant<W, B, true>(tmap, args, grid, smem, s);
    SAMD_CONV_CASE(1) SAMD_CONV_CASE(2) SAMD_CONV_CASE(3) SAMD_CONV_CASE(4)
    SAMD_CONV_CASE(5) SAMD_CONV_CASE(6) SAMD_CONV_CASE(7) SAMD_CONV_CASE(8)
#undef SAMD_CONV_CASE
    default:
      return cudaErrorInvalidValue;
  }
}

samd_fmt none_fmt() { return samd_fmt{0, 0, 0, 0}; }

}  // namespace

size_t conv2d_workspace_size(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw) {
  // the channel blocking depends on the output format only above 128/256
  // channels: report the largest size over every output format
  Plan p;
  if (make_plan(d, fa, fw, none_fmt(), p) != SAMD_OK) return 0;
  size_t best = p.ws_bytes;
  for (int wb : {32, 64})
    for (int bits = 1; bits <= 8; ++bits)
      for (int sp = 0; sp + bits <= 16 && sp <= 8; ++sp) {
        samd_fmt fo{static_cast<uint8_t>(bits), 0, static_cast<uint8_t>(sp), static_cast<uint8_t>(wb)};
        Plan q;
        if (make_plan(d, fa, fw, fo, q) == SAMD_OK && q.ws_bytes > best) best = q.ws_bytes;
      }
  return best;
}

samd_status conv2d_check(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw) {
  Plan p;
  return make_plan(d, fa, fw, none_fmt(), p);
}

samd_status conv2d_prepare(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, const void *wt, samd_fmt fo,
                           void *prepared, size_t prepared_bytes, cudaStream_t s) {
  Plan p;
  samd_status st = make_plan(d, fa, fw, fo, p);
  if (st != SAMD_OK) return st;
  if (prepared_bytes < p.ws_bytes) return SAMD_ESHAPE;
  WPrepArgs wa;
  wa.K = d->K;
  wa.C = d->C;
  wa.RS = d->R * d->S;
  wa.bits_w = fw.bits;
  wa.signed_w = fw.is_signed;
  wa.lane_w_w = fw.bits + fw.spacer;
  wa.Lw = lanes_per_word(fw);
  wa.wpr_w = static_cast<int>(words_per_row(fw, d->C));
  wa.bits_a = fa.bits;
  wa.La = p.La;
  wa.WC = p.WC;
  wa.wpr_a = p.wpr;
  wa.words_total = p.words_total;
  wa.Kpad = p.Kpad;
  wa.n_mma = p.n_mma;
  wa.mma_n = p.mma_n;
  wa.NBc = p.NBc;
  wa.split = p.split;
  wa.halo = p.halo;
  wa.taps = p.taps;
  wa.rows_total = static_cast<long long>(p.nblocks) * p.mma_n;
  const long long total = wa.rows_total * wa.Kpad;
  const int grid = grid_for(total, 256, sm_count() * 8);
  __half *B = static_cast<__half *>(prepared);
  if (fw.word_bits == 32)
    wprep_kernel<uint32_t><<<grid, 256, 0, s>>>(static_cast<const uint32_t *>(wt), B, wa);
  else
    wprep_kernel<uint64_t><<<grid, 256, 0, s>>>(static_cast<const uint64_t *>(wt), B, wa);
  return cudaGetLastError() == cudaSuccess ? SAMD_OK : SAMD_ECUDA;
}

samd_status conv2d_run(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, const void *act, const void *prepared,
                       size_t prepared_bytes, int32_t *acc_out, samd_fmt fo, void *packed_out, int shift,
                       cudaStream_t s) {
  Plan p;
  samd_status st = make_plan(d, fa, fw, fo, p);
  if (st != SAMD_OK) return st;
  if (prepared_bytes < p.ws_bytes) return SAMD_ESHAPE;
  if (p.M == 0) return SAMD_OK;
  EncodeTiledFn enc = encode_tiled();
  if (!enc) return SAMD_ECUDA;

  // tensor map over the widened weights: [nblocks * mma_n][Kpad] fp16, tiles
  // of mma_n rows x 64 elements, 128-byte swizzle
  CUtensorMap tmap;
  const long long rows_total = static_cast<long long>(p.nblocks) * p.mma_n;
  cuuint64_t gdim[2] = {static_cast<cuuint64_t>(p.Kpad), static_cast<cuuint64_t>(rows_total)};
  cuuint64_t gstride[1] = {static_cast<cuuint64_t>(p.Kpad) * sizeof(__half)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(p.mma_n)};
  cuuint32_t estride[2] = {1, 1};
  CUresult cr = enc(&tmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void *>(prepared), gdim, gstride, box,
                    estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return SAMD_ECUDA;

  ConvArgs a;
  a.act = act;
  a.acc_out = acc_out;
  a.packed_out = packed_out;
  a.N = d->N;
  a.C = d->C;
  a.H = d->H;
  a.W = d->W;
  a.K = d->K;
  a.R = d->R;
  a.S = d->S;
  a.stride = d->stride;
  a.pad = d->pad;
  a.Ho = p.Ho;
  a.Wo = p.Wo;
  a.M = p.M;
  a.wpr = p.wpr;
  a.words_total = p.words_total;
  a.nchunks = p.nchunks;
  a.NBc = p.NBc;
  a.n_mma = p.n_mma;
  a.mma_n = p.mma_n;
  a.split = p.split;
  a.stages = p.stages;
  a.stages_a = p.stages_a;
  a.b_resident = p.b_resident;
  a.grid_m = p.grid_m;
  a.nblocks = p.nblocks;
  a.gather_vec = p.gather_vec;
  a.tmem_cols = p.tmem_cols;
  a.out_bits = packed_out ? fo.bits : 8;
  a.out_signed = packed_out ? fo.is_signed : 1;
  a.out_lane_w = packed_out ? fo.bits + fo.spacer : 8;
  a.out_L = packed_out ? lanes_per_word(fo) : 1;
  a.out_word64 = packed_out ? (fo.word_bits == 64) : 0;
  a.out_wpr = packed_out ? static_cast<int>(words_per_row(fo, d->K)) : 0;
  {
    const int Lo = a.out_L;
    const bool fast = packed_out && (fo.word_bits == 32 ? (Lo == 4 || Lo == 8 || Lo == 16 || Lo == 32)
                                                        : (Lo == 8 || Lo == 16 || Lo == 32));
    a.out_fast = fast ? Lo : 0;
  }
  a.shift = shift;
  a.Hv = p.Hv;
  a.Wp = p.Wp;
  a.HR = p.halo ? p.HR : 0;  // 0 selects the gather kernel
  a.nck = p.nck;
  a.taps = p.taps;
  // the kernel's index math runs in 32 bits
  if (static_cast<long long>(d->N) * p.Hv * p.Wp + p.HR + BM >= (1LL << 31) || p.M >= (1LL << 31) ||
      p.grid_m * p.nblocks >= (1LL << 31))
    return SAMD_EUNSUP;
  a.fd_plane = make_fastdiv(static_cast<uint32_t>(p.Hv * p.Wp));
  a.fd_wp = make_fastdiv(static_cast<uint32_t>(p.Wp));
  a.fd_wo = make_fastdiv(static_cast<uint32_t>(p.Wo));
  a.fd_ho = make_fastdiv(static_cast<uint32_t>(p.Ho));
  a.fd_gm = make_fastdiv(static_cast<uint32_t>(p.grid_m));
  const long long total_tiles = p.grid_m * p.nblocks;
  long long ctas = sm_count();
  if (ctas > total_tiles) ctas = total_tiles;
  dim3 grid(static_cast<unsigned>(ctas));
  cudaError_t e = fa.word_bits == 32 ? launch_conv_word<uint32_t>(fa, tmap, a, grid, p.smem_bytes, s)
                                     : launch_conv_word<uint64_t>(fa, tmap, a, grid, p.smem_bytes, s);
  return e == cudaSuccess ? SAMD_OK : SAMD_ECUDA;
}

samd_status conv2d_nhwc(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                        int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, void *workspace,
                        size_t workspace_bytes, cudaStream_t s) {
  const samd_fmt fplan = packed_out ? fo : none_fmt();
  samd_status st = conv2d_prepare(d, fa, fw, wt, fplan, workspace, workspace_bytes, s);
  if (st != SAMD_OK) return st;
  return conv2d_run(d, fa, fw, act, workspace, workspace_bytes, acc_out, fplan, packed_out, shift, s);
}

namespace {
// Device address of g_noalloc_scratch for each device, looked up once with
// that device current (the symbol's host-side name is not a device address).
std::mutex g_scratch_mu;
void *g_scratch_ptr[64] = {nullptr};

cudaError_t noalloc_scratch(void **ptr) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_ptr[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_ptr[dev] = p;
  }
  *ptr = g_scratch_ptr[dev];
  return cudaSuccess;
}
}  // namespace

samd_status conv2d_nhwc_noalloc(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                                int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, cudaStream_t s) {
  Plan p;
  samd_status st = make_plan(d, fa, fw, packed_out ? fo : none_fmt(), p);
  if (st != SAMD_OK) return st;
  if (p.ws_bytes > kNoallocScratchBytes) return SAMD_EUNSUP;  // the layer's weights do not fit the static scratch
  void *scratch = nullptr;
  if (noalloc_scratch(&scratch) != cudaSuccess) return SAMD_ECUDA;
  // prepare writes every byte of the widened weights that run then reads, so
  // nothing left over from an earlier call is ever used
  return conv2d_nhwc(d, fa, act, fw, wt, acc_out, fo, packed_out, shift, scratch, kNoallocScratchBytes, s);
}

cudaError_t read_device_status(int *status, int reset, cudaStream_t s) {
  int v = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_conv_status, sizeof(int), 0, cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return e;
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return e;
  *status = v;
  if (reset && v != 0) {
    int zero = 0;
    e = cudaMemcpyToSymbolAsync(g_conv_status, &zero, sizeof(int), 0, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  }
  return e;
}

}  // namespace samd
