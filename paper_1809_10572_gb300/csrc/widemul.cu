// widemul.cu -- the convolution of NCHW tensors packed along W by the
// paper's own engine (section 5.1): every 1D sub-convolution of Fig. 12 (the
// x-loop over a row of the image against a row of the kernel) is one wide
// integer multiply of two packed words. Lanes are placed in fields of F bits,
// wide enough that no sum of products can overflow into the next field, so
// the 128-bit product of a word of nx inputs and a word of the S kernel taps
// holds nx + S - 1 coefficients of the polynomial product. Signed lanes are
// sign-extended through their fields (Fig. 10); the borrow a negative lane
// leaves in the field above is repaired when coefficients are read (Fig. 11).
//
// This runs on the CUDA cores (64 x 64 -> 128-bit multiplies, which the GPU
// builds from 32-bit multiply-adds); it is the paper's engine kept as a
// comparison point next to the tensor-core path of conv_kernel.cuh, and the
// path for the NCHW layout.
//
// Plan (host): bound = R*S*C*max|a|*max|w| (no partial or final sum exceeds
// it), F = bits(bound) + 1, nx = floor(64 / F) input positions per word,
// S*F <= 64 (the kernel row is one word), stride 1.
//
// Buffers (the caller's workspace):
//   X[n][c][h][g]  int64: the inputs xs[g*nx .. g*nx + nx) of row (n, c, h),
//                  xs[p] = act[p - pad] (zero outside the row), one per F-bit
//                  field, as the integer sum_i xs[g*nx + i] * 2^(F*i);
//   KR[m][c][r]    int64: the kernel row reversed, sum_t wt[m][c][r][S-1-t] * 2^(F*t).
// The full convolution z[q] = sum_t xs[q - t] * kr[t] gives the output
// y[j] = z[j + S - 1] (cross-correlation with padding, as in Fig. 12).
#include "samd_internal.cuh"

namespace samd {
namespace wm {

struct Geometry {
  int F, nx, G, Ho, Wo;
  long long bound;
};

int bit_length(long long v) {
  int b = 0;
  while (v >> b) ++b;
  return b;
}

long long max_abs(samd_fmt f) { return f.is_signed ? (1LL << (f.bits - 1)) : ((1LL << f.bits) - 1); }

samd_status plan(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, Geometry &g) {
  if (d->stride != 1) return SAMD_EUNSUP;  // a polynomial product slides by one position
  g.bound = static_cast<long long>(d->R) * d->S * d->C * max_abs(fa) * max_abs(fw);
  if (g.bound >= (1LL << 31)) return SAMD_EUNSUP;  // int32 results
  g.F = bit_length(g.bound) + 1;                   // |z| <= bound < 2^(F-1)
  const int wider = fa.bits > fw.bits ? fa.bits : fw.bits;
  if (g.F < wider + 1) g.F = wider + 1;            // a field holds a lane and its sign extension
  if (d->S * g.F > 64) return SAMD_EUNSUP;         // the kernel row is one 64-bit word
  g.nx = 64 / g.F;                                 // >= S >= S - 1: a segment's carries reach only the next one
  g.Ho = d->H + 2 * d->pad - d->R + 1;
  g.Wo = d->W + 2 * d->pad - d->S + 1;
  g.G = (g.Wo + d->S - 1 + g.nx - 1) / g.nx;
  return SAMD_OK;
}

size_t x_words(const samd_conv_desc *d, const Geometry &g) {
  return static_cast<size_t>(d->N) * d->C * d->H * g.G;
}

size_t workspace_bytes(const samd_conv_desc *d, const Geometry &g) {
  return 8 * (x_words(d, g) + static_cast<size_t>(d->K) * d->C * d->R);
}

// Lane p of a packed row (pattern in the low `bits` bits).
template <typename W>
__device__ __forceinline__ uint64_t row_lane(const W *row, int p, int L, int bits) {
  const W w = row[p / L];
  return static_cast<uint64_t>(w >> ((p % L) * bits)) & ((1ull << bits) - 1);
}

// Fig. 10: each lane's sign bit, moved one place up, is subtracted from the
// word; a negative lane's pattern v + 2^bits becomes v and the borrow runs
// through the field into the lane above, so the word equals sum_i v_i 2^(F i).
__device__ __forceinline__ uint64_t sign_extend4mul(uint64_t word, uint64_t sign_bits) {
  return word - ((word & sign_bits) << 1);
}

struct PrepArgs {
  int rows, G, nx, F, bits, is_signed, L, len, wpr, pad, reverse;
  uint64_t sign_bits;  // bit F*i + bits - 1 of every field
};

// One word per (row, segment g): fields i < nx hold row position
// g*nx + i - pad (X), or, with `reverse`, kernel tap len - 1 - i (KR, G = 1).
template <typename W>
__global__ void __launch_bounds__(256) wm_prep_kernel(const W *__restrict__ src, int64_t *__restrict__ dst,
                                                      const PrepArgs a) {
  const long long total = static_cast<long long>(a.rows) * a.G;
  for (long long t = blockIdx.x * (long long)blockDim.x + threadIdx.x; t < total;
       t += (long long)gridDim.x * blockDim.x) {
    const long long row = t / a.G;
    const int g = static_cast<int>(t - row * a.G);
    const W *r = src + row * a.wpr;
    uint64_t word = 0;
    for (int i = 0; i < a.nx; ++i) {
      const int p = a.reverse ? a.len - 1 - i : g * a.nx + i - a.pad;
      if (p >= 0 && p < a.len) word |= row_lane<W>(r, p, a.L, a.bits) << (a.F * i);
    }
    if (a.is_signed) word = sign_extend4mul(word, a.sign_bits);
    dst[t] = static_cast<int64_t>(word);
  }
}

struct ConvArgs {
  const int64_t *X, *KR;
  int32_t *acc_out;
  void *packed_out;
  int N, C, H, K, R, S, pad, Ho, Wo, G, F, nx;
  uint64_t msb_lo, msb_hi;  // the top bit of every F-bit field of a 128-bit value
  int out_bits, out_signed, out_lane_w, out_L, out_wpr, out_word64, shift;
  int row_bytes;            // bytes of the per-warp row buffer (>= Wo)
};

// Fig. 11: adding each field's top bit to itself carries +1 into the field
// above wherever the field reads negative (repaying the borrow that lane took
// from it); xoring the top bits back restores the fields' own top bits. Every
// field then holds its coefficient as F-bit two's complement.
__device__ __forceinline__ unsigned __int128 repair(unsigned __int128 v, unsigned __int128 msb) {
  const unsigned __int128 s = v & msb;
  return (v + s) ^ s;
}

__device__ __forceinline__ int field(unsigned __int128 r, int i, int F) {
  const int64_t f = static_cast<int64_t>(static_cast<uint64_t>(r >> (F * i)));
  return static_cast<int>((f << (64 - F)) >> (64 - F));  // sign-extended from F bits
}

constexpr int kWarps = 4;

// One warp per output row (n, m, ho). The row's segments are taken 31 at a
// time: lane l of chunk k sums, over channels and kernel rows, the products
// of segment g = 31 k + l - 1; lane l >= 1 then adds the part of segment
// g - 1's sum (its lane l - 1 neighbour) that reaches into its own fields
// and reads nx finished coefficients.
template <typename WO>
__global__ void __launch_bounds__(32 * kWarps) wm_conv_kernel(const ConvArgs a) {
  extern __shared__ uint8_t row_buf[];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long row_id = static_cast<long long>(blockIdx.x) * kWarps + warp;  // (n * K + m) * Ho + ho
  const long long rows = static_cast<long long>(a.N) * a.K * a.Ho;
  if (row_id >= rows) return;  // whole warps
  const int ho = static_cast<int>(row_id % a.Ho);
  const long long nm = row_id / a.Ho;
  const int m = static_cast<int>(nm % a.K), n = static_cast<int>(nm / a.K);
  const unsigned __int128 msb = (static_cast<unsigned __int128>(a.msb_hi) << 64) | a.msb_lo;
  uint8_t *q8 = row_buf + warp * a.row_bytes;
  const int lo = lane_lo(a.out_bits, a.out_signed), hi = lane_hi(a.out_bits, a.out_signed);
  const uint32_t omask = (1u << a.out_bits) - 1;
  const int shift_nx = a.F * a.nx;
  for (int chunk = 0; chunk * 31 < a.G; ++chunk) {
    const int g = chunk * 31 + lane - 1;
    unsigned __int128 acc = 0;
    if (g >= 0 && g < a.G) {
      for (int c = 0; c < a.C; ++c) {
        const int64_t *xc = a.X + (static_cast<long long>(n) * a.C + c) * a.H * a.G + g;
        const int64_t *kc = a.KR + (static_cast<long long>(m) * a.C + c) * a.R;
        for (int r = 0; r < a.R; ++r) {
          const int h = ho + r - a.pad;
          if (h < 0 || h >= a.H) continue;
          // section 5.1: one signed 64 x 64 -> 128-bit multiply is the 1D
          // convolution of nx inputs with the S taps
          acc += static_cast<unsigned __int128>(static_cast<__int128>(__ldg(xc + static_cast<long long>(h) * a.G)) *
                                                static_cast<__int128>(__ldg(kc + r)));
        }
      }
    }
    // the neighbour's sum: segment g - 1
    const uint64_t plo = __shfl_up_sync(0xffffffffu, static_cast<uint64_t>(acc), 1);
    const uint64_t phi = __shfl_up_sync(0xffffffffu, static_cast<uint64_t>(acc >> 64), 1);
    if (lane == 0 || g >= a.G) continue;
    const unsigned __int128 prev = (static_cast<unsigned __int128>(phi) << 64) | plo;
    // its fields nx .. nx + S - 2 belong to this segment: subtract its own
    // nx coefficients and shift the rest down (exact: the difference is a
    // multiple of 2^(F nx))
    const unsigned __int128 rp = repair(prev, msb);
    __int128 low = 0;
    for (int i = a.nx - 1; i >= 0; --i) low = low * (static_cast<__int128>(1) << a.F) + field(rp, i, a.F);
    const __int128 carry_in = (static_cast<__int128>(prev) - low) >> shift_nx;
    const unsigned __int128 r = repair(acc + static_cast<unsigned __int128>(carry_in), msb);
    for (int i = 0; i < a.nx; ++i) {
      const int j = g * a.nx + i - (a.S - 1);
      if (j < 0 || j >= a.Wo) continue;
      const int z = field(r, i, a.F);
      if (a.acc_out) a.acc_out[row_id * a.Wo + j] = z;
      if (a.packed_out) q8[j] = static_cast<uint8_t>(static_cast<uint32_t>(clamp_int(z >> a.shift, lo, hi)) & omask);
    }
  }
  if (!a.packed_out) return;
  __syncwarp();
  // the requantized row, packed along W in words of out_L lanes
  WO *dst = static_cast<WO *>(a.packed_out) + row_id * a.out_wpr;
  for (int w = lane; w < a.out_wpr; w += 32) {
    WO word = 0;
    for (int l = 0; l < a.out_L; ++l) {
      const int j = w * a.out_L + l;
      if (j < a.Wo) word |= static_cast<WO>(q8[j]) << (l * a.out_lane_w);
    }
    dst[w] = word;
  }
}

uint64_t field_bits(int F, int nfields, int bit, int word_bits, bool high_half) {
  uint64_t m = 0;
  for (int i = 0; i < nfields; ++i) {
    const int b = F * i + bit;
    if (b >= word_bits) break;
    if (!high_half && b < 64) m |= 1ull << b;
    if (high_half && b >= 64) m |= 1ull << (b - 64);
  }
  return m;
}

template <typename W>
cudaError_t launch_prep(const void *src, int64_t *dst, const PrepArgs &a, cudaStream_t s) {
  const long long total = static_cast<long long>(a.rows) * a.G;
  const int grid = grid_for(total, 256, sm_count() * 8);
  wm_prep_kernel<W><<<grid, 256, 0, s>>>(static_cast<const W *>(src), dst, a);
  return cudaGetLastError();
}

}  // namespace wm

samd_status conv2d_nchw_check(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo, size_t *ws_bytes) {
  wm::Geometry g;
  const samd_status st = wm::plan(d, fa, fw, g);
  if (st != SAMD_OK) return st;
  if (fo.bits != 0 && static_cast<size_t>(g.Wo) * wm::kWarps > 48 * 1024) return SAMD_EUNSUP;  // row buffers
  if (ws_bytes) *ws_bytes = wm::workspace_bytes(d, g);
  return SAMD_OK;
}

samd_status conv2d_nchw(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                        int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, void *workspace,
                        size_t workspace_bytes, cudaStream_t s) {
  using namespace wm;
  Geometry g;
  samd_status st = plan(d, fa, fw, g);
  if (st != SAMD_OK) return st;
  if (workspace_bytes < wm::workspace_bytes(d, g)) return SAMD_ESHAPE;
  if (packed_out && static_cast<size_t>(g.Wo) * kWarps > 48 * 1024) return SAMD_EUNSUP;  // row buffers
  const long long rows = static_cast<long long>(d->N) * d->K * g.Ho;
  if (rows == 0) return SAMD_OK;
  if ((rows + kWarps - 1) / kWarps >= (1LL << 31)) return SAMD_EUNSUP;
  int64_t *X = static_cast<int64_t *>(workspace);
  int64_t *KR = X + x_words(d, g);

  PrepArgs pa;
  pa.nx = g.nx;
  pa.F = g.F;
  // activations: rows (n, c, h) of W lanes
  pa.rows = d->N * d->C * d->H;
  pa.G = g.G;
  pa.bits = fa.bits;
  pa.is_signed = fa.is_signed;
  pa.L = lanes_per_word(fa);
  pa.len = d->W;
  pa.wpr = static_cast<int>(words_per_row(fa, d->W));
  pa.pad = d->pad;
  pa.reverse = 0;
  pa.sign_bits = field_bits(g.F, g.nx, fa.bits - 1, 64, false);
  cudaError_t e = fa.word_bits == 32 ? launch_prep<uint32_t>(act, X, pa, s) : launch_prep<uint64_t>(act, X, pa, s);
  if (e != cudaSuccess) return SAMD_ECUDA;
  // weights: rows (m, c, r) of S lanes, reversed into one word each
  PrepArgs pk = pa;
  pk.rows = d->K * d->C * d->R;
  pk.G = 1;
  pk.nx = d->S;
  pk.bits = fw.bits;
  pk.is_signed = fw.is_signed;
  pk.L = lanes_per_word(fw);
  pk.len = d->S;
  pk.wpr = static_cast<int>(words_per_row(fw, d->S));
  pk.pad = 0;
  pk.reverse = 1;
  pk.sign_bits = field_bits(g.F, d->S, fw.bits - 1, 64, false);
  e = fw.word_bits == 32 ? launch_prep<uint32_t>(wt, KR, pk, s) : launch_prep<uint64_t>(wt, KR, pk, s);
  if (e != cudaSuccess) return SAMD_ECUDA;

  ConvArgs a;
  a.X = X;
  a.KR = KR;
  a.acc_out = acc_out;
  a.packed_out = packed_out;
  a.N = d->N;
  a.C = d->C;
  a.H = d->H;
  a.K = d->K;
  a.R = d->R;
  a.S = d->S;
  a.pad = d->pad;
  a.Ho = g.Ho;
  a.Wo = g.Wo;
  a.G = g.G;
  a.F = g.F;
  a.nx = g.nx;
  a.msb_lo = field_bits(g.F, 128 / g.F, g.F - 1, 128, false);
  a.msb_hi = field_bits(g.F, 128 / g.F, g.F - 1, 128, true);
  a.out_bits = packed_out ? fo.bits : 8;
  a.out_signed = packed_out ? fo.is_signed : 1;
  a.out_lane_w = packed_out ? fo.bits + fo.spacer : 8;
  a.out_L = packed_out ? lanes_per_word(fo) : 1;
  a.out_wpr = packed_out ? static_cast<int>(words_per_row(fo, g.Wo)) : 0;
  a.out_word64 = packed_out ? (fo.word_bits == 64) : 0;
  a.shift = shift;
  a.row_bytes = packed_out ? (g.Wo + 15) / 16 * 16 : 0;
  const unsigned grid = static_cast<unsigned>((rows + kWarps - 1) / kWarps);
  const size_t smem = static_cast<size_t>(a.row_bytes) * kWarps;
  if (a.out_word64)
    wm_conv_kernel<uint64_t><<<grid, 32 * kWarps, smem, s>>>(a);
  else
    wm_conv_kernel<uint32_t><<<grid, 32 * kWarps, smem, s>>>(a);
  return cudaGetLastError() == cudaSuccess ? SAMD_OK : SAMD_ECUDA;
}

}  // namespace samd
