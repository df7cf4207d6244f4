// maxpool.cu -- lane-wise 2x2 max-pool, stride 2, on NHWC tensors packed
// along C (used between the VGG-16 blocks; the paper has no pooling).
//
// One thread per output word. For spacer-free lanes the max of two words is
// taken for all lanes at once: a lane-wise subtract with the MSBs as
// temporary spacers (section 3, Fig. 5) yields each lane's borrow, i.e.
// a < b, which selects the larger lane. Signed lanes are compared after
// flipping their sign bits (two's complement order = offset-binary order).
#include "samd_internal.cuh"

namespace samd {
namespace {

constexpr int kThreads = 256;

template <typename W, int BITS>
struct PoolMasks {
  static constexpr int L = WordTraits<W>::kBits / BITS;
  static constexpr W msb() {
    W m = 0;
    for (int i = 0; i < L; ++i) m |= W(1) << (i * BITS + BITS - 1);
    return m;
  }
  static constexpr W kMsb = msb();
};

template <typename W, int BITS>
__device__ __forceinline__ W swar_max(W a, W b, W flip) {
  constexpr W M = PoolMasks<W, BITS>::kMsb;
  W x = a ^ flip, y = b ^ flip;                        // offset-binary for signed lanes
  W d = ((x ^ y) & M) ^ ((x | M) - (y & ~M)) ^ M;       // lane-wise x - y
  W lt = ((~x & y) | ((~x | y) & d)) & M;               // borrow out of the lane: x < y
  W E = (lt - (lt >> (BITS - 1))) | lt;                 // whole lanes where x < y
  return (b & E) | (a & ~E);
}

template <typename W, int BITS>
__global__ void __launch_bounds__(kThreads) maxpool_swar_kernel(const W *__restrict__ in, W *__restrict__ out,
                                                                int N, int H, int W_, int wpr, int is_signed) {
  const int Ho = H / 2, Wo = W_ / 2;
  const int64_t total = (int64_t)N * Ho * Wo * wpr;
  const W flip = is_signed ? PoolMasks<W, BITS>::kMsb : W(0);
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
    int64_t px = t / wpr;
    int wi = static_cast<int>(t - px * wpr);
    int j = static_cast<int>(px % Wo);
    int64_t r = px / Wo;
    int i = static_cast<int>(r % Ho);
    int64_t n = r / Ho;
    int64_t base = ((n * H + 2 * i) * W_ + 2 * j) * wpr + wi;
    W m = swar_max<W, BITS>(__ldg(in + base), __ldg(in + base + wpr), flip);
    W m2 = swar_max<W, BITS>(__ldg(in + base + (int64_t)W_ * wpr), __ldg(in + base + (int64_t)W_ * wpr + wpr), flip);
    out[t] = swar_max<W, BITS>(m, m2, flip);
  }
}

template <typename W>
__global__ void __launch_bounds__(kThreads) maxpool_lane_kernel(const W *__restrict__ in, W *__restrict__ out, int N,
                                                                int H, int W_, int wpr, int bits, int is_signed,
                                                                int lane_w, int L) {
  const int Ho = H / 2, Wo = W_ / 2;
  const int64_t total = (int64_t)N * Ho * Wo * wpr;
  const uint32_t lm = (1u << bits) - 1;
  for (int64_t t = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; t < total; t += (int64_t)gridDim.x * blockDim.x) {
    int64_t px = t / wpr;
    int wi = static_cast<int>(t - px * wpr);
    int j = static_cast<int>(px % Wo);
    int64_t r = px / Wo;
    int i = static_cast<int>(r % Ho);
    int64_t n = r / Ho;
    int64_t base = ((n * H + 2 * i) * W_ + 2 * j) * wpr + wi;
    W w[4] = {in[base], in[base + wpr], in[base + (int64_t)W_ * wpr], in[base + (int64_t)W_ * wpr + wpr]};
    W o = 0;
    for (int l = 0; l < L; ++l) {
      int best = lane_value(static_cast<uint32_t>(w[0] >> (l * lane_w)) & lm, bits, is_signed);
      for (int k = 1; k < 4; ++k) {
        int v = lane_value(static_cast<uint32_t>(w[k] >> (l * lane_w)) & lm, bits, is_signed);
        best = v > best ? v : best;
      }
      o |= W(static_cast<uint32_t>(best) & lm) << (l * lane_w);
    }
    out[t] = o;
  }
}

template <typename W>
cudaError_t pool_dispatch(samd_fmt f, const void *in, void *out, int N, int C, int H, int W_, cudaStream_t s) {
  int wpr = static_cast<int>(words_per_row(f, C));
  int64_t total = (int64_t)N * (H / 2) * (W_ / 2) * wpr;
  int grid = grid_for(total, kThreads, sm_count() * 16);
  const W *pi = static_cast<const W *>(in);
  W *po = static_cast<W *>(out);
  if (f.spacer != 0) {
    maxpool_lane_kernel<W><<<grid, kThreads, 0, s>>>(pi, po, N, H, W_, wpr, f.bits, f.is_signed, f.bits + f.spacer,
                                                     lanes_per_word(f));
    return cudaGetLastError();
  }
  switch (f.bits) {
#define SAMD_POOL_CASE(B) \
  case B:                 \
    maxpool_swar_kernel<W, B><<<grid, kThreads, 0, s>>>(pi, po, N, H, W_, wpr, f.is_signed); \
    break;
    SAMD_POOL_CASE(1) SAMD_POOL_CASE(2) SAMD_POOL_CASE(3) SAMD_POOL_CASE(4)
    SAMD_POOL_CASE(5) SAMD_POOL_CASE(6) SAMD_POOL_CASE(7) SAMD_POOL_CASE(8)
#undef SAMD_POOL_CASE
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_maxpool2x2_nhwc(samd_fmt f, const void *in, void *out, int N, int C, int H, int W_,
                                   cudaStream_t s) {
  if (f.word_bits == 32) return pool_dispatch<uint32_t>(f, in, out, N, C, H, W_, s);
  return pool_dispatch<uint64_t>(f, in, out, N, C, H, W_, s);
}

}  // namespace samd
