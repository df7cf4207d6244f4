// maxpool.cu -- lane-wise 2x2 max-pool, stride 2, on NHWC tensors packed
// along C (used between the VGG-16 blocks; the paper has no pooling).
//
// The max of two words is taken for all lanes at once. Spacer-free lanes: a
// lane-wise subtract with the MSBs as temporary spacers (section 3, Fig. 5)
// yields each lane's borrow, i.e. a < b, which selects the larger lane.
// Lanes with permanent spacer bits (Fig. 2) read a >= b from the first
// spacer bit of (a | carry) - b. Signed lanes are compared after flipping
// their sign bits (two's complement order = offset-binary order).
#include <cstring>

#include "samd_internal.cuh"

namespace samd {
namespace {

constexpr int kThreads = 256;

template <typename W, int BITS>
__device__ __forceinline__ W swar_max(W a, W b, W flip) {
  return swar_lane_max<W, BITS>(a, b, flip);
}

// Blocks loop over output rows (image n, row i); threads run over the row's
// (pixel, unit) pairs, a unit being V consecutive words of a pixel (V = 4
// 32-bit or 2 64-bit words, one 16-byte vector, when a pixel's words allow;
// else V = 1). Index math stays in 32 bits.
template <typename W, int BITS, int V>
__global__ void __launch_bounds__(kThreads) maxpool_swar_kernel(const W *__restrict__ in, W *__restrict__ out, int Ho,
                                                                int Wo, int H, int W_, int wpr, int is_signed, int rows) {
  const int upp = wpr / V;  // units per pixel
  const int units = Wo * upp;
  const W flip = is_signed ? LaneMsb<W, BITS>::kValue : W(0);
  for (int row = blockIdx.x; row < rows; row += gridDim.x) {  // row = n * Ho + i
  const int n = row / Ho, i = row - (row / Ho) * Ho;
  const W *top = in + (static_cast<long long>(n) * H + 2 * i) * W_ * wpr;
  const W *bot = top + static_cast<long long>(W_) * wpr;
  W *dst = out + static_cast<long long>(row) * Wo * wpr;
  for (int u = blockIdx.y * blockDim.x + threadIdx.x; u < units; u += gridDim.y * blockDim.x) {
    const int j = u / upp, q = u - (u / upp) * upp;
    const int off = 2 * j * wpr + q * V;
    if constexpr (V == 1) {
      const W m1 = swar_max<W, BITS>(__ldcs(top + off), __ldcs(top + off + wpr), flip);
      const W m2 = swar_max<W, BITS>(__ldcs(bot + off), __ldcs(bot + off + wpr), flip);
      dst[j * wpr + q] = swar_max<W, BITS>(m1, m2, flip);
    } else {
      const uint4 a = __ldcs(reinterpret_cast<const uint4 *>(top + off));
      const uint4 b = __ldcs(reinterpret_cast<const uint4 *>(top + off + wpr));
      const uint4 c = __ldcs(reinterpret_cast<const uint4 *>(bot + off));
      const uint4 d = __ldcs(reinterpret_cast<const uint4 *>(bot + off + wpr));
      W wa[V], wbv[V], wc[V], wd[V], wo[V];
      memcpy(wa, &a, 16);
      memcpy(wbv, &b, 16);
      memcpy(wc, &c, 16);
      memcpy(wd, &d, 16);
#pragma unroll
      for (int k = 0; k < V; ++k)
        wo[k] = swar_max<W, BITS>(swar_max<W, BITS>(wa[k], wbv[k], flip), swar_max<W, BITS>(wc[k], wd[k], flip), flip);
      uint4 o;
      memcpy(&o, wo, 16);
      __stcs(reinterpret_cast<uint4 *>(dst + j * wpr + q * V), o);
    }
  }
  }
}

// Formats with permanent spacer bits: the same row walk, one word per
// (pixel, word) pair, lane-wise max by field_max.
template <typename W>
__global__ void __launch_bounds__(kThreads) maxpool_field_kernel(const W *__restrict__ in, W *__restrict__ out, int Ho,
                                                                 int Wo, int H, int W_, int wpr, int is_signed,
                                                                 int rows, const FieldMasks<W> f) {
  const int units = Wo * wpr;
  const W flip = is_signed ? f.msb : W(0);
  for (int row = blockIdx.x; row < rows; row += gridDim.x) {  // row = n * Ho + i
    const int n = row / Ho, i = row - (row / Ho) * Ho;
    const W *top = in + (static_cast<long long>(n) * H + 2 * i) * W_ * wpr;
    const W *bot = top + static_cast<long long>(W_) * wpr;
    W *dst = out + static_cast<long long>(row) * Wo * wpr;
    for (int u = blockIdx.y * blockDim.x + threadIdx.x; u < units; u += gridDim.y * blockDim.x) {
      const int j = u / wpr, q = u - (u / wpr) * wpr;
      const int off = 2 * j * wpr + q;
      const W m1 = field_max<W>(__ldcs(top + off), __ldcs(top + off + wpr), f, flip);
      const W m2 = field_max<W>(__ldcs(bot + off), __ldcs(bot + off + wpr), f, flip);
      dst[j * wpr + q] = field_max<W>(m1, m2, f, flip);
    }
  }
}

template <typename W>
cudaError_t pool_dispatch(samd_fmt f, const void *in, void *out, int N, int C, int H, int W_, cudaStream_t s) {
  int wpr = static_cast<int>(words_per_row(f, C));
  const W *pi = static_cast<const W *>(in);
  W *po = static_cast<W *>(out);
  const int Ho = H / 2, Wo = W_ / 2;
  constexpr int V16 = 16 / static_cast<int>(sizeof(W));
  const bool vec = f.spacer == 0 && (wpr % V16) == 0;
  const int units = Wo * (vec ? wpr / V16 : wpr);
  int gy = (units + kThreads - 1) / kThreads;
  if (gy > 65535) gy = 65535;
  if (static_cast<long long>(N) * Ho > 2147483647LL) return cudaErrorInvalidValue;
  const int rows = N * Ho;
  // enough blocks to fill the GPU (8 per SM), each looping over rows
  long long gx = (static_cast<long long>(sm_count()) * 8 + gy - 1) / gy;
  if (gx > rows) gx = rows;
  const dim3 pgrid(static_cast<unsigned>(gx), gy);
  if (f.spacer != 0) {
    maxpool_field_kernel<W><<<pgrid, kThreads, 0, s>>>(pi, po, Ho, Wo, H, W_, wpr, f.is_signed, rows,
                                                       field_masks<W>(f));
    return cudaGetLastError();
  }
  switch (f.bits * 2 + (vec ? 1 : 0)) {
#define SAMD_POOL_CASE(B)                                                                                   \
  case 2 * B:                                                                                               \
    maxpool_swar_kernel<W, B, 1><<<pgrid, kThreads, 0, s>>>(pi, po, Ho, Wo, H, W_, wpr, f.is_signed, rows); \
    break;                                                                                                  \
  case 2 * B + 1:                                                                                           \
    maxpool_swar_kernel<W, B, V16><<<pgrid, kThreads, 0, s>>>(pi, po, Ho, Wo, H, W_, wpr, f.is_signed, rows); \
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
