// pack.cu -- int8 bytes <-> packed b-bit lanes (section 2.1 of the paper:
// b-bit lanes laid side by side in a scalar word; section 7: unpacking to
// the native 8-bit type).
//
// One thread owns one packed word. When the word -> element map is affine
// (a single row, or rows whose length is a multiple of L) a full word's L
// bytes are moved with the widest aligned vector access that divides L;
// otherwise (a ragged row tail, or rows that do not end on a word boundary)
// the word's bytes are moved one at a time. Both forms produce the same
// canonical words.
#include "samd_internal.cuh"

namespace samd {
namespace {

constexpr int kThreads = 256;

// Largest power of two dividing n, capped at 16: the vector width in bytes
// for moving L consecutive bytes that start at a multiple of L.
__host__ __device__ constexpr int vec_bytes(int n) {
  return (n % 16 == 0) ? 16 : (n % 8 == 0) ? 8 : (n % 4 == 0) ? 4 : (n % 2 == 0) ? 2 : 1;
}

template <int VB>
struct Vec;
template <>
struct Vec<16> {
  using T = uint4;
};
template <>
struct Vec<8> {
  using T = uint2;
};
template <>
struct Vec<4> {
  using T = uint32_t;
};
template <>
struct Vec<2> {
  using T = uint16_t;
};
template <>
struct Vec<1> {
  using T = uint8_t;
};

// Copy n bytes (n a multiple of VB, src/dst VB-aligned) through registers.
template <int VB, int N>
__device__ __forceinline__ void load_bytes(const int8_t *src, uint8_t (&buf)[N]) {
  using T = typename Vec<VB>::T;
  const T *p = reinterpret_cast<const T *>(src);
#pragma unroll
  for (int v = 0; v < N / VB; ++v) {
    T t = __ldg(p + v);
    const uint8_t *tb = reinterpret_cast<const uint8_t *>(&t);
#pragma unroll
    for (int j = 0; j < VB; ++j) buf[v * VB + j] = tb[j];
  }
}

template <int VB, int N>
__device__ __forceinline__ void store_bytes(int8_t *dst, const uint8_t (&buf)[N]) {
  using T = typename Vec<VB>::T;
  T *p = reinterpret_cast<T *>(dst);
#pragma unroll
  for (int v = 0; v < N / VB; ++v) {
    T t;
    uint8_t *tb = reinterpret_cast<uint8_t *>(&t);
#pragma unroll
    for (int j = 0; j < VB; ++j) tb[j] = buf[v * VB + j];
    p[v] = t;
  }
}

// ---- pack ------------------------------------------------------------------

template <typename W, int BITS>
__global__ void __launch_bounds__(kThreads) pack_kernel(const int8_t *__restrict__ src, W *__restrict__ dst,
                                                        int64_t total_words, int64_t inner, int64_t wpr,
                                                        int affine, int64_t n_elems) {
  constexpr int L = WordTraits<W>::kBits / BITS;
  constexpr int VB = vec_bytes(L);
  constexpr W kMask = (W(1) << BITS) - 1;
  for (int64_t w = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < total_words;
       w += (int64_t)gridDim.x * blockDim.x) {
    int64_t e0, count;
    if (affine) {
      e0 = w * L;
      count = n_elems - e0 < L ? n_elems - e0 : L;
    } else {
      int64_t row = w / wpr, wi = w - row * wpr;
      e0 = row * inner + wi * L;
      count = inner - wi * L < L ? inner - wi * L : L;
    }
    W word = 0;
    if (affine && count == L) {
      uint8_t buf[L];
      load_bytes<VB, L>(src + e0, buf);
#pragma unroll
      for (int i = 0; i < L; ++i) word |= (W(buf[i]) & kMask) << (i * BITS);
    } else {
      for (int i = 0; i < count; ++i) word |= (W(static_cast<uint8_t>(src[e0 + i])) & kMask) << (i * BITS);
    }
    dst[w] = word;
  }
}

// Any format, spacer bits included: lane i at bit i * (bits + spacer).
template <typename W>
__global__ void __launch_bounds__(kThreads) pack_generic_kernel(const int8_t *__restrict__ src, W *__restrict__ dst,
                                                                int64_t total_words, int64_t inner, int64_t wpr,
                                                                int bits, int lane_w, int L) {
  const W mask = (W(1) << bits) - 1;
  for (int64_t w = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < total_words;
       w += (int64_t)gridDim.x * blockDim.x) {
    int64_t row = w / wpr, wi = w - row * wpr;
    int64_t e0 = row * inner + wi * L;
    int64_t count = inner - wi * L < L ? inner - wi * L : L;
    W word = 0;
    for (int i = 0; i < count; ++i) word |= (W(static_cast<uint8_t>(src[e0 + i])) & mask) << (i * lane_w);
    dst[w] = word;
  }
}

// ---- unpack ----------------------------------------------------------------

template <typename W, int BITS, bool SIGNED>
__device__ __forceinline__ uint8_t lane_byte(W word, int i) {
  uint32_t p = static_cast<uint32_t>(word >> (i * BITS)) & ((1u << BITS) - 1);
  if (SIGNED) p = static_cast<uint32_t>(static_cast<int>(p << (32 - BITS)) >> (32 - BITS));
  return static_cast<uint8_t>(p);
}

template <typename W, int BITS, bool SIGNED>
__global__ void __launch_bounds__(kThreads) unpack_kernel(const W *__restrict__ src, int8_t *__restrict__ dst,
                                                          int64_t total_words, int64_t inner, int64_t wpr,
                                                          int affine, int64_t n_elems) {
  constexpr int L = WordTraits<W>::kBits / BITS;
  constexpr int VB = vec_bytes(L);
  for (int64_t w = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < total_words;
       w += (int64_t)gridDim.x * blockDim.x) {
    int64_t e0, count;
    if (affine) {
      e0 = w * L;
      count = n_elems - e0 < L ? n_elems - e0 : L;
    } else {
      int64_t row = w / wpr, wi = w - row * wpr;
      e0 = row * inner + wi * L;
      count = inner - wi * L < L ? inner - wi * L : L;
    }
    W word = __ldg(src + w);
    if (affine && count == L) {
      uint8_t buf[L];
#pragma unroll
      for (int i = 0; i < L; ++i) buf[i] = lane_byte<W, BITS, SIGNED>(word, i);
      store_bytes<VB, L>(dst + e0, buf);
    } else {
      for (int i = 0; i < count; ++i) dst[e0 + i] = static_cast<int8_t>(lane_byte<W, BITS, SIGNED>(word, i));
    }
  }
}

template <typename W>
__global__ void __launch_bounds__(kThreads) unpack_generic_kernel(const W *__restrict__ src, int8_t *__restrict__ dst,
                                                                  int64_t total_words, int64_t inner, int64_t wpr,
                                                                  int bits, int is_signed, int lane_w, int L) {
  for (int64_t w = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; w < total_words;
       w += (int64_t)gridDim.x * blockDim.x) {
    int64_t row = w / wpr, wi = w - row * wpr;
    int64_t e0 = row * inner + wi * L;
    int64_t count = inner - wi * L < L ? inner - wi * L : L;
    W word = __ldg(src + w);
    for (int i = 0; i < count; ++i) {
      uint32_t p = static_cast<uint32_t>(word >> (i * lane_w)) & ((1u << bits) - 1);
      dst[e0 + i] = static_cast<int8_t>(lane_value(p, bits, is_signed));
    }
  }
}

template <typename W>
cudaError_t pack_dispatch(samd_fmt f, const int8_t *src, W *dst, int64_t rows, int64_t inner, cudaStream_t s) {
  int L = lanes_per_word(f);
  int64_t wpr = words_per_row(f, inner);
  int64_t total = rows * wpr;
  int grid = grid_for(total, kThreads, sm_count() * 16);
  int affine = (rows == 1 || inner % L == 0) ? 1 : 0;
  int64_t n = rows * inner;
  if (f.spacer != 0) {
    pack_generic_kernel<W><<<grid, kThreads, 0, s>>>(src, dst, total, inner, wpr, f.bits, f.bits + f.spacer, L);
    return cudaGetLastError();
  }
  switch (f.bits) {
#define SAMD_PACK_CASE(B) \
  case B:                 \
    pack_kernel<W, B><<<grid, kThreads, 0, s>>>(src, dst, total, inner, wpr, affine, n); \
    break;
    SAMD_PACK_CASE(1) SAMD_PACK_CASE(2) SAMD_PACK_CASE(3) SAMD_PACK_CASE(4)
    SAMD_PACK_CASE(5) SAMD_PACK_CASE(6) SAMD_PACK_CASE(7) SAMD_PACK_CASE(8)
#undef SAMD_PACK_CASE
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

template <typename W>
cudaError_t unpack_dispatch(samd_fmt f, const W *src, int8_t *dst, int64_t rows, int64_t inner, cudaStream_t s) {
  int L = lanes_per_word(f);
  int64_t wpr = words_per_row(f, inner);
  int64_t total = rows * wpr;
  int grid = grid_for(total, kThreads, sm_count() * 16);
  int affine = (rows == 1 || inner % L == 0) ? 1 : 0;
  int64_t n = rows * inner;
  if (f.spacer != 0) {
    unpack_generic_kernel<W><<<grid, kThreads, 0, s>>>(src, dst, total, inner, wpr, f.bits, f.is_signed,
                                                       f.bits + f.spacer, L);
    return cudaGetLastError();
  }
  switch (f.bits * 2 + (f.is_signed ? 1 : 0)) {
#define SAMD_UNPACK_CASE(B)                                                                   \
  case 2 * B:                                                                                 \
    unpack_kernel<W, B, false><<<grid, kThreads, 0, s>>>(src, dst, total, inner, wpr, affine, n); \
    break;                                                                                    \
  case 2 * B + 1:                                                                             \
    unpack_kernel<W, B, true><<<grid, kThreads, 0, s>>>(src, dst, total, inner, wpr, affine, n);  \
    break;
    SAMD_UNPACK_CASE(1) SAMD_UNPACK_CASE(2) SAMD_UNPACK_CASE(3) SAMD_UNPACK_CASE(4)
    SAMD_UNPACK_CASE(5) SAMD_UNPACK_CASE(6) SAMD_UNPACK_CASE(7) SAMD_UNPACK_CASE(8)
#undef SAMD_UNPACK_CASE
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pack(samd_fmt f, const int8_t *src, void *dst, int64_t rows, int64_t inner, cudaStream_t s) {
  if (f.word_bits == 32) return pack_dispatch<uint32_t>(f, src, static_cast<uint32_t *>(dst), rows, inner, s);
  return pack_dispatch<uint64_t>(f, src, static_cast<uint64_t *>(dst), rows, inner, s);
}

cudaError_t launch_unpack(samd_fmt f, const void *src, int8_t *dst, int64_t rows, int64_t inner, cudaStream_t s) {
  if (f.word_bits == 32)
    return unpack_dispatch<uint32_t>(f, static_cast<const uint32_t *>(src), dst, rows, inner, s);
  return unpack_dispatch<uint64_t>(f, static_cast<const uint64_t *>(src), dst, rows, inner, s);
}

}  // namespace samd
