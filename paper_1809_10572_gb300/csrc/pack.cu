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

// Load/store NB consecutive 32-bit chunks with VB-byte vectors (VB >= 4,
// address VB-aligned).
template <int VB, int NB>
__device__ __forceinline__ void load_chunks(const void *src, uint32_t (&c)[NB]) {
  if constexpr (VB == 16) {
#pragma unroll
    for (int v = 0; v < NB / 4; ++v) {
      const uint4 t = __ldcs(reinterpret_cast<const uint4 *>(src) + v);
      c[4 * v] = t.x, c[4 * v + 1] = t.y, c[4 * v + 2] = t.z, c[4 * v + 3] = t.w;
    }
  } else if constexpr (VB == 8) {
#pragma unroll
    for (int v = 0; v < NB / 2; ++v) {
      const uint2 t = __ldcs(reinterpret_cast<const uint2 *>(src) + v);
      c[2 * v] = t.x, c[2 * v + 1] = t.y;
    }
  } else {
#pragma unroll
    for (int v = 0; v < NB; ++v) c[v] = __ldcs(reinterpret_cast<const uint32_t *>(src) + v);
  }
}

template <int VB, int NB>
__device__ __forceinline__ void store_chunks(void *dst, const uint32_t (&c)[NB]) {
  if constexpr (VB == 16) {
#pragma unroll
    for (int v = 0; v < NB / 4; ++v)
      __stcs(reinterpret_cast<uint4 *>(dst) + v, make_uint4(c[4 * v], c[4 * v + 1], c[4 * v + 2], c[4 * v + 3]));
  } else if constexpr (VB == 8) {
#pragma unroll
    for (int v = 0; v < NB / 2; ++v) __stcs(reinterpret_cast<uint2 *>(dst) + v, make_uint2(c[2 * v], c[2 * v + 1]));
  } else {
#pragma unroll
    for (int v = 0; v < NB; ++v) __stcs(reinterpret_cast<uint32_t *>(dst) + v, c[v]);
  }
}

__device__ __forceinline__ uint32_t bfe_u32(uint32_t x, int pos, int len) {
  uint32_t r;
  asm("bfe.u32 %0, %1, %2, %3;" : "=r"(r) : "r"(x), "r"(pos), "r"(len));
  return r;
}
__device__ __forceinline__ uint32_t bfe_s32(uint32_t x, int pos, int len) {
  uint32_t r;
  asm("bfe.s32 %0, %1, %2, %3;" : "=r"(r) : "r"(x), "r"(pos), "r"(len));
  return r;
}
__device__ __forceinline__ uint32_t bfi_b32(uint32_t src, uint32_t into, int pos, int len) {
  uint32_t r;
  asm("bfi.b32 %0, %1, %2, %3, %4;" : "=r"(r) : "r"(src), "r"(into), "r"(pos), "r"(len));
  return r;
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

// ---- single-row (or whole-word rows) 32-bit words: four words per thread ----
//
// A thread packs 4 consecutive words (one 16-byte store) from 4L consecutive
// bytes read with the widest aligned vector that divides 4L. For 1-, 4- and
// 8-bit lanes whole groups of lanes move at once:
//   b = 1: (x & 0x01010101) * 0x01020408 >> 24 gathers the low bits of four
//          bytes into a nibble (the partial products never meet below bit 24);
//   b = 4: x | x >> 4 puts nibble pairs in bytes 0 and 2 of each 32-bit chunk,
//          and one byte permute (PRMT) joins two chunks into a word;
//   b = 8: the bytes are the word.
// Other widths insert lane by lane with compile-time shifts.
template <int BITS>
__device__ __forceinline__ uint32_t pack_word32(const uint32_t *c) {  // c: the L bytes of the word as L/4 chunks
  constexpr int L = 32 / BITS;
  if constexpr (BITS == 8) {
    return c[0];
  } else if constexpr (BITS == 4) {
    const uint32_t a = c[0] & 0x0F0F0F0Fu, b = c[1] & 0x0F0F0F0Fu;
    return __byte_perm(a | (a >> 4), b | (b >> 4), 0x6420);
  } else if constexpr (BITS == 1) {
    uint32_t w = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) w |= (((c[i] & 0x01010101u) * 0x01020408u) >> 24) << (4 * i);
    return w;
  } else {
    (void)L;
    return 0u;  // not used: other widths take pack_lanes
  }
}

template <int BITS, int NB>
__device__ __forceinline__ void pack_lanes(const uint32_t (&in)[NB], uint32_t (&w)[4]) {
  constexpr int L = 32 / BITS;
  constexpr uint32_t M = (1u << BITS) - 1;
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    uint32_t word = 0;
#pragma unroll
    for (int l = 0; l < L; ++l) {
      const int e = k * L + l;
      word = bfi_b32(in[e / 4] >> (8 * (e % 4)), word, l * BITS, BITS);
      (void)M;
    }
    w[k] = word;
  }
}

// A warp packs 32 consecutive quads of words. Its 32 x 4L input bytes are one
// contiguous block, read with consecutive 16-byte loads into shared memory
// (rows padded by 16 bytes), from where each lane takes its own 4L bytes.
template <int BITS>
__global__ void __launch_bounds__(kThreads) pack32_staged_kernel(const int8_t *__restrict__ src,
                                                                 uint32_t *__restrict__ dst, int64_t nwarp_tiles) {
  constexpr int L = 32 / BITS;
  constexpr int IB = 4 * L;  // input bytes per lane
  constexpr int NB = IB / 4;
  constexpr int ROW = IB + 16;
  constexpr int TILE16 = 2 * IB;
  __shared__ __align__(16) uint8_t stage[kThreads / 32][32 * ROW];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  uint8_t *my = stage[wib];
  const int64_t warps_total = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t wt = blockIdx.x * (int64_t)(blockDim.x >> 5) + wib; wt < nwarp_tiles; wt += warps_total) {
    const uint4 *in16 = reinterpret_cast<const uint4 *>(src + wt * 32 * IB);
#pragma unroll
    for (int p = lane; p < TILE16; p += 32) {
      const uint4 t = __ldcs(in16 + p);
      const uint32_t tw[4] = {t.x, t.y, t.z, t.w};
      const int byte = p * 16, r = byte / IB, off = byte - r * IB;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int b = off + 4 * k, rr = r + b / IB, oo = b - (b / IB) * IB;
        *reinterpret_cast<uint32_t *>(my + rr * ROW + oo) = tw[k];
      }
    }
    __syncwarp();
    uint32_t in[NB];
#pragma unroll
    for (int i = 0; i < NB; ++i) in[i] = *reinterpret_cast<const uint32_t *>(my + lane * ROW + 4 * i);
    __syncwarp();
    uint32_t w[4];
    if constexpr (BITS == 1 || BITS == 4 || BITS == 8) {
#pragma unroll
      for (int k = 0; k < 4; ++k) w[k] = pack_word32<BITS>(in + k * (L / 4));
    } else {
      pack_lanes<BITS, NB>(in, w);
    }
    __stcs(reinterpret_cast<uint4 *>(dst) + wt * 32 + lane, make_uint4(w[0], w[1], w[2], w[3]));
  }
}

// Lanes of 2 bits and more read their 4L bytes directly (at most 64 bytes a
// lane; the L1 cache merges a warp's neighbouring lines).
template <int BITS>
__global__ void __launch_bounds__(kThreads) pack32_vec_kernel(const int8_t *__restrict__ src, uint32_t *__restrict__ dst,
                                                              int64_t nquads) {
  constexpr int L = 32 / BITS;
  constexpr int IB = 4 * L;
  constexpr int VB = vec_bytes(IB);
  constexpr int NB = IB / 4;
  for (int64_t q = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; q < nquads; q += (int64_t)gridDim.x * blockDim.x) {
    uint32_t in[NB];
    load_chunks<VB, NB>(src + q * IB, in);
    uint32_t w[4];
    if constexpr (BITS == 4 || BITS == 8) {
#pragma unroll
      for (int k = 0; k < 4; ++k) w[k] = pack_word32<BITS>(in + k * (L / 4));
    } else {
      pack_lanes<BITS, NB>(in, w);
    }
    __stcs(reinterpret_cast<uint4 *>(dst) + q, make_uint4(w[0], w[1], w[2], w[3]));
  }
}

// Unpack of 4 words per thread into 4L bytes, written with the widest aligned
// vector. b = 8: the word is its bytes. b = 4: the low and high nibbles of
// each byte are masked apart and interleaved by byte permutes; signed nibbles
// are extended by or-ing 0xF0 into bytes whose bit 3 is set
// ((x & 0x08080808) * 0x1E). b = 1: (nibble * 0x00204081) & 0x01010101
// spreads four bits into four bytes; signed 1-bit lanes are -bit (x 0xFF).
template <int BITS, bool SIGNED>
__device__ __forceinline__ void unpack_word32(uint32_t w, uint32_t *out) {  // out: L/4 chunks of 4 bytes
  constexpr int L = 32 / BITS;
  if constexpr (BITS == 8) {
    out[0] = w;
  } else if constexpr (BITS == 4) {
    uint32_t lo = w & 0x0F0F0F0Fu, hi = (w >> 4) & 0x0F0F0F0Fu;
    if constexpr (SIGNED) {
      lo |= (lo & 0x08080808u) * 0x1Eu;
      hi |= (hi & 0x08080808u) * 0x1Eu;
    }
    out[0] = __byte_perm(lo, hi, 0x5140);
    out[1] = __byte_perm(lo, hi, 0x7362);
  } else if constexpr (BITS == 1) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      uint32_t t = (((w >> (4 * i)) & 0xFu) * 0x00204081u) & 0x01010101u;
      if constexpr (SIGNED) t *= 0xFFu;
      out[i] = t;
    }
  } else {
#pragma unroll
    for (int j = 0; j < L / 4 + (L % 4 ? 1 : 0); ++j) out[j] = 0;
    (void)w;
  }
}

// A warp expands 32 consecutive quads of words; its 32 x 4L output bytes are
// one contiguous block. Each lane stages its 4L bytes in shared memory (rows
// padded by 16 bytes so the lanes' 16-byte writes spread over the banks),
// then the warp writes the block with consecutive 16-byte stores.
template <int BITS, bool SIGNED>
__global__ void __launch_bounds__(kThreads) unpack32_vec_kernel(const uint32_t *__restrict__ src,
                                                                int8_t *__restrict__ dst, int64_t nwarp_tiles) {
  constexpr int L = 32 / BITS;
  constexpr int OB = 4 * L;          // output bytes per lane
  constexpr int NC = OB / 4;
  constexpr int ROW = OB + 16;       // staged row pitch (16-byte aligned)
  constexpr int TILE16 = 2 * OB;     // 16-byte vectors per warp block (32 * OB / 16)
  __shared__ __align__(16) uint8_t stage[kThreads / 32][32 * ROW];
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  uint8_t *my = stage[wib];
  const int64_t warps_total = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t wt = blockIdx.x * (int64_t)(blockDim.x >> 5) + wib; wt < nwarp_tiles; wt += warps_total) {
    const int64_t q = wt * 32 + lane;
    const uint4 v = __ldcs(reinterpret_cast<const uint4 *>(src) + q);
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t c[NC];
    if constexpr (BITS == 1 || BITS == 4 || BITS == 8) {
#pragma unroll
      for (int k = 0; k < 4; ++k) unpack_word32<BITS, SIGNED>(w[k], c + k * (L / 4));
    } else {
#pragma unroll
      for (int i = 0; i < NC; ++i) c[i] = 0;
#pragma unroll
      for (int k = 0; k < 4; ++k)
#pragma unroll
        for (int l = 0; l < L; ++l) {
          const int e = k * L + l;
          const uint32_t p = SIGNED ? bfe_s32(w[k], l * BITS, BITS) : bfe_u32(w[k], l * BITS, BITS);
          c[e / 4] = bfi_b32(p, c[e / 4], 8 * (e % 4), 8);
        }
    }
    // stage: lane's row holds its OB bytes (4-byte stores; OB may be 20 or 40)
#pragma unroll
    for (int i = 0; i < NC; ++i) *reinterpret_cast<uint32_t *>(my + lane * ROW + 4 * i) = c[i];
    __syncwarp();
    uint4 *out = reinterpret_cast<uint4 *>(dst + wt * 32 * OB);
#pragma unroll
    for (int p = lane; p < TILE16; p += 32) {
      const int byte = p * 16, r = byte / OB, off = byte - r * OB;  // 16-byte vector p of the block
      uint32_t t[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        // OB is a multiple of 4, so a 4-byte piece never straddles two rows
        const int b = off + 4 * k, rr = r + b / OB, oo = b - (b / OB) * OB;
        t[k] = *reinterpret_cast<const uint32_t *>(my + rr * ROW + oo);
      }
      __stcs(out + p, make_uint4(t[0], t[1], t[2], t[3]));
    }
    __syncwarp();
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

template <int BITS>
cudaError_t launch_pack32_vec(const int8_t *src, uint32_t *dst, int64_t ntiles, cudaStream_t s) {
  if (BITS == 1)
    pack32_staged_kernel<BITS><<<resident_grid<pack32_staged_kernel<BITS>>(ntiles * 32, kThreads), kThreads, 0, s>>>(
        src, dst, ntiles);
  else
    pack32_vec_kernel<BITS><<<resident_grid<pack32_vec_kernel<BITS>>(ntiles * 32, kThreads), kThreads, 0, s>>>(
        src, dst, ntiles * 32);
  return cudaGetLastError();
}

template <int BITS, bool SIGNED>
cudaError_t launch_unpack32_vec(const uint32_t *src, int8_t *dst, int64_t ntiles, cudaStream_t s) {
  const int grid = resident_grid<unpack32_vec_kernel<BITS, SIGNED>>(ntiles * 32, kThreads);
  unpack32_vec_kernel<BITS, SIGNED><<<grid, kThreads, 0, s>>>(src, dst, ntiles);
  return cudaGetLastError();
}

template <typename W>
cudaError_t pack_dispatch(samd_fmt f, const int8_t *src, W *dst, int64_t rows, int64_t inner, cudaStream_t s) {
  int L = lanes_per_word(f);
  int64_t wpr = words_per_row(f, inner);
  int64_t total = rows * wpr;
  int grid = grid_for(total, kThreads, sm_count() * 16);
  int affine = (rows == 1 || inner % L == 0) ? 1 : 0;
  int64_t n = rows * inner;
  // bulk of a spacer-free 32-bit affine array: 4 full words per thread; the
  // remaining words (partial quad, ragged last word) by the word kernel below
  if (sizeof(W) == 4 && f.spacer == 0 && affine) {
    const int64_t ntiles = (n / L) / 128;  // warp tiles of 32 quads of words
    const int64_t nquads = ntiles * 32;
    if (ntiles > 0) {
      cudaError_t e;
      uint32_t *d32 = reinterpret_cast<uint32_t *>(dst);
      switch (f.bits) {
        case 1: e = launch_pack32_vec<1>(src, d32, ntiles, s); break;
        case 2: e = launch_pack32_vec<2>(src, d32, ntiles, s); break;
        case 3: e = launch_pack32_vec<3>(src, d32, ntiles, s); break;
        case 4: e = launch_pack32_vec<4>(src, d32, ntiles, s); break;
        case 5: e = launch_pack32_vec<5>(src, d32, ntiles, s); break;
        case 6: e = launch_pack32_vec<6>(src, d32, ntiles, s); break;
        case 7: e = launch_pack32_vec<7>(src, d32, ntiles, s); break;
        default: e = launch_pack32_vec<8>(src, d32, ntiles, s); break;
      }
      if (e != cudaSuccess) return e;
      const int64_t done_words = nquads * 4;
      if (done_words == total) return cudaSuccess;
      // the tail: words [done_words, total) of the single (affine) row
      const int64_t tail = total - done_words;
      src += done_words * L;
      dst += done_words;
      n -= done_words * L;
      total = tail;
      rows = 1;
      inner = n;
      wpr = total;
      grid = grid_for(total, kThreads, sm_count() * 16);
    }
  }
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
  if (sizeof(W) == 4 && f.spacer == 0 && affine) {
    const int64_t ntiles = (n / L) / 128;
    const int64_t nquads = ntiles * 32;
    if (ntiles > 0) {
      cudaError_t e;
      const uint32_t *s32 = reinterpret_cast<const uint32_t *>(src);
      switch (f.bits * 2 + (f.is_signed ? 1 : 0)) {
#define SAMD_UV(B)                                                                      \
  case 2 * B: e = launch_unpack32_vec<B, false>(s32, dst, ntiles, s); break;           \
  case 2 * B + 1: e = launch_unpack32_vec<B, true>(s32, dst, ntiles, s); break;
        SAMD_UV(1) SAMD_UV(2) SAMD_UV(3) SAMD_UV(4) SAMD_UV(5) SAMD_UV(6) SAMD_UV(7) SAMD_UV(8)
#undef SAMD_UV
        default: return cudaErrorInvalidValue;
      }
      if (e != cudaSuccess) return e;
      const int64_t done_words = nquads * 4;
      if (done_words == total) return cudaSuccess;
      const int64_t tail = total - done_words;
      src += done_words;
      dst += done_words * L;
      n -= done_words * L;
      total = tail;
      rows = 1;
      inner = n;
      wpr = total;
      grid = grid_for(total, kThreads, sm_count() * 16);
    }
  }
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
