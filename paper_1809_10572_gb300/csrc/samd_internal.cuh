// samd_internal.cuh -- helpers shared by the libsamd translation units.
//
// Packed format (section 2.1 of the paper; Fig. 2 for spacer bits): lane i
// of a row sits in word i / L at bit offset (i % L) * (bits + spacer), least
// significant lane first; two's complement for signed lanes (section 6).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/samd.h"

namespace samd {

// ---- host-side format arithmetic -----------------------------------------

inline bool fmt_valid(samd_fmt f) {
  return f.bits >= 1 && f.bits <= 8 && f.spacer <= 8 && (f.word_bits == 32 || f.word_bits == 64) &&
         f.is_signed <= 1 && f.bits + f.spacer <= f.word_bits;
}

inline int lanes_per_word(samd_fmt f) { return fmt_valid(f) ? f.word_bits / (f.bits + f.spacer) : 0; }

inline int64_t words_per_row(samd_fmt f, int64_t inner) {
  int L = lanes_per_word(f);
  return (inner + L - 1) / L;
}

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline bool same_fmt(samd_fmt a, samd_fmt b) {
  return a.bits == b.bits && a.is_signed == b.is_signed && a.spacer == b.spacer && a.word_bits == b.word_bits;
}

inline int grid_for(int64_t work_items, int threads, int max_blocks) {
  int64_t blocks = (work_items + threads - 1) / threads;
  if (blocks < 1) blocks = 1;
  if (blocks > max_blocks) blocks = max_blocks;
  return static_cast<int>(blocks);
}

// Number of SMs of the current device (cached per device).
int sm_count();

// CTAs of `Kernel` resident on one SM at `threads` threads and `smem`
// dynamic shared bytes (its registers and static shared memory decide), at
// least 1; asked once per kernel.
template <auto Kernel>
int resident_ctas(int threads, size_t smem = 0) {
  static const int n = [threads, smem] {
    int r = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&r, Kernel, threads, smem) != cudaSuccess) {
      (void)cudaGetLastError();  // the query's own error; the launch reports any other
      r = 0;
    }
    return r < 1 ? 1 : r;
  }();
  return n;
}

// Grid of a grid-stride kernel: enough CTAs for the work, at most one full
// wave of resident CTAs (sm_count() x resident_ctas). A grid of 8 CTAs per SM
// for a kernel of which only 6 fit leaves a third of a wave to start late and
// run its share on an emptier GPU.
template <auto Kernel>
int resident_grid(int64_t work_items, int threads, size_t smem = 0) {
  return grid_for(work_items, threads, sm_count() * resident_ctas<Kernel>(threads, smem));
}

// ---- device-side lane helpers ----------------------------------------------

template <typename W>
struct WordTraits;
template <>
struct WordTraits<uint32_t> {
  static constexpr int kBits = 32;
};
template <>
struct WordTraits<uint64_t> {
  static constexpr int kBits = 64;
};

// Lane range of a b-bit lane.
__host__ __device__ inline int lane_lo(int bits, bool is_signed) { return is_signed ? -(1 << (bits - 1)) : 0; }
__host__ __device__ inline int lane_hi(int bits, bool is_signed) {
  return is_signed ? (1 << (bits - 1)) - 1 : (1 << bits) - 1;
}

// Value of a lane pattern (low `bits` bits of p).
__device__ __forceinline__ int lane_value(uint32_t p, int bits, bool is_signed) {
  return is_signed ? (static_cast<int>(p << (32 - bits)) >> (32 - bits)) : static_cast<int>(p);
}

__device__ __forceinline__ int clamp_int(int v, int lo, int hi) { return v < lo ? lo : (v > hi ? hi : v); }

// Masks over the lane fields of a format with permanent spacer bits (section
// 2.1, Fig. 2): a field is `bits` data bits and `spacer` zero bits above
// them, L fields per word.
template <typename W>
struct FieldMasks {
  W lsb;    // bit 0 of every field
  W msb;    // the top data bit (bits - 1) of every field
  W carry;  // the first spacer bit (bit `bits`) of every field
  W live;   // the data bits of every field
  int bits, fw, L;  // data bits, field width, fields per word
};

template <typename W>
inline FieldMasks<W> field_masks(samd_fmt f) {
  FieldMasks<W> m;
  m.bits = f.bits;
  m.fw = f.bits + f.spacer;
  m.L = lanes_per_word(f);
  m.lsb = 0;
  for (int i = 0; i < m.L; ++i) m.lsb |= W(1) << (i * m.fw);
  m.msb = m.lsb << (f.bits - 1);
  m.carry = m.lsb << f.bits;
  m.live = m.lsb * ((W(1) << f.bits) - 1);
  return m;
}

// Spread a mask of field bits at position p over the field's bits below p
// (and p itself): m - (m >> p) sets bits [0, p), or-ing m keeps bit p.
template <typename W>
__device__ __forceinline__ W spread_down(W m, int p) {
  return (m - (m >> p)) | m;
}

// Lane-wise max of two words of spacer-separated fields (spacer >= 1), flip
// = the msb mask for signed lanes (offset binary orders like two's
// complement), else 0: in (x | carry) - y every field computes 2^bits + x - y
// > 0, so no borrow crosses a field and the carry bit stays set exactly
// where x >= y.
template <typename W>
__device__ __forceinline__ W field_max(W a, W b, const FieldMasks<W> &f, W flip) {
  const W x = a ^ flip, y = b ^ flip;
  const W ge = ((x | f.carry) - y) & f.carry;
  const W E = ge - (ge >> f.bits);  // the data bits of the lanes where x >= y
  return (a & E) | (b & ~E & f.live);
}

// The top bit of every lane of a spacer-free word of BITS-bit lanes.
template <typename W, int BITS>
struct LaneMsb {
  static constexpr W mask() {
    W m = 0;
    for (int i = 0; i < WordTraits<W>::kBits / BITS; ++i) m |= W(1) << (i * BITS + BITS - 1);
    return m;
  }
  static constexpr W kValue = mask();
};

// Lane-wise max of two words of spacer-free BITS-bit lanes, flip = the msb
// mask for signed lanes (offset binary orders like two's complement), else
// 0. A lane-wise subtract with the lane MSBs as temporary spacers (section 3,
// Fig. 5) gives each lane's borrow, i.e. x < y, which selects the larger
// lane.
template <typename W, int BITS>
__device__ __forceinline__ W swar_lane_max(W a, W b, W flip) {
  constexpr W M = LaneMsb<W, BITS>::kValue;
  const W x = a ^ flip, y = b ^ flip;
  const W d = ((x ^ y) & M) ^ ((x | M) - (y & ~M)) ^ M;  // lane-wise x - y
  const W lt = ((~x & y) | ((~x | y) & d)) & M;          // borrow out of the lane: x < y
  const W E = (lt - (lt >> (BITS - 1))) | lt;            // whole lanes where x < y
  return (b & E) | (a & ~E);
}

}  // namespace samd

// ---- launchers implemented in the kernel translation units ----------------

namespace samd {
cudaError_t launch_pack(samd_fmt f, const int8_t *src, void *dst, int64_t rows, int64_t inner, cudaStream_t s);
cudaError_t launch_unpack(samd_fmt f, const void *src, int8_t *dst, int64_t rows, int64_t inner, cudaStream_t s);
cudaError_t launch_elementwise(samd_op op, samd_fmt fa, const void *a, const void *b, samd_fmt fo, void *out,
                               int64_t n, int shift, int saturate, cudaStream_t s);
cudaError_t launch_maxpool2x2_nhwc(samd_fmt f, const void *in, void *out, int N, int C, int H, int W,
                                   cudaStream_t s);

samd_status conv2d_check(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw);
samd_status conv2d_prepare(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, const void *wt, samd_fmt fo,
                           void *prepared, size_t prepared_bytes, cudaStream_t s);
samd_status conv2d_run(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, const void *act, const void *prepared,
                       size_t prepared_bytes, int32_t *acc_out, samd_fmt fo, void *packed_out, int shift,
                       cudaStream_t s, void *pooled_out = nullptr);
samd_status conv2d_nhwc(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                        int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, void *workspace,
                        size_t workspace_bytes, cudaStream_t s);
size_t conv2d_workspace_size(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw);
int conv2d_operand_bits(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw);
int conv2d_pool_supported(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo);
void conv2d_set_min_tiles_per_cta(int tiles);
constexpr size_t kNoallocScratchBytes = size_t(8) << 20;  // static scratch of samd_conv2d_noalloc
samd_status conv2d_noalloc(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                                int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, cudaStream_t s);
// NCHW packed along W: the wide-multiply engine of widemul.cu
samd_status conv2d_nchw_check(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo, size_t *ws_bytes);
samd_status conv2d_nchw(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                        int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, void *workspace,
                        size_t workspace_bytes, cudaStream_t s);
cudaError_t read_device_status(int *status, int reset, cudaStream_t s);
cudaError_t selftest_wait_timeout(uint64_t limit_ns, cudaStream_t s);
}  // namespace samd
