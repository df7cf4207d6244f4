// conv_inst.cu -- one instantiation unit of the convolution kernel. The build
// compiles this file once per (operand type, activation word width, lane
// width), selected by SAMD_INST_FP8 (0: fp16, 1: e4m3), SAMD_INST_WB (32 or
// 64) and SAMD_INST_BITS (1..8), so that the units compile in parallel.
// Without those macros it compiles to nothing.
#include "conv_kernel.cuh"

#if defined(SAMD_INST_FP8) && defined(SAMD_INST_WB) && defined(SAMD_INST_BITS)

namespace samd {
namespace conv {

#define SAMD_CAT2(a, b, c) launch_conv_##a##_w##b##_b##c
#define SAMD_CAT(a, b, c) SAMD_CAT2(a, b, c)  // expands the arguments first
#if SAMD_INST_FP8
#define SAMD_INST_FN SAMD_CAT(f8, SAMD_INST_WB, SAMD_INST_BITS)
#else
#define SAMD_INST_FN SAMD_CAT(f16, SAMD_INST_WB, SAMD_INST_BITS)
#endif

cudaError_t SAMD_INST_FN(bool is_signed, const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid,
                         size_t smem, cudaStream_t s) {
  using W = std::conditional_t<SAMD_INST_WB == 64, uint64_t, uint32_t>;
  constexpr bool kFp8 = SAMD_INST_FP8 != 0;
  constexpr int kBits = SAMD_INST_BITS;
  // e4m3 holds unsigned lanes of up to 4 bits and signed lanes of up to 5
  if (is_signed) return launch_conv<W, kBits, true, kFp8>(tmap, args, halo, grid, smem, s);
  if constexpr (!kFp8 || kBits <= 4) return launch_conv<W, kBits, false, kFp8>(tmap, args, halo, grid, smem, s);
  return cudaErrorInvalidValue;
}

}  // namespace conv
}  // namespace samd

#endif
