// conv_f16_w32b.cu -- instantiates the convolution kernel for fp16 operands from 32-bit words of 5-8-bit lanes.
#include "conv_kernel.cuh"

namespace samd {
namespace conv {

cudaError_t launch_conv_f16_w32b(int bits, bool is_signed, const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid,
                      size_t smem, cudaStream_t s) {
  switch (bits * 2 + (is_signed ? 1 : 0)) {
    case 10: return launch_conv<uint32_t, 5, false, false>(tmap, args, halo, grid, smem, s);
    case 11: return launch_conv<uint32_t, 5, true, false>(tmap, args, halo, grid, smem, s);
    case 12: return launch_conv<uint32_t, 6, false, false>(tmap, args, halo, grid, smem, s);
    case 13: return launch_conv<uint32_t, 6, true, false>(tmap, args, halo, grid, smem, s);
    case 14: return launch_conv<uint32_t, 7, false, false>(tmap, args, halo, grid, smem, s);
    case 15: return launch_conv<uint32_t, 7, true, false>(tmap, args, halo, grid, smem, s);
    case 16: return launch_conv<uint32_t, 8, false, false>(tmap, args, halo, grid, smem, s);
    case 17: return launch_conv<uint32_t, 8, true, false>(tmap, args, halo, grid, smem, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace conv
}  // namespace samd
