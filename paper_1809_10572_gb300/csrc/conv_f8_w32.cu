// conv_f8_w32.cu -- instantiates the convolution kernel for e4m3 operands from 32-bit words (lanes with |a| <= 16).
#include "conv_kernel.cuh"

namespace samd {
namespace conv {

cudaError_t launch_conv_f8_w32(int bits, bool is_signed, const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid,
                     size_t smem, cudaStream_t s) {
  switch (bits * 2 + (is_signed ? 1 : 0)) {
    case 2: return launch_conv<uint32_t, 1, false, true>(tmap, args, halo, grid, smem, s);
    case 3: return launch_conv<uint32_t, 1, true, true>(tmap, args, halo, grid, smem, s);
    case 4: return launch_conv<uint32_t, 2, false, true>(tmap, args, halo, grid, smem, s);
    case 5: return launch_conv<uint32_t, 2, true, true>(tmap, args, halo, grid, smem, s);
    case 6: return launch_conv<uint32_t, 3, false, true>(tmap, args, halo, grid, smem, s);
    case 7: return launch_conv<uint32_t, 3, true, true>(tmap, args, halo, grid, smem, s);
    case 8: return launch_conv<uint32_t, 4, false, true>(tmap, args, halo, grid, smem, s);
    case 9: return launch_conv<uint32_t, 4, true, true>(tmap, args, halo, grid, smem, s);
    case 11: return launch_conv<uint32_t, 5, true, true>(tmap, args, halo, grid, smem, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace conv
}  // namespace samd
