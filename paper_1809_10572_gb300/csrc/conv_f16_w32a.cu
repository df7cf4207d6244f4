// conv_f16_w32a.cu -- instantiates the convolution kernel for fp16 operands from 32-bit words of 1-4-bit lanes.
#include "conv_kernel.cuh"

namespace samd {
namespace conv {

cudaError_t launch_conv_f16_w32a(int bits, bool is_signed, const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid,
                      size_t smem, cudaStream_t s) {
  switch (bits * 2 + (is_signed ? 1 : 0)) {
    case 2: return launch_conv<uint32_t, 1, false, false>(tmap, args, halo, grid, smem, s);
    case 3: return launch_conv<uint32_t, 1, true, false>(tmap, args, halo, grid, smem, s);
    case 4: return launch_conv<uint32_t, 2, false, false>(tmap, args, halo, grid, smem, s);
    case 5: return launch_conv<uint32_t, 2, true, false>(tmap, args, halo, grid, smem, s);
    case 6: return launch_conv<uint32_t, 3, false, false>(tmap, args, halo, grid, smem, s);
    case 7: return launch_conv<uint32_t, 3, true, false>(tmap, args, halo, grid, smem, s);
    case 8: return launch_conv<uint32_t, 4, false, false>(tmap, args, halo, grid, smem, s);
    case 9: return launch_conv<uint32_t, 4, true, false>(tmap, args, halo, grid, smem, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace conv
}  // namespace samd
