// conv_f16_w64.cu -- instantiates the convolution kernel for fp16 operands from 64-bit words.
#include "conv_kernel.cuh"

namespace samd {
namespace conv {

cudaError_t launch_conv_f16_w64(int bits, bool is_signed, const CUtensorMap &tmap, const ConvArgs &args, bool halo, dim3 grid,
                      size_t smem, cudaStream_t s) {
  switch (bits * 2 + (is_signed ? 1 : 0)) {
    case 2: return launch_conv<uint64_t, 1, false, false>(tmap, args, halo, grid, smem, s);
    case 3: return launch_conv<uint64_t, 1, true, false>(tmap, args, halo, grid, smem, s);
    case 4: return launch_conv<uint64_t, 2, false, false>(tmap, args, halo, grid, smem, s);
    case 5: return launch_conv<uint64_t, 2, true, false>(tmap, args, halo, grid, smem, s);
    case 6: return launch_conv<uint64_t, 3, false, false>(tmap, args, halo, grid, smem, s);
    case 7: return launch_conv<uint64_t, 3, true, false>(tmap, args, halo, grid, smem, s);
    case 8: return launch_conv<uint64_t, 4, false, false>(tmap, args, halo, grid, smem, s);
    case 9: return launch_conv<uint64_t, 4, true, false>(tmap, args, halo, grid, smem, s);
    case 10: return launch_conv<uint64_t, 5, false, false>(tmap, args, halo, grid, smem, s);
    case 11: return launch_conv<uint64_t, 5, true, false>(tmap, args, halo, grid, smem, s);
    case 12: return launch_conv<uint64_t, 6, false, false>(tmap, args, halo, grid, smem, s);
    case 13: return launch_conv<uint64_t, 6, true, false>(tmap, args, halo, grid, smem, s);
    case 14: return launch_conv<uint64_t, 7, false, false>(tmap, args, halo, grid, smem, s);
    case 15: return launch_conv<uint64_t, 7, true, false>(tmap, args, halo, grid, smem, s);
    case 16: return launch_conv<uint64_t, 8, false, false>(tmap, args, halo, grid, smem, s);
    case 17: return launch_conv<uint64_t, 8, true, false>(tmap, args, halo, grid, smem, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace conv
}  // namespace samd
