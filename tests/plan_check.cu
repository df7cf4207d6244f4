// Host-only check of the convolution planner (conv2d.cu's make_plan and
// layout_ok) over a grid of shapes and formats: every plan it accepts fits
// the shared-memory and TMEM limits and its halo, staging and barrier areas
// do not overlap. Compiled and run by tests/test_plan_cpu.py; the kernel
// launchers are replaced by stubs (nothing is launched).
#include "../paper_1809_10572_gb300/csrc/conv2d.cu"

#define SAMD_STUB(name)                                                                                      \
  namespace samd {                                                                                           \
  namespace conv {                                                                                           \
  cudaError_t name(bool, const CUtensorMap &, const ConvArgs &, bool, dim3, size_t, cudaStream_t) {          \
    return cudaErrorInvalidValue;                                                                            \
  }                                                                                                          \
  }                                                                                                          \
  }
SAMD_STUB(launch_conv_f16_w32_b1) SAMD_STUB(launch_conv_f16_w32_b2) SAMD_STUB(launch_conv_f16_w32_b3)
SAMD_STUB(launch_conv_f16_w32_b4) SAMD_STUB(launch_conv_f16_w32_b5) SAMD_STUB(launch_conv_f16_w32_b6)
SAMD_STUB(launch_conv_f16_w32_b7) SAMD_STUB(launch_conv_f16_w32_b8) SAMD_STUB(launch_conv_f16_w64_b1)
SAMD_STUB(launch_conv_f16_w64_b2) SAMD_STUB(launch_conv_f16_w64_b3) SAMD_STUB(launch_conv_f16_w64_b4)
SAMD_STUB(launch_conv_f16_w64_b5) SAMD_STUB(launch_conv_f16_w64_b6) SAMD_STUB(launch_conv_f16_w64_b7)
SAMD_STUB(launch_conv_f16_w64_b8) SAMD_STUB(launch_conv_f8_w32_b1) SAMD_STUB(launch_conv_f8_w32_b2)
SAMD_STUB(launch_conv_f8_w32_b3) SAMD_STUB(launch_conv_f8_w32_b4) SAMD_STUB(launch_conv_f8_w32_b5)
SAMD_STUB(launch_conv_f8_w64_b1) SAMD_STUB(launch_conv_f8_w64_b2) SAMD_STUB(launch_conv_f8_w64_b3)
SAMD_STUB(launch_conv_f8_w64_b4) SAMD_STUB(launch_conv_f8_w64_b5)

namespace samd {
int sm_count() { return 152; }  // defined in samd_api.cu, not linked here
// the NCHW path lives in widemul.cu, not linked here
samd_status conv2d_nchw_check(const samd_conv_desc *, samd_fmt, samd_fmt, samd_fmt, size_t *) { return SAMD_EUNSUP; }
samd_status conv2d_nchw(const samd_conv_desc *, samd_fmt, const void *, samd_fmt, const void *, int32_t *, samd_fmt,
                        void *, int, void *, size_t, cudaStream_t) {
  return SAMD_EUNSUP;
}
}  // namespace samd

#include <cstdio>

int main() {
  using namespace samd;
  long long n = 0, bad = 0, halo = 0, seg = 0, fp8 = 0, res = 0, unsup = 0, hv2 = 0, win = 0, deep = 0, estg = 0, hv4 = 0;
  const int Cs[] = {1, 3, 16, 24, 64, 96, 128, 256, 512, 1024};
  const int Ks[] = {1, 16, 40, 64, 96, 128, 256, 300, 512, 1024};
  const int HWs[] = {1, 2, 7, 14, 28, 56, 224};
  for (int wb : {32, 64})
    for (int ba = 1; ba <= 8; ++ba)
      for (int sa = 0; sa < 2; ++sa)
        for (int bw = 1; bw <= 8; bw += (bw < 2 ? 1 : 2))
          for (int sw = 0; sw < 2; ++sw)
            for (int C : Cs)
              for (int K : Ks)
                for (int hw : HWs)
                  for (int rs : {1, 3, 5})
                    for (int st : {1, 2}) {
                      if (rs > hw + 2) continue;
                      samd_conv_desc d{hw >= 112 ? 16 : 2, C, hw, hw, K, rs, rs, st, rs / 2, SAMD_NHWC};  // batch 16 for large images (four-part tiles)
                      samd_fmt fa{(uint8_t)ba, (uint8_t)sa, 0, (uint8_t)wb};
                      samd_fmt fw{(uint8_t)bw, (uint8_t)sw, 0, (uint8_t)wb};
                      for (int fob : {0, 3, 4, 6}) {
                        samd_fmt fo{(uint8_t)fob, 0, 0, 32};
                        conv::Plan p;
                        const samd_status s = conv::make_plan(&d, fa, fw, fo, p);
                        ++n;
                        if (s != SAMD_OK) {
                          ++unsup;
                          continue;
                        }
                        if (p.M == 0) continue;
                        bool ok = conv::layout_ok(p) && p.smem_bytes <= 227 * 1024;
                        if (p.halo) {
                          ++halo;
                          if (p.nseg > 1) ++seg;
                          const int maxrow = (d.R - 1) * p.row_step + (d.S - 1) + 128 * p.hv - 1;
                          const int srow = (p.WC * wb / 8 + 15) / 16 * 16;
                          ok = ok && maxrow < p.nseg * p.seg_rows &&
                               p.nseg * p.seg_rows * static_cast<long long>(p.row_bytes) <= p.op_stride &&
                               p.gdepth >= 2 && p.gdepth <= 4 &&
                               static_cast<long long>(p.nseg) * p.seg_rows * srow <= p.g_stride;
                          if (p.gdepth == conv::kHaloGatherDepth) ++deep;
                        } else {
                          // gather staging: a producer group's ring of kGatherDepth x 128 rows
                          const int chunk_bytes = p.WC * wb / 8;
                          const int srow = (chunk_bytes + 15) / 16 * 16;
                          ok = ok && p.g_row >= srow && p.g_row % 16 == 0 &&
                               p.g_stride >= static_cast<uint32_t>(conv::kGatherDepth * conv::BM * p.g_row);
                          if (p.gather_win) {
                            ++win;
                            // (channel chunk, tap) chunks, each inside one pixel
                            ok = ok && p.g_row >= srow + 16 && (p.g_row / 16) % 2 == 1 &&
                                 p.nchunks == p.nck * p.taps && p.nck * p.WC >= p.wpr && (p.nck - 1) * p.WC < p.wpr;
                          }
                        }
                        if (p.fp8) ++fp8;
                        if (p.b_resident) ++res;
                        if (p.hv == 2) ++hv2;
                        if (p.hv == 4) ++hv4;
                        ok = ok && p.tmem_cols <= 512 && 2 * p.hv * p.mma_n <= static_cast<int>(p.tmem_cols);
                        if (p.e_stage) {
                          ++estg;
                          ok = ok && (fob == 3 || fob == 5 || fob == 6) && p.off_e + conv::kEpiStageBytes <= p.off_bar;
                        }
                        if (!ok && ++bad < 10)
                          printf("BAD C%d K%d hw%d rs%d st%d a%d%d w%d%d wb%d fo%d: smem %zu stages %d sta %d\n", C, K,
                                 hw, rs, st, ba, sa, bw, sw, wb, fob, p.smem_bytes, p.stages, p.stages_a);
                      }
                    }
  printf("plans %lld, bad %lld, unsupported %lld, halo %lld (segmented %lld), e4m3 %lld, resident %lld, "
         "two-half %lld, four-part %lld, window gather %lld, staging at the chosen depth %lld, staged epilogue %lld\n",
         n, bad, unsup, halo, seg, fp8, res, hv2, hv4, win, deep, estg);
  return bad != 0;
}
