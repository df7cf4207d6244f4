// samd_api.cu -- the extern "C" entry points of libsamd: argument checks on
// the host, then one launch (or two, for the convolution) on the caller's
// stream. See include/samd.h for the contract of each call.
#include <mutex>

#include "samd_internal.cuh"

namespace samd {

int sm_count() {
  static std::mutex mu;
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev] == 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    cache[dev] = n;
  }
  return cache[dev];
}

namespace {

samd_status from_cuda(cudaError_t e) { return e == cudaSuccess ? SAMD_OK : SAMD_ECUDA; }

bool shape_ok(int64_t rows, int64_t inner) { return rows >= 0 && inner >= 0 && (rows == 0 || inner <= INT64_MAX / rows); }

}  // namespace
}  // namespace samd

using namespace samd;

extern "C" {

size_t samd_lanes_per_word(samd_fmt f) { return static_cast<size_t>(lanes_per_word(f)); }

int64_t samd_packed_words(samd_fmt f, int64_t rows, int64_t inner) {
  if (!fmt_valid(f) || !shape_ok(rows, inner)) return -1;
  return rows * words_per_row(f, inner);
}

samd_status samd_pack(samd_fmt f, const int8_t *src, void *dst, int64_t rows, int64_t inner, samd_stream_t stream) {
  if (!fmt_valid(f)) return SAMD_EINVAL;
  if (!shape_ok(rows, inner)) return SAMD_ESHAPE;
  if (rows == 0 || inner == 0) return SAMD_OK;
  if (!src || !dst) return SAMD_EINVAL;
  if (!aligned16(src) || !aligned16(dst)) return SAMD_EALIGN;
  return from_cuda(launch_pack(f, src, dst, rows, inner, reinterpret_cast<cudaStream_t>(stream)));
}

samd_status samd_unpack(samd_fmt f, const void *src, int8_t *dst, int64_t rows, int64_t inner,
                        samd_stream_t stream) {
  if (!fmt_valid(f)) return SAMD_EINVAL;
  if (!shape_ok(rows, inner)) return SAMD_ESHAPE;
  if (rows == 0 || inner == 0) return SAMD_OK;
  if (!src || !dst) return SAMD_EINVAL;
  if (!aligned16(src) || !aligned16(dst)) return SAMD_EALIGN;
  return from_cuda(launch_unpack(f, src, dst, rows, inner, reinterpret_cast<cudaStream_t>(stream)));
}

samd_status samd_elementwise(samd_op op, samd_fmt fa, const void *a, const void *b, samd_fmt fo, void *out,
                             int64_t n, int shift, int saturate, samd_stream_t stream) {
  if (op < SAMD_ADD || op > SAMD_REQUANT) return SAMD_EINVAL;
  if (!fmt_valid(fa) || !fmt_valid(fo)) return SAMD_EINVAL;
  if (saturate != 0 && saturate != 1) return SAMD_EINVAL;
  if (op == SAMD_REQUANT) {
    if (shift < 0 || shift > 31) return SAMD_EINVAL;
  } else if (!same_fmt(fa, fo)) {
    return SAMD_EINVAL;
  }
  if (n < 0) return SAMD_ESHAPE;
  if (n == 0) return SAMD_OK;
  const bool binary = op == SAMD_ADD || op == SAMD_SUB || op == SAMD_MUL;
  if (!a || !out || (binary && !b)) return SAMD_EINVAL;
  if (!aligned16(a) || !aligned16(out) || (binary && !aligned16(b))) return SAMD_EALIGN;
  return from_cuda(launch_elementwise(op, fa, a, binary ? b : nullptr, fo, out, n, op == SAMD_REQUANT ? shift : 0,
                                      binary ? saturate : 0, reinterpret_cast<cudaStream_t>(stream)));
}

size_t samd_conv2d_workspace_size(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw) {
  if (!d || !fmt_valid(fa) || !fmt_valid(fw)) return 0;
  if (d->N < 0 || d->C < 1 || d->H < 1 || d->W < 1 || d->K < 1 || d->R < 1 || d->S < 1 || d->stride < 1 ||
      d->pad < 0)
    return 0;
  if (d->layout == SAMD_NCHW) {
    size_t ws = 0;
    if (fa.spacer != 0 || fw.spacer != 0 || d->R > 16 || d->S > 16) return 0;
    return conv2d_nchw_check(d, fa, fw, samd_fmt{0, 0, 0, 0}, &ws) == SAMD_OK ? ws : 0;
  }
  if (d->layout != SAMD_NHWC) return 0;
  return conv2d_workspace_size(d, fa, fw);
}

samd_status samd_conv2d_set_min_tiles_per_cta(int tiles) {
  if (tiles < 1 || tiles > 1024) return SAMD_EINVAL;
  conv2d_set_min_tiles_per_cta(tiles);
  return SAMD_OK;
}

int samd_conv2d_operand_bits(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw) {
  if (!d || !fmt_valid(fa) || !fmt_valid(fw) || fa.spacer != 0 || fw.spacer != 0) return 0;
  if (d->N < 0 || d->C < 1 || d->H < 1 || d->W < 1 || d->K < 1 || d->R < 1 || d->S < 1 || d->stride < 1 ||
      d->pad < 0 || d->R > 16 || d->S > 16)
    return 0;
  if (d->layout == SAMD_NCHW) return conv2d_nchw_check(d, fa, fw, samd_fmt{0, 0, 0, 0}, nullptr) == SAMD_OK ? 64 : 0;
  if (d->layout != SAMD_NHWC) return 0;
  return conv2d_operand_bits(d, fa, fw);
}

namespace {
// Checks shared by the three convolution entry points. fo.bits == 0 means no
// packed output format.
samd_status conv_common_checks(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo, int shift) {
  if (!d) return SAMD_EINVAL;
  if (!fmt_valid(fa) || !fmt_valid(fw)) return SAMD_EINVAL;
  if (fo.bits != 0 && !fmt_valid(fo)) return SAMD_EINVAL;
  if (shift < 0 || shift > 31) return SAMD_EINVAL;
  if (d->layout != SAMD_NHWC && d->layout != SAMD_NCHW) return SAMD_EINVAL;
  if (d->N < 0 || d->C < 1 || d->H < 1 || d->W < 1 || d->K < 1 || d->R < 1 || d->S < 1 || d->stride < 1 ||
      d->pad < 0)
    return SAMD_ESHAPE;
  if (d->H + 2 * d->pad < d->R || d->W + 2 * d->pad < d->S) return SAMD_ESHAPE;
  if (fa.spacer != 0 || fw.spacer != 0) return SAMD_EUNSUP;
  if (d->R > 16 || d->S > 16) return SAMD_EUNSUP;
  if (d->layout == SAMD_NCHW) return conv2d_nchw_check(d, fa, fw, fo, nullptr);  // wide-multiply engine limits
  return conv2d_check(d, fa, fw);  // exactness bound of the accumulation
}
}  // namespace

samd_status samd_conv2d(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                        int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, void *workspace,
                        size_t workspace_bytes, samd_stream_t stream) {
  if (!acc_out && !packed_out) return SAMD_EINVAL;
  const samd_fmt fplan = packed_out ? fo : samd_fmt{0, 0, 0, 0};
  samd_status st = conv_common_checks(d, fa, fw, fplan, packed_out ? shift : 0);
  if (st != SAMD_OK) return st;
  if (d->N == 0) return SAMD_OK;
  if (!act || !wt || !workspace) return SAMD_EINVAL;
  if (!aligned16(act) || !aligned16(wt) || !aligned16(workspace) || (acc_out && !aligned16(acc_out)) ||
      (packed_out && !aligned16(packed_out)))
    return SAMD_EALIGN;
  if (d->layout == SAMD_NCHW)
    return conv2d_nchw(d, fa, act, fw, wt, acc_out, fo, packed_out, shift, workspace, workspace_bytes,
                       reinterpret_cast<cudaStream_t>(stream));
  return conv2d_nhwc(d, fa, act, fw, wt, acc_out, fo, packed_out, shift, workspace, workspace_bytes,
                     reinterpret_cast<cudaStream_t>(stream));
}

samd_status samd_conv2d_noalloc(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                                int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, samd_stream_t stream) {
  if (!acc_out && !packed_out) return SAMD_EINVAL;
  const samd_fmt fplan = packed_out ? fo : samd_fmt{0, 0, 0, 0};
  samd_status st = conv_common_checks(d, fa, fw, fplan, packed_out ? shift : 0);
  if (st != SAMD_OK) return st;
  if (d->N == 0) return SAMD_OK;
  if (!act || !wt) return SAMD_EINVAL;
  if (!aligned16(act) || !aligned16(wt) || (acc_out && !aligned16(acc_out)) ||
      (packed_out && !aligned16(packed_out)))
    return SAMD_EALIGN;
  return conv2d_noalloc(d, fa, act, fw, wt, acc_out, fo, packed_out, shift,
                             reinterpret_cast<cudaStream_t>(stream));
}

samd_status samd_conv2d_prepare(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, const void *wt, samd_fmt fo,
                                void *prepared, size_t prepared_bytes, samd_stream_t stream) {
  samd_status st = conv_common_checks(d, fa, fw, fo, 0);
  if (st != SAMD_OK) return st;
  if (d->layout != SAMD_NHWC) return SAMD_EUNSUP;  // the NCHW engine widens its operands on every call
  if (!wt || !prepared) return SAMD_EINVAL;
  if (!aligned16(wt) || !aligned16(prepared)) return SAMD_EALIGN;
  return conv2d_prepare(d, fa, fw, wt, fo, prepared, prepared_bytes, reinterpret_cast<cudaStream_t>(stream));
}

samd_status samd_conv2d_prepared(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw,
                                 const void *prepared, size_t prepared_bytes, int32_t *acc_out, samd_fmt fo,
                                 void *packed_out, int shift, samd_stream_t stream) {
  if (!acc_out && !packed_out) return SAMD_EINVAL;
  if (packed_out && fo.bits == 0) return SAMD_EINVAL;
  samd_status st = conv_common_checks(d, fa, fw, fo, packed_out ? shift : 0);
  if (st != SAMD_OK) return st;
  if (d->layout != SAMD_NHWC) return SAMD_EUNSUP;
  if (d->N == 0) return SAMD_OK;
  if (!act || !prepared) return SAMD_EINVAL;
  if (!aligned16(act) || !aligned16(prepared) || (acc_out && !aligned16(acc_out)) ||
      (packed_out && !aligned16(packed_out)))
    return SAMD_EALIGN;
  return conv2d_run(d, fa, fw, act, prepared, prepared_bytes, acc_out, fo, packed_out, shift,
                    reinterpret_cast<cudaStream_t>(stream));
}

samd_status samd_conv2d_prepared_pool2x2(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw,
                                         const void *prepared, size_t prepared_bytes, samd_fmt fo, void *pooled_out,
                                         int shift, samd_stream_t stream) {
  if (!pooled_out || fo.bits == 0) return SAMD_EINVAL;
  samd_status st = conv_common_checks(d, fa, fw, fo, shift);
  if (st != SAMD_OK) return st;
  if (d->layout != SAMD_NHWC) return SAMD_EUNSUP;
  if (d->N == 0) return SAMD_OK;
  if (!conv2d_pool_supported(d, fa, fw, fo)) return SAMD_EUNSUP;
  if (!act || !prepared) return SAMD_EINVAL;
  if (!aligned16(act) || !aligned16(prepared) || !aligned16(pooled_out)) return SAMD_EALIGN;
  return conv2d_run(d, fa, fw, act, prepared, prepared_bytes, nullptr, fo, nullptr, shift,
                    reinterpret_cast<cudaStream_t>(stream), pooled_out);
}

int samd_conv2d_pool2x2_supported(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo) {
  if (!d || fo.bits == 0 || conv_common_checks(d, fa, fw, fo, 0) != SAMD_OK || d->layout != SAMD_NHWC) return 0;
  return conv2d_pool_supported(d, fa, fw, fo);
}

samd_status samd_maxpool2x2(samd_fmt f, const void *in, void *out, int N, int C, int H, int W, samd_layout layout,
                            samd_stream_t stream) {
  if (!fmt_valid(f)) return SAMD_EINVAL;
  if (layout != SAMD_NHWC && layout != SAMD_NCHW) return SAMD_EINVAL;
  if (N < 0 || C < 1 || H < 2 || W < 2 || (H & 1) || (W & 1)) return SAMD_ESHAPE;
  if (layout != SAMD_NHWC) return SAMD_EUNSUP;
  if (N == 0) return SAMD_OK;
  if (!in || !out) return SAMD_EINVAL;
  if (!aligned16(in) || !aligned16(out)) return SAMD_EALIGN;
  return from_cuda(launch_maxpool2x2_nhwc(f, in, out, N, C, H, W, reinterpret_cast<cudaStream_t>(stream)));
}

samd_status samd_device_status(int *status, int reset, samd_stream_t stream) {
  if (!status) return SAMD_EINVAL;
  return from_cuda(read_device_status(status, reset, reinterpret_cast<cudaStream_t>(stream)));
}

samd_status samd_selftest_wait_timeout(uint64_t limit_ns, samd_stream_t stream) {
  if (limit_ns < 1000ull || limit_ns > 2000000000ull) return SAMD_EINVAL;
  return from_cuda(selftest_wait_timeout(limit_ns, reinterpret_cast<cudaStream_t>(stream)));
}

const char *samd_status_str(samd_status s) {
  switch (s) {
    case SAMD_OK: return "SAMD_OK";
    case SAMD_EINVAL: return "SAMD_EINVAL: invalid argument";
    case SAMD_EALIGN: return "SAMD_EALIGN: pointer not 16-byte aligned";
    case SAMD_ESHAPE: return "SAMD_ESHAPE: invalid or inconsistent sizes";
    case SAMD_EUNSUP: return "SAMD_EUNSUP: not supported by the kernels";
    case SAMD_ECUDA: return "SAMD_ECUDA: CUDA error";
    case SAMD_ETIMEOUT: return "SAMD_ETIMEOUT: a kernel gave up on a bounded wait";
  }
  return "unknown samd_status";
}

const char *samd_version(void) { return "samd-gb300 0.1 (sm_103a)"; }

}  // extern "C"
