/*
 * samd.h -- C ABI of libsamd: bit-precise packed integer tensors on GB300.
 *
 * The operations follow "Scalar Arithmetic Multiple Data: Customizable
 * Precision for Deep Neural Networks" (Anderson, Doyle, Gregg; arXiv
 * 1809.10572). The paper packs b-bit integer lanes into scalar words and
 * computes on all lanes at once (section 2, "Emulating Vector
 * Architectures"); this library keeps that storage format on the GPU and
 * runs the lane arithmetic and the DNN convolution of section 7 (Fig. 12)
 * as CUDA kernels for sm_103a.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - All data pointers are DEVICE pointers owned by the caller; the library
 *   never allocates, frees or keeps them. Every call is asynchronous on the
 *   caller's stream `stream` (a cudaStream_t; NULL means the legacy default
 *   stream) and returns once the work is enqueued.
 * - Arguments are validated on the host before anything is launched. A
 *   non-SAMD_OK status means nothing was launched and no output was
 *   touched, except SAMD_ECUDA, which reports a failed launch.
 * - Data pointers must be 16-byte aligned (SAMD_EALIGN otherwise).
 * - Inputs are assumed canonical (see samd_fmt); outputs are always
 *   canonical.
 * - Sizes of zero are valid and launch nothing.
 *
 * Thread safety: entry points keep no host state except a per-device cache
 * of kernel attributes, guarded by a mutex.
 */
#ifndef SAMD_H_
#define SAMD_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define SAMD_API __attribute__((visibility("default")))
#else
#define SAMD_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without pulling in the CUDA headers. */
typedef struct CUstream_st *samd_stream_t;

typedef enum {
  SAMD_OK = 0,
  SAMD_EINVAL = 1,   /* bad enum, bit width, word width, shift or null pointer */
  SAMD_EALIGN = 2,   /* a data pointer is not 16-byte aligned */
  SAMD_ESHAPE = 3,   /* sizes are negative, inconsistent or overflow */
  SAMD_EUNSUP = 4,   /* valid request outside what the kernels implement */
  SAMD_ECUDA = 5,    /* a CUDA call or kernel launch failed */
  SAMD_ETIMEOUT = 6  /* a kernel gave up on a bounded wait (samd_device_status) */
} samd_status;

/*
 * Packed lane format (section 2.1, the SAMD vector; Fig. 2 for permanent
 * spacer bits).
 *   bits      lane width b, 1..8
 *   is_signed 1: two's complement in b bits (section 6); 0: unsigned
 *   spacer    zero bits kept above every lane, 0..8 (0 = no spacer)
 *   word_bits 32 or 64
 * Lane width w = bits + spacer; L = floor(word_bits / w) lanes per word.
 * A tensor of rows x inner elements is packed row by row; element i of a row
 * is lane (i mod L) of word floor(i / L) of that row, at bit offset
 * (i mod L) * w, least-significant lane first. Every row starts on a word
 * boundary, so a row takes ceil(inner / L) words. Canonical form: spacer
 * bits, the bits above the last whole lane and the lanes past the end of a
 * row are zero. Words are little-endian uint32/uint64.
 */
typedef struct {
  uint8_t bits;
  uint8_t is_signed;
  uint8_t spacer;
  uint8_t word_bits;
} samd_fmt;

/* floor(word_bits / (bits + spacer)), or 0 for an invalid format. */
SAMD_API size_t samd_lanes_per_word(samd_fmt f);

/* rows * ceil(inner / L) words, or -1 for an invalid format or size. */
SAMD_API int64_t samd_packed_words(samd_fmt f, int64_t rows, int64_t inner);

/*
 * samd_pack: src is rows x inner bytes (row-major, one value per byte; the
 * byte's low `bits` bits are kept, so unsigned 8-bit values use the uint8
 * bit pattern); dst receives samd_packed_words(f, rows, inner) words.
 * Section 2.1 (packing lanes into a scalar word); the inverse of the unpack
 * to native 8-bit integers described in section 7.
 */
SAMD_API samd_status samd_pack(samd_fmt f, const int8_t *src, void *dst, int64_t rows, int64_t inner,
                      samd_stream_t stream);

/*
 * samd_unpack: the inverse of samd_pack. Each lane is widened to one byte:
 * sign-extended for signed formats, zero-extended for unsigned ones (an
 * unsigned 8-bit lane fills the byte). Section 7: unpacking sub-8-bit values
 * to the closest native integer type.
 */
SAMD_API samd_status samd_unpack(samd_fmt f, const void *src, int8_t *dst, int64_t rows, int64_t inner,
                        samd_stream_t stream);

typedef enum {
  SAMD_ADD = 0,     /* section 3, Fig. 5: (a + b) mod 2^bits, or clamped if saturate */
  SAMD_SUB = 1,     /* section 3, Fig. 5: (a - b) mod 2^bits, or clamped if saturate */
  SAMD_MUL = 2,     /* section 3, Fig. 6: low bits of a * b (sign-agnostic, section 4.1), or clamped */
  SAMD_RELU = 3,    /* max(a, 0) for signed lanes; a copy for unsigned lanes */
  SAMD_REQUANT = 4  /* clamp_fo(floor(a / 2^shift)) into the output format fo */
} samd_op;

/*
 * samd_elementwise: lane-wise op over n elements packed as one row
 * (rows = 1, inner = n).
 *   a, b, out  packed arrays; b is read only by ADD/SUB/MUL (NULL otherwise)
 *              and has format fa. out may alias a or b.
 *   fo         output format: must equal fa for ADD/SUB/MUL/RELU; REQUANT
 *              may change bits and signedness (same word_bits and spacer).
 *   shift      REQUANT only, 0..31 (arithmetic shift for signed inputs).
 *   saturate   ADD/SUB/MUL: 0 wraps modulo 2^bits, 1 clamps to the lane range.
 */
SAMD_API samd_status samd_elementwise(samd_op op, samd_fmt fa, const void *a, const void *b, samd_fmt fo, void *out,
                             int64_t n, int shift, int saturate, samd_stream_t stream);

typedef enum { SAMD_NCHW = 0, SAMD_NHWC = 1 } samd_layout;

/*
 * Convolution shape. N images of C x H x W, K output channels, R x S taps,
 * one stride and one zero padding for both spatial dims.
 * Ho = (H + 2*pad - R) / stride + 1, Wo = (W + 2*pad - S) / stride + 1.
 */
typedef struct {
  int N, C, H, W;
  int K, R, S;
  int stride, pad;
  samd_layout layout;
} samd_conv_desc;

/*
 * samd_conv2d: the DNN convolution of section 7 (Fig. 12, direct-sum2d),
 * with a batch, stride, zero padding and K output channels:
 *   acc[n][k][ho][wo] = sum_{c,r,s} act[n][c][ho*stride-pad+r][wo*stride-pad+s] * wt[k][c][r][s]
 * (cross-correlation; taps outside the image read zero), computed exactly
 * in int32.
 * Layout SAMD_NHWC (the one implemented): act is N*H*W rows of C elements
 * packed along C with format fa; wt is K*R*S rows of C elements packed
 * along C with format fw ([K][R][S][C]). Outputs, each optional (NULL to
 * skip, but not both):
 *   acc_out     int32 [N][Ho][Wo][K]
 *   packed_out  N*Ho*Wo rows of K elements packed along K with format fo,
 *               each element clamp_fo(floor(acc / 2^shift)) (the requantize
 *               epilogue; an unsigned fo doubles as ReLU).
 * workspace / workspace_bytes: caller-owned device scratch of at least
 * samd_conv2d_workspace_size(...) bytes (16-byte aligned) that receives the
 * weights in the tensor-core operand layout on every call.
 * Exactness: the sum runs on the tensor cores with fp32 accumulation, exact
 * while every partial sum stays below 2^24, over e4m3 operands when
 * max|a| <= 16 and max|w| <= 16 (lanes of up to 4 bits, and signed 5-bit
 * lanes: every such integer is exact in e4m3) and over fp16 operands
 * otherwise (samd_conv2d_operand_bits tells which). If
 * R*S*C * max|a| * max|w| reaches 2^24 and the weights have 5-8 bits, the
 * weights are split into two 4-bit digits (two exact accumulators per
 * output); if R*S*C * max|a| * 16 also reaches 2^24, SAMD_EUNSUP.
 * Scheduling: a layer with less than T x (SM count) reference tiles of work
 * (T = samd_conv2d_set_min_tiles_per_cta, default 4) runs on fewer SMs, each
 * doing at least T reference tiles, so that independent layers issued on
 * other streams run beside it.
 * Other limits (SAMD_EUNSUP): spacer 0 for fa and fw; R, S <= 16.
 * A kernel that gives up on a bounded wait leaves its outputs undefined and
 * records SAMD_ETIMEOUT for samd_device_status.
 */
SAMD_API samd_status samd_conv2d(const samd_conv_desc *desc, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                        int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, void *workspace,
                        size_t workspace_bytes, samd_stream_t stream);

/* Bytes of workspace samd_conv2d needs for this shape and formats, for any
 * output format (0 on error). The same size suffices for
 * samd_conv2d_prepare. */
SAMD_API size_t samd_conv2d_workspace_size(const samd_conv_desc *desc, samd_fmt fa, samd_fmt fw);

/* Minimum work each SM does in one convolution launch, T, in reference
 * tiles: 128 output positions of a 3x3 convolution over 64 input and 64
 * output channels (4.7 M multiply-adds). A layer whose 128-position tiles
 * carry w times that work gets floor(T / w) tiles per SM, at least one
 * (process-wide, all devices, takes effect at the next launch). 1 spreads
 * every layer over all SMs (lowest latency of a single layer); larger values
 * leave SMs free for independent layers launched on other streams (higher
 * throughput when several small layers run at once). Default 4.
 * SAMD_EINVAL for values below 1 or above 1024. */
SAMD_API samd_status samd_conv2d_set_min_tiles_per_cta(int tiles);

/* Width in bits of the tensor-core operands samd_conv2d uses for this shape
 * and these formats: 8 (e4m3), 16 (fp16), or 0 if the convolution is
 * rejected (invalid arguments or SAMD_EUNSUP). Host-only; no GPU needed. */
SAMD_API int samd_conv2d_operand_bits(const samd_conv_desc *desc, samd_fmt fa, samd_fmt fw);

/*
 * Weights prepared once, used by many calls (the weights of an inference
 * layer do not change between batches). samd_conv2d_prepare widens the
 * packed weights wt ([K][R][S][C] along C, format fw) into `prepared`
 * (caller-owned, >= samd_conv2d_workspace_size bytes, 16-byte aligned);
 * samd_conv2d_prepared then runs the convolution of samd_conv2d without
 * touching wt, in one kernel launch. Both calls must get the same desc, fa,
 * fw and fo; fo may be {0,0,0,0} ("no packed output") in both. The
 * prepared buffer is only read by samd_conv2d_prepared, so concurrent calls
 * may share it.
 */
SAMD_API samd_status samd_conv2d_prepare(const samd_conv_desc *desc, samd_fmt fa, samd_fmt fw, const void *wt,
                                         samd_fmt fo, void *prepared, size_t prepared_bytes, samd_stream_t stream);
SAMD_API samd_status samd_conv2d_prepared(const samd_conv_desc *desc, samd_fmt fa, const void *act, samd_fmt fw,
                                          const void *prepared, size_t prepared_bytes, int32_t *acc_out,
                                          samd_fmt fo, void *packed_out, int shift, samd_stream_t stream);

/*
 * samd_conv2d_noalloc: samd_conv2d for callers that cannot allocate device
 * memory -- code that runs where cudaMalloc is off limits (inside a framework
 * that owns every allocation through its own pool, a plugin or real-time
 * path that must not allocate after start-up, a process whose memory pool
 * is already spoken for). The paper has no counterpart; this is an interface
 * convenience. Same arguments and results as samd_conv2d, without the
 * workspace: the widened weights go to a static device array of
 * 8 MiB (8388608 bytes) inside the library, held on every GPU that loads it
 * until the process exits. A call whose widened weights -- for its own desc,
 * fa, fw and output format fo -- need more than 8 MiB (e.g. 3x3
 * convolutions with far more than 512 x 512 channels) is rejected with
 * SAMD_EUNSUP before any launch; samd_conv2d_workspace_size, the largest
 * size over every output format, bounds that need from above, so a layer
 * with samd_conv2d_workspace_size <= 8 MiB is always accepted.
 * The first call in a CUDA context looks the array's device address up
 * (once per context, with that context current; a context created after
 * cudaDeviceReset looks it up again); make that first call before capturing
 * a stream into a CUDA graph. Every call reuses the same array and rewrites
 * the part it reads before reading it, so no earlier contents leak into a
 * result; but calls whose work overlaps on the GPU (different streams, no
 * ordering between them) race on the array: order them on one stream.
 * Neither this call nor anything it calls allocates or frees memory.
 */
SAMD_API samd_status samd_conv2d_noalloc(const samd_conv_desc *desc, samd_fmt fa, const void *act, samd_fmt fw,
                                         const void *wt, int32_t *acc_out, samd_fmt fo, void *packed_out, int shift,
                                         samd_stream_t stream);

/*
 * samd_conv2d_prepared_pool2x2: samd_conv2d_prepared followed by the 2x2
 * max-pool of samd_maxpool2x2, in one kernel (the paper has no pooling; the
 * VGG-16 stack pools after conv2, conv4, conv7, conv10 and conv13). The
 * convolution's packed rows never reach memory: pooled_out receives
 * N*(Ho/2)*(Wo/2) rows of K elements packed along K in format fo, row
 * (n, i, j) holding the lane-wise max over the 2x2 window at output rows
 * 2i, 2i+1 and columns 2j, 2j+1 of clamp_fo(floor(acc / 2^shift)) -- the
 * same words samd_conv2d_prepared and then samd_maxpool2x2 produce.
 * `prepared` is what samd_conv2d_prepare wrote for the same desc, fa, fw and
 * fo. Supported shapes (samd_conv2d_pool2x2_supported, host-only, tells;
 * else SAMD_EUNSUP and nothing is launched): NHWC, stride 1, Ho and Wo even,
 * 2 * (W + 2 * pad) <= 256 (a tile of 256 positions holds whole pairs of
 * padded image rows), fo of 1, 2, 4 or 8 bits in 32-bit words without
 * spacers, and a layer the kernel runs as halo tiles of two halves with
 * room for the tile's packed rows in shared memory. pooled_out: 16-byte
 * aligned, caller-owned.
 */
SAMD_API samd_status samd_conv2d_prepared_pool2x2(const samd_conv_desc *desc, samd_fmt fa, const void *act,
                                                  samd_fmt fw, const void *prepared, size_t prepared_bytes,
                                                  samd_fmt fo, void *pooled_out, int shift, samd_stream_t stream);
/* 1 if samd_conv2d_prepared_pool2x2 supports this shape and these formats,
 * else 0 (invalid arguments included). Host-only; no GPU needed. */
SAMD_API int samd_conv2d_pool2x2_supported(const samd_conv_desc *desc, samd_fmt fa, samd_fmt fw, samd_fmt fo);

/*
 * samd_maxpool2x2: lane-wise max over 2x2 windows with stride 2 (used
 * between the VGG-16 blocks; not in the paper). Layout SAMD_NHWC: in is
 * N*H*W rows of C elements packed along C, out is N*(H/2)*(W/2) rows.
 * H and W must be even.
 */
SAMD_API samd_status samd_maxpool2x2(samd_fmt f, const void *in, void *out, int N, int C, int H, int W,
                            samd_layout layout, samd_stream_t stream);

/*
 * samd_device_status: reads (and with reset=1 clears) the sticky status the
 * kernels of the current device record when a bounded wait runs out.
 * Synchronises `stream`. *status is SAMD_OK or SAMD_ETIMEOUT.
 */
SAMD_API samd_status samd_device_status(int *status, int reset, samd_stream_t stream);

/*
 * samd_selftest_wait_timeout: exercises the failure path of the bounded waits
 * without faulting the GPU. Launches one block on `stream` whose thread waits
 * on an mbarrier phase that nothing completes; after limit_ns nanoseconds
 * (1000 .. 2e9, else SAMD_EINVAL) the wait gives up and records
 * SAMD_ETIMEOUT in the sticky status read by samd_device_status, as a
 * convolution role that gives up does. The context stays usable. Asynchronous.
 */
SAMD_API samd_status samd_selftest_wait_timeout(uint64_t limit_ns, samd_stream_t stream);

/* A static string naming the status. */
SAMD_API const char *samd_status_str(samd_status s);

/* Library version string. */
SAMD_API const char *samd_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SAMD_H_ */
