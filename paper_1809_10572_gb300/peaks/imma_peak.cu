// imma_peak.cu -- the dense int8 tensor-core rate of the legacy warp-level
// path (mma.sync m16n8k32, s8 x s8 -> s32), measured by a kernel that does
// nothing else: every warp keeps eight independent accumulator tiles in
// registers and issues `iters` rounds of eight MMAs on register operands,
// with no memory traffic inside the loop. This is the denominator of the
// "fraction of int8 tensor-core peak" the convolution is reported against
// (sm_103a has no integer tcgen05.mma, so this is the chip's int8 MMA path).
//
// Built into libsamd_peaks.so, separate from libsamd: it is a measurement
// tool, not part of the hot path.
#include <cuda_runtime.h>

#include <cstdint>

namespace {

constexpr int kChains = 8;

__global__ void __launch_bounds__(256) imma_loop_kernel(int iters, int seed, int *out) {
  // operands from the thread index, so the compiler cannot fold the loop
  uint32_t a0 = 0x01010101u * (threadIdx.x & 7) + seed, a1 = a0 ^ 0x02020202u, a2 = a0 + 3u, a3 = a0 ^ 0x7F7F7F7Fu;
  uint32_t b0 = 0x01000100u + threadIdx.x, b1 = b0 ^ 0x00050005u;
  int d[kChains][4];
#pragma unroll
  for (int c = 0; c < kChains; ++c) d[c][0] = d[c][1] = d[c][2] = d[c][3] = 0;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kChains; ++c) {
      asm volatile(
          "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
          "{%0, %1, %2, %3};"
          : "+r"(d[c][0]), "+r"(d[c][1]), "+r"(d[c][2]), "+r"(d[c][3])
          : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
  }
  int s = 0;
#pragma unroll
  for (int c = 0; c < kChains; ++c) s += d[c][0] ^ d[c][1] ^ d[c][2] ^ d[c][3];
  if (s == 0x12345678) out[0] = s;  // keeps the results live; practically never taken
}

// A binary path for 1-2-bit lanes: mma.sync m16n8k256 on b1
// operands with AND + popcount accumulation into s32 (a 1-bit x 1-bit
// product per bit pair). A b-bit x b-bit multiply-add built from bit planes
// takes b^2 of these products, so this rate bounds such a convolution.
__global__ void __launch_bounds__(256) bmma_loop_kernel(int iters, int seed, int *out) {
  uint32_t a0 = 0x9E3779B9u * (threadIdx.x + 1) + seed, a1 = a0 ^ 0x5A5A5A5Au, a2 = a0 + 0x01234567u,
           a3 = ~a0;
  uint32_t b0 = 0x7F4A7C15u ^ threadIdx.x, b1 = b0 * 3u;
  int d[kChains][4];
#pragma unroll
  for (int c = 0; c < kChains; ++c) d[c][0] = d[c][1] = d[c][2] = d[c][3] = 0;
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < kChains; ++c) {
      asm volatile(
          "mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.and.popc {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
          "{%8, %9}, {%0, %1, %2, %3};"
          : "+r"(d[c][0]), "+r"(d[c][1]), "+r"(d[c][2]), "+r"(d[c][3])
          : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    }
  }
  int s = 0;
#pragma unroll
  for (int c = 0; c < kChains; ++c) s += d[c][0] ^ d[c][1] ^ d[c][2] ^ d[c][3];
  if (s == 0x12345678) out[0] = s;
}

using LoopKernel = void (*)(int, int, int *);

int time_loop(LoopKernel k, int blocks, int iters, int *scratch, float *ms) {
  cudaEvent_t e0, e1;
  cudaError_t e = cudaEventCreate(&e0);
  if (e != cudaSuccess) return static_cast<int>(e);
  e = cudaEventCreate(&e1);
  if (e != cudaSuccess) {
    cudaEventDestroy(e0);
    return static_cast<int>(e);
  }
  k<<<blocks, 256>>>(iters, 1, scratch);
  cudaEventRecord(e0);
  k<<<blocks, 256>>>(iters, 2, scratch);
  cudaEventRecord(e1);
  e = cudaEventSynchronize(e1);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaEventElapsedTime(ms, e0, e1);
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  return static_cast<int>(e);
}

}  // namespace

extern "C" {

// Runs the loop kernel on `blocks` blocks of 256 threads, `iters` rounds,
// on the current device and the legacy default stream, timed with CUDA
// events after one warm-up launch. Writes the kernel time in milliseconds
// and the number of multiply-adds it performed (16 x 8 x 32 per MMA).
// `scratch` is a device int that the kernel may write. Returns 0 on success,
// else the CUDA error code.
__attribute__((visibility("default"))) int samd_peak_imma_s8(int blocks, int iters, int *scratch, float *ms,
                                                             double *macs) {
  if (blocks < 1 || iters < 1 || !scratch || !ms || !macs) return static_cast<int>(cudaErrorInvalidValue);
  *macs = static_cast<double>(blocks) * (256 / 32) * static_cast<double>(iters) * kChains * 16.0 * 8.0 * 32.0;
  return time_loop(imma_loop_kernel, blocks, iters, scratch, ms);
}

// The same for the binary MMA (m16n8k256 b1, AND + popcount): `ops` is the
// number of 1-bit x 1-bit products (16 x 8 x 256 per MMA).
__attribute__((visibility("default"))) int samd_peak_bmma_b1(int blocks, int iters, int *scratch, float *ms,
                                                             double *ops) {
  if (blocks < 1 || iters < 1 || !scratch || !ms || !ops) return static_cast<int>(cudaErrorInvalidValue);
  *ops = static_cast<double>(blocks) * (256 / 32) * static_cast<double>(iters) * kChains * 16.0 * 8.0 * 256.0;
  return time_loop(bmma_loop_kernel, blocks, iters, scratch, ms);
}

}  // extern "C"
