// conv2d.cu -- host side of the bit-precise convolution: planning (operand
// type, tiling, halo geometry, shared-memory carve-up), weight widening into
// the prepared workspace, and the launch. The kernel is in conv_kernel.cuh.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include <atomic>
#include <cstring>
#include <mutex>

#include "conv_kernel.cuh"

namespace samd {

// Sticky record of a bounded wait that ran out (SAMD_ETIMEOUT), per device.
__device__ int g_conv_status;

// Scratch of samd_conv2d_noalloc: the widened weights of one layer. Every GPU
// that loads the library holds these bytes until the process exits.
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

namespace conv {

// Identity of the current CUDA context (cuCtxGetId), unique for the life of
// the process: a cache entry made for one context is never taken for a
// context created later, such as the primary context a device gets again
// after cudaDeviceReset (which reloads the module: kernel attributes and
// symbol addresses change). If the runtime has not made a context current
// yet, cudaSetDevice makes the device's primary context current (no
// allocation).
cudaError_t current_context_id(unsigned long long *id) {
  using GetCurrentFn = CUresult (*)(CUcontext *);
  using GetIdFn = CUresult (*)(CUcontext, unsigned long long *);
  static GetCurrentFn get_current = nullptr;
  static GetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 4000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<GetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<GetIdFn>(p);
  });
  if (!get_current || !get_id) return cudaErrorNotSupported;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
  if (!ctx) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaSetDevice(dev);
    if (e != cudaSuccess) return e;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return cudaErrorDeviceUninitialized;
  }
  return get_id(ctx, id) == CUDA_SUCCESS ? cudaSuccess : cudaErrorDeviceUninitialized;
}

// cudaFuncSetAttribute once per (kernel, context), so that launches made
// while a stream is being captured into a graph issue no other CUDA call.
// The dynamic limit is the per-block maximum minus the kernel's static
// shared memory. Returns cudaErrorInvalidValue if `smem` does not fit.
cudaError_t ensure_smem_attr(const void *kern, size_t smem) {
  constexpr int kSlots = 512;
  static std::mutex mu;
  static const void *done_fn[kSlots];
  static unsigned long long done_ctx[kSlots];
  static size_t done_smem[kSlots];
  static int n_done = 0, next_slot = 0;
  unsigned long long ctx = 0;
  cudaError_t e = current_context_id(&ctx);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < n_done; ++i)
    if (done_fn[i] == kern && done_ctx[i] == ctx) return smem <= done_smem[i] ? cudaSuccess : cudaErrorInvalidValue;
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  int optin = 0;
  e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  cudaFuncAttributes fa;
  e = cudaFuncGetAttributes(&fa, kern);
  if (e != cudaSuccess) return e;
  const size_t limit = static_cast<size_t>(optin) - fa.sharedSizeBytes;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(limit));
  if (e != cudaSuccess) return e;
  const int slot = n_done < kSlots ? n_done++ : next_slot;  // when full, entries are replaced in turn
  if (n_done == kSlots) next_slot = (slot + 1) % kSlots;
  done_fn[slot] = kern;
  done_ctx[slot] = ctx;
  done_smem[slot] = limit;
  return smem <= limit ? cudaSuccess : cudaErrorInvalidValue;
}

namespace {

// ---- weight widening into the workspace ----------------------------------

struct WPrepArgs {
  int K, C, RS;
  int bits_w, signed_w, lane_w_w, Lw, wpr_w;  // weight format
  int bits_a, signed_a, fp8, La, WC, wpr_a, words_total;  // reduction order set by the activation format
  int Kpad, n_mma, mma_n, NBc, split;
  int halo, taps;  // halo: reduction order (chunk, tap, position); else (tap-major words, position)
  long long rows_total;
};

// an integer |v| <= 16 as e4m3 (exact)
__device__ __forceinline__ uint8_t int_to_e4m3(int v) {
  const float f = static_cast<float>(v);
  uint16_t r;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(f), "f"(f));
  return static_cast<uint8_t>(r & 0xFF);
}

// B[row][kpos] for row = nb * mma_n + (plane, output channel), kpos over the
// reduction order of the activation operand; every element of every tile is
// written (zeros in padding), so nothing left over in the workspace is read.
template <typename WW, bool FP8>
__global__ void __launch_bounds__(256) wprep_kernel(const WW *__restrict__ wt, void *__restrict__ Bv,
                                                    const WPrepArgs a) {
  const long long total = a.rows_total * a.Kpad;
  const uint32_t mask = (1u << a.bits_w) - 1;
  for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
       idx += (long long)gridDim.x * blockDim.x) {
    const long long rowi = idx / a.Kpad;
    const int kpos = static_cast<int>(idx - rowi * a.Kpad);
    const int nb = static_cast<int>(rowi / a.mma_n), rb = static_cast<int>(rowi % a.mma_n);
    const int plane = a.split ? rb / a.n_mma : -1;  // 0: high digit, 1: low digit
    const int r = a.split ? rb % a.n_mma : rb;
    const int k = nb * a.NBc + r;
    const int chunk = kpos / BK, j = kpos % BK;
    const int q = j / a.La, pos = j % a.La;
    int v = 0;
    if (r < a.NBc && k < a.K && q < a.WC) {
      int tap, wi, kw;
      if (a.halo) {  // chunk = (channel chunk, tap)
        tap = chunk % a.taps;
        wi = (chunk / a.taps) * a.WC + q;
        kw = wi < a.wpr_a ? 0 : a.words_total;  // past the pixel's last word: zero
      } else {
        kw = chunk * a.WC + q;
        tap = kw / a.wpr_a;
        wi = kw % a.wpr_a;
      }
      if (kw < a.words_total) {
        const int ch = wi * a.La + kpos_lane_op(a.bits_a, a.signed_a != 0, a.fp8 != 0, pos);
        if (ch < a.C) {
          const long long wrow = static_cast<long long>(k) * a.RS + tap;
          const WW word = wt[wrow * a.wpr_w + ch / a.Lw];
          const uint32_t p = static_cast<uint32_t>(word >> ((ch % a.Lw) * a.lane_w_w)) & mask;
          v = lane_value(p, a.bits_w, a.signed_w);
          if (plane == 0) v >>= 4;       // floor(v / 16)
          else if (plane == 1) v &= 15;  // v - 16 * floor(v / 16)
        }
      }
    }
    if constexpr (FP8)
      static_cast<uint8_t *>(Bv)[idx] = int_to_e4m3(v);
    else
      static_cast<__half *>(Bv)[idx] = __int2half_rn(v);
  }
}

// ---- host side -------------------------------------------------------------

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_tiled() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

struct Plan {
  int fp8;        // e4m3 operands (kind::f8f6f4); else fp16
  int full;       // one chunk holds all of a pixel's words (AUnpack FULL)
  int hv;         // tile of hv halves of 128 output positions
  int row_bytes;  // operand row: 64 (e4m3) or 128 (fp16) bytes
  int wpr, words_total, La, WC, nchunks, Kpad, NBc, n_mma, mma_n, split, nblocks, stages, Ho, Wo, gather_vec;
  int gather_win;  // gather through 16-byte windows (AGather::issue_win); chunks = (channel chunk, tap)
  int g_row;       // gather staging row pitch in bytes
  int halo, Hv, Wp, nck, taps;
  int nseg, seg_rows, seg_used, row_step;  // halo geometry (see ConvArgs)
  long long grid_m;                        // 128-position tiles along the output
  int stages_a, b_resident;
  int gdepth;  // HALO: packed staging slots (items gathered gdepth - 1 ahead of the widening)
  int hbufs;   // HALO: widened halo buffers (2 or 3)
  int e_stage; // kEpiStageBytes at off_e stage the epilogue's 3/5/6-bit packed rows
  int pool, pool_rows, pool_nw, pool_pitch, pool_tpi;  // fused 2x2 max-pool (ConvArgs::pool)
  long long M;
  long long bound;  // R*S*C * max|a| * max|w|: no accumulator exceeds it
  uint32_t tmem_cols;
  uint32_t op_stride, off_b, b_bytes, off_g, g_stride, off_e, off_bar;
  size_t smem_bytes;
  size_t ws_bytes;
};

long long max_abs(samd_fmt f) { return f.is_signed ? (1LL << (f.bits - 1)) : ((1LL << f.bits) - 1); }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

constexpr int kMaxHaloRows = 1024;
constexpr int kHaloGatherDepth = 2;  // packed staging slots of the halo producers (2..4)
// minimum 128-pixel tiles per CTA of a launch (samd_conv2d_set_min_tiles_per_cta)
std::atomic<int> g_min_tiles_per_cta{4};

// Tiling, reduction order, operand type and exactness mode for one
// convolution. fo.bits == 0 means no packed output. Returns SAMD_EUNSUP when
// no mode keeps every accumulator below 2^24.
samd_status make_plan(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo, Plan &p, bool pool = false) {
  p.La = lanes_per_word(fa);
  if (p.La == 0) return SAMD_EINVAL;
  const long long taps = static_cast<long long>(d->R) * d->S * d->C;
  const long long bound = taps * max_abs(fa) * max_abs(fw);
  p.bound = bound;
  p.split = 0;
  if (bound >= (1LL << 24)) {
    // two 4-bit weight digits: each accumulator sums at most taps * max|a| * 16
    if (fw.bits <= 4 || taps * max_abs(fa) * 16 >= (1LL << 24)) return SAMD_EUNSUP;
    p.split = 1;
  }
  // e4m3 holds every integer of [-16, 16] exactly
  p.fp8 = (!p.split && max_abs(fa) <= 16 && max_abs(fw) <= 16) ? 1 : 0;
  p.row_bytes = p.fp8 ? 64 : 128;
  p.wpr = static_cast<int>((d->C + p.La - 1) / p.La);
  // FULL chunking (see AUnpack): lanes per word not dividing 64, and the
  // pixel's words hold at most 64 channels in exactly ceil(64 / L) words
  p.full = (BK % p.La != 0 && d->C <= BK && p.wpr == (BK + p.La - 1) / p.La) ? 1 : 0;
  p.WC = p.full ? p.wpr : BK / p.La;
  p.words_total = d->R * d->S * p.wpr;
  p.nchunks = (p.words_total + p.WC - 1) / p.WC;
  p.Kpad = p.nchunks * BK;
  p.Ho = (d->H + 2 * d->pad - d->R) / d->stride + 1;
  p.Wo = (d->W + 2 * d->pad - d->S) / d->stride + 1;
  p.M = static_cast<long long>(d->N) * p.Ho * p.Wo;
  // A channel block must cover whole output words so that no packed word is
  // shared by two CTAs.
  // Channel blocks of up to 256 MMA columns (128 with split digits). (Blocks
  // of 128 for layers with few output positions, which doubles their CTAs,
  // measured slower: every block gathers and widens the whole A operand
  // again, and those layers are bound by that work.)
  const int limit = p.split ? 128 : 256;
  if (d->K <= limit) {
    p.NBc = d->K;
  } else {
    const int Lo = fo.bits ? lanes_per_word(fo) : 1;
    p.NBc = (limit / Lo) * Lo;
  }
  p.n_mma = (p.NBc + 15) / 16 * 16;
  p.mma_n = p.split ? 2 * p.n_mma : p.n_mma;
  p.nblocks = (d->K + p.NBc - 1) / p.NBc;
  // ---- shared memory (the kernel uses these offsets from a 1024-aligned base)
  const int wb = fa.word_bits / 8;
  const int chunk_bytes = p.WC * wb;
  const int srow = (chunk_bytes + 15) / 16 * 16;  // Staging::kRowBytes
  const int vec = chunk_bytes % 16 == 0 ? 16 : (chunk_bytes % 8 == 0 ? 8 : wb);
  p.gather_vec = (p.wpr % p.WC == 0) && ((static_cast<long long>(p.wpr) * wb) % vec == 0) ? 1 : 0;
  // A gather layer whose chunks are not whole 16-byte vectors copies each
  // chunk through the 16-byte-aligned window around it: one more 16-byte
  // piece than the chunk, and an odd number of pieces per staging row, so
  // that a quarter-warp's 16-byte accesses to eight rows hit distinct banks.
  // Its chunks are (channel chunk, tap) pairs, each inside one pixel (as in
  // the halo path), so that a chunk is one contiguous run of a pixel's words
  // however the pixel's word count divides into chunks (strided 3x3 layers
  // whose chunks would otherwise straddle pixels and be copied word by word).
  p.gather_win = (p.gather_vec && vec == 16) ? 0 : 1;
  int win_pieces = srow / 16 + 1;
  if (win_pieces % 2 == 0) ++win_pieces;
  const int grow = p.gather_win ? win_pieces * 16 : srow;
  p.g_row = grow;
  p.b_bytes = static_cast<uint32_t>(p.mma_n) * p.row_bytes;  // a multiple of 1024
  const size_t bst = p.b_bytes;
  const size_t e_bytes = 0;  // the epilogue packs in registers
  // mbarriers: full_b and empty_b per weight stage, opfull and opempty per
  // operand stage, two accumulator pairs, the drain barrier and two
  // epilogue group barriers; then the TMEM address word
  auto bar_bytes = [](int stages, int op_stages) {
    return round_up(static_cast<size_t>(2 * stages + 2 * op_stages + 7) * 8 + 4, 16);
  };
  const size_t kBudget = 224 * 1024;  // below the 227 KB opt-in limit minus static shared memory
  auto finish = [&](size_t op_bytes, size_t g_bytes, int op_stages) {
    p.off_b = static_cast<uint32_t>(op_bytes);
    p.off_g = static_cast<uint32_t>(op_bytes + p.stages * bst);
    p.off_e = static_cast<uint32_t>(round_up(p.off_g + g_bytes, 16));
    p.off_bar = static_cast<uint32_t>(round_up(p.off_e + e_bytes, 16));
    p.smem_bytes = 1024 + p.off_bar + bar_bytes(p.stages, op_stages);  // + alignment slack of the base
  };
  p.taps = d->R * d->S;
  p.nck = (p.wpr + p.WC - 1) / p.WC;
  if (p.gather_win) {  // (channel chunk, tap) chunks
    p.nchunks = p.nck * p.taps;
    p.Kpad = p.nchunks * BK;
  }
  p.Hv = d->H + 2 * d->pad;
  p.Wp = d->W + 2 * d->pad;
  const int nchunks_gather = p.nchunks;
  // One configuration: operand mode (halo or gather) and tile halves hv.
  // Returns false if it does not fit, or if `need_resident` and the weights
  // would not stay resident.
  auto place = [&](bool halo, int hv, bool need_resident) -> bool {
    const int bmt = BM * hv;
    p.hv = hv;
    p.halo = 0;
    p.gdepth = 2;
    p.hbufs = 2;
    p.b_resident = 0;
    p.stages_a = 0;
    p.nseg = p.seg_rows = p.seg_used = p.row_step = 0;
    p.nchunks = nchunks_gather;
    p.Kpad = p.nchunks * BK;
    p.grid_m = (p.M + bmt - 1) / bmt;
    if (halo) {
      // Halo mode: stride 1, several taps, little padded-grid waste, halo
      // fits. The halo is either the contiguous run of virtual rows the tile
      // touches, or (wide images) one segment of bmt + S - 1 rows per filter
      // row.
      if (d->stride != 1 || p.taps < 2 || p.M == 0) return false;
      const int contig = bmt + (d->R - 1) * p.Wp + (d->S - 1);
      const int seg_used = bmt + d->S - 1, seg_rows = (seg_used + 7) / 8 * 8;
      if (d->R * seg_rows < (contig + 7) / 8 * 8) {
        p.nseg = d->R;
        p.seg_rows = seg_rows;
        p.seg_used = seg_used;
        p.row_step = seg_rows;
      } else {
        p.nseg = 1;
        p.seg_rows = (contig + 7) / 8 * 8;
        p.seg_used = contig;
        p.row_step = p.Wp;
      }
      const int halo_rows = p.nseg * p.seg_rows;
      const double waste = static_cast<double>(d->N) * p.Hv * p.Wp / static_cast<double>(p.M);
      const size_t halo_bytes = round_up(static_cast<size_t>(halo_rows) * p.row_bytes, 1024);
      const size_t stage_g = round_up(static_cast<size_t>(halo_rows) * srow, 16);
      const int ntiles_b = p.nck * p.taps;
      if (halo_rows > kMaxHaloRows || waste > 1.16) return false;
      // The packed staging ring: with depth D the gathers run D - 1 items
      // ahead of the widening. Depth 2 is used: per-role timelines show the
      // halo producers finishing a tile's operands microseconds before its
      // MMAs start, and the sweep step measured 6% slower at depth 4 (the
      // kernel takes depths up to 4).
      // Widened halo buffers: the producers widen item k into buffer
      // k mod hbufs once the MMAs of item k - hbufs are done. fp16 layers
      // take three when their weights stay resident as well. (A 6-bit sweep
      // layer's tiles came 2.9 -> 2.2 us apart with three buffers and
      // streamed weights, but the layer as a whole, four tiles per CTA, ran
      // 10-20% slower without resident weights; e4m3 layers, whose halo is
      // half as large and cheaper to widen, showed no gain.)
      size_t fixed = 0;
      bool res = false;
      int depth = kHaloGatherDepth, hbufs = 2;
      auto fits = [&](int nb, int dp, bool want_res) {
        fixed = nb * halo_bytes + dp * stage_g + e_bytes + 1024;
        if (fixed + 2 * bst + bar_bytes(2, nb) > kBudget) return false;
        res = p.nblocks == 1 && fixed + ntiles_b * bst + bar_bytes(ntiles_b, nb) <= kBudget;
        return !(want_res && !res);
      };
      bool ok3 = !p.fp8 && fits(3, depth, true);
      if (ok3) {
        hbufs = 3;
      } else {
        for (; depth >= 2; --depth)
          if (fits(2, depth, need_resident)) break;
        if (depth < 2) return false;
      }
      p.gdepth = depth;
      p.hbufs = hbufs;
      p.halo = 1;
      p.nchunks = ntiles_b;
      p.Kpad = ntiles_b * BK;
      p.grid_m = (static_cast<long long>(d->N) * p.Hv * p.Wp + bmt - 1) / bmt;
      if (res) {
        p.b_resident = 1;
        p.stages = ntiles_b;
      } else {
        long long st = static_cast<long long>((kBudget - fixed - bar_bytes(8, hbufs)) / bst);
        p.stages = static_cast<int>(st > 8 ? 8 : st);
      }
      p.op_stride = static_cast<uint32_t>(halo_bytes);
      p.g_stride = static_cast<uint32_t>(stage_g);
      finish(hbufs * halo_bytes, depth * stage_g, hbufs);
      return true;
    }
    const size_t tile_bytes = static_cast<size_t>(bmt) * p.row_bytes;
    const size_t group_slots = static_cast<size_t>(kGatherDepth) * BM * grow;  // one producer group's ring
    for (int sta = 4; sta >= 2; --sta) {
      const size_t fixed = sta * tile_bytes + 2 * group_slots + e_bytes + 1024;
      if (fixed + 2 * bst + bar_bytes(2, sta) > kBudget) continue;
      const bool res = p.nblocks == 1 && fixed + p.nchunks * bst + bar_bytes(p.nchunks, sta) <= kBudget;
      if (need_resident && !res) continue;
      p.stages_a = sta;
      if (res) {
        p.b_resident = 1;
        p.stages = p.nchunks;
      } else {
        long long st = static_cast<long long>((kBudget - fixed - bar_bytes(8, sta)) / bst);
        p.stages = static_cast<int>(st > 8 ? 8 : st);
      }
      p.op_stride = static_cast<uint32_t>(tile_bytes);
      p.g_stride = static_cast<uint32_t>(group_slots);
      finish(sta * tile_bytes, 2 * group_slots, sta);
      return true;
    }
    return false;
  };
  // Preference: resident weights, then halo over gather, then the most
  // 128-row parts per tile: four (e4m3 halo layers with at most 64 MMA
  // columns: two accumulators of 4 x 64 TMEM columns), two (mma_n <= 128),
  // one. A tile pays a fixed cost (its operand and accumulator handshakes,
  // about 0.7 us measured) whatever its MMA count, so larger tiles of small-N
  // layers spend more of their time in the MMAs -- when every SM gets many
  // of them: four-part tiles are taken for layers of at least four per SM
  // (VGG-16 conv2: 530 -> 622 TMAC/s); small layers, whose CTAs run a few
  // tiles after a start-up of about 3 us, measured no gain or a loss.
  const bool two = p.mma_n <= 128;
  const long long virt = static_cast<long long>(d->N) * (d->H + 2 * d->pad) * (d->W + 2 * d->pad);
  const bool four = p.fp8 && p.mma_n <= 64 && (virt + 4 * BM - 1) / (4 * BM) >= 4LL * sm_count();
  bool placed = false;
  const int kModes[5][2] = {{1, 4}, {1, 2}, {1, 1}, {0, 2}, {0, 1}};  // (halo, parts)
  for (int need_res = (p.nblocks == 1 ? 1 : 0); need_res >= 0 && !placed; --need_res)
    for (int mode = 0; mode < 5 && !placed; ++mode) {
      const bool halo = kModes[mode][0] != 0;
      const int hv = kModes[mode][1];
      if ((hv == 2 && !two) || (hv == 4 && !four)) continue;
      placed = place(halo, hv, need_res != 0);
    }
  if (!placed) return SAMD_EUNSUP;  // operand tiles do not fit (not reached for N <= 256)
  // Fused 2x2 max-pool: tiles must hold whole pairs of padded image rows,
  // 2 Wp <= 128 hv. Halo layers are placed again with the most tile halves
  // that allow it (the weight layout of a halo layer does not depend on the
  // halves or on residency, so the same prepared weights serve both forms).
  if (pool) {
    if (!p.halo) return SAMD_EUNSUP;
    placed = false;
    for (int hv = 2; hv >= 1 && !placed; --hv) {
      if ((hv == 2 && !two) || 2 * p.Wp > BM * hv) continue;
      for (int need_res = 1; need_res >= 0 && !placed; --need_res) placed = place(true, hv, need_res != 0);
    }
    if (!placed) return SAMD_EUNSUP;
  }
  // 3-, 5- and 6-bit packed outputs (32-bit words, no spacer) stage their
  // rows in shared memory when a channel block's row holds at least one
  // whole packing period (lcm(32, L) channels: 160 for L = 5 or 10, 96 for
  // L = 6) and the buffer fits beside the placement chosen above (which it
  // never changes), so that stores are contiguous within a row. Shorter rows
  // (64 channels: 7 to 13 words) measured faster stored directly.
  p.e_stage = 0;
  const int period_ch = fo.bits == 5 ? 96 : 160;
  if ((fo.bits == 3 || fo.bits == 5 || fo.bits == 6) && fo.spacer == 0 && fo.word_bits == 32 &&
      p.NBc >= period_ch && p.smem_bytes + round_up(kEpiStageBytes, 16) <= kBudget) {
    p.e_stage = 1;
    p.off_bar = static_cast<uint32_t>(round_up(p.off_e + kEpiStageBytes, 16));
    p.smem_bytes = 1024 + p.off_bar + bar_bytes(p.stages, p.halo ? p.hbufs : p.stages_a);
  }
  // Fused 2x2 max-pool (placed above): even output sizes, outputs of 1, 2, 4
  // or 8 bits in 32-bit words. A tile is q = 128 hv / (2 Wp) row pairs of
  // one image; its packed rows are staged in 256 rows of pool_pitch words
  // (odd, so that the epilogue threads' word stores spread over the banks)
  // after the other regions: one buffer of 256 rows for two-half tiles, one
  // of 128 rows per epilogue set for one-half tiles.
  p.pool = 0;
  if (pool) {
    const int Ho = p.Ho, Wo = p.Wo;
    if (!p.halo || d->stride != 1 || (Ho & 1) || (Wo & 1) || Ho < 2 || 2 * p.Wp > BM * p.hv || fo.spacer != 0 ||
        fo.word_bits != 32 || (fo.bits != 1 && fo.bits != 2 && fo.bits != 4 && fo.bits != 8))
      return SAMD_EUNSUP;
    int q = (BM * p.hv) / (2 * p.Wp);
    if (q > Ho / 2) q = Ho / 2;
    const int Lo = 32 / fo.bits;
    p.pool_rows = 2 * q;
    p.pool_tpi = (Ho / 2 + q - 1) / q;
    p.pool_nw = (p.NBc + Lo - 1) / Lo;
    p.pool_pitch = p.pool_nw | 1;
    const size_t pool_bytes = static_cast<size_t>(2 * BM) * p.pool_pitch * 4;
    if (p.e_stage) return SAMD_EUNSUP;  // not reached: e_stage is for 3/5/6-bit outputs
    // the buffer goes after the packed staging ring, made shallower if need
    // be (the ring's depth does not change the weight layout)
    int depth = p.gdepth;
    size_t off_e = 0;
    for (; depth >= 2; --depth) {
      off_e = round_up(p.off_g + static_cast<size_t>(depth) * p.g_stride, 16);
      if (1024 + round_up(off_e + pool_bytes, 16) + bar_bytes(p.stages, p.hbufs) <= kBudget) break;
    }
    if (depth < 2) return SAMD_EUNSUP;
    p.pool = 1;
    p.gdepth = depth;
    p.grid_m = static_cast<long long>(d->N) * p.pool_tpi;
    p.off_e = static_cast<uint32_t>(off_e);
    p.off_bar = static_cast<uint32_t>(round_up(off_e + pool_bytes, 16));
    p.smem_bytes = 1024 + p.off_bar + bar_bytes(p.stages, p.hbufs);
  }
  uint32_t cols = 32;
  while (cols < static_cast<uint32_t>(2 * p.hv * p.mma_n)) cols <<= 1;  // two accumulators of hv halves
  p.tmem_cols = cols;
  p.ws_bytes = static_cast<size_t>(p.nblocks) * p.mma_n * p.Kpad * (p.fp8 ? 1 : 2);
  return SAMD_OK;
}

samd_fmt none_fmt() { return samd_fmt{0, 0, 0, 0}; }

// Every shared-memory region of the plan lies inside its allocation (checked
// before each launch; a planning mistake becomes SAMD_EUNSUP, not a fault).
bool layout_ok(const Plan &p) {
  const size_t NO = p.halo ? static_cast<size_t>(p.hbufs) : static_cast<size_t>(p.stages_a);
  const size_t op_bytes = NO * p.op_stride;
  const size_t bars = (2 * static_cast<size_t>(p.stages) + 2 * NO + 7) * 8 + 4;
  return p.stages >= 1 && NO >= 2 && op_bytes <= p.off_b &&
         p.off_b + static_cast<size_t>(p.stages) * p.b_bytes <= p.off_g && p.off_g + static_cast<size_t>(p.halo ? p.gdepth : 2) * p.g_stride <= p.off_e &&
         p.off_e <= p.off_bar && 1023 + p.off_bar + bars <= p.smem_bytes && p.op_stride % 1024 == 0 &&
         p.off_b % 1024 == 0 && p.b_bytes % 1024 == 0 && p.off_bar % 8 == 0 && 2 * p.hv * p.mma_n <= 512 &&
         (p.hv == 1 || p.hv == 2 || (p.hv == 4 && p.halo && p.fp8 && p.mma_n <= 64)) && (!p.halo || (p.gdepth >= 2 && p.gdepth <= 4 && (p.hbufs == 2 || p.hbufs == 3))) &&
         (!p.e_stage || p.off_e + kEpiStageBytes <= p.off_bar) &&
         (!p.pool || (p.halo && 2 * p.Wp <= BM * p.hv && !p.e_stage && p.pool_pitch >= p.pool_nw &&
                      p.off_e + static_cast<size_t>(2 * BM) * p.pool_pitch * 4 <= p.off_bar));
}

// Device address of a __device__ symbol in the current context, looked up
// once per context (the symbol's host-side name is not a device address; a
// context made after a device reset loads the module again, at a new address).
struct SymbolAddr {
  static constexpr int kSlots = 64;
  std::mutex mu;
  unsigned long long ctx[kSlots] = {0};
  void *ptr[kSlots] = {nullptr};
  int n = 0, next = 0;
  cudaError_t get(const void *symbol, void **out) {
    unsigned long long id = 0;
    cudaError_t e = current_context_id(&id);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < n; ++i)
      if (ctx[i] == id) {
        *out = ptr[i];
        return cudaSuccess;
      }
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, symbol);
    if (e != cudaSuccess) return e;
    const int slot = n < kSlots ? n++ : next;  // when full, entries are replaced in turn
    if (n == kSlots) next = (slot + 1) % kSlots;
    ctx[slot] = id;
    ptr[slot] = p;
    *out = p;
    return cudaSuccess;
  }
};
SymbolAddr g_status_addr, g_scratch_addr;

}  // namespace
}  // namespace conv

size_t conv2d_workspace_size(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw) {
  // the channel blocking depends on the output format only above 128/256
  // channels: report the largest size over every output format
  conv::Plan p;
  if (conv::make_plan(d, fa, fw, conv::none_fmt(), p) != SAMD_OK) return 0;
  size_t best = p.ws_bytes;
  for (int wb : {32, 64})
    for (int bits = 1; bits <= 8; ++bits)
      for (int sp = 0; sp + bits <= 16 && sp <= 8; ++sp) {
        samd_fmt fo{static_cast<uint8_t>(bits), 0, static_cast<uint8_t>(sp), static_cast<uint8_t>(wb)};
        conv::Plan q;
        if (conv::make_plan(d, fa, fw, fo, q) == SAMD_OK && q.ws_bytes > best) best = q.ws_bytes;
      }
  return best;
}

void conv2d_set_min_tiles_per_cta(int tiles) { conv::g_min_tiles_per_cta.store(tiles, std::memory_order_relaxed); }

int conv2d_operand_bits(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw) {
  conv::Plan p;
  if (conv::make_plan(d, fa, fw, conv::none_fmt(), p) != SAMD_OK) return 0;
  return p.fp8 ? 8 : 16;
}

int conv2d_pool_supported(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, samd_fmt fo) {
  conv::Plan p;
  return (conv::make_plan(d, fa, fw, fo, p, true) == SAMD_OK && conv::layout_ok(p)) ? 1 : 0;
}

samd_status conv2d_check(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw) {
  conv::Plan p;
  return conv::make_plan(d, fa, fw, conv::none_fmt(), p);
}

samd_status conv2d_prepare(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, const void *wt, samd_fmt fo,
                           void *prepared, size_t prepared_bytes, cudaStream_t s) {
  using namespace conv;
  Plan p;
  samd_status st = make_plan(d, fa, fw, fo, p);
  if (st != SAMD_OK) return st;
  if (prepared_bytes < p.ws_bytes) return SAMD_ESHAPE;
  WPrepArgs wa;
  wa.K = d->K;
  wa.C = d->C;
  wa.RS = d->R * d->S;
  wa.bits_w = fw.bits;
  wa.signed_w = fw.is_signed;
  wa.lane_w_w = fw.bits + fw.spacer;
  wa.Lw = lanes_per_word(fw);
  wa.wpr_w = static_cast<int>(words_per_row(fw, d->C));
  wa.bits_a = fa.bits;
  wa.signed_a = fa.is_signed;
  wa.fp8 = p.fp8;
  wa.La = p.La;
  wa.WC = p.WC;
  wa.wpr_a = p.wpr;
  wa.words_total = p.words_total;
  wa.Kpad = p.Kpad;
  wa.n_mma = p.n_mma;
  wa.mma_n = p.mma_n;
  wa.NBc = p.NBc;
  wa.split = p.split;
  wa.halo = p.halo || p.gather_win;  // reduction order (channel chunk, tap, position)
  wa.taps = p.taps;
  wa.rows_total = static_cast<long long>(p.nblocks) * p.mma_n;
  const long long total = wa.rows_total * wa.Kpad;
  const int grid = grid_for(total, 256, sm_count() * 8);
  if (fw.word_bits == 32) {
    if (p.fp8)
      wprep_kernel<uint32_t, true><<<grid, 256, 0, s>>>(static_cast<const uint32_t *>(wt), prepared, wa);
    else
      wprep_kernel<uint32_t, false><<<grid, 256, 0, s>>>(static_cast<const uint32_t *>(wt), prepared, wa);
  } else {
    if (p.fp8)
      wprep_kernel<uint64_t, true><<<grid, 256, 0, s>>>(static_cast<const uint64_t *>(wt), prepared, wa);
    else
      wprep_kernel<uint64_t, false><<<grid, 256, 0, s>>>(static_cast<const uint64_t *>(wt), prepared, wa);
  }
  return cudaGetLastError() == cudaSuccess ? SAMD_OK : SAMD_ECUDA;
}

samd_status conv2d_run(const samd_conv_desc *d, samd_fmt fa, samd_fmt fw, const void *act, const void *prepared,
                       size_t prepared_bytes, int32_t *acc_out, samd_fmt fo, void *packed_out, int shift,
                       cudaStream_t s, void *pooled_out) {
  using namespace conv;
  Plan p;
  // pooled_out: the 2x2 max-pool of the packed output is the only output
  const bool pool = pooled_out != nullptr;
  if (pool && (acc_out || packed_out)) return SAMD_EINVAL;
  if (pool) packed_out = pooled_out;
  samd_status st = make_plan(d, fa, fw, fo, p, pool);
  if (st != SAMD_OK) return st;
  if (prepared_bytes < p.ws_bytes) return SAMD_ESHAPE;
  if (p.M == 0) return SAMD_OK;
  if (!layout_ok(p)) return SAMD_EUNSUP;
  EncodeTiledFn enc = encode_tiled();
  if (!enc) return SAMD_ECUDA;
  void *status_ptr = nullptr;
  if (g_status_addr.get(reinterpret_cast<const void *>(&g_conv_status), &status_ptr) != cudaSuccess) return SAMD_ECUDA;

  // tensor map over the widened weights: [nblocks * mma_n][Kpad] elements,
  // tiles of mma_n rows x 64 elements, swizzled like the A operand rows
  CUtensorMap tmap;
  const long long rows_total = static_cast<long long>(p.nblocks) * p.mma_n;
  const int esize = p.fp8 ? 1 : 2;
  cuuint64_t gdim[2] = {static_cast<cuuint64_t>(p.Kpad), static_cast<cuuint64_t>(rows_total)};
  cuuint64_t gstride[1] = {static_cast<cuuint64_t>(p.Kpad) * esize};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(p.mma_n)};
  cuuint32_t estride[2] = {1, 1};
  CUresult cr = enc(&tmap, p.fp8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2,
                    const_cast<void *>(prepared), gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    p.fp8 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return SAMD_ECUDA;

  ConvArgs a;
  a.act = act;
  a.acc_out = acc_out;
  a.packed_out = packed_out;
  a.status = static_cast<int *>(status_ptr);
  a.N = d->N;
  a.C = d->C;
  a.H = d->H;
  a.W = d->W;
  a.K = d->K;
  a.R = d->R;
  a.S = d->S;
  a.stride = d->stride;
  a.pad = d->pad;
  a.Ho = p.Ho;
  a.Wo = p.Wo;
  a.M = p.M;
  a.wpr = p.wpr;
  a.words_total = p.words_total;
  a.nchunks = p.nchunks;
  a.NBc = p.NBc;
  a.n_mma = p.n_mma;
  a.mma_n = p.mma_n;
  a.split = p.split;
  a.stages = p.stages;
  a.stages_a = p.stages_a;
  a.b_resident = p.b_resident;
  a.grid_m = p.grid_m;
  a.nblocks = p.nblocks;
  a.gather_vec = p.gather_vec;
  a.gather_win = p.gather_win;
  a.g_row = p.g_row;
  a.act_bytes = static_cast<long long>(d->N) * d->H * d->W * p.wpr * (fa.word_bits / 8);
  a.tmem_cols = p.tmem_cols;
  a.out_bits = packed_out ? fo.bits : 8;
  a.out_signed = packed_out ? fo.is_signed : 1;
  a.out_lane_w = packed_out ? fo.bits + fo.spacer : 8;
  a.out_L = packed_out ? lanes_per_word(fo) : 1;
  a.out_word64 = packed_out ? (fo.word_bits == 64) : 0;
  a.out_wpr = packed_out ? static_cast<int>(words_per_row(fo, d->K)) : 0;
  {
    const int Lo = a.out_L;
    const bool fast = packed_out && (fo.word_bits == 32 ? (Lo == 4 || Lo == 8 || Lo == 16 || Lo == 32)
                                                        : (Lo == 8 || Lo == 16 || Lo == 32));
    a.out_fast = fast ? Lo : 0;
  }
  a.shift = shift;
  a.out_scale = ldexpf(1.0f, -shift);
  a.fast_req = (!p.split && (p.bound >> shift) < (1LL << 22)) ? 1 : 0;
  a.fast_acc = (!p.split && p.bound < (1LL << 22)) ? 1 : 0;
  a.Hv = p.Hv;
  a.Wp = p.Wp;
  a.nseg = p.nseg;
  a.seg_rows = p.seg_rows;
  a.seg_used = p.seg_used;
  a.row_step = p.row_step;
  a.nck = p.nck;
  a.full = p.full;
  a.hv = p.hv;
  a.taps = p.taps;
  // the kernel's index math runs in 32 bits
  if (static_cast<long long>(d->N) * p.Hv * p.Wp + (p.nseg + 1) * static_cast<long long>(p.Wp) + kMaxHaloRows + 2 * BM >=
          (1LL << 31) ||
      p.M >= (1LL << 31) || p.grid_m * p.nblocks >= (1LL << 31))
    return SAMD_EUNSUP;
  a.fd_plane = make_fastdiv(static_cast<uint32_t>(p.Hv * p.Wp));
  a.fd_wp = make_fastdiv(static_cast<uint32_t>(p.Wp));
  a.fd_seg = make_fastdiv(static_cast<uint32_t>(p.seg_rows > 0 ? p.seg_rows : 1));
  a.fd_wo = make_fastdiv(static_cast<uint32_t>(p.Wo));
  a.fd_ho = make_fastdiv(static_cast<uint32_t>(p.Ho));
  a.fd_gm = make_fastdiv(static_cast<uint32_t>(p.grid_m));
  a.op_stride = p.op_stride;
  a.off_b = p.off_b;
  a.b_bytes = p.b_bytes;
  a.off_g = p.off_g;
  a.g_stride = p.g_stride;
  a.gdepth = p.gdepth;
  a.hbufs = p.hbufs;
  a.off_e = p.off_e;
  a.e_stage = p.e_stage;
  a.pool = p.pool;
  a.pool_rows = p.pool ? p.pool_rows : 0;
  a.pool_nw = p.pool ? p.pool_nw : 0;
  a.pool_pitch = p.pool ? p.pool_pitch : 0;
  a.fd_tpi = make_fastdiv(static_cast<uint32_t>(p.pool ? p.pool_tpi : 1));
  a.off_bar = p.off_bar;
  // A small layer gives each CTA at least T reference tiles of work (T from
  // samd_conv2d_set_min_tiles_per_cta; a reference tile is 128 positions of
  // a 3x3 convolution over 64 input and 64 output channels: 9 operand rows of
  // 64 positions, 64 MMA columns), leaving SMs to independent layers issued
  // on other streams. A tile of this layer weighs hv * nchunks * mma_n of
  // those 9 * 64, so layers with long reductions or many output channels
  // spread over more SMs.
  const long long total_tiles = p.grid_m * p.nblocks;
  const long long ref_work = static_cast<long long>(g_min_tiles_per_cta.load(std::memory_order_relaxed)) * 9 * 64;
  long long tile_work = static_cast<long long>(p.hv) * p.nchunks * p.mma_n;
  // A gather tile with a short reduction (1x1 layers over few channels) is
  // bound by widening its lanes and packing its outputs, not by its MMAs:
  // it counts as at least one reference tile per half.
  if (!p.halo && tile_work < static_cast<long long>(p.hv) * 9 * 64) tile_work = static_cast<long long>(p.hv) * 9 * 64;
  long long min_tiles = ref_work / tile_work;
  if (min_tiles < 1) min_tiles = 1;
  long long ctas = (total_tiles + min_tiles - 1) / min_tiles;
  if (ctas > sm_count()) ctas = sm_count();
  dim3 grid(static_cast<unsigned>(ctas));
  static const LaunchFn kF16[2][8] = {
      {launch_conv_f16_w32_b1, launch_conv_f16_w32_b2, launch_conv_f16_w32_b3, launch_conv_f16_w32_b4,
       launch_conv_f16_w32_b5, launch_conv_f16_w32_b6, launch_conv_f16_w32_b7, launch_conv_f16_w32_b8},
      {launch_conv_f16_w64_b1, launch_conv_f16_w64_b2, launch_conv_f16_w64_b3, launch_conv_f16_w64_b4,
       launch_conv_f16_w64_b5, launch_conv_f16_w64_b6, launch_conv_f16_w64_b7, launch_conv_f16_w64_b8}};
  static const LaunchFn kF8[2][5] = {
      {launch_conv_f8_w32_b1, launch_conv_f8_w32_b2, launch_conv_f8_w32_b3, launch_conv_f8_w32_b4,
       launch_conv_f8_w32_b5},
      {launch_conv_f8_w64_b1, launch_conv_f8_w64_b2, launch_conv_f8_w64_b3, launch_conv_f8_w64_b4,
       launch_conv_f8_w64_b5}};
  const int wi = fa.word_bits == 64 ? 1 : 0;
  if (p.fp8 && fa.bits > 5) return SAMD_EUNSUP;  // not reached: e4m3 only for |a| <= 16
  const LaunchFn fn = p.fp8 ? kF8[wi][fa.bits - 1] : kF16[wi][fa.bits - 1];
  const cudaError_t e = fn(fa.is_signed != 0, tmap, a, p.halo != 0, grid, p.smem_bytes, s);
  return e == cudaSuccess ? SAMD_OK : SAMD_ECUDA;
}

samd_status conv2d_nhwc(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                        int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, void *workspace,
                        size_t workspace_bytes, cudaStream_t s) {
  const samd_fmt fplan = packed_out ? fo : conv::none_fmt();
  samd_status st = conv2d_prepare(d, fa, fw, wt, fplan, workspace, workspace_bytes, s);
  if (st != SAMD_OK) return st;
  return conv2d_run(d, fa, fw, act, workspace, workspace_bytes, acc_out, fplan, packed_out, shift, s);
}

samd_status conv2d_noalloc(const samd_conv_desc *d, samd_fmt fa, const void *act, samd_fmt fw, const void *wt,
                           int32_t *acc_out, samd_fmt fo, void *packed_out, int shift, cudaStream_t s) {
  size_t need = 0;
  if (d->layout == SAMD_NCHW) {
    samd_status st = conv2d_nchw_check(d, fa, fw, packed_out ? fo : conv::none_fmt(), &need);
    if (st != SAMD_OK) return st;
  } else {
    conv::Plan p;
    samd_status st = conv::make_plan(d, fa, fw, packed_out ? fo : conv::none_fmt(), p);
    if (st != SAMD_OK) return st;
    need = p.ws_bytes;
  }
  // the scratch this call needs (for its shape, formats and output format) must fit
  if (need > kNoallocScratchBytes) return SAMD_EUNSUP;
  void *scratch = nullptr;
  if (conv::g_scratch_addr.get(reinterpret_cast<const void *>(&g_noalloc_scratch), &scratch) != cudaSuccess)
    return SAMD_ECUDA;
  // the calls below write every byte of scratch they then read, so nothing
  // left over from an earlier call is ever used
  if (d->layout == SAMD_NCHW)
    return conv2d_nchw(d, fa, act, fw, wt, acc_out, fo, packed_out, shift, scratch, kNoallocScratchBytes, s);
  return conv2d_nhwc(d, fa, act, fw, wt, acc_out, fo, packed_out, shift, scratch, kNoallocScratchBytes, s);
}

// One thread waits, bounded by limit_ns, on an mbarrier phase that nothing
// completes; the wait runs out and the thread records SAMD_ETIMEOUT exactly as
// a convolution role that gives up does. Nothing is in flight when it returns.
__global__ void wait_timeout_kernel(uint64_t limit_ns) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    ptx::mbar_init(ptx::smem_addr(&bar), 1);
    ptx::fence_barrier_init();
    int quiet = 0;
    if (!ptx::mbar_wait_bounded(ptx::smem_addr(&bar), 0, &quiet, limit_ns))
      atomicOr(&g_conv_status, static_cast<int>(SAMD_ETIMEOUT));
  }
}

cudaError_t selftest_wait_timeout(uint64_t limit_ns, cudaStream_t s) {
  wait_timeout_kernel<<<1, 32, 0, s>>>(limit_ns);
  return cudaGetLastError();
}

cudaError_t read_device_status(int *status, int reset, cudaStream_t s) {
  int v = 0;
  cudaError_t e = cudaMemcpyFromSymbolAsync(&v, g_conv_status, sizeof(int), 0, cudaMemcpyDeviceToHost, s);
  if (e != cudaSuccess) return e;
  e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return e;
  *status = v;
  if (reset && v != 0) {
    int zero = 0;
    e = cudaMemcpyToSymbolAsync(g_conv_status, &zero, sizeof(int), 0, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  }
  return e;
}

}  // namespace samd
