// Dense and zero-skipping implicit-GEMM kernel on the 5th-generation tensor
// cores (tcgen05, accumulators in tensor memory), sm_103a.
//
// Persistent: one CTA per SM walks the output tiles (128 rows x BN columns)
// of y = epilogue(A * B^T) with a static round-robin schedule.  Two tensor-
// memory accumulators alternate between tiles, so the epilogue of tile i
// (TMEM -> registers -> swizzled shared memory -> TMA store) overlaps the MMAs
// of tile i + 1, and the shared-memory stage ring never drains between tiles.
//
// B [N, K] holds the weights (K-major; [C_out][kh][kw][C] for a convolution)
// and is loaded by TMA.  A (128 rows of K) comes in one of three ways:
//   mode 0  GEMM: A = x[M, K] row-major; rows m0..m0+127; 2-D TMA box.
//   mode 2  convolution, C % BK == 0: the 128 rows are a spatial output tile
//           of bw x bh pixels in bn images; for K block (tap r,s; BK channels)
//           one 4-D TMA box {BK channels, bw, bh, bn} of the NHWC input at the
//           shifted, strided origin (element strides = conv stride) is the A
//           tile; out-of-range coordinates read zeros, which is the padding.
//   mode 1  convolution, any C % 8 == 0 (the RGB stem): 128 consecutive output
//           pixels, gathered by 128 producer threads with cp.async.
// K advances in BK-wide blocks: BK = 64 with the 128-byte swizzle (four
// tcgen05.mma of K = 16 per stage) or BK = 32 with the 64-byte swizzle.
//
// Threshold dispatch (Sec. 3 rule, thresholds as parameters) is evaluated in
// the kernel prologue from the input's Eq. 1 count, so no host round trip
// separates statistics and compute.  On the zero-skip path each tile leaves
// out the K blocks whose activations are all zero over its 128 rows (Sec. 2.1:
// products with zero activations can be skipped without changing the result):
//   GEMM: from the 128-row block-column mask of x (one word per 32 columns);
//   conv: from the row bitmaps of the tile's shifted input pixels, reduced
//         per tile into a per-tap mask of occupied 64-channel tiles.
// The epilogue applies bias / batch norm / residual / activation, stores y and
// writes y's Eq. 1 count and occupancy bitmaps for the next operator.
//
// Warp roles (416 threads): warps 0-3 producers (the skip masks; thread 0
// issues TMA; all 128 gather in mode 1), warps 4-11 epilogue (two per TMEM
// lane quarter, each taking 32 of every 64 accumulator columns), warp 12 TMEM
// allocation and MMA issue (lane 0).
//
// Each tile shape is compiled three times: the general kernel, and lean ones
// for modes 0 and 2 without a K split or fp32 output, without a residual and
// with one (N % 8 == 0).  With small K the
// epilogue is the whole cost of a tile and runs at a fraction of an
// instruction per cycle (few warps, long dependency chains); the lean kernel's
// smaller, branch-free epilogue issues fewer instructions per tile and misses
// the instruction cache less.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "sparoa_kernels.h"

namespace sparoa {

namespace {

constexpr int kEpiWarps = 8;
constexpr int kMaxSplit = 4;  // K split: at most this many units per output tile                   // two per TMEM lane quarter, 32 of each 64 columns
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kMmaWarp = 4 + kEpiWarps;
constexpr int kThreads = 32 * (kMmaWarp + 1);  // 4 producer warps, epilogue warps, MMA warp
constexpr int kBM = 128;
constexpr int kMaxKWords = 128;  // K-block occupancy bits: up to 4096 blocks
constexpr int kMaxTaps = 64;
constexpr int kStgBytes = 128 * 128;  // output staging: per epilogue warp 2 blocks of 32 rows x 64 bytes
constexpr int kWarpStgBytes = 32 * 64;
constexpr int kMaxAccCols = 4096;     // per-CTA column counters (output occupancy)

template <int BN, int BK>
struct Cfg {
  static constexpr int kAStage = kBM * BK * 2;
  static constexpr int kBStage = BN * BK * 2;
  static constexpr int kStageBytes = kAStage + kBStage;
  // Stage ring: about 200 KB of shared memory in all; a deeper ring made the
  // latency-bound small GEMMs and convs slower on GB300 (256 x 3072 x 768:
  // 13.6 -> 16.4 us).  192-wide tiles take all of the 227 KB for a fourth
  // 40 KB stage (4096 x 3072 x 768: 26.1 -> 22.3 us).  kFixed is everything
  // but the ring (barriers and flags of at most 12 stages) plus the 1024 bytes
  // of alignment slack.
  static constexpr int kFixed = 2 * kStgBytes + (2 * 12 + 5) * 8 + (12 + 8) * 4 + 16 + kMaxKWords * 4 +
                                kMaxTaps * 8 + 4 * BN * 4 + 4 * BN * 4 + kMaxAccCols * 4 + 2 * kBM * 8 +
                                2 * (BN / 32) * 4 + 16 + 1024;
  static constexpr int kBudget =
      BN == 192 ? 227 * 1024 - kFixed : 200 * 1024 - 2 * kStgBytes - 6 * 1024 - kMaxAccCols * 4;
  static constexpr int kStagesRaw = kBudget / kStageBytes;
  static constexpr int kStages = kStagesRaw > 12 ? 12 : kStagesRaw;
  static constexpr int kLag = kStages - 2;  // cp.async stages in flight (mode 1)
  static constexpr int kAOff = 0;
  static constexpr int kBOff = kAOff + kStages * kAStage;
  static constexpr int kStgOff = kBOff + kStages * kBStage;          // 1024-aligned
  static constexpr int kBarOff = kStgOff + 2 * kStgBytes;
  static constexpr int kNumBars = 2 * kStages + 5;                   // full, empty, accf[2], acce[2], drain
  static constexpr int kFlagOff = kBarOff + kNumBars * 8;
  static constexpr int kKBitsOff = (kFlagOff + (kStages + 8) * 4 + 15) & ~15;
  static constexpr int kTapOff = kKBitsOff + kMaxKWords * 4;
  static constexpr int kScaleOff = kTapOff + kMaxTaps * 8;
  static constexpr int kShiftOff = kScaleOff + 2 * BN * 4;  // scale / shift: [2 accumulators][BN]
  static constexpr int kCntOff = kShiftOff + 2 * BN * 4;
  static constexpr int kAccOff = kCntOff + 4 * BN * 4;
  static constexpr int kRowOff = kAccOff + kMaxAccCols * 4;   // [2][128] row bits of the tile
  static constexpr int kBlkOff = kRowOff + 2 * kBM * 8;       // [2][BN / 32] block-mask words
  static constexpr int kBytes = kBlkOff + 2 * (BN / 32) * 4 + 16;
  static constexpr int kSmem = kBytes + 1024;  // slack for 1024-byte alignment
  // TMEM: accumulator b starts at column b * kAccCols (BN rounded up to a
  // power of two, so each starts on a power-of-two column); the allocation
  // covers both
  static constexpr uint32_t kAccCols = BN <= 64 ? 64u : (BN <= 128 ? 128u : 256u);
  static constexpr uint32_t kTmemCols = 2 * kAccCols;
  static_assert(kStages >= 2, "stages");
  static_assert(kSmem <= 227 * 1024, "shared memory");
};

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const void* tmap, uint32_t bar, int c0,
                                            int c1, int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
      : "memory");
}

// Launch geometry copied out of the kernel parameters into registers once:
// reading IgemmArgs fields through a reference is a memory load, and every
// asm statement with a memory clobber would force it again.
struct Geo {
  int conv, M, N, Nimg, H, W, Cp, Ho, Wo, kh, kw, stride, pad, bw, bh, bn, tw, th, Ktot;
};

__device__ __forceinline__ Geo make_geo(const IgemmArgs& a) {
  Geo g;
  g.conv = a.conv; g.M = a.M; g.N = a.N; g.Nimg = a.Nimg; g.H = a.H; g.W = a.W; g.Cp = a.Cp;
  g.Ho = a.Ho; g.Wo = a.Wo; g.kh = a.kh; g.kw = a.kw; g.stride = a.stride; g.pad = a.pad;
  g.bw = a.bw; g.bh = a.bh; g.bn = a.bn; g.tw = a.tw; g.th = a.th; g.Ktot = a.Ktot;
  return g;
}

struct TileGeo {
  int m0, tn0, th0, tw0, n0;
};

__device__ __forceinline__ TileGeo tile_geo(const Geo& p, int t, int nt, int BN) {
  TileGeo g;
  const int mi = nt == 1 ? t : t / nt;
  g.n0 = (t - mi * nt) * BN;
  g.m0 = 0;
  g.tn0 = g.th0 = g.tw0 = 0;
  if (p.conv == 2) {
    const int per_img = p.th * p.tw;
    g.tn0 = (mi / per_img) * p.bn;
    const int rem = mi - (mi / per_img) * per_img;
    g.th0 = (rem / p.tw) * p.bh;
    g.tw0 = (rem - (rem / p.tw) * p.tw) * p.bw;
  } else {
    g.m0 = mi * kBM;
  }
  return g;
}

// Output pixel / row of tile row r and whether it exists.
__device__ __forceinline__ int64_t tile_row(const Geo& p, const TileGeo& g, int r, bool& valid,
                                            int& img, int& oh, int& ow) {
  if (p.conv == 2) {
    const int wl = r % p.bw, hl = (r / p.bw) % p.bh, nl = r / (p.bw * p.bh);
    img = g.tn0 + nl;
    oh = g.th0 + hl;
    ow = g.tw0 + wl;
    valid = img < p.Nimg && oh < p.Ho && ow < p.Wo;
    return ((int64_t)img * p.Ho + oh) * p.Wo + ow;
  }
  const int64_t m = (int64_t)g.m0 + r;
  valid = m < p.M;
  if (p.conv == 1) {
    const int hw = p.Ho * p.Wo;
    img = valid ? (int)(m / hw) : 0;
    const int rem = (int)(m - (int64_t)img * hw);
    oh = valid ? rem / p.Wo : 0;
    ow = valid ? rem - oh * p.Wo : 0;
  } else {
    img = oh = ow = 0;
  }
  return m;
}

// One row's 32 accumulator values (fp32 bits) through the column affine
// (scale and shift from shared memory; none when sc is null), the residual
// (bf16 at rp, none when rp is null; only the first rvalid of the 32 columns
// are read, rvalid a multiple of 8) and the activation, packed to 16 bf16
// pairs: fp32x2 FMAs, ReLU folded into the conversion.  The same operations
// in the same order as the general epilogue (fmaf, then + residual, then the
// activation, then round to bf16).
template <int ACT, bool RES>
__device__ __forceinline__ void affine_act_pack32(const uint32_t (&raw)[32], const float* sc, const float* sh,
                                                  const uint4* rp, int rvalid, uint32_t (&pk)[16]) {
  uint4 rv = make_uint4(0u, 0u, 0u, 0u);  // residual values 8 (i / 2) .. + 7
  if (!RES) rp = nullptr;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    if (RES && rp && (i & 1) == 0) rv = 8 * (i >> 1) < rvalid ? rp[i >> 1] : make_uint4(0u, 0u, 0u, 0u);
    if (sc == nullptr && rp == nullptr) {  // the accumulators as they are
      pk[2 * i] = act_pack2<ACT>(__uint_as_float(raw[4 * i]), __uint_as_float(raw[4 * i + 1]));
      pk[2 * i + 1] = act_pack2<ACT>(__uint_as_float(raw[4 * i + 2]), __uint_as_float(raw[4 * i + 3]));
      continue;
    }
    if (sc == nullptr) {
      float a = __uint_as_float(raw[4 * i]), b = __uint_as_float(raw[4 * i + 1]);
      float c = __uint_as_float(raw[4 * i + 2]), d = __uint_as_float(raw[4 * i + 3]);
      const uint32_t w0 = (i & 1) ? rv.z : rv.x, w1 = (i & 1) ? rv.w : rv.y;
      a += __uint_as_float(w0 << 16);
      b += __uint_as_float(w0 & 0xFFFF0000u);
      c += __uint_as_float(w1 << 16);
      d += __uint_as_float(w1 & 0xFFFF0000u);
      pk[2 * i] = act_pack2<ACT>(a, b);
      pk[2 * i + 1] = act_pack2<ACT>(c, d);
      continue;
    }
    const float4 s4 = reinterpret_cast<const float4*>(sc)[i];
    const float4 h4 = reinterpret_cast<const float4*>(sh)[i];
    float a, b, c, d;
    f2_split(ffma2(f2(__uint_as_float(raw[4 * i]), __uint_as_float(raw[4 * i + 1])), f2(s4.x, s4.y),
                   f2(h4.x, h4.y)),
             a, b);
    f2_split(ffma2(f2(__uint_as_float(raw[4 * i + 2]), __uint_as_float(raw[4 * i + 3])), f2(s4.z, s4.w),
                   f2(h4.z, h4.w)),
             c, d);
    if (RES && rp) {
      const uint32_t w0 = (i & 1) ? rv.z : rv.x, w1 = (i & 1) ? rv.w : rv.y;
      a += __uint_as_float(w0 << 16);
      b += __uint_as_float(w0 & 0xFFFF0000u);
      c += __uint_as_float(w1 << 16);
      d += __uint_as_float(w1 & 0xFFFF0000u);
    }
    pk[2 * i] = act_pack2<ACT>(a, b);
    pk[2 * i + 1] = act_pack2<ACT>(c, d);
  }
}

// Bit c of the result: bf16 value c of the 16 packed pairs is non-zero.  Per
// two words: the non-zero flags of their four halves (bits 15 and 31 after
// nz_pairs' carry trick) are gathered into one word's byte tops (bits 7, 15,
// 23, 31) by a byte permute, and the multiply by 1 + 2^7 + 2^14 + 2^21 moves
// them, without carries, to bits 28..31.
__device__ __forceinline__ uint32_t nz_mask32(const uint32_t (&pk)[16]) {
  uint32_t m = 0u;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const uint32_t ta = (pk[2 * i] & 0x7FFF7FFFu) + 0x7FFF7FFFu;
    const uint32_t tb = (pk[2 * i + 1] & 0x7FFF7FFFu) + 0x7FFF7FFFu;
    const uint32_t x = __byte_perm(ta, tb, 0x7531) & 0x80808080u;
    m |= ((x * 0x00204081u) >> 28) << (4 * i);
  }
  return m;
}

// Everything a producer thread needs to know about work unit u (tile u / ks,
// K range u % ks): pure arithmetic on the parameters, 32-bit throughout.
struct UnitGeo {
  int t, ks, kb0, kb1;
  TileGeo g;
  bool rvalid;
  int img, oh, ow;
  int cb, rr, ss;  // conv = 2: channel block and tap (row, column) of block kb0
  int iy0, ix0;    // conv = 2: input origin of the tile
};

__device__ __forceinline__ UnitGeo unit_geo(const Geo& p, int u, int KS, int kblocks, int nt, int BN,
                                            int BK, int r) {
  UnitGeo q;
  q.t = u / KS;
  q.ks = u - q.t * KS;
  q.kb0 = q.ks * kblocks / KS;
  q.kb1 = (q.ks + 1) * kblocks / KS;
  q.g = tile_geo(p, q.t, nt, BN);
  tile_row(p, q.g, r, q.rvalid, q.img, q.oh, q.ow);
  q.cb = q.rr = q.ss = 0;
  if (p.conv == 2) {
    const int cb_per_tap = p.Cp / BK;
    const int tap = q.kb0 / cb_per_tap;
    q.cb = q.kb0 - tap * cb_per_tap;
    q.rr = tap / p.kw;
    q.ss = tap - q.rr * p.kw;
  }
  q.iy0 = q.g.th0 * p.stride - p.pad;
  q.ix0 = q.g.tw0 * p.stride - p.pad;
  return q;
}

template <int BN, int BK, int LEAN>
__global__ void __launch_bounds__(kThreads, 1)
    igemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                 const __grid_constant__ CUtensorMap tmY, const __grid_constant__ CUtensorMap tmA32,
                 const __grid_constant__ CUtensorMap tmB32, const IgemmArgs P) {
  using C = Cfg<BN, BK>;
  const Geo p = make_geo(P);
  // lean kernels (LEAN 1: no residual, 2: a residual and N % 8 == 0): TMA
  // producers only (mode 0 or 2), no K split, bf16 output (the host launches
  // them only then)
  if (LEAN) __builtin_assume(p.conv != 1);
  const EpiDev ep = P.ep;
  const int act = P.ep.act;
  const __nv_bfloat16* const residual = LEAN == 1 ? nullptr : P.ep.residual;
  const int y_f32 = LEAN ? 0 : P.y_f32;
  const int emit = P.emit;
  const long long wlim = P.wait_limit > 0 ? P.wait_limit : kWaitLimitCycles;
  const __nv_bfloat16* const xin = P.x;
  const uint32_t* const in_blk = P.in_blk;
  const int in_C32 = P.in_C32;
  const unsigned long long* const in_rowbm = P.in_rowbm;
  const int in_W64 = P.in_W64;
  uint32_t* const err = P.err;
  void* const yout = P.y;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sA = sbase + C::kAOff;
  const uint32_t sB = sbase + C::kBOff;
  const uint32_t sStg = sbase + C::kStgOff;
  const uint32_t bar_full = sbase + C::kBarOff;  // + 8*s
  const uint32_t bar_empty = bar_full + 8 * S;   // + 8*s
  const uint32_t bar_accf = bar_empty + 8 * S;   // + 8*b
  const uint32_t bar_acce = bar_accf + 16;       // + 8*b
  const uint32_t bar_drain = bar_acce + 16;      // after an abort: the MMAs issued so far are done
  int* flags = reinterpret_cast<int*>(smem + C::kFlagOff);
  int* stage_last = flags;                // [S]: 1 = last stage of its tile
  volatile int* s_abort = flags + S;      // CTA-wide abort request
  volatile int* s_last = flags + S + 2;   // [2] split K: this unit finishes its tile
  int* s_issued = flags + S + 4;          // stages the producer filled (for the drain after an abort)
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(flags + S + 1);
  uint32_t* s_kbits = reinterpret_cast<uint32_t*>(smem + C::kKBitsOff);
  unsigned long long* s_tap = reinterpret_cast<unsigned long long*>(smem + C::kTapOff);
  float* s_scale = reinterpret_cast<float*>(smem + C::kScaleOff);
  float* s_shift = reinterpret_cast<float*>(smem + C::kShiftOff);
  const uint32_t sScale = sbase + C::kScaleOff;
  const uint32_t sShift = sbase + C::kShiftOff;
  uint32_t* s_cnt = reinterpret_cast<uint32_t*>(smem + C::kCntOff);  // [4][BN]
  uint32_t* s_acc = reinterpret_cast<uint32_t*>(smem + C::kAccOff);  // [N] non-zeros per column
  unsigned long long* s_rowbm = reinterpret_cast<unsigned long long*>(smem + C::kRowOff);
  uint32_t* s_blk = reinterpret_cast<uint32_t*>(smem + C::kBlkOff);
  // Column counts of all tiles a CTA handles are summed here and flushed once
  // (atomics on one address from every tile would serialise in L2).
  const bool acc_smem = emit && p.N <= kMaxAccCols;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int kblocks = (p.Ktot + BK - 1) / BK;
  const int kgroups = (p.Ktot + 31) / 32;  // 32-column groups of K (compacted zero-skip GEMM)
  const int nt = (p.N + BN - 1) / BN;
  const int mtiles = p.conv == 2 ? ((p.Nimg + p.bn - 1) / p.bn) * p.th * p.tw : (p.M + kBM - 1) / kBM;
  const int tiles = mtiles * nt;
  // split K: work unit u = (tile u / KS, K range u % KS); KS consecutive units
  // (run by neighbouring CTAs at the same time) share one output tile
  const int KS = (!LEAN && P.ksplit > 1) ? P.ksplit : 1;
  const int units = tiles * KS;

  if (!LEAN && P.dense_only) {
    // launched next to the fused small-FC kernel, which handles the zero-skip
    // path: decide first, and leave before any set-up when it is not ours
    pdl_wait();
    if (decide_path(P.disp) == 2) {
      pdl_trigger();
      return;
    }
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(bar_full + 8 * s, (!LEAN && p.conv == 1) ? 129u : 1u);
      mbar_init(bar_empty + 8 * s, 1u);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_accf + 8 * b, 1u);
      mbar_init(bar_acce + 8 * b, (uint32_t)kEpiThreads);
    }
    mbar_init(bar_drain, 1u);
    *s_abort = 0;
    fence_mbar_init();
    if (p.conv != 1) prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    if (p.conv == 0 && BK == 64) {
      prefetch_tmap(&tmA32);
      prefetch_tmap(&tmB32);
    }
    if (!y_f32) prefetch_tmap(&tmY);
  }
  if (warp == kMmaWarp) tmem_alloc(smem_u32(s_tmem), C::kTmemCols);
  if (acc_smem && warp >= 4 && warp < kMmaWarp)
    for (int c = threadIdx.x - 128; c < p.N; c += kEpiThreads) s_acc[c] = 0u;
  if (warp >= 4 && warp < kMmaWarp) {
    for (int i = threadIdx.x - 128; i < 2 * kBM; i += kEpiThreads) s_rowbm[i] = 0ull;
    for (int i = threadIdx.x - 128; i < 2 * (BN / 32); i += kEpiThreads) s_blk[i] = 0u;
  }
  // The producers' first work unit is laid out before the grid dependency
  // wait: no memory is read, and under programmatic dependent launch this
  // overlaps the tail of the kernel before.
  UnitGeo ug{};
  if (warp < 4 && (int)blockIdx.x < units) ug = unit_geo(p, blockIdx.x, KS, kblocks, nt, BN, BK, threadIdx.x);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;
  pdl_wait();
  pdl_trigger();
  const int path = decide_path(P.disp);
  // with dense_only the zero-skip kernel of this launch runs instead
  const bool run = !(!LEAN && P.dense_only && path == 2);
  if (run) record_path(P.disp, path);
  const bool skip = (path == 2);
  // zero-skip GEMM with 64-wide K blocks: stages hold two occupied 32-column
  // groups each (compacted), loaded as 32-column boxes with the 64-byte swizzle
  const bool compact = skip && p.conv == 0 && BK == 64 && kgroups <= kMaxKWords * 32 && in_blk != nullptr;

  if (!run) {
    // nothing to do; fall through to the common exit (TMEM is freed there)
  } else if (warp < 4) {
    // ------------------------------------------------------------------ producers
    const int r = threadIdx.x;
    const int cb_per_tap = p.Cp / BK;
    int it = 0;        // stages filled so far (ring position)
    int pending = 0;   // mode 1: filled stages whose A arrivals are still owed
    bool ok = true;
    // dense TMA modes: thread 0 issues everything, the other producer threads
    // have no part in the loop (their tile geometry would only take issue
    // slots from the epilogue warps on the same schedulers)
    const bool lone = !skip && (LEAN || p.conv != 1);
    for (int u = (lone && r != 0) ? units : (int)blockIdx.x; u < units; u += gridDim.x) {
      if (u != (int)blockIdx.x) ug = unit_geo(p, u, KS, kblocks, nt, BN, BK, r);
      const int kb0 = ug.kb0, kb1 = ug.kb1;
      const TileGeo g = ug.g;
      const bool rvalid = ug.rvalid;
      const int img = ug.img, oh = ug.oh, ow = ug.ow;
      int last = kb1 - 1;
      if (skip) {
        // ---- occupied K blocks of this tile
        named_bar_sync(1, 128);  // thread 0 is done with the previous tile's bits
        if (compact) {
          // occupied 32-column groups of this unit's K range in the tile's
          // 128-row block: one bit per group
          const int g0 = 2 * kb0, g1 = 2 * kb1 < kgroups ? 2 * kb1 : kgroups;
          const uint32_t* words = in_blk + (int64_t)(g.m0 >> 7) * in_C32;
          for (int w0 = 0; w0 < kgroups && w0 < kMaxKWords * 32; w0 += 128) {
            const int gi = w0 + r;
            const bool occ = gi >= g0 && gi < g1 && words[gi] != 0u;
            const uint32_t bits = __ballot_sync(0xffffffffu, occ);
            if (lane == 0 && (w0 >> 5) + warp < kMaxKWords) s_kbits[(w0 >> 5) + warp] = bits;
          }
        } else if (p.conv == 0) {
          for (int w0 = 0; w0 < kblocks && w0 < kMaxKWords * 32; w0 += 128) {
            const int kb = w0 + r;
            // a K block covers BK / 32 words of the 128-row block-column mask
            // (an input without block masks, such as the im2col rows of a
            // narrow stem, keeps every block)
            bool occ = false;
            if (kb < kblocks && in_blk == nullptr) {
              occ = true;
            } else if (kb < kblocks) {
              const uint32_t* words = in_blk + (int64_t)(g.m0 >> 7) * in_C32;
              occ = words[kb * (BK / 32)] != 0u;
              if (BK == 64 && kb * 2 + 1 < in_C32) occ |= words[kb * 2 + 1] != 0u;
            }
            const uint32_t bits = __ballot_sync(0xffffffffu, occ);
            if (lane == 0 && (w0 >> 5) + warp < kMaxKWords) s_kbits[(w0 >> 5) + warp] = bits;
          }
        } else {
          if (r < kMaxTaps) s_tap[r] = 0ull;
          named_bar_sync(1, 128);
          const int taps = p.kh * p.kw < kMaxTaps ? p.kh * p.kw : kMaxTaps;
          for (int t0 = 0; t0 < taps; t0 += 8) {
            unsigned long long wv[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {  // issue 8 taps' loads before reducing any
              const int tp = t0 + u;
              const int ih = oh * p.stride - p.pad + tp / p.kw;
              const int iw = ow * p.stride - p.pad + tp % p.kw;
              wv[u] = 0ull;
              if (in_rowbm && tp < taps && rvalid && ih >= 0 && ih < p.H && iw >= 0 && iw < p.W)
                wv[u] = in_rowbm[(((int64_t)img * p.H + ih) * p.W + iw) * in_W64];
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              unsigned long long w = wv[u];
#pragma unroll
              for (int s = 16; s > 0; s >>= 1) w |= __shfl_xor_sync(0xffffffffu, w, s);
              if (lane == 0 && w) atomicOr(&s_tap[t0 + u], w);
            }
          }
          named_bar_sync(1, 128);
          // no per-tap masks (too many taps, wide rows, or an input given without
          // row bitmaps): keep every block
          const bool many = p.kh * p.kw > kMaxTaps || in_W64 > 1 || in_rowbm == nullptr;
          for (int w0 = 0; w0 < kblocks && w0 < kMaxKWords * 32; w0 += 128) {
            const int kb = w0 + r;
            bool occ = false;
            if (kb < kblocks) {
              if (many) {
                occ = true;
              } else {
#pragma unroll
                for (int j = 0; j < BK / 8; ++j) {
                  const int flat = kb * BK + 8 * j;
                  if (flat >= p.Ktot) break;
                  const int tp = flat / p.Cp;
                  const int c = flat - tp * p.Cp;
                  occ |= ((s_tap[tp] >> (c >> 6)) & 1ull) != 0ull;
                }
              }
            }
            const uint32_t bits = __ballot_sync(0xffffffffu, occ);
            if (lane == 0 && (w0 >> 5) + warp < kMaxKWords) s_kbits[(w0 >> 5) + warp] = bits;
          }
        }
        named_bar_sync(1, 128);
        // last occupied block of this unit's K range; a range with none still
        // runs its first block (whose data is all zero)
        last = kb0;
        if (compact) last = kb1 - 1;  // unused: the compacted loop tracks its own last stage
        for (int kb = kb1 - 1; kb > kb0; --kb) {
          if (kb >= kMaxKWords * 32 || ((s_kbits[kb >> 5] >> (kb & 31)) & 1u)) {
            last = kb;
            break;
          }
        }
      }
      if (!ok) continue;  // keep the skip-mask barriers in step; issue nothing more
      if (compact) {
        if (r == 0) {
          // pairs of occupied groups in increasing order; an odd last group
          // takes a stage alone; a unit with none runs group g0 (all zero) so
          // that its accumulator is written
          const int g0 = 2 * kb0, g1 = 2 * kb1 < kgroups ? 2 * kb1 : kgroups;
          int cnt = 0;
          for (int wd = g0 >> 5; wd <= (g1 - 1) >> 5; ++wd) cnt += __popc(s_kbits[wd]);
          const int nst = cnt ? (cnt + 1) / 2 : 1;
          int slot = it % S;
          uint32_t ph = (uint32_t)((it / S) & 1);
          int st = 0, pend = -1;
          auto issue = [&](int ga, int gb) -> bool {
            if (it >= S && !mbar_wait(bar_empty + 8 * slot, ph ^ 1u, err, s_abort, kErrTimeoutEmpty, wlim)) return false;
            const uint32_t fb = bar_full + 8 * slot;
            const int nh = gb >= 0 ? 2 : 1;
            stage_last[slot] = (st == nst - 1 ? 1 : 0) | (nh == 1 ? 2 : 0);
            mbar_arrive_expect_tx(fb, (uint32_t)(nh * (kBM * 64 + BN * 64)));
            tma_load_2d(sA + slot * C::kAStage, &tmA32, fb, ga * 32, g.m0);
            tma_load_2d(sB + slot * C::kBStage, &tmB32, fb, ga * 32, g.n0);
            if (nh == 2) {
              tma_load_2d(sA + slot * C::kAStage + kBM * 64, &tmA32, fb, gb * 32, g.m0);
              tma_load_2d(sB + slot * C::kBStage + BN * 64, &tmB32, fb, gb * 32, g.n0);
            }
            ++st;
            ++it;
            if (++slot == S) {
              slot = 0;
              ph ^= 1u;
            }
            return true;
          };
          if (cnt == 0) {
            ok = issue(g0, -1);
          } else {
            for (int wd = g0 >> 5; wd <= (g1 - 1) >> 5 && ok; ++wd) {
              uint32_t bits = s_kbits[wd];
              while (bits && ok) {
                const int gi = wd * 32 + __ffs(bits) - 1;
                bits &= bits - 1u;
                if (pend < 0) {
                  pend = gi;
                } else {
                  ok = issue(pend, gi);
                  pend = -1;
                }
              }
            }
            if (ok && pend >= 0) ok = issue(pend, -1);
          }
        }
      } else if (LEAN || p.conv != 1) {
        if (r == 0) {
          // The issuing lane is slow at anything but issuing: ring slot, phase
          // and the (tap, channel block) of each K block advance incrementally,
          // with no divisions in the loop, and the ring's first lap (whose
          // slots are free by construction) waits for nothing.
          int slot = it % S;
          uint32_t ph = (uint32_t)((it / S) & 1);
          int cb = ug.cb, rr = ug.rr, ss = ug.ss;  // conv = 2: channel block and tap of block kb
          const int iy0 = ug.iy0, ix0 = ug.ix0;
          const uint32_t fb0 = bar_full, eb0 = bar_empty;
          for (int kb = kb0; kb <= last; ++kb) {
            const bool issue =
                !(skip && kb != last && kb < kMaxKWords * 32 && !((s_kbits[kb >> 5] >> (kb & 31)) & 1u));
            if (issue) {
              if (it >= S && !mbar_wait(eb0 + 8 * slot, ph ^ 1u, err, s_abort, kErrTimeoutEmpty, wlim)) {
                ok = false;
                break;
              }
              const uint32_t fb = fb0 + 8 * slot;
              stage_last[slot] = (kb == last) ? 1 : 0;
              mbar_arrive_expect_tx(fb, (uint32_t)C::kStageBytes);
              if (p.conv == 0)
                tma_load_2d(sA + slot * C::kAStage, &tmA, fb, kb * BK, g.m0);
              else
                tma_load_4d(sA + slot * C::kAStage, &tmA, fb, cb * BK, ix0 + ss, iy0 + rr, g.tn0);
              tma_load_2d(sB + slot * C::kBStage, &tmB, fb, kb * BK, g.n0);
              ++it;
              if (++slot == S) {
                slot = 0;
                ph ^= 1u;
              }
            }
            if (p.conv == 2 && ++cb == cb_per_tap) {
              cb = 0;
              if (++ss == p.kw) {
                ss = 0;
                ++rr;
              }
            }
          }
        }
      } else {
        // Implicit-GEMM gather: row r is output pixel m0 + r.
        const int ih0 = oh * p.stride - p.pad;
        const int iw0 = ow * p.stride - p.pad;
        const __nv_bfloat16* ximg = xin + (int64_t)img * p.H * p.W * p.Cp;
        for (int kb = kb0; kb <= last; ++kb) {
          if (skip && kb != last && kb < kMaxKWords * 32 && !((s_kbits[kb >> 5] >> (kb & 31)) & 1u))
            continue;
          const int slot = it % S;
          const uint32_t ph = (uint32_t)((it / S) & 1);
          if (!mbar_wait(bar_empty + 8 * slot, ph ^ 1u, err, s_abort, kErrTimeoutEmpty, wlim)) {
            ok = false;
            break;
          }
          if (r == 0) {
            stage_last[slot] = (kb == last) ? 1 : 0;
            mbar_arrive_expect_tx(bar_full + 8 * slot, (uint32_t)C::kBStage);
            tma_load_2d(sB + slot * C::kBStage, &tmB, bar_full + 8 * slot, kb * BK, g.n0);
          }
          const uint32_t dst = sA + slot * C::kAStage;
          // (tap, channel) of the block's first 8-channel chunk by division,
          // the block's other chunks by stepping (C % 8 == 0)
          const int flat0 = kb * BK;
          const int tp0 = flat0 / p.Cp;
          int c = flat0 - tp0 * p.Cp;
          int rr = tp0 / p.kw;
          int ss = tp0 - rr * p.kw;
#pragma unroll
          for (int j = 0; j < BK / 8; ++j) {
            const int flat = flat0 + 8 * j;
            const int ih = ih0 + rr, iw = iw0 + ss;
            const bool val = rvalid && flat < p.Ktot && ih >= 0 && ih < p.H && iw >= 0 && iw < p.W;
            const __nv_bfloat16* src = val ? ximg + ((int64_t)ih * p.W + iw) * p.Cp + c : xin;
            cp_async_16(dst + swz_offset<BK>(r, j), src, val ? 16u : 0u);
            c += 8;
            if (c == p.Cp) {
              c = 0;
              if (++ss == p.kw) {
                ss = 0;
                ++rr;
              }
            }
          }
          cp_async_commit();
          ++it;
          ++pending;
          if (pending > C::kLag) {
            cp_async_wait<C::kLag>();
            fence_proxy_async_smem();
            mbar_arrive(bar_full + 8 * ((it - 1 - C::kLag) % S));
            --pending;
          }
        }
      }
    }
    if (r == 0) *s_issued = it;  // stages this CTA filled (TMA copies issued)
    if (!LEAN && p.conv == 1) {
      cp_async_wait<0>();
      fence_proxy_async_smem();
      for (int q = pending; q > 0; --q) mbar_arrive(bar_full + 8 * ((it - q) % S));
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------------ MMA issue
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, BN);
      int it = 0, j = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x, ++j) {
        const int b = j & 1;
        if (!mbar_wait(bar_acce + 8 * b, (uint32_t)(((j >> 1) & 1) ^ 1), err, s_abort,
                       kErrTimeoutAcc, wlim))
          break;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)b * C::kAccCols;
        bool first = true;
        int slot = it % S;
        uint32_t ph = (uint32_t)((it / S) & 1);
        while (true) {
          if (!mbar_wait(bar_full + 8 * slot, ph, err, s_abort, kErrTimeoutFull, wlim)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const int sflags = stage_last[slot];
          const bool last = (sflags & 1) != 0;
          const uint32_t a = sA + slot * C::kAStage;
          const uint32_t bb = sB + slot * C::kBStage;
          if (compact) {
            // one or two 32-column groups, each 128 (A) / BN (B) rows of 64
            // bytes with the 64-byte swizzle: two k-steps of 16 per group
            const uint64_t a0 = smem_desc_sw64(a), b0 = smem_desc_sw64(bb);
            if (first) tc_mma_bf16(d, a0, b0, idesc, 0u);
            else tc_mma_bf16(d, a0, b0, idesc, 1u);
            tc_mma_bf16(d, a0 + 2, b0 + 2, idesc, 1u);
            if (!(sflags & 2)) {
              const uint64_t a1 = smem_desc_sw64(a + kBM * 64), b1 = smem_desc_sw64(bb + BN * 64);
              tc_mma_bf16(d, a1, b1, idesc, 1u);
              tc_mma_bf16(d, a1 + 2, b1 + 2, idesc, 1u);
            }
            first = false;
            tc_commit(bar_empty + 8 * slot);
            ++it;
            if (++slot == S) {
              slot = 0;
              ph ^= 1u;
            }
            if (last) break;
            continue;
          }
          // k-steps advance the start-address field by 32 B (2 units); the
          // accumulate flags are constants on both branches (a per-MMA flag
          // computed at run time roughly halves the issue rate)
          const uint64_t ad = smem_desc_kmajor<BK>(a), bd = smem_desc_kmajor<BK>(bb);
          if (first) {
            tc_mma_bf16(d, ad, bd, idesc, 0u);
#pragma unroll
            for (int k = 1; k < BK / 16; ++k)
              tc_mma_bf16(d, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, 1u);
          } else {
#pragma unroll
            for (int k = 0; k < BK / 16; ++k)
              tc_mma_bf16(d, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc, 1u);
          }
          first = false;
          tc_commit(bar_empty + 8 * slot);
          ++it;
          if (++slot == S) {
            slot = 0;
            ph ^= 1u;
          }
          if (last) break;
        }
        // (the fault injection of the error-path tests leaves the first
        // accumulator unsignalled: the epilogue's bounded wait runs out)
        if (ok && !(P.fault == kFaultSkipFirstAccCommit && j == 0)) tc_commit(bar_accf + 8 * b);
      }
    }
  } else if constexpr (LEAN) {
    // ------------------------------------------------------------- lean epilogue
    // The general epilogue's blocks (32 rows of one TMEM lane quarter x 32
    // columns, staged with the 64-byte swizzle, one TMA store each) without
    // K split or fp32 output, and with one barrier per tile: the
    // output occupancy a tile leaves in shared memory (row bitmaps and block-
    // column words, buffer j & 1) is written out after the next tile's
    // barrier, and column counts go straight into the CTA's column sums.
    const int q = warp & 3;
    const int hf = (warp - 4) >> 2;
    const int ew = warp - 4;
    const int r = q * 32 + lane;
    const int et = threadIdx.x - 128;
    int sw_ = 0, sh_ = 0, sn_ = 0;
    if (p.conv == 2) {
      const int rho = q * 32;
      sw_ = rho % p.bw;
      sh_ = (rho / p.bw) % p.bh;
      sn_ = rho / (p.bw * p.bh);
    }
    const uint32_t stg_base = sStg + (uint32_t)(ew * 2 * kWarpStgBytes);
    const bool fixed_cols = nt == 1 || (int)gridDim.x % nt == 0 || units <= (int)gridDim.x;
    if (fixed_cols && (int)blockIdx.x < units) {
      const int n0 = ((int)blockIdx.x % nt) * BN;
      for (int c = et; c < BN; c += kEpiThreads) {
        float sc = 1.f, sh = 0.f;
        if (n0 + c < p.N) epi_affine(ep, p.N, n0 + c, sc, sh);
        s_scale[c] = sc;
        s_shift[c] = sh;
      }
    }
    const bool affine = ep.bias != nullptr || ep.bn != nullptr;  // else the column affine is 1, 0
    const OccDev o = P.out_occ;
    // Writes out the occupancy that tile (m0, n0) left in buffer pb: the row
    // bitmap word of row r (its half-0 thread) and the block-column words of
    // its 128-row block (mode 0: the tile is that block).
    auto flush_tile = [&](int pb, int64_t m_t, bool v_t, int m0_t, int n0_t) {
      if (hf == 0) {
        unsigned long long* const srow = s_rowbm + pb * kBM + r;
        const unsigned long long v = *srow;
        *srow = 0ull;
        if (v_t) {
          unsigned long long* dst = &o.row_bm[m_t * o.W64 + (n0_t >> 12)];
          if (nt == 1) *dst = v;  // the tile spans the row's whole bitmap word
          else if (v) atomicOr(dst, v);
        }
      }
      if (p.conv != 2 && et < BN / 32) {
        uint32_t* const sb = s_blk + pb * (BN / 32) + et;
        const uint32_t v = *sb;
        *sb = 0u;
        const int word = (n0_t >> 5) + et;
        if (word < o.C32) o.blk_mask[(m0_t >> 7) * o.C32 + word] = v;
      }
    };
    int j = 0;
    int stg_count = 0;
    int64_t m_prev = 0;
    bool v_prev = false;
    int m0_prev = 0, n0_prev = 0;
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++j) {
      const int b = j & 1;
      const TileGeo g = tile_geo(p, u, nt, BN);
      bool mvalid;
      int img, oh, ow;
      const int64_t m = tile_row(p, g, r, mvalid, img, oh, ow);
      if (LEAN == 2 && mvalid) {
        // this row's residual segments into L1 while the accumulator is pending
        const __nv_bfloat16* rrow = residual + m * p.N + g.n0 + hf * 32;
        for (int gc = 0; gc < BN / 64; ++gc)
          if (g.n0 + gc * 64 + hf * 32 < p.N) prefetch_l1(rrow + gc * 64);
      }
      float* const scb = s_scale + (fixed_cols ? 0 : b * BN);
      float* const shb = s_shift + (fixed_cols ? 0 : b * BN);
      if (!fixed_cols) {
        for (int c = et; c < BN; c += kEpiThreads) {
          float sc = 1.f, sh = 0.f;
          if (g.n0 + c < p.N) epi_affine(ep, p.N, g.n0 + c, sc, sh);
          scb[c] = sc;
          shb[c] = sh;
        }
      }
      const bool ok = mbar_wait(bar_accf + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutAcc, wlim);
      if (named_bar_or(2, kEpiThreads, !ok)) break;
      if (emit && j > 0) flush_tile(b ^ 1, m_prev, v_prev, m0_prev, n0_prev);
      tc_fence_after();
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)b * C::kAccCols;
      const int blk = mvalid ? (int)(m >> 7) : -1;
      const uint32_t grp = p.conv == 2 ? __match_any_sync(0xffffffffu, blk) : 0xffffffffu;
      const bool leader = (__ffs(grp) - 1) == lane;
      unsigned long long tl = 0ull;
      // One block: columns ncol0..+31 of 64-column group gcol, accumulator
      // values in raw, staged in buffer stg; the TMA store and this block's
      // share of the output occupancy.
      auto block = [&](const uint32_t (&raw)[32], int gcol, uint32_t stg) {
        const int nbase = g.n0 + gcol * 64;
        const int ncol0 = nbase + hf * 32;
        const float* scg = affine ? scb + gcol * 64 + hf * 32 : nullptr;
        const float* shg = shb + gcol * 64 + hf * 32;
        const uint4* rp =
            residual && mvalid ? reinterpret_cast<const uint4*>(residual + m * p.N + ncol0) : nullptr;
        const int rvalid = p.N - ncol0 < 32 ? p.N - ncol0 : 32;
        uint32_t pk[16];
        constexpr bool kRes = LEAN == 2;
        if (act == 1) affine_act_pack32<1, kRes>(raw, scg, shg, rp, rvalid, pk);
        else if (act == 2) affine_act_pack32<2, kRes>(raw, scg, shg, rp, rvalid, pk);
        else if (act == 0) affine_act_pack32<0, kRes>(raw, scg, shg, rp, rvalid, pk);
        else affine_act_pack32<3, kRes>(raw, scg, shg, rp, rvalid, pk);
        const uint32_t row_addr = stg + (uint32_t)lane * 64u;
        const int sx = (lane >> 1) & 3;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          sts_u4(row_addr + (uint32_t)((k ^ sx) << 4), make_uint4(pk[4 * k], pk[4 * k + 1], pk[4 * k + 2], pk[4 * k + 3]));
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (p.conv == 2)
            tma_store_4d(&tmY, stg, ncol0, g.tw0 + sw_, g.th0 + sh_, g.tn0 + sn_);
          else
            tma_store_2d(&tmY, stg, ncol0, g.m0 + q * 32);
          bulk_commit();
        }
        if (emit) {
          uint32_t rw = nz_mask32(pk);  // bit c: column ncol0 + c of row r is non-zero
          const int nvalid = p.N - ncol0;
          if (!mvalid) rw = 0u;
          else if (nvalid < 32) rw &= nvalid > 0 ? ((1u << nvalid) - 1u) : 0u;
          if (rw) tl |= 1ull << ((nbase >> 6) & 63);
          const uint32_t bits = __reduce_or_sync(grp, rw);
          const int word = ncol0 >> 5;
          if (leader && blk >= 0 && bits && word < o.C32) {
            if (p.conv == 2) atomicOr(&o.blk_mask[blk * o.C32 + word], bits);
            else atomicOr(&s_blk[b * (BN / 32) + gcol * 2 + hf], bits);  // the tile is the whole block
          }
          // lane c: non-zeros of column ncol0 + c in the warp's 32 rows
          const uint32_t cnt = __popc(warp_transpose32(rw));
          const int col = ncol0 + lane;
          if (acc_smem) {
            if (cnt) atomicAdd(&s_acc[col], cnt);
          } else if (col < o.C) {
            if (cnt) atomicAdd(&o.col_nnz[col], cnt);
            const uint32_t sum = __reduce_add_sync(0xffffffffu, cnt);
            if (lane == 0 && sum) {
              atomicAdd(&o.tile_nnz[ncol0 >> 6], sum);
              atomicAdd(o.nnz, (unsigned long long)sum);
            }
          }
        }
      };
      // This warp's blocks of the tile (32-column halves past N have none).
      // (Two blocks per step, both accumulator loads in flight first, made
      // the kernel spill and was slower.)
      int nblk = 0;
      for (int gc = 0; gc < BN / 64; ++gc) nblk += (g.n0 + gc * 64 + hf * 32 < p.N) ? 1 : 0;
#pragma unroll 1
      for (int gcol = 0; gcol < nblk; ++gcol) {
        const uint32_t stg = stg_base + (uint32_t)((stg_count & 1) * kWarpStgBytes);
        if (lane == 0) bulk_wait_read<1>();  // the store that used this buffer has read it
        __syncwarp();
        uint32_t raw[32];
        tmem_ld32_nowait(tbase + (uint32_t)(gcol * 64 + hf * 32), raw);
        tmem_wait_ld32(raw);
        block(raw, gcol, stg);
        ++stg_count;
      }
      // accumulator b is free for the MMA of tile j + 2
      tc_fence_before();
      mbar_arrive(bar_acce + 8 * b);
      if (emit) {
        if (tl) atomicOr(&s_rowbm[b * kBM + r], tl);
        m_prev = m;
        v_prev = mvalid;
        m0_prev = g.m0;
        n0_prev = g.n0;
      }
    }
    if (emit) {
      named_bar_sync(2, kEpiThreads);  // the last tile's shared-memory occupancy is complete
      if (j > 0) flush_tile((j - 1) & 1, m_prev, v_prev, m0_prev, n0_prev);
    }
    if (acc_smem) {
      named_bar_sync(2, kEpiThreads);
      unsigned long long total = 0ull;
      for (int c0 = 0; c0 < p.N; c0 += kEpiThreads) {
        const int c = c0 + et;
        const uint32_t cnt = c < p.N ? s_acc[c] : 0u;
        if (cnt) atomicAdd(&o.col_nnz[c], cnt);
        uint32_t sum = cnt;
#pragma unroll
        for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
        total += sum;
        if (lane == 0 && sum) atomicAdd(&o.tile_nnz[c >> 6], sum);
      }
      if (lane == 0 && total) atomicAdd(o.nnz, total);
    }
    if (lane == 0) bulk_wait_all();
  } else {
    // ------------------------------------------------------------------ epilogue
    // Each epilogue warp owns a 32-row x 32-column block of every 64-column
    // group (rows from its TMEM lane quarter, columns from its half) and
    // stores it on its own: staging in shared memory with the 64-byte swizzle
    // and one TMA store per block, so the warps never wait for each other
    // inside a tile.  The only barrier per tile publishes the column affine
    // (double-buffered by accumulator), plus one for the output occupancy.
    const int q = warp & 3;            // TMEM lane quarter of this warp
    const int hf = (warp - 4) >> 2;    // which 32 columns of each 64-column group
    const int ew = warp - 4;           // epilogue warp index
    const int r = q * 32 + lane;       // tile row
    const int et = threadIdx.x - 128;  // 0..kEpiThreads-1
    const bool vec = (p.N % 8) == 0;
    const bool affine = ep.bias != nullptr || ep.bn != nullptr;  // else the column affine is 1, 0
    // this warp's 32-row sub-box of the tile: {32 channels, bw', bh', bn'} for
    // spatial tiles, 32 consecutive rows otherwise
    int sw_ = 0, sh_ = 0, sn_ = 0;
    if (p.conv == 2) {
      const int rho = q * 32;
      sw_ = rho % p.bw;
      sh_ = (rho / p.bw) % p.bh;
      sn_ = rho / (p.bw * p.bh);
    }
    const uint32_t stg_base = sStg + (uint32_t)(ew * 2 * kWarpStgBytes);
    // Tile t covers columns (t % nt) BN..; when every tile of this CTA has the
    // same columns (one column tile, or a grid that is a multiple of the column
    // tiles) the column affine is computed once, into buffer 0, instead of per
    // tile (its global loads would otherwise sit on every tile's critical path)
    const bool fixed_cols = KS == 1 && (nt == 1 || (int)gridDim.x % nt == 0 || units <= (int)gridDim.x);
    if (fixed_cols && (int)blockIdx.x < units) {
      const int n0 = ((int)blockIdx.x % nt) * BN;
      for (int c = et; c < BN; c += kEpiThreads) {
        float sc = 1.f, sh = 0.f;
        if (n0 + c < p.N) epi_affine(ep, p.N, n0 + c, sc, sh);
        s_scale[c] = sc;
        s_shift[c] = sh;
      }
    }
    int j = 0;
    int stg_count = 0;  // blocks this warp handed to TMA so far
    for (int u = blockIdx.x; u < units; u += gridDim.x, ++j) {
      const int t = u / KS, ks = u - (u / KS) * KS;
      const int b = j & 1;
      const TileGeo g = tile_geo(p, t, nt, BN);
      bool mvalid;
      int img, oh, ow;
      const int64_t m = tile_row(p, g, r, mvalid, img, oh, ow);
      float* const scb = s_scale + (fixed_cols ? 0 : b * BN);
      float* const shb = s_shift + (fixed_cols ? 0 : b * BN);
      // column affine of this tile into buffer b (its readers of tile j - 2
      // passed tile j - 1's barrier before any thread gets here)
      if (!fixed_cols) {
        for (int c = et; c < BN; c += kEpiThreads) {
          float sc = 1.f, sh = 0.f;
          if (g.n0 + c < p.N) epi_affine(ep, p.N, g.n0 + c, sc, sh);
          scb[c] = sc;
          shb[c] = sh;
        }
      }
      const bool ok = mbar_wait(bar_accf + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutAcc, wlim);
      // publishes the affine, and makes the abort decision the same for every
      // epilogue warp (a warp that left alone would strand the others at a barrier)
      if (named_bar_or(2, kEpiThreads, !ok)) break;
      tc_fence_after();
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)b * C::kAccCols;
      // split K: every unit stores its fp32 partial tile, then takes a ticket;
      // the unit that arrives last adds the others' partials and finishes the
      // tile (nobody waits for anybody)
      float* const ws_tile = KS > 1 ? P.ws + (int64_t)t * KS * kBM * BN : nullptr;
      if (KS > 1) {
        float* const mine = ws_tile + ((int64_t)ks * kBM + r) * BN + hf * 32;
#pragma unroll 1
        for (int gcol = 0; gcol < BN / 64; ++gcol) {
          uint32_t raw[32];
          tmem_ld32_nowait(tbase + (uint32_t)(gcol * 64 + hf * 32), raw);
          tmem_wait_ld32(raw);
          float4* dst = reinterpret_cast<float4*>(mine + gcol * 64);
#pragma unroll
          for (int i = 0; i < 8; ++i)
            __stcg(dst + i, make_float4(__uint_as_float(raw[4 * i]), __uint_as_float(raw[4 * i + 1]),
                                        __uint_as_float(raw[4 * i + 2]), __uint_as_float(raw[4 * i + 3])));
        }
        // One thread publishes the partial and takes the ticket: the barrier
        // orders every epilogue thread's stores before that thread's fence
        // (fences are cumulative), and the last arriver's fence after the
        // ticket orders the other units' partials before the reads below,
        // which the second barrier hands on to every thread.
        named_bar_sync(2, kEpiThreads);
        if (et == 0) {
          __threadfence();
          const int lst = atomicAdd(&P.ws_cnt[t], 1u) == (unsigned)(KS - 1) ? 1 : 0;
          if (lst) {
            __threadfence();
            P.ws_cnt[t] = 0u;  // every unit of the tile has arrived: ready for reuse
          }
          s_last[b] = lst;
        }
        named_bar_sync(2, kEpiThreads);
        if (!s_last[b]) {
          tc_fence_before();
          mbar_arrive(bar_acce + 8 * b);  // this unit's share is in the partial
          continue;
        }
      }
      const OccDev o = P.out_occ;  // registers, not parameter-space loads
      const int blk = mvalid ? (int)(m >> 7) : -1;
      const uint32_t grp = p.conv == 2 ? __match_any_sync(0xffffffffu, blk) : 0xffffffffu;
      const bool leader = (__ffs(grp) - 1) == lane;
      unsigned long long tl = 0ull;  // this row's occupied 64-column tiles
      // One 64-column group per iteration, kept as a loop (not unrolled) so the
      // epilogue's instructions stay in the instruction cache across groups.
#pragma unroll 1
      for (int gcol = 0; gcol < BN / 64; ++gcol) {
        const int nbase = g.n0 + gcol * 64;
        if (nbase >= p.N) break;  // uniform across the epilogue warps
        const int ncol0 = nbase + hf * 32;  // first column of this warp's block
        uint32_t stg = 0;
        if (!y_f32) {
          stg = stg_base + (uint32_t)((stg_count & 1) * kWarpStgBytes);
          if (lane == 0) bulk_wait_read<1>();  // the store that used this buffer has read it
          __syncwarp();
        }
        uint32_t raw[32];
        tmem_ld32_nowait(tbase + (uint32_t)(gcol * 64 + hf * 32), raw);
        tmem_wait_ld32(raw);
        if (KS > 1) {
          // the other units' partials of this row's 32 columns, in two halves:
          // every load of a half in flight before the first is used, added in
          // unit order
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            float4 pv[kMaxSplit - 1][4];
#pragma unroll
            for (int k2i = 0; k2i < kMaxSplit - 1; ++k2i) {
              const int k2 = k2i < ks ? k2i : k2i + 1;
              if (k2 < KS) {
                const float4* src = reinterpret_cast<const float4*>(
                    ws_tile + ((int64_t)k2 * kBM + r) * BN + gcol * 64 + hf * 32 + h * 16);
#pragma unroll
                for (int i = 0; i < 4; ++i) pv[k2i][i] = __ldcg(src + i);
              }
            }
#pragma unroll
            for (int k2i = 0; k2i < kMaxSplit - 1; ++k2i) {
              const int k2 = k2i < ks ? k2i : k2i + 1;
              if (k2 < KS) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                  uint32_t* q4 = raw + h * 16 + 4 * i;
                  q4[0] = __float_as_uint(__uint_as_float(q4[0]) + pv[k2i][i].x);
                  q4[1] = __float_as_uint(__uint_as_float(q4[1]) + pv[k2i][i].y);
                  q4[2] = __float_as_uint(__uint_as_float(q4[2]) + pv[k2i][i].z);
                  q4[3] = __float_as_uint(__uint_as_float(q4[3]) + pv[k2i][i].w);
                }
              }
            }
          }
        }
        uint32_t rw = 0u;  // non-zero bits of this row in the warp's 32 columns
        const float* scg = scb + gcol * 64 + hf * 32;
        const float* shg = shb + gcol * 64 + hf * 32;
#pragma unroll
        for (int c16s = 0; c16s < 2; ++c16s) {
          const int nb = ncol0 + c16s * 16;
          const bool full = vec && (nb + 16 <= p.N);
          const float4* sc4 = reinterpret_cast<const float4*>(scg + c16s * 16);
          const float4* sh4 = reinterpret_cast<const float4*>(shg + c16s * 16);
          float o32[16];
          if (affine) {
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
              const float4 sc = sc4[q4];
              const float4 sh = sh4[q4];
              o32[4 * q4 + 0] = fmaf(__uint_as_float(raw[c16s * 16 + 4 * q4 + 0]), sc.x, sh.x);
              o32[4 * q4 + 1] = fmaf(__uint_as_float(raw[c16s * 16 + 4 * q4 + 1]), sc.y, sh.y);
              o32[4 * q4 + 2] = fmaf(__uint_as_float(raw[c16s * 16 + 4 * q4 + 2]), sc.z, sh.z);
              o32[4 * q4 + 3] = fmaf(__uint_as_float(raw[c16s * 16 + 4 * q4 + 3]), sc.w, sh.w);
            }
          } else {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) o32[jj] = __uint_as_float(raw[c16s * 16 + jj]);
          }
          if (residual && mvalid) {
            const __nv_bfloat16* rp = residual + m * p.N + nb;
            if (full) {
              const uint4 r0 = *reinterpret_cast<const uint4*>(rp);
              const uint4 r1 = *reinterpret_cast<const uint4*>(rp + 8);
              const __nv_bfloat162* h0 = reinterpret_cast<const __nv_bfloat162*>(&r0);
              const __nv_bfloat162* h1 = reinterpret_cast<const __nv_bfloat162*>(&r1);
#pragma unroll
              for (int jj = 0; jj < 4; ++jj) {
                const float2 a0 = __bfloat1622float2(h0[jj]);
                const float2 a1 = __bfloat1622float2(h1[jj]);
                o32[2 * jj] += a0.x;
                o32[2 * jj + 1] += a0.y;
                o32[8 + 2 * jj] += a1.x;
                o32[8 + 2 * jj + 1] += a1.y;
              }
            } else {
              for (int jj = 0; jj < 16; ++jj)
                if (nb + jj < p.N) o32[jj] += __bfloat162float(rp[jj]);
            }
          }
          if (act == 1) {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) o32[jj] = fmaxf(o32[jj], 0.f);
          } else if (act == 2) {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) o32[jj] = fminf(fmaxf(o32[jj], 0.f), 6.f);
          } else if (act == 3) {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) o32[jj] = gelu_f(o32[jj]);
          }
          if (y_f32) {
            if (mvalid) {
              float* yp = reinterpret_cast<float*>(yout) + m * p.N + nb;
              if (full && (p.N % 4) == 0) {
#pragma unroll
                for (int jj = 0; jj < 16; jj += 4)
                  *reinterpret_cast<float4*>(yp + jj) = make_float4(o32[jj], o32[jj + 1], o32[jj + 2], o32[jj + 3]);
              } else {
                for (int jj = 0; jj < 16; ++jj)
                  if (nb + jj < p.N) yp[jj] = o32[jj];
              }
            }
          } else {
            uint32_t pk[8];
#pragma unroll
            for (int jj = 0; jj < 8; ++jj) {
              const __nv_bfloat162 h2 = __floats2bfloat162_rn(o32[2 * jj], o32[2 * jj + 1]);
              pk[jj] = *reinterpret_cast<const uint32_t*>(&h2);
            }
            if (emit) {
              uint32_t nzbits = 0u;
#pragma unroll
              for (int jj = 0; jj < 8; ++jj) {
                nzbits |= ((pk[jj] & 0x7FFFu) ? 1u : 0u) << (2 * jj);
                nzbits |= ((pk[jj] & 0x7FFF0000u) ? 1u : 0u) << (2 * jj + 1);
              }
              const int nvalid = p.N - nb;  // columns of this chunk inside the tensor
              if (!mvalid) nzbits = 0u;
              else if (nvalid < 16) nzbits &= nvalid > 0 ? ((1u << nvalid) - 1u) : 0u;
              rw |= nzbits << (c16s * 16);
            }
            // staging block: 32 rows x 64 bytes, 16-byte chunk k of row `lane` at
            // chunk k ^ ((lane >> 1) & 3) (the TMA 64-byte swizzle)
            const uint32_t row_addr = stg + (uint32_t)lane * 64u;
            const int k0 = c16s * 2;
            const int sx = (lane >> 1) & 3;
            sts_u4(row_addr + (uint32_t)((k0 ^ sx) << 4), make_uint4(pk[0], pk[1], pk[2], pk[3]));
            sts_u4(row_addr + (uint32_t)(((k0 + 1) ^ sx) << 4), make_uint4(pk[4], pk[5], pk[6], pk[7]));
          }
        }
        if (!y_f32) {
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            if (p.conv == 2)
              tma_store_4d(&tmY, stg, ncol0, g.tw0 + sw_, g.th0 + sh_, g.tn0 + sn_);
            else
              tma_store_2d(&tmY, stg, ncol0, g.m0 + q * 32);
            bulk_commit();
          }
          ++stg_count;
        }
        if (emit) {
          // this block's share of the output occupancy
          if (rw) tl |= 1ull << ((nbase >> 6) & 63);
          const uint32_t bits = __reduce_or_sync(grp, rw);
          const int word = (nbase >> 5) + hf;
          if (leader && blk >= 0 && bits && word < o.C32) {
            if (p.conv == 2) atomicOr(&o.blk_mask[blk * o.C32 + word], bits);
            else atomicOr(&s_blk[gcol * 2 + hf], bits);  // the tile is the whole block
          }
          // lane j: non-zeros of column 32 hf + j of this group in the warp's 32 rows
          s_cnt[q * BN + gcol * 64 + hf * 32 + lane] = __popc(warp_transpose32(rw));
        }
      }
      // accumulator b is free for the MMA of tile j + 2
      tc_fence_before();
      mbar_arrive(bar_acce + 8 * b);
      if (emit) {
        // both column halves of a row meet in shared memory; the half-0 thread of
        // the row then writes it once (a plain store when the tile spans every
        // column of the row's bitmap word, i.e. the word is this tile's alone)
        if (tl) atomicOr(&s_rowbm[r], tl);
        named_bar_sync(2, kEpiThreads);
        if (hf == 0) {
          const unsigned long long v = s_rowbm[r];
          s_rowbm[r] = 0ull;
          if (mvalid) {
            unsigned long long* dst = &o.row_bm[m * o.W64 + ((g.n0 >> 6) >> 6)];
            if (nt == 1) *dst = v;
            else if (v) atomicOr(dst, v);
          }
        }
        if (p.conv != 2 && et < BN / 32) {
          const uint32_t v = s_blk[et];
          s_blk[et] = 0u;
          const int word = (g.n0 >> 5) + et;
          // rows m0.. m0+127 are one whole block and columns n0.. are this tile's
          if (word < o.C32) o.blk_mask[(g.m0 >> 7) * o.C32 + word] = v;
        }
        for (int c = et; c < BN; c += kEpiThreads) {
          const bool live = g.n0 + c < o.C;
          const uint32_t cnt =
              live ? s_cnt[c] + s_cnt[BN + c] + s_cnt[2 * BN + c] + s_cnt[3 * BN + c] : 0u;
          if (acc_smem) {
            if (live) s_acc[g.n0 + c] += cnt;  // one thread per column of this tile
          } else {
            if (cnt) atomicAdd(&o.col_nnz[g.n0 + c], cnt);
            uint32_t sum = cnt;
#pragma unroll
            for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
            if (lane == 0 && sum) {
              atomicAdd(&o.tile_nnz[(g.n0 + c) >> 6], sum);
              atomicAdd(o.nnz, (unsigned long long)sum);
            }
          }
        }
      }
    }
    if (acc_smem) {
      // flush the CTA's column counts: per column, per 64-column tile, total
      named_bar_sync(2, kEpiThreads);
      const OccDev& o = P.out_occ;
      unsigned long long total = 0ull;
      for (int c0 = 0; c0 < p.N; c0 += kEpiThreads) {
        const int c = c0 + et;
        const uint32_t cnt = c < p.N ? s_acc[c] : 0u;
        if (cnt) atomicAdd(&o.col_nnz[c], cnt);
        uint32_t sum = cnt;
#pragma unroll
        for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
        total += sum;
        if (lane == 0 && sum) atomicAdd(&o.tile_nnz[c >> 6], sum);
      }
      if (lane == 0 && total) atomicAdd(o.nnz, total);
    }
    if (lane == 0) bulk_wait_all();
  }

  __syncwarp();  // lanes that finished early wait for their warp's working lane
  tc_fence_before();
  __syncthreads();
  if (*s_abort) {
    // a bounded wait ran out: before shared and tensor memory are released,
    // the copies into the last stage of every ring slot have landed and the
    // MMAs issued so far are done (each wait bounded again)
    if (threadIdx.x == 0) {
      const int issued = *s_issued;
      for (int k = 0; k < S && k < issued; ++k) {
        const int i = issued - 1 - k;
        mbar_drain(bar_full + 8 * (i % S), (uint32_t)((i / S) & 1), wlim);
      }
    }
    if (warp == kMmaWarp && lane == 0) {
      tc_commit(bar_drain);
      mbar_drain(bar_drain, 0u, wlim);
    }
    __syncthreads();
  }
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

CUtensorMapSwizzle swz_of(int inner_bytes) {
  return inner_bytes == 128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B;
}

// 2-D bf16 tensor [rows, cols] (cols contiguous), box {box_cols, box_rows}.
bool make_tmap_2d(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
                  uint32_t box_rows) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz_of((int)box_cols * 2),
                   CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// 4-D NHWC bf16 tensor [n, h, w, c], box {box_c, bw, bh, bn} traversed with
// element strides {1, stride, stride, 1}.
bool make_tmap_nhwc(CUtensorMap* m, const void* base, int n, int h, int w, int c, int box_c, int bw,
                    int bh, int bn, int stride) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[4] = {(cuuint64_t)c, (cuuint64_t)w, (cuuint64_t)h, (cuuint64_t)n};
  cuuint64_t strides[3] = {(cuuint64_t)c * 2, (cuuint64_t)w * c * 2, (cuuint64_t)h * w * c * 2};
  cuuint32_t box[4] = {(cuuint32_t)box_c, (cuuint32_t)(bw * stride), (cuuint32_t)(bh * stride),
                       (cuuint32_t)bn};
  cuuint32_t estr[4] = {1, (cuuint32_t)stride, (cuuint32_t)stride, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz_of(box_c * 2),
                   CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN, int BK, int LEAN>
cudaError_t launch_cfg(const IgemmArgs& a, const CUtensorMap& tA, const CUtensorMap& tB,
                       const CUtensorMap& tY, const CUtensorMap& tA32, const CUtensorMap& tB32,
                       int64_t tiles, cudaStream_t s) {
  cudaError_t e0 =
      smem_optin(reinterpret_cast<const void*>(igemm_kernel<BN, BK, LEAN>), (size_t)Cfg<BN, BK>::kSmem);
  if (e0 != cudaSuccess) return e0;
  const int64_t units = tiles * (a.ksplit > 1 ? a.ksplit : 1);
  const int64_t grid = units < device_sm_count() ? units : device_sm_count();
  cudaError_t e = launch_kernel(igemm_kernel<BN, BK, LEAN>, dim3((unsigned)grid), dim3(kThreads),
                                (size_t)Cfg<BN, BK>::kSmem, s, tA, tB, tY, tA32, tB32, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int LEAN>
cudaError_t launch_bn(const IgemmArgs& a, int bn, int bk, const CUtensorMap& tA, const CUtensorMap& tB,
                      const CUtensorMap& tY, const CUtensorMap& tA32, const CUtensorMap& tB32, int64_t tiles,
                      cudaStream_t s) {
  if (bk == 64) {
    switch (bn) {
      case 64: return launch_cfg<64, 64, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
      case 128: return launch_cfg<128, 64, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
      case 192: return launch_cfg<192, 64, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
      default: return launch_cfg<256, 64, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
    }
  }
  switch (bn) {
    case 64: return launch_cfg<64, 32, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
    case 128: return launch_cfg<128, 32, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
    case 192: return launch_cfg<192, 32, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
    default: return launch_cfg<256, 32, LEAN>(a, tA, tB, tY, tA32, tB32, tiles, s);
  }
}

}  // namespace

PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder() { return get_encode(); }

void choose_spatial_tile(IgemmArgs& a) {
  int64_t best = -1;
  for (int bw = 1; bw <= 128; bw *= 2) {
    if (bw * a.stride > 256) break;
    for (int bh = 1; bw * bh <= 128; bh *= 2) {
      if (bh * a.stride > 256) break;
      const int bn = 128 / (bw * bh);
      const int64_t tw = (a.Wo + bw - 1) / bw, th = (a.Ho + bh - 1) / bh,
                    tn = (a.Nimg + bn - 1) / bn;
      const int64_t cost = tw * bw * th * bh * tn * bn;
      // fewest padded pixels; then the widest (most contiguous) box
      if (best < 0 || cost < best || (cost == best && bw > a.bw)) {
        best = cost;
        a.bw = bw;
        a.bh = bh;
        a.bn = bn;
        a.tw = (int)tw;
        a.th = (int)th;
      }
    }
  }
}

// N tile and K split.  The main loop is bound by shared-memory traffic: a
// K block of a 128 x BN tile is written by TMA and read back by the MMAs,
// (128 + BN) rows each way, so a tile costs about (128 + BN) per K block and
// the tiles take ceil(tiles / SMs) rounds over the SMs.  Of 128, 192 and 256
// wide tiles the cheapest total wins, ties going to the narrower (a shorter
// epilogue); 64 wide ones when 128 wide tiles would fill under half of the
// SMs.  On GB300, GEMMs with M 1024..8192, K 768..3072 and N 768..3072 follow
// this ordering.  K blocks are 64 wide (128-byte swizzle) wherever the
// channel layout allows: 32 wide ones were slower at every tile width.
// Splitting K pays only while the tiles leave SMs idle, at most 4 ways and
// with at least 8 K blocks per unit (the tile's last unit reads the other
// partials alone); splitting further to even out the rounds was slower (the
// partial stores and reads cost more than the main-loop time they save).
static int k_block(const IgemmArgs& a) { return (a.conv == 2 ? (a.Cp % 64 == 0) : (a.Ktot > 32)) ? 64 : 32; }

void choose_tiles(const IgemmArgs& a, int64_t mtiles, int* bn_out, int* ks_out) {
  const int sms = device_sm_count();
  int bn = a.N > 64 ? 128 : 64;
  int64_t tiles = mtiles * ((a.N + bn - 1) / bn);
  if (bn == 128) {
    int64_t best = ((tiles + sms - 1) / sms) * (128 + 128);
    for (int cand = 192; cand <= 256 && cand <= a.N; cand += 64) {
      const int64_t t = mtiles * ((a.N + cand - 1) / cand);
      const int64_t cost = ((t + sms - 1) / sms) * (128 + cand);
      if (cost < best) {
        best = cost;
        bn = cand;
        tiles = t;
      }
    }
    if (bn == 128 && tiles < sms / 2) {
      bn = 64;
      tiles = mtiles * ((a.N + bn - 1) / bn);
    }
  }
  const int bk = k_block(a);
  const int kblocks = (a.Ktot + bk - 1) / bk;
  int ks = 1;
  if (a.ws && a.ws_cnt && tiles < sms && tiles <= a.ws_cnt_len) {
    ks = (int)(sms / tiles);
    if (ks > kMaxSplit) ks = kMaxSplit;
    while (ks > 1 && (kblocks < 8 * ks || (size_t)tiles * ks * kBM * bn * 4 > a.ws_bytes)) --ks;
  }
  *bn_out = bn;
  *ks_out = ks;
}

cudaError_t launch_igemm(const IgemmArgs& a_in, cudaStream_t s) {
  IgemmArgs a = a_in;
  if (a.M <= 0 || a.N <= 0) return cudaSuccess;
  if (a.conv == 2 && (a.Cp % 32 != 0 || a.bw * a.bh * a.bn != 128)) return cudaErrorInvalidValue;
  const int64_t mtiles =
      a.conv == 2 ? (int64_t)((a.Nimg + a.bn - 1) / a.bn) * a.th * a.tw : (a.M + kBM - 1) / kBM;
  int bn = 64, ks = 1;
  choose_tiles(a, mtiles, &bn, &ks);
  a.ksplit = ks;
  const int bk = k_block(a);
  CUtensorMap tA, tB, tY;
  memset(&tA, 0, sizeof(tA));
  memset(&tY, 0, sizeof(tY));
  if (a.conv == 0) {
    if (!make_tmap_2d(&tA, a.x, (uint64_t)a.M, (uint64_t)a.Ktot, (uint32_t)bk, kBM))
      return cudaErrorInvalidValue;
  } else if (a.conv == 2) {
    if (!make_tmap_nhwc(&tA, a.x, a.Nimg, a.H, a.W, a.Cp, bk, a.bw, a.bh, a.bn, a.stride))
      return cudaErrorInvalidValue;
  }
  if (!make_tmap_2d(&tB, a.w, (uint64_t)a.N, (uint64_t)a.Ktot, (uint32_t)bk, (uint32_t)bn))
    return cudaErrorInvalidValue;
  if (!a.y_f32) {
    // one epilogue warp's block: 32 columns x 32 tile rows (for spatial tiles
    // the sub-box {bw', bh', bn'} of 32 pixels that the rows form)
    const int sbw = a.bw < 32 ? a.bw : 32;
    const int sbh = a.bh < 32 / sbw ? a.bh : 32 / sbw;
    const int sbn = 32 / (sbw * sbh);
    bool okY = a.conv == 2
                   ? make_tmap_nhwc(&tY, a.y, a.Nimg, a.Ho, a.Wo, a.N, 32, sbw, sbh, sbn, 1)
                   : make_tmap_2d(&tY, a.y, (uint64_t)a.M, (uint64_t)a.N, 32, 32);
    if (!okY) return cudaErrorInvalidValue;
  }
  if (a.conv == 1) tA = tB;  // unused by the gather producers
  // 32-column boxes (64-byte swizzle) of the compacted zero-skip GEMM
  CUtensorMap tA32 = tB, tB32 = tB;
  if (a.conv == 0 && bk == 64) {
    if (!make_tmap_2d(&tA32, a.x, (uint64_t)a.M, (uint64_t)a.Ktot, 32, kBM) ||
        !make_tmap_2d(&tB32, a.w, (uint64_t)a.N, (uint64_t)a.Ktot, 32, (uint32_t)bn))
      return cudaErrorInvalidValue;
  }
  const int64_t tiles = mtiles * ((a.N + bn - 1) / bn);
  const bool lean = a.conv != 1 && ks == 1 && !a.y_f32 && !a.dense_only &&
                    (a.ep.residual == nullptr ||
                     (a.N % 8 == 0 && (reinterpret_cast<uintptr_t>(a.ep.residual) & 15u) == 0));
  if (!lean) return launch_bn<0>(a, bn, bk, tA, tB, tY, tA32, tB32, tiles, s);
  return a.ep.residual ? launch_bn<2>(a, bn, bk, tA, tB, tY, tA32, tB32, tiles, s)
                       : launch_bn<1>(a, bn, bk, tA, tB, tY, tA32, tB32, tiles, s);
}

}  // namespace sparoa
