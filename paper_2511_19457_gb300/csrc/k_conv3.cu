// 3x3, stride-1, pad-1 convolution on the tcgen05 tensor cores with the
// input halo loaded once per tile and the weights resident in shared memory.
//
// Output positions are numbered in the zero-padded input's row pitch
// Wp = W + 2: q = oh * Wp + ow (ow < W valid, ow = W, W + 1 are junk columns
// that are computed and dropped).  Then the input pixel that tap (r, s) needs
// for position q is the padded-input pixel q + r * Wp + s: every tap of a tile
// of 128 consecutive positions reads a contiguous run of the padded input.
// Per tile the kernel loads that run once (a "slab" of whole padded rows, one
// 4-D TMA box of 64 channels per channel block; out-of-range rows / columns
// read zeros, which is the padding) in the 128-byte-swizzled K-major layout
//   slab[channel block of 64][pixel][64 channels]   (one 128-byte row per pixel)
// so that the A operand of tap (r, s) is the same slab with its descriptor's
// start address moved by (r * Wp + s) whole rows (the swizzle is a function of
// the absolute shared-memory address, so a row-aligned move keeps it).  All
// 9 taps x C/16 MMAs of a tile read one slab; the weights [tap][channel block]
// [C_out][64] (same layout) are loaded once per CTA.
//
// Dispatch and zero skipping as in the implicit-GEMM kernel (Sec. 3 rule
// evaluated on the device; Sec. 2.1 zero-valued products skipped): on the
// zero-skip path one warp reads the input's 128-row block-column masks over
// the whole input rows each tap row of a tile touches, and the MMA warp
// leaves out the taps of a tap row whose activations are all zero there.
// Epilogue: bias / batch norm / residual / activation, bf16 store, output
// occupancy (column counts kept in registers across tiles, row flags of the
// two column halves combined at one 64-thread barrier per lane quarter).
//
// Warp roles (352 threads, persistent CTAs): warp 0 lane 0 issues the slab
// TMA loads, warp 1 computes the skip masks, warp 2 lane 0 issues the MMAs,
// warps 3-10 epilogue (two per TMEM lane quarter -- warp w reads lanes
// 32 (w % 4).. -- 32 columns each).
//
// Overlap with the statistics kernel launched before it: at most 128
// registers a thread (45,056 a CTA) leave room on an SM for one CTA of that
// kernel, so these CTAs become resident while it runs; when the host
// launched a kernel of this library between the producers of x / w and this
// grid (IgemmArgs::early), the weights, the first slab and the epilogue's
// column affine are loaded before griddepcontrol.wait.  After the wait one
// thread reads the input's count for the rule and warp 1 reads the first
// tile's block masks, side by side.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "sparoa_kernels.h"

namespace sparoa {

PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder();  // k_igemm.cu

namespace {
// Slab rows: a tile's 128 positions plus the two extra rows and two columns
// of the 3x3 window must fit: R * Wp >= (Wp - 1) + 2 * Wp + 2 + 128.
int slab_rows(int Wp) { return 3 + (129 + Wp - 1) / Wp; }
int block_stride(int Wp) { return (128 * Wp * slab_rows(Wp) + 1023) / 1024 * 1024; }
constexpr int kCtlBytes = 2048;  // barriers, flags, masks, row flags, column affine and counts
int conv3_smem(int C, int Co, int W) {
  return 9 * C * Co * 2 + 2 * (C / 64) * block_stride(W + 2) + kCtlBytes + 1024;
}

constexpr int kEpiWarps = 8;                      // two per TMEM lane quarter, 32 columns each
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kMmaWarp = 2;
constexpr int kFirstEpiWarp = 3;
constexpr int kThreads = 32 * (kFirstEpiWarp + kEpiWarps);  // slab loads, masks, MMA, epilogue
constexpr int kBM = 128;
constexpr int kMaxPos = 1024;  // slab positions (bounds the slab size)

struct Conv3Geo {
  int N, H, W, C, Co, Wp, R, tiles_per_img, chunk_stride, slab_bytes, w_bytes;
};

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const void* tmap, uint32_t bar, int c0,
                                            int c1, int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const void* tmap, uint32_t bar, int c0,
                                            int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
      : "memory");
}

// Two fp32 values to a bf16 pair (round to nearest even), `lo` in the low
// half; with relu, negative results become zero in the same instruction.
template <bool RELU>
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  if (RELU)
    asm("cvt.rn.relu.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  else
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

// Bits 0 and 1 of the result: the low / high bf16 of w is non-zero (not +-0).
__device__ __forceinline__ uint32_t nz_pair(uint32_t w) {
  const uint32_t t = ((w & 0x7FFF7FFFu) + 0x7FFF7FFFu) & 0x80008000u;
  return ((t >> 15) & 1u) | (t >> 30);
}

// Occupied tap rows of tile t (zero-skip path), from the input's 128-row
// block-column masks: tap row r of the tile reads input rows
// [oh_first + r - 1, oh_last + r - 1] of its image, and is occupied unless
// every 128-row block covering those whole rows is all zero in all channels.
// Executed by one whole warp; returns the 9-bit tap mask (bit 3 r + s).
__device__ __forceinline__ uint32_t conv3_tap_mask(const Conv3Geo& G, const uint32_t* in_blk, int in_C32,
                                                   int t, int lane) {
  const int img = t / G.tiles_per_img;
  const int q0 = (t - img * G.tiles_per_img) * kBM;
  const int oh_first = q0 / G.Wp;
  int oh_last = (q0 + kBM - 1) / G.Wp;
  if (oh_last > G.H - 1) oh_last = G.H - 1;
  const int64_t base = (int64_t)img * G.H * G.W;
  const int lo_row = oh_first - 1 < 0 ? 0 : oh_first - 1;
  const int hi_row = oh_last + 1 > G.H - 1 ? G.H - 1 : oh_last + 1;
  const int64_t B_lo = (base + (int64_t)lo_row * G.W) >> 7;
  const int64_t B_hi = (base + (int64_t)hi_row * G.W + G.W - 1) >> 7;
  const int nb = (int)(B_hi - B_lo + 1);
  if (nb > 32) return 0x1FFu;  // wider than one warp's reach: keep every tap
  bool nz = false;
  if (lane < nb) {
    const uint32_t* wd = in_blk + (B_lo + lane) * in_C32;
    for (int k = 0; k < in_C32; ++k) nz |= wd[k] != 0u;
  }
  const uint32_t occ = __ballot_sync(0xffffffffu, nz);
  uint32_t mask = 0u;
#pragma unroll
  for (int r = 0; r < 3; ++r) {
    const int ih_lo = oh_first + r - 1 < 0 ? 0 : oh_first + r - 1;
    const int ih_hi = oh_last + r - 1 > G.H - 1 ? G.H - 1 : oh_last + r - 1;
    if (ih_lo > ih_hi) continue;
    const int b0 = (int)(((base + (int64_t)ih_lo * G.W) >> 7) - B_lo);
    const int b1 = (int)(((base + (int64_t)ih_hi * G.W + G.W - 1) >> 7) - B_lo);
    const uint32_t span = (b1 - b0 + 1 >= 32) ? 0xffffffffu : ((1u << (b1 - b0 + 1)) - 1u);
    if ((occ >> b0) & span) mask |= 7u << (3 * r);
  }
  return mask;
}

// The per-tile MMAs: 9 taps x 4 k-steps of 128 x CO x 16, the A operand the
// slab shifted by the tap's row offset.  `tapmask` leaves out taps whose
// activations are all zero; accumulate flags are compile-time constants (the
// first issued MMA of the tile is peeled).
template <int CO>
__device__ __forceinline__ void conv3_issue(uint32_t d, uint64_t adesc0, uint64_t bdesc0, int Wp, uint32_t tapmask) {
  constexpr uint32_t idesc = idesc_bf16_f32(kBM, CO);
  if (tapmask == 0x1FFu) {
    tc_mma_bf16(d, adesc0, bdesc0, idesc, 0u);
#pragma unroll
    for (int i = 1; i < 36; ++i) {
      const int tap = i >> 2, ks = i & 3;
      tc_mma_bf16(d, adesc0 + (uint64_t)((((tap / 3) * Wp + (tap % 3)) * 128) >> 4) + (uint64_t)(2 * ks),
                  bdesc0 + (uint64_t)((tap * CO * 128) >> 4) + (uint64_t)(2 * ks), idesc, 1u);
    }
    return;
  }
  if (tapmask == 0u) {
    // no occupied tap: tap 0's activations are all zero, so one
    // non-accumulating MMA on them writes the zero accumulator
    tc_mma_bf16(d, adesc0, bdesc0, idesc, 0u);
    return;
  }
  const int ftap = __ffs((int)tapmask) - 1;
  {
    const uint64_t ad = adesc0 + (uint64_t)((((ftap / 3) * Wp + (ftap % 3)) * 128) >> 4);
    const uint64_t bd = bdesc0 + (uint64_t)((ftap * CO * 128) >> 4);
    tc_mma_bf16(d, ad, bd, idesc, 0u);
#pragma unroll
    for (int ks = 1; ks < 4; ++ks) tc_mma_bf16(d, ad + (uint64_t)(2 * ks), bd + (uint64_t)(2 * ks), idesc, 1u);
  }
#pragma unroll
  for (int tap = 1; tap < 9; ++tap) {
    if (tap <= ftap || !((tapmask >> tap) & 1u)) continue;
    const uint64_t ad = adesc0 + (uint64_t)((((tap / 3) * Wp + (tap % 3)) * 128) >> 4);
    const uint64_t bd = bdesc0 + (uint64_t)((tap * CO * 128) >> 4);
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) tc_mma_bf16(d, ad + (uint64_t)(2 * ks), bd + (uint64_t)(2 * ks), idesc, 1u);
  }
}

template <int CO>
__global__ void __maxnreg__(128)
    conv3_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                 const IgemmArgs P, const Conv3Geo G) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sW = sbase;                            // weights [9][C/64][CO][64]
  const uint32_t sSlab = sW + (uint32_t)G.w_bytes;      // 2 slabs
  uint8_t* ctl = smem + G.w_bytes + 2 * G.slab_bytes;
  const uint32_t sCtl = sSlab + 2u * (uint32_t)G.slab_bytes;
  // control block: mbarriers (8 bytes each) w (+ 8 spare), full[2], empty[2], accf[2],
  // acce[2], mask[2]; then flags, masks, row flags, column affine and counts
  const uint32_t bar_w = sCtl;
  const uint32_t bar_full = sCtl + 72;
  const uint32_t bar_empty = sCtl + 88;
  const uint32_t bar_accf = sCtl + 104;
  const uint32_t bar_acce = sCtl + 120;
  const uint32_t bar_mask = sCtl + 136;
  const uint32_t bar_drain = sCtl + 168;  // after an abort: the MMAs issued so far are done
  volatile int* s_abort = reinterpret_cast<volatile int*>(ctl + 152);
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(ctl + 156);
  uint32_t* s_tapm = reinterpret_cast<uint32_t*>(ctl + 160);          // [2] 9-bit occupied-tap masks
  int* s_slabs = reinterpret_cast<int*>(ctl + 176);                    // slabs issued (drain after an abort)
  volatile int* s_path = reinterpret_cast<volatile int*>(ctl + 180);   // the rule's decision
  uint8_t* s_rowf = ctl + 256;                                         // [3][2][128] row has a non-zero
  float* s_scale = reinterpret_cast<float*>(ctl + 1024);              // [CO]
  float* s_shift = s_scale + CO;                                       // [CO]
  uint32_t* s_acc = reinterpret_cast<uint32_t*>(s_shift + CO);         // [CO] non-zeros per column

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int N = G.N, H = G.H, W = G.W, C = G.C, Wp = G.Wp;
  const int tiles = N * G.tiles_per_img;
  uint32_t* const err = P.err;
  const int emit = P.emit;
  const long long wlim = P.wait_limit > 0 ? P.wait_limit : kWaitLimitCycles;

  // on-chip prologue, overlapping the previous grid on the stream
  if (threadIdx.x == 0) {
    mbar_init(bar_w, 1u);
    mbar_init(bar_drain, 1u);
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_full + 8 * b, 1u);
      mbar_init(bar_mask + 8 * b, 1u);
      mbar_init(bar_empty + 8 * b, 1u);
      mbar_init(bar_accf + 8 * b, 1u);
      mbar_init(bar_acce + 8 * b, (uint32_t)kEpiThreads);
    }
    *s_abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmX);
    prefetch_tmap(&tmW);
  }
  if (warp == kMmaWarp) tmem_alloc(smem_u32(s_tmem), (uint32_t)(2 * CO));
  if (warp >= kFirstEpiWarp)
    for (int c = threadIdx.x - 32 * kFirstEpiWarp; c < CO; c += kEpiThreads) s_acc[c] = 0u;
  // the first tile's slab origin (arithmetic on the parameters only)
  const int t_first = blockIdx.x;
  const int img_first = t_first / G.tiles_per_img;
  const int oh0_first = (t_first - img_first * G.tiles_per_img) * kBM / Wp;
  auto issue_first = [&]() {
    // The first tile's slab goes out first, then the weights (the same 72 KB
    // for every CTA, from L2; the larger and slower of the two).
    mbar_arrive_expect_tx(bar_full, (uint32_t)(C / 64 * 128 * Wp * G.R));
    for (int cb = 0; cb < C / 64; ++cb)
      tma_load_4d(sSlab + (uint32_t)(cb * G.chunk_stride), &tmX, bar_full, cb * 64, -1, oh0_first - 1,
                  img_first);
    mbar_arrive_expect_tx(bar_w, (uint32_t)(9 * (C / 64) * CO * 128));
    for (int tap = 0; tap < 9; ++tap)
      for (int cb = 0; cb < C / 64; ++cb)
        tma_load_3d(sW + (uint32_t)((tap * (C / 64) + cb) * CO * 128), &tmW, bar_w, cb * 64, tap, 0);
  };
  auto load_affine = [&]() {  // epilogue threads: the column affine into shared memory
    for (int c = threadIdx.x - 32 * kFirstEpiWarp; c < CO; c += kEpiThreads) {
      float sc = 1.f, sh = 0.f;
      if (c < G.Co) epi_affine(P.ep, G.Co, c, sc, sh);
      s_scale[c] = sc;
      s_shift[c] = sh;
    }
  };
  if (P.early) {
    if (threadIdx.x == 0 && t_first < tiles) issue_first();
    if (warp >= kFirstEpiWarp) load_affine();
  }
  pdl_wait();
  pdl_trigger();
  if (!P.early && threadIdx.x == 0 && t_first < tiles) issue_first();
  // the rule (one read of the input's count per CTA) and, side by side, the
  // first tile's occupied taps (used on the zero-skip path only)
  uint32_t first_mask = 0x1FFu;
  if (threadIdx.x == 0) {
    const int pth = decide_path(P.disp);
    record_path(P.disp, pth);
    *s_path = pth;
  } else if (warp == 1 && t_first < tiles && P.disp.force != 1 && P.in_blk) {
    first_mask = conv3_tap_mask(G, P.in_blk, P.in_C32, t_first, lane);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const bool skip = *s_path == 2;
  const uint32_t tmem = *s_tmem;

  if (warp == 0) {
    // -------------------------------------------------------------- slab loads
    if (lane == 0) {
      int j = 1;
      *s_slabs = t_first < tiles ? 1 : 0;  // the first went out in the prologue
      for (int t = blockIdx.x + gridDim.x; t < tiles; t += gridDim.x, ++j) {
        const int b = j & 1;
        if (!mbar_wait(bar_empty + 8 * b, (uint32_t)(((j >> 1) & 1) ^ 1), err, s_abort, kErrTimeoutEmpty, wlim))
          break;
        const int img = t / G.tiles_per_img;
        const int oh0 = (t - img * G.tiles_per_img) * kBM / Wp;
        const uint32_t dst = sSlab + (uint32_t)(b * G.slab_bytes);
        mbar_arrive_expect_tx(bar_full + 8 * b, (uint32_t)(C / 64 * 128 * Wp * G.R));
        for (int cb = 0; cb < C / 64; ++cb)
          tma_load_4d(dst + (uint32_t)(cb * G.chunk_stride), &tmX, bar_full + 8 * b, cb * 64, -1, oh0 - 1, img);
        *s_slabs = j + 1;
      }
    }
  } else if (warp == 1) {
    // -------------------------------------------------------------- skip masks
    if (skip) {
      int j = 0;
      for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++j) {
        const int b = j & 1;
        bool ok = true;
        // mask buffer b was read by the MMA issue of tile j - 2, before that
        // tile's commit to the slab-empty barrier
        if (lane == 0 && j >= 2)
          ok = mbar_wait(bar_empty + 8 * b, (uint32_t)(((j >> 1) & 1) ^ 1), err, s_abort, kErrTimeoutEmpty, wlim);
        if (!__shfl_sync(0xffffffffu, ok ? 1 : 0, 0)) break;
        const uint32_t m = j == 0 ? first_mask : conv3_tap_mask(G, P.in_blk, P.in_C32, t, lane);
        if (lane == 0) {
          s_tapm[b] = m;
          mbar_arrive(bar_mask + 8 * b);
        }
      }
    }
  } else if (warp == kMmaWarp) {
    // -------------------------------------------------------------- MMA issue
    if (lane == 0) {
      int j = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++j) {
        const int b = j & 1;
        ok = mbar_wait_spin(bar_acce + 8 * b, (uint32_t)(((j >> 1) & 1) ^ 1), err, s_abort, kErrTimeoutAcc, wlim) &&
             mbar_wait_spin(bar_full + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutFull, wlim) &&
             (!skip || mbar_wait_spin(bar_mask + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutFull, wlim));
        if (!ok) break;
        tc_fence_after();
        const int q0 = (t - (t / G.tiles_per_img) * G.tiles_per_img) * kBM;
        const int qoff = q0 - (q0 / Wp) * Wp;
        const uint32_t d = tmem + (uint32_t)(b * CO);
        const uint32_t slab = sSlab + (uint32_t)(b * G.slab_bytes);
        // descriptors of tap 0 / k-step 0; the others differ only in the
        // start-address field (byte offset >> 4), which never carries out
        const uint64_t adesc0 = smem_desc_kmajor<64>(slab + (uint32_t)(qoff * 128));
        const uint64_t bdesc0 = smem_desc_kmajor<64>(sW);
        const uint32_t tapmask = skip ? s_tapm[b] : 0x1FFu;
        if (j == 0) {
          ok = mbar_wait_spin(bar_w, 0u, err, s_abort, kErrTimeoutFull, wlim);
          if (!ok) break;
          tc_fence_after();
        }
        conv3_issue<CO>(d, adesc0, bdesc0, Wp, tapmask);
        tc_commit(bar_empty + 8 * b);  // slab and mask buffer free once these MMAs are done
        // (the fault injection of the error-path tests leaves the first
        // accumulator unsignalled: the epilogue's bounded wait runs out)
        if (!(P.fault == kFaultSkipFirstAccCommit && j == 0)) tc_commit(bar_accf + 8 * b);
      }
      // TMEM is freed below only after the epilogue has read the last two
      // accumulators (the waits a further two tiles would make)
      for (int k = 0; k < 2 && ok; ++k, ++j)
        ok = mbar_wait(bar_acce + 8 * (j & 1), (uint32_t)(((j >> 1) & 1) ^ 1), err, s_abort, kErrTimeoutAcc, wlim);
    }
  } else if (warp >= kFirstEpiWarp) {
    // -------------------------------------------------------------- epilogue
    // warp w reads TMEM lanes 32 (w % 4).. (its quarter of the tile's rows) and
    // the 32 accumulator columns 32 ((w - 3) / 4)..; the two warps of a lane
    // quarter meet at one 64-thread named barrier per tile (id 3 + quarter)
    const int q = warp & 3, r = q * 32 + lane, et = threadIdx.x - 32 * kFirstEpiWarp;
    const int hf = (warp - kFirstEpiWarp) >> 2;
    const int c0 = hf * 32;
    const int pair_bar = 3 + q;
    const OccDev o = P.out_occ;
    const int act = P.ep.act;
    const __nv_bfloat16* const residual = P.ep.residual;
    // without the early loads the column affine is read here, after the CTA
    // barrier, so that its global loads do not hold up the first MMAs
    if (!P.early) load_affine();
    named_bar_sync(2, kEpiThreads);
    // this warp's 32 columns of the affine stay in registers for every tile
    float sc[32], sh[32];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float4 a = reinterpret_cast<const float4*>(s_scale + c0)[i];
      const float4 bq = reinterpret_cast<const float4*>(s_shift + c0)[i];
      sc[4 * i] = a.x; sc[4 * i + 1] = a.y; sc[4 * i + 2] = a.z; sc[4 * i + 3] = a.w;
      sh[4 * i] = bq.x; sh[4 * i + 1] = bq.y; sh[4 * i + 2] = bq.z; sh[4 * i + 3] = bq.w;
    }
    uint32_t colcnt = 0u;    // non-zeros of column c0 + lane over this warp's rows of every tile
    int64_t prev_m = -1;     // the previous tile's output row of this thread (its row flag is pending)
    int j = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++j) {
      const int b = j & 1;
      const int img = t / G.tiles_per_img;
      const int qq = (t - img * G.tiles_per_img) * kBM + r;
      const int oh = qq / Wp, ow = qq - (qq / Wp) * Wp;
      const bool mvalid = oh < H && ow < W;
      const int64_t m = ((int64_t)img * H + oh) * W + ow;
      const bool ok = mbar_wait(bar_accf + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutAcc, wlim);
      // the pair agrees on an abort, and the row flags of the previous tile
      // (written before this barrier by both warps) can be combined after it
      if (named_bar_or(pair_bar, 64, !ok)) break;
      if (emit && hf == 0 && prev_m >= 0) {
        const int fb = (j - 1) % 3;
        o.row_bm[prev_m * o.W64] = (s_rowf[(fb * 2 + 0) * 128 + r] | s_rowf[(fb * 2 + 1) * 128 + r]) ? 1ull : 0ull;
      }
      tc_fence_after();
      uint32_t raw[32];
      tmem_ld32_nowait(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * CO + c0), raw);
      tmem_wait_ld32(raw);
      float v[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) v[i] = fmaf(__uint_as_float(raw[i]), sc[i], sh[i]);
      tc_fence_before();
      mbar_arrive(bar_acce + 8 * b);  // the accumulator is in registers
      if (residual && mvalid) {
        const uint4* rp = reinterpret_cast<const uint4*>(residual + m * G.Co + c0);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint4 rv = rp[k];
          const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&rv);
#pragma unroll
          for (int jj = 0; jj < 4; ++jj) {
            const float2 a = __bfloat1622float2(h[jj]);
            v[8 * k + 2 * jj] += a.x;
            v[8 * k + 2 * jj + 1] += a.y;
          }
        }
      }
      uint32_t pk[16];
      if (act == 1) {
#pragma unroll
        for (int i = 0; i < 16; ++i) pk[i] = pack_bf16x2<true>(v[2 * i], v[2 * i + 1]);
      } else {
        if (act == 2) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = fminf(fmaxf(v[i], 0.f), 6.f);
        } else if (act == 3) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = gelu_f(v[i]);
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) pk[i] = pack_bf16x2<false>(v[2 * i], v[2 * i + 1]);
      }
      if (mvalid) {
        uint4* yp = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(P.y) + m * G.Co + c0);
#pragma unroll
        for (int k = 0; k < 4; ++k) yp[k] = make_uint4(pk[4 * k], pk[4 * k + 1], pk[4 * k + 2], pk[4 * k + 3]);
      }
      if (emit) {
        uint32_t nzw = 0u;  // bit i: column c0 + i of this row is non-zero
#pragma unroll
        for (int i = 0; i < 16; ++i) nzw |= nz_pair(pk[i]) << (2 * i);
        if (!mvalid) nzw = 0u;
        // block-column mask: the warp's 32 positions cover at most two
        // 128-row blocks of the output (the first and the last valid row's)
        const int blk = mvalid ? (int)(m >> 7) : -1;
        const uint32_t vmask = __ballot_sync(0xffffffffu, mvalid);
        if (vmask) {
          const int lo = __shfl_sync(0xffffffffu, blk, __ffs(vmask) - 1);
          const int hi = __shfl_sync(0xffffffffu, blk, 31 - __clz(vmask));
          const uint32_t b_lo = __reduce_or_sync(0xffffffffu, blk == lo ? nzw : 0u);
          const uint32_t b_hi = hi != lo ? __reduce_or_sync(0xffffffffu, blk == hi ? nzw : 0u) : 0u;
          if (lane == 0 && b_lo) atomicOr(&o.blk_mask[lo * o.C32 + (c0 >> 5)], b_lo);
          if (lane == 1 && b_hi) atomicOr(&o.blk_mask[hi * o.C32 + (c0 >> 5)], b_hi);
        }
        colcnt += __popc(warp_transpose32(nzw));
        s_rowf[((j % 3) * 2 + hf) * 128 + r] = nzw ? 1 : 0;
      }
      prev_m = mvalid ? m : -1;
    }
    // the last tile's row flags
    named_bar_sync(pair_bar, 64);
    if (emit && hf == 0 && prev_m >= 0) {
      const int fb = (j - 1) % 3;
      o.row_bm[prev_m * o.W64] = (s_rowf[(fb * 2 + 0) * 128 + r] | s_rowf[(fb * 2 + 1) * 128 + r]) ? 1ull : 0ull;
    }
    if (emit) {
      // column counts: the four lane quarters meet in shared memory, then one
      // atomic per column, per 64-column tile and for the total
      if (colcnt) atomicAdd(&s_acc[c0 + lane], colcnt);
      named_bar_sync(2, kEpiThreads);
      if (et < CO) {
        const uint32_t cnt = s_acc[et];
        if (cnt) atomicAdd(&o.col_nnz[et], cnt);
        uint32_t sum = cnt;
#pragma unroll
        for (int sft = 16; sft > 0; sft >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, sft);
        if (lane == 0 && sum) {
          atomicAdd(&o.tile_nnz[et >> 6], sum);
          atomicAdd(o.nnz, (unsigned long long)sum);
        }
      }
    }
  }

  __syncwarp();  // lanes that finished early wait for their warp's working lane
  tc_fence_before();
  __syncthreads();
  if (*s_abort) {
    // a bounded wait ran out: before shared and tensor memory are released,
    // the weights and the last slab of each buffer have landed and the MMAs
    // issued so far are done (each wait bounded again)
    if (threadIdx.x == 0 && t_first < tiles) {
      mbar_drain(bar_w, 0u, wlim);
      const int n = *s_slabs;
      for (int k = 0; k < 2 && k < n; ++k) {
        const int i = n - 1 - k;
        mbar_drain(bar_full + 8 * (i & 1), (uint32_t)((i >> 1) & 1), wlim);
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
    tmem_dealloc(tmem, (uint32_t)(2 * CO));
  }
}

template <int CO>
cudaError_t launch_co(const CUtensorMap& tX, const CUtensorMap& tW, const IgemmArgs& a,
                      const Conv3Geo& g, int smem, cudaStream_t s) {
  cudaError_t e0 = smem_optin(reinterpret_cast<const void*>(conv3_kernel<CO>), (size_t)smem);
  if (e0 != cudaSuccess) return e0;
  const int tiles = g.N * g.tiles_per_img;
  const int grid = tiles < device_sm_count() ? tiles : device_sm_count();
  cudaError_t e = launch_kernel(conv3_kernel<CO>, dim3(grid), dim3(kThreads), (size_t)smem, s, tX, tW, a, g);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

bool conv3_supported(const IgemmArgs& a) {
  if (a.kh != 3 || a.kw != 3 || a.stride != 1 || a.pad != 1) return false;
  // one 64-channel block in and out: the weights (72 KB) stay resident next to
  // two halo slabs
  if (a.Cp != 64 || a.N != 64 || a.W + 2 > 256) return false;
  const int w_bytes = 9 * a.Cp * a.N * 2;
  const int Wp = a.W + 2;
  return w_bytes <= 96 * 1024 && conv3_smem(a.Cp, a.N, a.W) <= 220 * 1024 &&
         slab_rows(Wp) * Wp <= kMaxPos;
}

cudaError_t launch_conv3(const IgemmArgs& a, cudaStream_t s) {
  if (a.M <= 0) return cudaSuccess;
  Conv3Geo g;
  g.N = a.Nimg;
  g.H = a.H;
  g.W = a.W;
  g.C = a.Cp;
  g.Co = a.N;
  g.Wp = a.W + 2;
  g.R = slab_rows(g.Wp);
  g.tiles_per_img = (a.H * g.Wp + kBM - 1) / kBM;
  g.chunk_stride = block_stride(g.Wp);
  g.slab_bytes = (g.C / 64) * g.chunk_stride;
  g.w_bytes = 9 * g.C * g.Co * 2;
  const int smem = conv3_smem(g.C, g.Co, g.W);
  auto enc = tmap_encoder();
  if (!enc) return cudaErrorInvalidValue;
  CUtensorMap tX, tW;
  {
    cuuint64_t dims[4] = {(cuuint64_t)g.C, (cuuint64_t)g.W, (cuuint64_t)g.H, (cuuint64_t)g.N};
    cuuint64_t strides[3] = {(cuuint64_t)g.C * 2, (cuuint64_t)g.W * g.C * 2,
                             (cuuint64_t)g.H * g.W * g.C * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)g.Wp, (cuuint32_t)g.R, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    if (enc(&tX, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>((const void*)a.x), dims,
            strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  {
    cuuint64_t dims[3] = {(cuuint64_t)g.C, 9, (cuuint64_t)g.Co};
    cuuint64_t strides[2] = {(cuuint64_t)g.C * 2, (cuuint64_t)9 * g.C * 2};
    cuuint32_t box[3] = {64, 1, (cuuint32_t)g.Co};
    cuuint32_t estr[3] = {1, 1, 1};
    if (enc(&tW, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>((const void*)a.w), dims,
            strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
      return cudaErrorInvalidValue;
  }
  if (g.C != 64 || g.Co != 64) return cudaErrorInvalidValue;
  return launch_co<64>(tX, tW, a, g, smem, s);
}

}  // namespace sparoa
