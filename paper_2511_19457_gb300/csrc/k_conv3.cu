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
// [C_out][64] (same layout) are loaded once per CTA.  Compared with gathering A per (tap, channel block), the shared-memory
// traffic per tile drops about tenfold.
//
// Dispatch and zero skipping as in the implicit-GEMM kernel (Sec. 3 rule
// evaluated on the device; Sec. 2.1 zero-valued products skipped): on the
// zero-skip path the producers OR the input row bitmaps of each tap's 128
// shifted pixels, and the MMA warp leaves out the (tap, 64-channel tile) MMAs
// whose activations are all zero.  Epilogue: bias / batch norm / residual /
// activation, bf16 store, output occupancy.
//
// Warp roles (416 threads, persistent CTAs): warps 0-3 producers (thread 0
// issues TMA; all compute skip masks), warps 4-11 epilogue (two per TMEM lane
// quarter, 32 columns each), warp 12 MMA.
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
int conv3_smem(int C, int Co, int W) {
  const int ctl = 512 + 2 * Co * 4 + 4 * Co * 4 + Co * 4 + 16 + 1024 * 8;
  return 9 * C * Co * 2 + 2 * (C / 64) * block_stride(W + 2) + ctl + 1024;
}
}  // namespace

namespace {

constexpr int kEpiWarps = 8;                      // two per TMEM lane quarter, 32 columns each
constexpr int kEpiThreads = 32 * kEpiWarps;
constexpr int kMmaWarp = 4 + kEpiWarps;
constexpr int kThreads = 32 * (kMmaWarp + 1);     // 4 producer warps, epilogue warps, MMA warp
constexpr int kBM = 128;
constexpr int kMaxPos = 1024;  // slab positions for the skip masks

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

template <int CO>
__global__ void __launch_bounds__(kThreads, 1)
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
  // control block: bars(8 each): w, slab_full[2], slab_empty[2], accf[2], acce[2]
  const uint32_t bar_w = sCtl;
  const uint32_t bar_full = sCtl + 8;
  const uint32_t bar_empty = sCtl + 24;
  const uint32_t bar_accf = sCtl + 40;
  const uint32_t bar_acce = sCtl + 56;
  const uint32_t bar_mask = sCtl + 80;  // [2] zero-skip: the 128 mask threads of a slab's tile are done
  volatile int* s_abort = reinterpret_cast<volatile int*>(ctl + 72);
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(ctl + 76);
  uint32_t* s_tapm = reinterpret_cast<uint32_t*>(ctl + 128);  // [3] 9-bit occupied-tap masks
  float* s_scale = reinterpret_cast<float*>(ctl + 512);                          // [CO]
  float* s_shift = s_scale + CO;                                                 // [CO]
  uint32_t* s_cnt = reinterpret_cast<uint32_t*>(s_shift + CO);                   // [4][CO]
  uint32_t* s_acc = s_cnt + 4 * CO;                                              // [CO]
  uint8_t* s_pos = reinterpret_cast<uint8_t*>(s_acc + CO);  // [kMaxPos] 1 = input pixel has a non-zero
  unsigned long long* s_rowbm = reinterpret_cast<unsigned long long*>(s_pos + kMaxPos);  // [128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int N = G.N, H = G.H, W = G.W, C = G.C, Wp = G.Wp;
  const int tiles = N * G.tiles_per_img;
  const int act = P.ep.act;
  const __nv_bfloat16* const residual = P.ep.residual;
  const unsigned long long* const in_rowbm = P.in_rowbm;
  const int in_W64 = P.in_W64;
  uint32_t* const err = P.err;
  const int emit = P.emit;

  // on-chip prologue, overlapping the previous grid on the stream
  if (threadIdx.x == 0) {
    mbar_init(bar_w, 1u);
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar_full + 8 * b, 1u);
      mbar_init(bar_mask + 8 * b, 128u);
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
  // the first tile's slab origin (arithmetic on the parameters only)
  const int t_first = blockIdx.x;
  const int img_first = t_first / G.tiles_per_img;
  const int oh0_first = (t_first - img_first * G.tiles_per_img) * kBM / Wp;
  pdl_wait();
  pdl_trigger();
  if (threadIdx.x == 0 && t_first < tiles) {
    // The first slab and the weights go out before anything else: the slab
    // comes from HBM and gates the first MMAs.  Either path needs them.
    mbar_arrive_expect_tx(bar_full, (uint32_t)(C / 64 * 128 * Wp * G.R));
    for (int cb = 0; cb < C / 64; ++cb)
      tma_load_4d(sSlab + (uint32_t)(cb * G.chunk_stride), &tmX, bar_full, cb * 64, -1, oh0_first - 1,
                  img_first);
    mbar_arrive_expect_tx(bar_w, (uint32_t)G.w_bytes);
    for (int tap = 0; tap < 9; ++tap)
      for (int cb = 0; cb < C / 64; ++cb)
        tma_load_3d(sW + (uint32_t)((tap * (C / 64) + cb) * CO * 128), &tmW, bar_w, cb * 64, tap, 0);
  }
  const int path = decide_path(P.disp);
  record_path(P.disp, path);
  const bool skip = path == 2;
  if (warp >= 4 && warp < kMmaWarp) {
    const int et = threadIdx.x - 128;
    for (int c = et; c < CO; c += kEpiThreads) s_acc[c] = 0u;
    for (int i = et; i < kBM; i += kEpiThreads) s_rowbm[i] = 0ull;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;

  if (warp < 4) {
    // -------------------------------------------------------------- producers
    const int t_ = threadIdx.x;
    int j = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++j) {
      if (!skip && warp != 0) break;  // dense path: warp 0 walks the tiles, lane 0 streams the slabs
      const int b = j & 1;
      const int mb = j % 3;  // mask buffer: the MMAs of tile j - 3 are issued by now
      const int img = t / G.tiles_per_img;
      const int q0 = (t - img * G.tiles_per_img) * kBM;
      const int oh0 = q0 / Wp;
      // the slab first, so that its load overlaps the mask computation below
      bool ok = true;
      if (t_ == 0 && j > 0) {  // the first slab went out with the weights
        ok = mbar_wait(bar_empty + 8 * b, (uint32_t)(((j >> 1) & 1) ^ 1), err, s_abort, kErrTimeoutEmpty);
        if (ok) {
          const uint32_t dst = sSlab + (uint32_t)(b * G.slab_bytes);
          mbar_arrive_expect_tx(bar_full + 8 * b, (uint32_t)(C / 64 * 128 * Wp * G.R));
          for (int cb = 0; cb < C / 64; ++cb)
            tma_load_4d(dst + (uint32_t)(cb * G.chunk_stride), &tmX, bar_full + 8 * b, cb * 64, -1,
                        oh0 - 1, img);
        }
      }
      if (skip) {
        // zero-skip masks of this tile: per tap, OR of the row bitmaps of the
        // tile's 128 shifted pixels (the mask buffer of tile j - 3 is free: the
        // empty-slot wait of tile j - 1 saw those MMAs complete)
        // One 64-channel block (C == 64): a pixel's row bitmap word is its bit 0.
        // All of this thread's bitmap loads are issued before any is used.
        const int npos = G.R * Wp < kMaxPos ? G.R * Wp : kMaxPos;
        uint32_t nzb = 0u;  // bit k: slab position t_ + 128 k is a non-zero pixel
#pragma unroll
        for (int k = 0; k < kMaxPos / 128; ++k) {
          const int pp = t_ + 128 * k;
          const int prr = pp / Wp;
          const int pr = oh0 - 1 + prr, pc = pp - prr * Wp - 1;  // input pixel of slab position pp
          unsigned long long w = 0ull;
          if (pp < npos && pr >= 0 && pr < H && pc >= 0 && pc < W)
            w = in_rowbm[(((int64_t)img * H + pr) * W + pc) * in_W64];
          nzb |= (uint32_t)(w & 1ull) << k;
        }
#pragma unroll
        for (int k = 0; k < kMaxPos / 128; ++k)
          if (t_ + 128 * k < npos) s_pos[t_ + 128 * k] = (uint8_t)((nzb >> k) & 1u);
        if (t_ == 0) s_tapm[mb] = 0u;
        named_bar_sync(1, 128);
        const int qoff = q0 - oh0 * Wp;
        const bool rvalid = q0 + t_ < H * Wp;
        uint32_t tb = 0u;  // bit tap: this output position reads a non-zero pixel under that tap
#pragma unroll
        for (int tap = 0; tap < 9; ++tap) {
          const int pp = qoff + t_ + (tap / 3) * Wp + (tap % 3);
          if (rvalid && pp < kMaxPos && s_pos[pp]) tb |= 1u << tap;
        }
        tb = __reduce_or_sync(0xffffffffu, tb);
        if (lane == 0 && tb) atomicOr(&s_tapm[mb], tb);
      }
      if (!skip) {
        if (__shfl_sync(0xffffffffu, ok ? 1 : 0, 0) == 0) break;
        continue;
      }
      // all masks written (and s_pos free for the next tile); uniform abort decision
      if (named_bar_or(1, 128, !ok)) break;
      mbar_arrive(bar_mask + 8 * b);  // this tile's masks are written
    }
  } else if (warp == kMmaWarp) {
    // -------------------------------------------------------------- MMA issue
    // The whole warp walks the tiles so that it stays converged between tiles;
    // lane 0 waits, issues the MMAs and commits.
    constexpr uint32_t idesc = idesc_bf16_f32(kBM, CO);
    bool ok = true;
    if (lane == 0) ok = mbar_wait(bar_w, 0u, err, s_abort, kErrTimeoutFull);
    ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    tc_fence_after();
    int j = 0;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++j) {
      const int b = j & 1;
      if (lane == 0) {
        ok = mbar_wait(bar_acce + 8 * b, (uint32_t)(((j >> 1) & 1) ^ 1), err, s_abort, kErrTimeoutAcc) &&
             mbar_wait(bar_full + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutFull) &&
             (!skip || mbar_wait(bar_mask + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutFull));
      }
      if (lane == 0 && ok) {
        const int q0 = (t - (t / G.tiles_per_img) * G.tiles_per_img) * kBM;
        const int qoff = q0 - (q0 / Wp) * Wp;
        tc_fence_after();
        const uint32_t d = tmem + (uint32_t)(b * CO);
        const uint32_t slab = sSlab + (uint32_t)(b * G.slab_bytes);
        // descriptors of tap 0 / channel block 0 / k-step 0; the others differ only
        // in the start-address field (byte offset >> 4), which never carries out
        const uint64_t adesc0 = smem_desc_kmajor<64>(slab + (uint32_t)(qoff * 128));
        const uint64_t bdesc0 = smem_desc_kmajor<64>(sW);
        // Occupied taps as a 9-bit mask (one 64-channel block: C == 64). The
        // lane issuing MMAs is slow at anything else, so the dense case is a
        // straight run of 36 MMAs and the zero-skip case one branch per tap;
        // every accumulate flag is a constant (the first occupied tap's first
        // k-step is the only non-accumulating MMA).
        uint32_t tapmask = skip ? s_tapm[j % 3] : 0x1FFu;
        if (tapmask == 0x1FFu) {
          tc_mma_bf16(d, adesc0, bdesc0, idesc, 0u);
#pragma unroll
          for (int i = 1; i < 36; ++i) {
            const int tap = i >> 2, ks = i & 3;
            tc_mma_bf16(d, adesc0 + (uint64_t)((((tap / 3) * Wp + (tap % 3)) * 128) >> 4) + (uint64_t)(2 * ks),
                        bdesc0 + (uint64_t)((tap * CO * 128) >> 4) + (uint64_t)(2 * ks), idesc, 1u);
          }
        } else if (tapmask == 0u) {
          // no tap is occupied: tap 0's activations are all zero, so one
          // non-accumulating MMA on them writes the zero accumulator
          tc_mma_bf16(d, adesc0, bdesc0, idesc, 0u);
        } else {
          const int ftap = __ffs((int)tapmask) - 1;
          tapmask &= ~(1u << ftap);
          {
            const uint64_t ad = adesc0 + (uint64_t)((((ftap / 3) * Wp + (ftap % 3)) * 128) >> 4);
            const uint64_t bd = bdesc0 + (uint64_t)((ftap * CO * 128) >> 4);
            tc_mma_bf16(d, ad, bd, idesc, 0u);
#pragma unroll
            for (int ks = 1; ks < 4; ++ks)
              tc_mma_bf16(d, ad + (uint64_t)(2 * ks), bd + (uint64_t)(2 * ks), idesc, 1u);
          }
#pragma unroll
          for (int tap = 0; tap < 9; ++tap) {
            if (!((tapmask >> tap) & 1u)) continue;  // all-zero activations, or the peeled tap
            const uint64_t ad = adesc0 + (uint64_t)((((tap / 3) * Wp + (tap % 3)) * 128) >> 4);
            const uint64_t bd = bdesc0 + (uint64_t)((tap * CO * 128) >> 4);
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)
              tc_mma_bf16(d, ad + (uint64_t)(2 * ks), bd + (uint64_t)(2 * ks), idesc, 1u);
          }
        }
        tc_commit(bar_empty + 8 * b);  // slab free once these MMAs are done
        tc_commit(bar_accf + 8 * b);
      }
      ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
    }
  } else {
    // -------------------------------------------------------------- epilogue
    // warp w reads TMEM lanes 32 (w % 4).. (its quarter of the tile's rows) and
    // the 32 accumulator columns 32 ((w - 4) / 4)..
    const int q = warp & 3, r = q * 32 + lane, et = threadIdx.x - 128;
    const int c0 = ((warp - 4) >> 2) * 32;
    const OccDev o = P.out_occ;
    const bool acc_smem = emit != 0;
    const bool affine = P.ep.bias != nullptr || P.ep.bn != nullptr;  // else the column affine is 1, 0
    // the column affine, read here rather than before the CTA barrier so that
    // its global loads do not hold up the first MMAs
    for (int c = et; c < CO; c += kEpiThreads) {
      float sc = 1.f, sh = 0.f;
      if (c < G.Co) epi_affine(P.ep, G.Co, c, sc, sh);
      s_scale[c] = sc;
      s_shift[c] = sh;
    }
    named_bar_sync(2, kEpiThreads);
    int j = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++j) {
      const int b = j & 1;
      const int img = t / G.tiles_per_img;
      const int qq = (t - img * G.tiles_per_img) * kBM + r;
      const int oh = qq / Wp, ow = qq - (qq / Wp) * Wp;
      const bool mvalid = oh < H && ow < W;
      const int64_t m = ((int64_t)img * H + oh) * W + ow;
      const bool ok = mbar_wait(bar_accf + 8 * b, (uint32_t)((j >> 1) & 1), err, s_abort, kErrTimeoutAcc);
      // the same abort decision for every epilogue warp (one that left alone
      // would strand the others at the occupancy barrier)
      if (named_bar_or(2, kEpiThreads, !ok)) break;
      tc_fence_after();
      const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * CO);
      const int blk = mvalid ? (int)(m >> 7) : -1;
      const uint32_t grp = __match_any_sync(0xffffffffu, blk);
      const bool leader = (__ffs(grp) - 1) == lane;
      unsigned long long tl = 0ull;
      {
        uint32_t raw[32];
        tmem_ld32_nowait(tbase + (uint32_t)c0, raw);
        tmem_wait_ld32(raw);
        uint32_t nzw = 0u;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int cc = c0 + h * 16;
          float v[16];
          if (affine) {
#pragma unroll
            for (int q4 = 0; q4 < 4; ++q4) {
              const float4 sc = reinterpret_cast<const float4*>(s_scale + cc)[q4];
              const float4 sh = reinterpret_cast<const float4*>(s_shift + cc)[q4];
              v[4 * q4 + 0] = fmaf(__uint_as_float(raw[h * 16 + 4 * q4 + 0]), sc.x, sh.x);
              v[4 * q4 + 1] = fmaf(__uint_as_float(raw[h * 16 + 4 * q4 + 1]), sc.y, sh.y);
              v[4 * q4 + 2] = fmaf(__uint_as_float(raw[h * 16 + 4 * q4 + 2]), sc.z, sh.z);
              v[4 * q4 + 3] = fmaf(__uint_as_float(raw[h * 16 + 4 * q4 + 3]), sc.w, sh.w);
            }
          } else {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) v[jj] = __uint_as_float(raw[h * 16 + jj]);
          }
          if (residual && mvalid) {
            const uint4* rp = reinterpret_cast<const uint4*>(residual + m * G.Co + cc);
            const uint4 r0 = rp[0], r1 = rp[1];
            const __nv_bfloat162* h0 = reinterpret_cast<const __nv_bfloat162*>(&r0);
            const __nv_bfloat162* h1 = reinterpret_cast<const __nv_bfloat162*>(&r1);
#pragma unroll
            for (int jj = 0; jj < 4; ++jj) {
              const float2 a0 = __bfloat1622float2(h0[jj]);
              const float2 a1 = __bfloat1622float2(h1[jj]);
              v[2 * jj] += a0.x;
              v[2 * jj + 1] += a0.y;
              v[8 + 2 * jj] += a1.x;
              v[8 + 2 * jj + 1] += a1.y;
            }
          }
          if (act == 1) {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) v[jj] = v[jj] > 0.f ? v[jj] : 0.f;
          } else if (act == 2) {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) v[jj] = v[jj] > 0.f ? (v[jj] < 6.f ? v[jj] : 6.f) : 0.f;
          } else if (act == 3) {
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) v[jj] = gelu_f(v[jj]);
          }
          uint32_t pk[8];
#pragma unroll
          for (int jj = 0; jj < 8; ++jj) {
            const __nv_bfloat162 h2 = __floats2bfloat162_rn(v[2 * jj], v[2 * jj + 1]);
            pk[jj] = *reinterpret_cast<const uint32_t*>(&h2);
            nzw |= ((pk[jj] & 0x7FFFu) ? 1u : 0u) << (h * 16 + 2 * jj);
            nzw |= ((pk[jj] & 0x7FFF0000u) ? 1u : 0u) << (h * 16 + 2 * jj + 1);
          }
          if (mvalid) {
            uint4* yp = reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(P.y) + m * G.Co + cc);
            yp[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            yp[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
          }
        }
        if (!mvalid) nzw = 0u;
        if (emit) {
          if (nzw) tl |= 1ull << ((c0 >> 6) & 63);
          const uint32_t bits = __reduce_or_sync(grp, nzw);
          const int word = c0 >> 5;
          if (leader && blk >= 0 && bits) atomicOr(&o.blk_mask[blk * o.C32 + word], bits);
          s_cnt[q * CO + c0 + lane] = __popc(warp_transpose32(nzw));
        }
      }
      tc_fence_before();
      mbar_arrive(bar_acce + 8 * b);
      if (emit) {
        // both column halves of a row meet in shared memory; the tile owns its
        // output rows, so the half-0 thread stores the word once
        if (tl) atomicOr(&s_rowbm[r], tl);
        named_bar_sync(2, kEpiThreads);
        if (c0 == 0) {
          const unsigned long long v = s_rowbm[r];
          s_rowbm[r] = 0ull;
          if (mvalid) o.row_bm[m * o.W64] = v;
        }
        for (int c = et; c < CO; c += kEpiThreads)
          s_acc[c] += s_cnt[c] + s_cnt[CO + c] + s_cnt[2 * CO + c] + s_cnt[3 * CO + c];
        named_bar_sync(2, kEpiThreads);
      }
    }
    if (emit && acc_smem) {
      unsigned long long total = 0ull;
      for (int cb0 = 0; cb0 < CO; cb0 += kEpiThreads) {
        const int c = cb0 + et;
        const uint32_t cnt = c < CO ? s_acc[c] : 0u;
        if (cnt) atomicAdd(&o.col_nnz[c], cnt);
        uint32_t sum = cnt;
#pragma unroll
        for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
        total += sum;
        if (lane == 0 && sum) atomicAdd(&o.tile_nnz[c >> 6], sum);
      }
      if (lane == 0 && total) atomicAdd(o.nnz, total);
    }
  }

  __syncwarp();  // lanes that finished early wait for their warp's working lane
  tc_fence_before();
  __syncthreads();
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
