// Depthwise 3x3 convolution, pad 1, stride S in {1, 2} (every depthwise layer
// of MobileNetV2), with folded batch norm, activation, optional residual and
// the output's occupancy (Eq. 1 count and bitmaps, Sec. 3.1).
//
// A CTA computes output tiles of kTH x kTW pixels of one image and one
// 64-channel slice.  Each tile's input window with its halo is one 4-D TMA box
// {64 channels, IW, IH, 1} (coordinates outside the image read zeros, which is
// the padding) into shared memory laid out [IH][IW][64]; stride-1 CTAs keep
// two windows in flight.  The weights and the column affine of every channel
// sit in shared memory as fp32 for the whole kernel.
//
// Thread layout: warp w computes output row w of the tile; lanes 8 s .. 8 s + 7
// the 4 pixels 4 s .. 4 s + 3 of it, lane l channels 8 (l % 8) .. + 7 of the
// slice.  Channels go in pairs through packed fp32x2 FMAs (two products of
// the same rounding as two scalar FMAs, in the same order: kernel row, then
// kernel column), bf16 inputs are widened by shifts, and the activation is
// fused into the packing conversion.
//
// Work: with enough pixel tiles to fill the GPU a CTA runs every channel
// slice of its pixel tiles one after the other (the slices of a window share
// DRAM lines, which stay in L2), and owns those pixels' occupancy: row bits
// and 128-row block masks gather in shared memory and reach global memory
// once per pixel tile (row words as plain stores).  Otherwise an item is one
// (slice, pixel tile) and the bits go to global memory directly.  Column
// counts: per-thread 16-bit counters (two channels per word), kept in
// registers per slice for up to kRegSlices slices and reduced through shared
// memory into one global atomic per column per CTA; with more slices they are
// reduced after every step.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "sparoa_kernels.h"

namespace sparoa {

PFN_cuTensorMapEncodeTiled_v12000 tmap_encoder();  // k_igemm.cu

namespace {

constexpr int kThreads = 256;
constexpr int kTH = 8, kTW = 16;  // output tile: 8 rows (one per warp) x 16 pixels
constexpr int kMaxBlk = 16;       // 128-row blocks one output tile touches (Wo up to ~230)
constexpr int kRegSlices = 3;     // column counters kept in registers for up to 3 slices

template <int S>
struct Dw3Shape {
  static constexpr int IH = (kTH - 1) * S + 3, IW = (kTW - 1) * S + 3;
  static constexpr int NCOL = 3 * S + 3;         // input columns of a 4-pixel strip
  static constexpr int NB = S == 1 ? 2 : 1;      // input windows in flight
  static constexpr int kWinBytes = IH * IW * 128;
};

struct Dw3Geo {
  int Cp;            // channels rounded up to whole 64-channel slices
  int ctn;           // slices
  int tiles_h, tiles_w;
  int nsp;           // pixel tiles: N * tiles_h * tiles_w
  int own;           // a CTA runs every slice of its pixel tiles
  long long items;   // own ? nsp : nsp * ctn (item i: slice i / nsp of tile i % nsp)
  int win_off, w_off, aff_off, blk_off;  // shared-memory carve (bytes)
};

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const void* tmap, uint32_t bar, int c0, int c1,
                                            int c2, int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
      : "memory");
}

// a bf16 pair widened to fp32 (exact)
__device__ __forceinline__ f2_t widen(uint32_t w) {
  return f2(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}



struct Step {
  long long item;
  int n, ty, tx, ct, ct_end;
};

template <int S, int ACT>
__global__ void __launch_bounds__(kThreads, 2)
    dw3_kernel(const __grid_constant__ CUtensorMap tmX, const DwArgs a, const Dw3Geo G) {
  using Sh = Dw3Shape<S>;
  constexpr int IW = Sh::IW, NCOL = Sh::NCOL, NB = Sh::NB;
  extern __shared__ uint8_t dsm_raw[];
  uint8_t* dsm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 127) & ~uintptr_t(127));
  const uint32_t s_win = smem_u32(dsm + G.win_off);            // [NB][IH][IW][64] bf16
  const float* s_w = reinterpret_cast<const float*>(dsm + G.w_off);  // [9][Cp] weights
  float* s_wm = reinterpret_cast<float*>(dsm + G.w_off);
  float* s_sc = reinterpret_cast<float*>(dsm + G.aff_off);     // [Cp] affine scale
  float* s_sh = s_sc + G.Cp;                                   // [Cp] affine shift
  uint32_t* s_blk = reinterpret_cast<uint32_t*>(dsm + G.blk_off);  // [kMaxBlk][C32] (owned tiles)
  __shared__ __align__(8) unsigned long long s_bar[2];
  __shared__ uint32_t s_cnt[kThreads / 32][64];  // per-warp column counts of a slice
  __shared__ uint32_t s_row[kTH * kTW];          // row bits of an owned tile (slice ct: bit ct)
  __shared__ int s_abort;

  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int cg = lane & 7, st = lane >> 3;
  const OccDev o = a.out_occ;
  const bool emit = a.emit != 0;
  const bool own = G.own != 0;
  const bool reg_cnt = G.ctn <= kRegSlices;
  const long long wlim = a.wait_limit > 0 ? a.wait_limit : kWaitLimitCycles;
  const uint32_t bar0 = smem_u32(&s_bar[0]);

  if (threadIdx.x == 0) {
    for (int b = 0; b < NB; ++b) mbar_init(bar0 + 8 * b, 1u);
    s_abort = 0;
    fence_mbar_init();
    prefetch_tmap(&tmX);
  }
  if (own && emit) {
    for (int i = threadIdx.x; i < kMaxBlk * o.C32; i += kThreads) s_blk[i] = 0u;
    if (threadIdx.x < kTH * kTW) s_row[threadIdx.x] = 0u;
  }
  pdl_wait();
  pdl_trigger();
  if (a.path_out && blockIdx.x == 0 && threadIdx.x == 0) *a.path_out = 3;

  // steps of this CTA in order: items blockIdx.x, + gridDim.x, ...; every
  // slice of an owned item, else the item's one slice
  auto make_step = [&](long long item) {
    Step q;
    q.item = item;
    const int per_img = G.tiles_h * G.tiles_w;
    int ct_begin = 0;
    long long rest = item;
    if (!own) {
      ct_begin = (int)(item / G.nsp);
      rest = item - (long long)ct_begin * G.nsp;
    }
    q.ct = ct_begin;
    q.ct_end = own ? G.ctn : ct_begin + 1;
    q.n = (int)(rest / per_img);
    const int r2 = (int)(rest - (long long)q.n * per_img);
    q.ty = r2 / G.tiles_w;
    q.tx = r2 - q.ty * G.tiles_w;
    return q;
  };
  auto next_step = [&](const Step& q) {
    if (q.ct + 1 < q.ct_end) {
      Step r = q;
      r.ct = q.ct + 1;
      return r;
    }
    return make_step(q.item + gridDim.x);
  };
  auto issue = [&](const Step& q, int buf) {  // thread 0: one TMA box per input window
    const uint32_t bar = bar0 + 8 * buf;
    mbar_arrive_expect_tx(bar, (uint32_t)Sh::kWinBytes);
    tma_load_4d(s_win + (uint32_t)(buf * Sh::kWinBytes), &tmX, bar, q.ct * 64, q.tx * kTW * S - 1,
                q.ty * kTH * S - 1, q.n);
  };

  Step cur = make_step(blockIdx.x);
  Step iss = cur;  // thread 0: the next step whose window is to be loaded
  int issued = 0;
  if (threadIdx.x == 0) {
    for (int b = 0; b < NB && iss.item < G.items; ++b) {
      issue(iss, b);
      ++issued;
      iss = next_step(iss);
    }
  }
  // weights and affine of every channel, fp32 (zero / identity past C)
  for (int i = threadIdx.x; i < 9 * G.Cp; i += kThreads) {
    const int t = i / G.Cp, c = i - t * G.Cp;
    s_wm[i] = c < a.C ? __bfloat162float(a.w[c * 9 + t]) : 0.f;
  }
  for (int c = threadIdx.x; c < G.Cp; c += kThreads) {
    float sc = 1.f, sh = 0.f;
    if (c < a.C) epi_affine(a.ep, a.C, c, sc, sh);
    s_sc[c] = sc;
    s_sh[c] = sh;
  }
  __syncthreads();

  // column counts: cnt = this step's, 16-bit halves (channels 2p / 2p + 1);
  // cntr[k] = slice k's, kept while the CTA runs (reg_cnt); flush_counts
  // adds cnt of slice cnt_ct to global memory (every thread calls it)
  uint32_t cnt[4] = {0u, 0u, 0u, 0u};
  uint32_t cntr[kRegSlices][4];
#pragma unroll
  for (int k = 0; k < kRegSlices; ++k)
#pragma unroll
    for (int p = 0; p < 4; ++p) cntr[k][p] = 0u;
  int cnt_ct = 0, cnt_steps = 0;
  auto flush_counts = [&]() {
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      cnt[p] += __shfl_xor_sync(0xffffffffu, cnt[p], 8);   // the 4 strips of the warp
      cnt[p] += __shfl_xor_sync(0xffffffffu, cnt[p], 16);
    }
    if (st == 0) {
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        s_cnt[warp][cg * 8 + 2 * p] = cnt[p] & 0xFFFFu;
        s_cnt[warp][cg * 8 + 2 * p + 1] = cnt[p] >> 16;
      }
    }
#pragma unroll
    for (int p = 0; p < 4; ++p) cnt[p] = 0u;
    __syncthreads();
    if (threadIdx.x < 64) {
      uint32_t v = 0u;
#pragma unroll
      for (int w = 0; w < kThreads / 32; ++w) v += s_cnt[w][threadIdx.x];
      const int c = cnt_ct * 64 + threadIdx.x;
      if (c < a.C && v) atomicAdd(&o.col_nnz[c], v);
      uint32_t sum = v;
#pragma unroll
      for (int sft = 16; sft > 0; sft >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, sft);
      if (lane == 0 && sum) {
        atomicAdd(&o.tile_nnz[cnt_ct], sum);
        atomicAdd(o.nnz, (unsigned long long)sum);
      }
    }
    __syncthreads();
    cnt_steps = 0;
  };
  bool aborted = false;
  for (int sj = 0; cur.item < G.items; ++sj) {
    const int buf = NB == 2 ? (sj & 1) : 0;
    const uint32_t parity = (uint32_t)((NB == 2 ? (sj >> 1) : sj) & 1);
    const bool ok = mbar_wait(bar0 + 8 * buf, parity, a.err, &s_abort, kErrTimeoutFull, wlim);
    if (__syncthreads_or(!ok)) {
      aborted = true;
      break;
    }
    if (emit && reg_cnt && cnt_steps >= 4000) {  // before a 16-bit counter could overflow
      for (int k = 0; k < G.ctn; ++k) {
#pragma unroll
        for (int p = 0; p < 4; ++p) cnt[p] = k == 0 ? cntr[0][p] : (k == 1 ? cntr[1][p] : cntr[2][p]);
        cnt_ct = k;
        flush_counts();
      }
#pragma unroll
      for (int k = 0; k < kRegSlices; ++k)
#pragma unroll
        for (int p = 0; p < 4; ++p) cntr[k][p] = 0u;
    }
    const int n = cur.n, ty = cur.ty, tx = cur.tx, ct = cur.ct;
    const int c0 = ct * 64 + cg * 8;
    const int oy = warp, ox0 = st * 4;
    // ---------------------------------------------------------------- compute
    f2_t acc[4][4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int p = 0; p < 4; ++p) acc[j][p] = 0ull;
    const uint8_t* win = dsm + G.win_off + buf * Sh::kWinBytes;
#pragma unroll
    for (int r = 0; r < 3; ++r) {
      f2_t wr[3][4];
#pragma unroll
      for (int kc = 0; kc < 3; ++kc) {
        const ulonglong2 w01 = *reinterpret_cast<const ulonglong2*>(&s_w[(r * 3 + kc) * G.Cp + c0]);
        const ulonglong2 w23 = *reinterpret_cast<const ulonglong2*>(&s_w[(r * 3 + kc) * G.Cp + c0 + 4]);
        wr[kc][0] = w01.x;
        wr[kc][1] = w01.y;
        wr[kc][2] = w23.x;
        wr[kc][3] = w23.y;
      }
      const uint8_t* rowp = win + ((oy * S + r) * IW + ox0 * S) * 128 + cg * 16;
#pragma unroll
      for (int q = 0; q < NCOL; ++q) {
        const uint4 v = *reinterpret_cast<const uint4*>(rowp + q * 128);
        const f2_t in[4] = {widen(v.x), widen(v.y), widen(v.z), widen(v.w)};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int kc = q - j * S;  // kernel column pixel j applies to this input column
          if (kc >= 0 && kc < 3) {
#pragma unroll
            for (int p = 0; p < 4; ++p) acc[j][p] = ffma2(in[p], wr[kc][p], acc[j][p]);
          }
        }
      }
    }
    __syncthreads();  // every thread is done with this window: the next one may land there
    if (threadIdx.x == 0 && iss.item < G.items) {
      issue(iss, buf);
      ++issued;
      iss = next_step(iss);
    }
    // ---------------------------------------------------------------- epilogue
    const bool cvalid = c0 < a.C;
    f2_t sc2[4], sh2[4];
    {
      const ulonglong2 s01 = *reinterpret_cast<const ulonglong2*>(&s_sc[c0]);
      const ulonglong2 s23 = *reinterpret_cast<const ulonglong2*>(&s_sc[c0 + 4]);
      const ulonglong2 h01 = *reinterpret_cast<const ulonglong2*>(&s_sh[c0]);
      const ulonglong2 h23 = *reinterpret_cast<const ulonglong2*>(&s_sh[c0 + 4]);
      sc2[0] = s01.x; sc2[1] = s01.y; sc2[2] = s23.x; sc2[3] = s23.y;
      sh2[0] = h01.x; sh2[1] = h01.y; sh2[2] = h23.x; sh2[3] = h23.y;
    }
    const int oh = ty * kTH + oy;
    const uint32_t m_base = ((uint32_t)n * a.Ho + (oh < a.Ho ? oh : 0)) * a.Wo;
    uint32_t flags = 0u;                  // bit j: pixel j has a non-zero
    uint32_t blo_or[4] = {0u, 0u, 0u, 0u};  // non-zero pairs of pixels in the first pixel's block
    uint32_t bhi_or[4] = {0u, 0u, 0u, 0u};  // ... in the block after it
    const int ow0 = tx * kTW + ox0;
    const uint32_t blk_first = (m_base + (uint32_t)(ow0 < a.Wo ? ow0 : 0)) >> 7;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int ow = ow0 + j;
      const bool live = cvalid && oh < a.Ho && ow < a.Wo;
      const uint32_t m = m_base + (uint32_t)(ow < a.Wo ? ow : 0);
      uint4 res = make_uint4(0u, 0u, 0u, 0u);
      if (a.ep.residual && live) res = *reinterpret_cast<const uint4*>(a.ep.residual + (int64_t)m * a.C + c0);
      const uint32_t rw[4] = {res.x, res.y, res.z, res.w};
      uint32_t pk[4];
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        float lo, hi;
        f2_split(ffma2(acc[j][p], sc2[p], sh2[p]), lo, hi);
        if (a.ep.residual) {
          lo += __uint_as_float(rw[p] << 16);
          hi += __uint_as_float(rw[p] & 0xFFFF0000u);
        }
        pk[p] = act_pack2<ACT>(lo, hi);
      }
      if (live) {
        *reinterpret_cast<uint4*>(a.y + (int64_t)m * a.C + c0) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        if (emit) {
          const bool hi_blk = (m >> 7) != blk_first;
          uint32_t any = 0u;
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const uint32_t z = nz_pairs(pk[p]);
            cnt[p] += z;
            any |= z;
            if (hi_blk) bhi_or[p] |= z;
            else blo_or[p] |= z;
          }
          if (any) flags |= 1u << j;
        }
      }
    }
    if (emit) {
      // row bits: the pixel's 64 channels of this slice sit in the strip's 8 lanes
      uint32_t f = flags;
      f |= __shfl_xor_sync(0xffffffffu, f, 1);
      f |= __shfl_xor_sync(0xffffffffu, f, 2);
      f |= __shfl_xor_sync(0xffffffffu, f, 4);
      if (cg == 0 && f) {
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if (!((f >> j) & 1u)) continue;
          if (own && G.ctn <= 32)
            atomicOr(&s_row[oy * kTW + ox0 + j], 1u << ct);
          else
            atomicOr(&o.row_bm[(int64_t)(m_base + (uint32_t)(ow0 + j)) * o.W64 + (ct >> 6)], 1ull << (ct & 63));
        }
      }
      // block masks: this lane's 8 channels as bits 8 (cg % 4) .. of the
      // 32-channel word, OR-ed over the 4 lanes of the word
      auto bits8 = [](const uint32_t (&z)[4]) {
        uint32_t m8 = 0u;
#pragma unroll
        for (int p = 0; p < 4; ++p) m8 |= ((z[p] & 1u) | ((z[p] >> 15) & 2u)) << (2 * p);
        return m8;
      };
      uint32_t wlo = bits8(blo_or) << ((cg & 3) * 8), whi = bits8(bhi_or) << ((cg & 3) * 8);
      wlo |= __shfl_xor_sync(0xffffffffu, wlo, 1);
      wlo |= __shfl_xor_sync(0xffffffffu, wlo, 2);
      whi |= __shfl_xor_sync(0xffffffffu, whi, 1);
      whi |= __shfl_xor_sync(0xffffffffu, whi, 2);
      const int word = ct * 2 + (cg >> 2);
      if ((cg & 3) == 0 && word < o.C32) {
        const int b0 = (int)((((uint32_t)n * a.Ho + ty * kTH) * a.Wo + tx * kTW) >> 7);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const uint32_t v = h ? whi : wlo;
          if (!v) continue;
          const int blk = (int)blk_first + h;
          const int lb = blk - b0;
          if (own && lb >= 0 && lb < kMaxBlk) atomicOr(&s_blk[lb * o.C32 + word], v);
          else atomicOr(&o.blk_mask[(int64_t)blk * o.C32 + word], v);
        }
      }
      // this step's column counts: into slice ct's registers, or reduced now
      if (reg_cnt) {
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          if (ct == 0) cntr[0][p] += cnt[p];
          else if (ct == 1) cntr[1][p] += cnt[p];
          else cntr[2][p] += cnt[p];
          cnt[p] = 0u;
        }
        ++cnt_steps;
      } else {
        cnt_ct = ct;
        flush_counts();
      }
      if (own && cur.ct + 1 == cur.ct_end) {
        // the pixel tile is complete: its row words (plain stores) and its
        // block-mask words
        __syncthreads();
        if (G.ctn <= 32 && threadIdx.x < kTH * kTW) {
          const int py = threadIdx.x / kTW, px = threadIdx.x - py * kTW;
          const int ohh = ty * kTH + py, oww = tx * kTW + px;
          if (ohh < a.Ho && oww < a.Wo)
            o.row_bm[(int64_t)(((uint32_t)n * a.Ho + ohh) * a.Wo + oww) * o.W64] = s_row[threadIdx.x];
          s_row[threadIdx.x] = 0u;
        }
        const int b0 = (int)((((uint32_t)n * a.Ho + ty * kTH) * a.Wo + tx * kTW) >> 7);
        for (int i = threadIdx.x; i < kMaxBlk * o.C32; i += kThreads) {
          const uint32_t v = s_blk[i];
          if (v) {
            const int lb = i / o.C32, w = i - lb * o.C32;
            atomicOr(&o.blk_mask[(int64_t)(b0 + lb) * o.C32 + w], v);
            s_blk[i] = 0u;
          }
        }
      }
    }
    cur = next_step(cur);
  }
  if (aborted) {
    // a bounded wait ran out: the windows still in flight land before the
    // shared memory is released (each wait bounded again)
    if (threadIdx.x == 0) {
      for (int k = 0; k < NB && k < issued; ++k) {
        const int i = issued - 1 - k;
        const int b = NB == 2 ? (i & 1) : 0;
        mbar_drain(bar0 + 8 * b, (uint32_t)((NB == 2 ? (i >> 1) : i) & 1), wlim);
      }
    }
    return;
  }
  if (emit && reg_cnt) {
    for (int k = 0; k < G.ctn; ++k) {
#pragma unroll
      for (int p = 0; p < 4; ++p) cnt[p] = k == 0 ? cntr[0][p] : (k == 1 ? cntr[1][p] : cntr[2][p]);
      cnt_ct = k;
      flush_counts();
    }
  }
}

template <int S, int ACT>
cudaError_t launch_one(const CUtensorMap& tm, const DwArgs& a, const Dw3Geo& g, unsigned grid, size_t smem,
                       cudaStream_t s) {
  const void* fn = reinterpret_cast<const void*>(dw3_kernel<S, ACT>);
  cudaError_t e = smem_optin(fn, smem);
  if (e != cudaSuccess) return e;
  return launch_kernel(dw3_kernel<S, ACT>, dim3(grid), dim3(kThreads), smem, s, tm, a, g);
}

}  // namespace

bool dw3_supported(const DwArgs& a) {
  if (!(a.kh == 3 && a.kw == 3 && a.pad == 1 && (a.stride == 1 || a.stride == 2) && a.C % 8 == 0)) return false;
  if ((reinterpret_cast<uintptr_t>(a.x) & 15u) != 0) return false;  // TMA: 16-byte aligned base
  if (a.ep.act < 0 || a.ep.act > 3) return false;
  const int Cp = (a.C + 63) / 64 * 64, C32 = (a.C + 31) / 32;
  const int win = a.stride == 1 ? 2 * Dw3Shape<1>::kWinBytes : Dw3Shape<2>::kWinBytes;
  const size_t smem = 128 + (size_t)win + sizeof(float) * 11 * (size_t)Cp + sizeof(uint32_t) * (size_t)kMaxBlk * C32;
  return smem <= 110 * 1024;  // two CTAs per SM
}

cudaError_t launch_dw3(const DwArgs& a, cudaStream_t s) {
  Dw3Geo g;
  g.Cp = (a.C + 63) / 64 * 64;
  g.ctn = g.Cp / 64;
  g.tiles_h = (a.Ho + kTH - 1) / kTH;
  g.tiles_w = (a.Wo + kTW - 1) / kTW;
  const long long nsp = (long long)a.N * g.tiles_h * g.tiles_w;
  if (nsp * g.ctn >= (1ll << 31)) return cudaErrorInvalidValue;
  g.nsp = (int)nsp;
  g.own = (nsp >= 2ll * device_sm_count() && a.C <= 4096) ? 1 : 0;
  g.items = g.own ? nsp : nsp * g.ctn;
  const int C32 = (a.C + 31) / 32;
  const int win = a.stride == 1 ? 2 * Dw3Shape<1>::kWinBytes : Dw3Shape<2>::kWinBytes;
  g.win_off = 0;
  g.w_off = win;
  g.aff_off = g.w_off + (int)sizeof(float) * 9 * g.Cp;
  g.blk_off = g.aff_off + (int)sizeof(float) * 2 * g.Cp;
  const size_t smem = 128 + (size_t)g.blk_off + sizeof(uint32_t) * (size_t)kMaxBlk * C32;
  const long long cap = 2ll * device_sm_count();
  const unsigned grid = (unsigned)(g.items < cap ? g.items : cap);

  auto enc = tmap_encoder();
  if (!enc) return cudaErrorInvalidValue;
  CUtensorMap tm;
  const int IH = a.stride == 1 ? Dw3Shape<1>::IH : Dw3Shape<2>::IH;
  const int IW = a.stride == 1 ? Dw3Shape<1>::IW : Dw3Shape<2>::IW;
  cuuint64_t dims[4] = {(cuuint64_t)a.C, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.N};
  cuuint64_t strides[3] = {(cuuint64_t)a.C * 2, (cuuint64_t)a.W * a.C * 2, (cuuint64_t)a.H * a.W * a.C * 2};
  cuuint32_t box[4] = {64, (cuuint32_t)IW, (cuuint32_t)IH, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  if (enc(&tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>((const void*)a.x), dims, strides, box, estr,
          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_128B,
          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  const int act = a.ep.act;
  if (a.stride == 1) {
    if (act == 0) return launch_one<1, 0>(tm, a, g, grid, smem, s);
    if (act == 1) return launch_one<1, 1>(tm, a, g, grid, smem, s);
    if (act == 2) return launch_one<1, 2>(tm, a, g, grid, smem, s);
    return launch_one<1, 3>(tm, a, g, grid, smem, s);
  }
  if (act == 0) return launch_one<2, 0>(tm, a, g, grid, smem, s);
  if (act == 1) return launch_one<2, 1>(tm, a, g, grid, smem, s);
  if (act == 2) return launch_one<2, 2>(tm, a, g, grid, smem, s);
  return launch_one<2, 3>(tm, a, g, grid, smem, s);
}

}  // namespace sparoa
