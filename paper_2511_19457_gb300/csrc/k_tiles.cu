// Memory-bound kernels of the path.  Most work on 128-row x 64-channel tiles
// with 256 threads, thread t owning channels [8*(t%8), 8*(t%8)+8) of the tile
// (one 16-byte vector) in rows t/8 + 32*i, i = 0..3; the 3x3 depthwise and the
// global average pool lay their threads out as their comments say.  Each
// kernel fuses the occupancy emission of its output (Eq. 1 count and bitmaps,
// Sec. 3.1) so the next operator's dispatch reads them without another pass
// over HBM.
//   stats_kernel    Eq. 1 count and bitmaps of an existing tensor (C % 8 == 0;
//                   stats_scalar_kernel for other widths)
//   dwconv_kernel   depthwise convolutions other than the 3x3 shapes of
//                   k_dw3.cu
//   maxpool_kernel  k x k max pooling
//   avgpool_kernel  global average pooling
//   bn_act_kernel   stand-alone bias / batch norm / residual / activation
#include "sparoa_kernels.h"

namespace sparoa {

namespace {

constexpr int kTileThreads = 256;

__device__ __forceinline__ uint32_t nz_mask8(const uint4& u) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
  uint32_t m = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    if (w[j] & 0x7FFFu) m |= 1u << (2 * j);
    if (w[j] & 0x7FFF0000u) m |= 1u << (2 * j + 1);
  }
  return m;
}


// Occupancy of the 128-row x 64-column tiles a CTA produces.  Each thread
// holds an 8-bit non-zero mask per row it owns (lanes 8k..8k+7 of a warp share
// a row).  row() sets the row's bit in the row bitmap and counts columns in
// registers; tile_done() writes the tile's block-column mask words and adds
// its column counts to the CTA's shared counters s_acc[C]; cta_done() flushes
// those counters once (column, 64-column tile and total counts), so the
// atomics on one address number one per CTA, not one per tile.  Tensors wider
// than kMaxAccCols columns flush per tile instead.
constexpr int kMaxAccCols = 4096;

struct TileEmit {
  uint32_t cnt[8];
  __device__ __forceinline__ void init() {
#pragma unroll
    for (int j = 0; j < 8; ++j) cnt[j] = 0u;
  }
  // Every thread of the CTA calls this with its mask (0 outside the tensor).
  __device__ __forceinline__ void row(uint32_t mask, int64_t grow, int col0, const OccDev& o) {
    const int lane = threadIdx.x & 31;
    const uint32_t b = __ballot_sync(0xffffffffu, mask != 0u);
    if ((lane & 7) == 0 && ((b >> lane) & 0xFFu) != 0u)
      atomicOr(&o.row_bm[grow * o.W64 + (col0 >> 12)], 1ull << ((col0 >> 6) & 63));
#pragma unroll
    for (int j = 0; j < 8; ++j) cnt[j] += (mask >> j) & 1u;
  }
  // All threads; s_cnt holds 8 warps x 64 columns.
  __device__ __forceinline__ void tile_done(int64_t row0, int col0, const OccDev& o,
                                            uint32_t* s_cnt, uint32_t* s_acc, bool acc) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, cg = threadIdx.x & 7;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      cnt[j] += __shfl_xor_sync(0xffffffffu, cnt[j], 8);
      cnt[j] += __shfl_xor_sync(0xffffffffu, cnt[j], 16);
    }
    if (lane < 8) {
#pragma unroll
      for (int j = 0; j < 8; ++j) s_cnt[warp * 64 + cg * 8 + j] = cnt[j];
    }
    __syncthreads();
    if (threadIdx.x < 64) {
      uint32_t c = 0;
#pragma unroll
      for (int w = 0; w < kTileThreads / 32; ++w) c += s_cnt[w * 64 + threadIdx.x];
      const int col = col0 + threadIdx.x;
      const uint32_t word = __ballot_sync(0xffffffffu, c != 0u);
      const int w = (col0 >> 5) + (threadIdx.x >> 5);
      if (lane == 0 && word && w < o.C32) atomicOr(&o.blk_mask[(row0 >> 7) * o.C32 + w], word);
      if (acc) {
        if (col < o.C) s_acc[col] += c;
      } else {
        if (c && col < o.C) atomicAdd(&o.col_nnz[col], c);
        uint32_t sum = c;
#pragma unroll
        for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
        if (lane == 0 && sum) {
          atomicAdd(&o.tile_nnz[col0 >> 6], sum);
          atomicAdd(o.nnz, (unsigned long long)sum);
        }
      }
    }
    __syncthreads();
    init();
  }
};

__device__ __forceinline__ void acc_init(uint32_t* s_acc, int C, bool acc) {
  if (acc)
    for (int c = threadIdx.x; c < C; c += kTileThreads) s_acc[c] = 0u;
  __syncthreads();
}

__device__ __forceinline__ void cta_done(const OccDev& o, const uint32_t* s_acc, bool acc) {
  if (!acc) return;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  unsigned long long total = 0ull;
  for (int c0 = 0; c0 < o.C; c0 += kTileThreads) {
    const int c = c0 + threadIdx.x;
    const uint32_t cnt = c < o.C ? s_acc[c] : 0u;
    if (cnt) atomicAdd(&o.col_nnz[c], cnt);
    uint32_t sum = cnt;
#pragma unroll
    for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
    total += sum;
    if (lane == 0 && sum) atomicAdd(&o.tile_nnz[c >> 6], sum);
  }
  if (lane == 0 && total) atomicAdd(o.nnz, total);
}

// Tiles of a [R, C] output: rt = t / ct_count row tile, ct = t % ct_count column tile.
#define SPAROA_TILE_LOOP(R, C)                                                   \
  const int ctn = ((C) + 63) / 64;                                               \
  const int64_t ntiles = (((R) + 127) / 128) * (int64_t)ctn;                     \
  for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x)

// ---------------------------------------------------------------------------
// Eq. 1 count and bitmaps of a tensor of any width (the RGB input of a
// network among them; stats_kernel below takes C % 8 == 0).  A work item is a 128-row
// block x a chunk of up to kStatsChunk 64-column tiles; the next tile's loads
// are issued before the current one is reduced.  Block masks are owned by
// their item (plain stores); a row's bitmap word is stored whole when one
// chunk covers all of the row's tiles, else OR-ed in (the caller then clears
// the row bitmaps too).  Column counts gather in shared memory (C words,
// dynamic) and reach global memory once per CTA.
constexpr int kStatsChunk = kStatsWholeRowCols / 64;

__device__ __forceinline__ void stats_load(const __nv_bfloat16* __restrict__ x, int64_t R, int C,
                                           bool vec, int64_t row0, int col0, int cg, int rs,
                                           uint4 (&u)[4], uint32_t (&m)[4]) {
  const int c0 = col0 + cg * 8;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t r = row0 + rs + 32 * i;
    m[i] = 0u;
    u[i] = make_uint4(0u, 0u, 0u, 0u);
    if (r < R && c0 < C) {
      const __nv_bfloat16* p = x + r * C + c0;
      if (vec) {
        u[i] = __ldg(reinterpret_cast<const uint4*>(p));
      } else {
        for (int j = 0; j < 8 && c0 + j < C; ++j)
          if (bf16_nz(__bfloat16_as_ushort(p[j]))) m[i] |= 1u << j;
      }
    }
  }
}

__global__ void __launch_bounds__(kTileThreads, 3) stats_scalar_kernel(const __nv_bfloat16* __restrict__ x,
                                                                       int64_t R, int C, OccDev o_param,
                                                                       int chunk) {
  const OccDev o = o_param;  // registers, not parameter-space loads
  extern __shared__ uint32_t s_acc[];  // [C] when acc
  __shared__ uint32_t s_cnt[8 * 64];
  const bool acc = C <= kMaxAccCols;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const bool vec = (C & 7) == 0;
  const int ctn = (C + 63) / 64;
  const int nch = (ctn + chunk - 1) / chunk;
  const bool own_row = nch == 1;  // one chunk holds every tile of a row
  const int64_t nrb = (R + 127) / 128;
  const int64_t items = nrb * nch;
  if (acc)
    for (int c = threadIdx.x; c < C; c += kTileThreads) s_acc[c] = 0u;
  __syncthreads();
  pdl_wait();
  pdl_trigger();
  // The loads of the next tile -- of this item, else the first of the CTA's
  // next item -- are in flight while the current one is reduced.
  uint4 u[4];
  uint32_t m[4];
  if ((int64_t)blockIdx.x < items) {
    const int64_t rb = blockIdx.x / nch;
    stats_load(x, R, C, vec, rb * 128, (int)(blockIdx.x - rb * nch) * chunk * 64, cg, rs, u, m);
  }
  for (int64_t item = blockIdx.x; item < items; item += gridDim.x) {
    const int64_t rb = item / nch;
    const int ch = (int)(item - rb * nch);
    const int64_t row0 = rb * 128;
    const int ct0 = ch * chunk;
    const int ct1 = ct0 + chunk < ctn ? ct0 + chunk : ctn;
    unsigned long long rw[4] = {0ull, 0ull, 0ull, 0ull};  // row bitmap bits of this chunk, per owned row
    for (int ct = ct0; ct < ct1; ++ct) {
      const int col0 = ct * 64;
      if (vec) {
#pragma unroll
        for (int i = 0; i < 4; ++i) m[i] = nz_mask8(u[i]);
      }
      uint32_t mc[4] = {m[0], m[1], m[2], m[3]};
      if (ct + 1 < ct1) {
        stats_load(x, R, C, vec, row0, col0 + 64, cg, rs, u, m);  // next tile in flight
      } else if (item + gridDim.x < items) {
        const int64_t ni = item + gridDim.x, nrb2 = ni / nch;
        stats_load(x, R, C, vec, nrb2 * 128, (int)(ni - nrb2 * nch) * chunk * 64, cg, rs, u, m);
      }
      // row bits: lanes 8k..8k+7 share a row
      uint32_t cnt[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) cnt[j] = 0u;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t bl = __ballot_sync(0xffffffffu, mc[i] != 0u);
        if ((bl >> (lane & ~7)) & 0xFFu) rw[i] |= 1ull << (ct & 63);
#pragma unroll
        for (int j = 0; j < 8; ++j) cnt[j] += (mc[i] >> j) & 1u;
      }
      if ((ct & 63) == 63 || ct == ct1 - 1) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int64_t r = row0 + rs + 32 * i;
          if (cg == 0 && r < R) {
            unsigned long long* dst = &o.row_bm[r * o.W64 + (ct >> 6)];
            if (own_row) *dst = rw[i];
            else if (rw[i]) atomicOr(dst, rw[i]);
          }
          rw[i] = 0ull;
        }
      }
      // column counts of the tile: 8 warps x 64 columns through shared memory
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        cnt[j] += __shfl_xor_sync(0xffffffffu, cnt[j], 8);
        cnt[j] += __shfl_xor_sync(0xffffffffu, cnt[j], 16);
      }
      if (lane < 8) {
#pragma unroll
        for (int j = 0; j < 8; ++j) s_cnt[warp * 64 + cg * 8 + j] = cnt[j];
      }
      __syncthreads();
      if (threadIdx.x < 64) {
        uint32_t c = 0;
#pragma unroll
        for (int w = 0; w < kTileThreads / 32; ++w) c += s_cnt[w * 64 + threadIdx.x];
        const int col = col0 + threadIdx.x;
        const uint32_t word = __ballot_sync(0xffffffffu, c != 0u);
        const int w = (col0 >> 5) + (threadIdx.x >> 5);
        if (lane == 0 && w < o.C32) o.blk_mask[rb * o.C32 + w] = word;  // this item owns the word
        if (acc) {
          if (col < C) s_acc[col] += c;
        } else {
          // c is 0 for columns past C; all 32 lanes of both warps take part
          if (c) atomicAdd(&o.col_nnz[col], c);
          uint32_t sum = c;
#pragma unroll
          for (int s = 16; s > 0; s >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, s);
          if (lane == 0 && sum) {
            atomicAdd(&o.tile_nnz[ct], sum);
            atomicAdd(o.nnz, (unsigned long long)sum);
          }
        }
      }
      __syncthreads();
    }
  }
  cta_done(o, s_acc, acc);
}

// ---------------------------------------------------------------------------
// Eq. 1 count and bitmaps of a [R, C] tensor with C % 8 == 0, streamed with no
// barrier per tile.  The 128 x 64 tiles are numbered column tile first
// (L = ct * row_blocks + rb) and each CTA takes one contiguous range of them,
// so that it stays on one column tile for long runs: its column counts stay
// in registers (two 16-bit counters per 32-bit word) and reach global memory
// once per run (a barrier reduction, one atomic per column).  Per tile and
// row, the non-zero test is branch-free on pairs of bf16 values; row bits come
// from a ballot (the row's word stored whole when the tensor has one column
// tile, else OR-ed in); each warp ORs its block-column mask words into global
// memory.  Two register buffers alternate, so the next tile's loads are in
// flight while a tile is reduced.
constexpr int kStatsRunTiles = 8192;  // tiles per run: 4 rows each, under the 16-bit counters' 65535


// Grid-stride zeroing of up to five word ranges.
__device__ __forceinline__ void zero_ranges(const ClearArgs& a) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    uint32_t* p = a.p[k];
    const int64_t n = a.words[k];
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) p[i] = 0u;
  }
}

__global__ void __launch_bounds__(kTileThreads, 3) stats_kernel(const __nv_bfloat16* __restrict__ x,
                                                                int64_t R, int C, OccDev o_param,
                                                                int early, const ClearArgs zero) {
  const OccDev o = o_param;  // registers, not parameter-space loads
  __shared__ uint32_t s_cnt[8 * 64];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int ctn = (C + 63) / 64;
  const int64_t nrb = (R + 127) / 128;
  const int64_t P = nrb * ctn;
  const int64_t L0 = (int64_t)blockIdx.x * P / gridDim.x, L1 = ((int64_t)blockIdx.x + 1) * P / gridDim.x;
  const bool own_row = ctn == 1;  // the row's bitmap word is this tile's bit alone
  // (column tile, row block) of the first tile; later ones by stepping (no
  // 64-bit division per tile)
  const int ct0 = L0 < L1 ? (int)(L0 / nrb) : 0;
  const int64_t rb0 = L0 - (int64_t)ct0 * nrb;
  int64_t Ln = L0;  // next tile to load, at (l_ct, l_rb)
  int l_ct = ct0;
  int64_t l_rb = rb0;
  auto load = [&](uint4 (&u)[4]) {
    if (Ln < L1) {
      const int64_t r0 = l_rb * 128 + rs;
      const int c0 = l_ct * 64 + cg * 8;
      const __nv_bfloat16* p = x + r0 * C + c0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        u[i] = (r0 + 32 * i < R && c0 < C) ? __ldg(reinterpret_cast<const uint4*>(p))
                                           : make_uint4(0u, 0u, 0u, 0u);
        p += 32 * (int64_t)C;
      }
    }
    ++Ln;
    if (++l_rb == nrb) {
      l_rb = 0;
      ++l_ct;
    }
  };
  uint32_t cnt[4] = {0u, 0u, 0u, 0u};  // columns cg*8 + 2w (low half), + 2w + 1 (high half)
  auto flush = [&](int ct) {
    uint32_t c8[8];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      c8[2 * w] = cnt[w] & 0xFFFFu;
      c8[2 * w + 1] = cnt[w] >> 16;
      cnt[w] = 0u;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      c8[j] += __shfl_xor_sync(0xffffffffu, c8[j], 8);
      c8[j] += __shfl_xor_sync(0xffffffffu, c8[j], 16);
    }
    if (lane < 8) {
#pragma unroll
      for (int j = 0; j < 8; ++j) s_cnt[warp * 64 + lane * 8 + j] = c8[j];
    }
    __syncthreads();
    if (threadIdx.x < 64) {
      uint32_t c = 0u;
#pragma unroll
      for (int w = 0; w < kTileThreads / 32; ++w) c += s_cnt[w * 64 + threadIdx.x];
      if (c) atomicAdd(&o.col_nnz[ct * 64 + threadIdx.x], c);  // 0 for columns past C
      uint32_t sum = c;
#pragma unroll
      for (int sh = 16; sh > 0; sh >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, sh);
      if (lane == 0 && sum) {
        atomicAdd(&o.tile_nnz[ct], sum);
        atomicAdd(o.nnz, (unsigned long long)sum);
      }
    }
    __syncthreads();
  };
  int run_ct = ct0;
  int run_tiles = 0;
  int t_ct = ct0;  // the tile being reduced
  int64_t t_rb = rb0;
  auto tile = [&](uint4 (&u)[4]) {
    const int ct = t_ct;
    const int64_t row0 = t_rb * 128;
    if (++t_rb == nrb) {
      t_rb = 0;
      ++t_ct;
    }
    if (ct != run_ct || run_tiles == kStatsRunTiles) {  // the same for every thread
      flush(run_ct);
      run_ct = ct;
      run_tiles = 0;
    }
    ++run_tiles;
    uint32_t n[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      n[i][0] = nz_pairs(u[i].x);
      n[i][1] = nz_pairs(u[i].y);
      n[i][2] = nz_pairs(u[i].z);
      n[i][3] = nz_pairs(u[i].w);
    }
    load(u);  // the tile two ahead
    uint32_t o4[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      cnt[w] += (n[0][w] + n[1][w]) + (n[2][w] + n[3][w]);  // at most 4 per 16-bit half
      o4[w] = (n[0][w] | n[1][w]) | (n[2][w] | n[3][w]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const uint32_t b = __ballot_sync(0xffffffffu, (n[i][0] | n[i][1] | n[i][2] | n[i][3]) != 0u);
      const int64_t r = row0 + rs + 32 * i;
      if ((lane & 7) == 0 && r < R) {
        const bool nzr = ((b >> lane) & 0xFFu) != 0u;
        if (own_row) o.row_bm[r] = nzr ? 1ull : 0ull;
        else if (nzr) atomicOr(&o.row_bm[r * o.W64 + (ct >> 6)], 1ull << (ct & 63));
      }
    }
    // block-column mask: this thread's 8 columns over its 4 rows, then OR-ed over
    // the warp's lanes of the same 32 columns; lanes 0 and 4 hold the two words
    const uint32_t m8 = (o4[0] & 1u) | ((o4[0] >> 15) & 2u) | ((o4[1] << 2) & 4u) | ((o4[1] >> 13) & 8u) |
                        ((o4[2] << 4) & 16u) | ((o4[2] >> 11) & 32u) | ((o4[3] << 6) & 64u) |
                        ((o4[3] >> 9) & 128u);
    uint32_t v = m8 << ((cg & 3) * 8);
    v |= __shfl_xor_sync(0xffffffffu, v, 1);
    v |= __shfl_xor_sync(0xffffffffu, v, 2);
    v |= __shfl_xor_sync(0xffffffffu, v, 8);
    v |= __shfl_xor_sync(0xffffffffu, v, 16);
    if ((lane & 27) == 0 && v) {  // lanes 0 and 4
      const int w = ct * 2 + (lane >> 2);
      if (w < o.C32) atomicOr(&o.blk_mask[(row0 >> 7) * o.C32 + w], v);
    }
  };
  // with `early` (x complete when the grid starts) the first two tiles are in
  // flight while griddepcontrol.wait waits for the clear of the counters
  uint4 ua[4], ub[4];
  if (early) {
    load(ua);
    load(ub);
    pdl_wait();
    pdl_trigger();
  } else {
    pdl_wait();
    pdl_trigger();
    load(ua);
    load(ub);
  }
  zero_ranges(zero);  // another block's counters and masks (the loads are in flight)
  for (int64_t L = L0; L < L1; ++L) {
    tile(ua);
    if (++L >= L1) break;
    tile(ub);
  }
  flush(run_ct);
}

// ---------------------------------------------------------------------------
// Streamed element-wise producers: the stats kernel's tile order and
// occupancy scheme (contiguous runs of column-tile-major 128 x 64 tiles per
// CTA, column counts in 16-bit register halves flushed once per run, row bits
// by ballot, block-column masks OR-ed per warp) with the tile's values made
// and stored first.  No barrier per tile; the next tile's loads are in flight
// while a tile is transformed.
struct StreamEmit {
  uint32_t cnt[4];  // columns cg*8 + 2w (low half) and + 2w + 1 (high half)
  int run_ct, run_tiles;
};

__device__ __forceinline__ void stream_flush(StreamEmit& e, uint32_t* s_cnt, const OccDev& o) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t c8[8];
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    c8[2 * w] = e.cnt[w] & 0xFFFFu;
    c8[2 * w + 1] = e.cnt[w] >> 16;
    e.cnt[w] = 0u;
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    c8[j] += __shfl_xor_sync(0xffffffffu, c8[j], 8);
    c8[j] += __shfl_xor_sync(0xffffffffu, c8[j], 16);
  }
  if (lane < 8) {
#pragma unroll
    for (int j = 0; j < 8; ++j) s_cnt[warp * 64 + lane * 8 + j] = c8[j];
  }
  __syncthreads();
  if (threadIdx.x < 64) {
    uint32_t c = 0u;
#pragma unroll
    for (int w = 0; w < kTileThreads / 32; ++w) c += s_cnt[w * 64 + threadIdx.x];
    if (c) atomicAdd(&o.col_nnz[e.run_ct * 64 + threadIdx.x], c);  // 0 for columns past C
    uint32_t sum = c;
#pragma unroll
    for (int sh = 16; sh > 0; sh >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, sh);
    if (lane == 0 && sum) {
      atomicAdd(&o.tile_nnz[e.run_ct], sum);
      atomicAdd(o.nnz, (unsigned long long)sum);
    }
  }
  __syncthreads();
}

// n[i][w]: nz_pairs of word w of this thread's row i (0 outside the tensor).
// Called by every thread with the same tile sequence.
__device__ __forceinline__ void stream_tile(StreamEmit& e, const uint32_t (&n)[4][4], int ct, int64_t row0,
                                            int64_t R, bool own_row, uint32_t* s_cnt, const OccDev& o) {
  const int lane = threadIdx.x & 31, cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  if (ct != e.run_ct || e.run_tiles == kStatsRunTiles) {
    stream_flush(e, s_cnt, o);
    e.run_ct = ct;
    e.run_tiles = 0;
  }
  ++e.run_tiles;
  uint32_t o4[4];
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    e.cnt[w] += (n[0][w] + n[1][w]) + (n[2][w] + n[3][w]);
    o4[w] = (n[0][w] | n[1][w]) | (n[2][w] | n[3][w]);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t b = __ballot_sync(0xffffffffu, (n[i][0] | n[i][1] | n[i][2] | n[i][3]) != 0u);
    const int64_t r = row0 + rs + 32 * i;
    if ((lane & 7) == 0 && r < R) {
      const bool nzr = ((b >> lane) & 0xFFu) != 0u;
      if (own_row) o.row_bm[r] = nzr ? 1ull : 0ull;
      else if (nzr) atomicOr(&o.row_bm[r * o.W64 + (ct >> 6)], 1ull << (ct & 63));
    }
  }
  const uint32_t m8 = (o4[0] & 1u) | ((o4[0] >> 15) & 2u) | ((o4[1] << 2) & 4u) | ((o4[1] >> 13) & 8u) |
                      ((o4[2] << 4) & 16u) | ((o4[2] >> 11) & 32u) | ((o4[3] << 6) & 64u) |
                      ((o4[3] >> 9) & 128u);
  uint32_t v = m8 << ((cg & 3) * 8);
  v |= __shfl_xor_sync(0xffffffffu, v, 1);
  v |= __shfl_xor_sync(0xffffffffu, v, 2);
  v |= __shfl_xor_sync(0xffffffffu, v, 8);
  v |= __shfl_xor_sync(0xffffffffu, v, 16);
  if ((lane & 27) == 0 && v) {  // lanes 0 and 4
    const int w = ct * 2 + (lane >> 2);
    if (w < o.C32) atomicOr(&o.blk_mask[(row0 >> 7) * o.C32 + w], v);
  }
}


// Stand-alone bias / batch norm / residual / activation over [R, C] (C % 8
// == 0), y and its occupancy.  The activation and the presence of a residual
// are compile-time parameters, so that a tile's 32 values per thread go
// through straight-line code (bf16 halves widened by shifts, one FMA each,
// the activation fused into the packing conversion).
template <int ACT, bool RES>
__global__ void __launch_bounds__(kTileThreads, 2) bn_act_kernel(const __nv_bfloat16* __restrict__ x, int64_t R,
                                                                 int C, EpiDev ep_param,
                                                                 __nv_bfloat16* __restrict__ y, OccDev o_param,
                                                                 int emit) {
  const OccDev o = o_param;
  const EpiDev ep = ep_param;
  __shared__ uint32_t s_cnt[8 * 64];
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int ctn = (C + 63) / 64;
  const int64_t nrb = (R + 127) / 128;
  const int64_t P = nrb * ctn;
  const int64_t L0 = (int64_t)blockIdx.x * P / gridDim.x, L1 = ((int64_t)blockIdx.x + 1) * P / gridDim.x;
  const bool own_row = ctn == 1;
  const int ct0 = L0 < L1 ? (int)(L0 / nrb) : 0;
  const int64_t rb0 = L0 - (int64_t)ct0 * nrb;
  const __nv_bfloat16* const res = ep.residual;
  pdl_wait();
  pdl_trigger();
  int64_t Ln = L0;
  int l_ct = ct0;
  int64_t l_rb = rb0;
  auto load = [&](uint4 (&u)[4]) {
    if (Ln < L1) {
      const int64_t r0 = l_rb * 128 + rs;
      const int c0 = l_ct * 64 + cg * 8;
      const int64_t off = r0 * C + c0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const bool ok = r0 + 32 * i < R && c0 < C;
        u[i] = ok ? __ldg(reinterpret_cast<const uint4*>(x + off + 32 * i * (int64_t)C)) : make_uint4(0u, 0u, 0u, 0u);
      }
    }
    ++Ln;
    if (++l_rb == nrb) {
      l_rb = 0;
      ++l_ct;
    }
  };
  StreamEmit e;
#pragma unroll
  for (int w = 0; w < 4; ++w) e.cnt[w] = 0u;
  e.run_ct = ct0;
  e.run_tiles = 0;
  int aff_ct = -1;
  float sc[8], sh[8];
  int t_ct = ct0;
  int64_t t_rb = rb0;
  auto tile = [&](uint4 (&u)[4]) {
    const int ct = t_ct;
    const int64_t row0 = t_rb * 128;
    if (++t_rb == nrb) {
      t_rb = 0;
      ++t_ct;
    }
    const int c0 = ct * 64 + cg * 8;
    if (ct != aff_ct) {  // the column affine of this thread's 8 columns
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        sc[j] = 1.f;
        sh[j] = 0.f;
        if (c0 + j < C) epi_affine(ep, C, c0 + j, sc[j], sh[j]);
      }
      aff_ct = ct;
    }
    uint4 ur[4];  // the residual rows, all in flight together
    if (RES) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int64_t r = row0 + rs + 32 * i;
        ur[i] = (r < R && c0 < C) ? *reinterpret_cast<const uint4*>(res + r * C + c0) : make_uint4(0u, 0u, 0u, 0u);
      }
    }
    uint32_t n[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t r = row0 + rs + 32 * i;
      const uint32_t* xw = reinterpret_cast<const uint32_t*>(&u[i]);
      const uint32_t* rw = reinterpret_cast<const uint32_t*>(&ur[i]);
      uint4 pk;
      uint32_t* pw = reinterpret_cast<uint32_t*>(&pk);
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        float lo = fmaf(__uint_as_float(xw[w] << 16), sc[2 * w], sh[2 * w]);
        float hi = fmaf(__uint_as_float(xw[w] & 0xFFFF0000u), sc[2 * w + 1], sh[2 * w + 1]);
        if (RES) {
          lo += __uint_as_float(rw[w] << 16);
          hi += __uint_as_float(rw[w] & 0xFFFF0000u);
        }
        pw[w] = act_pack2<ACT>(lo, hi);
      }
      const bool ok = r < R && c0 < C;
      if (ok) *reinterpret_cast<uint4*>(y + r * C + c0) = pk;
      n[i][0] = ok ? nz_pairs(pk.x) : 0u;
      n[i][1] = ok ? nz_pairs(pk.y) : 0u;
      n[i][2] = ok ? nz_pairs(pk.z) : 0u;
      n[i][3] = ok ? nz_pairs(pk.w) : 0u;
    }
    load(u);  // the tile two ahead
    if (emit) stream_tile(e, n, ct, row0, R, own_row, s_cnt, o);
  };
  uint4 ua[4], ub[4];
  load(ua);
  load(ub);
  for (int64_t L = L0; L < L1; ++L) {
    tile(ua);
    if (++L >= L1) break;
    tile(ub);
  }
  if (emit) stream_flush(e, s_cnt, o);
}

// k x k max pooling (C % 8 == 0), y [N, Ho, Wo, C] and its occupancy: per
// output row and 8 channels, the window's taps are loaded together (addresses
// clamped into the image; taps outside it count as -inf) and reduced with
// packed bf16 maxima.
__global__ void __launch_bounds__(kTileThreads, 3)
    maxpool_kernel(const __nv_bfloat16* __restrict__ x, int N, int H, int W, int C, int k,
                   int stride, int pad, int Ho, int Wo, __nv_bfloat16* __restrict__ y, OccDev o_param,
                   int emit) {
  const OccDev o = o_param;
  __shared__ uint32_t s_cnt[8 * 64];
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int64_t R = (int64_t)N * Ho * Wo;
  const int ctn = (C + 63) / 64;
  const int64_t nrb = (R + 127) / 128;
  const int64_t P = nrb * ctn;
  const int64_t L0 = (int64_t)blockIdx.x * P / gridDim.x, L1 = ((int64_t)blockIdx.x + 1) * P / gridDim.x;
  const bool own_row = ctn == 1;
  const int hw = Ho * Wo;
  pdl_wait();
  pdl_trigger();
  StreamEmit e;
#pragma unroll
  for (int w = 0; w < 4; ++w) e.cnt[w] = 0u;
  e.run_ct = L0 < L1 ? (int)(L0 / nrb) : 0;
  e.run_tiles = 0;
  const __nv_bfloat162 ninf = __halves2bfloat162(__ushort_as_bfloat16(0xFF80u), __ushort_as_bfloat16(0xFF80u));
  for (int64_t L = L0; L < L1; ++L) {
    const int ct = (int)(L / nrb);
    const int64_t row0 = (L - (int64_t)ct * nrb) * 128;
    const int c0 = ct * 64 + cg * 8;
    uint32_t n[4][4];
    uint4 outv[4];
    bool okr[4];
    if (k == 3) {
      // This thread's output rows row0 + rs + 32 i: (image, oh, ow) by one
      // division for the first and stepping for the others; an output whose
      // 3 x 3 window lies inside the image loads its taps at fixed offsets
      // from one address, a border output clamps each tap and leaves the
      // outside ones out.  Two outputs at a time: 18 loads in flight.
      const int64_t m0 = row0 + rs;
      int img = 0, oh = 0, ow = 0;
      if (m0 < R) {
        const int mr = (int)m0;
        img = mr / hw;
        const int rem = mr - img * hw;
        oh = rem / Wo;
        ow = rem - oh * Wo;
      }
      const int64_t rowC = (int64_t)W * C;
#pragma unroll
      for (int i0 = 0; i0 < 4; i0 += 2) {
        uint4 u[2][9];
        uint32_t inb[2];
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
          const int i = i0 + ii;
          if (i > 0) {  // the next output row of this thread: 32 positions on
            ow += 32;
            while (ow >= Wo) {
              ow -= Wo;
              if (++oh == Ho) {
                oh = 0;
                ++img;
              }
            }
          }
          okr[i] = m0 + 32 * i < R && c0 < C;
          const int ih0 = oh * stride - pad, iw0 = ow * stride - pad;
          const bool inner = ih0 >= 0 && ih0 + 2 < H && iw0 >= 0 && iw0 + 2 < W;
          inb[ii] = 0x1FFu;
          if (!okr[i]) {
#pragma unroll
            for (int t = 0; t < 9; ++t) u[ii][t] = make_uint4(0u, 0u, 0u, 0u);
          } else if (inner) {
            const __nv_bfloat16* p = x + (((int64_t)img * H + ih0) * W + iw0) * C + c0;
#pragma unroll
            for (int r = 0; r < 3; ++r)
#pragma unroll
              for (int s2 = 0; s2 < 3; ++s2)
                u[ii][r * 3 + s2] = __ldg(reinterpret_cast<const uint4*>(p + r * rowC + s2 * C));
          } else {
            inb[ii] = 0u;
#pragma unroll
            for (int r = 0; r < 3; ++r) {
              const int ih = ih0 + r;
              const int ihc = ih < 0 ? 0 : (ih >= H ? H - 1 : ih);
#pragma unroll
              for (int s2 = 0; s2 < 3; ++s2) {
                const int iw = iw0 + s2;
                const int iwc = iw < 0 ? 0 : (iw >= W ? W - 1 : iw);
                if (ih == ihc && iw == iwc) inb[ii] |= 1u << (r * 3 + s2);
                u[ii][r * 3 + s2] =
                    __ldg(reinterpret_cast<const uint4*>(x + (((int64_t)img * H + ihc) * W + iwc) * C + c0));
              }
            }
          }
        }
#pragma unroll
        for (int ii = 0; ii < 2; ++ii) {
          __nv_bfloat162 m[4] = {ninf, ninf, ninf, ninf};
#pragma unroll
          for (int t = 0; t < 9; ++t) {
            if (!((inb[ii] >> t) & 1u)) continue;
            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u[ii][t]);
#pragma unroll
            for (int w = 0; w < 4; ++w) m[w] = __hmax2(m[w], h[w]);
          }
          outv[i0 + ii] = make_uint4(*reinterpret_cast<uint32_t*>(&m[0]), *reinterpret_cast<uint32_t*>(&m[1]),
                                     *reinterpret_cast<uint32_t*>(&m[2]), *reinterpret_cast<uint32_t*>(&m[3]));
        }
      }
    } else {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int64_t mrow = row0 + rs + 32 * i;
        okr[i] = mrow < R && c0 < C;
        __nv_bfloat162 m[4] = {ninf, ninf, ninf, ninf};
        if (okr[i]) {
          const int mr = (int)mrow;
          const int img = mr / hw, rem = mr - (mr / hw) * hw;
          const int oh = rem / Wo, ow = rem - (rem / Wo) * Wo;
          for (int r = 0; r < k; ++r) {
            const int ih = oh * stride - pad + r;
            if (ih < 0 || ih >= H) continue;
            for (int s2 = 0; s2 < k; ++s2) {
              const int iw = ow * stride - pad + s2;
              if (iw < 0 || iw >= W) continue;
              const uint4 v = __ldg(reinterpret_cast<const uint4*>(x + (((int64_t)img * H + ih) * W + iw) * C + c0));
              const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
              for (int w = 0; w < 4; ++w) m[w] = __hmax2(m[w], h[w]);
            }
          }
        }
        outv[i] = make_uint4(*reinterpret_cast<uint32_t*>(&m[0]), *reinterpret_cast<uint32_t*>(&m[1]),
                             *reinterpret_cast<uint32_t*>(&m[2]), *reinterpret_cast<uint32_t*>(&m[3]));
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t mrow = row0 + rs + 32 * i;
      if (okr[i]) *reinterpret_cast<uint4*>(y + mrow * C + c0) = outv[i];
      n[i][0] = okr[i] ? nz_pairs(outv[i].x) : 0u;
      n[i][1] = okr[i] ? nz_pairs(outv[i].y) : 0u;
      n[i][2] = okr[i] ? nz_pairs(outv[i].z) : 0u;
      n[i][3] = okr[i] ? nz_pairs(outv[i].w) : 0u;
    }
    if (emit) stream_tile(e, n, ct, row0, R, own_row, s_cnt, o);
  }
  if (emit) stream_flush(e, s_cnt, o);
}

// ---------------------------------------------------------------------------
// ---------------------------------------------------------------------------
// Narrow tensors (C < 8 channels, the RGB input): a thread takes groups of 8
// consecutive rows = C 16-byte words (the group starts on a 16-byte boundary
// when x does), so every load is a full vector.  Element e of a group is row
// e / C, channel e % C; its non-zero bit goes to bit e of a 64-bit mask, and
// the channel counts are population counts of the mask under a constant
// per-channel pattern.
template <int C>
struct NarrowMasks {
  static constexpr unsigned long long chan(int c) {
    unsigned long long m = 0ull;
    for (int p = 0; p < 8; ++p) m |= 1ull << (p * C + c);
    return m;
  }
};

template <int C>
__device__ __forceinline__ bool narrow_load(const __nv_bfloat16* __restrict__ x, int64_t R, int64_t g,
                                            uint32_t (&w)[4 * C]) {
  const int64_t r0 = g * 8;
  if (r0 + 8 <= R) {
    const uint4* p = reinterpret_cast<const uint4*>(x + r0 * C);
#pragma unroll
    for (int k = 0; k < C; ++k) {
      const uint4 v = __ldg(p + k);
      w[4 * k] = v.x;
      w[4 * k + 1] = v.y;
      w[4 * k + 2] = v.z;
      w[4 * k + 3] = v.w;
    }
    return true;
  }
  // the last, partial group: element by element, zero past the tensor
  const uint16_t* q = reinterpret_cast<const uint16_t*>(x);
  const int64_t n = (R - r0) * C;
#pragma unroll
  for (int k = 0; k < 4 * C; ++k) {
    const uint32_t lo = 2 * k < n ? q[r0 * C + 2 * k] : 0u;
    const uint32_t hi = 2 * k + 1 < n ? q[r0 * C + 2 * k + 1] : 0u;
    w[k] = lo | (hi << 16);
  }
  return false;
}

// Eq. 1 count and occupancy of an [R, C] tensor with C < 8.  Rows are whole
// words of the row bitmap (one column tile) and a half warp's 16 groups are
// one 128-row block, so row words and block masks are plain stores; the
// counts meet in shared memory and reach global memory once per CTA.
template <int C>
__global__ void __launch_bounds__(256) stats_narrow_kernel(const __nv_bfloat16* __restrict__ x, int64_t R,
                                                           OccDev o, int early) {
  __shared__ uint32_t s_cnt[C];
  const int lane = threadIdx.x & 31;
  if (threadIdx.x < C) s_cnt[threadIdx.x] = 0u;
  __syncthreads();
  if (!early) {
    pdl_wait();
    pdl_trigger();
  }
  const int64_t groups = (R + 7) / 8;
  const int64_t RB = (R + 127) / 128;
  uint32_t cnt[C];
#pragma unroll
  for (int c = 0; c < C; ++c) cnt[c] = 0u;
  bool waited = !early;
  // whole warps step together (32 groups = two 128-row blocks per step)
  const int64_t wstride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); g0 < groups; g0 += wstride) {
    const int64_t g = g0 + lane;
    uint32_t w[4 * C];
    if (g < groups) narrow_load<C>(x, R, g, w);
    else
#pragma unroll
      for (int k = 0; k < 4 * C; ++k) w[k] = 0u;
    if (!waited) {  // the loads of the first step were issued before the wait
      pdl_wait();
      pdl_trigger();
      waited = true;
    }
    unsigned long long m = 0ull;
#pragma unroll
    for (int k = 0; k < 4 * C; ++k) {
      const uint32_t t = ((w[k] & 0x7FFF7FFFu) + 0x7FFF7FFFu) >> 15;
      m |= (unsigned long long)(t & 1u) << (2 * k);
      m |= (unsigned long long)((t >> 16) & 1u) << (2 * k + 1);
    }
    uint32_t chbits = 0u;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const unsigned long long mc = m & NarrowMasks<C>::chan(c);
      cnt[c] += (uint32_t)__popcll(mc);
      chbits |= (mc != 0ull ? 1u : 0u) << c;
    }
    if (g < groups) {
      const int64_t r0 = g * 8;
#pragma unroll
      for (int p = 0; p < 8; ++p)
        if (r0 + p < R) o.row_bm[r0 + p] = ((m >> (p * C)) & ((1ull << C) - 1ull)) ? 1ull : 0ull;
    }
    // block masks: lanes 0-15 and 16-31 are the blocks g0 / 16 and g0 / 16 + 1
    const uint32_t blo = __reduce_or_sync(0xffffffffu, lane < 16 ? chbits : 0u);
    const uint32_t bhi = __reduce_or_sync(0xffffffffu, lane >= 16 ? chbits : 0u);
    const int64_t b = g0 / 16;
    if (lane == 0 && b < RB) o.blk_mask[b] = blo;
    if (lane == 16 && b + 1 < RB) o.blk_mask[b + 1] = bhi;
  }
  if (!waited) {
    pdl_wait();
    pdl_trigger();
  }
#pragma unroll
  for (int c = 0; c < C; ++c) {
    const uint32_t v = __reduce_add_sync(0xffffffffu, cnt[c]);
    if (lane == 0 && v) atomicAdd(&s_cnt[c], v);
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t tot = 0u;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const uint32_t v = s_cnt[c];
      if (v) atomicAdd(&o.col_nnz[c], v);
      tot += v;
    }
    if (tot) {
      atomicAdd(&o.tile_nnz[0], tot);
      atomicAdd(o.nnz, (unsigned long long)tot);
    }
  }
}

// [P, C] -> [P, 8] (C < 8, zero channels appended): C 16-byte loads and 8
// 16-byte stores per group of 8 rows.
template <int C>
__global__ void __launch_bounds__(256) pad8_kernel(const __nv_bfloat16* __restrict__ x, int64_t P,
                                                   __nv_bfloat16* __restrict__ y) {
  pdl_wait();
  pdl_trigger();
  const int64_t groups = (P + 7) / 8;
  for (int64_t g = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g < groups;
       g += (int64_t)gridDim.x * blockDim.x) {
    uint32_t w[4 * C];
    narrow_load<C>(x, P, g, w);
    const uint16_t* h = reinterpret_cast<const uint16_t*>(w);
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      if (g * 8 + p >= P) break;
      uint32_t o4[4] = {0u, 0u, 0u, 0u};
#pragma unroll
      for (int c = 0; c < C; ++c) o4[c >> 1] |= (uint32_t)h[p * C + c] << (16 * (c & 1));
      reinterpret_cast<uint4*>(y)[g * 8 + p] = make_uint4(o4[0], o4[1], o4[2], o4[3]);
    }
  }
}

// im2col for a convolution with few input channels (the RGB stems):
// x [N, H, W, C] -> xc [N Ho Wo, Kp], row (n, oh, ow) = the kh x kw x C window
// of output pixel (n, oh, ow) in [kh][kw][C] order (zero outside the image),
// columns Kc = kh kw C .. Kp - 1 zero (Kp = Kc rounded up to 32).  The
// convolution is then a plain GEMM of xc with the weights [C_out][Kc] padded to
// Kp, whose A rows the implicit GEMM loads with 2-D TMA boxes of 128-byte rows.
// One CTA per output row (n, oh): the kh zero-padded input rows it needs are
// staged in shared memory (row r at r RLp + pre, `pre` placing the image part
// of each row on a 16-byte boundary so that aligned rows are copied in 16-byte
// pieces), where window element k of pixel ow sits at off[k] + ow S C.  Each
// thread owns one 16-byte chunk position q of the output rows (its eight
// offsets in registers) and writes that chunk for every (256 / Q)-th pixel.
__global__ void __launch_bounds__(256) im2col_kernel(const __nv_bfloat16* __restrict__ x, int N, int H, int W,
                                                     int C, int kh, int kw, int S, int P, int Ho, int Wo, int Kp,
                                                     __nv_bfloat16* __restrict__ xc) {
  extern __shared__ uint4 s_v4[];
  const int RL = (W + 2 * P) * C;               // elements of one padded input row
  const int pre = (8 - (P * C) % 8) % 8;        // leading slack: image part 16-byte aligned
  const int RLp = (pre + RL + 7) / 8 * 8;       // row pitch (elements)
  const int Kc = kh * kw * C, Q = Kp / 8;
  uint16_t* s_rows = reinterpret_cast<uint16_t*>(s_v4);
  const int ppc = (int)blockDim.x / Q;          // pixels per pass
  const int q = (int)threadIdx.x % Q, p0 = (int)threadIdx.x / Q;
  int off[8];
#pragma unroll
  for (int t = 0; t < 8; ++t) {
    const int k = 8 * q + t;
    off[t] = -1;
    if (k < Kc) {
      const int c = k % C, tap = k / C;
      off[t] = (tap / kw) * RLp + pre + (tap % kw) * C + c;
    }
  }
  pdl_wait();
  pdl_trigger();
  const uint16_t* xs = reinterpret_cast<const uint16_t*>(x);
  const bool vec = (W * C) % 8 == 0 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0;
  const int img0 = pre + P * C, img1 = img0 + W * C;  // image part of a staged row
  for (int64_t row = blockIdx.x; row < (int64_t)N * Ho; row += gridDim.x) {
    const int n = (int)(row / Ho), oh = (int)(row - (int64_t)n * Ho);
    __syncthreads();  // the previous row's readers are done
    for (int r = 0; r < kh; ++r) {
      const int ih = oh * S - P + r;
      uint16_t* dst = s_rows + r * RLp;
      if (ih < 0 || ih >= H) {
        for (int i = threadIdx.x; i < RLp / 8; i += blockDim.x) reinterpret_cast<uint4*>(dst)[i] = make_uint4(0, 0, 0, 0);
        continue;
      }
      const uint16_t* src = xs + ((int64_t)n * H + ih) * W * C;
      for (int i = threadIdx.x; i < img0; i += blockDim.x) dst[i] = 0;
      for (int i = img1 + threadIdx.x; i < RLp; i += blockDim.x) dst[i] = 0;
      if (vec) {
        for (int i = threadIdx.x; i < W * C / 8; i += blockDim.x)
          reinterpret_cast<uint4*>(dst + img0)[i] = reinterpret_cast<const uint4*>(src)[i];
      } else {
        for (int i = threadIdx.x; i < W * C; i += blockDim.x) dst[img0 + i] = src[i];
      }
    }
    __syncthreads();
    if (p0 >= ppc) continue;  // threads past the last whole pass of pixels
    uint4* out = reinterpret_cast<uint4*>(xc + row * Wo * Kp) + q;
    for (int ow = p0; ow < Wo; ow += ppc) {
      const int base = ow * S * C;
      uint32_t o[4];
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        const uint32_t lo = off[2 * t] >= 0 ? s_rows[off[2 * t] + base] : 0u;
        const uint32_t hi = off[2 * t + 1] >= 0 ? s_rows[off[2 * t + 1] + base] : 0u;
        o[t] = lo | (hi << 16);
      }
      out[(int64_t)ow * Q] = make_uint4(o[0], o[1], o[2], o[3]);
    }
  }
}

__global__ void pad_kernel(const __nv_bfloat16* __restrict__ x, int64_t P, int C, int Cp,
                           __nv_bfloat16* __restrict__ y) {
  pdl_wait();
  pdl_trigger();
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= P * Cp) return;
  const int64_t p = i / Cp;
  const int c = (int)(i - p * Cp);
  y[i] = c < C ? x[p * C + c] : __float2bfloat16_rn(0.f);
}

// ---------------------------------------------------------------------------
// Depthwise 3x3 convolution (stride 1 or 2, any padding) + epilogue.
__global__ void __launch_bounds__(kTileThreads) dwconv_kernel(const DwArgs a_param) {
  const DwArgs a = a_param;  // registers, not parameter-space loads
  __shared__ uint32_t s_cnt[8 * 64];
  extern __shared__ uint32_t s_acc[];  // [C] when acc (dynamic)
  __shared__ __align__(16) float s_w[9][64];
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int64_t R = (int64_t)a.N * a.Ho * a.Wo;
  const bool acc = a.emit && a.C <= kMaxAccCols;
  acc_init(s_acc, a.C, acc);
  pdl_wait();
  pdl_trigger();
  if (a.path_out && blockIdx.x == 0 && threadIdx.x == 0) *a.path_out = 3;
  TileEmit e;
  e.init();
  const int hw = a.Ho * a.Wo;
  const int64_t img_elems = (int64_t)a.H * a.W * a.C;
  int cur_col0 = -1;
  float sc[8], sh[8];
  // channel slice major: a CTA's consecutive tiles share their weights and affine
  const int ctn = (a.C + 63) / 64;
  const int64_t nrt = (R + 127) / 128;
  const int64_t ntiles = nrt * ctn;
  for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
    const int64_t row0 = (tile % nrt) * 128;
    const int col0 = (int)(tile / nrt) * 64;
    const int c0 = col0 + cg * 8;
    const bool cvalid = c0 < a.C;
    if (col0 != cur_col0) {  // (uniform) new channel slice: weights and affine
      __syncthreads();
      for (int idx = threadIdx.x; idx < 9 * 64; idx += kTileThreads) {
        const int t = idx / 64, c = idx % 64;
        s_w[t][c] = (col0 + c < a.C) ? __bfloat162float(a.w[(int64_t)(col0 + c) * 9 + t]) : 0.f;
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        sc[j] = 1.f;
        sh[j] = 0.f;
        if (cvalid) epi_affine(a.ep, a.C, c0 + j, sc[j], sh[j]);
      }
      __syncthreads();
      cur_col0 = col0;
    }
    // Every tap's load is unconditional (its address clamped into the image;
    // out-of-range taps are zeroed afterwards), so a row's 9 loads, and the
    // next row's, are in flight together instead of one latency each.
#pragma unroll 2
    for (int i = 0; i < 4; ++i) {
      const int64_t mrow_raw = row0 + rs + 32 * i;
      const bool live = cvalid && mrow_raw < R;
      const int64_t mrow = live ? mrow_raw : 0;
      uint32_t mask = 0;
      {
        // 32-bit index math (output rows and in-image offsets stay below 2^31;
        // the launcher checks), 64-bit only for the image base
        const uint32_t m32 = (uint32_t)mrow;
        const uint32_t img = m32 / (uint32_t)hw;
        const uint32_t rem = m32 - img * (uint32_t)hw;
        const int oh = (int)(rem / (uint32_t)a.Wo), ow = (int)(rem - (rem / (uint32_t)a.Wo) * (uint32_t)a.Wo);
        const __nv_bfloat16* xi = a.x + (int64_t)img * img_elems + (cvalid ? c0 : 0);
        uint4 u[9];
        uint32_t inb = 0u;
#pragma unroll
        for (int r = 0; r < 3; ++r) {
          const int ih = oh * a.stride - a.pad + r;
          const int ihc = ih < 0 ? 0 : (ih >= a.H ? a.H - 1 : ih);
#pragma unroll
          for (int s = 0; s < 3; ++s) {
            const int iw = ow * a.stride - a.pad + s;
            const int iwc = iw < 0 ? 0 : (iw >= a.W ? a.W - 1 : iw);
            if (ih == ihc && iw == iwc) inb |= 1u << (r * 3 + s);
            u[r * 3 + s] = __ldg(reinterpret_cast<const uint4*>(xi + (uint32_t)(ihc * a.W + iwc) * (uint32_t)a.C));
          }
        }
        float accv[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) accv[j] = 0.f;
#pragma unroll
        for (int t = 0; t < 9; ++t) {
          float f[8];
          unpack8(((inb >> t) & 1u) ? u[t] : make_uint4(0u, 0u, 0u, 0u), f);
          const float4 w0 = *reinterpret_cast<const float4*>(&s_w[t][cg * 8]);
          const float4 w1 = *reinterpret_cast<const float4*>(&s_w[t][cg * 8 + 4]);
          const float wv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
#pragma unroll
          for (int j = 0; j < 8; ++j) accv[j] = fmaf(f[j], wv[j], accv[j]);
        }
        float rv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (a.ep.residual && live) unpack8(*reinterpret_cast<const uint4*>(a.ep.residual + mrow * a.C + c0), rv);
        float o[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) o[j] = epi_act(fmaf(accv[j], sc[j], sh[j]) + rv[j], a.ep.act);
        const uint4 uo = pack8(o);
        if (live) {
          *reinterpret_cast<uint4*>(a.y + mrow * a.C + c0) = uo;
          mask = nz_mask8(uo);
        }
      }
      if (a.emit) e.row(mask, mrow_raw, col0, a.out_occ);
    }
    if (a.emit) e.tile_done(row0, col0, a.out_occ, s_cnt, s_acc, acc);
  }
  if (a.emit) cta_done(a.out_occ, s_acc, acc);
}

// ---------------------------------------------------------------------------
// Global average pooling [N, HW, C] -> [N, C] (C % 8 == 0): one CTA per (image,
// 64-channel slice).  Lane l of warp w sums pixels 4 w + l / 8 + 32 k of the 8
// channels 8 (l % 8) .. + 7, so every load of the CTA is in flight at once;
// the 32 pixel partial sums of a channel meet by shuffles and in shared
// memory, and threads 0..63 finish one channel each: the mean, its bf16 value
// and the output occupancy (atomics into the cleared block: row bit, column,
// tile and total counts, block-column mask words).
__global__ void __launch_bounds__(kTileThreads)
    avgpool_kernel(const __nv_bfloat16* __restrict__ x, int N, int HW, int C,
                   __nv_bfloat16* __restrict__ y, OccDev o_param, int emit) {
  const OccDev o = o_param;
  __shared__ float s_part[8 * 64];  // [warp][channel of the slice]
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int cg = lane & 7, pq = warp * 4 + (lane >> 3);  // channel group, pixel lane 0..31
  const int ctn = (C + 63) / 64;
  const int n = (int)(blockIdx.x / ctn), ct = (int)(blockIdx.x - (blockIdx.x / ctn) * ctn);
  const int c0 = ct * 64 + cg * 8;
  pdl_wait();
  pdl_trigger();
  float a8[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (c0 < C) {
    const __nv_bfloat16* p = x + (int64_t)n * HW * C + c0;
    for (int q = pq; q < HW; q += 32) {
      float f[8];
      unpack8(__ldg(reinterpret_cast<const uint4*>(p + (int64_t)q * C)), f);
#pragma unroll
      for (int j = 0; j < 8; ++j) a8[j] += f[j];
    }
  }
  // lanes cg, cg + 8, cg + 16, cg + 24 of a warp hold the same channels
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    a8[j] += __shfl_xor_sync(0xffffffffu, a8[j], 8);
    a8[j] += __shfl_xor_sync(0xffffffffu, a8[j], 16);
  }
  if (lane < 8) {
#pragma unroll
    for (int j = 0; j < 8; ++j) s_part[warp * 64 + lane * 8 + j] = a8[j];
  }
  __syncthreads();
  if (threadIdx.x < 64) {  // two full warps
    const int c = ct * 64 + (int)threadIdx.x;
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kTileThreads / 32; ++w) sum += s_part[w * 64 + threadIdx.x];
    const __nv_bfloat16 b = __float2bfloat16_rn(sum / (float)HW);
    const bool live = c < C;
    if (live) y[(int64_t)n * C + c] = b;
    const bool nz = live && (__bfloat16_as_ushort(b) & 0x7FFFu) != 0u;
    if (emit) {
      const uint32_t word = __ballot_sync(0xffffffffu, nz);  // this warp's 32 columns
      if (nz) atomicAdd(&o.col_nnz[c], 1u);
      if (lane == 0 && word) {
        const int w = ct * 2 + (int)(threadIdx.x >> 5);
        if (w < o.C32) atomicOr(&o.blk_mask[(int64_t)(n >> 7) * o.C32 + w], word);
        atomicAdd(&o.tile_nnz[ct], (uint32_t)__popc(word));
        atomicAdd(o.nnz, (unsigned long long)__popc(word));
        atomicOr(&o.row_bm[(int64_t)n * o.W64 + (ct >> 6)], 1ull << (ct & 63));
      }
    }
  }
}

// Dynamic shared memory of a tile kernel: the per-CTA column counters.
size_t acc_smem(int emit, int C) {
  return (emit && C <= kMaxAccCols) ? sizeof(uint32_t) * (size_t)C : 0;
}

// Zero the word ranges of a ClearArgs (grid-stride over the longest range).
__global__ void __launch_bounds__(256) clear_kernel(const ClearArgs a) {
  pdl_wait();
  pdl_trigger();
  zero_ranges(a);
}

// Grid-stride over 128 x 64 tiles with at most 4 CTAs per SM.
unsigned tile_grid(int64_t R, int C) {
  const int64_t tiles = ((R + 127) / 128) * ((C + 63) / 64);
  const int64_t cap = 4LL * device_sm_count();
  return (unsigned)(tiles < cap ? tiles : cap);
}

// Column tiles per stats work item: whole chunks while the row blocks alone
// give the GPU enough items, single tiles for short tensors.
int stats_chunk(int64_t R, int C) {
  const int64_t nrb = (R + 127) / 128;
  return (C > 64 && nrb < device_sm_count()) ? 1 : kStatsChunk;
}

}  // namespace

bool stats_writes_rows_whole(int64_t R, int C) {
  (void)R;
  return C <= 64;  // one column tile: both kernels store each row's word whole
}

// CTAs of the stats kernel for an [R, C] tensor.
unsigned stats_grid(int64_t R, int C) {
  const int64_t tiles = ((R + 127) / 128) * ((C + 63) / 64);
  if (C % 8 != 0) {
    const int chunk = stats_chunk(R, C);
    const int64_t items = ((R + 127) / 128) * ((((C + 63) / 64) + chunk - 1) / chunk);
    const int64_t cap = 3LL * device_sm_count();
    return (unsigned)(items < cap ? items : cap);
  }
  const int64_t cap = 3LL * device_sm_count();  // the resident CTAs (3 per SM) split the tiles
  return (unsigned)(tiles < cap ? tiles : cap);
}

cudaError_t launch_stats(const __nv_bfloat16* x, int64_t R, int C, const OccDev& o, cudaStream_t s,
                         bool early, const ClearArgs* zero) {
  if (R <= 0 || C <= 0) return cudaSuccess;
  ClearArgs z = {};
  if (zero) z = *zero;
  if (C % 8 == 0) {
    const unsigned grid = stats_grid(R, C);
    return launch_kernel(stats_kernel, dim3(grid), dim3(kTileThreads), 0, s, x, R, C, o, early ? 1 : 0, z);
  }
  if (zero) {  // the kernels below zero nothing: a clear launch first
    const cudaError_t e = launch_clear(z, s);
    if (e != cudaSuccess) return e;
  }
  if (C < 8 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0) {
    const int64_t groups = (R + 7) / 8;
    const int64_t cap = 4LL * device_sm_count();
    int64_t blocks = (groups + 255) / 256;
    blocks = blocks < cap ? blocks : cap;
    const int e1 = early ? 1 : 0;
    switch (C) {
      case 1: return launch_kernel(stats_narrow_kernel<1>, dim3((unsigned)blocks), dim3(256), 0, s, x, R, o, e1);
      case 2: return launch_kernel(stats_narrow_kernel<2>, dim3((unsigned)blocks), dim3(256), 0, s, x, R, o, e1);
      case 3: return launch_kernel(stats_narrow_kernel<3>, dim3((unsigned)blocks), dim3(256), 0, s, x, R, o, e1);
      case 4: return launch_kernel(stats_narrow_kernel<4>, dim3((unsigned)blocks), dim3(256), 0, s, x, R, o, e1);
      case 5: return launch_kernel(stats_narrow_kernel<5>, dim3((unsigned)blocks), dim3(256), 0, s, x, R, o, e1);
      case 6: return launch_kernel(stats_narrow_kernel<6>, dim3((unsigned)blocks), dim3(256), 0, s, x, R, o, e1);
      default: return launch_kernel(stats_narrow_kernel<7>, dim3((unsigned)blocks), dim3(256), 0, s, x, R, o, e1);
    }
  }
  const int chunk = stats_chunk(R, C);
  const unsigned grid = stats_grid(R, C);  // the resident CTAs (3 per SM) loop over the items
  const size_t smem = C <= kMaxAccCols ? sizeof(uint32_t) * (size_t)C : 0;
  return launch_kernel(stats_scalar_kernel, dim3(grid), dim3(kTileThreads), smem, s, x, R, C, o, chunk);
}

cudaError_t launch_clear(const ClearArgs& a, cudaStream_t s) {
  int64_t mx = 0;
  for (int k = 0; k < 5; ++k) mx = a.words[k] > mx ? a.words[k] : mx;
  if (mx <= 0) return cudaSuccess;
  const int64_t blocks = (mx + 255) / 256;
  const int64_t cap = 2LL * device_sm_count();
  return launch_kernel(clear_kernel, dim3((unsigned)(blocks < cap ? blocks : cap)), dim3(256), 0, s, a);
}

static size_t im2col_smem(int W, int C, int kh, int P) {
  const int64_t pre = (8 - (P * C) % 8) % 8;
  const int64_t RLp = (pre + (int64_t)(W + 2 * P) * C + 7) / 8 * 8;
  return sizeof(uint16_t) * (size_t)(kh * RLp);
}

int im2col_width(int C, int kh, int kw) { return (kh * kw * C + 31) / 32 * 32; }

bool im2col_applies(int C, int kh, int kw, int groups, int W, int P) {
  if (groups != 1 || C >= 8 || kh * kw <= 1) return false;
  const int Kp = im2col_width(C, kh, kw);
  return Kp <= 512 && im2col_smem(W, C, kh, P) <= 48 * 1024;
}

cudaError_t launch_im2col(const __nv_bfloat16* x, int N, int H, int W, int C, int kh, int kw, int S, int P,
                          __nv_bfloat16* xc, cudaStream_t s) {
  const int Ho = (H + 2 * P - kh) / S + 1, Wo = (W + 2 * P - kw) / S + 1;
  const int64_t rows = (int64_t)N * Ho;
  if (rows <= 0 || Wo <= 0) return cudaSuccess;
  if (!im2col_applies(C, kh, kw, 1, W, P) || (reinterpret_cast<uintptr_t>(xc) & 15u) != 0)
    return cudaErrorInvalidValue;
  const int Kp = im2col_width(C, kh, kw);
  const int64_t cap = 8LL * device_sm_count();
  return launch_kernel(im2col_kernel, dim3((unsigned)(rows < cap ? rows : cap)), dim3(256),
                       im2col_smem(W, C, kh, P), s, x, N, H, W, C, kh, kw, S, P, Ho, Wo, Kp, xc);
}

cudaError_t launch_pad_channels(const __nv_bfloat16* x, int64_t P, int C, int Cp,
                                __nv_bfloat16* y, cudaStream_t s) {
  const int64_t n = P * Cp;
  if (n <= 0) return cudaSuccess;
  if (Cp == 8 && C < 8 && (reinterpret_cast<uintptr_t>(x) & 15u) == 0 && (reinterpret_cast<uintptr_t>(y) & 15u) == 0) {
    const int64_t groups = (P + 7) / 8;
    const int64_t cap = 4LL * device_sm_count();
    int64_t blocks = (groups + 255) / 256;
    const dim3 grid((unsigned)(blocks < cap ? blocks : cap));
    switch (C) {
      case 1: return launch_kernel(pad8_kernel<1>, grid, dim3(256), 0, s, x, P, y);
      case 2: return launch_kernel(pad8_kernel<2>, grid, dim3(256), 0, s, x, P, y);
      case 3: return launch_kernel(pad8_kernel<3>, grid, dim3(256), 0, s, x, P, y);
      case 4: return launch_kernel(pad8_kernel<4>, grid, dim3(256), 0, s, x, P, y);
      case 5: return launch_kernel(pad8_kernel<5>, grid, dim3(256), 0, s, x, P, y);
      case 6: return launch_kernel(pad8_kernel<6>, grid, dim3(256), 0, s, x, P, y);
      default: return launch_kernel(pad8_kernel<7>, grid, dim3(256), 0, s, x, P, y);
    }
  }
  return launch_kernel(pad_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, x, P, C, Cp, y);
}

cudaError_t launch_dwconv(const DwArgs& a, cudaStream_t s) {
  const int64_t R = (int64_t)a.N * a.Ho * a.Wo;
  if (R <= 0) return cudaSuccess;
  // the kernels' 32-bit index math: output rows and one image's elements
  if (R >= ((int64_t)1 << 31) || (int64_t)a.H * a.W * a.C >= ((int64_t)1 << 31)) return cudaErrorInvalidValue;
  if (dw3_supported(a)) return launch_dw3(a, s);
  return launch_kernel(dwconv_kernel, dim3(tile_grid(R, a.C)), dim3(kTileThreads),
                       acc_smem(a.emit, a.C), s, a);
}

cudaError_t launch_maxpool(const __nv_bfloat16* x, int N, int H, int W, int C, int k, int stride,
                           int pad, int Ho, int Wo, __nv_bfloat16* y, const OccDev& o, int emit,
                           cudaStream_t s) {
  const int64_t R = (int64_t)N * Ho * Wo;
  if (R <= 0) return cudaSuccess;
  if (C % 8) return cudaErrorInvalidValue;
  const int64_t tiles = ((R + 127) / 128) * ((C + 63) / 64);
  const int64_t cap = 3LL * device_sm_count();  // the resident CTAs split the tiles
  return launch_kernel(maxpool_kernel, dim3((unsigned)(tiles < cap ? tiles : cap)), dim3(kTileThreads), 0,
                       s, x, N, H, W, C, k, stride, pad, Ho, Wo, y, o, emit);
}

cudaError_t launch_avgpool(const __nv_bfloat16* x, int N, int HW, int C, __nv_bfloat16* y,
                           const OccDev& o, int emit, cudaStream_t s) {
  if (N <= 0) return cudaSuccess;
  if (C % 8) return cudaErrorInvalidValue;
  const int64_t ctas = (int64_t)N * ((C + 63) / 64);
  if (ctas >= ((int64_t)1 << 31)) return cudaErrorInvalidValue;
  return launch_kernel(avgpool_kernel, dim3((unsigned)ctas), dim3(kTileThreads), 0, s, x, N, HW, C, y, o,
                       emit);
}

cudaError_t launch_bn_act(const __nv_bfloat16* x, int64_t R, int C, const EpiDev& ep,
                          __nv_bfloat16* y, const OccDev& o, int emit, cudaStream_t s) {
  if (R <= 0) return cudaSuccess;
  if (C % 8) return cudaErrorInvalidValue;
  const int64_t tiles = ((R + 127) / 128) * ((C + 63) / 64);
  const int64_t cap2 = 2LL * device_sm_count();  // the resident CTAs (two per SM) split the tiles
  const dim3 grid((unsigned)(tiles < cap2 ? tiles : cap2));
  const bool res = ep.residual != nullptr;
  switch (ep.act * 2 + (res ? 1 : 0)) {
    case 0: return launch_kernel(bn_act_kernel<0, false>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    case 1: return launch_kernel(bn_act_kernel<0, true>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    case 2: return launch_kernel(bn_act_kernel<1, false>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    case 3: return launch_kernel(bn_act_kernel<1, true>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    case 4: return launch_kernel(bn_act_kernel<2, false>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    case 5: return launch_kernel(bn_act_kernel<2, true>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    case 6: return launch_kernel(bn_act_kernel<3, false>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    case 7: return launch_kernel(bn_act_kernel<3, true>, grid, dim3(kTileThreads), 0, s, x, R, C, ep, y, o, emit);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace sparoa
