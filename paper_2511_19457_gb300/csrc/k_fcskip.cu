// Column-compacting zero-skip fully connected kernel for few rows.
//
// y[M, N] = epilogue(x[M, K] * W[N, K]^T) where, per 128-row block of x, only
// the columns k that hold a non-zero in that block take part (Sec. 2.1:
// products with a zero activation are skipped without changing the output).
// The block-column mask of x (one bit per column per 128-row block) gives the
// occupied columns; the kernel compacts them into a list and reads only the
// matching rows of W stored as [K, N] (each a contiguous run of N values, so
// skipped columns cost no HBM traffic), accumulating in fp32 on the CUDA
// cores.  This is the path for small-M layers (a batch of feature vectors),
// which are bound by the weight bytes and by latency, not by arithmetic.
//
// CTA = 64 rows x 16 output columns (many CTAs even for a handful of rows),
// 256 threads.  Per window of kKW columns of K the CTA stages its x rows whole
// (coalesced cp.async; the first window is in flight while the occupied
// columns are listed) and the W-row slices of the window's occupied columns
// (bf16), then the threads split the occupied columns four ways: thread
// (slice, row group, column group) accumulates a 4-row x 4-column outer
// product over every fourth occupied column, reading x straight from the
// staged rows (no compaction pass).  The four slices' sums meet in shared
// memory, where every thread takes one row x 4 columns for the epilogue.
#include "sparoa_kernels.h"

namespace sparoa {

namespace {

constexpr int kThreads = 256;
constexpr int kTM = 64;           // rows per CTA
constexpr int kTN = 16;           // output columns per CTA
constexpr int kKW = 512;          // K window staged at once
constexpr int kPitch = kKW + 8;   // bf16 elements per staged x row (16-byte multiple; rows 1..7
                                  // apart fall in different banks)
constexpr int kSlices = 4;        // ways the occupied columns are split
constexpr int kMaxWin = 32;       // K windows (K <= kMaxWin * kKW)

struct FcSmem {
  static constexpr size_t kX = (size_t)kTM * kPitch * 2;   // x window, bf16, rows whole
  static constexpr size_t kW = (size_t)kKW * kTN * 2;      // occupied W rows, bf16; then the slice sums
  static_assert(kW >= (size_t)kSlices * kTM * kTN * 4, "slice sums fit the W buffer");
  static constexpr size_t kBytes = kX + kW + (kMaxWin + 2) * 4;  // + window starts, count
};

__device__ __forceinline__ void stage_x(uint32_t xs_u32, const FcSkipArgs& a, int64_t m0, int k0, int kw,
                                        int tid) {
  const int chunks = kw / 8;  // K % 8 == 0
  for (int idx = tid; idx < kTM * chunks; idx += kThreads) {
    const int r = idx / chunks, c = idx - (idx / chunks) * chunks;
    const bool ok = m0 + r < a.M;
    const __nv_bfloat16* src = ok ? a.x + (m0 + r) * a.K + k0 + c * 8 : a.x;
    cp_async_16(xs_u32 + (uint32_t)((r * kPitch + c * 8) * 2), src, ok ? 16u : 0u);
  }
  cp_async_commit();
}

__global__ void __launch_bounds__(kThreads) fcskip_kernel(const FcSkipArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(smem);                   // [kTM][kPitch]
  __nv_bfloat16* wsb = reinterpret_cast<__nv_bfloat16*>(smem + FcSmem::kX);     // [kk][kTN]
  float* red = reinterpret_cast<float*>(smem + FcSmem::kX);                     // [slice][kTM][kTN]
  int* s_misc = reinterpret_cast<int*>(smem + FcSmem::kX + FcSmem::kW);  // [0] count, [1..] window starts
  short* s_col = reinterpret_cast<short*>(smem + FcSmem::kBytes);               // [K] occupied columns (< 32768)
  __shared__ uint32_t s_cnt[kTN];
  __shared__ uint32_t s_blk;

  pdl_wait();
  pdl_trigger();
  const int path = decide_path(a.disp);
  if (path != 2) return;  // the dense kernel of this launch runs instead
  record_path(a.disp, path);

  const int n0 = blockIdx.x * kTN;
  const int64_t m0 = (int64_t)blockIdx.y * kTM;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int row = tid >> 2, cq = tid & 3;  // epilogue: this thread's row and 4-column group
  const int64_t m = m0 + row;
  // accumulation: slice sl takes occupied columns sl, sl + 4, ...; rows rg + 16 i, columns 4 cg ..
  const int sl = tid >> 6, u = tid & 63, rg = u >> 2, cg = u & 3;
  const uint32_t xs_u32 = smem_u32(xs);
  const int nwin = (a.K + kKW - 1) / kKW;

  // 0. the first x window is loaded while the occupied columns are listed
  stage_x(xs_u32, a, m0, 0, a.K < kKW ? a.K : kKW, tid);

  // 1. occupied columns of the rows' 128-row block, in increasing order
  if (warp == 0) {
    const int rb = (int)(m0 >> 7);
    int base = 0;
    for (int w0 = 0; w0 < a.in_C32; w0 += 32) {
      uint32_t word = (w0 + lane < a.in_C32) ? a.in_blk[(int64_t)rb * a.in_C32 + w0 + lane] : 0u;
      const int cnt = __popc(word);
      int incl = cnt;
#pragma unroll
      for (int s = 1; s < 32; s <<= 1) {
        const int v = __shfl_up_sync(0xffffffffu, incl, s);
        if (lane >= s) incl += v;
      }
      int off = base + incl - cnt;
      while (word) {
        const int b = __ffs(word) - 1;
        const int k = (w0 + lane) * 32 + b;
        if (k < a.K) s_col[off++] = (short)k;
        word &= word - 1;
      }
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) s_misc[0] = base < a.K ? base : a.K;
  }
  if (tid < kTN) s_cnt[tid] = 0u;
  if (tid == 0) s_blk = 0u;
  __syncthreads();
  const int nocc = s_misc[0];
  // where each K window starts in the (sorted) occupied list: binary search
  if (tid <= nwin) {
    const int bound = tid * kKW;
    int lo = 0, hi = nocc;
    while (lo < hi) {
      const int mid = (lo + hi) >> 1;
      if (s_col[mid] < bound) lo = mid + 1;
      else hi = mid;
    }
    s_misc[1 + tid] = lo;
  }
  __syncthreads();

  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  for (int win = 0; win < nwin; ++win) {
    const int k0 = win * kKW;
    const int kw = a.K - k0 < kKW ? a.K - k0 : kKW;
    const int oc = s_misc[1 + win];
    const int nk = s_misc[2 + win] - oc;  // occupied columns of this window
    if (win > 0 && nk > 0) stage_x(xs_u32, a, m0, k0, kw, tid);
    if (nk > 0) {
      // 2a. W rows of the window's occupied columns, columns n0 .. n0 + 16 (bf16)
      for (int idx = tid; idx < nk * (kTN / 8); idx += kThreads) {
        const int kk = idx >> 1, h = idx & 1;
        const int n = n0 + h * 8;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (n + 8 <= a.N) v = __ldg(reinterpret_cast<const uint4*>(a.w_kn + (int64_t)s_col[oc + kk] * a.N + n));
        *reinterpret_cast<uint4*>(wsb + kk * kTN + h * 8) = v;
      }
    }
    cp_async_wait<0>();
    __syncthreads();
    if (nk > 0) {
      // 2b. this slice's occupied columns: 4 rows x 4 columns per column
      const __nv_bfloat16* xr = xs + rg * kPitch - k0;
#pragma unroll 4
      for (int kk = sl; kk < nk; kk += kSlices) {
        const int col = s_col[oc + kk];
        const uint2 wv = *reinterpret_cast<const uint2*>(wsb + kk * kTN + cg * 4);
        const float2 w01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wv.x));
        const float2 w23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wv.y));
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float xv = __bfloat162float(xr[i * 16 * kPitch + col]);
          acc[i][0] = fmaf(xv, w01.x, acc[i][0]);
          acc[i][1] = fmaf(xv, w01.y, acc[i][1]);
          acc[i][2] = fmaf(xv, w23.x, acc[i][2]);
          acc[i][3] = fmaf(xv, w23.y, acc[i][3]);
        }
      }
    }
    __syncthreads();  // window buffers free for the next window
  }
  // 2c. the slices' sums meet in shared memory (the W buffer is free now)
#pragma unroll
  for (int i = 0; i < 4; ++i)
    *reinterpret_cast<float4*>(red + ((sl * kTM) + rg + 16 * i) * kTN + cg * 4) =
        make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
  __syncthreads();
  float sum4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int s2 = 0; s2 < kSlices; ++s2) {
    const float4 v = *reinterpret_cast<const float4*>(red + ((s2 * kTM) + row) * kTN + cq * 4);
    sum4[0] += v.x;
    sum4[1] += v.y;
    sum4[2] += v.z;
    sum4[3] += v.w;
  }

  // 3. epilogue
  uint32_t bits = 0u;
  if (m < a.M) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + cq * 4 + j;
      if (n >= a.N) continue;
      float scv = 1.f, shv = 0.f;
      epi_affine(a.ep, a.N, n, scv, shv);
      float v = fmaf(sum4[j], scv, shv);
      if (a.ep.residual) v += __bfloat162float(a.ep.residual[m * a.N + n]);
      v = epi_act(v, a.ep.act);
      if (a.y_f32) {
        reinterpret_cast<float*>(a.y)[m * a.N + n] = v;
      } else {
        const __nv_bfloat16 o = __float2bfloat16_rn(v);
        reinterpret_cast<__nv_bfloat16*>(a.y)[m * a.N + n] = o;
        if (bf16_nz(__bfloat16_as_ushort(o))) bits |= 1u << j;
      }
    }
  }
  if (a.emit) {
    const OccDev o = a.out_occ;
    // the row's 16 columns: 4 lanes (cq) per row
    uint32_t rb16 = bits << (cq * 4);
    rb16 |= __shfl_xor_sync(0xffffffffu, rb16, 1);
    rb16 |= __shfl_xor_sync(0xffffffffu, rb16, 2);
    if (cq == 0 && rb16 && m < a.M)
      atomicOr(&o.row_bm[m * o.W64 + (n0 >> 12)], 1ull << ((n0 >> 6) & 63));
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if ((bits >> j) & 1u) atomicAdd(&s_cnt[cq * 4 + j], 1u);
    // block mask: the 16 columns' bits over the CTA's rows (one 128-row block)
    const uint32_t wbits = __reduce_or_sync(0xffffffffu, rb16);
    if (lane == 0 && wbits) atomicOr(&s_blk, wbits);
    __syncthreads();
    if (tid < kTN) {
      const uint32_t c = s_cnt[tid];
      const int n = n0 + tid;
      if (c && n < a.N) atomicAdd(&o.col_nnz[n], c);
    }
    if (tid == 0) {
      uint32_t sum = 0u;
      for (int j = 0; j < kTN; ++j) sum += s_cnt[j];
      const int w = n0 >> 5;
      if (s_blk && w < o.C32) atomicOr(&o.blk_mask[(m0 >> 7) * o.C32 + w], s_blk << (n0 & 31));
      if (sum) {
        atomicAdd(&o.tile_nnz[n0 >> 6], sum);
        atomicAdd(o.nnz, (unsigned long long)sum);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Fused small FC: statistics, dispatch and the zero-skip product in one launch
// ---------------------------------------------------------------------------
// For inputs small enough to sit in shared memory whole (M <= 128 rows,
// M * (K + 8) * 2 bytes within kSmallXBytes) every CTA loads x once and
// derives from it what the separate statistics kernel would: the Eq. 1
// non-zero count (Sec. 3.1) and which columns hold a non-zero.  All CTAs reach
// the same decision (Sec. 3 rule); on the zero-skip path each CTA multiplies
// the occupied columns of x by the matching rows of W_kn for its 16 output
// columns on the tensor cores (mma.sync m16n8k16, fp32 accumulation), the
// columns compacted into dense k-steps of 16 (Sec. 2.1: zero activations
// take no part); on the dense path every column takes part.  A 128-row
// tcgen05 tile would be mostly empty at these sizes, so both paths of a
// small FC run here, in one launch.  CTA 0 writes the count and the path
// for the host record.
constexpr int kSmallTN = 16;
constexpr size_t kSmallXBytes = 160 * 1024;

__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

constexpr int kSmallThreads = 1024;  // 32 warps: short dependency chains per warp
constexpr int kSmallWarps = kSmallThreads / 32;

struct SmallGeo {
  int xpitch;   // bf16 elements per staged x row: K + 8 (column K stays zero)
  int mp8;      // rows staged: M rounded up to 8 (the extra rows zero)
  int kc;       // compacted K bound: K rounded up to 16
  size_t x_off, any_off, w_off, red_off, col_off, misc_off, bytes;
};

__host__ __device__ inline SmallGeo small_geo(int M, int K) {
  SmallGeo g;
  g.xpitch = K + 8;
  g.mp8 = (M + 7) / 8 * 8;
  g.kc = (K + 15) / 16 * 16;
  g.x_off = 0;
  g.any_off = ((size_t)g.mp8 * g.xpitch * 2 + 15) / 16 * 16;          // [K / 2] u32: pair occupancy
  g.w_off = (g.any_off + (size_t)(K / 2) * 4 + 15) / 16 * 16;        // [kc][16] bf16: W rows taken
  g.red_off = g.w_off + (size_t)g.kc * kSmallTN * 2;                 // [32][16][16] fp32 partial sums
  g.col_off = g.red_off + (size_t)kSmallWarps * 16 * kSmallTN * 4;   // [kc] columns taken
  g.misc_off = (g.col_off + (size_t)g.kc * 2 + 15) / 16 * 16;
  g.bytes = g.misc_off + 256;  // count, path, per-warp counts [32], per-column output counts [16]
  return g;
}

__global__ void __launch_bounds__(kSmallThreads) fcsmall_kernel(const FcSkipArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int M = a.M, K = a.K, N = a.N;
  const SmallGeo G = small_geo(M, K);
  __nv_bfloat16* xs = reinterpret_cast<__nv_bfloat16*>(smem + G.x_off);
  uint32_t* s_any = reinterpret_cast<uint32_t*>(smem + G.any_off);
  __nv_bfloat16* wc = reinterpret_cast<__nv_bfloat16*>(smem + G.w_off);
  float* red = reinterpret_cast<float*>(smem + G.red_off);
  short* s_col = reinterpret_cast<short*>(smem + G.col_off);
  uint32_t* s_cnt32 = reinterpret_cast<uint32_t*>(smem + G.misc_off);  // x's non-zeros
  int* s_path = reinterpret_cast<int*>(smem + G.misc_off + 8);
  int* s_wsum = reinterpret_cast<int*>(smem + G.misc_off + 16);     // [32]
  uint32_t* s_cnt = reinterpret_cast<uint32_t*>(smem + G.misc_off + 144);  // [16]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n0 = blockIdx.x * kSmallTN;
  const int KP = K / 2;  // column pairs

  for (int i = tid; i < KP; i += kSmallThreads) s_any[i] = 0u;
  if (tid == 0) *s_cnt32 = 0u;
  if (tid < kSmallTN) s_cnt[tid] = 0u;
  pdl_wait();
  pdl_trigger();
  // the epilogue's column affine, fetched now: thread t < 4 Mp takes row
  // t / 4 and the four columns n0 + 4 (t % 4) ..
  float e_sc[4], e_sh[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int n = n0 + (tid & 3) * 4 + j;
    e_sc[j] = 1.f;
    e_sh[j] = 0.f;
    if (n < N) epi_affine(a.ep, N, n, e_sc[j], e_sh[j]);
  }
  // 1. x whole into shared memory (16-byte copies, all in flight); rows
  //    M .. mp8 - 1 and column K zero
  const uint32_t xs_u32 = smem_u32(xs);
  const int chunks = K / 8;
  for (int idx = tid; idx < M * chunks; idx += kSmallThreads) {
    const int r = idx / chunks, c = idx - (idx / chunks) * chunks;
    cp_async_16(xs_u32 + (uint32_t)((r * G.xpitch + c * 8) * 2), a.x + (int64_t)r * K + c * 8, 16u);
  }
  cp_async_commit();
  for (int idx = tid; idx < (G.mp8 - M) * (chunks + 1); idx += kSmallThreads) {
    const int r = M + idx / (chunks + 1), c = idx - (idx / (chunks + 1)) * (chunks + 1);
    *reinterpret_cast<uint4*>(xs + r * G.xpitch + c * 8) = make_uint4(0u, 0u, 0u, 0u);
  }
  for (int r = tid; r < M; r += kSmallThreads)
    *reinterpret_cast<uint4*>(xs + r * G.xpitch + K) = make_uint4(0u, 0u, 0u, 0u);
  cp_async_wait<0>();
  __syncthreads();

  // 2. Eq. 1 count and occupied column pairs: unit = (pair, 8 rows); the
  //    non-zero bits of a bf16 pair land on bits 15 / 31
  const uint32_t* x32 = reinterpret_cast<const uint32_t*>(xs);
  const int pitch32 = G.xpitch / 2;
  uint32_t cnt = 0u;
  const int units = KP * (G.mp8 / 8);
  for (int u = tid; u < units; u += kSmallThreads) {
    const int oct = u / KP, cp = u - oct * KP;
    const uint32_t* col = x32 + oct * 8 * pitch32 + cp;
    uint32_t wv[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) wv[i] = col[i * pitch32];
    uint32_t any = 0u;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const uint32_t t = ((wv[i] & 0x7FFF7FFFu) + 0x7FFF7FFFu) & 0x80008000u;
      any |= t;
      cnt += __popc(t);
    }
    if (any) atomicOr(&s_any[cp], any);
  }
#pragma unroll
  for (int sft = 16; sft > 0; sft >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, sft);
  if (lane == 0 && cnt) atomicAdd(s_cnt32, cnt);  // M * K < 2^31: a 32-bit count
  __syncthreads();

  // 3. the rule (every CTA reaches the same decision)
  const unsigned long long nnz = *s_cnt32;
  if (tid == 0) {
    int path;
    if (a.disp.force == 1) path = 1;
    else if (a.disp.force == 2) path = 2;
    else {
      const double numel = (double)((unsigned long long)M * (unsigned long long)K);
      const double zeros = numel - (double)nnz;
      path = zeros >= __dmul_rn(a.disp.s_thr, numel) ? 2 : (a.disp.fpb_ok ? 1 : 2);
    }
    *s_path = path;
    if (blockIdx.x == 0) {
      if (a.nnz_out) *a.nnz_out = nnz;
      if (a.disp.path_out) *a.disp.path_out = path;
    }
  }
  __syncthreads();
  const int path = *s_path;

  // 4. the columns that take part, in increasing order: every column on the
  //    dense path; on the zero-skip path the occupied ones, numbered from the
  //    warps' ballots and a prefix over the warps, a pass of 1024 pairs at a
  //    time
  int nocc = 0;
  if (path == 2) {
    for (int pass0 = 0; pass0 < KP; pass0 += kSmallThreads) {
      const int cp = pass0 + tid;
      const uint32_t any = cp < KP ? s_any[cp] : 0u;
      const bool f_lo = (any >> 15) & 1u, f_hi = any >> 31;
      const uint32_t b_lo = __ballot_sync(0xffffffffu, f_lo), b_hi = __ballot_sync(0xffffffffu, f_hi);
      const uint32_t lt = (1u << lane) - 1u;
      if (lane == 0) s_wsum[warp] = __popc(b_lo) + __popc(b_hi);
      __syncthreads();
      // exclusive prefix of the 32 warps' counts: one load per lane, a scan
      // by shuffles
      const int wv = s_wsum[lane];
      int incl = wv;
#pragma unroll
      for (int sft = 1; sft < 32; sft <<= 1) {
        const int t2 = __shfl_up_sync(0xffffffffu, incl, sft);
        if (lane >= sft) incl += t2;
      }
      const int total = __shfl_sync(0xffffffffu, incl, 31);
      int off = nocc + __shfl_sync(0xffffffffu, incl - wv, warp) + __popc(b_lo & lt) + __popc(b_hi & lt);
      if (f_lo) s_col[off++] = (short)(2 * cp);
      if (f_hi) s_col[off] = (short)(2 * cp + 1);
      nocc += total;
      __syncthreads();  // s_wsum is reused by the next pass
    }
  } else {
    for (int k = tid; k < K; k += kSmallThreads) s_col[k] = (short)k;
    nocc = K;
  }
  const int kc = (nocc + 15) / 16 * 16;
  for (int k = nocc + tid; k < kc; k += kSmallThreads) s_col[k] = (short)K;  // the zero column
  __syncthreads();
  // W rows of the columns taken: W_kn[col][n0 .. n0 + 16), zero for the padding
  for (int idx = tid; idx < kc * 2; idx += kSmallThreads) {
    const int kk = idx >> 1, h = idx & 1;
    const int col = s_col[kk];
    uint4 v = make_uint4(0u, 0u, 0u, 0u);
    if (col < K && n0 + h * 8 + 8 <= N) v = __ldg(reinterpret_cast<const uint4*>(a.w_kn + (int64_t)col * N + n0 + h * 8));
    *reinterpret_cast<uint4*>(wc + kk * kSmallTN + h * 8) = v;
  }
  __syncthreads();

  // 5. tensor-core product over the k-steps of 16 taken columns: warp w takes
  //    row group w % RG (16 rows) and every KS-th k-step from w / RG
  const int RG = (M + 15) / 16;
  const int KS = kSmallWarps / RG;
  const int rg = warp % RG, ks0 = warp / RG;
  const int g = lane >> 2, tq = lane & 3;
  const int Mp = RG * 16;
  if (ks0 < KS) {
    float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
    const int r0 = rg * 16 + g, r1 = r0 + 8;
    const bool v0 = r0 < M, v1 = r1 < M;
    const __nv_bfloat16* xr0 = xs + (v0 ? r0 : 0) * G.xpitch;
    const __nv_bfloat16* xr1 = xs + (v1 ? r1 : 0) * G.xpitch;
    const uint32_t w_lane = smem_u32(wc) + (uint32_t)(((lane & 15) * kSmallTN + (lane >> 4) * 8) * 2);
    for (int k0 = ks0 * 16; k0 < kc; k0 += KS * 16) {
      const uint32_t p01 = *reinterpret_cast<const uint32_t*>(s_col + k0 + 2 * tq);
      const uint32_t p23 = *reinterpret_cast<const uint32_t*>(s_col + k0 + 2 * tq + 8);
      const int c0 = (int)(p01 & 0xFFFFu), c1 = (int)(p01 >> 16);
      const int c2 = (int)(p23 & 0xFFFFu), c3 = (int)(p23 >> 16);
      uint32_t af[4];
      af[0] = v0 ? ((uint32_t)__bfloat16_as_ushort(xr0[c0]) | ((uint32_t)__bfloat16_as_ushort(xr0[c1]) << 16)) : 0u;
      af[1] = v1 ? ((uint32_t)__bfloat16_as_ushort(xr1[c0]) | ((uint32_t)__bfloat16_as_ushort(xr1[c1]) << 16)) : 0u;
      af[2] = v0 ? ((uint32_t)__bfloat16_as_ushort(xr0[c2]) | ((uint32_t)__bfloat16_as_ushort(xr0[c3]) << 16)) : 0u;
      af[3] = v1 ? ((uint32_t)__bfloat16_as_ushort(xr1[c2]) | ((uint32_t)__bfloat16_as_ushort(xr1[c3]) << 16)) : 0u;
      uint32_t b0, b1, b2, b3;
      ldsm_x4_t(w_lane + (uint32_t)(k0 * kSmallTN * 2), b0, b1, b2, b3);
      mma_16816(acc[0], af, b0, b1);
      mma_16816(acc[1], af, b2, b3);
    }
    // partial sums of this k-step group: red[ks][row][16]
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      float* rb = red + ((size_t)ks0 * Mp + rg * 16) * kSmallTN + j * 8 + 2 * tq;
      rb[g * kSmallTN] = acc[j][0];
      rb[g * kSmallTN + 1] = acc[j][1];
      rb[(g + 8) * kSmallTN] = acc[j][2];
      rb[(g + 8) * kSmallTN + 1] = acc[j][3];
    }
  }
  __syncthreads();

  // 6. epilogue: thread t < 4 Mp = (row t / 4, columns n0 + 4 (t % 4) ..)
  const OccDev o = a.out_occ;
  if (tid < Mp * 4) {
    const int row = tid >> 2, cq = tid & 3;
    const int64_t m = row;
    float v4[4] = {0.f, 0.f, 0.f, 0.f};
    for (int k2 = 0; k2 < KS; ++k2) {
      const float4 pv = *reinterpret_cast<const float4*>(red + ((size_t)k2 * Mp + row) * kSmallTN + cq * 4);
      v4[0] += pv.x;
      v4[1] += pv.y;
      v4[2] += pv.z;
      v4[3] += pv.w;
    }
    uint32_t bits = 0u;
    if (row < M) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int n = n0 + cq * 4 + j;
        if (n >= N) continue;
        float v = fmaf(v4[j], e_sc[j], e_sh[j]);
        if (a.ep.residual) v += __bfloat162float(a.ep.residual[m * N + n]);
        v = epi_act(v, a.ep.act);
        if (a.y_f32) {
          reinterpret_cast<float*>(a.y)[m * N + n] = v;
        } else {
          const __nv_bfloat16 ob = __float2bfloat16_rn(v);
          reinterpret_cast<__nv_bfloat16*>(a.y)[m * N + n] = ob;
          if (bf16_nz(__bfloat16_as_ushort(ob))) bits |= 1u << j;
        }
      }
    }
    if (a.emit) {
      // the row's 16 columns are held by 4 consecutive threads (one warp)
      uint32_t rb16 = bits << (cq * 4);
      rb16 |= __shfl_xor_sync(0xffffffffu, rb16, 1);
      rb16 |= __shfl_xor_sync(0xffffffffu, rb16, 2);
      if (cq == 0 && rb16 && row < M) atomicOr(&o.row_bm[m * o.W64 + (n0 >> 12)], 1ull << ((n0 >> 6) & 63));
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if ((bits >> j) & 1u) atomicAdd(&s_cnt[cq * 4 + j], 1u);
      const uint32_t wbits = __reduce_or_sync(0xffffffffu, rb16);
      const int w = n0 >> 5;
      if (lane == 0 && wbits && w < o.C32) atomicOr(&o.blk_mask[w], wbits << (n0 & 31));
    }
  }
  if (a.emit) {
    __syncthreads();
    if (tid < kSmallTN) {
      const uint32_t c = s_cnt[tid];
      const int n = n0 + tid;
      if (c && n < N) atomicAdd(&o.col_nnz[n], c);
    }
    if (tid == 0) {
      uint32_t sum = 0u;
      for (int j = 0; j < kSmallTN; ++j) sum += s_cnt[j];
      if (sum) {
        atomicAdd(&o.tile_nnz[n0 >> 6], sum);
        atomicAdd(o.nnz, (unsigned long long)sum);
      }
    }
  }
}

}  // namespace

cudaError_t launch_fcskip(const FcSkipArgs& a, cudaStream_t s) {
  if (a.M <= 0 || a.N <= 0) return cudaSuccess;
  if (a.K % 8 != 0 || a.N % 8 != 0 || a.K > kMaxWin * kKW) return cudaErrorInvalidValue;
  const size_t smem = FcSmem::kBytes + (size_t)a.K * sizeof(short);
  // opt in above the 48 KB default, which also counts the static shared memory
  if (smem > 40 * 1024) {
    cudaError_t e = smem_optin(reinterpret_cast<const void*>(fcskip_kernel), smem);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((a.N + kTN - 1) / kTN, (a.M + kTM - 1) / kTM);
  return launch_kernel(fcskip_kernel, grid, dim3(kThreads), smem, s, a);
}

bool fcsmall_supported(int M, int K, int N) {
  return M > 0 && M <= 128 && K % 8 == 0 && N % 8 == 0 && K < 32760 &&
         (size_t)M * (K + 8) * 2 <= kSmallXBytes && small_geo(M, K).bytes <= 220 * 1024;
}

cudaError_t launch_fcsmall(const FcSkipArgs& a, cudaStream_t s) {
  if (a.M <= 0 || a.N <= 0) return cudaSuccess;
  if (!fcsmall_supported(a.M, a.K, a.N)) return cudaErrorInvalidValue;
  const size_t smem = small_geo(a.M, a.K).bytes;
  if (smem > 40 * 1024) {
    cudaError_t e = smem_optin(reinterpret_cast<const void*>(fcsmall_kernel), smem);
    if (e != cudaSuccess) return e;
  }
  dim3 grid((a.N + kSmallTN - 1) / kSmallTN);
  return launch_kernel(fcsmall_kernel, grid, dim3(kSmallThreads), smem, s, a);
}

}  // namespace sparoa
