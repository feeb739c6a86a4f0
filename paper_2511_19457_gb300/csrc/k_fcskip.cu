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

}  // namespace sparoa
