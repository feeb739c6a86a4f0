// Column-compacting zero-skip fully connected kernel for few rows.
//
// y[M, N] = epilogue(x[M, K] * W[N, K]^T) where, per 128-row block of x, only
// the columns k that hold a non-zero in that block take part (Sec. 2.1:
// products with a zero activation are skipped without changing the output).
// The block-column mask of x (one bit per column per 128-row block) gives the
// occupied columns; the kernel compacts them into a list, gathers those
// columns of x and the matching rows of W stored as [K, N] (each a contiguous
// run of N values, so skipped columns cost no HBM traffic), and accumulates in
// fp32 on the CUDA cores.  This is the path for small-M layers (a batch of
// feature vectors), which are bound by the weight bytes, not by arithmetic.
//
// CTA = 128 rows x 64 output columns, 256 threads, each owning 8 x 4 outputs.
#include "sparoa_kernels.h"

namespace sparoa {

namespace {

constexpr int kThreads = 256;
constexpr int kKC = 32;   // compacted columns per chunk

__global__ void __launch_bounds__(kThreads) fcskip_kernel(const FcSkipArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  float* xs = reinterpret_cast<float*>(smem);               // [kKC][128]
  float* ws = xs + kKC * 128;                               // [kKC][64]
  uint64_t* s_nz = reinterpret_cast<uint64_t*>(ws + kKC * 64);  // [128]
  int* s_cnt = reinterpret_cast<int*>(s_nz + 128);
  int* cols = s_cnt + 4;                                    // [K]

  pdl_wait();
  pdl_trigger();
  const int path = decide_path(a.disp);
  if (path != 2) return;  // the dense kernel of this launch runs instead
  record_path(a.disp, path);

  const int n0 = blockIdx.x * 64;
  const int64_t m0 = (int64_t)blockIdx.y * 128;
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;

  // 1. occupied columns of this row block, in increasing order
  if (warp == 0) {
    int base = 0;
    for (int w0 = 0; w0 < a.in_C32; w0 += 32) {
      uint32_t word = (w0 + lane < a.in_C32) ? a.in_blk[blockIdx.y * a.in_C32 + w0 + lane] : 0u;
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
        cols[off++] = (w0 + lane) * 32 + b;
        word &= word - 1;
      }
      base += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) *s_cnt = base;
  }
  if (tid < 128) s_nz[tid] = 0ull;
  __syncthreads();
  const int kc_total = *s_cnt;

  const int rg = tid >> 4;   // rows rg*8 .. +8
  const int cq = tid & 15;   // cols cq*4 .. +4
  float acc[8][4];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;

  for (int kc = 0; kc < kc_total; kc += kKC) {
    // 2a. gather x[m0 + row, cols[kc + k]] -> xs[k][row]
    {
      const int row = tid >> 1, half = tid & 1;
      const int64_t m = m0 + row;
#pragma unroll 4
      for (int j = 0; j < 16; ++j) {
        const int k = kc + half * 16 + j;
        float v = 0.f;
        if (k < kc_total && m < a.M) v = __bfloat162float(a.x[m * a.K + cols[k]]);
        xs[(half * 16 + j) * 128 + row] = v;
      }
    }
    // 2b. W_kn[cols[kc + kr], n0 .. n0+64) -> ws[kr][*]
    {
      const int kr = tid >> 3, cg = tid & 7;
      const int k = kc + kr;
      const int n = n0 + cg * 8;
      float f[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      if (k < kc_total && n < a.N) {
        const uint4 u = __ldg(reinterpret_cast<const uint4*>(a.w_kn + (int64_t)cols[k] * a.N + n));
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const float2 t = __bfloat1622float2(h[j]);
          f[2 * j] = t.x;
          f[2 * j + 1] = t.y;
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) ws[kr * 64 + cg * 8 + j] = f[j];
    }
    __syncthreads();
    // 2c. accumulate
#pragma unroll 8
    for (int k = 0; k < kKC; ++k) {
      const float4 a0 = *reinterpret_cast<const float4*>(&xs[k * 128 + rg * 8]);
      const float4 a1 = *reinterpret_cast<const float4*>(&xs[k * 128 + rg * 8 + 4]);
      const float4 b = *reinterpret_cast<const float4*>(&ws[k * 64 + cq * 4]);
      const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      const float bv[4] = {b.x, b.y, b.z, b.w};
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }

  // 3. epilogue
  float sc[4], sh[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    sc[j] = 1.f;
    sh[j] = 0.f;
    const int n = n0 + cq * 4 + j;
    if (n < a.N) epi_affine(a.ep, a.N, n, sc[j], sh[j]);
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int row = rg * 8 + i;
    const int64_t m = m0 + row;
    if (m >= a.M) continue;
    uint32_t bits = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + cq * 4 + j;
      if (n >= a.N) continue;
      float v = fmaf(acc[i][j], sc[j], sh[j]);
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
    if (a.emit && bits) atomicOr(reinterpret_cast<unsigned long long*>(&s_nz[row]),
                                 (unsigned long long)bits << (cq * 4));
  }
  if (a.emit) {
    __syncthreads();
    flush_tile(s_nz, m0, n0, a.out_occ, tid, kThreads);
  }
}

}  // namespace

cudaError_t launch_fcskip(const FcSkipArgs& a, cudaStream_t s) {
  if (a.M <= 0 || a.N <= 0) return cudaSuccess;
  const size_t smem = (size_t)kKC * 128 * 4 + (size_t)kKC * 64 * 4 + 128 * 8 + 16 + (size_t)a.K * 4;
  static size_t attr = 0;
  if (smem > 48 * 1024 && smem > attr) {
    cudaError_t e = cudaFuncSetAttribute(fcskip_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    attr = smem;
  }
  dim3 grid((a.N + 63) / 64, (a.M + 127) / 128);
  return launch_kernel(fcskip_kernel, grid, dim3(kThreads), smem, s, a);
}

}  // namespace sparoa
