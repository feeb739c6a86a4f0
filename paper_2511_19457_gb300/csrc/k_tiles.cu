// Memory-bound kernels of the path, all on the same 128-row x 64-channel tile:
// 256 threads, thread t owns channels [8*(t%8), 8*(t%8)+8) of the tile (one
// 16-byte vector) in rows t/8 + 32*i, i = 0..3.  Each kernel fuses the
// occupancy emission of its output (Eq. 1 count and bitmaps, Sec. 3.1) so the
// next operator's dispatch reads them without another pass over HBM.
//   stats_kernel    Eq. 1 count and bitmaps of an existing tensor
//   dwconv_kernel   depthwise k x k convolution + epilogue (MobileNetV2 layers)
//   maxpool_kernel  k x k max pooling
//   avgpool_kernel  global average pooling
//   bn_act_kernel   stand-alone bias / batch norm / residual / activation
#include "sparoa_kernels.h"

namespace sparoa {

namespace {

constexpr int kTileThreads = 256;

__device__ __forceinline__ void unpack8(const uint4& u, float (&f)[8]) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 t = __bfloat1622float2(h[j]);
    f[2 * j] = t.x;
    f[2 * j + 1] = t.y;
  }
}

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

// Pack 8 floats to bf16 (round to nearest even); returns the vector.
__device__ __forceinline__ uint4 pack8(const float (&f)[8]) {
  uint4 u;
  uint32_t* w = reinterpret_cast<uint32_t*>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(f[2 * j]));
    const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(f[2 * j + 1]));
    w[j] = lo | (hi << 16);
  }
  return u;
}

// Combine the 8-bit masks of the 8 lanes that share a row into the row's
// 64-bit tile word and store it (lane with t%8 == 0).
__device__ __forceinline__ void put_row_bits(uint64_t* s_nz, int row, uint32_t mask8) {
  const int cg = threadIdx.x & 7;
  uint32_t lo = cg < 4 ? (mask8 << (8 * cg)) : 0u;
  uint32_t hi = cg >= 4 ? (mask8 << (8 * (cg - 4))) : 0u;
#pragma unroll
  for (int s = 1; s < 8; s <<= 1) {
    lo |= __shfl_xor_sync(0xffffffffu, lo, s);
    hi |= __shfl_xor_sync(0xffffffffu, hi, s);
  }
  if (cg == 0) s_nz[row] = (uint64_t)lo | ((uint64_t)hi << 32);
}

__device__ __forceinline__ void zero_rows(uint64_t* s_nz) {
  if (threadIdx.x < 128) s_nz[threadIdx.x] = 0ull;
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kTileThreads) stats_kernel(const __nv_bfloat16* __restrict__ x,
                                                             int64_t R, int C, OccDev o) {
  __shared__ uint64_t s_nz[128];
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int64_t row0 = (int64_t)blockIdx.x * 128;
  const int c0 = blockIdx.y * 64 + cg * 8;
  const bool vec = (C & 7) == 0;
  uint32_t m[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t r = row0 + rs + 32 * i;
    m[i] = 0;
    if (r < R && c0 < C) {
      const __nv_bfloat16* p = x + r * C + c0;
      if (vec) {
        m[i] = nz_mask8(__ldg(reinterpret_cast<const uint4*>(p)));
      } else {
        for (int j = 0; j < 8 && c0 + j < C; ++j)
          if (bf16_nz(__bfloat16_as_ushort(p[j]))) m[i] |= 1u << j;
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) put_row_bits(s_nz, rs + 32 * i, m[i]);
  __syncthreads();
  flush_tile(s_nz, row0, blockIdx.y * 64, o, threadIdx.x, kTileThreads);
}

// ---------------------------------------------------------------------------
__global__ void pad_kernel(const __nv_bfloat16* __restrict__ x, int64_t P, int C, int Cp,
                           __nv_bfloat16* __restrict__ y) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= P * Cp) return;
  const int64_t p = i / Cp;
  const int c = (int)(i - p * Cp);
  y[i] = c < C ? x[p * C + c] : __float2bfloat16_rn(0.f);
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kTileThreads) dwconv_kernel(const DwArgs a) {
  __shared__ uint64_t s_nz[128];
  zero_rows(s_nz);
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int64_t row0 = (int64_t)blockIdx.x * 128;
  const int c0 = blockIdx.y * 64 + cg * 8;
  const int64_t R = (int64_t)a.N * a.Ho * a.Wo;
  const int taps = a.kh * a.kw;
  if (a.path_out && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) *a.path_out = 3;
  __syncthreads();
  const bool cvalid = c0 < a.C;
  float wr[9][8];
  float sc[8], sh[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    sc[j] = 1.f;
    sh[j] = 0.f;
    if (cvalid) epi_affine(a.ep, a.C, c0 + j, sc[j], sh[j]);
#pragma unroll
    for (int t = 0; t < 9; ++t)
      wr[t][j] = (cvalid && t < taps) ? __bfloat162float(a.w[(int64_t)(c0 + j) * taps + t]) : 0.f;
  }
  for (int i = 0; i < 4; ++i) {
    const int row = rs + 32 * i;
    const int64_t mrow = row0 + row;
    uint32_t mask = 0;
    if (cvalid && mrow < R) {
      const int hw = a.Ho * a.Wo;
      const int img = (int)(mrow / hw);
      const int rem = (int)(mrow - (int64_t)img * hw);
      const int oh = rem / a.Wo, ow = rem - (rem / a.Wo) * a.Wo;
      float acc[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = 0.f;
      for (int r = 0; r < a.kh; ++r) {
        const int ih = oh * a.stride - a.pad + r;
        if (ih < 0 || ih >= a.H) continue;
        for (int s = 0; s < a.kw; ++s) {
          const int iw = ow * a.stride - a.pad + s;
          if (iw < 0 || iw >= a.W) continue;
          const uint4 u = __ldg(reinterpret_cast<const uint4*>(
              a.x + (((int64_t)img * a.H + ih) * a.W + iw) * a.C + c0));
          float f[8];
          unpack8(u, f);
          const int t = r * a.kw + s;
#pragma unroll
          for (int j = 0; j < 8; ++j) acc[j] = fmaf(f[j], wr[t][j], acc[j]);
        }
      }
      float rv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      if (a.ep.residual) unpack8(*reinterpret_cast<const uint4*>(a.ep.residual + mrow * a.C + c0), rv);
      float o[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) o[j] = epi_act(fmaf(acc[j], sc[j], sh[j]) + rv[j], a.ep.act);
      const uint4 u = pack8(o);
      *reinterpret_cast<uint4*>(a.y + mrow * a.C + c0) = u;
      mask = nz_mask8(u);
    }
    if (a.emit) put_row_bits(s_nz, row, mask);
  }
  if (a.emit) {
    __syncthreads();
    flush_tile(s_nz, row0, blockIdx.y * 64, a.out_occ, threadIdx.x, kTileThreads);
  }
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kTileThreads)
    maxpool_kernel(const __nv_bfloat16* __restrict__ x, int N, int H, int W, int C, int k,
                   int stride, int pad, int Ho, int Wo, __nv_bfloat16* __restrict__ y, OccDev o,
                   int emit) {
  __shared__ uint64_t s_nz[128];
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int64_t row0 = (int64_t)blockIdx.x * 128;
  const int c0 = blockIdx.y * 64 + cg * 8;
  const int64_t R = (int64_t)N * Ho * Wo;
  for (int i = 0; i < 4; ++i) {
    const int row = rs + 32 * i;
    const int64_t mrow = row0 + row;
    uint32_t mask = 0;
    if (mrow < R && c0 < C) {
      const int hw = Ho * Wo;
      const int img = (int)(mrow / hw);
      const int rem = (int)(mrow - (int64_t)img * hw);
      const int oh = rem / Wo, ow = rem - (rem / Wo) * Wo;
      float mx[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) mx[j] = -INFINITY;
      for (int r = 0; r < k; ++r) {
        const int ih = oh * stride - pad + r;
        if (ih < 0 || ih >= H) continue;
        for (int s = 0; s < k; ++s) {
          const int iw = ow * stride - pad + s;
          if (iw < 0 || iw >= W) continue;
          float f[8];
          unpack8(__ldg(reinterpret_cast<const uint4*>(x + (((int64_t)img * H + ih) * W + iw) * C + c0)), f);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            if (f[j] > mx[j]) mx[j] = f[j];
        }
      }
      const uint4 u = pack8(mx);
      *reinterpret_cast<uint4*>(y + mrow * C + c0) = u;
      mask = nz_mask8(u);
    }
    if (emit) put_row_bits(s_nz, row, mask);
  }
  if (emit) {
    __syncthreads();
    flush_tile(s_nz, row0, blockIdx.y * 64, o, threadIdx.x, kTileThreads);
  }
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kTileThreads)
    avgpool_kernel(const __nv_bfloat16* __restrict__ x, int N, int HW, int C,
                   __nv_bfloat16* __restrict__ y, OccDev o, int emit) {
  __shared__ uint64_t s_nz[128];
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int64_t row0 = (int64_t)blockIdx.x * 128;
  const int c0 = blockIdx.y * 64 + cg * 8;
  for (int i = 0; i < 4; ++i) {
    const int row = rs + 32 * i;
    const int64_t n = row0 + row;
    uint32_t mask = 0;
    if (n < N && c0 < C) {
      float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      const __nv_bfloat16* p = x + n * (int64_t)HW * C + c0;
      for (int q = 0; q < HW; ++q) {
        float f[8];
        unpack8(__ldg(reinterpret_cast<const uint4*>(p + (int64_t)q * C)), f);
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] += f[j];
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = acc[j] / (float)HW;
      const uint4 u = pack8(acc);
      *reinterpret_cast<uint4*>(y + n * C + c0) = u;
      mask = nz_mask8(u);
    }
    if (emit) put_row_bits(s_nz, row, mask);
  }
  if (emit) {
    __syncthreads();
    flush_tile(s_nz, row0, blockIdx.y * 64, o, threadIdx.x, kTileThreads);
  }
}

// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kTileThreads)
    bn_act_kernel(const __nv_bfloat16* __restrict__ x, int64_t R, int C, EpiDev ep,
                  __nv_bfloat16* __restrict__ y, OccDev o, int emit) {
  __shared__ uint64_t s_nz[128];
  const int cg = threadIdx.x & 7, rs = threadIdx.x >> 3;
  const int64_t row0 = (int64_t)blockIdx.x * 128;
  const int c0 = blockIdx.y * 64 + cg * 8;
  float sc[8], sh[8];
  if (c0 < C) {
#pragma unroll
    for (int j = 0; j < 8; ++j) epi_affine(ep, C, c0 + j, sc[j], sh[j]);
  }
  for (int i = 0; i < 4; ++i) {
    const int row = rs + 32 * i;
    const int64_t r = row0 + row;
    uint32_t mask = 0;
    if (r < R && c0 < C) {
      float f[8], rv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
      unpack8(__ldg(reinterpret_cast<const uint4*>(x + r * C + c0)), f);
      if (ep.residual) unpack8(*reinterpret_cast<const uint4*>(ep.residual + r * C + c0), rv);
#pragma unroll
      for (int j = 0; j < 8; ++j) f[j] = epi_act(fmaf(f[j], sc[j], sh[j]) + rv[j], ep.act);
      const uint4 u = pack8(f);
      *reinterpret_cast<uint4*>(y + r * C + c0) = u;
      mask = nz_mask8(u);
    }
    if (emit) put_row_bits(s_nz, row, mask);
  }
  if (emit) {
    __syncthreads();
    flush_tile(s_nz, row0, blockIdx.y * 64, o, threadIdx.x, kTileThreads);
  }
}

dim3 tile_grid(int64_t R, int C) { return dim3((unsigned)((R + 127) / 128), (unsigned)((C + 63) / 64)); }

}  // namespace

cudaError_t launch_stats(const __nv_bfloat16* x, int64_t R, int C, const OccDev& o, cudaStream_t s) {
  if (R <= 0 || C <= 0) return cudaSuccess;
  stats_kernel<<<tile_grid(R, C), kTileThreads, 0, s>>>(x, R, C, o);
  return cudaGetLastError();
}

cudaError_t launch_pad_channels(const __nv_bfloat16* x, int64_t P, int C, int Cp,
                                __nv_bfloat16* y, cudaStream_t s) {
  const int64_t n = P * Cp;
  if (n <= 0) return cudaSuccess;
  pad_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(x, P, C, Cp, y);
  return cudaGetLastError();
}

cudaError_t launch_dwconv(const DwArgs& a, cudaStream_t s) {
  const int64_t R = (int64_t)a.N * a.Ho * a.Wo;
  if (R <= 0) return cudaSuccess;
  dwconv_kernel<<<tile_grid(R, a.C), kTileThreads, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_maxpool(const __nv_bfloat16* x, int N, int H, int W, int C, int k, int stride,
                           int pad, int Ho, int Wo, __nv_bfloat16* y, const OccDev& o, int emit,
                           cudaStream_t s) {
  const int64_t R = (int64_t)N * Ho * Wo;
  if (R <= 0) return cudaSuccess;
  maxpool_kernel<<<tile_grid(R, C), kTileThreads, 0, s>>>(x, N, H, W, C, k, stride, pad, Ho, Wo,
                                                          y, o, emit);
  return cudaGetLastError();
}

cudaError_t launch_avgpool(const __nv_bfloat16* x, int N, int HW, int C, __nv_bfloat16* y,
                           const OccDev& o, int emit, cudaStream_t s) {
  if (N <= 0) return cudaSuccess;
  avgpool_kernel<<<tile_grid(N, C), kTileThreads, 0, s>>>(x, N, HW, C, y, o, emit);
  return cudaGetLastError();
}

cudaError_t launch_bn_act(const __nv_bfloat16* x, int64_t R, int C, const EpiDev& ep,
                          __nv_bfloat16* y, const OccDev& o, int emit, cudaStream_t s) {
  if (R <= 0) return cudaSuccess;
  bn_act_kernel<<<tile_grid(R, C), kTileThreads, 0, s>>>(x, R, C, ep, y, o, emit);
  return cudaGetLastError();
}

}  // namespace sparoa
