// Vision-transformer operators (the attention-based models of Sec. 6, Table 2:
// ViT-B16): layer normalisation, multi-head self-attention, the token sequence
// of a patch embedding, and token selection.  The token-wise linear layers of
// a transformer are 1x1 convolutions over [N, 1, T, C] and run on the
// threshold-dispatched GEMM path; these kernels are the rest.  Their outputs'
// Eq. 1 statistics are measured by the stats kernel afterwards.
#include "sparoa_kernels.h"

namespace sparoa {

namespace {

constexpr int kVitThreads = 256;

// ---------------------------------------------------------------------------
// Layer normalisation: one warp per row of C values (C % 8 == 0), two passes
// over the row (mean, then the variance of the deviations), fp32.
__global__ void __launch_bounds__(kVitThreads) layernorm_kernel(const __nv_bfloat16* __restrict__ x,
                                                                int64_t R, int C,
                                                                const float* __restrict__ gb, float eps,
                                                                __nv_bfloat16* __restrict__ y) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kVitThreads / 32);
  const int chunks = C / 8;
  for (int64_t r = (int64_t)blockIdx.x * (kVitThreads / 32) + (threadIdx.x >> 5); r < R; r += warps) {
    const __nv_bfloat16* xr = x + r * C;
    float s = 0.f;
    for (int c = lane; c < chunks; c += 32) {
      float f[8];
      unpack8(*reinterpret_cast<const uint4*>(xr + c * 8), f);
#pragma unroll
      for (int k = 0; k < 8; ++k) s += f[k];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mean = s / (float)C;
    float q = 0.f;
    for (int c = lane; c < chunks; c += 32) {
      float f[8];
      unpack8(*reinterpret_cast<const uint4*>(xr + c * 8), f);
#pragma unroll
      for (int k = 0; k < 8; ++k) q = fmaf(f[k] - mean, f[k] - mean, q);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    const float rstd = rsqrtf(q / (float)C + eps);
    for (int c = lane; c < chunks; c += 32) {
      float f[8];
      unpack8(*reinterpret_cast<const uint4*>(xr + c * 8), f);
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        float v = (f[k] - mean) * rstd;
        if (gb) v = fmaf(v, gb[c * 8 + k], gb[C + c * 8 + k]);
        f[k] = v;
      }
      *reinterpret_cast<uint4*>(y + r * C + c * 8) = pack8(f);
    }
  }
}

// ---------------------------------------------------------------------------
// Multi-head self-attention.  Input rows (one per token) hold q | k | v, each
// heads x hd values; CTA = (image, head, block of 64 queries).  The head's K
// and V (T rows of hd bf16, rows padded by 16 bytes so that lanes reading
// different rows hit different banks) are staged in shared memory; each warp
// takes 8 queries in turn: lane j scores keys j, j + 32, ... against the query
// (held in registers), the warp forms the softmax, and lane l accumulates
// output dimensions 2l, 2l + 1 over all keys.
constexpr int kAttnQ = 64;       // queries per CTA
constexpr int kAttnMaxT = 512;   // tokens (16 scores per lane)
constexpr int kAttnMaxHd = 64;   // head dimension held per lane (2 per lane)

__global__ void __launch_bounds__(kVitThreads) attention_kernel(const __nv_bfloat16* __restrict__ qkv, int T,
                                                                int heads, int hd,
                                                                __nv_bfloat16* __restrict__ y) {
  extern __shared__ __align__(16) uint8_t smem[];
  const int pitch = hd * 2 + 16;  // bytes per staged row
  uint8_t* sK = smem;
  uint8_t* sV = smem + (size_t)T * pitch;
  const int n = blockIdx.x / heads, h = blockIdx.x - (blockIdx.x / heads) * heads;
  const int D = heads * hd, row3 = 3 * D;
  const __nv_bfloat16* base = qkv + (int64_t)n * T * row3;
  pdl_wait();
  pdl_trigger();
  // stage K and V of this head: 16-byte chunks
  const int cpr = hd / 8;  // chunks per row
  for (int idx = threadIdx.x; idx < T * cpr; idx += kVitThreads) {
    const int t = idx / cpr, c = idx - (idx / cpr) * cpr;
    const __nv_bfloat16* src = base + (int64_t)t * row3 + h * hd + c * 8;
    *reinterpret_cast<uint4*>(sK + t * pitch + c * 16) = *reinterpret_cast<const uint4*>(src + D);
    *reinterpret_cast<uint4*>(sV + t * pitch + c * 16) = *reinterpret_cast<const uint4*>(src + 2 * D);
  }
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const float scale = rsqrtf((float)hd);
  for (int qi = 0; qi < kAttnQ / 8; ++qi) {
    const int t = blockIdx.y * kAttnQ + warp * (kAttnQ / 8) + qi;
    if (t >= T) break;  // uniform across the warp
    float q[kAttnMaxHd];
    const __nv_bfloat16* qr = base + (int64_t)t * row3 + h * hd;
#pragma unroll
    for (int c = 0; c < kAttnMaxHd / 8; ++c) {
      if (c < cpr) {
        float f[8];
        unpack8(*reinterpret_cast<const uint4*>(qr + c * 8), f);
#pragma unroll
        for (int k = 0; k < 8; ++k) q[c * 8 + k] = f[k] * scale;
      } else {
#pragma unroll
        for (int k = 0; k < 8; ++k) q[c * 8 + k] = 0.f;
      }
    }
    // scores of keys lane, lane + 32, ...
    float sc[kAttnMaxT / 32];
    float mx = -3.402823466e38f;
#pragma unroll
    for (int i = 0; i < kAttnMaxT / 32; ++i) {
      const int j = lane + 32 * i;
      float sv = -3.402823466e38f;
      if (j < T) {
        sv = 0.f;
        const uint8_t* kr = sK + j * pitch;
#pragma unroll
        for (int c = 0; c < kAttnMaxHd / 8; ++c) {
          if (c < cpr) {
            float f[8];
            unpack8(*reinterpret_cast<const uint4*>(kr + c * 16), f);
#pragma unroll
            for (int k = 0; k < 8; ++k) sv = fmaf(q[c * 8 + k], f[k], sv);
          }
        }
      }
      sc[i] = sv;
      mx = fmaxf(mx, sv);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.f;
#pragma unroll
    for (int i = 0; i < kAttnMaxT / 32; ++i) {
      const int j = lane + 32 * i;
      const float e = j < T ? expf(sc[i] - mx) : 0.f;
      sc[i] = e;
      sum += e;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    const float inv = 1.f / sum;
    // output dims 2 lane, 2 lane + 1: sum over keys of p_j v_j
    float o0 = 0.f, o1 = 0.f;
    const bool dl = 2 * lane < hd;
#pragma unroll
    for (int i = 0; i < kAttnMaxT / 32; ++i) {
      if (32 * i >= T) break;
      const float pi = sc[i];
      const int jn = T - 32 * i < 32 ? T - 32 * i : 32;
      for (int l2 = 0; l2 < jn; ++l2) {
        const float p = __shfl_sync(0xffffffffu, pi, l2);
        if (dl) {
          const float2 v = __bfloat1622float2(
              *reinterpret_cast<const __nv_bfloat162*>(sV + (32 * i + l2) * pitch + lane * 4));
          o0 = fmaf(p, v.x, o0);
          o1 = fmaf(p, v.y, o1);
        }
      }
    }
    if (dl)
      *reinterpret_cast<__nv_bfloat162*>(y + ((int64_t)n * T + t) * D + h * hd + 2 * lane) =
          __floats2bfloat162_rn(o0 * inv, o1 * inv);
  }
}

// ---------------------------------------------------------------------------
// Token sequence: row 0 the class token, rows 1..P the patch vectors, each
// plus its position embedding (fp32 [1 + P][D]); 8 values per thread.
__global__ void __launch_bounds__(kVitThreads) tokens_kernel(const __nv_bfloat16* __restrict__ x, int N,
                                                             int P, int D,
                                                             const __nv_bfloat16* __restrict__ cls,
                                                             const float* __restrict__ pos,
                                                             __nv_bfloat16* __restrict__ y) {
  pdl_wait();
  pdl_trigger();
  const int cpr = D / 8;
  const int64_t total = (int64_t)N * (P + 1) * cpr;
  for (int64_t i = (int64_t)blockIdx.x * kVitThreads + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * kVitThreads) {
    const int c = (int)(i % cpr);
    const int64_t rt = i / cpr;
    const int t = (int)(rt % (P + 1));
    const int n = (int)(rt / (P + 1));
    const __nv_bfloat16* src = t == 0 ? cls + c * 8 : x + ((int64_t)n * P + (t - 1)) * D + c * 8;
    float f[8];
    unpack8(*reinterpret_cast<const uint4*>(src), f);
    const float* pp = pos + (int64_t)t * D + c * 8;
#pragma unroll
    for (int k = 0; k < 8; ++k) f[k] += pp[k];
    *reinterpret_cast<uint4*>(y + rt * D + c * 8) = pack8(f);
  }
}

// Token `index` of every image: [N, T, D] -> [N, D].
__global__ void __launch_bounds__(kVitThreads) select_kernel(const __nv_bfloat16* __restrict__ x, int N, int T,
                                                             int D, int index, __nv_bfloat16* __restrict__ y) {
  pdl_wait();
  pdl_trigger();
  const int cpr = D / 8;
  const int64_t total = (int64_t)N * cpr;
  for (int64_t i = (int64_t)blockIdx.x * kVitThreads + threadIdx.x; i < total;
       i += (int64_t)gridDim.x * kVitThreads) {
    const int c = (int)(i % cpr);
    const int n = (int)(i / cpr);
    *reinterpret_cast<uint4*>(y + (int64_t)n * D + c * 8) =
        *reinterpret_cast<const uint4*>(x + ((int64_t)n * T + index) * D + c * 8);
  }
}

unsigned grid_for(int64_t work, int per_cta) {
  const int64_t b = (work + per_cta - 1) / per_cta;
  const int64_t cap = 8LL * device_sm_count();
  return (unsigned)(b < 1 ? 1 : (b < cap ? b : cap));
}

}  // namespace

size_t attention_smem(int T, int hd) { return (size_t)2 * T * (hd * 2 + 16); }

cudaError_t launch_layernorm(const __nv_bfloat16* x, int64_t R, int C, const float* gb, float eps,
                             __nv_bfloat16* y, cudaStream_t s) {
  if (R <= 0) return cudaSuccess;
  if (C % 8) return cudaErrorInvalidValue;
  return launch_kernel(layernorm_kernel, dim3(grid_for(R, kVitThreads / 32)), dim3(kVitThreads), 0, s, x, R,
                       C, gb, eps, y);
}

cudaError_t launch_attention(const __nv_bfloat16* qkv, int N, int T, int heads, int hd, __nv_bfloat16* y,
                             cudaStream_t s) {
  if (N <= 0 || T <= 0) return cudaSuccess;
  if (T > kAttnMaxT || hd > kAttnMaxHd || hd % 8 || heads <= 0) return cudaErrorInvalidValue;
  const size_t smem = attention_smem(T, hd);
  static size_t attr = 0;
  if (smem > 40 * 1024 && smem > attr) {
    cudaError_t e = cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    attr = smem;
  }
  dim3 grid((unsigned)(N * heads), (unsigned)((T + kAttnQ - 1) / kAttnQ));
  return launch_kernel(attention_kernel, grid, dim3(kVitThreads), smem, s, qkv, T, heads, hd, y);
}

cudaError_t launch_tokens(const __nv_bfloat16* x, int N, int P, int D, const __nv_bfloat16* cls,
                          const float* pos, __nv_bfloat16* y, cudaStream_t s) {
  if (N <= 0) return cudaSuccess;
  if (D % 8) return cudaErrorInvalidValue;
  return launch_kernel(tokens_kernel, dim3(grid_for((int64_t)N * (P + 1) * (D / 8), kVitThreads)),
                       dim3(kVitThreads), 0, s, x, N, P, D, cls, pos, y);
}

cudaError_t launch_select(const __nv_bfloat16* x, int N, int T, int D, int index, __nv_bfloat16* y,
                          cudaStream_t s) {
  if (N <= 0) return cudaSuccess;
  if (D % 8 || index < 0 || index >= T) return cudaErrorInvalidValue;
  return launch_kernel(select_kernel, dim3(grid_for((int64_t)N * (D / 8), kVitThreads)), dim3(kVitThreads), 0,
                       s, x, N, T, D, index, y);
}

}  // namespace sparoa
