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
// Layer normalisation: one warp per row of C values (C % 8 == 0), fp32: the
// mean, then the mean square of the deviations.  Rows of up to 1024 values
// are held in registers (every load of the row in flight at once, one pass
// over memory); longer rows are re-read for each of the three steps.
constexpr int kLnRegChunks = 4;  // 8-value chunks per lane held in registers

__device__ __forceinline__ void ln_store(__nv_bfloat16* __restrict__ yr, const float* __restrict__ gb, int C,
                                         int c, float (&f)[8], float mean, float rstd) {
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    float v = (f[k] - mean) * rstd;
    if (gb) v = fmaf(v, gb[c * 8 + k], gb[C + c * 8 + k]);
    f[k] = v;
  }
  *reinterpret_cast<uint4*>(yr + c * 8) = pack8(f);
}

__global__ void __launch_bounds__(kVitThreads) layernorm_kernel(const __nv_bfloat16* __restrict__ x,
                                                                int64_t R, int C,
                                                                const float* __restrict__ gb, float eps,
                                                                __nv_bfloat16* __restrict__ y) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (kVitThreads / 32);
  const int chunks = C / 8;
  const float inv_c = 1.f / (float)C;
  for (int64_t r = (int64_t)blockIdx.x * (kVitThreads / 32) + (threadIdx.x >> 5); r < R; r += warps) {
    const __nv_bfloat16* xr = x + r * C;
    __nv_bfloat16* yr = y + r * C;
    if (chunks <= 32 * kLnRegChunks) {
      uint4 u[kLnRegChunks];
#pragma unroll
      for (int i = 0; i < kLnRegChunks; ++i) {
        const int c = lane + 32 * i;
        u[i] = c < chunks ? *reinterpret_cast<const uint4*>(xr + c * 8) : make_uint4(0u, 0u, 0u, 0u);
      }
      float s = 0.f;
#pragma unroll
      for (int i = 0; i < kLnRegChunks; ++i) {
        float f[8];
        unpack8(u[i], f);
#pragma unroll
        for (int k = 0; k < 8; ++k) s += f[k];
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
      const float mean = s * inv_c;
      float q = 0.f;
#pragma unroll
      for (int i = 0; i < kLnRegChunks; ++i) {
        if (lane + 32 * i < chunks) {
          float f[8];
          unpack8(u[i], f);
#pragma unroll
          for (int k = 0; k < 8; ++k) q = fmaf(f[k] - mean, f[k] - mean, q);
        }
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
      const float rstd = rsqrtf(q * inv_c + eps);
#pragma unroll
      for (int i = 0; i < kLnRegChunks; ++i) {
        const int c = lane + 32 * i;
        if (c < chunks) {
          float f[8];
          unpack8(u[i], f);
          ln_store(yr, gb, C, c, f, mean, rstd);
        }
      }
      continue;
    }
    float s = 0.f;
    for (int c = lane; c < chunks; c += 32) {
      float f[8];
      unpack8(*reinterpret_cast<const uint4*>(xr + c * 8), f);
#pragma unroll
      for (int k = 0; k < 8; ++k) s += f[k];
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    const float mean = s * inv_c;
    float q = 0.f;
    for (int c = lane; c < chunks; c += 32) {
      float f[8];
      unpack8(*reinterpret_cast<const uint4*>(xr + c * 8), f);
#pragma unroll
      for (int k = 0; k < 8; ++k) q = fmaf(f[k] - mean, f[k] - mean, q);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) q += __shfl_xor_sync(0xffffffffu, q, o);
    const float rstd = rsqrtf(q * inv_c + eps);
    for (int c = lane; c < chunks; c += 32) {
      float f[8];
      unpack8(*reinterpret_cast<const uint4*>(xr + c * 8), f);
      ln_store(yr, gb, C, c, f, mean, rstd);
    }
  }
}

// ---------------------------------------------------------------------------
// Multi-head self-attention on the tensor cores (mma.sync m16n8k16, bf16 in,
// fp32 accumulate), flash-attention style.  Input rows (one per token) hold
// q | k | v, each heads x HD values.  One CTA per (image, head): the head's K
// and V rows are copied once into shared memory by cp.async (row pitch HD + 8
// elements, so the 8 rows of a fragment load fall in distinct banks; rows past
// T up to the next multiple of 16 zero-filled), then the 4 warps take the
// 16-query tiles in turn.  When the (image, head) pairs are fewer than the
// resident CTAs, each pair's query tiles are split over gridDim.y CTAs (each
// stages K and V itself).  A warp walks the keys in blocks of 64: S = Q K^T
// (Q fragments in registers, K fragments read as pairs of consecutive
// dimensions), an online softmax per query row (running maximum and sum,
// rescaling the output), and O += P V with P taken straight from the S
// accumulators (their layout is the A-operand layout of the next MMA) and the
// V fragments read by ldmatrix.trans from the row-major V.  Key tiles wholly
// at or past T are not computed.  O / sum is stored as bf16.
constexpr int kAttnThreads = 128;  // 4 warps
constexpr int kAttnMaxT = 512;
constexpr int kAttnKB = 64;        // keys per block

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
      "{%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// four 8x8 b16 matrices, transposed on the way: lanes 8i..8i+7 address the
// rows of matrix i, register i receives its fragment
__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                              uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr)
               : "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

template <int HD>
__global__ void __launch_bounds__(kAttnThreads, 3) attention_kernel(const __nv_bfloat16* __restrict__ qkv, int T,
                                                                    int heads, __nv_bfloat16* __restrict__ y) {
  extern __shared__ __align__(16) uint8_t smem[];
  constexpr int KP = HD + 8;  // row pitch of K and V (elements)
  const int T16 = (T + 15) & ~15;
  __nv_bfloat16* sK = reinterpret_cast<__nv_bfloat16*>(smem);  // [T16][KP]
  __nv_bfloat16* sV = sK + (size_t)T16 * KP;                     // [T16][KP]
  const int n = blockIdx.x / heads, h = blockIdx.x - (blockIdx.x / heads) * heads;
  const int D = heads * HD, row3 = 3 * D;
  const __nv_bfloat16* base = qkv + (int64_t)n * T * row3;
  pdl_wait();
  pdl_trigger();
  // K and V rows of the head: 16-byte copies, all in flight at once
  for (int idx = threadIdx.x; idx < T16 * (HD / 8); idx += kAttnThreads) {
    const int t = idx / (HD / 8), c = idx - (idx / (HD / 8)) * (HD / 8);
    const bool live = t < T;
    const __nv_bfloat16* src = base + (int64_t)(live ? t : 0) * row3 + h * HD + c * 8;
    cp_async_16(smem_u32(sK + t * KP + c * 8), src + D, live ? 16u : 0u);
    cp_async_16(smem_u32(sV + t * KP + c * 8), src + 2 * D, live ? 16u : 0u);
  }
  cp_async_commit();
  cp_async_wait<0>();
  __syncthreads();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int g = lane >> 2, tq = lane & 3;
  const float sl2 = rsqrtf((float)HD) * 1.4426950408889634f;  // 1/sqrt(HD) * log2(e)
  // ldmatrix.trans lane address within a (16 keys x 16 dimensions) V block:
  // matrices (keys 0-7, dims 0-7), (keys 8-15, dims 0-7), (keys 0-7, dims
  // 8-15), (keys 8-15, dims 8-15) -> b0, b1 of one 8-dimension n-tile, then
  // b0, b1 of the next
  const uint32_t v_lane = smem_u32(sV) + (uint32_t)(((lane & 15) * KP + (lane >> 4) * 8) * 2);
  const int qtn = (T + 15) >> 4;  // 16-query tiles
  const int per = (qtn + (int)gridDim.y - 1) / (int)gridDim.y;
  const int qt_end = min(qtn, ((int)blockIdx.y + 1) * per);
  for (int qt = (int)blockIdx.y * per + warp; qt < qt_end; qt += 4) {
    const int q0 = qt * 16;
    // Q fragments (A operand, rows g and g + 8, HD / 16 k-steps), zero past T
    uint32_t qa[HD / 16][4];
    {
      const int r0 = q0 + g, r1 = q0 + g + 8;
      const __nv_bfloat16* p0 = base + (int64_t)(r0 < T ? r0 : 0) * row3 + h * HD;
      const __nv_bfloat16* p1 = base + (int64_t)(r1 < T ? r1 : 0) * row3 + h * HD;
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk) {
        const int c = kk * 16 + 2 * tq;
        qa[kk][0] = r0 < T ? *reinterpret_cast<const uint32_t*>(p0 + c) : 0u;
        qa[kk][1] = r1 < T ? *reinterpret_cast<const uint32_t*>(p1 + c) : 0u;
        qa[kk][2] = r0 < T ? *reinterpret_cast<const uint32_t*>(p0 + c + 8) : 0u;
        qa[kk][3] = r1 < T ? *reinterpret_cast<const uint32_t*>(p1 + c + 8) : 0u;
      }
    }
    float o[HD / 8][4];
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
    float m0 = -3.0e38f, m1 = -3.0e38f, l0 = 0.f, l1 = 0.f;  // rows g, g + 8
    for (int kb = 0; kb < T; kb += kAttnKB) {
      // S = Q K^T for up to 64 keys: 8 n-tiles of 8 keys
      float s[kAttnKB / 8][4];
#pragma unroll
      for (int nt = 0; nt < kAttnKB / 8; ++nt) {
        s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
        if (kb + nt * 8 < T) {  // uniform across the warp
          const __nv_bfloat16* kr = sK + (kb + nt * 8 + g) * KP + 2 * tq;
#pragma unroll
          for (int kk = 0; kk < HD / 16; ++kk) {
            const uint32_t b0 = *reinterpret_cast<const uint32_t*>(kr + kk * 16);
            const uint32_t b1 = *reinterpret_cast<const uint32_t*>(kr + kk * 16 + 8);
            mma_bf16_16816(s[nt], qa[kk], b0, b1);
          }
        }
      }
      // keys past T do not take part
      if (kb + kAttnKB > T) {
#pragma unroll
        for (int nt = 0; nt < kAttnKB / 8; ++nt) {
          const int key = kb + nt * 8 + 2 * tq;
          if (key >= T) s[nt][0] = s[nt][2] = -3.0e38f;
          if (key + 1 >= T) s[nt][1] = s[nt][3] = -3.0e38f;
        }
      }
      // online softmax: block maxima of rows g and g + 8 over the 4 lanes of a quad
      float bm0 = -3.0e38f, bm1 = -3.0e38f;
#pragma unroll
      for (int nt = 0; nt < kAttnKB / 8; ++nt) {
        bm0 = fmaxf(bm0, fmaxf(s[nt][0], s[nt][1]));
        bm1 = fmaxf(bm1, fmaxf(s[nt][2], s[nt][3]));
      }
      bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 1));
      bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 2));
      bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 1));
      bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 2));
      const float nm0 = fmaxf(m0, bm0), nm1 = fmaxf(m1, bm1);
      const float c0 = exp2f((m0 - nm0) * sl2), c1 = exp2f((m1 - nm1) * sl2);
      m0 = nm0;
      m1 = nm1;
      float rs0 = 0.f, rs1 = 0.f;
      uint32_t pa[kAttnKB / 16][4];  // P as A fragments of the P V MMAs
#pragma unroll
      for (int nt = 0; nt < kAttnKB / 8; ++nt) {
        const float p0 = exp2f((s[nt][0] - nm0) * sl2), p1 = exp2f((s[nt][1] - nm0) * sl2);
        const float p2 = exp2f((s[nt][2] - nm1) * sl2), p3 = exp2f((s[nt][3] - nm1) * sl2);
        rs0 += p0 + p1;
        rs1 += p2 + p3;
        pa[nt >> 1][(nt & 1) * 2 + 0] = pack_bf16x2(p0, p1);
        pa[nt >> 1][(nt & 1) * 2 + 1] = pack_bf16x2(p2, p3);
      }
      l0 = l0 * c0 + rs0;
      l1 = l1 * c1 + rs1;
#pragma unroll
      for (int j = 0; j < HD / 8; ++j) {
        o[j][0] *= c0;
        o[j][1] *= c0;
        o[j][2] *= c1;
        o[j][3] *= c1;
      }
      // O += P V: k-steps of 16 keys (those starting before T), two 8-dimension
      // n-tiles per ldmatrix
#pragma unroll
      for (int kk = 0; kk < kAttnKB / 16; ++kk) {
        if (kb + kk * 16 < T) {  // uniform across the warp
          const uint32_t va = v_lane + (uint32_t)((kb + kk * 16) * KP * 2);
#pragma unroll
          for (int j = 0; j < HD / 8; j += 2) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4_trans(va + (uint32_t)(j * 8 * 2), b0, b1, b2, b3);
            mma_bf16_16816(o[j], pa[kk], b0, b1);
            mma_bf16_16816(o[j + 1], pa[kk], b2, b3);
          }
        }
      }
    }
    // row sums over the quad, then O / sum
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    const float i0 = 1.f / l0, i1 = 1.f / l1;
    const int r0 = q0 + g, r1 = q0 + g + 8;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      const int c = h * HD + j * 8 + 2 * tq;
      if (r0 < T)
        *reinterpret_cast<uint32_t*>(y + ((int64_t)n * T + r0) * D + c) = pack_bf16x2(o[j][0] * i0, o[j][1] * i0);
      if (r1 < T)
        *reinterpret_cast<uint32_t*>(y + ((int64_t)n * T + r1) * D + c) = pack_bf16x2(o[j][2] * i1, o[j][3] * i1);
    }
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

size_t attention_smem(int T, int hd) {
  const size_t T16 = (size_t)(T + 15) / 16 * 16;
  return 2 * 2 * T16 * (size_t)(hd + 8);  // K and V, bf16
}

namespace {

template <int HD>
cudaError_t launch_attention_hd(const __nv_bfloat16* qkv, int N, int T, int heads, __nv_bfloat16* y,
                                cudaStream_t s) {
  const size_t smem = attention_smem(T, HD);
  if (smem > 40 * 1024) {
    cudaError_t e = smem_optin(reinterpret_cast<const void*>(attention_kernel<HD>), smem);
    if (e != cudaSuccess) return e;
  }
  // split the query tiles while the (image, head) pairs leave resident CTA
  // slots (3 per SM) empty, down to one tile per warp
  const int pairs = N * heads;
  const int qsplit_max = ((T + 15) / 16 + 3) / 4;
  int qsplit = 3 * device_sm_count() / pairs;
  qsplit = qsplit < 1 ? 1 : (qsplit > qsplit_max ? qsplit_max : qsplit);
  dim3 grid((unsigned)pairs, (unsigned)qsplit);
  return launch_kernel(attention_kernel<HD>, grid, dim3(kAttnThreads), smem, s, qkv, T, heads, y);
}

}  // namespace

cudaError_t launch_attention(const __nv_bfloat16* qkv, int N, int T, int heads, int hd, __nv_bfloat16* y,
                             cudaStream_t s) {
  if (N <= 0 || T <= 0) return cudaSuccess;
  if (T > kAttnMaxT || heads <= 0) return cudaErrorInvalidValue;
  switch (hd) {
    case 16: return launch_attention_hd<16>(qkv, N, T, heads, y, s);
    case 32: return launch_attention_hd<32>(qkv, N, T, heads, y, s);
    case 64: return launch_attention_hd<64>(qkv, N, T, heads, y, s);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_layernorm(const __nv_bfloat16* x, int64_t R, int C, const float* gb, float eps,
                             __nv_bfloat16* y, cudaStream_t s) {
  if (R <= 0) return cudaSuccess;
  if (C % 8) return cudaErrorInvalidValue;
  return launch_kernel(layernorm_kernel, dim3(grid_for(R, kVitThreads / 32)), dim3(kVitThreads), 0, s, x, R,
                       C, gb, eps, y);
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
