// Dense and zero-skipping implicit-GEMM kernel on the 5th-generation tensor
// cores (tcgen05, accumulators in tensor memory), sm_103a.
//
// One CTA computes a 128 x BN tile of y = epilogue(A * B^T):
//   A [M, K]  GEMM: the activation matrix, loaded by TMA (64-byte swizzle).
//             Conv: gathered from the NHWC activation (implicit GEMM; K runs
//             over (tap, channel) in [kh][kw][C] order) by 128 producer
//             threads with cp.async, written in the same swizzled layout.
//   B [N, K]  the weights, K-major, loaded by TMA.
// K advances in 32-wide blocks (one 64-byte swizzle row, two MMAs of K = 16).
//
// Threshold dispatch (Sec. 3 rule, thresholds as parameters) happens inside
// the kernel: every CTA reads the Eq. 1 non-zero count of its input and
// evaluates the rule, so no host round trip separates statistics and compute.
// On the zero-skip path the producers leave out every K block whose
// activations are all zero over the tile's 128 rows (Sec. 2.1: zero-valued
// operations can be skipped without changing the output):
//   GEMM: K block kb of row block b is skipped iff word kb of the input's
//         block-column mask is 0 (no non-zero in those 32 columns x 128 rows);
//   conv: a (tap, channel) block is skipped iff none of the 128 shifted input
//         pixels has an occupied 64-channel tile there (row bitmaps; padding
//         counts as unoccupied).
// The epilogue applies bias / batch norm / residual / activation, stores y and
// writes y's Eq. 1 count and occupancy bitmaps for the next operator.
//
// Warp roles (288 threads): warps 0-3 producers, warps 4-7 epilogue (TMEM lane
// quarters 0-3), warp 8 TMEM allocation + MMA issue (lane 0).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "sparoa_kernels.h"

namespace sparoa {

namespace {

constexpr int kThreads = 288;
constexpr int kBM = 128;
constexpr int kBK = 32;                   // K elements per stage
constexpr int kAStageBytes = kBM * kBK * 2;  // 8 KiB
constexpr int kLag = 2;                   // cp.async stages in flight per producer

template <int BN>
struct Cfg {
  static constexpr int kStages = BN == 64 ? 8 : (BN == 128 ? 6 : 4);
  static constexpr int kBStageBytes = BN * kBK * 2;
  static constexpr int kAOff = 0;
  static constexpr int kBOff = kAOff + kStages * kAStageBytes;
  static constexpr int kBarOff = kBOff + kStages * kBStageBytes;    // 1024-aligned
  static constexpr int kFlagOff = kBarOff + (2 * kStages + 1) * 8;
  static constexpr int kScaleOff = (kFlagOff + (kStages + 8) * 4 + 15) & ~15;
  static constexpr int kShiftOff = kScaleOff + BN * 4;
  static constexpr int kNzOff = (kShiftOff + BN * 4 + 15) & ~15;
  static constexpr int kBytes = kNzOff + (BN / 64) * 128 * 8;
  static constexpr int kSmem = kBytes + 1024;  // slack for 1024-byte alignment
};

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
    igemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                 const IgemmArgs p) {
  using C = Cfg<BN>;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t sA = sbase + C::kAOff;
  const uint32_t sB = sbase + C::kBOff;
  const uint32_t bar_full = sbase + C::kBarOff;            // + 8*s
  const uint32_t bar_empty = bar_full + 8 * S;             // + 8*s
  const uint32_t bar_acc = bar_empty + 8 * S;
  int* flags = reinterpret_cast<int*>(smem + C::kFlagOff);
  int* stage_end = flags;                  // [S]
  volatile int* s_abort = flags + S;       // CTA-wide abort request
  int* s_acc_has = flags + S + 1;          // accumulator holds MMA results
  uint32_t* s_tmem = reinterpret_cast<uint32_t*>(flags + S + 2);
  volatile int* s_go = flags + S + 3;      // [2] producer broadcast
  float* s_scale = reinterpret_cast<float*>(smem + C::kScaleOff);
  float* s_shift = reinterpret_cast<float*>(smem + C::kShiftOff);
  uint64_t* s_nz = reinterpret_cast<uint64_t*>(smem + C::kNzOff);  // [BN/64][128]

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int path = decide_path(p.disp);
  if (p.dense_only && path == 2) return;  // the zero-skip kernel of this launch runs instead
  record_path(p.disp, path);
  const bool skip = (path == 2);
  const int m0 = blockIdx.x * kBM;
  const int n0 = blockIdx.y * BN;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(bar_full + 8 * s, p.conv ? 129u : 1u);
      mbar_init(bar_empty + 8 * s, 1u);
    }
    mbar_init(bar_acc, 1u);
    *s_abort = 0;
    *s_acc_has = 1;
    fence_mbar_init();
    if (!p.conv) prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
  }
  if (warp == 8) tmem_alloc(smem_u32(s_tmem), (uint32_t)BN);
  if (warp >= 4 && warp < 8) {
    const int et = threadIdx.x - 128;
    for (int c = et; c < BN; c += 128) {
      float sc = 1.f, sh = 0.f;
      if (n0 + c < p.N) epi_affine(p.ep, p.N, n0 + c, sc, sh);
      s_scale[c] = sc;
      s_shift[c] = sh;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *s_tmem;

  if (warp < 4) {
    // ------------------------------------------------------------------ producers
    const int r = threadIdx.x;  // A-tile row owned in conv mode
    if (!p.conv) {
      if (r == 0) {
        int i = 0;
        bool ok = true;
        for (int kb = 0; kb * kBK < p.Ktot; ++kb) {
          if (skip && p.in_blk[blockIdx.x * p.in_C32 + kb] == 0u) continue;
          const int slot = i % S;
          const uint32_t ph = (uint32_t)((i / S) & 1);
          if (!mbar_wait(bar_empty + 8 * slot, ph ^ 1u, p.err, s_abort, kErrTimeoutEmpty)) {
            ok = false;
            break;
          }
          stage_end[slot] = 0;
          mbar_arrive_expect_tx(bar_full + 8 * slot, (uint32_t)(kAStageBytes + C::kBStageBytes));
          tma_load_2d(sA + slot * kAStageBytes, &tmA, bar_full + 8 * slot, kb * kBK, m0);
          tma_load_2d(sB + slot * C::kBStageBytes, &tmB, bar_full + 8 * slot, kb * kBK, n0);
          ++i;
        }
        if (ok) {
          const int slot = i % S;
          const uint32_t ph = (uint32_t)((i / S) & 1);
          if (mbar_wait(bar_empty + 8 * slot, ph ^ 1u, p.err, s_abort, kErrTimeoutEmpty)) {
            stage_end[slot] = 1;
            mbar_arrive(bar_full + 8 * slot);
          }
        }
      }
    } else {
      // Implicit GEMM gather.  Row r of the tile is output pixel m0 + r.
      const int m = m0 + r;
      const bool mvalid = m < p.M;
      int img = 0, oh = 0, ow = 0;
      if (mvalid) {
        const int hw = p.Ho * p.Wo;
        img = m / hw;
        const int rem = m - img * hw;
        oh = rem / p.Wo;
        ow = rem - oh * p.Wo;
      }
      const int ih0 = oh * p.stride - p.pad;
      const int iw0 = ow * p.stride - p.pad;
      const __nv_bfloat16* ximg = p.x + (int64_t)img * p.H * p.W * p.Cp;
      const int64_t pix0 = (int64_t)img * p.H * p.W;
      const bool cp32 = (p.Cp % 32) == 0;
      int i = 0;           // stages filled
      int pending = 0;     // filled stages whose A arrivals are still owed
      bool ok = true;
      for (int kb = 0; kb * kBK < p.Ktot; ++kb) {
        // geometry of this thread's four 16-byte chunks
        const __nv_bfloat16* src[4];
        bool val[4];
        bool occ = false;
        int tap = 0, cbase = 0;
        if (cp32) {
          const int flat = kb * kBK;
          tap = flat / p.Cp;
          cbase = flat - tap * p.Cp;
        }
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          int t, c;
          const int flat = kb * kBK + 8 * j;
          if (cp32) {
            t = tap;
            c = cbase + 8 * j;
          } else {
            t = flat / p.Cp;
            c = flat - t * p.Cp;
          }
          const int rr = t / p.kw;
          const int ss = t - rr * p.kw;
          const int ih = ih0 + rr, iw = iw0 + ss;
          val[j] = mvalid && flat < p.Ktot && ih >= 0 && ih < p.H && iw >= 0 && iw < p.W;
          src[j] = val[j] ? ximg + ((int64_t)ih * p.W + iw) * p.Cp + c : p.x;
          if (skip && val[j]) {
            const int tile = c >> 6;
            const unsigned long long wbits =
                p.in_rowbm[(pix0 + (int64_t)ih * p.W + iw) * p.in_W64 + (tile >> 6)];
            occ |= ((wbits >> (tile & 63)) & 1ull) != 0ull;
          }
        }
        if (skip && !named_bar_or(1, 128, occ)) continue;
        const int slot = i % S;
        const uint32_t ph = (uint32_t)((i / S) & 1);
        if (r == 0) {
          const bool go = mbar_wait(bar_empty + 8 * slot, ph ^ 1u, p.err, s_abort, kErrTimeoutEmpty);
          s_go[i & 1] = go ? 1 : 0;
          if (go) {
            stage_end[slot] = 0;
            mbar_arrive_expect_tx(bar_full + 8 * slot, (uint32_t)C::kBStageBytes);
            tma_load_2d(sB + slot * C::kBStageBytes, &tmB, bar_full + 8 * slot, kb * kBK, n0);
          }
        }
        named_bar_sync(1, 128);
        if (!s_go[i & 1]) {
          ok = false;
          break;
        }
        const uint32_t dst = sA + slot * kAStageBytes;
#pragma unroll
        for (int j = 0; j < 4; ++j) cp_async_16(dst + sw64_offset(r, j), src[j], val[j] ? 16u : 0u);
        cp_async_commit();
        ++i;
        ++pending;
        if (pending > kLag) {
          cp_async_wait<kLag>();
          fence_proxy_async_smem();
          mbar_arrive(bar_full + 8 * ((i - 1 - kLag) % S));
          --pending;
        }
      }
      cp_async_wait<0>();
      fence_proxy_async_smem();
      for (int q = pending; q > 0; --q) mbar_arrive(bar_full + 8 * ((i - q) % S));
      named_bar_sync(1, 128);
      if (ok && r == 0) {
        const int slot = i % S;
        const uint32_t ph = (uint32_t)((i / S) & 1);
        if (mbar_wait(bar_empty + 8 * slot, ph ^ 1u, p.err, s_abort, kErrTimeoutEmpty)) {
          stage_end[slot] = 1;
          asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0], %1;" ::"r"(bar_full + 8 * slot),
                       "r"(129)
                       : "memory");
        }
      }
    }
  } else if (warp == 8) {
    // ------------------------------------------------------------------ MMA issue
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kBM, BN);
      int i = 0;
      bool any = false;
      while (true) {
        const int slot = i % S;
        const uint32_t ph = (uint32_t)((i / S) & 1);
        if (!mbar_wait(bar_full + 8 * slot, ph, p.err, s_abort, kErrTimeoutFull)) break;
        if (stage_end[slot]) break;
        tc_fence_after();
        const uint32_t a = sA + slot * kAStageBytes;
        const uint32_t b = sB + slot * C::kBStageBytes;
#pragma unroll
        for (int k = 0; k < kBK / 16; ++k)
          tc_mma_bf16(tmem, smem_desc_sw64(a + 32 * k), smem_desc_sw64(b + 32 * k), idesc,
                      (any || k > 0) ? 1u : 0u);
        any = true;
        tc_commit(bar_empty + 8 * slot);
        ++i;
      }
      if (any) {
        tc_commit(bar_acc);
      } else {
        *s_acc_has = 0;
        mbar_arrive(bar_acc);
      }
    }
  } else {
    // ------------------------------------------------------------------ epilogue
    const int q = warp & 3;            // TMEM lane quarter of this warp
    const int r = q * 32 + lane;       // tile row
    const int et = threadIdx.x - 128;  // 0..127
    const int64_t m = (int64_t)m0 + r;
    const bool mvalid = m < p.M;
    bool ok = mbar_wait(bar_acc, 0u, p.err, s_abort, kErrTimeoutAcc);
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();
    const bool has = ok && (*s_acc_has != 0);
    const bool vec = (p.N % 8) == 0;
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      if (has) {
        tmem_ld16(tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)c0, v);
      } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) v[j] = 0.f;
      }
      const int nb = n0 + c0;
      const bool full = vec && (nb + 16 <= p.N);
      float res[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) res[j] = 0.f;
      if (p.ep.residual && mvalid) {
        const __nv_bfloat16* rp = p.ep.residual + m * p.N + nb;
        if (full) {
          const uint4 r0 = *reinterpret_cast<const uint4*>(rp);
          const uint4 r1 = *reinterpret_cast<const uint4*>(rp + 8);
          const __nv_bfloat16* h0 = reinterpret_cast<const __nv_bfloat16*>(&r0);
          const __nv_bfloat16* h1 = reinterpret_cast<const __nv_bfloat16*>(&r1);
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            res[j] = __bfloat162float(h0[j]);
            res[8 + j] = __bfloat162float(h1[j]);
          }
        } else {
          for (int j = 0; j < 16; ++j)
            if (nb + j < p.N) res[j] = __bfloat162float(rp[j]);
        }
      }
      uint32_t nzbits = 0;
      if (p.y_f32) {
        float o[16];
#pragma unroll
        for (int j = 0; j < 16; ++j)
          o[j] = epi_act(fmaf(v[j], s_scale[c0 + j], s_shift[c0 + j]) + res[j], p.ep.act);
        if (mvalid) {
          float* yp = reinterpret_cast<float*>(p.y) + m * p.N + nb;
          if (full && (p.N % 4) == 0) {
#pragma unroll
            for (int j = 0; j < 16; j += 4)
              *reinterpret_cast<float4*>(yp + j) = make_float4(o[j], o[j + 1], o[j + 2], o[j + 3]);
          } else {
            for (int j = 0; j < 16; ++j)
              if (nb + j < p.N) yp[j] = o[j];
          }
        }
      } else {
        __align__(16) __nv_bfloat16 o[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          o[j] = __float2bfloat16_rn(
              epi_act(fmaf(v[j], s_scale[c0 + j], s_shift[c0 + j]) + res[j], p.ep.act));
          const uint16_t bits = __bfloat16_as_ushort(o[j]);
          if (mvalid && nb + j < p.N && bf16_nz(bits)) nzbits |= 1u << j;
        }
        if (mvalid) {
          __nv_bfloat16* yp = reinterpret_cast<__nv_bfloat16*>(p.y) + m * p.N + nb;
          if (full) {
            *reinterpret_cast<uint4*>(yp) = *reinterpret_cast<const uint4*>(&o[0]);
            *reinterpret_cast<uint4*>(yp + 8) = *reinterpret_cast<const uint4*>(&o[8]);
          } else {
            for (int j = 0; j < 16; ++j)
              if (nb + j < p.N) yp[j] = o[j];
          }
        }
      }
      if (p.emit) {
        uint64_t* w = &s_nz[(c0 >> 6) * 128 + r];
        const int sh = c0 & 63;
        if (sh == 0) *w = (uint64_t)nzbits;
        else *w |= (uint64_t)nzbits << sh;
      }
    }
    if (p.emit) {
      tc_fence_before();
      named_bar_sync(2, 128);
      for (int g = 0; g < BN / 64; ++g) {
        if (n0 + 64 * g < p.N) flush_tile(&s_nz[g * 128], m0, n0 + 64 * g, p.out_occ, et, 128);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 8) {
    tc_fence_after();
    tmem_dealloc(tmem, (uint32_t)BN);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 get_encode() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 2-D bf16 tensor [rows, cols] (cols contiguous), box {32, box_rows}, 64-byte swizzle.
bool make_tmap(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  auto enc = get_encode();
  if (!enc) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {32, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                   box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int BN>
cudaError_t launch_bn(const IgemmArgs& a, const CUtensorMap& tA, const CUtensorMap& tB,
                      cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(igemm_kernel<BN>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Cfg<BN>::kSmem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  dim3 grid((a.M + kBM - 1) / kBM, (a.N + BN - 1) / BN);
  igemm_kernel<BN><<<grid, kThreads, Cfg<BN>::kSmem, s>>>(tA, tB, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_igemm(const IgemmArgs& a, cudaStream_t s) {
  if (a.M <= 0 || a.N <= 0) return cudaSuccess;
  const int mt = (a.M + kBM - 1) / kBM;
  int bn = 64;
  if (a.N > 64) {
    bn = 256;
    while (bn > 64 && (bn / 2 >= a.N || (int64_t)mt * ((a.N + bn - 1) / bn) < 148)) bn /= 2;
  }
  CUtensorMap tA, tB;
  memset(&tA, 0, sizeof(tA));
  if (!a.conv) {
    if (!make_tmap(&tA, a.x, (uint64_t)a.M, (uint64_t)a.Ktot, kBM)) return cudaErrorInvalidValue;
  }
  if (!make_tmap(&tB, a.w, (uint64_t)a.N, (uint64_t)a.Ktot, (uint32_t)bn))
    return cudaErrorInvalidValue;
  if (a.conv) tA = tB;  // unused by the gather producers
  switch (bn) {
    case 64: return launch_bn<64>(a, tA, tB, s);
    case 128: return launch_bn<128>(a, tA, tB, s);
    default: return launch_bn<256>(a, tA, tB, s);
  }
}

}  // namespace sparoa
