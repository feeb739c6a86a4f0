// Host-side launch interface of the libsparoa kernels (internal to the library).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "sparoa_dev.cuh"

namespace sparoa {

// Whether launches made by the calling host thread carry the programmatic
// stream serialization attribute (set per C-ABI call from its context).
bool pdl_enabled();
void set_pdl_enabled(bool on);

// Launch `kernel` on `s`, overlapping its prologue with the previous grid on
// the stream when enabled (the kernel must call pdl_wait() before touching
// global memory).
template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// Zero up to five word ranges (the fields of an occupancy block) in one launch.
struct ClearArgs {
  uint32_t* p[5];
  int64_t words[5];
};
cudaError_t launch_clear(const ClearArgs& a, cudaStream_t s);

// ----------------------------------------------------------------------------
// Implicit-GEMM tensor-core kernel (dense path and zero-skip path)
// ----------------------------------------------------------------------------
struct IgemmArgs {
  // Output y[M, N] (conv: M = images * Ho * Wo output pixels, N = C_out).
  int M = 0, N = 0;
  // conv = 0: A = x[M, K] row-major, loaded by TMA.  K = Ktot, K % 8 == 0.
  // conv = 1: A gathered from NHWC x (implicit GEMM over (tap, channel)).
  // conv = 2: A loaded by 4-D TMA boxes over a spatial output tile (Cp % 32 == 0).
  int conv = 0;
  const __nv_bfloat16* x = nullptr;
  int Nimg = 1, H = 1, W = 1, Cp = 0;  // conv input geometry; Cp = channel pitch (% 8 == 0)
  int Ho = 1, Wo = 1, kh = 1, kw = 1, stride = 1, pad = 0;
  int bw = 0, bh = 0, bn = 0;        // conv = 2: output tile of bw x bh pixels in bn images
  int tw = 0, th = 0;                // conv = 2: tiles along W and H
  int Ktot = 0;                      // GEMM K, or kh*kw*Cp
  const __nv_bfloat16* w = nullptr;  // [N, Ktot] K-major
  EpiDev ep{};
  void* y = nullptr;
  int y_f32 = 0;
  DispatchDev disp{};
  int dense_only = 0;                // 1: exit when the rule picks zero-skip
  // occupancy of the input (zero-skip path)
  const uint32_t* in_blk = nullptr;            // GEMM: blk_mask of x
  int in_C32 = 0;
  const unsigned long long* in_rowbm = nullptr;  // conv: row_bm of x
  int in_W64 = 0;
  // occupancy of the output
  OccDev out_occ{};
  int emit = 0;
  uint32_t* err = nullptr;
  long long wait_limit = 0;          // cycles before a bounded wait gives up (0: the default)
  int fault = 0;                     // error-path tests: kFaultSkipFirstAccCommit or 0
  // 1: the host launched a kernel of this library between the producers of
  // x, w and the epilogue's parameters and this grid, so they are complete
  // when this grid starts and may be read before griddepcontrol.wait (every
  // kernel here triggers its dependents only after its own wait)
  int early = 0;
  // split K (set by launch_igemm from the scratch offered here): fp32 partial
  // tiles [tiles][ksplit][128][BN] in `ws` (ws_bytes), one zeroed arrival
  // counter per output tile in `ws_cnt` (ws_cnt_len), left zero again
  int ksplit = 1;
  float* ws = nullptr;
  size_t ws_bytes = 0;
  unsigned* ws_cnt = nullptr;
  int ws_cnt_len = 0;
};

// Picks the N tile and the K split, encodes the tensor maps and launches.
cudaError_t launch_igemm(const IgemmArgs& a, cudaStream_t s);

// Streaming multiprocessors of the current device (cached per device).
int device_sm_count();

// Opt `func` in to `bytes` of dynamic shared memory on the current device.
// The attribute belongs to the device, so the largest size set so far is
// remembered per (device, kernel); the record is guarded by a mutex, so host
// threads may launch concurrently.
cudaError_t smem_optin(const void* func, size_t bytes);

// conv = 2: the bw x bh x bn (= 128) output tile with the fewest padded pixels.
void choose_spatial_tile(IgemmArgs& a);

// 3x3 stride-1 pad-1 convolution with resident weights and per-tile input
// slabs (k_conv3.cu); the same IgemmArgs (conv geometry, epilogue, dispatch,
// occupancy).  conv3_supported() says whether the shape fits.
bool conv3_supported(const IgemmArgs& a);
cudaError_t launch_conv3(const IgemmArgs& a, cudaStream_t s);

// ----------------------------------------------------------------------------
// Column-compacting zero-skip FC for few rows (M <= 128 per row block)
// ----------------------------------------------------------------------------
struct FcSkipArgs {
  const __nv_bfloat16* x = nullptr;   // [M, K]
  const __nv_bfloat16* w_kn = nullptr;  // [K, N]
  int M = 0, K = 0, N = 0;
  const uint32_t* in_blk = nullptr;   // blk_mask of x, [ceil(M/128)][ceil(K/32)]
  int in_C32 = 0;
  EpiDev ep{};
  void* y = nullptr;
  int y_f32 = 0;
  DispatchDev disp{};
  OccDev out_occ{};
  int emit = 0;
  unsigned long long* nnz_out = nullptr;  // fcsmall: where CTA 0 writes x's Eq. 1 count
};
cudaError_t launch_fcskip(const FcSkipArgs& a, cudaStream_t s);

// Fused statistics + dispatch + FC for an x that fits shared memory whole
// (M <= 128): counts x's non-zeros and occupied columns itself, writes the
// count to nnz_out (nullable) and the path to disp.path_out, and multiplies
// on the tensor cores (mma.sync) the occupied columns (zero-skip path) or all
// of them (dense path).
bool fcsmall_supported(int M, int K, int N);
cudaError_t launch_fcsmall(const FcSkipArgs& a, cudaStream_t s);

// ----------------------------------------------------------------------------
// Vision-transformer operators (k_vit.cu)
// ----------------------------------------------------------------------------
// y[r, :] = LN(x[r, :]) over C (C % 8 == 0); gb fp32 [2][C] gamma, beta or NULL.
cudaError_t launch_layernorm(const __nv_bfloat16* x, int64_t R, int C, const float* gb, float eps,
                             __nv_bfloat16* y, cudaStream_t s);
// qkv [N, T, 3 D] (q | k | v per token, D = heads * hd) -> y [N, T, D];
// T <= 512, hd 16, 32 or 64.
cudaError_t launch_attention(const __nv_bfloat16* qkv, int N, int T, int heads, int hd, __nv_bfloat16* y,
                             cudaStream_t s);
size_t attention_smem(int T, int hd);
// x [N, P, D] -> y [N, 1 + P, D]: class token row, then the patches; + pos [1 + P][D].
cudaError_t launch_tokens(const __nv_bfloat16* x, int N, int P, int D, const __nv_bfloat16* cls,
                          const float* pos, __nv_bfloat16* y, cudaStream_t s);
// x [N, T, D] -> y [N, D]: token `index`.
cudaError_t launch_select(const __nv_bfloat16* x, int N, int T, int D, int index, __nv_bfloat16* y,
                          cudaStream_t s);

// ----------------------------------------------------------------------------
// Memory-bound kernels (128-row x 64-channel tiles, occupancy fused)
// ----------------------------------------------------------------------------
// Eq. 1 statistics and bitmaps of x viewed as [R, C].  The row bitmaps are
// written whole when stats_writes_rows_whole(R, C) (one 64-column tile); the
// counters (nnz, col_nnz, tile_nnz), the block masks, and otherwise the row
// bitmaps, are accumulated and must be zero on entry.
constexpr int kStatsWholeRowCols = 512;
bool stats_writes_rows_whole(int64_t R, int C);
// early: x is complete when the kernel starts (a kernel of this library was
// launched between its producer and this one), so its first tiles are loaded
// before griddepcontrol.wait.  zero: word ranges the kernel zeroes after its
// wait, besides its own work (blocks that a later kernel accumulates into;
// not `o`).
cudaError_t launch_stats(const __nv_bfloat16* x, int64_t R, int C, const OccDev& o, cudaStream_t s,
                         bool early = false, const ClearArgs* zero = nullptr);

// im2col for a convolution with few input channels (k_tiles.cu): x [N, H, W,
// C] -> xc [N Ho Wo, Kp], each row the [kh][kw][C] window of one output pixel,
// zero-padded to Kp = im2col_width(C, kh, kw) (see im2col_kernel); for groups
// == 1, C < 8, kh kw > 1 and small enough windows (im2col_applies).
int im2col_width(int C, int kh, int kw);
bool im2col_applies(int C, int kh, int kw, int groups, int W, int P);
cudaError_t launch_im2col(const __nv_bfloat16* x, int N, int H, int W, int C, int kh, int kw, int S, int P,
                          __nv_bfloat16* xc, cudaStream_t s);

// Copy [P, C] to [P, Cp] with zero channels C..Cp-1.
cudaError_t launch_pad_channels(const __nv_bfloat16* x, int64_t P, int C, int Cp,
                                __nv_bfloat16* y, cudaStream_t s);

struct DwArgs {
  const __nv_bfloat16* x = nullptr;  // [N, H, W, C]
  const __nv_bfloat16* w = nullptr;  // [C, kh, kw]
  int N = 0, H = 0, W = 0, C = 0, kh = 3, kw = 3, stride = 1, pad = 1, Ho = 0, Wo = 0;
  EpiDev ep{};
  __nv_bfloat16* y = nullptr;
  OccDev out_occ{};
  int emit = 0;
  int32_t* path_out = nullptr;
  uint32_t* err = nullptr;           // bounded waits: error bits (k_dw3.cu)
  long long wait_limit = 0;          // cycles before a bounded wait gives up (0: the default)
};
cudaError_t launch_dwconv(const DwArgs& a, cudaStream_t s);
// The TMA-staged 3x3 depthwise kernel (k_dw3.cu): stride 1 or 2, pad 1,
// C % 8 == 0, a 16-byte aligned input and the weights of every channel in
// shared memory.
bool dw3_supported(const DwArgs& a);
cudaError_t launch_dw3(const DwArgs& a, cudaStream_t s);

cudaError_t launch_maxpool(const __nv_bfloat16* x, int N, int H, int W, int C, int k, int stride,
                           int pad, int Ho, int Wo, __nv_bfloat16* y, const OccDev& o, int emit,
                           cudaStream_t s);

cudaError_t launch_avgpool(const __nv_bfloat16* x, int N, int HW, int C, __nv_bfloat16* y,
                           const OccDev& o, int emit, cudaStream_t s);

cudaError_t launch_bn_act(const __nv_bfloat16* x, int64_t R, int C, const EpiDev& ep,
                          __nv_bfloat16* y, const OccDev& o, int emit, cudaStream_t s);

}  // namespace sparoa
