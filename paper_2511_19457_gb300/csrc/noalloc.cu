// sparoa_gemm_noalloc: the fully connected operator with threshold dispatch,
// for callers that must not allocate device memory.
//
// Who needs this: plugins that run inside another framework whose caching
// allocator owns all device memory, and latency-critical loops whose memory
// budget is fixed at start-up and where an allocation (slow, implicitly
// synchronising, or able to fail in the middle of a run) is not acceptable.  sparoa_gemm needs a context, whose
// creation allocates, and it measures the input's occupancy into context
// scratch that grows on demand.  This entry point instead keeps that scratch
// in one statically sized __device__ array that every GPU loading the library
// holds until the process exits.
//
// Use: the first call on a device resolves the array's device address with
// cudaGetSymbolAddress (the device must be current) and keeps it for the
// process, so a device reset after that call is not supported.  Every call
// shares the one array, and the
// array keeps the previous call's contents: each call clears the part it uses
// before writing.  Calls whose work overlaps on the GPU (several streams, or
// several host threads) race on the array; serialise them.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/sparoa.h"
#include "sparoa_kernels.h"

namespace sparoa {
namespace {

// 256 bytes of control words (error flag, path code) + the input occupancy.
constexpr size_t kCtrlBytes = 256;
constexpr size_t kStaticScratchBytes = (size_t)SPAROA_NOALLOC_SCRATCH_BYTES;
static __device__ __align__(256) unsigned char g_noalloc_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
void* g_scratch_addr[kMaxDevices] = {};
std::mutex g_scratch_mu;

size_t round16(size_t v) { return (v + 15) / 16 * 16; }

// Same carving as every other occupancy block of the library.
size_t carve(char* base, int64_t R, int64_t C, OccDev* o) {
  const int64_t T = (C + 63) / 64, W64 = (T + 63) / 64, RB = (R + 127) / 128, C32 = (C + 31) / 32;
  const size_t col = 16;
  const size_t tile = round16(col + 4 * (size_t)C);
  const size_t row = round16(tile + 4 * (size_t)T);
  const size_t blk = round16(row + 8 * (size_t)(R * W64));
  const size_t total = round16(blk + 4 * (size_t)(RB * C32));
  if (base) {
    o->nnz = reinterpret_cast<unsigned long long*>(base);
    o->col_nnz = reinterpret_cast<uint32_t*>(base + col);
    o->tile_nnz = reinterpret_cast<uint32_t*>(base + tile);
    o->row_bm = reinterpret_cast<unsigned long long*>(base + row);
    o->blk_mask = reinterpret_cast<uint32_t*>(base + blk);
    o->R = R;
    o->C = (int32_t)C;
    o->W64 = (int32_t)W64;
    o->C32 = (int32_t)C32;
  }
  return total;
}

}  // namespace
}  // namespace sparoa

using namespace sparoa;

extern "C" sparoa_status sparoa_gemm_noalloc(void* stream, const void* x, int64_t M, int64_t K,
                                             const void* W, const void* W_kn, int64_t N,
                                             const sparoa_epilogue* ep,
                                             const sparoa_thresholds* thr, void* y,
                                             int32_t y_dtype, sparoa_stats* host_out) {
  if (M < 0 || K <= 0 || N <= 0 || K % 8 || N % 8) return SPAROA_ERR_INVALID_ARG;
  if (M > ((int64_t)1 << 30) || K > (1 << 30) || N > (1 << 30)) return SPAROA_ERR_UNSUPPORTED;
  if (M > 0 && (!x || !W || !y)) return SPAROA_ERR_INVALID_ARG;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!al16(x) || !al16(W) || !al16(y) || (W_kn && !al16(W_kn))) return SPAROA_ERR_INVALID_ARG;
  if (y_dtype != SPAROA_BF16 && y_dtype != SPAROA_F32) return SPAROA_ERR_INVALID_ARG;
  if (ep && (ep->act < 0 || ep->act > 3 || (ep->residual && !al16(ep->residual))))
    return SPAROA_ERR_INVALID_ARG;
  sparoa_thresholds t;
  if (thr) {
    t = *thr;
  } else {
    t.s_thr = 0.5;
    t.c_thr = 32.0;
    t.intensity_mode = 0;
    t.force_path = 0;
  }
  if (!(t.s_thr == t.s_thr) || !(t.c_thr == t.c_thr) || t.intensity_mode < 0 ||
      t.intensity_mode > 1 || t.force_path < 0 || t.force_path > 2)
    return SPAROA_ERR_INVALID_ARG;
  // the control words and the input occupancy must fit the static array
  const size_t occ_bytes = carve(nullptr, M, K, nullptr);
  if (kCtrlBytes + occ_bytes > kStaticScratchBytes) return SPAROA_ERR_UNSUPPORTED;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return SPAROA_ERR_CUDA;
  void* base = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_addr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) {
        cudaGetLastError();
        return SPAROA_ERR_CUDA;
      }
      g_scratch_addr[dev] = p;
    }
    base = g_scratch_addr[dev];
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  char* b = static_cast<char*>(base);
  uint32_t* err = reinterpret_cast<uint32_t*>(b);
  int32_t* path_slot = reinterpret_cast<int32_t*>(b + 16);
  OccDev xo;
  carve(b + kCtrlBytes, M, K, &xo);
  {
    // control words, the Eq. 1 counters (which start the occupancy block) and
    // the block masks; the row bitmaps too unless the stats kernel writes them
    // whole (K <= 64)
    ClearArgs z = {};
    const int64_t blk_words = ((M + 127) / 128) * ((K + 31) / 32);
    z.p[0] = reinterpret_cast<uint32_t*>(b);
    if (stats_writes_rows_whole(M, (int)K)) {
      z.words[0] = (int64_t)((reinterpret_cast<char*>(xo.row_bm) - b) / 4);
      z.p[1] = xo.blk_mask;
      z.words[1] = blk_words;
    } else {
      z.words[0] = (int64_t)((reinterpret_cast<char*>(xo.blk_mask) - b) / 4) + blk_words;
    }
    if (launch_clear(z, s) != cudaSuccess) return SPAROA_ERR_CUDA;
  }

  const uint64_t flops = (uint64_t)2 * M * K * N;
  const uint64_t in_bytes = (uint64_t)M * K * 2;
  const double fpb = in_bytes ? (double)flops / (double)in_bytes : 0.0;
  const double intensity = t.intensity_mode == 1 ? (double)(K * N) : fpb;
  EpiDev e;
  e.bias = ep ? ep->bias : nullptr;
  e.bn = ep ? ep->bn : nullptr;
  e.eps = ep ? ep->bn_eps : 1e-5f;
  e.act = ep ? ep->act : 0;
  e.residual = ep ? static_cast<const __nv_bfloat16*>(ep->residual) : nullptr;
  DispatchDev d;
  d.in_nnz = xo.nnz;
  d.numel = (unsigned long long)(M * K);
  d.s_thr = t.s_thr;
  d.fpb_ok = intensity >= t.c_thr ? 1 : 0;
  d.force = t.force_path;
  d.path_out = path_slot;
  if (M > 0) {
    if (launch_stats(static_cast<const __nv_bfloat16*>(x), M, (int)K, xo, s) != cudaSuccess)
      return SPAROA_ERR_CUDA;
    const bool small_skip = M <= 128 && W_kn != nullptr && K <= 8192;
    if (!(small_skip && t.force_path == 2)) {
      IgemmArgs a;
      a.M = (int)M;
      a.N = (int)N;
      a.conv = 0;
      a.x = static_cast<const __nv_bfloat16*>(x);
      a.Ktot = (int)K;
      a.w = static_cast<const __nv_bfloat16*>(W);
      a.ep = e;
      a.y = y;
      a.y_f32 = y_dtype == SPAROA_F32;
      a.disp = d;
      a.dense_only = small_skip ? 1 : 0;
      a.in_blk = xo.blk_mask;
      a.in_C32 = xo.C32;
      a.emit = 0;
      a.err = err;
      if (launch_igemm(a, s) != cudaSuccess) return SPAROA_ERR_CUDA;
    }
    if (small_skip && t.force_path != 1) {
      FcSkipArgs f;
      f.x = static_cast<const __nv_bfloat16*>(x);
      f.w_kn = static_cast<const __nv_bfloat16*>(W_kn);
      f.M = (int)M;
      f.K = (int)K;
      f.N = (int)N;
      f.in_blk = xo.blk_mask;
      f.in_C32 = xo.C32;
      f.ep = e;
      f.y = y;
      f.y_f32 = y_dtype == SPAROA_F32;
      f.disp = d;
      f.emit = 0;
      if (launch_fcskip(f, s) != cudaSuccess) return SPAROA_ERR_CUDA;
    }
  }
  if (!host_out) return SPAROA_OK;
  unsigned long long nnz = 0;
  int32_t path = 0;
  uint32_t errv = 0;
  if (cudaMemcpyAsync(&nnz, xo.nnz, 8, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemcpyAsync(&path, path_slot, 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaMemcpyAsync(&errv, err, 4, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
      cudaStreamSynchronize(s) != cudaSuccess)
    return SPAROA_ERR_CUDA;
  if (errv) return SPAROA_ERR_TIMEOUT;
  const uint64_t numel = (uint64_t)(M * K);
  if (M == 0)  // no kernel ran; an empty input has no zeros to fall short of s_thr
    path = t.force_path == 1 ? SPAROA_PATH_DENSE_TC : SPAROA_PATH_ZERO_SKIP;
  host_out->numel = numel;
  host_out->nnz = nnz;
  host_out->sparsity = numel ? 1.0 - (double)nnz / (double)numel : 0.0;
  host_out->flops = flops;
  host_out->macs_eq2 = (uint64_t)(K * N);
  host_out->input_bytes = in_bytes;
  host_out->flops_per_byte = fpb;
  host_out->B = (int32_t)M;
  host_out->C_in = (int32_t)K;
  host_out->H = 1;
  host_out->W = 1;
  host_out->path = path;
  host_out->reserved = 0;
  return SPAROA_OK;
}
