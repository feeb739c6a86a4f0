// libsparoa C ABI: argument checks, workspace, launch plans and the graph walk.
// Declarations and documentation: include/sparoa.h.
#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/sparoa.h"
#include "sparoa_kernels.h"

namespace sparoa {
namespace {
thread_local bool t_pdl = true;

// Per-device launch facts: SM count, and per kernel the dynamic shared memory
// it has been opted in to on that device.
struct DeviceFacts {
  int sms = 0;
  std::map<const void*, size_t> optin;
};
std::mutex g_facts_mu;
std::map<int, DeviceFacts> g_facts;

int current_device() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    dev = 0;
  }
  return dev;
}
}  // namespace
bool pdl_enabled() { return t_pdl; }
void set_pdl_enabled(bool on) { t_pdl = on; }

int device_sm_count() {
  const int dev = current_device();
  std::lock_guard<std::mutex> lock(g_facts_mu);
  DeviceFacts& f = g_facts[dev];
  if (f.sms <= 0) {
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
      cudaGetLastError();
      return 152;  // grid sizing only; not remembered, so the next call asks again
    }
    f.sms = n;
  }
  return f.sms;
}

cudaError_t smem_optin(const void* func, size_t bytes) {
  const int dev = current_device();
  std::lock_guard<std::mutex> lock(g_facts_mu);
  size_t& have = g_facts[dev].optin[func];
  if (bytes <= have) return cudaSuccess;
  const cudaError_t e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e != cudaSuccess) return e;
  have = bytes;
  return cudaSuccess;
}
}  // namespace sparoa

using namespace sparoa;

namespace {

struct DevBuf {
  void* p = nullptr;
  size_t bytes = 0;
};

}  // namespace

struct sparoa_ctx {
  int device = 0;
  cudaStream_t stream = nullptr;
  std::string last_error;
  DevBuf small;       // u32 error flag, i32 path slot, padding
  DevBuf occ;         // occupancy of inputs measured inside a call
  DevBuf pad_x, pad_w;
  DevBuf arena;       // sparoa_run_graph activations, occupancies, paths
  DevBuf splitk;      // split-K arrival counters (kept zero) + fp32 partial tiles
  std::vector<sparoa_occupancy> graph_occ;
  int overlap = 1;    // programmatic dependent launch between consecutive kernels
  int64_t wait_limit = 0;  // SM cycles before a kernel's bounded wait gives up (0: default)
  int fault = 0;           // error-path tests: 1 MMA signal withheld, 2 next allocation fails
  cudaStream_t aux = nullptr;                        // second stream of split execution
  cudaEvent_t ev_fork = nullptr, ev_join = nullptr;  // its fork / join with `stream`
  uint32_t* d_err() const { return reinterpret_cast<uint32_t*>(small.p); }
  int32_t* d_path() const { return reinterpret_cast<int32_t*>(reinterpret_cast<char*>(small.p) + 16); }
  // Eq. 1 count of an FC input that the fused small-FC kernel measures itself
  uint64_t* d_count() const { return reinterpret_cast<uint64_t*>(reinterpret_cast<char*>(small.p) + 32); }
};

namespace {

constexpr size_t kAlign = 256;
size_t align_up(size_t v, size_t a = kAlign) { return (v + a - 1) / a * a; }

sparoa_status fail(sparoa_ctx* ctx, sparoa_status st, const char* fmt, ...) {
  if (ctx) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    ctx->last_error = buf;
  }
  return st;
}

#define SP_CUDA(call)                                                                   \
  do {                                                                                  \
    cudaError_t e_ = (call);                                                            \
    if (e_ != cudaSuccess)                                                              \
      return fail(ctx, SPAROA_ERR_CUDA, "%s: %s", #call, cudaGetErrorString(e_));      \
  } while (0)

#define SP_TRY(expr)                       \
  do {                                     \
    sparoa_status s_ = (expr);             \
    if (s_ != SPAROA_OK) return s_;        \
  } while (0)

// Make `device` current for the duration of a call and restore the caller's;
// launches made meanwhile follow the context's overlap setting.
struct DeviceGuard {
  int prev = -1;
  bool changed = false;
  bool pdl_prev = true;
  explicit DeviceGuard(int dev, int overlap = 1) {
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) changed = cudaSetDevice(dev) == cudaSuccess;
    pdl_prev = pdl_enabled();
    set_pdl_enabled(overlap != 0);
  }
  ~DeviceGuard() {
    set_pdl_enabled(pdl_prev);
    if (changed) cudaSetDevice(prev);
  }
};

sparoa_status ensure(sparoa_ctx* ctx, DevBuf& b, size_t bytes) {
  if (bytes <= b.bytes) return SPAROA_OK;
  if (ctx->fault == 2) {  // injected for the error-path tests: this allocation fails, once
    ctx->fault = 0;
    return fail(ctx, SPAROA_ERR_OOM, "workspace allocation of %zu bytes failed (injected)", bytes);
  }
  if (b.p) {
    SP_CUDA(cudaStreamSynchronize(ctx->stream));
    cudaFree(b.p);
    b.p = nullptr;
    b.bytes = 0;
  }
  const size_t want = align_up(bytes, 1 << 20);
  if (cudaMalloc(&b.p, want) != cudaSuccess) {
    cudaGetLastError();
    return fail(ctx, SPAROA_ERR_OOM, "workspace allocation of %zu bytes failed", want);
  }
  b.bytes = want;
  return SPAROA_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// ---------------------------------------------------------------------------
// occupancy layout
// ---------------------------------------------------------------------------
struct OccLayout {
  size_t nnz, col, tile, row, blk, total;
};

OccLayout occ_layout(int64_t R, int64_t C) {
  const int64_t T = (C + 63) / 64, W64 = (T + 63) / 64, RB = (R + 127) / 128, C32 = (C + 31) / 32;
  OccLayout l;
  l.nnz = 0;
  l.col = 16;
  l.tile = align_up(l.col + sizeof(uint32_t) * (size_t)C, 16);
  l.row = align_up(l.tile + sizeof(uint32_t) * (size_t)T, 16);
  l.blk = align_up(l.row + sizeof(uint64_t) * (size_t)(R * W64), 16);
  l.total = align_up(l.blk + sizeof(uint32_t) * (size_t)(RB * C32), 16);
  return l;
}

void occ_carve(void* base, int64_t R, int64_t C, sparoa_occupancy* o) {
  const OccLayout l = occ_layout(R, C);
  char* b = static_cast<char*>(base);
  o->nnz = reinterpret_cast<uint64_t*>(b + l.nnz);
  o->col_nnz = reinterpret_cast<uint32_t*>(b + l.col);
  o->tile_nnz = reinterpret_cast<uint32_t*>(b + l.tile);
  o->row_bm = reinterpret_cast<uint64_t*>(b + l.row);
  o->blk_mask = reinterpret_cast<uint32_t*>(b + l.blk);
  o->R = R;
  o->C = C;
  o->bytes = l.total;
}

OccDev to_dev(const sparoa_occupancy& o) {
  OccDev d;
  d.nnz = reinterpret_cast<unsigned long long*>(o.nnz);
  d.col_nnz = o.col_nnz;
  d.tile_nnz = o.tile_nnz;
  d.row_bm = reinterpret_cast<unsigned long long*>(o.row_bm);
  d.blk_mask = o.blk_mask;
  d.R = o.R;
  d.C = (int32_t)o.C;
  const int64_t T = (o.C + 63) / 64;
  d.W64 = (int32_t)((T + 63) / 64);
  d.C32 = (int32_t)((o.C + 31) / 32);
  return d;
}

sparoa_status check_occ(sparoa_ctx* ctx, const sparoa_occupancy* o, int64_t R, int64_t C,
                        const char* what) {
  if (!o) return SPAROA_OK;
  if (!o->nnz || !o->col_nnz || !o->tile_nnz || !o->row_bm || !o->blk_mask)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "%s: occupancy has a NULL field", what);
  if (o->R != R || o->C != C)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "%s: occupancy is [%lld, %lld], tensor is [%lld, %lld]",
                what, (long long)o->R, (long long)o->C, (long long)R, (long long)C);
  return SPAROA_OK;
}

// Clear an occupancy block with the clear kernel (a kernel, not a memset, so
// that consecutive launches keep overlapping).  rows_whole: everything but the
// row bitmaps (the stats kernel writes those whole).
sparoa_status occ_clear(sparoa_ctx* ctx, const sparoa_occupancy& o, bool rows_whole = false) {
  const int64_t T = (o.C + 63) / 64, W64 = (T + 63) / 64, RB = (o.R + 127) / 128,
                C32 = (o.C + 31) / 32;
  ClearArgs a = {};
  a.p[0] = reinterpret_cast<uint32_t*>(o.nnz);
  a.words[0] = 2;
  a.p[1] = o.col_nnz;
  a.words[1] = o.C;
  a.p[2] = o.tile_nnz;
  a.words[2] = T;
  if (!rows_whole) {
    a.p[3] = reinterpret_cast<uint32_t*>(o.row_bm);
    a.words[3] = 2 * o.R * W64;
  }
  a.p[4] = o.blk_mask;
  a.words[4] = RB * C32;
  SP_CUDA(launch_clear(a, ctx->stream));
  return SPAROA_OK;
}

// Word ranges that clear an occupancy block (rows_whole: all but the row
// bitmaps).  A block carved by sparoa_occupancy_init is contiguous and takes
// one range (two with rows_whole); any other block one range per field.
void occ_ranges(const sparoa_occupancy& o, bool rows_whole, std::vector<std::pair<uint32_t*, int64_t>>* out) {
  const OccLayout l = occ_layout(o.R, o.C);
  char* base = reinterpret_cast<char*>(o.nnz);
  const int64_t T = (o.C + 63) / 64, W64 = (T + 63) / 64, RB = (o.R + 127) / 128, C32 = (o.C + 31) / 32;
  const bool contiguous = reinterpret_cast<char*>(o.col_nnz) == base + l.col &&
                          reinterpret_cast<char*>(o.tile_nnz) == base + l.tile &&
                          reinterpret_cast<char*>(o.row_bm) == base + l.row &&
                          reinterpret_cast<char*>(o.blk_mask) == base + l.blk;
  if (contiguous) {
    if (rows_whole) {
      out->push_back({reinterpret_cast<uint32_t*>(base), (int64_t)(l.row / 4)});
      out->push_back({o.blk_mask, (int64_t)((l.total - l.blk) / 4)});
    } else {
      out->push_back({reinterpret_cast<uint32_t*>(base), (int64_t)(l.total / 4)});
    }
    return;
  }
  out->push_back({reinterpret_cast<uint32_t*>(o.nnz), 2});
  out->push_back({o.col_nnz, o.C});
  out->push_back({o.tile_nnz, T});
  if (!rows_whole) out->push_back({reinterpret_cast<uint32_t*>(o.row_bm), 2 * o.R * W64});
  out->push_back({o.blk_mask, RB * C32});
}

// Clear the given word ranges, five per launch.
sparoa_status clear_ranges(sparoa_ctx* ctx, const std::vector<std::pair<uint32_t*, int64_t>>& rg) {
  for (size_t i = 0; i < rg.size(); i += 5) {
    ClearArgs a = {};
    for (size_t k = 0; k < 5 && i + k < rg.size(); ++k) {
      a.p[k] = rg[i + k].first;
      a.words[k] = rg[i + k].second;
    }
    SP_CUDA(launch_clear(a, ctx->stream));
  }
  return SPAROA_OK;
}

// Split-K scratch offered to the implicit-GEMM kernel: 65536 arrival counters
// (zeroed once when allocated; every launch leaves them zero) and 64 MiB of
// fp32 partial tiles.  Allocated with the context.
constexpr int kSplitCounters = 65536;
constexpr size_t kSplitCntBytes = sizeof(unsigned) * kSplitCounters;
constexpr size_t kSplitWsBytes = (size_t)64 << 20;

// slot -1: the whole scratch; 0 / 1: disjoint halves, for two launches that
// may run at the same time (split execution)
sparoa_status offer_splitk(sparoa_ctx* ctx, IgemmArgs* a, int slot = -1) {
  if (!ctx->splitk.p) return SPAROA_OK;  // no split K
  a->ws_cnt = static_cast<unsigned*>(ctx->splitk.p);
  a->ws_cnt_len = kSplitCounters;
  a->ws = reinterpret_cast<float*>(static_cast<char*>(ctx->splitk.p) + kSplitCntBytes);
  a->ws_bytes = kSplitWsBytes;
  if (slot >= 0) {
    a->ws_cnt_len = kSplitCounters / 2;
    a->ws_cnt += slot * (kSplitCounters / 2);
    a->ws_bytes = kSplitWsBytes / 2;
    a->ws += slot * (kSplitWsBytes / 2 / sizeof(float));
  }
  return SPAROA_OK;
}

// Eq. 1 count and bitmaps of x [R, C] into `o` (counters and masks cleared
// first; the row bitmaps too unless the stats kernel writes them whole).
sparoa_status run_stats(sparoa_ctx* ctx, const void* x, int64_t R, int64_t C,
                        const sparoa_occupancy& o) {
  SP_TRY(occ_clear(ctx, o, stats_writes_rows_whole(R, (int)C)));
  SP_CUDA(launch_stats(static_cast<const __nv_bfloat16*>(x), R, (int)C, to_dev(o), ctx->stream, true));
  return SPAROA_OK;
}

// Occupancy of an input measured into context scratch.
sparoa_status measure(sparoa_ctx* ctx, const void* x, int64_t R, int64_t C, sparoa_occupancy* out) {
  const OccLayout l = occ_layout(R, C);
  SP_TRY(ensure(ctx, ctx->occ, l.total));
  occ_carve(ctx->occ.p, R, C, out);
  return run_stats(ctx, x, R, C, *out);
}

// ---------------------------------------------------------------------------
// Eq. 2 work and the rule on the host
// ---------------------------------------------------------------------------
struct Work {
  uint64_t flops = 0, macs = 0, in_bytes = 0;
  double fpb = 0.0;
};

Work conv_work(int64_t N, int64_t H, int64_t W, int64_t Cin, int64_t Cout, int64_t kh, int64_t kw,
               int64_t Ho, int64_t Wo, int64_t groups) {
  Work w;
  w.flops = (uint64_t)2 * N * Ho * Wo * Cout * (Cin / groups) * kh * kw;
  w.macs = (uint64_t)kh * kw * Cin * Cout * Ho * Wo;
  w.in_bytes = (uint64_t)N * H * W * Cin * 2;
  w.fpb = w.in_bytes ? (double)w.flops / (double)w.in_bytes : 0.0;
  return w;
}

Work fc_work(int64_t M, int64_t K, int64_t N) {
  Work w;
  w.flops = (uint64_t)2 * M * K * N;
  w.macs = (uint64_t)K * N;
  w.in_bytes = (uint64_t)M * K * 2;
  w.fpb = w.in_bytes ? (double)w.flops / (double)w.in_bytes : 0.0;
  return w;
}

// Q K^T and P V of every head: 2 T^2 D MACs per sequence; input bytes of q, k, v.
Work attention_work(int64_t N, int64_t T, int64_t D) {
  Work w;
  w.macs = (uint64_t)(2 * N * T * T * D);
  w.flops = 2 * w.macs;
  w.in_bytes = (uint64_t)(N * T * 3 * D * 2);
  w.fpb = w.in_bytes ? (double)w.flops / (double)w.in_bytes : 0.0;
  return w;
}

sparoa_thresholds thr_or_default(const sparoa_thresholds* t) {
  if (t) return *t;
  sparoa_thresholds d;
  d.s_thr = 0.5;
  d.c_thr = 32.0;
  d.intensity_mode = 0;
  d.force_path = 0;
  return d;
}

int intensity_ok(const sparoa_thresholds& t, const Work& w) {
  const double I = t.intensity_mode == 1 ? (double)w.macs : w.fpb;
  return I >= t.c_thr ? 1 : 0;
}

int host_rule(const sparoa_thresholds& t, uint64_t numel, uint64_t nnz, const Work& w) {
  if (t.force_path == 1) return SPAROA_PATH_DENSE_TC;
  if (t.force_path == 2) return SPAROA_PATH_ZERO_SKIP;
  const double zeros = (double)(numel - nnz);
  if (zeros >= t.s_thr * (double)numel) return SPAROA_PATH_ZERO_SKIP;
  return intensity_ok(t, w) ? SPAROA_PATH_DENSE_TC : SPAROA_PATH_ZERO_SKIP;
}

sparoa_status check_thr(sparoa_ctx* ctx, const sparoa_thresholds& t) {
  if (!(t.s_thr == t.s_thr) || !(t.c_thr == t.c_thr))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "thresholds must not be NaN");
  if (t.intensity_mode != 0 && t.intensity_mode != 1)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "intensity_mode must be 0 or 1");
  if (t.force_path < 0 || t.force_path > 2)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "force_path must be 0, 1 or 2");
  return SPAROA_OK;
}

EpiDev to_dev(const sparoa_epilogue* ep) {
  EpiDev e;
  e.bias = ep ? ep->bias : nullptr;
  e.bn = ep ? ep->bn : nullptr;
  e.eps = ep ? ep->bn_eps : 1e-5f;
  e.act = ep ? ep->act : 0;
  e.residual = ep ? static_cast<const __nv_bfloat16*>(ep->residual) : nullptr;
  return e;
}

sparoa_status check_ep(sparoa_ctx* ctx, const sparoa_epilogue* ep) {
  if (ep && (ep->act < 0 || ep->act > 3)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "bad activation");
  if (ep && ep->residual && !aligned16(ep->residual))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "residual must be 16-byte aligned");
  return SPAROA_OK;
}

sparoa_status read_device_error(sparoa_ctx* ctx) {
  uint32_t err = 0;
  SP_CUDA(cudaMemcpyAsync(&err, ctx->d_err(), 4, cudaMemcpyDeviceToHost, ctx->stream));
  SP_CUDA(cudaStreamSynchronize(ctx->stream));
  if (err) {
    SP_CUDA(cudaMemsetAsync(ctx->d_err(), 0, 4, ctx->stream));
    SP_CUDA(cudaStreamSynchronize(ctx->stream));
    return fail(ctx, SPAROA_ERR_TIMEOUT, "a kernel's bounded wait ran out (code 0x%x)", err);
  }
  return SPAROA_OK;
}

void fill_stats(sparoa_stats* s, uint64_t numel, uint64_t nnz, const Work& w, int B, int Cin, int H,
                int W, int path) {
  s->numel = numel;
  s->nnz = nnz;
  s->sparsity = numel ? 1.0 - (double)nnz / (double)numel : 0.0;
  s->flops = w.flops;
  s->macs_eq2 = w.macs;
  s->input_bytes = w.in_bytes ? w.in_bytes : numel * 2;
  s->flops_per_byte = w.fpb;
  s->B = B;
  s->C_in = Cin;
  s->H = H;
  s->W = W;
  s->path = path;
  s->reserved = 0;
}

// ---------------------------------------------------------------------------
// shared launch plans
// ---------------------------------------------------------------------------
struct GemmPlan {
  const void* x;
  int64_t M, K, N;
  const void* W;
  const void* W_kn;
  EpiDev ep;
  void* y;
  int y_f32;
  sparoa_occupancy xo;  // occupancy of x (device)
  const sparoa_occupancy* yo;
  DispatchDev disp;
};

// count_out: the input's Eq. 1 count is not known yet; the fused small-FC
// kernel measures it into count_out (which g.disp.in_nnz points at).
sparoa_status run_gemm(sparoa_ctx* ctx, const GemmPlan& g, cudaStream_t stream, int ws_slot = -1,
                       unsigned long long* count_out = nullptr) {
  const bool small_skip = g.M <= 128 && g.W_kn != nullptr && g.K <= 8192 && (g.N % 8) == 0;
  // small inputs: statistics, dispatch and either path's product in one kernel
  const bool fused = small_skip && fcsmall_supported((int)g.M, (int)g.K, (int)g.N);
  const int force = g.disp.force;
  OccDev yo{};
  if (g.yo) yo = to_dev(*g.yo);
  if (fused) {
    // both paths of a small FC in one launch (count, dispatch, product)
    FcSkipArgs f;
    f.x = static_cast<const __nv_bfloat16*>(g.x);
    f.w_kn = static_cast<const __nv_bfloat16*>(g.W_kn);
    f.M = (int)g.M;
    f.K = (int)g.K;
    f.N = (int)g.N;
    f.ep = g.ep;
    f.y = g.y;
    f.y_f32 = g.y_f32;
    f.disp = g.disp;
    f.out_occ = yo;
    f.emit = g.yo ? 1 : 0;
    f.nnz_out = count_out;
    SP_CUDA(launch_fcsmall(f, stream));
    return SPAROA_OK;
  }
  if (small_skip && force != 1) {
    FcSkipArgs f;
    f.x = static_cast<const __nv_bfloat16*>(g.x);
    f.w_kn = static_cast<const __nv_bfloat16*>(g.W_kn);
    f.M = (int)g.M;
    f.K = (int)g.K;
    f.N = (int)g.N;
    f.in_blk = g.xo.blk_mask;
    f.in_C32 = (int)((g.K + 31) / 32);
    f.ep = g.ep;
    f.y = g.y;
    f.y_f32 = g.y_f32;
    f.disp = g.disp;
    f.out_occ = yo;
    f.emit = g.yo ? 1 : 0;
    SP_CUDA(launch_fcskip(f, stream));
  }
  if (!(small_skip && force == 2)) {
    IgemmArgs a;
    a.M = (int)g.M;
    a.N = (int)g.N;
    a.conv = 0;
    a.x = static_cast<const __nv_bfloat16*>(g.x);
    a.Ktot = (int)g.K;
    a.w = static_cast<const __nv_bfloat16*>(g.W);
    a.ep = g.ep;
    a.y = g.y;
    a.y_f32 = g.y_f32;
    a.disp = g.disp;
    a.dense_only = small_skip ? 1 : 0;
    a.in_blk = g.xo.blk_mask;
    a.in_C32 = (int)((g.K + 31) / 32);
    a.out_occ = yo;
    a.emit = g.yo ? 1 : 0;
    a.err = ctx->d_err();
    a.wait_limit = ctx->wait_limit;
    a.fault = ctx->fault == 1 ? kFaultSkipFirstAccCommit : 0;
    SP_TRY(offer_splitk(ctx, &a, ws_slot));
    SP_CUDA(launch_igemm(a, stream));
  }
  return SPAROA_OK;
}

struct ConvPlan {
  const void* x;     // NHWC, channel pitch Cp
  int64_t N, H, W, Cin, Cp;
  const void* w;     // [Cout][kh][kw][Cp]
  int64_t Cout;
  int kh, kw, stride, pad;
  int64_t Ho, Wo;
  EpiDev ep;
  void* y;
  sparoa_occupancy xo;
  const sparoa_occupancy* yo;
  DispatchDev disp;
  // a kernel of this library was launched between the producers of x, w and
  // the epilogue's parameters and the conv (IgemmArgs::early)
  int early = 0;
};

sparoa_status run_conv(sparoa_ctx* ctx, const ConvPlan& c) {
  IgemmArgs a;
  const bool pointwise = c.kh == 1 && c.kw == 1 && c.stride == 1 && c.pad == 0;
  a.M = (int)(c.N * c.Ho * c.Wo);
  a.N = (int)c.Cout;
  a.conv = pointwise ? 0 : ((c.Cp % 32) == 0 ? 2 : 1);
  a.x = static_cast<const __nv_bfloat16*>(c.x);
  a.Nimg = (int)c.N;
  a.H = (int)c.H;
  a.W = (int)c.W;
  a.Cp = (int)c.Cp;
  a.Ho = (int)c.Ho;
  a.Wo = (int)c.Wo;
  a.kh = c.kh;
  a.kw = c.kw;
  a.stride = c.stride;
  a.pad = c.pad;
  a.Ktot = (int)(c.kh * c.kw * c.Cp);
  a.w = static_cast<const __nv_bfloat16*>(c.w);
  a.ep = c.ep;
  a.y = c.y;
  a.y_f32 = 0;
  a.disp = c.disp;
  a.dense_only = 0;
  a.in_blk = c.xo.blk_mask;
  a.in_C32 = (int)((c.Cin + 31) / 32);
  a.in_rowbm = reinterpret_cast<const unsigned long long*>(c.xo.row_bm);
  a.in_W64 = (int)((((c.Cin + 63) / 64) + 63) / 64);
  if (c.yo) a.out_occ = to_dev(*c.yo);
  a.emit = c.yo ? 1 : 0;
  a.err = ctx->d_err();
  a.wait_limit = ctx->wait_limit;
  a.fault = ctx->fault == 1 ? kFaultSkipFirstAccCommit : 0;
  a.early = c.early;
  if (!pointwise && conv3_supported(a)) {
    SP_CUDA(launch_conv3(a, ctx->stream));
    return SPAROA_OK;
  }
  if (a.conv == 2) choose_spatial_tile(a);
  SP_TRY(offer_splitk(ctx, &a));
  SP_CUDA(launch_igemm(a, ctx->stream));
  return SPAROA_OK;
}

int64_t out_dim(int64_t in, int k, int s, int p) { return (in + 2 * p - k) / s + 1; }

}  // namespace

// ===========================================================================
// C ABI
// ===========================================================================
extern "C" {

const char* sparoa_status_str(sparoa_status s) {
  switch (s) {
    case SPAROA_OK: return "ok";
    case SPAROA_ERR_INVALID_ARG: return "invalid argument";
    case SPAROA_ERR_UNSUPPORTED: return "unsupported";
    case SPAROA_ERR_OOM: return "out of device memory";
    case SPAROA_ERR_CUDA: return "CUDA error";
    case SPAROA_ERR_TIMEOUT: return "device wait timed out";
  }
  return "unknown status";
}

const char* sparoa_last_error(const sparoa_ctx* ctx) { return ctx ? ctx->last_error.c_str() : ""; }

sparoa_status sparoa_create(sparoa_ctx** out, int device, void* stream) {
  if (!out) return SPAROA_ERR_INVALID_ARG;
  *out = nullptr;
  int n = 0;
  if (cudaGetDeviceCount(&n) != cudaSuccess) {
    cudaGetLastError();
    return SPAROA_ERR_CUDA;
  }
  if (device < 0 || device >= n) return SPAROA_ERR_INVALID_ARG;
  DeviceGuard g(device);
  sparoa_ctx* ctx = new sparoa_ctx();
  ctx->device = device;
  ctx->stream = static_cast<cudaStream_t>(stream);
  if (cudaMalloc(&ctx->small.p, 256) != cudaSuccess) {
    cudaGetLastError();
    delete ctx;
    return SPAROA_ERR_OOM;
  }
  ctx->small.bytes = 256;
  if (cudaMemset(ctx->small.p, 0, 256) != cudaSuccess) {
    cudaFree(ctx->small.p);
    delete ctx;
    return SPAROA_ERR_CUDA;
  }
  // the split-K scratch is allocated here, not on first use, so that a
  // context's first conv/GEMM can be recorded by stream capture
  if (cudaMalloc(&ctx->splitk.p, kSplitCntBytes + kSplitWsBytes) != cudaSuccess) {
    cudaGetLastError();
    cudaFree(ctx->small.p);
    delete ctx;
    return SPAROA_ERR_OOM;
  }
  ctx->splitk.bytes = kSplitCntBytes + kSplitWsBytes;
  if (cudaStreamCreateWithFlags(&ctx->aux, cudaStreamNonBlocking) != cudaSuccess ||
      cudaEventCreateWithFlags(&ctx->ev_fork, cudaEventDisableTiming) != cudaSuccess ||
      cudaEventCreateWithFlags(&ctx->ev_join, cudaEventDisableTiming) != cudaSuccess) {
    cudaGetLastError();
    if (ctx->ev_fork) cudaEventDestroy(ctx->ev_fork);
    if (ctx->aux) cudaStreamDestroy(ctx->aux);
    cudaFree(ctx->splitk.p);
    cudaFree(ctx->small.p);
    delete ctx;
    return SPAROA_ERR_CUDA;
  }
  if (cudaMemset(ctx->splitk.p, 0, kSplitCntBytes) != cudaSuccess || cudaStreamSynchronize(0) != cudaSuccess) {
    cudaEventDestroy(ctx->ev_join);
    cudaEventDestroy(ctx->ev_fork);
    cudaStreamDestroy(ctx->aux);
    cudaFree(ctx->splitk.p);
    cudaFree(ctx->small.p);
    delete ctx;
    return SPAROA_ERR_CUDA;
  }
  *out = ctx;
  return SPAROA_OK;
}

sparoa_status sparoa_destroy(sparoa_ctx* ctx) {
  if (!ctx) return SPAROA_OK;
  DeviceGuard g(ctx->device, ctx->overlap);
  cudaStreamSynchronize(ctx->stream);
  if (ctx->aux) cudaStreamSynchronize(ctx->aux);
  for (DevBuf* b : {&ctx->small, &ctx->occ, &ctx->pad_x, &ctx->pad_w, &ctx->arena, &ctx->splitk})
    if (b->p) cudaFree(b->p);
  if (ctx->ev_fork) cudaEventDestroy(ctx->ev_fork);
  if (ctx->ev_join) cudaEventDestroy(ctx->ev_join);
  if (ctx->aux) cudaStreamDestroy(ctx->aux);
  delete ctx;
  return SPAROA_OK;
}

sparoa_status sparoa_set_overlap(sparoa_ctx* ctx, int32_t enable) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  ctx->overlap = enable ? 1 : 0;
  return SPAROA_OK;
}

sparoa_status sparoa_set_stream(sparoa_ctx* ctx, void* stream) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  ctx->stream = static_cast<cudaStream_t>(stream);
  return SPAROA_OK;
}

sparoa_status sparoa_last_path(sparoa_ctx* ctx, int32_t* path) {
  if (!ctx || !path) return SPAROA_ERR_INVALID_ARG;
  DeviceGuard g(ctx->device, ctx->overlap);
  int32_t p = 0;
  SP_CUDA(cudaMemcpyAsync(&p, ctx->d_path(), 4, cudaMemcpyDeviceToHost, ctx->stream));
  SP_TRY(read_device_error(ctx));
  *path = p;
  return SPAROA_OK;
}

sparoa_status sparoa_set_wait_limit(sparoa_ctx* ctx, int64_t cycles) {
  if (!ctx || cycles < 0) return SPAROA_ERR_INVALID_ARG;
  ctx->wait_limit = cycles;
  return SPAROA_OK;
}

sparoa_status sparoa_set_fault(sparoa_ctx* ctx, int32_t code) {
  if (!ctx || code < 0 || code > 2) return SPAROA_ERR_INVALID_ARG;
  ctx->fault = code;
  return SPAROA_OK;
}

sparoa_status sparoa_sync(sparoa_ctx* ctx) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  DeviceGuard g(ctx->device, ctx->overlap);
  return read_device_error(ctx);
}

uint64_t sparoa_occupancy_bytes(int64_t R, int64_t C) {
  if (R < 0 || C < 0) return 0;
  return occ_layout(R, C).total;
}

sparoa_status sparoa_occupancy_init(void* dev_buf, uint64_t bytes, int64_t R, int64_t C,
                                    sparoa_occupancy* out) {
  if (!dev_buf || !out || R < 0 || C <= 0 || !aligned16(dev_buf)) return SPAROA_ERR_INVALID_ARG;
  if (bytes < occ_layout(R, C).total) return SPAROA_ERR_INVALID_ARG;
  occ_carve(dev_buf, R, C, out);
  return SPAROA_OK;
}

sparoa_status sparoa_op_stats(sparoa_ctx* ctx, const void* x, int64_t N, int64_t H, int64_t W,
                              int64_t C, const sparoa_op* consumer, const sparoa_occupancy* occ,
                              sparoa_stats* host_out) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (N < 0 || H < 0 || W < 0 || C <= 0)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "op_stats: bad shape");
  const int64_t R = N * H * W;
  if (R > 0 && !x) return fail(ctx, SPAROA_ERR_INVALID_ARG, "op_stats: x is NULL");
  if (R > 0 && (C % 8) == 0 && !aligned16(x))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "op_stats: x must be 16-byte aligned");
  SP_TRY(check_occ(ctx, occ, R, C, "op_stats"));
  DeviceGuard g(ctx->device, ctx->overlap);
  sparoa_occupancy o;
  if (occ) {
    o = *occ;
    SP_TRY(run_stats(ctx, x, R, C, o));
  } else {
    SP_TRY(measure(ctx, x, R, C, &o));
  }
  if (!host_out) return SPAROA_OK;
  uint64_t nnz = 0;
  SP_CUDA(cudaMemcpyAsync(&nnz, o.nnz, 8, cudaMemcpyDeviceToHost, ctx->stream));
  SP_TRY(read_device_error(ctx));
  Work w;
  int path = SPAROA_PATH_NONE;
  if (consumer) {
    const sparoa_thresholds t = thr_or_default(&consumer->thr);
    if (consumer->kind == SPAROA_OP_CONV2D) {
      if (consumer->kh <= 0 || consumer->kw <= 0 || consumer->stride <= 0 || consumer->groups <= 0)
        return fail(ctx, SPAROA_ERR_INVALID_ARG, "op_stats: bad consumer geometry");
      const int64_t Ho = out_dim(H, consumer->kh, consumer->stride, consumer->pad);
      const int64_t Wo = out_dim(W, consumer->kw, consumer->stride, consumer->pad);
      w = conv_work(N, H, W, C, consumer->c_out, consumer->kh, consumer->kw, Ho, Wo,
                    consumer->groups);
      path = consumer->groups == 1 ? host_rule(t, (uint64_t)(R * C), nnz, w) : SPAROA_PATH_DEPTHWISE;
    } else if (consumer->kind == SPAROA_OP_FC) {
      w = fc_work(N, H * W * C, consumer->c_out);
      path = host_rule(t, (uint64_t)(R * C), nnz, w);
    }
  }
  fill_stats(host_out, (uint64_t)(R * C), nnz, w, (int)N, (int)C, (int)H, (int)W, path);
  return SPAROA_OK;
}

sparoa_status sparoa_gemm(sparoa_ctx* ctx, const void* x, int64_t M, int64_t K, const void* W,
                          const void* W_kn, int64_t N, const sparoa_epilogue* ep,
                          const sparoa_thresholds* thr, void* y, int32_t y_dtype,
                          const sparoa_occupancy* x_occ, const sparoa_occupancy* y_occ,
                          sparoa_stats* host_out) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (M < 0 || K <= 0 || N <= 0) return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm: bad shape");
  if (M > (int64_t)1 << 30 || K > (1 << 30) || N > (1 << 30))
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "gemm: dimension too large");
  if (K % 8 || N % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm: K and N must be multiples of 8");
  if (M > 0 && (!x || !W || !y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm: NULL tensor");
  if (!aligned16(x) || !aligned16(W) || !aligned16(y) || (W_kn && !aligned16(W_kn)))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm: tensors must be 16-byte aligned");
  if (y_dtype != SPAROA_BF16 && y_dtype != SPAROA_F32)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm: bad y_dtype");
  if (y_occ && y_dtype != SPAROA_BF16)
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "gemm: occupancy of an fp32 output");
  const sparoa_thresholds t = thr_or_default(thr);
  SP_TRY(check_thr(ctx, t));
  SP_TRY(check_ep(ctx, ep));
  SP_TRY(check_occ(ctx, x_occ, M, K, "gemm x_occ"));
  SP_TRY(check_occ(ctx, y_occ, M, N, "gemm y_occ"));
  DeviceGuard g(ctx->device, ctx->overlap);
  const Work w = fc_work(M, K, N);
  GemmPlan p;
  p.x = x;
  p.M = M;
  p.K = K;
  p.N = N;
  p.W = W;
  p.W_kn = W_kn;
  p.ep = to_dev(ep);
  p.y = y;
  p.y_f32 = y_dtype == SPAROA_F32;
  p.yo = y_occ;
  // a small input with its [K, N] weights is measured by the fused FC kernel
  // itself (count only); otherwise by the statistics kernel
  const bool fused_count = !x_occ && M > 0 && M <= 128 && W_kn && K <= 8192 &&
                           fcsmall_supported((int)M, (int)K, (int)N);
  if (x_occ) {
    p.xo = *x_occ;
  } else if (fused_count) {
    memset(&p.xo, 0, sizeof(p.xo));
    p.xo.nnz = ctx->d_count();
    p.xo.R = M;
    p.xo.C = K;
  } else {
    SP_TRY(measure(ctx, x, M, K, &p.xo));
  }
  if (y_occ) SP_TRY(occ_clear(ctx, *y_occ));
  p.disp.in_nnz = reinterpret_cast<const unsigned long long*>(p.xo.nnz);
  p.disp.numel = (unsigned long long)(M * K);
  p.disp.s_thr = t.s_thr;
  p.disp.fpb_ok = intensity_ok(t, w);
  p.disp.force = t.force_path;
  p.disp.path_out = ctx->d_path();
  if (M > 0)
    SP_TRY(run_gemm(ctx, p, ctx->stream, -1,
                    fused_count ? reinterpret_cast<unsigned long long*>(ctx->d_count()) : nullptr));
  if (!host_out) return SPAROA_OK;
  uint64_t nnz = 0;
  int32_t path = 0;
  SP_CUDA(cudaMemcpyAsync(&nnz, p.xo.nnz, 8, cudaMemcpyDeviceToHost, ctx->stream));
  SP_CUDA(cudaMemcpyAsync(&path, ctx->d_path(), 4, cudaMemcpyDeviceToHost, ctx->stream));
  SP_TRY(read_device_error(ctx));
  if (M == 0) path = host_rule(t, 0, 0, w);
  fill_stats(host_out, (uint64_t)(M * K), nnz, w, (int)M, (int)K, 1, 1, path);
  return SPAROA_OK;
}

namespace {

// The occupancy of rows [r0, R) of a tensor whose occupancy is `o`: the row
// bitmaps and block-column masks of those rows (r0 a multiple of 128, so the
// blocks align), the Eq. 1 counters shared.
sparoa_occupancy occ_rows(const sparoa_occupancy& o, int64_t r0) {
  sparoa_occupancy v = o;
  const int64_t T = (o.C + 63) / 64, W64 = (T + 63) / 64, C32 = (o.C + 31) / 32;
  v.row_bm = o.row_bm + r0 * W64;
  v.blk_mask = o.blk_mask + (r0 / 128) * C32;
  v.R = o.R - r0;
  return v;
}

}  // namespace

sparoa_status sparoa_gemm_split(sparoa_ctx* ctx, const void* x, int64_t M, int64_t K, const void* W,
                                const void* W_kn, int64_t N, const sparoa_epilogue* ep, double xi,
                                void* y, int32_t y_dtype, const sparoa_occupancy* x_occ,
                                const sparoa_occupancy* y_occ) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (M < 0 || K <= 0 || N <= 0) return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm_split: bad shape");
  if (M > (int64_t)1 << 30 || K > (1 << 30) || N > (1 << 30))
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "gemm_split: dimension too large");
  if (K % 8 || N % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm_split: K and N must be multiples of 8");
  if (M > 0 && (!x || !W || !y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm_split: NULL tensor");
  if (!aligned16(x) || !aligned16(W) || !aligned16(y) || (W_kn && !aligned16(W_kn)))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm_split: tensors must be 16-byte aligned");
  if (y_dtype != SPAROA_BF16 && y_dtype != SPAROA_F32)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm_split: bad y_dtype");
  if (y_occ && y_dtype != SPAROA_BF16)
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "gemm_split: occupancy of an fp32 output");
  if (!(xi >= 0.0 && xi <= 1.0)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "gemm_split: xi outside [0, 1]");
  SP_TRY(check_ep(ctx, ep));
  SP_TRY(check_occ(ctx, x_occ, M, K, "gemm_split x_occ"));
  SP_TRY(check_occ(ctx, y_occ, M, N, "gemm_split y_occ"));
  if (M == 0) return SPAROA_OK;
  DeviceGuard g(ctx->device, ctx->overlap);
  // rows [0, Ms) zero-skip, [Ms, M) dense; Ms whole 128-row blocks
  int64_t Ms = (int64_t)llround(xi * (double)M / 128.0) * 128;
  if (Ms > M) Ms = M;
  GemmPlan p;
  p.x = x;
  p.M = M;
  p.K = K;
  p.N = N;
  p.W = W;
  p.W_kn = W_kn;
  p.ep = to_dev(ep);
  p.y = y;
  p.y_f32 = y_dtype == SPAROA_F32;
  p.yo = nullptr;
  if (x_occ) p.xo = *x_occ;
  else SP_TRY(measure(ctx, x, M, K, &p.xo));
  if (y_occ) SP_TRY(occ_clear(ctx, *y_occ));
  p.disp.in_nnz = reinterpret_cast<const unsigned long long*>(p.xo.nnz);
  p.disp.numel = (unsigned long long)(M * K);
  p.disp.s_thr = 0.5;
  p.disp.fpb_ok = 1;
  p.disp.path_out = nullptr;
  const size_t ysz = p.y_f32 ? 4 : 2;
  sparoa_occupancy yo_a, yo_b;
  GemmPlan a = p, b = p;
  a.M = Ms;
  a.disp.force = 2;  // zero-skip
  if (y_occ) {
    yo_a = *y_occ;
    yo_a.R = Ms;
    a.yo = &yo_a;
  }
  b.x = static_cast<const char*>(x) + Ms * K * 2;
  b.y = static_cast<char*>(y) + Ms * N * ysz;
  b.M = M - Ms;
  b.xo = occ_rows(p.xo, Ms);
  b.disp.force = 1;  // dense
  if (y_occ) {
    yo_b = occ_rows(*y_occ, Ms);
    b.yo = &yo_b;
  }
  if (Ms == 0) return run_gemm(ctx, b, ctx->stream);
  if (Ms == M) return run_gemm(ctx, a, ctx->stream);
  // the two parts on two streams (each takes half of the split-K scratch),
  // forked from and joined back into the context stream
  SP_CUDA(cudaEventRecord(ctx->ev_fork, ctx->stream));
  SP_CUDA(cudaStreamWaitEvent(ctx->aux, ctx->ev_fork, 0));
  SP_TRY(run_gemm(ctx, a, ctx->aux, 1));
  SP_TRY(run_gemm(ctx, b, ctx->stream, 0));
  SP_CUDA(cudaEventRecord(ctx->ev_join, ctx->aux));
  SP_CUDA(cudaStreamWaitEvent(ctx->stream, ctx->ev_join, 0));
  return SPAROA_OK;
}

sparoa_status sparoa_conv2d(sparoa_ctx* ctx, const void* x, int64_t N, int64_t H, int64_t W,
                            int64_t C_in, const void* w, int64_t C_out, int32_t kh, int32_t kw,
                            int32_t stride, int32_t pad, int32_t groups,
                            const sparoa_epilogue* ep, const sparoa_thresholds* thr, void* y,
                            const sparoa_occupancy* x_occ, const sparoa_occupancy* y_occ,
                            sparoa_stats* host_out) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (N < 0 || H <= 0 || W <= 0 || C_in <= 0 || C_out <= 0 || kh <= 0 || kw <= 0 || stride <= 0 ||
      pad < 0 || groups <= 0)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "conv2d: bad shape or geometry");
  const int64_t Ho = out_dim(H, kh, stride, pad), Wo = out_dim(W, kw, stride, pad);
  if (Ho <= 0 || Wo <= 0 || H + 2 * pad < kh || W + 2 * pad < kw)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "conv2d: empty output");
  if (N * H * W > ((int64_t)1 << 31) - 1 || N * Ho * Wo > ((int64_t)1 << 31) - 1 ||
      (int64_t)kh * kw * ((C_in + 7) / 8 * 8) > ((int64_t)1 << 30))
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "conv2d: problem too large");
  if (N > 0 && (!x || !w || !y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "conv2d: NULL tensor");
  if (!aligned16(w) || !aligned16(y) || ((C_in % 8) == 0 && !aligned16(x)))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "conv2d: tensors must be 16-byte aligned");
  const sparoa_thresholds t = thr_or_default(thr);
  SP_TRY(check_thr(ctx, t));
  SP_TRY(check_ep(ctx, ep));
  SP_TRY(check_occ(ctx, x_occ, N * H * W, C_in, "conv2d x_occ"));
  SP_TRY(check_occ(ctx, y_occ, N * Ho * Wo, C_out, "conv2d y_occ"));
  const bool depthwise = groups > 1 && groups == C_in && groups == C_out;
  if (groups > 1 && !depthwise)
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "conv2d: grouped convolution other than depthwise");
  if (depthwise && (C_in % 8 || kh != 3 || kw != 3))
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "conv2d: depthwise needs C %% 8 == 0 and a 3x3 kernel");
  if (!depthwise && (C_out % 8))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "conv2d: C_out must be a multiple of 8");
  DeviceGuard g(ctx->device, ctx->overlap);
  const Work wk = conv_work(N, H, W, C_in, C_out, kh, kw, Ho, Wo, groups);
  sparoa_occupancy xo;
  const bool need_x_occ = !depthwise || host_out;
  bool launched = false;  // a kernel of this call runs before the operator's
  if (need_x_occ && !x_occ && N > 0) {
    // The input's occupancy is measured into context scratch: one small
    // clear launch (the counters and block masks; the stats kernel writes the
    // row bitmaps whole when C_in <= 64), then the stats kernel, which also
    // zeroes the output's occupancy block.  The clear comes between x's
    // producer and the stats kernel, so that kernel may read x before its
    // griddepcontrol.wait.
    const int64_t R = N * H * W;
    SP_TRY(ensure(ctx, ctx->occ, occ_layout(R, C_in).total));
    occ_carve(ctx->occ.p, R, C_in, &xo);
    std::vector<std::pair<uint32_t*, int64_t>> pre, yr;
    occ_ranges(xo, stats_writes_rows_whole(R, (int)C_in), &pre);
    if (y_occ) occ_ranges(*y_occ, false, &yr);
    if (yr.size() > 5) {  // a caller block in separate fields: cleared with the input's
      pre.insert(pre.end(), yr.begin(), yr.end());
      yr.clear();
    }
    ClearArgs z = {};
    for (size_t k = 0; k < yr.size(); ++k) {
      z.p[k] = yr[k].first;
      z.words[k] = yr[k].second;
    }
    SP_TRY(clear_ranges(ctx, pre));
    SP_CUDA(launch_stats(static_cast<const __nv_bfloat16*>(x), R, (int)C_in, to_dev(xo), ctx->stream, true,
                         &z));
    launched = true;
  } else {
    if (need_x_occ && x_occ) xo = *x_occ;
    if (y_occ) {
      SP_TRY(occ_clear(ctx, *y_occ));
      launched = true;
    }
  }
  if (N > 0) {
    if (depthwise) {
      DwArgs a;
      a.x = static_cast<const __nv_bfloat16*>(x);
      a.w = static_cast<const __nv_bfloat16*>(w);
      a.N = (int)N;
      a.H = (int)H;
      a.W = (int)W;
      a.C = (int)C_in;
      a.kh = kh;
      a.kw = kw;
      a.stride = stride;
      a.pad = pad;
      a.Ho = (int)Ho;
      a.Wo = (int)Wo;
      a.ep = to_dev(ep);
      a.y = static_cast<__nv_bfloat16*>(y);
      if (y_occ) a.out_occ = to_dev(*y_occ);
      a.emit = y_occ ? 1 : 0;
      a.path_out = ctx->d_path();
      a.err = ctx->d_err();
      a.wait_limit = ctx->wait_limit;
      SP_CUDA(launch_dwconv(a, ctx->stream));
    } else {
      ConvPlan c;
      c.N = N;
      c.H = H;
      c.W = W;
      c.Cin = C_in;
      c.Cp = (C_in + 7) / 8 * 8;
      c.x = x;
      c.w = w;
      int ckh = kh, ckw = kw, cstride = stride, cpad = pad;
      bool cols = false;
      if (im2col_applies((int)C_in, kh, kw, groups, (int)W, pad)) {
        // a narrow stem as a GEMM of its im2col rows (a 1 x 1 conv over Kp channels)
        const int Kp = im2col_width((int)C_in, kh, kw);
        SP_TRY(ensure(ctx, ctx->pad_x, (size_t)(N * Ho * Wo * Kp * 2)));
        SP_TRY(ensure(ctx, ctx->pad_w, (size_t)(C_out * Kp * 2)));
        SP_CUDA(launch_im2col(static_cast<const __nv_bfloat16*>(x), (int)N, (int)H, (int)W, (int)C_in, kh, kw,
                              stride, pad, static_cast<__nv_bfloat16*>(ctx->pad_x.p), ctx->stream));
        SP_CUDA(launch_pad_channels(static_cast<const __nv_bfloat16*>(w), C_out, kh * kw * (int)C_in, Kp,
                                    static_cast<__nv_bfloat16*>(ctx->pad_w.p), ctx->stream));
        c.x = ctx->pad_x.p;
        c.w = ctx->pad_w.p;
        c.H = Ho;
        c.W = Wo;
        c.Cin = Kp;
        c.Cp = Kp;
        ckh = ckw = cstride = 1;
        cpad = 0;
        cols = true;
      } else if (c.Cp != C_in) {
        const int64_t P = N * H * W, Q = C_out * kh * kw;
        SP_TRY(ensure(ctx, ctx->pad_x, (size_t)(P * c.Cp * 2)));
        SP_TRY(ensure(ctx, ctx->pad_w, (size_t)(Q * c.Cp * 2)));
        SP_CUDA(launch_pad_channels(static_cast<const __nv_bfloat16*>(x), P, (int)C_in, (int)c.Cp,
                                    static_cast<__nv_bfloat16*>(ctx->pad_x.p), ctx->stream));
        SP_CUDA(launch_pad_channels(static_cast<const __nv_bfloat16*>(w), Q, (int)C_in, (int)c.Cp,
                                    static_cast<__nv_bfloat16*>(ctx->pad_w.p), ctx->stream));
        c.x = ctx->pad_x.p;
        c.w = ctx->pad_w.p;
      }
      c.Cout = C_out;
      c.kh = ckh;
      c.kw = ckw;
      c.stride = cstride;
      c.pad = cpad;
      c.Ho = Ho;
      c.Wo = Wo;
      c.ep = to_dev(ep);
      c.y = y;
      c.xo = xo;
      if (cols) {  // the im2col rows have no occupancy: every K block is kept
        c.xo.blk_mask = nullptr;
        c.xo.row_bm = nullptr;
      }
      c.yo = y_occ;
      c.disp.in_nnz = reinterpret_cast<const unsigned long long*>(xo.nnz);
      c.disp.numel = (unsigned long long)(N * H * W * C_in);
      c.disp.s_thr = t.s_thr;
      c.disp.fpb_ok = intensity_ok(t, wk);
      c.disp.force = t.force_path;
      c.disp.path_out = ctx->d_path();
      c.early = launched && c.Cp == C_in ? 1 : 0;  // (padding launches write x and w)
      SP_TRY(run_conv(ctx, c));
    }
  }
  if (!host_out) return SPAROA_OK;
  uint64_t nnz = 0;
  int32_t path = depthwise ? SPAROA_PATH_DEPTHWISE : 0;
  if (N > 0) {
    SP_CUDA(cudaMemcpyAsync(&nnz, xo.nnz, 8, cudaMemcpyDeviceToHost, ctx->stream));
    if (!depthwise)
      SP_CUDA(cudaMemcpyAsync(&path, ctx->d_path(), 4, cudaMemcpyDeviceToHost, ctx->stream));
  } else if (!depthwise) {
    path = host_rule(t, 0, 0, wk);
  }
  SP_TRY(read_device_error(ctx));
  fill_stats(host_out, (uint64_t)(N * H * W * C_in), nnz, wk, (int)N, (int)C_in, (int)H, (int)W,
             path);
  return SPAROA_OK;
}

sparoa_status sparoa_maxpool2d(sparoa_ctx* ctx, const void* x, int64_t N, int64_t H, int64_t W,
                               int64_t C, int32_t k, int32_t stride, int32_t pad, void* y,
                               const sparoa_occupancy* y_occ) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (N < 0 || H <= 0 || W <= 0 || C <= 0 || k <= 0 || stride <= 0 || pad < 0 || pad >= k)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "maxpool: bad shape or geometry");
  if (C % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "maxpool: C must be a multiple of 8");
  const int64_t Ho = out_dim(H, k, stride, pad), Wo = out_dim(W, k, stride, pad);
  if (Ho <= 0 || Wo <= 0) return fail(ctx, SPAROA_ERR_INVALID_ARG, "maxpool: empty output");
  if (N > 0 && (!x || !y || !aligned16(x) || !aligned16(y)))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "maxpool: NULL or misaligned tensor");
  SP_TRY(check_occ(ctx, y_occ, N * Ho * Wo, C, "maxpool y_occ"));
  DeviceGuard g(ctx->device, ctx->overlap);
  if (y_occ) SP_TRY(occ_clear(ctx, *y_occ));
  OccDev o{};
  if (y_occ) o = to_dev(*y_occ);
  SP_CUDA(launch_maxpool(static_cast<const __nv_bfloat16*>(x), (int)N, (int)H, (int)W, (int)C, k,
                         stride, pad, (int)Ho, (int)Wo, static_cast<__nv_bfloat16*>(y), o,
                         y_occ ? 1 : 0, ctx->stream));
  return SPAROA_OK;
}

sparoa_status sparoa_avgpool_global(sparoa_ctx* ctx, const void* x, int64_t N, int64_t H,
                                    int64_t W, int64_t C, void* y,
                                    const sparoa_occupancy* y_occ) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (N < 0 || H <= 0 || W <= 0 || C <= 0)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "avgpool: bad shape");
  if (C % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "avgpool: C must be a multiple of 8");
  if (N > 0 && (!x || !y || !aligned16(x) || !aligned16(y)))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "avgpool: NULL or misaligned tensor");
  SP_TRY(check_occ(ctx, y_occ, N, C, "avgpool y_occ"));
  DeviceGuard g(ctx->device, ctx->overlap);
  if (y_occ) SP_TRY(occ_clear(ctx, *y_occ));
  OccDev o{};
  if (y_occ) o = to_dev(*y_occ);
  SP_CUDA(launch_avgpool(static_cast<const __nv_bfloat16*>(x), (int)N, (int)(H * W), (int)C,
                         static_cast<__nv_bfloat16*>(y), o, y_occ ? 1 : 0, ctx->stream));
  return SPAROA_OK;
}

sparoa_status sparoa_layernorm(sparoa_ctx* ctx, const void* x, int64_t R, int64_t C,
                               const float* gamma_beta, float eps, void* y,
                               const sparoa_occupancy* y_occ) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (R < 0 || C <= 0 || C % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "layernorm: bad shape");
  if (R > 0 && (!x || !y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "layernorm: NULL tensor");
  if (!aligned16(x) || !aligned16(y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "layernorm: misaligned");
  if (!(eps >= 0.f)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "layernorm: eps");
  SP_TRY(check_occ(ctx, y_occ, R, C, "layernorm y_occ"));
  DeviceGuard g(ctx->device, ctx->overlap);
  SP_CUDA(launch_layernorm(static_cast<const __nv_bfloat16*>(x), R, (int)C, gamma_beta, eps,
                           static_cast<__nv_bfloat16*>(y), ctx->stream));
  if (y_occ) SP_TRY(run_stats(ctx, y, R, C, *y_occ));
  return SPAROA_OK;
}

sparoa_status sparoa_attention(sparoa_ctx* ctx, const void* qkv, int64_t N, int64_t T, int32_t heads,
                               int32_t head_dim, void* y, const sparoa_occupancy* y_occ) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (N < 0 || T <= 0 || heads <= 0 || head_dim <= 0)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "attention: bad shape");
  if (T > 512 || (head_dim != 16 && head_dim != 32 && head_dim != 64))
    return fail(ctx, SPAROA_ERR_UNSUPPORTED, "attention: T <= 512 and head_dim 16, 32 or 64 only");
  if (N > 0 && (!qkv || !y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "attention: NULL tensor");
  if (!aligned16(qkv) || !aligned16(y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "attention: misaligned");
  const int64_t D = (int64_t)heads * head_dim;
  SP_TRY(check_occ(ctx, y_occ, N * T, D, "attention y_occ"));
  DeviceGuard g(ctx->device, ctx->overlap);
  SP_CUDA(launch_attention(static_cast<const __nv_bfloat16*>(qkv), (int)N, (int)T, heads, head_dim,
                           static_cast<__nv_bfloat16*>(y), ctx->stream));
  if (y_occ) SP_TRY(run_stats(ctx, y, N * T, D, *y_occ));
  return SPAROA_OK;
}

sparoa_status sparoa_bn_act(sparoa_ctx* ctx, const void* x, int64_t R, int64_t C,
                            const sparoa_epilogue* ep, void* y, const sparoa_occupancy* y_occ) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (R < 0 || C <= 0) return fail(ctx, SPAROA_ERR_INVALID_ARG, "bn_act: bad shape");
  if (C % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "bn_act: C must be a multiple of 8");
  if (R > 0 && (!x || !y || !aligned16(x) || !aligned16(y)))
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "bn_act: NULL or misaligned tensor");
  SP_TRY(check_ep(ctx, ep));
  SP_TRY(check_occ(ctx, y_occ, R, C, "bn_act y_occ"));
  DeviceGuard g(ctx->device, ctx->overlap);
  if (y_occ) SP_TRY(occ_clear(ctx, *y_occ));
  OccDev o{};
  if (y_occ) o = to_dev(*y_occ);
  SP_CUDA(launch_bn_act(static_cast<const __nv_bfloat16*>(x), R, (int)C, to_dev(ep),
                        static_cast<__nv_bfloat16*>(y), o, y_occ ? 1 : 0, ctx->stream));
  return SPAROA_OK;
}

// ---------------------------------------------------------------------------
// graph walk
// ---------------------------------------------------------------------------
namespace {

// The graph walk's plan: every value's shape (checked against its operator),
// and the layout of the context arena that holds the occupancy blocks, the
// recorded paths, the activations and the channel-padded copies.
struct Val {
  int64_t n, h, w, c;
  size_t act_off = 0, occ_off = 0;
};
struct Aux {
  size_t padx = 0, padw = 0, fcocc = 0;
  int64_t cp = 0;
  bool cols = false;  // narrow stem as a GEMM of its im2col rows (im2col_applies)
  bool fc_view = false;
};
struct GraphPlan {
  std::vector<Val> vals;
  std::vector<Aux> aux;
  size_t nnz_off = 0, occ_end = 0, path_off = 0, total = 0;
};

sparoa_status plan_graph(sparoa_ctx* ctx, const sparoa_op* ops, int32_t n_ops, int64_t N, int64_t H,
                         int64_t W, int64_t C, GraphPlan& pl) {
  // ---- plan: shapes, checks and arena layout
  std::vector<Val>& vals = pl.vals;
  vals.assign((size_t)n_ops + 1, Val{});
  vals[0] = {N, H, W, C};
  std::vector<Aux>& aux = pl.aux;
  aux.assign((size_t)n_ops, Aux{});
  for (int i = 0; i < n_ops; ++i) {
    const sparoa_op& op = ops[i];
    if (op.input < 0 || op.input > i)
      return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d reads value %d", i, op.input);
    if (op.residual < -1 || op.residual > i)
      return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d residual %d", i, op.residual);
    const Val& in = vals[(size_t)op.input];
    Val out{};
    switch (op.kind) {
      case SPAROA_OP_CONV2D: {
        if (op.c_in != in.c || op.c_out <= 0 || op.kh <= 0 || op.kw <= 0 || op.stride <= 0 ||
            op.pad < 0 || op.groups <= 0 || !op.weight)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d conv geometry", i);
        const bool dw = op.groups > 1;
        if (dw && (op.groups != op.c_in || op.groups != op.c_out || op.c_in % 8 || op.kh != 3 || op.kw != 3))
          return fail(ctx, SPAROA_ERR_UNSUPPORTED, "run_graph: op %d grouped conv", i);
        if (!dw && op.c_out % 8)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d C_out %% 8", i);
        out = {in.n, out_dim(in.h, op.kh, op.stride, op.pad), out_dim(in.w, op.kw, op.stride, op.pad),
               op.c_out};
        if (out.h <= 0 || out.w <= 0)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d empty output", i);
        if (!dw && im2col_applies(op.c_in, op.kh, op.kw, op.groups, (int)in.w, op.pad)) {
          aux[(size_t)i].cols = true;
          aux[(size_t)i].cp = im2col_width(op.c_in, op.kh, op.kw);
        } else if (!dw && op.c_in % 8) {
          aux[(size_t)i].cp = (op.c_in + 7) / 8 * 8;
        }
        break;
      }
      case SPAROA_OP_FC: {
        const int64_t K = in.h * in.w * in.c;
        if (op.c_in != K || op.c_out <= 0 || op.c_out % 8 || K % 8 || !op.weight)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d fc shape", i);
        out = {in.n, 1, 1, op.c_out};
        aux[(size_t)i].fc_view = (in.h * in.w) != 1;
        break;
      }
      case SPAROA_OP_MAXPOOL:
        if (in.c % 8 || op.kh <= 0 || op.stride <= 0 || op.pad < 0 || op.pad >= op.kh)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d maxpool", i);
        out = {in.n, out_dim(in.h, op.kh, op.stride, op.pad), out_dim(in.w, op.kh, op.stride, op.pad),
               in.c};
        if (out.h <= 0 || out.w <= 0)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d empty output", i);
        break;
      case SPAROA_OP_AVGPOOL:
        if (in.c % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d avgpool", i);
        out = {in.n, 1, 1, in.c};
        break;
      case SPAROA_OP_BN_ACT:
        if (in.c % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d bn_act", i);
        out = {in.n, in.h, in.w, in.c};
        break;
      case SPAROA_OP_LAYERNORM:
        if (in.c % 8) return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d layernorm C %% 8", i);
        out = {in.n, in.h, in.w, in.c};
        break;
      case SPAROA_OP_ATTENTION: {
        const int64_t T = in.h * in.w;
        if (op.groups <= 0 || in.c % (3 * op.groups))
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d attention heads", i);
        const int64_t hd = in.c / 3 / op.groups;
        if (T > 512 || (hd != 16 && hd != 32 && hd != 64))
          return fail(ctx, SPAROA_ERR_UNSUPPORTED, "run_graph: op %d attention T %lld hd %lld", i,
                      (long long)T, (long long)hd);
        out = {in.n, in.h, in.w, in.c / 3};
        break;
      }
      case SPAROA_OP_TOKENS:
        if (in.c % 8 || !op.weight || !op.bias)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d tokens", i);
        out = {in.n, 1, 1 + in.h * in.w, in.c};
        break;
      case SPAROA_OP_SELECT:
        if (in.c % 8 || op.pad < 0 || op.pad >= in.h * in.w)
          return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d select", i);
        out = {in.n, 1, 1, in.c};
        break;
      default:
        return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d kind %d", i, op.kind);
    }
    if (op.act < 0 || op.act > 3)
      return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d activation %d", i, op.act);
    if (op.residual >= 0) {
      const Val& r = vals[(size_t)op.residual];
      if (r.n != out.n || r.h != out.h || r.w != out.w || r.c != out.c)
        return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: op %d residual shape", i);
    }
    if (out.n * out.h * out.w > ((int64_t)1 << 31) - 1)
      return fail(ctx, SPAROA_ERR_UNSUPPORTED, "run_graph: op %d too large", i);
    vals[(size_t)i + 1] = out;
  }
  size_t off = 0;
  const size_t nnz_off = off;  // all occupancy blocks first (one memset)
  for (auto& v : vals) {
    v.occ_off = off;
    off += align_up(occ_layout(v.n * v.h * v.w, v.c).total);
  }
  for (int i = 0; i < n_ops; ++i) {
    if (aux[(size_t)i].fc_view) {
      const Val& in = vals[(size_t)ops[i].input];
      aux[(size_t)i].fcocc = off;
      off += align_up(occ_layout(in.n, in.h * in.w * in.c).total);
    }
  }
  const size_t occ_end = off;
  const size_t path_off = off;
  off += align_up(sizeof(int32_t) * (size_t)n_ops);
  for (size_t v = 1; v < vals.size(); ++v) {
    vals[v].act_off = off;
    off += align_up((size_t)(vals[v].n * vals[v].h * vals[v].w * vals[v].c) * 2);
  }
  for (int i = 0; i < n_ops; ++i) {
    if (aux[(size_t)i].cols) {
      const Val& out = vals[(size_t)i + 1];
      aux[(size_t)i].padx = off;
      off += align_up((size_t)(out.n * out.h * out.w * aux[(size_t)i].cp) * 2);
      aux[(size_t)i].padw = off;
      off += align_up((size_t)(ops[i].c_out * aux[(size_t)i].cp) * 2);
    } else if (aux[(size_t)i].cp) {
      const Val& in = vals[(size_t)ops[i].input];
      aux[(size_t)i].padx = off;
      off += align_up((size_t)(in.n * in.h * in.w * aux[(size_t)i].cp) * 2);
      aux[(size_t)i].padw = off;
      off += align_up((size_t)(ops[i].c_out * ops[i].kh * ops[i].kw * aux[(size_t)i].cp) * 2);
    }
  }
  pl.nnz_off = nnz_off;
  pl.occ_end = occ_end;
  pl.path_off = path_off;
  pl.total = off;
  return SPAROA_OK;
}

}  // namespace

sparoa_status sparoa_graph_workspace(sparoa_ctx* ctx, const sparoa_op* ops, int32_t n_ops, int64_t N,
                                     int64_t H, int64_t W, int64_t C, uint64_t* bytes) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (!bytes) return fail(ctx, SPAROA_ERR_INVALID_ARG, "graph_workspace: NULL bytes");
  if (!ops || n_ops <= 0) return fail(ctx, SPAROA_ERR_INVALID_ARG, "graph_workspace: no operators");
  if (N <= 0 || H <= 0 || W <= 0 || C <= 0)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "graph_workspace: bad input");
  GraphPlan pl;
  SP_TRY(plan_graph(ctx, ops, n_ops, N, H, W, C, pl));
  *bytes = (uint64_t)pl.total;
  return SPAROA_OK;
}

sparoa_status sparoa_run_graph(sparoa_ctx* ctx, const sparoa_op* ops, int32_t n_ops,
                               const void* x, int64_t N, int64_t H, int64_t W, int64_t C, void* y,
                               uint64_t y_bytes, sparoa_record* records) {
  if (!ctx) return SPAROA_ERR_INVALID_ARG;
  if (!ops || n_ops <= 0) return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: no operators");
  if (N <= 0 || H <= 0 || W <= 0 || C <= 0 || !x)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: bad input");
  if (C % 8 == 0 && !aligned16(x)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: misaligned input");
  GraphPlan pl;
  SP_TRY(plan_graph(ctx, ops, n_ops, N, H, W, C, pl));
  std::vector<Val>& vals = pl.vals;
  std::vector<Aux>& aux = pl.aux;
  const size_t nnz_off = pl.nnz_off, occ_end = pl.occ_end, path_off = pl.path_off;
  const size_t off = pl.total;
  const Val& last = vals.back();
  const uint64_t out_bytes = (uint64_t)(last.n * last.h * last.w * last.c) * 2;
  if (y && y_bytes < out_bytes)
    return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: y holds %llu bytes, output needs %llu",
                (unsigned long long)y_bytes, (unsigned long long)out_bytes);
  if (y && !aligned16(y)) return fail(ctx, SPAROA_ERR_INVALID_ARG, "run_graph: misaligned y");
  DeviceGuard g(ctx->device, ctx->overlap);
  SP_TRY(ensure(ctx, ctx->arena, off));
  char* base = static_cast<char*>(ctx->arena.p);
  ctx->graph_occ.assign(vals.size(), sparoa_occupancy{});
  for (size_t v = 0; v < vals.size(); ++v)
    occ_carve(base + vals[v].occ_off, vals[v].n * vals[v].h * vals[v].w, vals[v].c, &ctx->graph_occ[v]);
  int32_t* d_paths = reinterpret_cast<int32_t*>(base + path_off);
  auto act = [&](int v) -> void* {
    return v == 0 ? const_cast<void*>(x) : static_cast<void*>(base + vals[(size_t)v].act_off);
  };
  // ---- execute
  {
    // every occupancy block and path slot of the walk, cleared in one launch
    ClearArgs z = {};
    z.p[0] = reinterpret_cast<uint32_t*>(base + nnz_off);
    z.words[0] = (int64_t)((occ_end - nnz_off + align_up(sizeof(int32_t) * (size_t)n_ops)) / 4);
    SP_CUDA(launch_clear(z, ctx->stream));
  }
  SP_TRY(run_stats(ctx, x, N * H * W, C, ctx->graph_occ[0]));
  for (int i = 0; i < n_ops; ++i) {
    const sparoa_op& op = ops[i];
    const Val& in = vals[(size_t)op.input];
    const Val& out = vals[(size_t)i + 1];
    const sparoa_occupancy& xo = ctx->graph_occ[(size_t)op.input];
    const sparoa_occupancy* yo = &ctx->graph_occ[(size_t)i + 1];
    EpiDev ep;
    ep.bias = op.bias;
    ep.bn = op.bn;
    ep.eps = op.bn_eps;
    ep.act = op.act;
    ep.residual = op.residual >= 0 ? static_cast<const __nv_bfloat16*>(act(op.residual)) : nullptr;
    const sparoa_thresholds t = op.thr;
    SP_TRY(check_thr(ctx, t));
    switch (op.kind) {
      case SPAROA_OP_CONV2D: {
        if (op.groups > 1) {
          DwArgs a;
          a.x = static_cast<const __nv_bfloat16*>(act(op.input));
          a.w = static_cast<const __nv_bfloat16*>(op.weight);
          a.N = (int)in.n;
          a.H = (int)in.h;
          a.W = (int)in.w;
          a.C = (int)in.c;
          a.kh = op.kh;
          a.kw = op.kw;
          a.stride = op.stride;
          a.pad = op.pad;
          a.Ho = (int)out.h;
          a.Wo = (int)out.w;
          a.ep = ep;
          a.y = static_cast<__nv_bfloat16*>(act(i + 1));
          a.out_occ = to_dev(*yo);
          a.emit = 1;
          a.path_out = d_paths + i;
          a.err = ctx->d_err();
          a.wait_limit = ctx->wait_limit;
          SP_CUDA(launch_dwconv(a, ctx->stream));
          break;
        }
        const Work wk = conv_work(in.n, in.h, in.w, in.c, op.c_out, op.kh, op.kw, out.h, out.w, 1);
        ConvPlan c;
        c.N = in.n;
        c.H = in.h;
        c.W = in.w;
        c.Cin = in.c;
        c.Cp = aux[(size_t)i].cp ? aux[(size_t)i].cp : in.c;
        c.x = act(op.input);
        c.w = op.weight;
        const bool cols = aux[(size_t)i].cols;
        if (cols) {  // a narrow stem as a GEMM of its im2col rows (a 1 x 1 conv over Kp channels)
          void* px = base + aux[(size_t)i].padx;
          void* pw = base + aux[(size_t)i].padw;
          SP_CUDA(launch_im2col(static_cast<const __nv_bfloat16*>(c.x), (int)in.n, (int)in.h, (int)in.w, (int)in.c,
                                op.kh, op.kw, op.stride, op.pad, static_cast<__nv_bfloat16*>(px), ctx->stream));
          SP_CUDA(launch_pad_channels(static_cast<const __nv_bfloat16*>(op.weight), (int64_t)op.c_out,
                                      op.kh * op.kw * (int)in.c, (int)c.Cp, static_cast<__nv_bfloat16*>(pw),
                                      ctx->stream));
          c.x = px;
          c.w = pw;
          c.H = out.h;
          c.W = out.w;
          c.Cin = c.Cp;
        } else if (aux[(size_t)i].cp) {
          const int64_t P = in.n * in.h * in.w, Q = (int64_t)op.c_out * op.kh * op.kw;
          void* px = base + aux[(size_t)i].padx;
          void* pw = base + aux[(size_t)i].padw;
          SP_CUDA(launch_pad_channels(static_cast<const __nv_bfloat16*>(c.x), P, (int)in.c, (int)c.Cp,
                                      static_cast<__nv_bfloat16*>(px), ctx->stream));
          SP_CUDA(launch_pad_channels(static_cast<const __nv_bfloat16*>(op.weight), Q, (int)in.c,
                                      (int)c.Cp, static_cast<__nv_bfloat16*>(pw), ctx->stream));
          c.x = px;
          c.w = pw;
        }
        c.Cout = op.c_out;
        c.kh = cols ? 1 : op.kh;
        c.kw = cols ? 1 : op.kw;
        c.stride = cols ? 1 : op.stride;
        c.pad = cols ? 0 : op.pad;
        c.Ho = out.h;
        c.Wo = out.w;
        c.ep = ep;
        c.y = act(i + 1);
        c.xo = xo;
        if (cols) {  // the im2col rows have no occupancy: every K block is kept
          c.xo.blk_mask = nullptr;
          c.xo.row_bm = nullptr;
        }
        c.yo = yo;
        c.disp.in_nnz = reinterpret_cast<const unsigned long long*>(xo.nnz);
        c.disp.numel = (unsigned long long)(in.n * in.h * in.w * in.c);
        c.disp.s_thr = t.s_thr;
        c.disp.fpb_ok = intensity_ok(t, wk);
        c.disp.force = t.force_path;
        c.disp.path_out = d_paths + i;
        SP_TRY(run_conv(ctx, c));
        break;
      }
      case SPAROA_OP_FC: {
        const int64_t M = in.n, K = in.h * in.w * in.c;
        const Work wk = fc_work(M, K, op.c_out);
        GemmPlan p;
        p.x = act(op.input);
        p.M = M;
        p.K = K;
        p.N = op.c_out;
        p.W = op.weight;
        p.W_kn = op.weight_kn;
        p.ep = ep;
        p.y = act(i + 1);
        p.y_f32 = 0;
        p.yo = yo;
        if (aux[(size_t)i].fc_view) {
          occ_carve(base + aux[(size_t)i].fcocc, M, K, &p.xo);
          SP_TRY(run_stats(ctx, p.x, M, K, p.xo));
        } else {
          p.xo = xo;
        }
        p.disp.in_nnz = reinterpret_cast<const unsigned long long*>(p.xo.nnz);
        p.disp.numel = (unsigned long long)(M * K);
        p.disp.s_thr = t.s_thr;
        p.disp.fpb_ok = intensity_ok(t, wk);
        p.disp.force = t.force_path;
        p.disp.path_out = d_paths + i;
        SP_TRY(run_gemm(ctx, p, ctx->stream));
        break;
      }
      case SPAROA_OP_MAXPOOL:
        SP_CUDA(launch_maxpool(static_cast<const __nv_bfloat16*>(act(op.input)), (int)in.n, (int)in.h,
                               (int)in.w, (int)in.c, op.kh, op.stride, op.pad, (int)out.h, (int)out.w,
                               static_cast<__nv_bfloat16*>(act(i + 1)), to_dev(*yo), 1, ctx->stream));
        break;
      case SPAROA_OP_AVGPOOL:
        SP_CUDA(launch_avgpool(static_cast<const __nv_bfloat16*>(act(op.input)), (int)in.n,
                               (int)(in.h * in.w), (int)in.c, static_cast<__nv_bfloat16*>(act(i + 1)),
                               to_dev(*yo), 1, ctx->stream));
        break;
      case SPAROA_OP_BN_ACT:
        SP_CUDA(launch_bn_act(static_cast<const __nv_bfloat16*>(act(op.input)), in.n * in.h * in.w,
                              (int)in.c, ep, static_cast<__nv_bfloat16*>(act(i + 1)), to_dev(*yo), 1,
                              ctx->stream));
        break;
      case SPAROA_OP_LAYERNORM:
        SP_CUDA(launch_layernorm(static_cast<const __nv_bfloat16*>(act(op.input)), in.n * in.h * in.w,
                                 (int)in.c, op.bn, op.bn_eps, static_cast<__nv_bfloat16*>(act(i + 1)),
                                 ctx->stream));
        break;
      case SPAROA_OP_ATTENTION:
        SP_CUDA(launch_attention(static_cast<const __nv_bfloat16*>(act(op.input)), (int)in.n,
                                 (int)(in.h * in.w), op.groups, (int)(in.c / 3 / op.groups),
                                 static_cast<__nv_bfloat16*>(act(i + 1)), ctx->stream));
        break;
      case SPAROA_OP_TOKENS:
        SP_CUDA(launch_tokens(static_cast<const __nv_bfloat16*>(act(op.input)), (int)in.n,
                              (int)(in.h * in.w), (int)in.c, static_cast<const __nv_bfloat16*>(op.weight),
                              op.bias, static_cast<__nv_bfloat16*>(act(i + 1)), ctx->stream));
        break;
      case SPAROA_OP_SELECT:
        SP_CUDA(launch_select(static_cast<const __nv_bfloat16*>(act(op.input)), (int)in.n,
                              (int)(in.h * in.w), (int)in.c, op.pad, static_cast<__nv_bfloat16*>(act(i + 1)),
                              ctx->stream));
        break;
    }
    if (op.kind >= SPAROA_OP_LAYERNORM) {
      // these kernels write no occupancy: the stats kernel measures the output
      // (the walk cleared every occupancy block when it started)
      SP_CUDA(launch_stats(static_cast<const __nv_bfloat16*>(act(i + 1)), out.n * out.h * out.w,
                           (int)out.c, to_dev(*yo), ctx->stream));
    }
  }
  if (y) SP_CUDA(cudaMemcpyAsync(y, act(n_ops), out_bytes, cudaMemcpyDeviceToDevice, ctx->stream));
  if (!records) return SPAROA_OK;
  std::vector<int32_t> paths((size_t)n_ops);
  std::vector<uint64_t> nnz(vals.size());
  SP_CUDA(cudaMemcpyAsync(paths.data(), d_paths, sizeof(int32_t) * (size_t)n_ops,
                          cudaMemcpyDeviceToHost, ctx->stream));
  for (size_t v = 0; v < vals.size(); ++v)
    SP_CUDA(cudaMemcpyAsync(&nnz[v], ctx->graph_occ[v].nnz, 8, cudaMemcpyDeviceToHost, ctx->stream));
  SP_TRY(read_device_error(ctx));
  for (int i = 0; i < n_ops; ++i) {
    const sparoa_op& op = ops[i];
    const Val& in = vals[(size_t)op.input];
    const Val& out = vals[(size_t)i + 1];
    Work wk;
    if (op.kind == SPAROA_OP_CONV2D)
      wk = conv_work(in.n, in.h, in.w, in.c, op.c_out, op.kh, op.kw, out.h, out.w, op.groups);
    else if (op.kind == SPAROA_OP_FC)
      wk = fc_work(in.n, in.h * in.w * in.c, op.c_out);
    else if (op.kind == SPAROA_OP_ATTENTION)
      wk = attention_work(in.n, in.h * in.w, in.c / 3);
    sparoa_record& r = records[i];
    fill_stats(&r.stats, (uint64_t)(in.n * in.h * in.w * in.c), nnz[(size_t)op.input], wk, (int)in.n,
               (int)in.c, (int)in.h, (int)in.w, paths[(size_t)i]);
    r.output = act(i + 1);
    r.out_shape[0] = out.n;
    r.out_shape[1] = out.h;
    r.out_shape[2] = out.w;
    r.out_shape[3] = out.c;
    r.out_occ = &ctx->graph_occ[(size_t)i + 1];
  }
  return SPAROA_OK;
}

}  // extern "C"
