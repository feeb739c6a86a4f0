// Device-side building blocks shared by the libsparoa kernels (sm_103a).
//
//  * PTX wrappers: mbarrier, TMA (cp.async.bulk.tensor), cp.async, tcgen05
//    (alloc / mma / commit / ld), proxy fences, named barriers.
//  * Bounded waits: every spin on an mbarrier gives up after kWaitLimitNs,
//    records an error bit in the context's device flag and lets the CTA
//    unwind, so a broken pipeline never hangs the GPU.
//  * Occupancy emission: every kernel that writes a bf16 activation builds, per
//    128-row x 64-column tile, a shared-memory bitmap (one 64-bit word per row,
//    bit c = element (r, c) is non-zero) and flushes it into the Eq. 1 count
//    and occupancy bitmaps of the output (Sec. 3.1 sparsity).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace sparoa {

// Bounded waits give up after about a second of SM clock cycles (the default;
// a context can set another limit, which its kernels receive as a parameter).
constexpr long long kWaitLimitCycles = 1ll << 31;

enum ErrBits : uint32_t {
  kErrTimeoutFull = 1u,
  kErrTimeoutEmpty = 2u,
  kErrTimeoutAcc = 4u,
};

// Occupancy outputs of a [R, C] bf16 tensor (mirrors sparoa_occupancy).
struct OccDev {
  unsigned long long* nnz;
  uint32_t* col_nnz;
  uint32_t* tile_nnz;
  unsigned long long* row_bm;
  uint32_t* blk_mask;
  int64_t R;
  int32_t C;
  int32_t W64;  // words per row of row_bm
  int32_t C32;  // words per 128-row block of blk_mask
};

// Inputs of the on-device dispatch decision.
struct DispatchDev {
  const unsigned long long* in_nnz;  // Eq. 1 count of the operator's input
  unsigned long long numel;
  double s_thr;
  int32_t fpb_ok;     // host: intensity >= c_thr
  int32_t force;      // 0 rule, 1 dense, 2 zero-skip
  int32_t* path_out;  // nullable; written once by CTA (0,0,0) thread 0
};

// The threshold rule, in IEEE double (path 1 = dense, 2 = zero-skip), for an
// input with `nnz` non-zeros.
__device__ __forceinline__ int decide_path_count(const DispatchDev& d, unsigned long long nnz) {
  if (d.force == 1) return 1;
  if (d.force == 2) return 2;
  const double zeros = (double)(d.numel - nnz);
  const double bound = __dmul_rn(d.s_thr, (double)d.numel);
  if (zeros >= bound) return 2;
  return d.fpb_ok ? 1 : 2;
}

__device__ __forceinline__ int decide_path(const DispatchDev& d) {
  if (d.force == 1) return 1;
  if (d.force == 2) return 2;
  return decide_path_count(d, *d.in_nnz);
}

__device__ __forceinline__ void record_path(const DispatchDev& d, int path) {
  if (d.path_out && blockIdx.x == 0 && blockIdx.y == 0 && blockIdx.z == 0 && threadIdx.x == 0)
    *d.path_out = path;
}

// bf16 zero test on the bit pattern: +0 and -0 are zero, everything else not.
__device__ __forceinline__ bool bf16_nz(uint16_t b) { return (b & 0x7FFFu) != 0; }

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// ---------------------------------------------------------------------------
// mbarrier
// ---------------------------------------------------------------------------
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// try_wait that suspends the thread in hardware until the phase completes or
// about `hint_ns` nanoseconds pass, so waiting warps leave the issue slots to
// the warps doing work on the same scheduler.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

// Wait for the phase with the given parity to complete.  Waiting threads are
// suspended by the hardware between polls (woken when the phase completes);
// the cycle counter and the CTA abort flag are checked every 16 polls.  Gives
// up after `limit` cycles (then it records `bit` in *err and raises *abort) or
// once another role of the CTA raised *abort; either way it returns false.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, uint32_t* err,
                                          volatile int* abort, uint32_t bit,
                                          long long limit = kWaitLimitCycles) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (uint32_t n = 1;; ++n) {
    if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if ((n & 15u) == 0u) {
      if (*abort) return false;
      if (clock64() - t0 > limit) {
        atomicOr(err, bit);
        *abort = 1;
        return false;
      }
    }
  }
}

// Non-blocking test of the phase with the given parity.
__device__ __forceinline__ bool mbar_test_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}

// mbar_wait for short waits on the critical path of a single issuing thread:
// polls without being suspended between polls (a suspended thread is woken
// some time after the phase completes), with the same limit and abort rule.
__device__ __forceinline__ bool mbar_wait_spin(uint32_t bar, uint32_t parity, uint32_t* err,
                                               volatile int* abort, uint32_t bit,
                                               long long limit = kWaitLimitCycles) {
  if (mbar_test_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (uint32_t n = 1;; ++n) {
    if (mbar_test_wait(bar, parity)) return true;
    if ((n & 255u) == 0u) {
      if (*abort) return false;
      if (clock64() - t0 > limit) {
        atomicOr(err, bit);
        *abort = 1;
        return false;
      }
    }
  }
}

// After an abort: wait, at most `limit` cycles and whatever the abort flag
// says, for a phase that asynchronous work already issued by this CTA (TMA
// copies into its shared memory, MMAs into its tensor memory) completes, so
// that the CTA does not release those resources while they are written.
__device__ __forceinline__ bool mbar_drain(uint32_t bar, uint32_t parity, long long limit) {
  if (mbar_test_wait(bar, parity)) return true;
  const long long t0 = clock64();
  for (uint32_t n = 1;; ++n) {
    if (mbar_try_wait_sleep(bar, parity, 2000u)) return true;
    if ((n & 15u) == 0u && clock64() - t0 > limit) return false;
  }
}

// Fault injection for tests of the error paths (IgemmArgs::fault): the MMA
// issuer never signals the first accumulator, so the epilogue's bounded wait
// runs out and the call reports a timeout.
constexpr int kFaultSkipFirstAccCommit = 1;

// ---------------------------------------------------------------------------
// TMA and cp.async
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, uint32_t bar, int x,
                                            int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(x), "r"(y), "r"(bar)
      : "memory");
}

// Shared -> global tensor stores (bulk-group completion).
__device__ __forceinline__ void tma_store_2d(const void* tmap, uint32_t src, int x, int y) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(src), "r"(x), "r"(y)
               : "memory");
}
__device__ __forceinline__ void tma_store_4d(const void* tmap, uint32_t src, int c0, int c1, int c2,
                                             int c3) {
  asm volatile(
      "cp.async.bulk.tensor.4d.global.shared::cta.bulk_group [%0, {%2, %3, %4, %5}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(tmap)),
      "r"(src), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
      : "memory");
}
__device__ __forceinline__ void bulk_commit() {
  asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// Wait until at most N committed store groups still read their shared source.
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void bulk_wait_all() {
  asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tmap)) : "memory");
}

// 16-byte async copy global -> shared; src_bytes 0 writes 16 zero bytes.
__device__ __forceinline__ void cp_async_16(uint32_t dst, const void* src, uint32_t src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
               "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Programmatic dependent launch.  Every kernel of the library runs its
// on-chip prologue (barrier init, TMEM allocation, tensor-map prefetch), then
// pdl_wait(): the grid launched before it on the stream has completed and its
// memory is visible.  No global memory is read or written before that wait.
// pdl_trigger() right after lets the next grid start its own prologue while
// this one works.  Both are no-ops for a launch without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Make generic-proxy writes to shared memory visible to the async proxy
// (tensor cores / TMA).
// Pull the 128-byte line holding p into L1 (no register result; a hint).
__device__ __forceinline__ void prefetch_l1(const void* p) {
  asm volatile("prefetch.global.L1 [%0];" ::"l"(p));
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Named barrier over `count` threads (whole warps).
__device__ __forceinline__ void named_bar_sync(int id, int count) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// OR of `pred` over the `count` threads of named barrier `id`.
__device__ __forceinline__ bool named_bar_or(int id, int count, bool pred) {
  uint32_t out;
  asm volatile(
      "{\n\t.reg .pred pi, po;\n\t"
      "setp.ne.u32 pi, %1, 0;\n\t"
      "bar.red.or.pred po, %2, %3, pi;\n\t"
      "selp.u32 %0, 1, 0, po;\n\t}"
      : "=r"(out)
      : "r"((uint32_t)pred), "r"(id), "r"(count)
      : "memory");
  return out != 0;
}

// ---------------------------------------------------------------------------
// tcgen05 (5th-generation tensor cores, accumulators in tensor memory)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 inputs, fp32 accumulate).
// Volatile (ordered with the barrier / commit asm) but without a memory
// clobber: the operands are read by the tensor cores, not by this thread.
__device__ __forceinline__ void tc_mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate));
}

// Arrive once on `bar` when every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

// Load 16 consecutive fp32 columns of this thread's TMEM lane.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32"
      " {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Issue a load of 32 consecutive fp32 columns of this thread's TMEM lane;
// the registers are valid after tmem_wait_ld().
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32"
      " {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]),
        "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]),
        "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]),
        "=r"(r[31])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// Wait for the loads into r[]; the registers are operands so that no use of
// them can be scheduled before the wait.
__device__ __forceinline__ void tmem_wait_ld32(uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.wait::ld.sync.aligned;"
      : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]),
        "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]),
        "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]), "+r"(r[17]), "+r"(r[18]),
        "+r"(r[19]), "+r"(r[20]), "+r"(r[21]), "+r"(r[22]), "+r"(r[23]), "+r"(r[24]),
        "+r"(r[25]), "+r"(r[26]), "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]),
        "+r"(r[31]));
}

// Shared-memory vector load / store that stay ordered with the other volatile
// asm (barriers, fences) but do not make the compiler reload unrelated memory.
__device__ __forceinline__ float4 lds_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr));
  return v;
}
__device__ __forceinline__ void sts_u4(uint32_t addr, const uint4& v) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w));
}

// 32 x 32 bit-matrix transpose across a warp: lane i holds row i on entry
// (bit j = element (i, j)) and column i on exit (bit j = element (j, i)).
// Five butterfly stages exchange ever smaller blocks between lane pairs.
__device__ __forceinline__ uint32_t warp_transpose32(uint32_t x) {
  const int lane = threadIdx.x & 31;
  const uint32_t masks[5] = {0x0000FFFFu, 0x00FF00FFu, 0x0F0F0F0Fu, 0x33333333u, 0x55555555u};
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    const int sft = 16 >> k;
    const uint32_t m = masks[k];
    const uint32_t y = __shfl_xor_sync(0xffffffffu, x, sft);
    x = (lane & sft) ? ((x & ~m) | ((y >> sft) & m)) : ((x & m) | ((y << sft) & ~m));
  }
  return x;
}

// Shared-memory matrix descriptor for a K-major operand tile written with the
// 64-byte swizzle: rows of 32 bf16 (64 B), 8-row core-matrix groups 512 B apart.
__device__ __forceinline__ uint64_t smem_desc_sw64(uint32_t addr) {
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFF);        // start address
  d |= (uint64_t)(16 >> 4) << 16;                // leading byte offset (unused here)
  d |= (uint64_t)(512 >> 4) << 32;               // stride byte offset: 8 rows * 64 B
  d |= (uint64_t)1 << 46;                        // descriptor version (sm_100 family)
  d |= (uint64_t)4 << 61;                        // layout: 64-byte swizzle
  return d;
}

// K-major operand tiles with BK bf16 of K per row: BK = 32 uses the 64-byte
// swizzle (8-row groups 512 B apart), BK = 64 the 128-byte swizzle (1024 B).
template <int BK>
__device__ __forceinline__ uint64_t smem_desc_kmajor(uint32_t addr) {
  static_assert(BK == 32 || BK == 64, "BK");
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFF);           // start address
  d |= (uint64_t)(16 >> 4) << 16;                   // leading byte offset (unused here)
  d |= (uint64_t)((BK * 2 * 8) >> 4) << 32;         // stride byte offset: 8 rows
  d |= (uint64_t)1 << 46;                           // descriptor version (sm_100 family)
  d |= (uint64_t)(BK == 32 ? 4 : 2) << 61;          // layout: 64- or 128-byte swizzle
  return d;
}

// Byte offset of 16-byte chunk j of row r in a BK-wide swizzled tile (the
// layout TMA writes with the matching CU_TENSOR_MAP_SWIZZLE_*): the chunk
// index is XORed with the row's position inside the swizzle period.
template <int BK>
__device__ __forceinline__ uint32_t swz_offset(int r, int j) {
  if (BK == 32) return (uint32_t)(r * 64 + ((j ^ ((r >> 1) & 3)) << 4));
  return (uint32_t)(r * 128 + ((j ^ (r & 7)) << 4));
}

// Instruction descriptor: kind::f16, A = B = bf16, D = fp32, both K-major.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
  return (1u << 4)                         // D format f32
         | (1u << 7)                       // A format bf16
         | (1u << 10)                      // B format bf16
         | ((uint32_t)(N >> 3) << 17)      // N / 8
         | ((uint32_t)(M >> 4) << 24);     // M / 16
}

// Byte offset of 16-byte chunk j (0..3) of row r in a 64-byte-swizzled tile
// (the layout TMA writes with CU_TENSOR_MAP_SWIZZLE_64B): address bits [4,6)
// are XORed with bits [7,9).
__device__ __forceinline__ uint32_t sw64_offset(int r, int j) {
  return (uint32_t)(r * 64 + ((j ^ ((r >> 1) & 3)) << 4));
}

// ---------------------------------------------------------------------------
// Epilogue math
// ---------------------------------------------------------------------------
struct EpiDev {
  const float* bias;   // [C]
  const float* bn;     // [4][C]
  float eps;
  int32_t act;
  const __nv_bfloat16* residual;  // same layout as the output
};

// Per-channel affine form of bias + batch norm: v * scale + shift.
__device__ __forceinline__ void epi_affine(const EpiDev& e, int C, int c, float& scale,
                                           float& shift) {
  const float b = e.bias ? e.bias[c] : 0.f;
  if (e.bn) {
    const float g = e.bn[c], beta = e.bn[C + c], mean = e.bn[2 * C + c], var = e.bn[3 * C + c];
    scale = g * rsqrtf(var + e.eps);
    shift = (b - mean) * scale + beta;
  } else {
    scale = 1.f;
    shift = b;
  }
}

// 8 bf16 values (one 16-byte chunk) to floats.
__device__ __forceinline__ void unpack8(const uint4& u, float (&f)[8]) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 t = __bfloat1622float2(h[j]);
    f[2 * j] = t.x;
    f[2 * j + 1] = t.y;
  }
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

// GELU in the tanh form of Hendrycks and Gimpel, 0.5 v (1 + tanh(sqrt(2/pi)
// (v + 0.044715 v^3))), with the hardware tanh approximation: within about
// 1e-3 of the exact form v * Phi(v), below the bf16 spacing of the result.
__device__ __forceinline__ float gelu_f(float v) {
  const float u = 0.7978845608028654f * fmaf(0.044715f * v, v * v, v);
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(u));
  return 0.5f * v * (1.f + t);
}

// Packed fp32 pairs for the fma.rn.f32x2 instruction (two independent
// fp32 FMAs, each rounded to nearest like fmaf).
typedef unsigned long long f2_t;  // two fp32 values (low: even channel)

__device__ __forceinline__ f2_t f2(float lo, float hi) {
  f2_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ void f2_split(f2_t v, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
__device__ __forceinline__ f2_t ffma2(f2_t a, f2_t b, f2_t c) {
  f2_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
// bit 0 / bit 16 set where the low / high bf16 of w is non-zero (any bit but
// the sign): adding 0x7FFF to a 15-bit magnitude carries into bit 15 exactly
// when the magnitude is not zero, and never out of its 16-bit half
__device__ __forceinline__ uint32_t nz_pairs(uint32_t w) {
  return (((w & 0x7FFF7FFFu) + 0x7FFF7FFFu) >> 15) & 0x00010001u;
}

// Two fp32 values through the activation to a bf16 pair (round to nearest
// even), `lo` in the low half; ReLU is applied by the conversion itself.
// ReLU6 clamps after the rounding: min(round(relu(v)), 6) = round(min(relu(v),
// 6)) because rounding is monotonic and 6 is a bf16 value.
template <int ACT>
__device__ __forceinline__ uint32_t act_pack2(float lo, float hi) {
  if (ACT == 3) {
    lo = gelu_f(lo);
    hi = gelu_f(hi);
  }
  uint32_t d;
  if (ACT == 1 || ACT == 2)
    asm("cvt.rn.relu.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  else
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  if (ACT == 2) asm("min.bf16x2 %0, %0, %1;" : "+r"(d) : "r"(0x40C040C0u));  // 6.0 in both halves
  return d;
}

__device__ __forceinline__ float epi_act(float v, int act) {
  if (act == 1) return v > 0.f ? v : 0.f;
  if (act == 2) return v > 0.f ? (v < 6.f ? v : 6.f) : 0.f;
  if (act == 3) return gelu_f(v);
  return v;
}


}  // namespace sparoa
