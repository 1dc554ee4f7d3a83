// dptq_device.cuh -- sm_103a device primitives used by the quantized-linear kernels:
// mbarriers with bounded waits, bulk (TMA) copies, tcgen05 MMA / TMEM access, PDL.
// Everything is inline PTX written for this library; no CUTLASS.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

namespace dptq {

// ------------------------------------------------------------------ tracing
// Built with -DDPTQ_TRACE (a separate library, see build.py), kernels record
// %globaltimer stamps per CTA at fixed slots of a 256-entry row of the buffer set by
// dptq_trace_set(); otherwise the trace points compile to nothing.
#ifdef DPTQ_TRACE
// One copy per translation unit; dptq_trace_set() sets the GEMM's.
static __device__ unsigned long long* g_dptq_trace = nullptr;
__device__ __forceinline__ unsigned long long trace_now() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
#ifdef DPTQ_TRACE_CLOCKS
// Stamps in SM cycles (cheap); the entry stamp also records %globaltimer (slot 0) and the
// cycle counter (slot 255) so that CTAs can be put on one time axis.
#define DPTQ_TRACE_POINT(buf, slot) \
  do {                              \
    if (buf) (buf)[blockIdx.x * 256 + (slot)] = (unsigned long long)clock64(); \
  } while (0)
#define DPTQ_TRACE_ENTRY(buf)                                                        \
  do {                                                                               \
    if (buf) {                                                                       \
      (buf)[blockIdx.x * 256 + 255] = (unsigned long long)clock64();                \
      (buf)[blockIdx.x * 256] = ::dptq::trace_now();                                \
    }                                                                                \
  } while (0)
#else
#define DPTQ_TRACE_POINT(buf, slot) \
  do {                              \
    if (buf) (buf)[blockIdx.x * 256 + (slot)] = ::dptq::trace_now(); \
  } while (0)
#define DPTQ_TRACE_ENTRY(buf) DPTQ_TRACE_POINT(buf, 0)
#endif
#define DPTQ_TRACE_VALUE(buf, slot, v) \
  do {                                 \
    if (buf) (buf)[blockIdx.x * 256 + (slot)] = (unsigned long long)(v); \
  } while (0)
#define DPTQ_TRACE_BUF() ::dptq::g_dptq_trace
#define DPTQ_TRACE_CLOCK(buf, slot) \
  do {                              \
    if (buf) (buf)[blockIdx.x * 256 + (slot)] = (unsigned long long)clock64(); \
  } while (0)
#else
#define DPTQ_TRACE_CLOCK(buf, slot) \
  do {                              \
  } while (0)
#define DPTQ_TRACE_POINT(buf, slot) \
  do {                              \
  } while (0)
#define DPTQ_TRACE_VALUE(buf, slot, v) \
  do {                                 \
  } while (0)
#define DPTQ_TRACE_BUF() nullptr
#define DPTQ_TRACE_ENTRY(buf) \
  do {                        \
  } while (0)
#endif

// Device error codes written to the library's error word (host maps them to status).
enum DeviceError : int {
  kDevOk = 0,
  kDevTimeoutFull = 0x101,     // waited too long for a bulk copy to land
  kDevTimeoutConv = 0x102,     // MMA waited too long for converted weights
  kDevTimeoutEmpty = 0x103,    // producer waited too long for a free stage
  kDevTimeoutTmemFull = 0x104, // epilogue waited too long for an accumulator
  kDevTimeoutTmemEmpty = 0x105,
  kDevTimeoutDrain = 0x106,
  kDevTimeoutGrid = 0x107,     // grid-wide phase barrier did not complete
  kDevTimeoutRowMax = 0x108,   // a row's parts did not all post their maxima
};

// ------------------------------------------------------------------ debug checks
// Built with -DDPTQ_DEBUG (a separate library, see build.py), DPTQ_CHECK(cond, err, site)
// tests the index arithmetic of a global access: when cond is false it records
// kDevBoundsCheck + site in the error word (the first failure wins) and evaluates to
// false, so that the caller skips the access.  Otherwise it is the constant true and the
// check compiles to nothing.  No check traps.
constexpr int kDevBoundsCheck = 0x200;
#ifdef DPTQ_DEBUG
#define DPTQ_CHECK(cond, err, site) \
  ((cond) ? true : (atomicCAS((err), 0, ::dptq::kDevBoundsCheck + (site)), false))
#else
#define DPTQ_CHECK(cond, err, site) true
#endif

// About one second at the GB300's ~2 GHz SM clock: any single wait longer than this
// means the pipeline is broken, so the kernel records an error and unwinds instead of
// spinning forever.
constexpr long long kWaitTimeoutCycles = 2000000000LL;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// ------------------------------------------------------------------ mbarrier
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait for the phase of `parity` to complete.  Returns false if the CTA-wide
// abort flag is raised or the wait times out after `limit` cycles (then the flag is
// raised and `code` is recorded in the global error word).
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          int* err, int code, long long limit = kWaitTimeoutCycles) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    __nanosleep(20);   // yield issue slots to the warps doing work
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) {
      *abort_flag = 1;
      atomicCAS(err, 0, code);
      return false;
    }
  }
}

// The same wait for a whole, converged warp: every lane polls, the result is the same
// for all lanes, and lane 0 decides a time-out.  The phase waited on must not be able to
// advance twice while the warp polls (true for every ring here: its next phase needs an
// action of this warp first).
__device__ __forceinline__ bool mbar_wait_warp(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                               int* err, int code, long long limit = kWaitTimeoutCycles) {
  if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
  const long long t0 = clock64();
  while (true) {
    if (__all_sync(0xffffffffu, mbar_try_wait(bar, parity))) return true;
    __nanosleep(20);
    int stop = 0;
    if ((threadIdx.x & 31) == 0) stop = *abort_flag ? 1 : (clock64() - t0 > limit ? 2 : 0);
    stop = __shfl_sync(0xffffffffu, stop, 0);
    if (stop) {
      if (stop == 2 && (threadIdx.x & 31) == 0) {
        *abort_flag = 1;
        atomicCAS(err, 0, code);
      }
      return false;
    }
  }
}

// One lane of a converged warp (the lowest) gets true.  Single-thread tcgen05 and bulk
// copy issue is much faster from an elected lane of a warp whose control flow is uniform
// than from a thread that runs its loop alone.
__device__ __forceinline__ bool elect_one() {
  uint32_t p = 0;
  asm volatile("{\n\t.reg .pred P;\n\telect.sync _|P, 0xffffffff;\n\tselp.b32 %0, 1, 0, P;\n\t}\n" : "=r"(p));
  return p != 0;
}

// ------------------------------------------------------------------ bulk copies (TMA engine)
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
// Contiguous global -> shared copy completing on `bar` (both addresses 16-byte aligned,
// bytes a multiple of 16).
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}

// Bring `bytes` of global memory at `src` into L2 without copying it anywhere (both
// 16-byte aligned / a multiple of 16); no completion is tracked.
__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(src), "r"(bytes) : "memory");
}

// ------------------------------------------------------------------ tcgen05 / TMEM
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Orders this thread's generic-proxy view of global memory (e.g. data another CTA
// published, acquired here) before its later async-proxy (bulk copy) accesses.
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, FP8 operands (kind::f8f6f4), fp32 accumulate.
__device__ __forceinline__ void mma_f8(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// D[tmem] (+)= A[tmem] * B[smem]^T: A read from tensor memory (one row per lane, four
// FP8 K-elements per 32-bit column, lowest K in the lowest byte).
__device__ __forceinline__ void mma_f8_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], [%1], %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive once on `bar` when every MMA issued so far by this thread has completed.
__device__ __forceinline__ void mma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

// Shared-memory matrix descriptor: K-major operand in the 128-byte swizzle layout
// (8-row x 128-byte atoms, rows 128 B apart, atoms 1024 B apart; base 1024-aligned).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu)   // start address >> 4
         | ((uint64_t)1 << 16)                 // leading byte offset (unused for SW128 K-major)
         | ((uint64_t)(1024 >> 4) << 32)       // stride byte offset: 8-row atom pitch
         | ((uint64_t)1 << 46)                 // descriptor version for tcgen05
         | ((uint64_t)2 << 61);                // swizzle mode: 128-byte
}

// Instruction descriptor: kind::f8f6f4, A = B = E4M3, D = F32, both K-major, M = 128.
__host__ __device__ constexpr uint32_t idesc_e4m3_m128(int n) {
  return (1u << 4)                        // D format F32
         | (0u << 7) | (0u << 10)         // A, B format E4M3
         | ((uint32_t)(n >> 3) << 17)     // N / 8
         | ((uint32_t)(128 >> 4) << 24);  // M / 16
}

// 32 TMEM lanes (one per thread of the warp) x 16 consecutive 32-bit columns.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
        "=r"(r[15])
      : "r"(taddr));
}
// 32 TMEM lanes (one per thread) x 32 consecutive 32-bit columns, from registers.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
      "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]), "r"(r[16]),
      "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]), "r"(r[24]),
      "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}
// 32 TMEM lanes (one per thread) x 16 consecutive 32-bit columns, from registers.
__device__ __forceinline__ void tmem_st16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// The same wait, tied to the registers of one load, so that no use of them can be
// scheduled before it (used when another load is issued before these are consumed).
__device__ __forceinline__ void tmem_ld_wait_regs(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                 "+r"(r[15])
               :
               : "memory");
}

// ------------------------------------------------------------------ PDL
// GPU-scope acquire load and acquire-release add (split-tile arrival counters).
__device__ __forceinline__ uint32_t ld_acquire_gpu(const uint32_t* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ uint32_t atom_add_acq_rel_gpu(uint32_t* p, uint32_t v) {
  uint32_t old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// Vector fp32 reduction into global memory (performed at L2, no return value).
__device__ __forceinline__ void red_add_v4_f32(float* p, float a, float b, float c, float d) {
  asm volatile("red.relaxed.gpu.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(a), "f"(b), "f"(c), "f"(d)
               : "memory");
}

// Release-add: this thread's earlier writes, and those it has synchronized with (a CTA
// barrier), are visible at GPU scope before the addition; no return value.
__device__ __forceinline__ void release_add_gpu(uint32_t* p, uint32_t v) {
  asm volatile("fence.acq_rel.gpu;\n\tred.relaxed.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

}  // namespace dptq
