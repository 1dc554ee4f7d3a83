// static_scratch.cu -- dptq_qlinear_static: the quantized linear layer for callers that
// cannot allocate device memory when they call it.
//
// dptq_qlinear grows a per-device scratch with cudaMalloc on first use.  Some callers
// must not allocate at call time: runtimes whose own memory pool owns every byte of the
// device, or hosts that forbid cudaMalloc once they have started serving.  This entry
// point runs the same two kernels (rotate + quantize, then the GEMM) with their scratch
// in one file-scope device array of fixed size, so it never calls cudaMalloc, cudaFree
// or an allocating library routine.
#include <cstdint>
#include <mutex>
#include <string>

#include <cuda_runtime.h>

#include "../../include/dptq.h"
#include "dptq_internal.h"

using namespace dptq;

namespace {

// Limits of the static scratch: up to 32 tokens, K up to 16384, 256 CTAs.
constexpr int kStaticMaxM = 32;
constexpr int kStaticMaxKPad = 16384;
constexpr int kStaticMaxGrid = 256;
constexpr int kStaticMaxNT = 32;   // token tile the GEMM picks for M <= 32

// Regions of the array (each a multiple of 256 bytes).
constexpr size_t kActOff = 0;                                                     // E4M3 operand planes
constexpr size_t kActBytes = (size_t)2 * kStaticMaxKPad * kStaticMaxM;           // 1 MiB
constexpr size_t kSaOff = kActOff + kActBytes;                                    // token scales
constexpr size_t kSaBytes = 256;
constexpr size_t kWsOff = kSaOff + kSaBytes;                                      // split-tile sums
constexpr size_t kWsBytes = (size_t)kStaticMaxGrid * kStaticMaxNT * 128 * sizeof(int32_t);   // 4 MiB
constexpr size_t kCntOff = kWsOff + kWsBytes;                                     // arrival counters
constexpr size_t kCntBytes = (size_t)kStaticMaxGrid * sizeof(uint32_t);
constexpr size_t kErrOff = kCntOff + kCntBytes;                                   // device error word
constexpr size_t kErrBytes = 256;
constexpr size_t kStaticBytes = kErrOff + kErrBytes;

}  // namespace

// The scratch itself (about 5 MiB): every GPU that loads the library holds it until the
// process exits.  In host code this name is only a host-side stand-in; kernels get the
// device address that cudaGetSymbolAddress returns.
static __device__ __align__(256) unsigned char g_dptq_static_scratch[kStaticBytes];

namespace {

struct StaticState {
  bool ready = false;
  unsigned char* base = nullptr;   // device address of g_dptq_static_scratch
  int num_sms = 0;
};
constexpr int kMaxDevices = 64;
std::mutex g_static_mu;
StaticState g_static_state[kMaxDevices];

dptq_status static_fail(dptq_status st, const std::string& m) {
  set_error_message(m);
  return st;
}

// Once per device, with that device current: look up the array's device address and
// zero the parts that must start at zero (split-tile sums, counters, error word).  The
// kernels leave those parts zeroed again after every call that completes.
dptq_status static_setup(int dev, StaticState** out) {
  if (dev < 0 || dev >= kMaxDevices) return static_fail(DPTQ_ERR_UNSUPPORTED, "device index above 63");
  std::lock_guard<std::mutex> lk(g_static_mu);
  StaticState& st = g_static_state[dev];
  if (!st.ready) {
    void* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&ptr, g_dptq_static_scratch);
    if (e != cudaSuccess)
      return static_fail(DPTQ_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    e = cudaDeviceGetAttribute(&st.num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess)
      return static_fail(DPTQ_ERR_CUDA, std::string("cudaDeviceGetAttribute: ") + cudaGetErrorString(e));
    e = cudaMemset(static_cast<unsigned char*>(ptr) + kWsOff, 0, kWsBytes + kCntBytes + kErrBytes);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return static_fail(DPTQ_ERR_CUDA, std::string("cudaMemset: ") + cudaGetErrorString(e));
    st.base = static_cast<unsigned char*>(ptr);
    st.ready = true;
  }
  *out = &st;
  return DPTQ_OK;
}

bool pow2(int v) { return v > 0 && (v & (v - 1)) == 0; }

}  // namespace

namespace dptq {
// A bounded wait that gave up inside dptq_qlinear_static leaves its error word, and
// possibly split-tile sums and arrival counters, in the fixed array; every later call
// would start from those.  dptq_last_device_error calls this (after synchronizing the
// device) to report the word and return the array to its clean state.  No allocation.
cudaError_t static_scratch_check_reset(int dev, int* word) {
  *word = 0;
  if (dev < 0 || dev >= kMaxDevices) return cudaSuccess;
  std::lock_guard<std::mutex> lk(g_static_mu);
  const StaticState& st = g_static_state[dev];
  if (!st.ready) return cudaSuccess;
  cudaError_t e = cudaMemcpy(word, st.base + kErrOff, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess || *word == 0) return e;
  e = cudaMemset(st.base + kWsOff, 0, kWsBytes + kCntBytes + kErrBytes);
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  return e;
}
}  // namespace dptq

extern "C" dptq_status dptq_qlinear_static(dptq_handle h, const void* x_fp16, int M, int bits, void* out_fp16,
                                           void* stream) {
  if (!h) return static_fail(DPTQ_ERR_INVALID_ARG, "null handle");
  if (bits != 4 && bits != 8) return static_fail(DPTQ_ERR_INVALID_ARG, "bits must be 4 or 8");
  if (M < 0) return static_fail(DPTQ_ERR_INVALID_ARG, "M must be >= 0");
  if (M > kStaticMaxM)
    return static_fail(DPTQ_ERR_UNSUPPORTED, "dptq_qlinear_static: M above the static limit of 32 tokens");
  if (h->K_pad > kStaticMaxKPad)
    return static_fail(DPTQ_ERR_UNSUPPORTED, "dptq_qlinear_static: K above the static limit of 16384");
  if (M == 0) return DPTQ_OK;
  if (!x_fp16 || !out_fp16) return static_fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return static_fail(DPTQ_ERR_CUDA, "cudaGetDevice failed");
  if (dev != h->device)
    return static_fail(DPTQ_ERR_INVALID_ARG, "handle belongs to another device than the current one");
  StaticState* st = nullptr;
  dptq_status s = static_setup(dev, &st);
  if (s != DPTQ_OK) return s;

  const int B = h->had_block;
  const int K = h->K;
  if (!pow2(B) || B > 4096) return static_fail(DPTQ_ERR_UNSUPPORTED, "bad had_block");
  const int nfull = K / B, tail = K % B;
  if (tail != 0 && !pow2(tail)) return static_fail(DPTQ_ERR_UNSUPPORTED, "bad Hadamard tail");
  int log2B = 0, log2T = 0;
  while ((1 << log2B) < B) ++log2B;
  while (tail && (1 << log2T) < tail) ++log2T;

  const int grid_cap = st->num_sms < kStaticMaxGrid ? st->num_sms : kStaticMaxGrid;
  GemmPlan plan;
  if (!plan_gemm(M, h->N, h->K_pad, bits, grid_cap, plan) || plan.nt > kStaticMaxNT || plan.grid > kStaticMaxGrid)
    return static_fail(DPTQ_ERR_UNSUPPORTED, "dptq_qlinear_static: shape outside the static scratch");

  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  float* sa = reinterpret_cast<float*>(st->base + kSaOff);
  uint8_t* act = st->base + kActOff;

  RQArgs a{};
  a.x = static_cast<const __half*>(x_fp16);
  a.rows_in = M;
  a.rows_out = plan.M_pad;
  a.K = K;
  a.KB = h->KB;
  a.B = B;
  a.log2B = log2B;
  a.nfull = nfull;
  a.tail = tail;
  a.log2T = log2T;
  a.chunk = 4096;
  const double r2 = 0.70710678118654752440;
  a.c_hi = (float)r2;
  a.c_lo = (float)(r2 - (double)a.c_hi);
  a.bits = bits;
  a.scales = sa;
  a.signs = h->signs;
  a.out = act;
  cudaError_t e = launch_rotate_quant(kRQAct, a, cs, true);
  if (e != cudaSuccess) return static_fail(DPTQ_ERR_CUDA, std::string("rotate_quant launch: ") + cudaGetErrorString(e));

  GemmArgs& g = plan.args;
  g.wt = h->wt;
  g.act = act;
  g.sa = sa;
  g.sw = h->sw;
  g.out = static_cast<__half*>(out_fp16);
  g.out_vec = (reinterpret_cast<uintptr_t>(out_fp16) & 15u) == 0;
  g.acc_out = nullptr;
  g.ws = reinterpret_cast<int32_t*>(st->base + kWsOff);
  g.counters = reinterpret_cast<uint32_t*>(st->base + kCntOff);
  g.err = reinterpret_cast<int*>(st->base + kErrOff);
  e = launch_gemm(plan, cs, true);
  if (e != cudaSuccess) return static_fail(DPTQ_ERR_CUDA, std::string("qgemm launch: ") + cudaGetErrorString(e));
  return DPTQ_OK;
}
