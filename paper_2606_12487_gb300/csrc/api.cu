// api.cu -- the C ABI of include/dptq.h: argument checks, the layer handle, the
// per-device scratch, and the launch sequence of each call.  No compute happens here;
// every step of the path runs in the kernels of rotate_quant.cu and qgemm.cu.
#include <cmath>
#include <cstdint>
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <atomic>
#include <map>
#include <mutex>
#include <set>
#include <utility>
#include <string>
#include <vector>

#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "../../include/dptq.h"
#include "dptq_internal.h"

using namespace dptq;

namespace {

thread_local std::string g_msg;

dptq_status fail(dptq_status st, const std::string& m) {
  g_msg = m;
  return st;
}
dptq_status cuda_fail(cudaError_t e, const char* where) {
  g_msg = std::string(where) + ": " + cudaGetErrorString(e);
  return e == cudaErrorMemoryAllocation ? DPTQ_ERR_OOM : DPTQ_ERR_CUDA;
}
#define DPTQ_CUDA(call, where)                      \
  do {                                              \
    cudaError_t e_ = (call);                        \
    if (e_ != cudaSuccess) return cuda_fail(e_, where); \
  } while (0)

bool is_pow2(int v) { return v > 0 && (v & (v - 1)) == 0; }

bool is_prime_int(int v) {
  if (v < 2) return false;
  for (int d = 2; d * d <= v; ++d)
    if (v % d == 0) return false;
  return true;
}

// A tail block of r elements is r = p 2^k: p = 1 for a power of two; otherwise p is the
// smallest Paley order (odd part of r times 2^m, m >= 2, with p - 1 prime) that divides r,
// and the tail's Hadamard matrix is H_p (x) H_(2^k) with H_p from Paley's first
// construction.  False when r is neither.
bool tail_factor(int r, int& p, int& k) {
  if (r <= 0) return false;
  if (is_pow2(r)) {
    p = 1;
    k = 0;
    while ((1 << k) < r) ++k;
    return true;
  }
  int tz = 0;
  while (((r >> tz) & 1) == 0) ++tz;
  const int odd = r >> tz;
  for (int m = 2; m <= tz; ++m) {
    if (is_prime_int((odd << m) - 1)) {
      p = odd << m;
      k = tz - m;
      return true;
    }
  }
  return false;
}

// Block layout of R along K: nfull blocks of B then a tail (or none) that is a power of
// two or a Paley order times a power of two.
bool hadamard_layout(int K, int B, int& nfull, int& tail, int& log2B) {
  if (!is_pow2(B) || K <= 0) return false;
  nfull = K / B;
  tail = K % B;
  int p, k;
  if (tail != 0 && !tail_factor(tail, p, k)) return false;
  log2B = 0;
  while ((1 << log2B) < B) ++log2B;
  return true;
}

// Elements per rotation pass: whole blocks, at least 4096 elements when K allows.
int rq_chunk(int K, int B) {
  int c = B;
  while (c < 4096 && c < K) c += B;
  return c < K ? c : K;
}

// Whether K's tail block is a power of two (or absent); the fused decode launch and the
// whole-row kernel handle only those.
bool pow2_tail(int K, int B) { return K % B == 0 || is_pow2(K % B); }

dptq_status check_shape(int K, int B, int& nfull, int& tail, int& log2B) {
  if (K % 32 != 0) return fail(DPTQ_ERR_UNSUPPORTED, "K must be a multiple of 32");
  if (B > 4096) return fail(DPTQ_ERR_UNSUPPORTED, "had_block above 4096 is not supported");
  if (!hadamard_layout(K, B, nfull, tail, log2B))
    return fail(DPTQ_ERR_UNSUPPORTED,
                "K must split into blocks of had_block (a power of two) plus a tail that is a power of two or a "
                "Paley order times a power of two");
  int p = 1, k = 0;
  if (tail != 0 && !is_pow2(tail)) {
    tail_factor(tail, p, k);
    if (p > 256) return fail(DPTQ_ERR_UNSUPPORTED, "the tail block's Paley order is above 256");
    // The tail must lie in the last 4096-element rotation pass.
    if (nfull * B < ((K - 1) / 4096) * 4096)
      return fail(DPTQ_ERR_UNSUPPORTED, "a non-power-of-two tail must lie in the last 4096 elements of K");
  }
  if (rotate_quant_smem(K, rq_chunk(K, B)) > kSmemPerBlock)
    return fail(DPTQ_ERR_UNSUPPORTED, "K and had_block exceed the shared memory of one CTA");
  return DPTQ_OK;
}

RQArgs make_rq(const void* x, int rows_in, int rows_out, int K, int KB, int B, int nfull, int tail, int log2B,
               int bits, float* scales, void* out) {
  RQArgs a{};
  a.x = static_cast<const __half*>(x);
  a.rows_in = rows_in;
  a.rows_out = rows_out;
  a.K = K;
  a.KB = KB;
  a.B = B;
  a.log2B = log2B;
  a.nfull = nfull;
  a.tail = tail;
  a.log2T = 0;
  a.tail_p = 1;
  a.tail_j = 0;
  int p = 1, k = 0;
  if (tail && tail_factor(tail, p, k)) {
    a.log2T = k;
    a.tail_p = p;
    if (p > 1) {   // y = S 2^-24 / sqrt(p 2^k) = S 2^-(24 + k/2) / sqrt(p 2^(k mod 2))
      const double t = 1.0 / std::sqrt((double)p * (double)(1 << (k & 1)));
      a.tail_j = k >> 1;
      a.t_hi = (float)t;
      a.t_lo = (float)(t - (double)a.t_hi);
    }
  }
  a.chunk = rq_chunk(K, B);
  const double r2 = 1.0 / std::sqrt(2.0);
  a.c_hi = (float)r2;
  a.c_lo = (float)(r2 - (double)a.c_hi);
  a.bits = bits;
  a.scales = scales;
  a.out = out;
  return a;
}

// Per-device scratch shared by the online calls: E4M3 activation planes, per-token
// scales, split-tile partial sums and their counters, and the device error word.
// Activation planes and scales grow on demand.  A buffer that growth supersedes is never
// freed: work enqueued earlier, or captured into a CUDA graph, may still read or write
// it, so it stays allocated (in `retired`) until the process exits.  Growth is geometric
// (at least doubling), so the retired buffers together hold less than the live ones.
struct Scratch {
  uint8_t* act = nullptr;
  size_t act_bytes = 0;
  float* sa = nullptr;
  size_t sa_count = 0;
  int32_t* ws = nullptr;
  // [SMs] split-tile arrivals, [2] fused-launch grid counters, then (128-byte aligned)
  // the row-maximum slots of the fused launch's row parts, [64][kRowMaxStride]
  uint32_t* counters = nullptr;
  size_t counter_words = 0;
  uint32_t* gsync = nullptr;
  uint32_t* pmax = nullptr;
  int* err = nullptr;
  int num_sms = 0;
  std::vector<std::pair<void*, size_t>> retired;   // superseded act / sa buffers, still allocated
};
std::mutex g_mu;
std::map<int, Scratch> g_scratch;

bool capturing(cudaStream_t s) {
  cudaStreamCaptureStatus st = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &st) != cudaSuccess) return false;
  return st != cudaStreamCaptureStatusNone;
}

constexpr int kMaxNT = 256;
// Rows of up to 16384 elements take the fused launch (each of a row's four parts rotates
// at most 4096 of them).
constexpr int kFusedMaxKPad = 16384;
// Counter words: split-tile arrivals and grid counters, then the row-maximum slots, one
// 128-byte line per row (only the parts of one row poll a line).
size_t pmax_offset(int sms) { return ((size_t)sms + 2 + 31) & ~(size_t)31; }
size_t counter_words(int sms) { return pmax_offset(sms) + (size_t)64 * kRowMaxStride; }

// Every device allocation of the library goes through here.  Host-side fault injection
// for tests of the out-of-memory path: with DPTQ_FAULT_ALLOC=n (n >= 1) in the
// environment, the n-th allocation the library attempts in this process fails as
// cudaErrorMemoryAllocation without calling cudaMalloc.
cudaError_t dev_malloc(void** p, size_t bytes) {
  static const long long fail_at = [] {
    const char* v = std::getenv("DPTQ_FAULT_ALLOC");
    return v ? std::atoll(v) : 0LL;
  }();
  static long long n = 0;
  if (fail_at > 0 && ++n == fail_at) {
    *p = nullptr;
    return cudaErrorMemoryAllocation;
  }
  return cudaMalloc(p, bytes);
}

// Make sure the device's scratch holds `act_bytes` of activation planes and `sa_count`
// scales.  Growth allocates, so it is refused while `s` is being captured.
dptq_status ensure_scratch(int dev, size_t act_bytes, size_t sa_count, cudaStream_t s, Scratch** out) {
  std::lock_guard<std::mutex> lk(g_mu);
  Scratch& sc = g_scratch[dev];
  const bool grow_act = act_bytes > sc.act_bytes;
  const bool grow_sa = sa_count > sc.sa_count;
  const bool first = sc.err == nullptr;
  if ((grow_act || grow_sa || first) && capturing(s))
    return fail(DPTQ_ERR_UNSUPPORTED, "scratch must grow during stream capture: call dptq_reserve first");
  if (first) {
    int sms = 0;
    DPTQ_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev), "cudaDeviceGetAttribute");
    const size_t ws_bytes = (size_t)sms * kMaxNT * 128 * sizeof(int32_t);
    int32_t* ws = nullptr;
    uint32_t* counters = nullptr;
    int* err = nullptr;
    cudaError_t e = dev_malloc(reinterpret_cast<void**>(&ws), ws_bytes);
    if (e == cudaSuccess) e = dev_malloc(reinterpret_cast<void**>(&counters), sizeof(uint32_t) * counter_words(sms));
    if (e == cudaSuccess) e = dev_malloc(reinterpret_cast<void**>(&err), sizeof(int));
    if (e == cudaSuccess) e = cudaMemset(ws, 0, ws_bytes);
    if (e == cudaSuccess) e = cudaMemset(counters, 0, sizeof(uint32_t) * counter_words(sms));
    if (e == cudaSuccess) e = cudaMemset(err, 0, sizeof(int));
    if (e != cudaSuccess) {   // nothing has used these yet: release them and stay uninitialized
      if (ws) cudaFree(ws);
      if (counters) cudaFree(counters);
      if (err) cudaFree(err);
      return cuda_fail(e, "scratch allocation");
    }
    sc.counter_words = counter_words(sms);
    sc.pmax = counters + pmax_offset(sms);
    // DPTQ_MAX_GRID=n caps the CTAs of a GEMM launch (tuning experiments; default: the
    // device's SMs).
    if (const char* v = std::getenv("DPTQ_MAX_GRID")) {
      const int cap = std::atoi(v);
      if (cap > 0 && cap < sms) sms = cap;
    }
    sc.num_sms = sms;
    sc.ws = ws;
    sc.counters = counters;
    sc.gsync = counters + sms;
    sc.err = err;
  }
  if (grow_act) {
    const size_t bytes = std::max(act_bytes, 2 * sc.act_bytes);
    void* p = nullptr;
    DPTQ_CUDA(dev_malloc(&p, bytes), "cudaMalloc(act)");
    if (sc.act) sc.retired.emplace_back(sc.act, sc.act_bytes);
    sc.act = static_cast<uint8_t*>(p);
    sc.act_bytes = bytes;
  }
  if (grow_sa) {
    const size_t count = std::max(sa_count, 2 * sc.sa_count);
    void* p = nullptr;
    DPTQ_CUDA(dev_malloc(&p, sizeof(float) * count), "cudaMalloc(sa)");
    if (sc.sa) sc.retired.emplace_back(sc.sa, sizeof(float) * sc.sa_count);
    sc.sa = static_cast<float*>(p);
    sc.sa_count = count;
  }
  *out = &sc;
  return DPTQ_OK;
}

dptq_status current_device(int* dev) {
  DPTQ_CUDA(cudaGetDevice(dev), "cudaGetDevice");
  return DPTQ_OK;
}

dptq_status check_handle(dptq_handle h, int* dev) {
  if (!h) return fail(DPTQ_ERR_INVALID_ARG, "null handle");
  dptq_status st = current_device(dev);
  if (st != DPTQ_OK) return st;
  if (*dev != h->device) return fail(DPTQ_ERR_INVALID_ARG, "handle belongs to another device than the current one");
  return DPTQ_OK;
}

// GEMM + epilogue from the E4M3 planes already in scratch.
dptq_status run_gemm(dptq_handle h, const GemmPlan& plan0, const uint8_t* act, const float* sa, void* out,
                     int32_t* acc, Scratch* sc, cudaStream_t s) {
  GemmPlan plan = plan0;
  GemmArgs& g = plan.args;
  g.wt = h->wt;
  g.act = act;
  g.sa = sa;
  g.sw = h->sw;
  g.out = static_cast<__half*>(out);
  g.out_vec = (reinterpret_cast<uintptr_t>(out) & 15u) == 0;
  g.acc_out = acc;
  g.ws = sc->ws;
  g.counters = sc->counters;
  g.gsync = sc->gsync;
  g.err = sc->err;
  g.wait_cycles = wait_cycles_setting();
  if (plan.fused) {
    g.rq_shortfall = take_rows_shortfall();
    g.pre_stages = pre_stages_setting();
  }
  DPTQ_CUDA(launch_gemm(plan, s, true), "qgemm launch");
  return DPTQ_OK;
}

}  // namespace

namespace dptq {
bool pdl_allowed() {
  static const bool on = [] {
    const char* v = std::getenv("DPTQ_PDL");
    return !(v && v[0] == '0');
  }();
  return on;
}

// NVTX ranges named after the entry points, around every call that launches work, for
// timelines in NVIDIA's tools (DPTQ_NVTX=1; off by default, when a range costs one load).
bool nvtx_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("DPTQ_NVTX");
    return v && v[0] == '1';
  }();
  return on;
}
struct NvtxRange {
  const bool on;
  explicit NvtxRange(const char* name) : on(nvtx_enabled()) {
    if (on) nvtxRangePushA(name);
  }
  ~NvtxRange() {
    if (on) nvtxRangePop();
  }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

bool fused_allowed() {
  static const bool on = [] {
    const char* v = std::getenv("DPTQ_FUSED");
    return !(v && v[0] == '0');
  }();
  return on;
}

bool l2_prefetch_allowed() {
  static const bool on = [] {
    const char* v = std::getenv("DPTQ_L2PF");
    return !(v && v[0] == '0');
  }();
  return on;
}

// Decode grids of one CTA per whole weight tile when the tiles fit the SMs (default), or,
// with DPTQ_DECODE_WHOLE_TILES=0, every SM with split tiles (tuning).
bool decode_whole_tiles() {
  static const bool on = [] {
    const char* v = std::getenv("DPTQ_DECODE_WHOLE_TILES");
    return !(v && v[0] == '0');
  }();
  return on;
}

// A8 prefill tiles: 192 tokens with the widened weights in tensor memory (default), or,
// with DPTQ_A8_TILE128=1, 128 tokens with the weights widened into shared memory.
bool a8_tile128() {
  static const bool on = [] {
    const char* v = std::getenv("DPTQ_A8_TILE128");
    return v && v[0] == '1';
  }();
  return on;
}

// Weight stages a fused launch requests before its token rows are ready (DPTQ_PRE_STAGES,
// a tuning knob; default 4: of 2, 3, 4 and 6 the fastest LLaMA-2-7B decode stack at
// M = 32).
int pre_stages_setting() {
  static const int v = [] {
    const char* e = std::getenv("DPTQ_PRE_STAGES");
    const int n = e ? std::atoi(e) : 4;
    return n < 1 ? 1 : n;
  }();
  return v;
}

long long wait_cycles_setting() {
  static const long long v = [] {
    const char* e = std::getenv("DPTQ_WAIT_CYCLES");
    const long long c = e ? std::atoll(e) : 0LL;
    return c > 0 ? c : 2000000000LL;
  }();
  return v;
}

int take_rows_shortfall() {
  static std::atomic<int> left{[] {
    const char* e = std::getenv("DPTQ_TEST_ROWS_SHORTFALL");
    return e ? std::atoi(e) : 0;
  }()};
  return left.exchange(0);
}

cudaError_t ensure_max_dyn_smem_impl(const void* fn) {
  // One entry per (kernel, device) whose ceiling is already raised.
  static std::mutex mu;
  static std::set<std::pair<const void*, int>> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lk(mu);
  if (done.count({fn, dev})) return cudaSuccess;
  // The ceiling is the device's opt-in maximum per block less the kernel's static shared
  // memory.
  int optin = 0;
  e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (e != cudaSuccess) return e;
  cudaFuncAttributes fa{};
  e = cudaFuncGetAttributes(&fa, fn);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, optin - (int)fa.sharedSizeBytes);
  if (e == cudaSuccess) done.insert({fn, dev});
  return e;
}

bool rows_kernel_allowed() {
  static const bool on = [] {
    const char* v = std::getenv("DPTQ_ROWS_KERNEL");
    return !(v && v[0] == '0');
  }();
  return on;
}

// Record the message returned by dptq_last_error_message for this thread.
void set_error_message(const std::string& m) { g_msg = m; }
}  // namespace dptq

extern "C" {

const char* dptq_status_str(dptq_status s) {
  switch (s) {
    case DPTQ_OK: return "ok";
    case DPTQ_ERR_INVALID_ARG: return "invalid argument";
    case DPTQ_ERR_UNSUPPORTED: return "unsupported shape";
    case DPTQ_ERR_CUDA: return "CUDA error";
    case DPTQ_ERR_OOM: return "out of device memory";
    case DPTQ_ERR_TIMEOUT: return "device wait timed out";
  }
  return "unknown status";
}

const char* dptq_last_error_message(void) { return g_msg.c_str(); }

namespace {
// Shared body of dptq_pack_weights and dptq_pack_weights_rh (signs_host null: plain).
dptq_status pack_weights_impl(const void* W_fp16, int N, int K, int had_block, const int8_t* signs_host,
                              int w_on_device, dptq_handle* out) {
  if (!W_fp16 || !out) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  *out = nullptr;
  if (N <= 0 || K <= 0 || had_block <= 0) return fail(DPTQ_ERR_INVALID_ARG, "sizes must be positive");
  if (N % 16 != 0) return fail(DPTQ_ERR_UNSUPPORTED, "N must be a multiple of 16");
  int nfull, tail, log2B;
  dptq_status st = check_shape(K, had_block, nfull, tail, log2B);
  if (st != DPTQ_OK) return st;
  int dev;
  if ((st = current_device(&dev)) != DPTQ_OK) return st;

  dptq_linear* h = new dptq_linear{};
  h->device = dev;
  h->N = N;
  h->K = K;
  h->K_pad = round_up(K, kKPad);
  h->KB = h->K_pad / kKBlock;
  h->N_pad = round_up(N, 128);
  h->had_block = had_block;
  if (signs_host != nullptr) {
    for (int k = 0; k < K; ++k)
      if (signs_host[k] != 1 && signs_host[k] != -1) {
        delete h;
        return fail(DPTQ_ERR_INVALID_ARG, "signs must be +1 or -1");
      }
  }
  const size_t wt_bytes = (size_t)(h->N_pad / 128) * h->KB * kWTileBytes;
  void* tmp = nullptr;
  cudaError_t e = dev_malloc(reinterpret_cast<void**>(&h->wt), wt_bytes);
  if (e == cudaSuccess) e = dev_malloc(reinterpret_cast<void**>(&h->sw), sizeof(float) * h->N_pad);
  if (e == cudaSuccess && signs_host != nullptr) {
    e = dev_malloc(reinterpret_cast<void**>(&h->signs), (size_t)h->K_pad);
    if (e == cudaSuccess) e = cudaMemset(h->signs, 1, (size_t)h->K_pad);
    if (e == cudaSuccess) e = cudaMemcpy(h->signs, signs_host, (size_t)K, cudaMemcpyHostToDevice);
  }
  const void* src = W_fp16;
  if (e == cudaSuccess && !w_on_device) {
    e = dev_malloc(&tmp, (size_t)N * K * 2);
    if (e == cudaSuccess) e = cudaMemcpy(tmp, W_fp16, (size_t)N * K * 2, cudaMemcpyHostToDevice);
    src = tmp;
  }
  if (e == cudaSuccess) {
    RQArgs a = make_rq(src, N, h->N_pad, K, h->KB, had_block, nfull, tail, log2B, 4, h->sw, h->wt);
    a.signs = h->signs;
    e = launch_rotate_quant(kRQWeights, a, 0, false);
  }
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (tmp) cudaFree(tmp);
  if (e != cudaSuccess) {
    dptq_destroy(h);
    return cuda_fail(e, "dptq_pack_weights");
  }
  *out = h;
  return DPTQ_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
}  // namespace

dptq_status dptq_pack_weights(const void* W_fp16, int N, int K, int had_block, int w_on_device, dptq_handle* out) {
  NvtxRange nvtx_range("dptq_pack_weights");
  return pack_weights_impl(W_fp16, N, K, had_block, nullptr, w_on_device, out);
}

dptq_status dptq_pack_weights_rh(const void* W_fp16, int N, int K, int had_block, const int8_t* signs_host,
                                 int w_on_device, dptq_handle* out) {
  NvtxRange nvtx_range("dptq_pack_weights_rh");
  if (!signs_host) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  return pack_weights_impl(W_fp16, N, K, had_block, signs_host, w_on_device, out);
}

dptq_status dptq_rotate_quant_act_rh(const void* x_fp16, int M, int K, int had_block, int bits,
                                     const int8_t* signs_dev, void* codes, float* scales, void* stream) {
  NvtxRange nvtx_range("dptq_rotate_quant_act_rh");
  if (bits != 4 && bits != 8) return fail(DPTQ_ERR_INVALID_ARG, "bits must be 4 or 8");
  if (M < 0 || K <= 0 || had_block <= 0) return fail(DPTQ_ERR_INVALID_ARG, "bad sizes");
  if (M == 0) return DPTQ_OK;
  if (!x_fp16 || !codes || !scales) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  if (signs_dev && !aligned16(signs_dev)) return fail(DPTQ_ERR_INVALID_ARG, "signs must be 16-byte aligned");
  int nfull, tail, log2B;
  dptq_status st = check_shape(K, had_block, nfull, tail, log2B);
  if (st != DPTQ_OK) return st;
  RQArgs a = make_rq(x_fp16, M, M, K, round_up(K, kKBlock) / kKBlock, had_block, nfull, tail, log2B, bits, scales,
                     codes);
  a.signs = signs_dev;
  DPTQ_CUDA(launch_rotate_quant(kRQPublic, a, static_cast<cudaStream_t>(stream), true), "rotate_quant launch");
  return DPTQ_OK;
}

dptq_status dptq_rotate_act_rh(const void* x_fp16, int M, int K, int had_block, const int8_t* signs_dev,
                               float* y_f32, void* stream) {
  NvtxRange nvtx_range("dptq_rotate_act_rh");
  if (M < 0 || K <= 0 || had_block <= 0) return fail(DPTQ_ERR_INVALID_ARG, "bad sizes");
  if (M == 0) return DPTQ_OK;
  if (!x_fp16 || !y_f32) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  if (signs_dev && !aligned16(signs_dev)) return fail(DPTQ_ERR_INVALID_ARG, "signs must be 16-byte aligned");
  int nfull, tail, log2B;
  dptq_status st = check_shape(K, had_block, nfull, tail, log2B);
  if (st != DPTQ_OK) return st;
  RQArgs a = make_rq(x_fp16, M, M, K, round_up(K, kKBlock) / kKBlock, had_block, nfull, tail, log2B, 4, nullptr,
                     y_f32);
  a.signs = signs_dev;
  DPTQ_CUDA(launch_rotate_quant(kRQY, a, static_cast<cudaStream_t>(stream), true), "rotate launch");
  return DPTQ_OK;
}

dptq_status dptq_rotate_quant_act(const void* x_fp16, int M, int K, int had_block, int bits, void* codes,
                                  float* scales, void* stream) {
  NvtxRange nvtx_range("dptq_rotate_quant_act");
  if (bits != 4 && bits != 8) return fail(DPTQ_ERR_INVALID_ARG, "bits must be 4 or 8");
  if (M < 0 || K <= 0 || had_block <= 0) return fail(DPTQ_ERR_INVALID_ARG, "bad sizes");
  if (M == 0) return DPTQ_OK;
  if (!x_fp16 || !codes || !scales) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  int nfull, tail, log2B;
  dptq_status st = check_shape(K, had_block, nfull, tail, log2B);
  if (st != DPTQ_OK) return st;
  RQArgs a = make_rq(x_fp16, M, M, K, round_up(K, kKBlock) / kKBlock, had_block, nfull, tail, log2B, bits, scales,
                     codes);
  DPTQ_CUDA(launch_rotate_quant(kRQPublic, a, static_cast<cudaStream_t>(stream), true), "rotate_quant launch");
  return DPTQ_OK;
}

dptq_status dptq_rotate_act(const void* x_fp16, int M, int K, int had_block, float* y_f32, void* stream) {
  NvtxRange nvtx_range("dptq_rotate_act");
  if (M < 0 || K <= 0 || had_block <= 0) return fail(DPTQ_ERR_INVALID_ARG, "bad sizes");
  if (M == 0) return DPTQ_OK;
  if (!x_fp16 || !y_f32) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  int nfull, tail, log2B;
  dptq_status st = check_shape(K, had_block, nfull, tail, log2B);
  if (st != DPTQ_OK) return st;
  RQArgs a = make_rq(x_fp16, M, M, K, round_up(K, kKBlock) / kKBlock, had_block, nfull, tail, log2B, 4, nullptr,
                     y_f32);
  DPTQ_CUDA(launch_rotate_quant(kRQY, a, static_cast<cudaStream_t>(stream), true), "rotate launch");
  return DPTQ_OK;
}

}  // extern "C"

namespace {

// Shape checks and scratch sizing shared by the qlinear entry points.
dptq_status prepare_qlinear(dptq_handle h, int M, int bits, cudaStream_t s, int* dev, GemmPlan* plan,
                            Scratch** sc) {
  if (bits != 4 && bits != 8) return fail(DPTQ_ERR_INVALID_ARG, "bits must be 4 or 8");
  if (M < 0) return fail(DPTQ_ERR_INVALID_ARG, "M must be >= 0");
  dptq_status st = check_handle(h, dev);
  if (st != DPTQ_OK) return st;
  if (M == 0) return DPTQ_OK;
  if ((st = ensure_scratch(*dev, 0, 0, s, sc)) != DPTQ_OK) return st;
  if (!plan_gemm(M, h->N, h->K_pad, bits, (*sc)->num_sms, *plan)) return fail(DPTQ_ERR_UNSUPPORTED, "no GEMM plan");
  const int planes = bits == 8 ? 2 : 1;
  return ensure_scratch(*dev, (size_t)planes * h->K_pad * plan->M_pad, plan->M_pad, s, sc);
}

dptq_status quantize_into_scratch(dptq_handle h, const void* x_fp16, int M, int bits, const GemmPlan& plan,
                                  Scratch* sc, cudaStream_t s) {
  int nfull, tail, log2B;
  dptq_status st = check_shape(h->K, h->had_block, nfull, tail, log2B);
  if (st != DPTQ_OK) return st;
  RQArgs a = make_rq(x_fp16, M, plan.M_pad, h->K, h->KB, h->had_block, nfull, tail, log2B, bits, sc->sa, sc->act);
  a.signs = h->signs;
  DPTQ_CUDA(launch_rotate_quant(kRQAct, a, s, true), "rotate_quant launch");
  return DPTQ_OK;
}

}  // namespace

extern "C" {

dptq_status dptq_qlinear(dptq_handle h, const void* x_fp16, int M, int bits, void* out_fp16, void* stream) {
  NvtxRange nvtx_range("dptq_qlinear");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int dev;
  GemmPlan plan;
  Scratch* sc = nullptr;
  dptq_status st = prepare_qlinear(h, M, bits, s, &dev, &plan, &sc);
  if (st != DPTQ_OK || M == 0) return st;
  if (!x_fp16 || !out_fp16) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  // Small M: one launch that rotates and quantizes the rows and runs the GEMM.
  GemmPlan fp;
  if (fused_allowed() && h->K_pad <= kFusedMaxKPad && pow2_tail(h->K, h->had_block) &&
      plan_gemm(M, h->N, h->K_pad, bits, sc->num_sms, fp, kRQPartSmemBytes) && fp.M_pad == plan.M_pad &&
      fp.M_pad <= 64 && fused_rotation_variant(h->K, h->had_block, h->K % h->had_block, fp.args.rq_np) >= 0) {
    int nfull, tail, log2B;
    if ((st = check_shape(h->K, h->had_block, nfull, tail, log2B)) != DPTQ_OK) return st;
    fp.args.rq = make_rq(x_fp16, M, fp.M_pad, h->K, h->KB, h->had_block, nfull, tail, log2B, bits, sc->sa, sc->act);
    fp.args.rq.signs = h->signs;
    fp.args.rq.np = fp.args.rq_np;
    fp.args.rq.pmax = sc->pmax;
    return run_gemm(h, fp, sc->act, sc->sa, out_fp16, nullptr, sc, s);
  }
  if ((st = quantize_into_scratch(h, x_fp16, M, bits, plan, sc, s)) != DPTQ_OK) return st;
  return run_gemm(h, plan, sc->act, sc->sa, out_fp16, nullptr, sc, s);
}

dptq_status dptq_qlinear_quantize(dptq_handle h, const void* x_fp16, int M, int bits, void* stream) {
  NvtxRange nvtx_range("dptq_qlinear_quantize");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int dev;
  GemmPlan plan;
  Scratch* sc = nullptr;
  dptq_status st = prepare_qlinear(h, M, bits, s, &dev, &plan, &sc);
  if (st != DPTQ_OK || M == 0) return st;
  if (!x_fp16) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  return quantize_into_scratch(h, x_fp16, M, bits, plan, sc, s);
}

dptq_status dptq_qlinear_gemm(dptq_handle h, int M, int bits, void* out_fp16, void* stream) {
  NvtxRange nvtx_range("dptq_qlinear_gemm");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int dev;
  GemmPlan plan;
  Scratch* sc = nullptr;
  dptq_status st = prepare_qlinear(h, M, bits, s, &dev, &plan, &sc);
  if (st != DPTQ_OK || M == 0) return st;
  if (!out_fp16) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  return run_gemm(h, plan, sc->act, sc->sa, out_fp16, nullptr, sc, s);
}

dptq_status dptq_qgemm_codes(dptq_handle h, const void* codes, const float* scales, int M, int bits, void* out_fp16,
                             int32_t* acc_i32, void* stream) {
  NvtxRange nvtx_range("dptq_qgemm_codes");
  if (bits != 4 && bits != 8) return fail(DPTQ_ERR_INVALID_ARG, "bits must be 4 or 8");
  if (M < 0) return fail(DPTQ_ERR_INVALID_ARG, "M must be >= 0");
  int dev;
  dptq_status st = check_handle(h, &dev);
  if (st != DPTQ_OK) return st;
  if (M == 0) return DPTQ_OK;
  if (!codes || !scales || !out_fp16) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Scratch* sc = nullptr;
  if ((st = ensure_scratch(dev, 0, 0, s, &sc)) != DPTQ_OK) return st;
  GemmPlan plan;
  if (!plan_gemm(M, h->N, h->K_pad, bits, sc->num_sms, plan)) return fail(DPTQ_ERR_UNSUPPORTED, "no GEMM plan");
  const int planes = bits == 8 ? 2 : 1;
  if ((st = ensure_scratch(dev, (size_t)planes * h->K_pad * plan.M_pad, 0, s, &sc)) != DPTQ_OK) return st;
  CodesArgs c{};
  c.codes = static_cast<const uint8_t*>(codes);
  c.M = M;
  c.M_pad = plan.M_pad;
  c.K = h->K;
  c.KB = h->KB;
  c.bits = bits;
  c.act = sc->act;
  DPTQ_CUDA(launch_codes_to_act(c, s), "codes_to_act launch");
  return run_gemm(h, plan, sc->act, scales, out_fp16, acc_i32, sc, s);
}

dptq_status dptq_kv4_quantize(const void* kv_fp16, int rows, int cols, int group, void* codes, float* scales,
                              void* stream) {
  NvtxRange nvtx_range("dptq_kv4_quantize");
  if (rows < 0 || cols <= 0 || group <= 0) return fail(DPTQ_ERR_INVALID_ARG, "bad sizes");
  if (rows == 0) return DPTQ_OK;
  if (!kv_fp16 || !codes || !scales) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(kv_fp16)) return fail(DPTQ_ERR_INVALID_ARG, "kv must be 16-byte aligned");
  if (group % 128 != 0 || group > 1024 || cols % group != 0)
    return fail(DPTQ_ERR_UNSUPPORTED, "group must be a multiple of 128 up to 1024 that divides cols");
  int dev;
  dptq_status st = current_device(&dev);
  if (st != DPTQ_OK) return st;
  int sms = 0;
  DPTQ_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev), "cudaDeviceGetAttribute");
  KvArgs a{static_cast<const __half*>(kv_fp16), rows, cols, group, static_cast<uint8_t*>(codes), scales};
  DPTQ_CUDA(launch_kv4(a, sms, static_cast<cudaStream_t>(stream)), "kv4 launch");
  return DPTQ_OK;
}

dptq_status dptq_sensitivity_policy(const float* x, const float* dx, int L, int T, int d, int bits, double eps,
                                    double tau_jr, double tau_snr, double* jr, double* snr, uint8_t* bits_out,
                                    void* stream) {
  NvtxRange nvtx_range("dptq_sensitivity_policy");
  if (bits != 4 && bits != 8) return fail(DPTQ_ERR_INVALID_ARG, "bits must be 4 or 8");
  if (L < 0 || T <= 0 || d <= 0 || !(eps >= 0.0)) return fail(DPTQ_ERR_INVALID_ARG, "bad sizes or eps");
  if (L == 0) return DPTQ_OK;
  if (!x || !dx || !jr || !snr || !bits_out) return fail(DPTQ_ERR_INVALID_ARG, "null pointer");
  if (!aligned16(x) || !aligned16(dx) || d % 4 != 0)
    return fail(DPTQ_ERR_INVALID_ARG, "x and dx must be 16-byte aligned and d a multiple of 4");
  int dev;
  dptq_status st = current_device(&dev);
  if (st != DPTQ_OK) return st;
  Scratch* sc = nullptr;
  st = ensure_scratch(dev, 0, 0, static_cast<cudaStream_t>(stream), &sc);
  if (st != DPTQ_OK) return st;
  PolicyArgs a{x, dx, L, T, d, bits, eps, tau_jr, tau_snr, jr, snr, bits_out, sc->err};
  DPTQ_CUDA(launch_policy(a, sc->num_sms, static_cast<cudaStream_t>(stream)), "policy launch");
  return DPTQ_OK;
}

dptq_status dptq_plan_info(int M, int N, int K, int bits, int num_sms, int fused, int* info, int info_len) {
  if (M < 1 || N < 1 || K < 1 || num_sms < 1) return fail(DPTQ_ERR_INVALID_ARG, "sizes must be >= 1");
  if (bits != 4 && bits != 8) return fail(DPTQ_ERR_INVALID_ARG, "bits must be 4 or 8");
  if (info == nullptr || info_len < DPTQ_PLAN_INFO_LEN) return fail(DPTQ_ERR_INVALID_ARG, "info too short");
  GemmPlan plan{};
  if (!plan_gemm(M, N, round_up(K, kKBlock), bits, num_sms, plan, fused ? kRQPartSmemBytes : 0))
    return fail(DPTQ_ERR_UNSUPPORTED, "no GEMM plan for this shape");
  const GemmArgs& g = plan.args;
  const long long sk = g.sk_iters;
  const int v[DPTQ_PLAN_INFO_LEN] = {plan.nt, plan.kps, plan.M_pad, plan.grid, plan.smem_bytes, g.stages,
                                     g.conv_slots, plan.a_tmem ? 1 : 0, g.nbuf, g.segs, g.seg_iters,
                                     (int)g.tmem_cols, (int)g.a_col0, g.KI, g.n_wtiles, g.m_tiles, g.dp_tiles,
                                     sk > 0x7fffffffLL ? 0x7fffffff : (int)sk, g.rq_np, plan.fused ? 1 : 0};
  for (int i = 0; i < DPTQ_PLAN_INFO_LEN; ++i) info[i] = v[i];
  return DPTQ_OK;
}

dptq_status dptq_reserve(int max_M, int max_K, int max_N) {
  NvtxRange nvtx_range("dptq_reserve");
  if (max_M < 0 || max_K < 0 || max_N < 0) return fail(DPTQ_ERR_INVALID_ARG, "sizes must be >= 0");
  int dev;
  dptq_status st = current_device(&dev);
  if (st != DPTQ_OK) return st;
  (void)max_N;
  // Rows of the widest token tile and of the 192-token prefill tile.
  const int m_res = max_M > 0 ? max_M : 1;
  const size_t M_pad = (size_t)std::max(round_up(m_res, kMaxNT), round_up(m_res, 192));
  const size_t K_pad = (size_t)round_up(max_K > 0 ? max_K : kKBlock, kKBlock);
  Scratch* sc = nullptr;
  st = ensure_scratch(dev, 2 * K_pad * M_pad, M_pad, 0, &sc);
  if (st != DPTQ_OK) return st;
  DPTQ_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
  return DPTQ_OK;
}

dptq_status dptq_get_packed(dptq_handle h, void* wq_host, float* sw_host) {
  int dev;
  dptq_status st = check_handle(h, &dev);
  if (st != DPTQ_OK) return st;
  if (sw_host) DPTQ_CUDA(cudaMemcpy(sw_host, h->sw, sizeof(float) * h->N, cudaMemcpyDeviceToHost), "cudaMemcpy(sw)");
  if (!wq_host) return DPTQ_OK;
  const size_t wt_bytes = (size_t)(h->N_pad / 128) * h->KB * kWTileBytes;
  std::vector<uint8_t> t(wt_bytes);
  DPTQ_CUDA(cudaMemcpy(t.data(), h->wt, wt_bytes, cudaMemcpyDeviceToHost), "cudaMemcpy(wt)");
  uint8_t* dst = static_cast<uint8_t*>(wq_host);
  for (int n = 0; n < h->N; ++n) {
    for (int k = 0; k < h->K; k += 2) {
      int code[2];
      for (int d = 0; d < 2; ++d) {
        const int kk = k + d;
        const int e = kk & 15;  // position in the 16-weight chunk
        const size_t chunk = (((size_t)(n >> 7) * h->KB + (kk >> 7)) * kWTileBytes) + ((kk & 127) >> 5) * 2048 +
                             (n & 127) * 16 + (((kk & 127) >> 4) & 1) * 8;
        const int word = e >> 3, i = e & 3, high = (e & 7) >= 4;
        const uint8_t byte = t[chunk + word * 4 + i];
        const int nib = high ? (byte >> 4) & 0xF : byte & 0xF;
        const int mag = nib & 7;
        code[d] = (nib & 8) ? -mag : mag;
      }
      dst[(size_t)n * (h->K / 2) + k / 2] = (uint8_t)((code[0] & 0xF) | ((code[1] & 0xF) << 4));
    }
  }
  return DPTQ_OK;
}

dptq_status dptq_get_shape(dptq_handle h, int* N, int* K, int* had_block) {
  if (!h) return fail(DPTQ_ERR_INVALID_ARG, "null handle");
  if (N) *N = h->N;
  if (K) *K = h->K;
  if (had_block) *had_block = h->had_block;
  return DPTQ_OK;
}

dptq_status dptq_last_device_error(dptq_handle h) {
  (void)h;
  int dev;
  dptq_status st = current_device(&dev);
  if (st != DPTQ_OK) return st;
  DPTQ_CUDA(cudaDeviceSynchronize(), "cudaDeviceSynchronize");
  int word = 0;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_scratch.find(dev);
    if (it != g_scratch.end() && it->second.err != nullptr) {
      Scratch& sc = it->second;
      DPTQ_CUDA(cudaMemcpy(&word, sc.err, sizeof(int), cudaMemcpyDeviceToHost), "cudaMemcpy(err)");
      if (word != 0) {
        // A wait gave up: clear the word, the split-tile sums and every counter (split-tile
        // arrivals, the fused launch's two grid counters and its row-maximum slots) the
        // aborted kernel may have left non-zero.
        DPTQ_CUDA(cudaMemset(sc.err, 0, sizeof(int)), "cudaMemset(err)");
        DPTQ_CUDA(cudaMemset(sc.ws, 0, (size_t)sc.num_sms * kMaxNT * 128 * sizeof(int32_t)), "cudaMemset(ws)");
        DPTQ_CUDA(cudaMemset(sc.counters, 0, sizeof(uint32_t) * sc.counter_words), "cudaMemset(counters)");
      }
    }
  }
  // The fixed scratch of dptq_qlinear_static keeps its own error word.
  int sword = 0;
  const cudaError_t e = static_scratch_check_reset(dev, &sword);
  if (e != cudaSuccess) return cuda_fail(e, "static scratch error word");
  if (word == 0) word = sword;
  if (word == 0) return DPTQ_OK;
  char buf[64];
  snprintf(buf, sizeof(buf), "device wait timed out (code 0x%x)", word);
  return fail(DPTQ_ERR_TIMEOUT, buf);
}

dptq_status dptq_scratch_buffers(void** ptrs, size_t* bytes, int* allocated, int max, int* count) {
  if (count == nullptr || max < 0 || (max > 0 && (ptrs == nullptr || bytes == nullptr || allocated == nullptr)))
    return fail(DPTQ_ERR_INVALID_ARG, "null pointer or negative max");
  int dev;
  dptq_status st = current_device(&dev);
  if (st != DPTQ_OK) return st;
  std::vector<std::pair<void*, size_t>> list;
  {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_scratch.find(dev);
    if (it != g_scratch.end()) {
      const Scratch& sc = it->second;
      if (sc.act) list.emplace_back(sc.act, sc.act_bytes);
      if (sc.sa) list.emplace_back(sc.sa, sizeof(float) * sc.sa_count);
      list.insert(list.end(), sc.retired.rbegin(), sc.retired.rend());
    }
  }
  *count = (int)list.size();
  for (int i = 0; i < (int)list.size() && i < max; ++i) {
    ptrs[i] = list[i].first;
    bytes[i] = list[i].second;
    cudaPointerAttributes at{};
    const cudaError_t e = cudaPointerGetAttributes(&at, list[i].first);
    allocated[i] = (e == cudaSuccess && at.type == cudaMemoryTypeDevice) ? 1 : 0;
    if (e != cudaSuccess) (void)cudaGetLastError();
  }
  return DPTQ_OK;
}

void dptq_destroy(dptq_handle h) {
  if (!h) return;
  if (h->wt) cudaFree(h->wt);
  if (h->sw) cudaFree(h->sw);
  if (h->signs) cudaFree(h->signs);
  delete h;
}

}  // extern "C"
