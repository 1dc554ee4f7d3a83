// kv_policy.cu -- two kernels next to the quantized linear layer:
//   * the group-wise symmetric 4-bit KV-cache quantizer (Section 4.2: KV cache quantized
//     group-wise with group size 128), and
//   * the sensitive-layer policy: Jump Ratio and historical-feature SNR per layer
//     (Section 3.1, Eqs. 8-11) thresholded into the 8-bit layer set (Section 3.3,
//     Eq. 20; Algorithm 1 step 2).
// Both are HBM-bound streams over their inputs; the per-group / per-token quantizer is
// the same exact quantizer as the activation path (rotate_row.cuh).
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "dptq_device.cuh"
#include "dptq_internal.h"
#include "rotate_row.cuh"

namespace dptq {

// ------------------------------------------------------------------ KV4
// One warp per (row, group) at a time.  Lane l holds columns 4l .. 4l + 3 of each
// 128-column block of the group (J = group / 128 blocks, at most 8): one 8-byte load per
// block, the group's absmax by shuffles, then four codes per block packed into 2 bytes
// (the warp stores 64 contiguous bytes per block).
constexpr int kKvWarps = 8;

// Quantize the 4 values of one lane (raw fp16 bits), given the group's absmax, into 4
// nibbles (low nibble first).
__device__ __forceinline__ uint32_t kv4_codes(uint2 raw, float s, float r, bool nz) {
  const __half2 h0 = *reinterpret_cast<const __half2*>(&raw.x);
  const __half2 h1 = *reinterpret_cast<const __half2*>(&raw.y);
  const float y[4] = {__low2float(h0), __high2float(h0), __low2float(h1), __high2float(h1)};
  float c[4] = {0.f, 0.f, 0.f, 0.f};
  if (nz) quant_code4(y, s, r, -8.f, 7.f, c);
  uint32_t packed = 0;
#pragma unroll
  for (int e = 0; e < 4; ++e) packed |= ((uint32_t)(int)c[e] & 0xFu) << (4 * e);
  return packed;
}

__device__ __forceinline__ float absmax4(uint2 raw) {
  const __half2 h0 = *reinterpret_cast<const __half2*>(&raw.x);
  const __half2 h1 = *reinterpret_cast<const __half2*>(&raw.y);
  return fmaxf(fmaxf(fabsf(__low2float(h0)), fabsf(__high2float(h0))),
               fmaxf(fabsf(__low2float(h1)), fabsf(__high2float(h1))));
}

// Groups of 128 (the paper's size): kKvQuads sets of four consecutive groups per warp and
// iteration, all loads issued first, so that each SM keeps enough bytes in flight.
//   * The four groups' maxima are reduced by one transposed butterfly (6 exchanges, not
//     20): afterwards lane l holds the maximum of group 2 (l >> 4) + ((l >> 3) & 1), so
//     every lane forms one scale and reciprocal and lanes 0, 8, 16, 24 hand them out.
//   * Codes: |y / s| <= 7 (1 + 2^-22), so no code needs the clamp.  y r + 1.5 * 2^23,
//     rounded once (an fma), holds round(y r) in its low mantissa bits (two's
//     complement, ties to even); the nibble is those bits.  Where y r lies within 2^-15
//     of a half-integer, the IEEE quotient y / s decides instead (|y r - y / s| and
//     |fl(y / s) - y / s| are both below 2^-21, so elsewhere the two agree).
constexpr float kRoundMagic = 12582912.0f;   // 1.5 * 2^23
constexpr int kKvQuads = 2;

__global__ void __launch_bounds__(kKvWarps * 32) kv4_quantize_g128_kernel(const KvArgs a) {
  const int lane = threadIdx.x & 31;
  const int my_g = ((lane >> 4) << 1) | ((lane >> 3) & 1);
  const bool up16 = (lane & 16) != 0, up8 = (lane & 8) != 0;
  const long long ngroups = (long long)a.rows * (a.cols >> 7);   // groups are consecutive in memory
  const long long nitems = (ngroups + 4 * kKvQuads - 1) / (4 * kKvQuads);
  const long long nwarps = (long long)gridDim.x * kKvWarps;
  for (long long w = (long long)blockIdx.x * kKvWarps + (threadIdx.x >> 5); w < nitems; w += nwarps) {
    uint2 raws[4 * kKvQuads];
#pragma unroll
    for (int i = 0; i < 4 * kKvQuads; ++i) {
      const long long g = 4 * kKvQuads * w + i;
      raws[i] = g < ngroups ? __ldg(reinterpret_cast<const uint2*>(a.kv + (size_t)g * 128 + 4 * lane))
                            : make_uint2(0u, 0u);
    }
#pragma unroll
    for (int q = 0; q < kKvQuads; ++q) {
      const long long g0 = 4 * kKvQuads * w + 4 * q;
      if (g0 >= ngroups) break;
      const int ng = ngroups - g0 < 4 ? (int)(ngroups - g0) : 4;
      const uint2* raw = raws + 4 * q;
      float m[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) m[i] = absmax4(raw[i]);
      float k0 = up16 ? m[2] : m[0], k1 = up16 ? m[3] : m[1];
      k0 = fmaxf(k0, __shfl_xor_sync(0xffffffffu, up16 ? m[0] : m[2], 16));
      k1 = fmaxf(k1, __shfl_xor_sync(0xffffffffu, up16 ? m[1] : m[3], 16));
      float amax = fmaxf(up8 ? k1 : k0, __shfl_xor_sync(0xffffffffu, up8 ? k0 : k1, 8));
#pragma unroll
      for (int o = 4; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
      const float s_mine = __fdiv_rn(amax, 7.f);   // 0 for an all-zero group
      const float r_mine = amax > 0.f ? __frcp_rn(s_mine) : 0.f;
      if ((lane & 7) == 0 && my_g < ng) a.scales[g0 + my_g] = s_mine;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float s = __shfl_sync(0xffffffffu, s_mine, 8 * i);
        const float r = __shfl_sync(0xffffffffu, r_mine, 8 * i);
        const __half2 h0 = *reinterpret_cast<const __half2*>(&raw[i].x);
        const __half2 h1 = *reinterpret_cast<const __half2*>(&raw[i].y);
        const float y[4] = {__low2float(h0), __high2float(h0), __low2float(h1), __high2float(h1)};
        float tb[4];
        uint32_t nearm = 0;
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          tb[e] = __fmaf_rn(y[e], r, kRoundMagic);
          const float f = __fmaf_rn(y[e], r, -__fsub_rn(tb[e], kRoundMagic));
          nearm |= fabsf(f) >= 0.5f - 0x1p-15f ? (1u << e) : 0u;
        }
        if (__any_sync(0xffffffffu, nearm != 0u)) {
#pragma unroll
          for (int e = 0; e < 4; ++e)
            if ((nearm >> e) & 1u) tb[e] = __fadd_rn(rintf(__fdiv_rn(y[e], s)), kRoundMagic);
        }
        const uint32_t packed = (__float_as_uint(tb[0]) & 0xFu) | ((__float_as_uint(tb[1]) & 0xFu) << 4) |
                                ((__float_as_uint(tb[2]) & 0xFu) << 8) | ((__float_as_uint(tb[3]) & 0xFu) << 12);
        if (i < ng) reinterpret_cast<uint16_t*>(a.codes + (size_t)(g0 + i) * 64)[lane] = (uint16_t)packed;
      }
    }
  }
}

__global__ void __launch_bounds__(kKvWarps * 32) kv4_quantize_kernel(const KvArgs a) {
  const int lane = threadIdx.x & 31;
  const int J = a.group >> 7;
  const int ng = a.cols / a.group;
  const long long ngroups = (long long)a.rows * ng;
  const long long nwarps = (long long)gridDim.x * kKvWarps;
  for (long long w = (long long)blockIdx.x * kKvWarps + (threadIdx.x >> 5); w < ngroups; w += nwarps) {
    const int row = (int)(w / ng);
    const int g = (int)(w - (long long)row * ng);
    const size_t base = (size_t)row * a.cols + (size_t)g * a.group;
    const __half* src = a.kv + base;
    uint2 raw[8];
    float amax = 0.f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (j < J) {
        raw[j] = __ldg(reinterpret_cast<const uint2*>(src + 128 * j + 4 * lane));
        const __half2 h0 = *reinterpret_cast<const __half2*>(&raw[j].x);
        const __half2 h1 = *reinterpret_cast<const __half2*>(&raw[j].y);
        amax = fmaxf(amax, fmaxf(fmaxf(fabsf(__low2float(h0)), fabsf(__high2float(h0))),
                                 fmaxf(fabsf(__low2float(h1)), fabsf(__high2float(h1)))));
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
    const float s = __fdiv_rn(amax, 7.f);
    const bool nz = amax > 0.f;
    const float r = nz ? __frcp_rn(s) : 0.f;
    if (lane == 0) a.scales[(size_t)row * ng + g] = nz ? s : 0.f;
    uint16_t* dst = reinterpret_cast<uint16_t*>(a.codes + base / 2);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (j < J) {
        const __half2 h0 = *reinterpret_cast<const __half2*>(&raw[j].x);
        const __half2 h1 = *reinterpret_cast<const __half2*>(&raw[j].y);
        const float y[4] = {__low2float(h0), __high2float(h0), __low2float(h1), __high2float(h1)};
        float c[4] = {0.f, 0.f, 0.f, 0.f};
        if (nz) quant_code4(y, s, r, -8.f, 7.f, c);
        uint32_t packed = 0;
#pragma unroll
        for (int e = 0; e < 4; ++e) packed |= ((uint32_t)(int)c[e] & 0xFu) << (4 * e);
        dst[32 * j + lane] = (uint16_t)packed;   // columns 128 j + 4 lane .. + 3, low nibble first
      }
    }
  }
}

cudaError_t launch_kv4(const KvArgs& a, int num_sms, cudaStream_t s) {
  const long long ngroups = (long long)a.rows * (a.cols / a.group);
  const long long work = a.group == 128 ? (ngroups + 4 * kKvQuads - 1) / (4 * kKvQuads) : ngroups;   // warps' items
  long long blocks = (work + kKvWarps - 1) / kKvWarps;
  int per_sm = 8;
  if (a.group == 128) {   // one wave of resident CTAs
    const cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kv4_quantize_g128_kernel,
                                                                        kKvWarps * 32, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) per_sm = 1;
  }
  const long long cap = (long long)num_sms * per_sm;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  if (a.group == 128)
    kv4_quantize_g128_kernel<<<(unsigned)blocks, kKvWarps * 32, 0, s>>>(a);
  else
    kv4_quantize_kernel<<<(unsigned)blocks, kKvWarps * 32, 0, s>>>(a);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ policy
// Tokens of more than 4096 values: one CTA of 256 threads per (layer, token) at a time,
// with plain loads.  Thread t holds columns
// 4t + 1024 i of the token (float4 loads of x and dx).  Per element, in fp32:
//   |x|^2 and |dx|^2; u = fl(x + dx) as the quantizer's input (the fp32 sum);
//   the reconstruction error xhat - x = s c - dx - x = (s c - u) - (x + dx - u): the
//   first term by one fma, the second, the rounding residue of x + dx, exactly
//   (two-sum), so that no cancellation against |x| is lost.
// The three sums go per thread in fp32, across the CTA in fp64.  Thread 0 adds the
// token's JR and SNR terms to per-layer fp64 sums; a second kernel averages them and
// applies the thresholds.
constexpr int kPolThreads = 256;

__device__ __forceinline__ double block_sum_f64(double v, double* red, int tid) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();   // red is reused
  if ((tid & 31) == 0) red[tid >> 5] = v;
  __syncthreads();
  double t = 0.0;
#pragma unroll
  for (int w = 0; w < kPolThreads / 32; ++w) t += red[w];
  return t;
}

__global__ void __launch_bounds__(kPolThreads) policy_stats_kernel(const PolicyArgs a) {
  __shared__ double red[kPolThreads / 32];
  __shared__ float redf[kPolThreads / 32];
  const int tid = threadIdx.x;
  const int qmax = (1 << (a.bits - 1)) - 1;
  const float qmaxf = (float)qmax, qminf = (float)(-(1 << (a.bits - 1)));
  const long long items = (long long)a.L * a.T;
  for (long long it = blockIdx.x; it < items; it += gridDim.x) {
    const int l = (int)(it / a.T);
    const float* x = a.x + (size_t)it * a.d;
    const float* dx = a.dx + (size_t)it * a.d;
    // pass 1: norms and the quantizer's absmax
    float nx = 0.f, nd = 0.f, am = 0.f;
    for (int k = 4 * tid; k < a.d; k += 4 * kPolThreads) {
      const float4 xv = __ldg(reinterpret_cast<const float4*>(x + k));
      const float4 dv = __ldg(reinterpret_cast<const float4*>(dx + k));
      const float xs[4] = {xv.x, xv.y, xv.z, xv.w}, ds[4] = {dv.x, dv.y, dv.z, dv.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        nx = __fmaf_rn(xs[e], xs[e], nx);
        nd = __fmaf_rn(ds[e], ds[e], nd);
        am = fmaxf(am, fabsf(__fadd_rn(xs[e], ds[e])));
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, o));
    __syncthreads();
    if ((tid & 31) == 0) redf[tid >> 5] = am;
    __syncthreads();
    float amax = redf[0];
#pragma unroll
    for (int w = 1; w < kPolThreads / 32; ++w) amax = fmaxf(amax, redf[w]);
    const float s = __fdiv_rn(amax, qmaxf);
    const bool nzs = amax > 0.f;
    const float r = nzs ? __frcp_rn(s) : 0.f;
    // pass 2 (the token's 8d bytes are still in L1/L2): the reconstruction error
    float ne = 0.f;
    auto err4 = [&](const float4 xv, const float4 dv) {
      const float xs[4] = {xv.x, xv.y, xv.z, xv.w}, ds[4] = {dv.x, dv.y, dv.z, dv.w};
      float u[4], c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int e = 0; e < 4; ++e) u[e] = __fadd_rn(xs[e], ds[e]);
      if (nzs) quant_code4(u, s, r, qminf, qmaxf, c);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float bv = __fsub_rn(u[e], xs[e]);
        const float av = __fsub_rn(u[e], bv);
        const float res = __fadd_rn(__fsub_rn(xs[e], av), __fsub_rn(ds[e], bv));   // x + dx - u, exact
        const float err = __fsub_rn(__fmaf_rn(s, c[e], -u[e]), res);
        ne = __fmaf_rn(err, err, ne);
      }
    };
    for (int k = 4 * tid; k < a.d; k += 4 * kPolThreads)
      err4(__ldg(reinterpret_cast<const float4*>(x + k)), __ldg(reinterpret_cast<const float4*>(dx + k)));
    const double nx2 = block_sum_f64((double)nx, red, tid);
    const double nd2 = block_sum_f64((double)nd, red, tid);
    const double ne2 = block_sum_f64((double)ne, red, tid);
    if (tid == 0) {
      atomicAdd(a.jr + l, sqrt(nd2) / (sqrt(nx2) + a.eps));
      atomicAdd(a.snr + l, 10.0 * log10(nx2 / (ne2 + a.eps)));
    }
  }
}

// Tokens of up to 4096 values: the staged form.  Each CTA takes a contiguous range of
// (layer, token) items; bulk copies put whole tokens (x, then dx: 8d bytes) into a ring of
// kPolStages shared-memory stages, up to kPolStages tokens ahead.  Iteration j runs pass 2
// of token j - 1 (its quantizer is known) and pass 1 of token j on the same threads, then
// one barrier publishes the per-warp partials of both; the stage of token j - 1 is
// refilled right after that barrier.  The per-element arithmetic is that of the kernel
// above.  All sums are of non-negative terms and stay in fp32 up to the token (per thread
// 16 elements, then the warp's tree, then 8 warps: a relative error below 30 units of
// 2^-24).  Thread 0 records each finished token's three sums; every 32 tokens the lanes
// of warp 0 form the tokens' JR and SNR terms in parallel (fp32; the fp64 unit of this
// GPU is far slower) and add them per layer to the fp64 outputs, one atomic per layer.
constexpr int kPolStages = 3;
constexpr int kPolMaxStagedD = 4096;

// Warp 0, converged: token i of the batch (i < nb, first item `item0`) has its sums in
// tok[i]; adds its terms to the per-layer outputs.
__device__ __forceinline__ void pol_batch(const PolicyArgs& a, const float (*tok)[3], long long item0, int nb,
                                          int lane) {
  float jr = 0.f, snr = 0.f;
  int l = -1;
  if (lane < nb) {
    const float nx = tok[lane][0], nd = tok[lane][1], ne = tok[lane][2];
    const float eps = (float)a.eps;
    jr = __fdiv_rn(sqrtf(nd), __fadd_rn(sqrtf(nx), eps));
    snr = 10.f * log10f(__fdiv_rn(nx, __fadd_rn(ne, eps)));
    l = (int)((item0 + lane) / a.T);
  }
  unsigned left = __ballot_sync(0xffffffffu, lane < nb);
  while (left) {   // one pass per layer present in the batch (the batch's items are consecutive)
    const int l0 = __shfl_sync(0xffffffffu, l, __ffs(left) - 1);
    const bool in = l == l0 && lane < nb;
    float vj = in ? jr : 0.f, vs = in ? snr : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      vj += __shfl_xor_sync(0xffffffffu, vj, o);
      vs += __shfl_xor_sync(0xffffffffu, vs, o);
    }
    if (lane == 0) {
      atomicAdd(a.jr + l0, (double)vj);
      atomicAdd(a.snr + l0, (double)vs);
    }
    left &= ~__ballot_sync(0xffffffffu, in);
  }
}

__global__ void __launch_bounds__(kPolThreads) policy_stats_staged_kernel(const PolicyArgs a) {
  extern __shared__ __align__(128) uint8_t pol_smem[];
  __shared__ uint64_t full[kPolStages];
  __shared__ float part[2][4][kPolThreads / 32];   // [iteration parity][amax, |x|^2, |dx|^2, |err|^2][warp]
  __shared__ float tok[32][3];                      // finished tokens' |x|^2, |dx|^2, |err|^2
  __shared__ int abort_flag;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const long long n = (long long)a.L * a.T;
  const long long t0 = n * blockIdx.x / gridDim.x;
  const int cnt = (int)(n * (blockIdx.x + 1) / gridDim.x - t0);
  const uint32_t half_bytes = 4u * (uint32_t)a.d, stage_bytes = 8u * (uint32_t)a.d;
  const float qmaxf = (float)((1 << (a.bits - 1)) - 1), qminf = (float)(-(1 << (a.bits - 1)));
  if (tid == 0) {
    for (int i = 0; i < kPolStages; ++i) mbar_init(&full[i], 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  const uint64_t pol = l2_policy_evict_first();
  auto issue = [&](int k) {   // token t0 + k into stage k % kPolStages (one thread)
    uint8_t* st = pol_smem + (size_t)(k % kPolStages) * stage_bytes;
    uint64_t* bar = &full[k % kPolStages];
    fence_proxy_async_smem();   // the stage's earlier generic reads come before the copy's writes
    mbar_arrive_expect_tx(bar, stage_bytes);
    bulk_g2s(st, a.x + (size_t)(t0 + k) * a.d, half_bytes, bar, pol);
    bulk_g2s(st + half_bytes, a.dx + (size_t)(t0 + k) * a.d, half_bytes, bar, pol);
  };
  int issued = 0;   // tokens whose copies were issued (meaningful in warp 0)
  if (warp == 0) {
    issued = cnt < kPolStages ? cnt : kPolStages;
    if (elect_one())
      for (int k = 0; k < issued; ++k) issue(k);
    __syncwarp();
  }
  float s = 0.f, r = 0.f;
  bool nzs = false;
  float tok_nx = 0.f, tok_nd = 0.f;   // thread 0: sums of token j - 1
  for (int j = 0; j <= cnt; ++j) {
    float am = 0.f, nx = 0.f, nd = 0.f, ne = 0.f;
    if (j >= 1) {   // pass 2 of token j - 1
      const float* xs = reinterpret_cast<const float*>(pol_smem + (size_t)((j - 1) % kPolStages) * stage_bytes);
      const float* ds = xs + a.d;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int k = 4 * (tid + kPolThreads * i);
        if (k < a.d) {
          const float4 xv = *reinterpret_cast<const float4*>(xs + k);
          const float4 dv = *reinterpret_cast<const float4*>(ds + k);
          const float xe[4] = {xv.x, xv.y, xv.z, xv.w}, de[4] = {dv.x, dv.y, dv.z, dv.w};
          float u[4], c[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int e = 0; e < 4; ++e) u[e] = __fadd_rn(xe[e], de[e]);
          if (nzs) quant_code4(u, s, r, qminf, qmaxf, c);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float bv = __fsub_rn(u[e], xe[e]);
            const float av = __fsub_rn(u[e], bv);
            const float res = __fadd_rn(__fsub_rn(xe[e], av), __fsub_rn(de[e], bv));   // x + dx - u, exact
            const float err = __fsub_rn(__fmaf_rn(s, c[e], -u[e]), res);
            ne = __fmaf_rn(err, err, ne);
          }
        }
      }
    }
    if (j < cnt) {   // pass 1 of token j
      const int st = j % kPolStages;
      if (mbar_wait_warp(&full[st], (uint32_t)(j / kPolStages) & 1u, &abort_flag, a.err, kDevTimeoutFull)) {
        const float* xs = reinterpret_cast<const float*>(pol_smem + (size_t)st * stage_bytes);
        const float* ds = xs + a.d;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int k = 4 * (tid + kPolThreads * i);
          if (k < a.d) {
            const float4 xv = *reinterpret_cast<const float4*>(xs + k);
            const float4 dv = *reinterpret_cast<const float4*>(ds + k);
            const float xe[4] = {xv.x, xv.y, xv.z, xv.w}, de[4] = {dv.x, dv.y, dv.z, dv.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              nx = __fmaf_rn(xe[e], xe[e], nx);
              nd = __fmaf_rn(de[e], de[e], nd);
              am = fmaxf(am, fabsf(__fadd_rn(xe[e], de[e])));
            }
          }
        }
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      am = fmaxf(am, __shfl_xor_sync(0xffffffffu, am, o));
      nx += __shfl_xor_sync(0xffffffffu, nx, o);
      nd += __shfl_xor_sync(0xffffffffu, nd, o);
      ne += __shfl_xor_sync(0xffffffffu, ne, o);
    }
    if (lane == 0) {
      part[j & 1][0][warp] = am;
      part[j & 1][1][warp] = nx;
      part[j & 1][2][warp] = nd;
      part[j & 1][3][warp] = ne;
    }
    __syncthreads();
    const bool aborted = __shfl_sync(0xffffffffu, *(volatile int*)&abort_flag, 0) != 0;
    if (warp == 0 && j >= 1 && j - 1 + kPolStages < cnt && !aborted) {   // refill the stage of token j - 1
      if (elect_one()) issue(j - 1 + kPolStages);
      __syncwarp();
      issued = j + kPolStages;
    }
    float amax = part[j & 1][0][0];
#pragma unroll
    for (int w = 1; w < kPolThreads / 32; ++w) amax = fmaxf(amax, part[j & 1][0][w]);
    s = __fdiv_rn(amax, qmaxf);
    nzs = amax > 0.f;
    r = nzs ? __frcp_rn(s) : 0.f;
    if (warp == 0) {
      if (lane == 0) {
        float sx = 0.f, sd = 0.f, se = 0.f;
#pragma unroll
        for (int w = 0; w < kPolThreads / 32; ++w) {
          sx += part[j & 1][1][w];
          sd += part[j & 1][2][w];
          se += part[j & 1][3][w];
        }
        if (j >= 1) {   // token j - 1 is complete
          tok[(j - 1) & 31][0] = tok_nx;
          tok[(j - 1) & 31][1] = tok_nd;
          tok[(j - 1) & 31][2] = se;
        }
        tok_nx = sx;
        tok_nd = sd;
      }
      __syncwarp();
      if (j >= 1 && (((j - 1) & 31) == 31 || j == cnt) && !aborted) {
        const int first = (j - 1) & ~31;
        pol_batch(a, tok, t0 + first, j - first, lane);
      }
      __syncwarp();
    }
  }
  if (abort_flag) {
    // A wait gave up (the outputs are incomplete; the error word says so): let the copies
    // already issued land before the CTA's shared memory is released (bounded, on the
    // tokens that may still be in flight).
    if (warp == 0) {
      volatile int no_abort = 0;
      const int lo = issued > kPolStages ? issued - kPolStages : 0;
      for (int k = lo; k < issued; ++k)
        mbar_wait_warp(&full[k % kPolStages], (uint32_t)(k / kPolStages) & 1u, &no_abort, a.err, kDevTimeoutDrain);
    }
  }
}

__global__ void policy_finish_kernel(const PolicyArgs a) {
  const int l = blockIdx.x * blockDim.x + threadIdx.x;
  if (l >= a.L) return;
  const double jr = a.jr[l] / a.T, snr = a.snr[l] / a.T;
  a.jr[l] = jr;
  a.snr[l] = snr;
  a.bits_out[l] = (jr > a.tau_jr && snr < a.tau_snr) ? 8 : 4;
}

cudaError_t launch_policy(const PolicyArgs& a, int num_sms, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(a.jr, 0, sizeof(double) * a.L, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(a.snr, 0, sizeof(double) * a.L, s);
  if (e != cudaSuccess) return e;
  const long long items = (long long)a.L * a.T;
  if (a.d <= kPolMaxStagedD) {
    const int smem = kPolStages * 8 * a.d;
    e = ensure_max_dyn_smem(policy_stats_staged_kernel);
    int per_sm = 0;
    if (e == cudaSuccess)
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, policy_stats_staged_kernel, kPolThreads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    long long blocks = (long long)num_sms * per_sm;
    if (blocks > items) blocks = items;
    policy_stats_staged_kernel<<<(unsigned)blocks, kPolThreads, smem, s>>>(a);
  } else {
    long long blocks = items < (long long)num_sms * 8 ? items : (long long)num_sms * 8;
    if (blocks < 1) blocks = 1;
    policy_stats_kernel<<<(unsigned)blocks, kPolThreads, 0, s>>>(a);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  policy_finish_kernel<<<(a.L + 127) / 128, 128, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace dptq
