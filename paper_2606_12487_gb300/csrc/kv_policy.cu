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

// Groups of 128 (the paper's size): four consecutive groups per warp and iteration, all
// four loads issued first, so that each SM keeps enough bytes in flight.
__global__ void __launch_bounds__(kKvWarps * 32) kv4_quantize_g128_kernel(const KvArgs a) {
  const int lane = threadIdx.x & 31;
  const long long ngroups = (long long)a.rows * (a.cols >> 7);   // groups are consecutive in memory
  const long long nquads = (ngroups + 3) >> 2;
  const long long nwarps = (long long)gridDim.x * kKvWarps;
  for (long long w = (long long)blockIdx.x * kKvWarps + (threadIdx.x >> 5); w < nquads; w += nwarps) {
    const long long g0 = 4 * w;
    uint2 raw[4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
      raw[i] = g0 + i < ngroups ? __ldg(reinterpret_cast<const uint2*>(a.kv + (size_t)(g0 + i) * 128 + 4 * lane))
                                : make_uint2(0u, 0u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (g0 + i >= ngroups) break;
      float amax = absmax4(raw[i]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
      const float s = __fdiv_rn(amax, 7.f);
      const bool nz = amax > 0.f;
      const float r = nz ? __frcp_rn(s) : 0.f;
      if (lane == 0) a.scales[g0 + i] = nz ? s : 0.f;
      reinterpret_cast<uint16_t*>(a.codes + (size_t)(g0 + i) * 64)[lane] = (uint16_t)kv4_codes(raw[i], s, r, nz);
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
  const long long work = a.group == 128 ? (ngroups + 3) / 4 : ngroups;   // warps' work items
  long long blocks = (work + kKvWarps - 1) / kKvWarps;
  const long long cap = (long long)num_sms * 8;
  if (blocks > cap) blocks = cap;
  if (blocks < 1) blocks = 1;
  if (a.group == 128)
    kv4_quantize_g128_kernel<<<(unsigned)blocks, kKvWarps * 32, 0, s>>>(a);
  else
    kv4_quantize_kernel<<<(unsigned)blocks, kKvWarps * 32, 0, s>>>(a);
  return cudaGetLastError();
}

// ------------------------------------------------------------------ policy
// One CTA of 256 threads per (layer, token) at a time.  Thread t holds columns
// 4t + 1024 i of the token (float4 loads of x and dx).  Per element, in fp32:
//   |x|^2 and |dx|^2; u = fl(x + dx) as the quantizer's input (the oracle's fp32 sum);
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
    // pass 1: norms and the quantizer's absmax (tokens of up to 4096 values stay in
    // registers for pass 2; all loads of a token are issued first)
    float nx = 0.f, nd = 0.f, am = 0.f;
    const bool cached = a.d <= 4 * 4 * kPolThreads;
    float4 xc[4], dc[4];
    if (cached) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int k = 4 * tid + 4 * kPolThreads * i;
        xc[i] = k < a.d ? __ldg(reinterpret_cast<const float4*>(x + k)) : make_float4(0.f, 0.f, 0.f, 0.f);
        dc[i] = k < a.d ? __ldg(reinterpret_cast<const float4*>(dx + k)) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float xs[4] = {xc[i].x, xc[i].y, xc[i].z, xc[i].w}, ds[4] = {dc[i].x, dc[i].y, dc[i].z, dc[i].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          nx = __fmaf_rn(xs[e], xs[e], nx);
          nd = __fmaf_rn(ds[e], ds[e], nd);
          am = fmaxf(am, fabsf(__fadd_rn(xs[e], ds[e])));
        }
      }
    } else {
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
    // pass 2: the reconstruction error (registers, or re-read from L1/L2)
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
    if (cached) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (4 * tid + 4 * kPolThreads * i < a.d) err4(xc[i], dc[i]);
    } else {
      for (int k = 4 * tid; k < a.d; k += 4 * kPolThreads)
        err4(__ldg(reinterpret_cast<const float4*>(x + k)), __ldg(reinterpret_cast<const float4*>(dx + k)));
    }
    const double nx2 = block_sum_f64((double)nx, red, tid);
    const double nd2 = block_sum_f64((double)nd, red, tid);
    const double ne2 = block_sum_f64((double)ne, red, tid);
    if (tid == 0) {
      atomicAdd(a.jr + l, sqrt(nd2) / (sqrt(nx2) + a.eps));
      atomicAdd(a.snr + l, 10.0 * log10(nx2 / (ne2 + a.eps)));
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
  long long blocks = items < (long long)num_sms * 8 ? items : (long long)num_sms * 8;
  if (blocks < 1) blocks = 1;
  policy_stats_kernel<<<(unsigned)blocks, kPolThreads, 0, s>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  policy_finish_kernel<<<(a.L + 127) / 128, 128, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace dptq
