// rotate_quant.cu -- standalone launches of the fused online block-Hadamard rotation +
// symmetric per-row quantization whose per-row body lives in rotate_row.cuh
// (Section 2, Eq. 4 then Eq. 2; Section 4.2): one CTA of 256 threads per row, in the
// four writer modes, and the converter of public codes into the GEMM's E4M3 planes.
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "dptq_device.cuh"
#include "dptq_internal.h"
#include "rotate_row.cuh"

namespace dptq {

// Three CTAs per SM (at most 85 registers a thread; the body needs 72 without spilling):
// many-row launches (prefill) are bound by the latency of each row's chain of steps, so
// rows in flight per SM set their throughput.
template <int MODE>
__global__ void __launch_bounds__(kRQThreads, 3) rotate_quant_kernel(const RQArgs a) {
  extern __shared__ __align__(16) unsigned char rq_smem[];
  __shared__ float red[kRQThreads / 32];
  pdl_launch_dependents();
  pdl_wait();
  rotate_quant_row<MODE>(a, blockIdx.x, rq_smem, red, threadIdx.x, [] { __syncthreads(); });
}

// ---------------------------------------------------------------- whole-row kernel (GEMM operand)
// Codes of 16 exact Hadamard sums (units of 2^-24) of one thread, without converting each
// sum exactly.  For a value of block-size class log2n, y = S 2^-24 / sqrt(2^log2n) and the
// oracle's code is rint(fl(y_f32 / s)), y_f32 the correctly rounded y.  Here
// t = fl(fl(S) r) with r = fl(fl(2^-(24 + j) [/sqrt 2]) / s-ish): every factor carries at most
// a few units of 2^-24, so |t - fl(y_f32 / s)| <= |y / s| 8 2^-24 <= |t| 2^-21 (1 + 2^-21).
// Both round to the same integer unless t lies within m = |t| 2^-20 + 2^-30 of a
// half-integer; only there (a warp-uniform rare branch) is y_f32 formed exactly and the
// IEEE quotient taken.  The results are clamped to [qmin, qmax] and -0 becomes +0.
__device__ __forceinline__ float s_to_float_approx(long long S) {
  // S = hi 2^24 + lo with 0 <= lo < 2^24 (exact in fp32); one rounding of hi, one of the fma.
  const int hi = (int)(S >> 24);
  const int lo = (int)(S & 0xFFFFFFLL);
  return __fmaf_rn((float)hi, 16777216.f, (float)lo);
}

template <int NCH>
__global__ void __launch_bounds__(kRQThreads * NCH, NCH == 1 ? 3 : 1) rotate_quant_rows_kernel(const RQArgs a) {
  // Group g (threads 256 g .. 256 g + 255) rotates chunk g of the row (4096 elements, whole
  // Hadamard blocks), keeps its 16 exact sums per thread in registers through the row
  // absmax, quantizes them directly and writes the GEMM operand planes.
  extern __shared__ __align__(16) unsigned char rqr_smem[];
  __shared__ float redf[kRQThreads * NCH / 32];
  pdl_launch_dependents();
  pdl_wait();
  const int g = threadIdx.x / kRQThreads;
  const int tid = threadIdx.x - g * kRQThreads;
  const int row = blockIdx.x;
  const int K = a.K;
  const int K_pad = a.KB * 128;
  const int bits = a.bits;
  const int c0 = g * kChunk;
  const int len = c0 < K ? min(kChunk, K - c0) : 0;
  long long* sx = reinterpret_cast<long long*>(rqr_smem + (size_t)g * kChunkPadded * 8);
  uint8_t* stg = reinterpret_cast<uint8_t*>(sx);   // staged codes once the butterflies are done
  uint8_t* act = static_cast<uint8_t*>(a.out);
  const size_t plane_stride = (size_t)a.KB * a.rows_out * 128;
  auto gsync = [g] { asm volatile("bar.sync %0, %1;" ::"r"(1 + g), "n"(kRQThreads) : "memory"); };
  auto store4 = [&](int k, uint32_t w0, uint32_t w1) {   // codes k .. k + 3 (k % 4 == 0)
    const int kb = k >> 7, j = (k >> 4) & 7;
    const size_t off = ((size_t)kb * a.rows_out + row) * 128 + ((j ^ (row & 7)) << 4) + (k & 15);
    *reinterpret_cast<uint32_t*>(act + off) = w0;
    if (bits == 8) *reinterpret_cast<uint32_t*>(act + plane_stride + off) = w1;
  };
  if (row >= a.rows_in) {   // padding row: zero codes and scale
    for (int w = threadIdx.x; w < K_pad / 4; w += kRQThreads * NCH) store4(4 * w, 0u, 0u);
    if (threadIdx.x == 0 && a.scales != nullptr) a.scales[row] = 0.f;
    return;
  }
  const int tail_start = a.nfull << a.log2B;
  long long f[16];
  int L = 0;
  long long mB = 0, mT = 0;
  if (len > 0) {
    const uint4* src = reinterpret_cast<const uint4*>(a.x + (size_t)row * K);
    uint4 u[2];
    rq_load16(src, c0, len, tid, u);
    rq_fix16(a, u, c0, len, tid, f);
    L = rq_bfly(a, c0, len, tail_start, f, sx, tid, gsync);
    if (len == kChunk && c0 + len <= tail_start) {
      long long m[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const long long p = f[e] < 0 ? -f[e] : f[e], q = f[e + 8] < 0 ? -f[e + 8] : f[e + 8];
        m[e] = p > q ? p : q;
      }
#pragma unroll
      for (int w = 4; w > 0; w >>= 1)
#pragma unroll
        for (int e = 0; e < w; ++e) m[e] = m[e] > m[e + w] ? m[e] : m[e + w];
      mB = m[0];
    } else {
#pragma unroll
      for (int e = 0; e < 16; ++e) {
        const int i = rq_pos(L, tid, e);
        const long long v = f[e] < 0 ? -f[e] : f[e];
        if (i < len) {
          if (c0 + i < tail_start)
            mB = v > mB ? v : mB;
          else
            mT = v > mT ? v : mT;
        }
      }
    }
  }
  // Row absmax: the fp32 of the largest |S| of each block size (odd, monotone conversion),
  // a warp redux on the bit patterns, then one step across the CTA's warps.
  const float yB = mB ? fixed_to_rotated(mB, a.log2B, a.c_hi, a.c_lo) : 0.f;
  const float yT = mT ? fixed_to_rotated(mT, a.log2T, a.c_hi, a.c_lo) : 0.f;
  const uint32_t wmax = __reduce_max_sync(0xffffffffu, __float_as_uint(fmaxf(yB, yT)));
  if ((threadIdx.x & 31) == 0) redf[threadIdx.x >> 5] = __uint_as_float(wmax);
  __syncthreads();
  float amax = redf[0];
#pragma unroll
  for (int w = 1; w < kRQThreads * NCH / 32; ++w) amax = fmaxf(amax, redf[w]);
  const int qmax = (1 << (bits - 1)) - 1;
  const float qmaxf = (float)qmax, qminf = (float)(-(1 << (bits - 1)));
  const float s = __fdiv_rn(amax, qmaxf);
  const bool nz = amax > 0.f;
  const float rs = nz ? __frcp_rn(s) : 0.f;
  if (threadIdx.x == 0 && a.scales != nullptr) a.scales[row] = nz ? s : 0.f;
  if (len > 0) {
    // Per block size: y = S 2^-(24 + j) [x 1/sqrt 2 for odd log2]; r = that factor / s.
    auto rfac = [&](int log2n) {
      const float p2 = __int_as_float((127 - 24 - (log2n >> 1)) << 23);
      return __fmul_rn((log2n & 1) ? __fmul_rn(p2, a.c_hi) : p2, rs);
    };
    const float rB = rfac(a.log2B), rT = rfac(a.log2T);
    const bool uni = len == kChunk && c0 + len <= tail_start;
#pragma unroll
    for (int e4 = 0; e4 < 16; e4 += 4) {
      float t[4], q[4];
      uint32_t nearm = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int e = e4 + j;
        const float r = (uni || c0 + rq_pos(L, tid, e) < tail_start) ? rB : rT;
        t[j] = __fmul_rn(s_to_float_approx(f[e]), r);
        q[j] = rintf(t[j]);
        const float m = __fmaf_rn(fabsf(t[j]), 0x1p-20f, 0x1p-30f);
        nearm |= (fabsf(__fsub_rn(t[j], q[j])) > 0.5f - m) ? (1u << j) : 0u;
      }
      if (__any_sync(0xffffffffu, nearm != 0u)) {
#pragma unroll 1
        for (int j = 0; j < 4; ++j) {
          if ((nearm >> j) & 1u) {
            const int e = e4 + j;
            long long v = f[0];
#pragma unroll
            for (int ee = 1; ee < 16; ++ee)
              if (ee == e) v = f[ee];
            const int lg = (uni || c0 + rq_pos(L, tid, e) < tail_start) ? a.log2B : a.log2T;
            const float qq = rintf(__fdiv_rn(fixed_to_rotated(v, lg, a.c_hi, a.c_lo), s));
            if (j == 0) q[0] = qq;
            if (j == 1) q[1] = qq;
            if (j == 2) q[2] = qq;
            if (j == 3) q[3] = qq;
          }
        }
      }
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = rq_pos(L, tid, e4 + j);
        const float c = nz ? __fadd_rn(fminf(fmaxf(q[j], qminf), qmaxf), 0.0f) : 0.f;
        if (i < len) {
          if (bits == 4) {
            stg[i] = (uint8_t)(e4m3x2(c, 0.f) & 0xFFu);
          } else {
            const float mm = fabsf(c);
            const float h = __fmul_rn(floorf(__fmul_rn(mm, 0.0625f)), 16.f);
            stg[i] = (uint8_t)(e4m3x2(__fadd_rn(copysignf(h, c), 0.0f), 0.f) & 0xFFu);
            stg[kChunk + i] = (uint8_t)(e4m3x2(__fadd_rn(copysignf(__fsub_rn(mm, h), c), 0.0f), 0.f) & 0xFFu);
          }
        }
      }
    }
  }
  gsync();   // the group's codes are staged (sx is free: the max step synchronized the CTA)
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int i = 4 * (j * kRQThreads + tid);
    if (i < len)
      store4(c0 + i, *reinterpret_cast<const uint32_t*>(stg + i), *reinterpret_cast<const uint32_t*>(stg + kChunk + i));
  }
  if (g == NCH - 1)   // k in [K, K_pad): zero codes
    for (int k = K + 4 * tid; k < K_pad; k += 4 * kRQThreads) store4(k, 0u, 0u);
}

// Whole-row kernel for the GEMM operand when the row fits in registers (K <= 16384, one
// group of 256 threads per 4096-element chunk); -1 when it does not apply.
int rows_kernel_chunks(const RQArgs& a) {
  if (a.B > kChunk || a.K > 4 * kChunk || a.tail_p > 1) return -1;
  const int nch = (a.K + kChunk - 1) / kChunk;
  return nch;
}

size_t rotate_quant_smem(int K, int chunk) {
  (void)chunk;
  // the fp32 row, the int64 transpose chunk, and a Paley tail's character table (<= 256 B)
  return (size_t)K * sizeof(float) + (size_t)kChunkPadded * sizeof(long long) + 256;
}

cudaError_t launch_rotate_quant(RQMode mode, const RQArgs& a, cudaStream_t s, bool pdl) {
  const size_t smem = rotate_quant_smem(a.K, a.chunk);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)a.rows_out);
  cfg.blockDim = dim3(kRQThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = (pdl && pdl_allowed()) ? 1 : 0;
  cudaError_t e = cudaSuccess;
  switch (mode) {
    case kRQPublic:
      e = ensure_max_dyn_smem(rotate_quant_kernel<kRQPublic>);
      if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_kernel<kRQPublic>, a);
      break;
    case kRQAct: {
      const int nch = rows_kernel_chunks(a);
      if (nch >= 1 && rows_kernel_allowed()) {
        cfg.blockDim = dim3(kRQThreads * nch);
        cfg.dynamicSmemBytes = (size_t)nch * kChunkPadded * 8;
        switch (nch) {
          case 1:
            e = ensure_max_dyn_smem(rotate_quant_rows_kernel<1>);
            if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_rows_kernel<1>, a);
            break;
          case 2:
            e = ensure_max_dyn_smem(rotate_quant_rows_kernel<2>);
            if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_rows_kernel<2>, a);
            break;
          case 3:
            e = ensure_max_dyn_smem(rotate_quant_rows_kernel<3>);
            if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_rows_kernel<3>, a);
            break;
          default:
            e = ensure_max_dyn_smem(rotate_quant_rows_kernel<4>);
            if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_rows_kernel<4>, a);
            break;
        }
        break;
      }
      e = ensure_max_dyn_smem(rotate_quant_kernel<kRQAct>);
      if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_kernel<kRQAct>, a);
      break;
    }
    case kRQY:
      e = ensure_max_dyn_smem(rotate_quant_kernel<kRQY>);
      if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_kernel<kRQY>, a);
      break;
    case kRQWeights:
      e = ensure_max_dyn_smem(rotate_quant_kernel<kRQWeights>);
      if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_kernel<kRQWeights>, a);
      break;
  }
  return e;
}

// ------------------------------------------------------------------ public codes -> E4M3 planes
__global__ void __launch_bounds__(256) codes_to_act_kernel(const CodesArgs a) {
  const int nchunks = a.KB * 8;
  const long long total = (long long)a.M_pad * nchunks;
  const size_t plane_stride = (size_t)a.KB * a.M_pad * 128;
  for (long long idx = blockIdx.x * 256LL + threadIdx.x; idx < total; idx += (long long)gridDim.x * 256) {
    const int row = (int)(idx / nchunks);
    const int ch = (int)(idx - (long long)row * nchunks);
    const int kb = ch >> 3, j = ch & 7;
    const int k0 = ch * 16;
    uint32_t p0[4] = {0, 0, 0, 0}, p1[4] = {0, 0, 0, 0};
    if (row < a.M && k0 < a.K) {
      // K % 32 == 0, so a 16-code chunk is either fully inside K or fully padding.
      if (a.bits == 4) {
        const uint2 w = *reinterpret_cast<const uint2*>(a.codes + (size_t)row * (a.K / 2) + k0 / 2);
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const uint32_t word = e < 8 ? w.x : w.y;
          int c = (int)((word >> (4 * (e & 7))) & 0xFu);
          c = c >= 8 ? c - 16 : c;
          p0[e >> 2] |= e4m3_small_int(c) << (8 * (e & 3));
        }
      } else {
        const uint4 w = *reinterpret_cast<const uint4*>(a.codes + (size_t)row * a.K + k0);
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int c = (int)(int8_t)((ws[e >> 2] >> (8 * (e & 3))) & 0xFFu);
          p0[e >> 2] |= e4m3_hi_plane(c) << (8 * (e & 3));
          p1[e >> 2] |= e4m3_lo_plane(c) << (8 * (e & 3));
        }
      }
    }
    const size_t off = ((size_t)kb * a.M_pad + row) * 128 + ((j ^ (row & 7)) << 4);
    *reinterpret_cast<uint4*>(a.act + off) = make_uint4(p0[0], p0[1], p0[2], p0[3]);
    if (a.bits == 8) *reinterpret_cast<uint4*>(a.act + plane_stride + off) = make_uint4(p1[0], p1[1], p1[2], p1[3]);
  }
}

cudaError_t launch_codes_to_act(const CodesArgs& a, cudaStream_t s) {
  const long long total = (long long)a.M_pad * a.KB * 8;
  long long blocks = (total + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  codes_to_act_kernel<<<(unsigned)blocks, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace dptq
