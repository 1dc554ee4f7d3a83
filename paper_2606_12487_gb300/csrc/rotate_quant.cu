// rotate_quant.cu -- fused online block-Hadamard rotation + symmetric per-row
// quantization (Section 2, Eq. 4 then Eq. 2; Section 4.2 per-token / per-channel
// symmetric).  One CTA per row: 128-bit loads of the fp16 row, Walsh-Hadamard
// butterflies per block (natural Sylvester order) on exact 64-bit fixed-point values
// in registers with two shared-memory transposes per 4096-element chunk, one correctly rounded conversion to fp32 including 1/sqrt(block),
// row absmax by warp shuffles, IEEE-division rounding to the
// integer grid, and one of four writers:
//   kRQPublic   public codes (A4 packed nibbles / A8 int8) + fp32 scales
//   kRQAct      E4M3 operand planes in the GEMM's pre-swizzled tile layout
//   kRQY        the rotated fp32 row (test hook)
//   kRQWeights  offline weight packing (Eq. 5 fold): sign-magnitude int4 tiles
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "dptq_device.cuh"
#include "dptq_internal.h"

namespace dptq {

constexpr int kRQThreads = 256;

// Exact FP8 E4M3 encoding of an integer with |v| <= 15 (bias 7, 3 mantissa bits).
__device__ __forceinline__ uint32_t e4m3_small_int(int v) {
  const uint32_t a = (uint32_t)(v < 0 ? -v : v);
  if (a == 0) return 0u;
  const int e = 31 - __clz(a);                 // floor(log2 a), 0..3
  const uint32_t m = ((a << 3) >> e) & 7u;     // fraction bits
  return (v < 0 ? 0x80u : 0u) | ((uint32_t)(e + 7) << 3) | m;
}

// An 8-bit code c = sign * (16 h + l) (h = |c| >> 4, l = |c| & 15) splits into two
// E4M3-exact planes: hi = sign * 16 h and lo = sign * l, with hi + lo = c.
__device__ __forceinline__ uint32_t e4m3_hi_plane(int c) {
  const int a = c < 0 ? -c : c;
  const int h = a >> 4;
  if (h == 0) return 0u;
  return e4m3_small_int(c < 0 ? -h : h) + (4u << 3);   // times 2^4: exponent + 4
}
__device__ __forceinline__ uint32_t e4m3_lo_plane(int c) {
  const int a = c < 0 ? -c : c;
  const int l = a & 15;
  return e4m3_small_int(c < 0 ? -l : l);
}

__device__ __forceinline__ int quantize(float y, float s, int qmin, int qmax) {
  const float t = __fdiv_rn(y, s);   // IEEE fp32 division
  int c = __float2int_rn(t);         // round half to even
  c = c > qmax ? qmax : c;
  c = c < qmin ? qmin : c;
  return c;
}

// fp16 -> signed fixed point in units of 2^-24 (every finite binary16 is an integer
// multiple of 2^-24 below 2^41 in magnitude).
__device__ __forceinline__ long long half_to_fixed(uint32_t h) {
  const int e = (int)((h >> 10) & 31u);
  const long long m = e ? (long long)(1024u + (h & 1023u)) : (long long)(h & 1023u);
  const long long v = m << (e ? e - 1 : 0);
  return (h & 0x8000u) ? -v : v;
}

// Correctly rounded fp32 of S * 2^-24 / sqrt(2^log2n) for an exact Hadamard sum S.
// Even log2n: one rounding of S, then an exact power-of-two scale.  Odd log2n: S and
// 1/sqrt(2) as fp32 pairs, the product formed with fma to ~2^-47 relative, and one
// final rounding.
__device__ __forceinline__ float fixed_to_rotated(long long S, int log2n, float c_hi, float c_lo) {
  const int j = log2n >> 1;
  const float scale = __int_as_float((127 - 24 - j) << 23);   // 2^-(24 + j), exact
  const float hi = __ll2float_rn(S);
  if ((log2n & 1) == 0) return __fmul_rn(hi, scale);
  const float lo = __ll2float_rn(S - __float2ll_rn(hi));
  const float p = __fmul_rn(hi, c_hi);
  const float e = __fmaf_rn(hi, c_hi, -p);
  const float t = __fmaf_rn(hi, c_lo, __fmaf_rn(lo, c_hi, e));
  return __fmul_rn(__fadd_rn(p, t), scale);
}

// The row is rotated in chunks of 4096 elements (whole Hadamard blocks; the last chunk
// may be shorter).  Thread t holds 16 values of a chunk at a time, as exact 64-bit
// fixed point, in three rounds that each cover 4 bits of the element index:
//   round A: i = 16 t + e          (butterfly strides 1, 2, 4, 8 inside the thread)
//   round B: i = 256 (t>>4) + 16 e + (t&15)   (strides 16 .. 128)
//   round C: i = 256 e + t                    (strides 256 .. 2048)
// with two transposes through shared memory in between (rows of 16 values padded by
// one slot, so every access pattern is free of bank conflicts).  A stride applies to an
// element only while it is below the size of the element's Hadamard block (B, or the
// row's tail block).
constexpr int kChunk = 4096;
constexpr int kChunkPadded = kChunk + kChunk / 16;

__device__ __forceinline__ int pad_idx(int i) { return i + (i >> 4); }

template <int MODE>
__global__ void __launch_bounds__(kRQThreads) rotate_quant_kernel(const RQArgs a) {
  extern __shared__ __align__(16) unsigned char rq_smem[];
  float* sy = reinterpret_cast<float*>(rq_smem);                                      // the row, K floats
  long long* sx = reinterpret_cast<long long*>(rq_smem + (size_t)a.K * sizeof(float));  // one padded chunk
  __shared__ float red[kRQThreads / 32];
  pdl_launch_dependents();
  pdl_wait();

  const int row = blockIdx.x;
  const int tid = threadIdx.x;
  const int K = a.K;
  const bool live = row < a.rows_in;
  const int tail_start = a.nfull << a.log2B;   // first element of the tail block

  if (live) {
    const uint4* src = reinterpret_cast<const uint4*>(a.x + (size_t)row * K);
    for (int c0 = 0; c0 < K; c0 += kChunk) {
      const int len = min(kChunk, K - c0);
      // log2 of the block size that element i of this chunk belongs to
      auto lg = [&](int i) { return (c0 + i < tail_start) ? a.log2B : a.log2T; };
      long long f[16];
      // ---- round A: load 16 consecutive fp16 values
      {
        const int i0 = tid * 16;
        if (i0 < len) {
          const uint4 u0 = src[(c0 + i0) / 8];
          const uint4 u1 = src[(c0 + i0) / 8 + 1];
          const uint32_t w[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            f[2 * k] = half_to_fixed(w[k] & 0xFFFFu);
            f[2 * k + 1] = half_to_fixed(w[k] >> 16);
          }
        } else {
#pragma unroll
          for (int k = 0; k < 16; ++k) f[k] = 0;
        }
        const int L = lg(i0 < len ? i0 : 0);
#pragma unroll
        for (int bit = 0; bit < 4; ++bit) {
          if (bit < L) {
            const int h = 1 << bit;
#pragma unroll
            for (int e = 0; e < 16; ++e)
              if ((e & h) == 0) {
                const long long p = f[e], q = f[e + h];
                f[e] = p + q;
                f[e + h] = p - q;
              }
          }
        }
      }
      const int maxlg = (c0 + len > tail_start) ? max(a.log2B, a.log2T) : a.log2B;
      const int iA = tid * 16;
      if (maxlg > 4) {
        // ---- transpose A -> B
        __syncthreads();   // the previous chunk's readers are done with sx
#pragma unroll
        for (int e = 0; e < 16; ++e) sx[pad_idx(iA + e)] = f[e];
        __syncthreads();
        const int iB = 256 * (tid >> 4) + (tid & 15);
#pragma unroll
        for (int e = 0; e < 16; ++e) f[e] = sx[pad_idx(iB + 16 * e)];
        const int L = lg(iB);
#pragma unroll
        for (int bit = 4; bit < 8; ++bit) {
          if (bit < L) {
            const int h = 1 << (bit - 4);
#pragma unroll
            for (int e = 0; e < 16; ++e)
              if ((e & h) == 0) {
                const long long p = f[e], q = f[e + h];
                f[e] = p + q;
                f[e + h] = p - q;
              }
          }
        }
        if (maxlg > 8) {
          // ---- transpose B -> C
#pragma unroll
          for (int e = 0; e < 16; ++e) sx[pad_idx(iB + 16 * e)] = f[e];
          __syncthreads();
#pragma unroll
          for (int e = 0; e < 16; ++e) f[e] = sx[pad_idx(256 * e + tid)];
#pragma unroll
          for (int bit = 8; bit < 12; ++bit) {
            const int h = 1 << (bit - 8);
#pragma unroll
            for (int e = 0; e < 16; ++e)
              if ((e & h) == 0 && bit < lg(256 * e + tid)) {
                const long long p = f[e], q = f[e + h];
                f[e] = p + q;
                f[e + h] = p - q;
              }
          }
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int i = 256 * e + tid;
            if (i < len) sy[c0 + i] = fixed_to_rotated(f[e], lg(i), a.c_hi, a.c_lo);
          }
        } else {
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int i = iB + 16 * e;
            if (i < len) sy[c0 + i] = fixed_to_rotated(f[e], lg(i), a.c_hi, a.c_lo);
          }
        }
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int i = iA + e;
          if (i < len) sy[c0 + i] = fixed_to_rotated(f[e], lg(i), a.c_hi, a.c_lo);
        }
      }
    }
    __syncthreads();
  }

  // Row absmax.
  float lmax = 0.f;
  if (live) {
    for (int k = tid; k < K; k += kRQThreads) lmax = fmaxf(lmax, fabsf(sy[k]));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
  if ((tid & 31) == 0) red[tid >> 5] = lmax;
  __syncthreads();
  float amax = red[0];
#pragma unroll
  for (int w = 1; w < kRQThreads / 32; ++w) amax = fmaxf(amax, red[w]);

  if constexpr (MODE == kRQY) {
    if (live) {
      float* dst = static_cast<float*>(a.out) + (size_t)row * K;
      for (int k = tid; k < K; k += kRQThreads) dst[k] = sy[k];
    }
    return;
  } else {
    const int qmax = (1 << (a.bits - 1)) - 1;
    const int qmin = -(1 << (a.bits - 1));
    const float s = __fdiv_rn(amax, (float)qmax);
    const bool nz = live && amax > 0.f;
    if (tid == 0 && a.scales != nullptr) a.scales[row] = nz ? s : 0.f;

    if constexpr (MODE == kRQPublic) {
      if (!live) return;
      if (a.bits == 4) {
        // 8 codes -> one 32-bit word: byte j = code 2j (bits 0-3) | code 2j+1 (bits 4-7)
        uint32_t* dst = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(a.out) + (size_t)row * (K / 2));
        for (int g = tid; g < K / 8; g += kRQThreads) {
          uint32_t word = 0;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const int c = nz ? quantize(sy[8 * g + e], s, qmin, qmax) : 0;
            word |= ((uint32_t)c & 0xFu) << (4 * e);
          }
          dst[g] = word;
        }
      } else {
        uint32_t* dst = reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(a.out) + (size_t)row * K);
        for (int g = tid; g < K / 4; g += kRQThreads) {
          uint32_t word = 0;
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int c = nz ? quantize(sy[4 * g + e], s, qmin, qmax) : 0;
            word |= ((uint32_t)c & 0xFFu) << (8 * e);
          }
          dst[g] = word;
        }
      }
    } else if constexpr (MODE == kRQAct) {
      // One 16-code chunk per iteration: chunk j of k-block kb of this row sits at
      // byte ((j ^ (row & 7)) * 16) of the row's 128-byte slot (128-byte swizzle).
      uint8_t* act = static_cast<uint8_t*>(a.out);
      const int nchunks = a.KB * 8;
      const size_t plane_stride = (size_t)a.KB * a.rows_out * 128;
      for (int ch = tid; ch < nchunks; ch += kRQThreads) {
        const int kb = ch >> 3, j = ch & 7;
        const int k0 = ch * 16;
        uint32_t p0[4] = {0, 0, 0, 0}, p1[4] = {0, 0, 0, 0};
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int k = k0 + e;
          const int c = (nz && k < K) ? quantize(sy[k], s, qmin, qmax) : 0;
          if (a.bits == 4) {
            p0[e >> 2] |= e4m3_small_int(c) << (8 * (e & 3));
          } else {
            p0[e >> 2] |= e4m3_hi_plane(c) << (8 * (e & 3));
            p1[e >> 2] |= e4m3_lo_plane(c) << (8 * (e & 3));
          }
        }
        const size_t off = ((size_t)kb * a.rows_out + row) * 128 + ((j ^ (row & 7)) << 4);
        *reinterpret_cast<uint4*>(act + off) = make_uint4(p0[0], p0[1], p0[2], p0[3]);
        if (a.bits == 8)
          *reinterpret_cast<uint4*>(act + plane_stride + off) = make_uint4(p1[0], p1[1], p1[2], p1[3]);
      }
    } else if constexpr (MODE == kRQWeights) {
      // 16 weights -> 8 bytes.  Nibble = sign (bit 3) | magnitude (bits 0-2); word 0
      // byte i holds k0+i (low nibble) and k0+4+i (high nibble), word 1 holds k0+8+i
      // and k0+12+i, so that the GEMM widens a word with two masks per half.  A tile of
      // 128 rows x 128 k is stored as 4 column chunks of 32 k, each [128 rows][16 B].
      uint8_t* wt = static_cast<uint8_t*>(a.out);
      const int nchunks = a.KB * 8;
      for (int ch = tid; ch < nchunks; ch += kRQThreads) {
        const int kb = ch >> 3, j = ch & 7;
        const int k0 = ch * 16;
        uint32_t nib[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int k = k0 + e;
          int c = (nz && k < K) ? quantize(sy[k], s, qmin, qmax) : 0;
          c = c < -7 ? -7 : c;   // unreachable for symmetric RTN (|W'/s| <= 7)
          nib[e] = (c < 0 ? 8u : 0u) | (uint32_t)(c < 0 ? -c : c);
        }
        uint32_t w0 = 0, w1 = 0;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          w0 |= (nib[i] | (nib[4 + i] << 4)) << (8 * i);
          w1 |= (nib[8 + i] | (nib[12 + i] << 4)) << (8 * i);
        }
        // tile [16-byte chunk j / 2][row][16 B]: the 32 rows a warp reads side by side
        // are contiguous
        const size_t off = (((size_t)(row >> 7) * a.KB + kb) * kWTileBytes) + (j >> 1) * 2048 + (row & 127) * 16 +
                           (j & 1) * 8;
        *reinterpret_cast<uint2*>(wt + off) = make_uint2(w0, w1);
      }
    }
  }
}

size_t rotate_quant_smem(int K, int chunk) {
  (void)chunk;
  return (size_t)K * sizeof(float) + (size_t)kChunkPadded * sizeof(long long);
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
      e = cudaFuncSetAttribute(rotate_quant_kernel<kRQPublic>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_kernel<kRQPublic>, a);
      break;
    case kRQAct:
      e = cudaFuncSetAttribute(rotate_quant_kernel<kRQAct>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_kernel<kRQAct>, a);
      break;
    case kRQY:
      e = cudaFuncSetAttribute(rotate_quant_kernel<kRQY>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e == cudaSuccess) e = cudaLaunchKernelEx(&cfg, rotate_quant_kernel<kRQY>, a);
      break;
    case kRQWeights:
      e = cudaFuncSetAttribute(rotate_quant_kernel<kRQWeights>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
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
