// rotate_row.cuh -- the per-row body of the fused online block-Hadamard rotation +
// symmetric per-row quantization (Section 2, Eq. 4 then Eq. 2; Section 4.2 per-token /
// per-channel symmetric), shared by the standalone kernel (rotate_quant.cu) and the
// fused decode GEMM (qgemm.cu).  Exact 64-bit fixed-point Walsh-Hadamard butterflies
// in registers with two shared-memory transposes per 4096-element chunk, one correctly
// rounded conversion to fp32 including 1/sqrt(block), row absmax by warp shuffles,
// IEEE-division rounding to the integer grid, and one of four writers:
//   kRQPublic   public codes (A4 packed nibbles / A8 int8) + fp32 scales
//   kRQAct      E4M3 operand planes in the GEMM's pre-swizzled tile layout
//   kRQY        the rotated fp32 row (test hook)
//   kRQWeights  offline weight packing (Eq. 5 fold): sign-magnitude int4 tiles
#pragma once
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

// Code of y on the grid of step s: the IEEE fp32 quotient y / s rounded half to even,
// clamped to [qmin, qmax], returned as a float (an integer, +0 for zero).
// The quotient is replaced by t = y * r with r = 1/s correctly rounded: t is within
// |y/s| * 2^-23 (1 + 2^-24) <= 2^-16 of the exact y/s for |y/s| <= 128, and the IEEE
// quotient within 2^-17 of it, so both round to the same integer unless t lies within
// 2^-16 + 2^-17 < 2^-15 of a half-integer.  Only there is the IEEE division computed.
// Called by whole warps (the division runs only when some lane of the warp needs it).
__device__ __forceinline__ float quant_code(float y, float s, float r, float qmin, float qmax) {
  const float t = __fmul_rn(y, r);
  float c = rintf(t);
  const bool near = fabsf(__fsub_rn(t, c)) >= 0.5f - 0x1p-15f;
  if (__any_sync(__activemask(), near)) {
    if (near) c = rintf(__fdiv_rn(y, s));
  }
  c = fminf(fmaxf(c, qmin), qmax);
  return __fadd_rn(c, 0.0f);   // -0 -> +0
}
__device__ __forceinline__ int quantize(float y, float s, float r, int qmin, int qmax) {
  return (int)quant_code(y, s, r, (float)qmin, (float)qmax);
}

// Two small integers (exact in E4M3) to FP8 E4M3 bytes: lo in bits 0-7, hi in 8-15.
__device__ __forceinline__ uint32_t e4m3x2(float lo, float hi) {
  uint16_t d;
  asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(d) : "f"(hi), "f"(lo));
  return d;
}

// fp16 -> signed fixed point in units of 2^-24 (every finite binary16 is an integer
// multiple of 2^-24 below 2^41 in magnitude).
__device__ __forceinline__ long long half_to_fixed(uint32_t h) {
  const int e = (int)((h >> 10) & 31u);
  const long long m = e ? (long long)(1024u + (h & 1023u)) : (long long)(h & 1023u);
  const long long v = m << (e ? e - 1 : 0);
  return (h & 0x8000u) ? -v : v;
}

// |S| < 2^53 to fp32, correctly rounded (round to nearest even), with one 32-bit
// conversion: |S| is shifted right by the n bits that do not fit in 32 (n = 0 below
// 2^32), every set bit shifted out is folded into the lowest kept bit (a sticky bit
// below the rounding position leaves round-to-nearest-even unchanged), and the rounded
// result is scaled by 2^n.  Branch-free: the 64-bit conversion instruction is several
// times slower on this part.
__device__ __forceinline__ float ll_to_float_rn(long long S) {
  const unsigned long long m = (unsigned long long)(S < 0 ? -S : S);
  const uint32_t hi = (uint32_t)(m >> 32), lo = (uint32_t)m;
  const int n = 32 - __clz(hi);   // 0..21
  const uint32_t top = (uint32_t)(m >> n) | ((lo & ((1u << n) - 1u)) != 0u);
  const float f = __fmul_rn(__uint2float_rn(top), __int_as_float((127 + n) << 23));   // exact scale by 2^n
  return S < 0 ? -f : f;
}

// Correctly rounded fp32 of S * 2^-24 / sqrt(2^log2n) for an exact Hadamard sum S.
// Even log2n: one rounding of S, then an exact power-of-two scale.  Odd log2n: S and
// 1/sqrt(2) as fp32 pairs, the product formed with fma to ~2^-47 relative, and one
// final rounding.
__device__ __forceinline__ float fixed_to_rotated(long long S, int log2n, float c_hi, float c_lo) {
  const int j = log2n >> 1;
  const float scale = __int_as_float((127 - 24 - j) << 23);   // 2^-(24 + j), exact
  const float hi = ll_to_float_rn(S);
  if ((log2n & 1) == 0) return __fmul_rn(hi, scale);
  // S - hi exactly: hi = +-(1.f) * 2^e with e <= 52 is the integer mag << (e - 23); the
  // remainder is below 2^29 in magnitude.
  const uint32_t hb = __float_as_uint(hi);
  const int e = (int)((hb >> 23) & 0xFFu) - 127;
  long long hi_int = 0;
  if (e >= 0) {
    const unsigned long long mag = (unsigned long long)((hb & 0x7FFFFFu) | 0x800000u);
    hi_int = (long long)(e >= 23 ? mag << (e - 23) : mag >> (23 - e));
    if (hb >> 31) hi_int = -hi_int;
  }
  const float lo = __int2float_rn((int)(S - hi_int));
  const float p = __fmul_rn(hi, c_hi);
  const float err = __fmaf_rn(hi, c_hi, -p);
  const float t = __fmaf_rn(hi, c_lo, __fmaf_rn(lo, c_hi, err));
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

// One row: rotate, find the absmax, quantize and write it in mode MODE.  Run by
// kRQThreads threads (thread index `tid`) that meet at `sync()`; `smem` holds
// rotate_quant_smem(K) bytes (16-byte aligned) and `red` kRQThreads / 32 floats.  The
// caller synchronizes before reusing `smem` for another row.
template <int MODE, class Sync>
__device__ __forceinline__ void rotate_quant_row(const RQArgs& a, int row, unsigned char* smem, float* red, int tid,
                                                 Sync sync) {
  float* sy = reinterpret_cast<float*>(smem);                                      // the row, K floats
  long long* sx = reinterpret_cast<long long*>(smem + (size_t)a.K * sizeof(float));  // one padded chunk
  unsigned long long* const tr = DPTQ_TRACE_BUF();
  (void)tr;
#define RQ_TRACE(slot) \
  do {                 \
    if (tid == 0) DPTQ_TRACE_POINT(tr, slot); \
  } while (0)
  const int K = a.K;
  const bool live = row < a.rows_in;
  const int tail_start = a.nfull << a.log2B;   // first element of the tail block
  float lmax = 0.f;   // this thread's largest |y|

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
        if (c0 == 0) RQ_TRACE(130);
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
      if (c0 == 0) RQ_TRACE(131);
      const int maxlg = (c0 + len > tail_start) ? max(a.log2B, a.log2T) : a.log2B;
      const int iA = tid * 16;
      if (maxlg > 4) {
        // ---- transpose A -> B
        sync();   // the previous chunk's readers are done with sx
#pragma unroll
        for (int e = 0; e < 16; ++e) sx[pad_idx(iA + e)] = f[e];
        sync();
        const int iB = 256 * (tid >> 4) + (tid & 15);
#pragma unroll
        for (int e = 0; e < 16; ++e) f[e] = sx[pad_idx(iB + 16 * e)];
        if (c0 == 0) RQ_TRACE(132);
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
        if (c0 == 0) RQ_TRACE(133);
        if (maxlg > 8) {
          // ---- transpose B -> C
#pragma unroll
          for (int e = 0; e < 16; ++e) sx[pad_idx(iB + 16 * e)] = f[e];
          sync();
#pragma unroll
          for (int e = 0; e < 16; ++e) f[e] = sx[pad_idx(256 * e + tid)];
          if (c0 == 0) RQ_TRACE(134);
          if (c0 + len <= tail_start) {
            // every element of the chunk lies in a block of size B: uniform strides
#pragma unroll
            for (int bit = 8; bit < 12; ++bit) {
              if (bit < a.log2B) {
                const int h = 1 << (bit - 8);
#pragma unroll
                for (int e = 0; e < 16; ++e)
                  if ((e & h) == 0) {
                    const long long p = f[e], q = f[e + h];
                    f[e] = p + q;
                    f[e + h] = p - q;
                  }
              }
            }
#pragma unroll
            for (int e = 0; e < 16; ++e) {
              const int i = 256 * e + tid;
              if (i < len) {
                const float yv = fixed_to_rotated(f[e], a.log2B, a.c_hi, a.c_lo);
                lmax = fmaxf(lmax, fabsf(yv));
                sy[c0 + i] = yv;
              }
            }
            if (c0 == 0) RQ_TRACE(135);
          } else {
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
              if (i < len) {
                const float yv = fixed_to_rotated(f[e], lg(i), a.c_hi, a.c_lo);
                lmax = fmaxf(lmax, fabsf(yv));
                sy[c0 + i] = yv;
              }
            }
          }
        } else {
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int i = iB + 16 * e;
            if (i < len) {
              const float yv = fixed_to_rotated(f[e], lg(i), a.c_hi, a.c_lo);
              lmax = fmaxf(lmax, fabsf(yv));
              sy[c0 + i] = yv;
            }
          }
        }
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int i = iA + e;
          if (i < len) {
            const float yv = fixed_to_rotated(f[e], lg(i), a.c_hi, a.c_lo);
            lmax = fmaxf(lmax, fabsf(yv));
            sy[c0 + i] = yv;
          }
        }
      }
    }
    sync();
  }
  RQ_TRACE(136);

  // Row absmax.
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) lmax = fmaxf(lmax, __shfl_xor_sync(0xffffffffu, lmax, o));
  if ((tid & 31) == 0) red[tid >> 5] = lmax;
  sync();
  float amax = red[0];
#pragma unroll
  for (int w = 1; w < kRQThreads / 32; ++w) amax = fmaxf(amax, red[w]);
  RQ_TRACE(137);

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
    const float rs = nz ? __frcp_rn(s) : 0.f;
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
            const int c = nz ? quantize(sy[8 * g + e], s, rs, qmin, qmax) : 0;
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
            const int c = nz ? quantize(sy[4 * g + e], s, rs, qmin, qmax) : 0;
            word |= ((uint32_t)c & 0xFFu) << (8 * e);
          }
          dst[g] = word;
        }
      }
    } else if constexpr (MODE == kRQAct) {
      // Thread t quantizes codes k = 4t + 1024 i (a conflict-free float4 read) and
      // stores them as one 32-bit word: chunk j of k-block kb of this row sits at byte
      // ((j ^ (row & 7)) * 16) of the row's 128-byte slot (128-byte swizzle); a warp
      // writes one k-block of the row.  Rows past rows_in and k past K get zeros.
      uint8_t* act = static_cast<uint8_t*>(a.out);
      const size_t plane_stride = (size_t)a.KB * a.rows_out * 128;
      const int K_pad = a.KB * 128;
      const float qminf = (float)qmin, qmaxf = (float)qmax;
      for (int k = 4 * tid; k < K_pad; k += 4 * kRQThreads) {
        float c[4] = {0.f, 0.f, 0.f, 0.f};
        if (nz && k < K) {   // K % 32 == 0: the four codes are all inside K or all padding
          const float4 y4 = *reinterpret_cast<const float4*>(sy + k);
          c[0] = quant_code(y4.x, s, rs, qminf, qmaxf);
          c[1] = quant_code(y4.y, s, rs, qminf, qmaxf);
          c[2] = quant_code(y4.z, s, rs, qminf, qmaxf);
          c[3] = quant_code(y4.w, s, rs, qminf, qmaxf);
        }
        const int kb = k >> 7, j = (k >> 4) & 7;
        const size_t off = ((size_t)kb * a.rows_out + row) * 128 + ((j ^ (row & 7)) << 4) + (k & 15);
        if (a.bits == 4) {
          *reinterpret_cast<uint32_t*>(act + off) = e4m3x2(c[0], c[1]) | (e4m3x2(c[2], c[3]) << 16);
        } else {
          // c = hi + lo with hi = sign * 16 * (|c| >> 4) and lo = sign * (|c| & 15)
          float hi[4], lo[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float m = fabsf(c[e]);
            const float h = __fmul_rn(floorf(__fmul_rn(m, 0.0625f)), 16.f);
            hi[e] = __fadd_rn(copysignf(h, c[e]), 0.0f);   // -0 -> +0
            lo[e] = __fadd_rn(copysignf(__fsub_rn(m, h), c[e]), 0.0f);
          }
          *reinterpret_cast<uint32_t*>(act + off) = e4m3x2(hi[0], hi[1]) | (e4m3x2(hi[2], hi[3]) << 16);
          *reinterpret_cast<uint32_t*>(act + plane_stride + off) = e4m3x2(lo[0], lo[1]) | (e4m3x2(lo[2], lo[3]) << 16);
        }
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
          int c = (nz && k < K) ? quantize(sy[k], s, rs, qmin, qmax) : 0;
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
#undef RQ_TRACE
}

}  // namespace dptq
