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

// The same for four values at once, by a whole warp: the reciprocal products for all
// four, then (only if some lane of the warp has a value near a half-integer) the IEEE
// quotients of those values, so that the common path carries no division code.
__device__ __forceinline__ void quant_code4(const float (&y)[4], float s, float r, float qmin, float qmax,
                                            float (&c)[4]) {
  uint32_t nearm = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float t = __fmul_rn(y[j], r);
    c[j] = rintf(t);
    nearm |= (fabsf(__fsub_rn(t, c[j])) >= 0.5f - 0x1p-15f) ? (1u << j) : 0u;
  }
  if (__any_sync(__activemask(), nearm != 0u)) {
#pragma unroll 1
    for (int j = 0; j < 4; ++j) {
      if ((nearm >> j) & 1u) {
        const float yj = j == 0 ? y[0] : j == 1 ? y[1] : j == 2 ? y[2] : y[3];
        const float q = rintf(__fdiv_rn(yj, s));
        if (j == 0) c[0] = q;
        if (j == 1) c[1] = q;
        if (j == 2) c[2] = q;
        if (j == 3) c[3] = q;
      }
    }
  }
#pragma unroll
  for (int j = 0; j < 4; ++j) c[j] = __fadd_rn(fminf(fmaxf(c[j], qmin), qmax), 0.0f);   // -0 -> +0
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

// Randomized Hadamard (QuaRot's diagonal, Sections 1 and 4.2): negate the values whose
// sign byte is negative (16 consecutive elements; `sg` 16-byte aligned).  Exact.
__device__ __forceinline__ void apply_signs(const int8_t* sg, long long (&f)[16]) {
  const uint4 v = *reinterpret_cast<const uint4*>(sg);
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int e = 0; e < 16; ++e)
    if ((w[e >> 2] >> (8 * (e & 3) + 7)) & 1u) f[e] = -f[e];
}

// fp32 of S * 2^-(24 + j) * c for an exact sum S and an fp32 pair c = c_hi + c_lo (an
// irrational constant to ~2^-48): S and c as fp32 pairs, their product formed with fma to
// ~2^-47 relative, and one final rounding (correctly rounded except within ~2^-47 of a
// rounding boundary).
__device__ __forceinline__ float fixed_times_const(long long S, int j, float c_hi, float c_lo) {
  const float scale = __int_as_float((127 - 24 - j) << 23);   // 2^-(24 + j), exact
  const float hi = ll_to_float_rn(S);
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

// Correctly rounded fp32 of S * 2^-24 / sqrt(2^log2n) for an exact Hadamard sum S.
// Even log2n: one rounding of S, then an exact power-of-two scale.  Odd log2n: the
// product with 1/sqrt(2) (c_hi + c_lo) of fixed_times_const.
__device__ __forceinline__ float fixed_to_rotated(long long S, int log2n, float c_hi, float c_lo) {
  const int j = log2n >> 1;
  if ((log2n & 1) == 0) return __fmul_rn(ll_to_float_rn(S), __int_as_float((127 - 24 - j) << 23));
  return fixed_times_const(S, j, c_hi, c_lo);
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

  // Non-power-of-two tail (tail_p > 1): the quadratic character mod q = tail_p - 1, one
  // byte per residue, after the transpose buffer; the tail's sums wait in sx until every
  // segment's H_(2^log2T) butterflies are done, then H_p mixes the segments.
  const bool ptail = a.tail_p > 1;
  signed char* chi = reinterpret_cast<signed char*>(smem + (size_t)K * sizeof(float) + (size_t)kChunkPadded * 8);
  if (live && ptail) {
    const int q = a.tail_p - 1;
    for (int d = tid; d < q; d += kRQThreads) {
      int r = 1, b = d, e = (q - 1) / 2;   // d^((q-1)/2) mod q (Euler's criterion)
      while (e) {
        if (e & 1) r = (r * b) % q;
        b = (b * b) % q;
        e >>= 1;
      }
      chi[d] = d == 0 ? 0 : (r == 1 ? 1 : -1);
    }
  }

  if (live) {
    const uint4* src = reinterpret_cast<const uint4*>(a.x + (size_t)row * K);
    for (int c0 = 0; c0 < K; c0 += kChunk) {
      const int len = min(kChunk, K - c0);
      // log2 of the block size that element i of this chunk belongs to
      auto lg = [&](int i) { return (c0 + i < tail_start) ? a.log2B : a.log2T; };
      // fp32 of the sum of element c0 + i into sy (a Paley tail's sums are mixed later)
      auto put = [&](long long S, int i) {
        if (ptail && c0 + i >= tail_start) return;
        const float yv = fixed_to_rotated(S, lg(i), a.c_hi, a.c_lo);
        lmax = fmaxf(lmax, fabsf(yv));
        sy[c0 + i] = yv;
      };
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
          if (a.signs != nullptr) apply_signs(a.signs + c0 + i0, f);
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
              if (i < len) put(f[e], i);
            }
          }
        } else {
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            const int i = iB + 16 * e;
            if (i < len) put(f[e], i);
          }
        }
      } else {
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int i = iA + e;
          if (i < len) put(f[e], i);
        }
      }
      if (ptail && c0 + len > tail_start) {
        // The tail lies in this (last) chunk: park its sums, in tail order, in sx once
        // every thread's transpose reads are done.
        sync();
        long long* tz = sx;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const int i = maxlg > 8 ? 256 * e + tid : maxlg > 4 ? 256 * (tid >> 4) + 16 * e + (tid & 15) : iA + e;
          if (i < len && c0 + i >= tail_start) tz[c0 + i - tail_start] = f[e];
        }
      }
    }
    if (ptail) {
      // y[a' 2^k + b'] = sum_a H_p[a][a'] z[a 2^k + b'] (exact), H_p[a][a'] = 1 on the
      // diagonal and in row 0, -1 in column 0, chi(a' - a) elsewhere (Paley I); then
      // y 2^-(24 + tail_j) (t_hi + t_lo) = S 2^-24 / sqrt(r).
      sync();
      const long long* tz = sx;
      const int r = K - tail_start, k = a.log2T, q = a.tail_p - 1;
      for (int j = tid; j < r; j += kRQThreads) {
        const int ap = j >> k, bp = j & ((1 << k) - 1);
        long long S = 0;
        for (int aa = 0; aa < a.tail_p; ++aa) {
          const long long z = tz[(aa << k) + bp];
          int h;
          if (aa == ap || aa == 0)
            h = 1;
          else if (ap == 0)
            h = -1;
          else
            h = chi[(ap - aa + q) % q];
          S += h > 0 ? z : -z;
        }
        const float yv = fixed_times_const(S, a.tail_j, a.t_hi, a.t_lo);
        lmax = fmaxf(lmax, fabsf(yv));
        sy[tail_start + j] = yv;
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
          const float yv[4] = {y4.x, y4.y, y4.z, y4.w};
          quant_code4(yv, s, rs, qminf, qmaxf, c);
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

// ---------------------------------------------------------------- fused decode launch
// Element index of value e of thread t in the layout the butterflies of a chunk end in:
// 0 = round A only (blocks of at most 16), 1 = rounds A and B (at most 256), 2 = all.
__device__ __forceinline__ int rq_pos(int layout, int t, int e) {
  return layout == 2 ? 256 * e + t : layout == 1 ? 256 * (t >> 4) + 16 * e + (t & 15) : 16 * t + e;
}

// Raw fp16 words of thread `tid`'s 16 consecutive values of the chunk at c0 (round A
// layout, i = 16 tid + e); zeros past the chunk's length.
__device__ __forceinline__ void rq_load16(const uint4* src, int c0, int len, int tid, uint4 (&u)[2]) {
  const int i0 = tid * 16;
  if (i0 < len) {
    u[0] = src[(c0 + i0) / 8];
    u[1] = src[(c0 + i0) / 8 + 1];
  } else {
    u[0] = make_uint4(0u, 0u, 0u, 0u);
    u[1] = u[0];
  }
}

// The 16 raw fp16 values to exact fixed point, with the randomized-Hadamard signs.
__device__ __forceinline__ void rq_fix16(const RQArgs& a, const uint4 (&u)[2], int c0, int len, int tid,
                                         long long (&f)[16]) {
  const uint32_t w[8] = {u[0].x, u[0].y, u[0].z, u[0].w, u[1].x, u[1].y, u[1].z, u[1].w};
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    f[2 * k] = half_to_fixed(w[k] & 0xFFFFu);
    f[2 * k + 1] = half_to_fixed(w[k] >> 16);
  }
  if (a.signs != nullptr && tid * 16 < len) apply_signs(a.signs + c0 + tid * 16, f);
}

// The exact butterflies of one chunk (elements c0 .. c0 + len - 1 of the row), starting
// from f[] in the round A layout; returns the layout f[] ends in (see rq_pos).
template <class Sync>
__device__ __forceinline__ int rq_bfly(const RQArgs& a, int c0, int len, int tail_start, long long (&f)[16],
                                       long long* sx, int tid, Sync sync) {
  unsigned long long* const tr = DPTQ_TRACE_BUF();
  (void)tr;
#define RQC_T(slot) \
  do {              \
    if (tid == 0 && c0 == 0) DPTQ_TRACE_CLOCK(tr, slot); \
  } while (0)
  auto lg = [&](int i) { return (c0 + i < tail_start) ? a.log2B : a.log2T; };
  auto bfly = [&](int h) {
#pragma unroll
    for (int e = 0; e < 16; ++e)
      if ((e & h) == 0) {
        const long long p = f[e], q = f[e + h];
        f[e] = p + q;
        f[e + h] = p - q;
      }
  };
  const int i0 = tid * 16;
  RQC_T(171);
  {
    const int L = lg(i0 < len ? i0 : 0);
    if (L >= 4) {
      bfly(1);
      bfly(2);
      bfly(4);
      bfly(8);
    } else {
#pragma unroll
      for (int bit = 0; bit < 4; ++bit)
        if (bit < L) bfly(1 << bit);
    }
  }
  RQC_T(172);
  const int maxlg = (c0 + len > tail_start) ? max(a.log2B, a.log2T) : a.log2B;
  if (maxlg <= 4) return 0;
  sync();   // the previous readers of sx are done
#pragma unroll
  for (int e = 0; e < 16; ++e) sx[pad_idx(i0 + e)] = f[e];
  sync();
  const int iB = 256 * (tid >> 4) + (tid & 15);
#pragma unroll
  for (int e = 0; e < 16; ++e) f[e] = sx[pad_idx(iB + 16 * e)];
  RQC_T(173);
  {
    const int L = lg(iB);
    if (L >= 8) {
      bfly(1);
      bfly(2);
      bfly(4);
      bfly(8);
    } else {
#pragma unroll
      for (int bit = 4; bit < 8; ++bit)
        if (bit < L) bfly(1 << (bit - 4));
    }
  }
  RQC_T(174);
  if (maxlg <= 8) return 1;
#pragma unroll
  for (int e = 0; e < 16; ++e) sx[pad_idx(iB + 16 * e)] = f[e];
  sync();
#pragma unroll
  for (int e = 0; e < 16; ++e) f[e] = sx[pad_idx(256 * e + tid)];
  RQC_T(175);
  if (c0 + len <= tail_start && a.log2B == 12) {
    bfly(1);
    bfly(2);
    bfly(4);
    bfly(8);
  } else if (c0 + len <= tail_start) {
#pragma unroll
    for (int bit = 8; bit < 12; ++bit)
      if (bit < a.log2B) bfly(1 << (bit - 8));
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
  }
  RQC_T(176);
#undef RQC_T
  return 2;
}

// Load, fix and butterflies of one chunk: the same arithmetic as rotate_quant_row.
template <class Sync>
__device__ __forceinline__ int rq_chunk(const RQArgs& a, const uint4* src, int c0, int len, int tail_start,
                                        long long (&f)[16], long long* sx, int tid, Sync sync) {
  uint4 u[2];
  rq_load16(src, c0, len, tid, u);
  rq_fix16(a, u, c0, len, tid, f);
  return rq_bfly(a, c0, len, tail_start, f, sx, tid, sync);
}

// The same butterflies as rq_bfly with a small code footprint, for code that runs once
// per launch (the fused decode rotation), where every instruction is fetched cold: the
// three rounds share one body (a transpose through sx between rounds, then the round's
// four levels on the 16 values in registers), so rounds B and C run from instructions
// that round A brought into the instruction cache.  Returns the layout f[] ends in.
template <class Sync>
__device__ __forceinline__ int rq_bfly_compact(const RQArgs& a, int c0, int len, int tail_start, long long (&f)[16],
                                            long long* sx, int tid, Sync sync) {
  const int maxlg = (c0 + len > tail_start) ? max(a.log2B, a.log2T) : a.log2B;
  const int rounds = maxlg <= 4 ? 1 : maxlg <= 8 ? 2 : 3;
  // Blocks are B-sized before tail_start and tail-sized after, so only chunks that reach
  // the tail can mix block sizes.
  const bool mixed = c0 + len > tail_start && a.log2T != a.log2B;
  // Padded index of value e of this thread in layout r: pad_idx(rq_pos(r, tid, e)) =
  // pb[r] + ps[r] e, since every layout is linear in e (strides 1, 16, 256) and the
  // padding adds one slot per 16 elements.
  const int pb0 = 17 * tid;
  const int ib1 = 256 * (tid >> 4) + (tid & 15);
  const int pb1 = ib1 + (ib1 >> 4);
  const int pb2 = tid + (tid >> 4);
#pragma unroll 1
  for (int r = 0; r < rounds; ++r) {
    if (r > 0) {
      const int wb = r == 1 ? pb0 : pb1, ws = r == 1 ? 1 : 17;
      const int rb = r == 1 ? pb1 : pb2, rs = r == 1 ? 17 : 272;
      sync();   // the previous readers of sx are done
      long long* wp = sx + wb;
#pragma unroll
      for (int e = 0; e < 16; ++e) wp[ws * e] = f[e];
      sync();
      const long long* rp = sx + rb;
#pragma unroll
      for (int e = 0; e < 16; ++e) f[e] = rp[rs * e];
    }
    const int base = 4 * r;
    if (!mixed && a.log2B >= base + 4) {   // every element's block spans the round's 4 levels
#pragma unroll
      for (int bit = 0; bit < 4; ++bit) {
        const int h = 1 << bit;
#pragma unroll
        for (int e = 0; e < 16; ++e)
          if ((e & h) == 0) {
            const long long p = f[e], q = f[e + h];
            f[e] = p + q;
            f[e + h] = p - q;
          }
      }
    } else {
      // A level applies to an element while it is below the log2 of the element's block.
#pragma unroll
      for (int bit = 0; bit < 4; ++bit) {
        const int lvl = base + bit;
        const int h = 1 << bit;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          if ((e & h) == 0) {
            const int i = rq_pos(r, tid, e);
            const int lg = (c0 + i < tail_start) ? a.log2B : a.log2T;
            if (lvl < lg) {
              const long long p = f[e], q = f[e + h];
              f[e] = p + q;
              f[e + h] = p - q;
            }
          }
        }
      }
    }
  }
  return rounds - 1;
}

__device__ __forceinline__ uint32_t e4m3_byte(float v) { return e4m3x2(v, 0.f) & 0xFFu; }

static_assert(kRQPartSmemBytes == kChunkPadded * 8 + 2 * kChunk + 16 * 8, "part scratch layout");

// ---- one row's rotation split over the parts of the fused decode launch
// Each of the np parts of a row rotates only its own outputs, so the parts share the
// work instead of repeating it; the row absmax, which every code depends on, is then
// exchanged between the parts through one slot per part in global memory.
//   * Whole blocks (kPartBlocks): the row splits into np ranges of whole 128-aligned
//     granules (a granule is max(B, 128) elements: whole Hadamard blocks), each at most
//     4096 elements, rotated like one chunk of rotate_quant_row.
//   * Block slices (kPartSlice4 / kPartSlice8): when a row has fewer blocks than parts,
//     each block of B = n L elements is shared by n parts.  With Sylvester's ordering
//     H_B = H_n (x) H_L, so output slice p' of the block is H_L applied to
//     v = sum_a H_n[p'][a] x_a, x_a the a-th L-element slice of the block's input: a part
//     combines the n input slices at its L positions (exact) and runs the L-point
//     butterflies, L = 256 V (V = 4 or 8 values per thread).
enum : int { kPartBlocks = 1, kPartSlice4 = 4, kPartSlice8 = 8 };

// Granule range [g0, g1) of `part` when ng granules are split over np parts.
__device__ __forceinline__ void part_granules(int ng, int np, int part, int& g0, int& g1) {
  g0 = part * ng / np;
  g1 = (part + 1) * ng / np;
}

// Row absmax over the parts.  Thread 0 of the part stores 1 + the bits of its own
// maximum (non-negative floats order as their bit patterns; 0 marks an empty slot) in
// slot [row][part] (one 128-byte line per row), then reads the row's first four slots,
// pausing between reads so that the pollers of a line leave the store of the last part
// a way in, until the first np are set; the
// slots are cleared for the next launch once every part of the launch is past this
// point.  A slot holds only its own value, so relaxed accesses suffice.  Bounded: on
// timeout the error word is set and the part's own maximum stands in.
__device__ __forceinline__ float part_absmax_exchange(uint32_t* slots, int np, int part, float mine,
                                                      long long wait_cycles, int* err) {
  asm volatile("st.relaxed.gpu.global.u32 [%0], %1;" ::"l"(slots + part), "r"(__float_as_uint(mine) + 1u) : "memory");
  const long long t0 = clock64();
  while (true) {
    uint32_t v[4];
    asm volatile("ld.relaxed.gpu.global.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3])
                 : "l"(slots)
                 : "memory");
    bool all = true;
    uint32_t m = 0u;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < np) {
        all = all && v[i] != 0u;
        m = v[i] > m ? v[i] : m;
      }
    if (all) return __uint_as_float(m - 1u);
    if (clock64() - t0 > wait_cycles) {
      atomicCAS(err, 0, (int)kDevTimeoutRowMax);
      return mine;
    }
    __nanosleep(100);
  }
}

// The part's largest |y| from the fp32 of each thread's largest |y| (`tmax`, >= 0): one
// redux per warp on the bit patterns, the 8 warp maxima through `redf`, then the
// exchange between the parts (thread 0) and its broadcast.  Two barriers.
template <class Sync>
__device__ __forceinline__ float part_row_absmax(const RQArgs& a, int row, int part, float tmax, float* redf, int tid,
                                                 Sync sync, long long wait_cycles, int* err) {
  const uint32_t wmax = __reduce_max_sync(0xffffffffu, __float_as_uint(tmax));
  if ((tid & 31) == 0) redf[tid >> 5] = __uint_as_float(wmax);
  sync();
  if (tid == 0) {
    float pm = redf[0];
#pragma unroll
    for (int w = 1; w < kRQThreads / 32; ++w) pm = fmaxf(pm, redf[w]);
    // debug builds: one of the 64 slot lines and a part of the row (site 6)
    redf[8] = DPTQ_CHECK(row < 64 && part < a.np && a.np <= 4, err, 6)
                  ? part_absmax_exchange(a.pmax + kRowMaxStride * row, a.np, part, pm, wait_cycles, err)
                  : pm;
  }
  sync();
  return redf[8];
}

// Codes k .. k + 3 of `row` (k % 4 == 0) into the GEMM operand planes (the 128-byte
// swizzled K-major layout of rotate_quant_row<kRQAct>).
__device__ __forceinline__ void part_store4(const RQArgs& a, int row, int k, uint32_t w0, uint32_t w1, int* err) {
  uint8_t* act = static_cast<uint8_t*>(a.out);
  // debug builds: inside the operand planes (site 4)
  if (!DPTQ_CHECK(row < a.rows_out && k >= 0 && k + 4 <= a.KB * 128 && (k & 3) == 0, err, 4)) return;
  const int kb = k >> 7, j = (k >> 4) & 7;
  const size_t off = ((size_t)kb * a.rows_out + row) * 128 + ((j ^ (row & 7)) << 4) + (k & 15);
  *reinterpret_cast<uint32_t*>(act + off) = w0;
  if (a.bits == 8) *reinterpret_cast<uint32_t*>(act + (size_t)a.KB * a.rows_out * 128 + off) = w1;
}

// Padding row (row >= rows_in): zero codes, the K_pad / 4 words split evenly over the
// parts, and a zero scale.
__device__ __forceinline__ void part_zero_row(const RQArgs& a, int row, int part, int tid, int* err) {
  const int W = a.KB * 32;
  for (int w = W * part / a.np + tid; w < W * (part + 1) / a.np; w += kRQThreads) part_store4(a, row, 4 * w, 0u, 0u, err);
  if (part == 0 && tid == 0 && a.scales != nullptr) a.scales[row] = 0.f;
}

// Staged E4M3 byte(s) of one code: plane 0 (A4, or the A8 hi part) and plane 1 (A8 lo).
__device__ __forceinline__ void part_code_bytes(float q, int bits, uint32_t& b0, uint32_t& b1) {
  if (bits == 4) {
    b0 = e4m3_byte(q);
    b1 = 0u;
  } else {
    const float m = fabsf(q);
    const float h = __fmul_rn(floorf(__fmul_rn(m, 0.0625f)), 16.f);
    b0 = e4m3_byte(__fadd_rn(copysignf(h, q), 0.0f));   // + 0: no negative zeros
    b1 = e4m3_byte(__fadd_rn(copysignf(__fsub_rn(m, h), q), 0.0f));
  }
}

// Whole blocks: this part's granules [c0, c0 + len) of the row (len <= 4096), rotated as
// one chunk (16 values per thread, the three-round butterflies of rq_bfly_compact), its
// codes staged in shared memory and stored as 32-bit words of four consecutive codes.
// smem: kRQPartSmemBytes, 16-byte aligned; 256 threads meet at sync(); the caller
// synchronizes before reusing smem.
template <class Sync>
__device__ __forceinline__ void rotate_quant_part_blocks(const RQArgs& a, int row, int part, unsigned char* smem,
                                                         int tid, Sync sync, long long wait_cycles, int* err) {
  long long* sx = reinterpret_cast<long long*>(smem);
  uint8_t* stg = smem;   // staged codes [2][4096] (plane 1 at +4096), in sx once its readers are done
  float* redf = reinterpret_cast<float*>(smem + (size_t)kChunkPadded * 8 + 2 * kChunk);
  unsigned long long* const tr = DPTQ_TRACE_BUF();
  (void)tr;
  if (row >= a.rows_in) {
    part_zero_row(a, row, part, tid, err);
    return;
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 170);
  const int K = a.K;
  const int tail_start = a.nfull << a.log2B;
  const int gr = a.B > 128 ? a.B : 128;
  int g0, g1;
  part_granules((K + gr - 1) / gr, a.np, part, g0, g1);
  const int c0 = min(K, g0 * gr);
  const int len = min(K, g1 * gr) - c0;   // 0 .. 4096, a multiple of 32
  long long f[16];
  {
    uint4 u[2];
    rq_load16(reinterpret_cast<const uint4*>(a.x + (size_t)row * K), c0, len, tid, u);
    rq_fix16(a, u, c0, len, tid, f);
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 171);
  const int L = len > 0 ? rq_bfly_compact(a, c0, len, tail_start, f, sx, tid, sync) : 2;
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 176);
  // Block size of the part's values: one size unless the part reaches into the tail
  // block from a whole block.  Values past len are zero (whole zero blocks).
  const bool mixed = c0 < tail_start && c0 + len > tail_start;
  const int lgp = c0 >= tail_start ? a.log2T : a.log2B;
  float tmax;
  if (!mixed) {
    long long m[8];   // pairwise tree of |S|
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const long long p = f[e] < 0 ? -f[e] : f[e], q = f[e + 8] < 0 ? -f[e + 8] : f[e + 8];
      m[e] = p > q ? p : q;
    }
#pragma unroll
    for (int w = 4; w > 0; w >>= 1)
#pragma unroll
      for (int e = 0; e < w; ++e) m[e] = m[e] > m[e + w] ? m[e] : m[e + w];
    tmax = m[0] ? fixed_to_rotated(m[0], lgp, a.c_hi, a.c_lo) : 0.f;
  } else {
    long long mB = 0, mT = 0;
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      const long long v = f[e] < 0 ? -f[e] : f[e];
      if (c0 + rq_pos(L, tid, e) < tail_start)
        mB = v > mB ? v : mB;
      else
        mT = v > mT ? v : mT;
    }
    tmax = fmaxf(mB ? fixed_to_rotated(mB, a.log2B, a.c_hi, a.c_lo) : 0.f,
                 mT ? fixed_to_rotated(mT, a.log2T, a.c_hi, a.c_lo) : 0.f);
  }
  // The fp32 values, converted before the exchange so that their arithmetic overlaps it
  // (the conversion is odd and monotone: the fp32 of the largest |S| is the largest |y|).
  // This code runs once per launch from a cold instruction cache, so the uniform choices
  // (one block size or two, even or odd log2) are taken once, outside the unrolled loops.
  float y[16];
  if (!mixed && (lgp & 1) == 0) {
    const float sc = __int_as_float((127 - 24 - (lgp >> 1)) << 23);   // 2^-(24 + lgp / 2), exact
#pragma unroll
    for (int e = 0; e < 16; ++e) y[e] = __fmul_rn(ll_to_float_rn(f[e]), sc);
  } else if (!mixed) {
#pragma unroll
    for (int e = 0; e < 16; ++e) y[e] = fixed_times_const(f[e], lgp >> 1, a.c_hi, a.c_lo);
  } else {   // a part that reaches from a whole block into the tail block (rare)
#pragma unroll
    for (int e = 0; e < 16; ++e)
      y[e] = fixed_to_rotated(f[e], (c0 + rq_pos(L, tid, e) < tail_start) ? a.log2B : a.log2T, a.c_hi, a.c_lo);
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 140);
  const float amax = part_row_absmax(a, row, part, tmax, redf, tid, sync, wait_cycles, err);   // also ends sx's reads
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 141);
  const int bits = a.bits;
  const float qmaxf = (float)((1 << (bits - 1)) - 1), qminf = -(float)(1 << (bits - 1));
  const float s = __fdiv_rn(amax, qmaxf);
  const bool nz = amax > 0.f;
  const float rs = nz ? __frcp_rn(s) : 0.f;
  if (part == 0 && tid == 0 && a.scales != nullptr) a.scales[row] = nz ? s : 0.f;
  // Codes into the staging bytes at their positions; A4 and A8 each in a loop of their own.
  const int ib = L == 2 ? tid : L == 1 ? 256 * (tid >> 4) + (tid & 15) : 16 * tid;   // position of value 0
  const int is = L == 2 ? 256 : L == 1 ? 16 : 1;                                       // and the stride
  if (bits == 4) {
#pragma unroll
    for (int g4 = 0; g4 < 4; ++g4) {
      const float yy[4] = {y[4 * g4], y[4 * g4 + 1], y[4 * g4 + 2], y[4 * g4 + 3]};
      float q[4] = {0.f, 0.f, 0.f, 0.f};
      if (nz) quant_code4(yy, s, rs, qminf, qmaxf, q);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = ib + is * (4 * g4 + j);
        if (i < len) stg[i] = (uint8_t)e4m3_byte(q[j]);
      }
    }
  } else {
#pragma unroll
    for (int g4 = 0; g4 < 4; ++g4) {
      const float yy[4] = {y[4 * g4], y[4 * g4 + 1], y[4 * g4 + 2], y[4 * g4 + 3]};
      float q[4] = {0.f, 0.f, 0.f, 0.f};
      if (nz) quant_code4(yy, s, rs, qminf, qmaxf, q);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int i = ib + is * (4 * g4 + j);
        if (i < len) {
          uint32_t b0, b1;
          part_code_bytes(q[j], 8, b0, b1);
          stg[i] = (uint8_t)b0;
          stg[kChunk + i] = (uint8_t)b1;
        }
      }
    }
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 142);
  sync();
  // Word j of this thread, found directly from the layout: L = 2 (value e at 256 e + t),
  // L = 1 (256 (t >> 4) + 16 e + (t & 15)), L = 0 (16 t + e).
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int i = L == 2 ? 4 * (j * kRQThreads + tid) : L == 1 ? 256 * (tid >> 4) + 4 * (j * 16 + (tid & 15)) : 16 * tid + 4 * j;
    if (i < len)
      part_store4(a, row, c0 + i, *reinterpret_cast<const uint32_t*>(stg + i),
                  *reinterpret_cast<const uint32_t*>(stg + kChunk + i), err);
  }
  if (part == a.np - 1)   // k in [K, K_pad): zero codes
    for (int k = K + 4 * tid; k < a.KB * 128; k += 4 * kRQThreads) part_store4(a, row, k, 0u, 0u, err);
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 143);
}

// Block slices: output slice ps of block blk (B = n L, L = 256 V), thread t owning slice
// positions V t .. V t + V - 1.  v = sum_a (-1)^popc(ps & a) x_a (exact), then the L-point
// butterflies: log2 V levels in registers, 5 across the lanes (shuffles), 3 across the 8
// warps (one exchange through shared memory, groups of 8 values on 32 V threads); the
// codes go out as words without staging.  smem as rotate_quant_part_blocks.
template <int V, class Sync>
__device__ __forceinline__ void rotate_quant_part_slice(const RQArgs& a, int row, int part, unsigned char* smem,
                                                        int tid, Sync sync, long long wait_cycles, int* err) {
  static_assert(V == 4 || V == 8, "4 or 8 values per thread");
  constexpr int L = 256 * V;
  constexpr int U = L / 8;   // threads of the warp-level step
  long long* sx = reinterpret_cast<long long*>(smem);   // [L], unpadded
  float* redf = reinterpret_cast<float*>(smem + (size_t)kChunkPadded * 8 + 2 * kChunk);
  unsigned long long* const tr = DPTQ_TRACE_BUF();
  (void)tr;
  if (row >= a.rows_in) {
    part_zero_row(a, row, part, tid, err);
    return;
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 170);
  const int n = a.B / L;   // parts per block: 2 or 4
  const int ps = part % n;
  const int k0 = (part / n) * a.B + V * tid;   // this thread's position in input slice 0
  // debug builds: the n slices lie inside the row (site 5); a failed check reads slice 0
  const bool in_row = DPTQ_CHECK(k0 + (n - 1) * L + V <= a.K && n <= 4, err, 5);
  const __half* xr = a.x + (size_t)row * a.K + (in_row ? k0 : 0);
  uint32_t raw[4][V / 2];   // the n slices' V fp16 values, all requested before any use
#pragma unroll
  for (int sl = 0; sl < 4; ++sl)
    if (sl < n) {
      if constexpr (V == 4) {
        const uint2 w = *reinterpret_cast<const uint2*>(xr + sl * L);
        raw[sl][0] = w.x;
        raw[sl][1] = w.y;
      } else {
        const uint4 w = *reinterpret_cast<const uint4*>(xr + sl * L);
        raw[sl][0] = w.x;
        raw[sl][1] = w.y;
        raw[sl][2] = w.z;
        raw[sl][3] = w.w;
      }
    }
  long long v[V];
#pragma unroll
  for (int i = 0; i < V; ++i) v[i] = 0;
#pragma unroll
  for (int sl = 0; sl < 4; ++sl)
    if (sl < n) {
      uint32_t sg = 0u;   // sign bits of the randomized Hadamard, one per value
      if (a.signs != nullptr) {
        const int8_t* sp = a.signs + k0 + sl * L;
#pragma unroll
        for (int i = 0; i < V; ++i) sg |= (sp[i] < 0 ? 1u : 0u) << i;
      }
      const bool neg = __popc(ps & sl) & 1;   // H_n[ps][sl] = -1
#pragma unroll
      for (int i = 0; i < V; ++i) {
        long long t = half_to_fixed(i & 1 ? raw[sl][i >> 1] >> 16 : raw[sl][i >> 1] & 0xFFFFu);
        if ((sg >> i) & 1u) t = -t;
        v[i] = neg ? v[i] - t : v[i] + t;
      }
    }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 171);
#pragma unroll
  for (int h = 1; h < V; h <<= 1)
#pragma unroll
    for (int i = 0; i < V; ++i)
      if ((i & h) == 0) {
        const long long p = v[i], q = v[i + h];
        v[i] = p + q;
        v[i + h] = p - q;
      }
  const int lane = tid & 31;
#pragma unroll
  for (int b = 0; b < 5; ++b) {
    const bool up = (lane >> b) & 1;   // the higher position of the pair
#pragma unroll
    for (int i = 0; i < V; ++i) {
      const long long o = __shfl_xor_sync(0xffffffffu, v[i], 1 << b);
      v[i] = up ? o - v[i] : v[i] + o;
    }
  }
#pragma unroll
  for (int i = 0; i < V; i += 2) *reinterpret_cast<longlong2*>(sx + V * tid + i) = make_longlong2(v[i], v[i + 1]);
  sync();
  if (tid < U) {
    long long w[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) w[k] = sx[tid + U * k];
#pragma unroll
    for (int h = 1; h < 8; h <<= 1)
#pragma unroll
      for (int k = 0; k < 8; ++k)
        if ((k & h) == 0) {
          const long long p = w[k], q = w[k + h];
          w[k] = p + q;
          w[k + h] = p - q;
        }
#pragma unroll
    for (int k = 0; k < 8; ++k) sx[tid + U * k] = w[k];
  }
  sync();
#pragma unroll
  for (int i = 0; i < V; i += 2) {
    const longlong2 t = *reinterpret_cast<const longlong2*>(sx + V * tid + i);
    v[i] = t.x;
    v[i + 1] = t.y;
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 176);
  long long mx = 0;
#pragma unroll
  for (int i = 0; i < V; ++i) {
    const long long t = v[i] < 0 ? -v[i] : v[i];
    mx = t > mx ? t : mx;
  }
  const float tmax = mx ? fixed_to_rotated(mx, a.log2B, a.c_hi, a.c_lo) : 0.f;
  float y[V];   // exact 0 for S = 0; even or odd log2 B chosen once, outside the loop
  if ((a.log2B & 1) == 0) {
    const float sc = __int_as_float((127 - 24 - (a.log2B >> 1)) << 23);
#pragma unroll
    for (int i = 0; i < V; ++i) y[i] = __fmul_rn(ll_to_float_rn(v[i]), sc);
  } else {
#pragma unroll
    for (int i = 0; i < V; ++i) y[i] = fixed_times_const(v[i], a.log2B >> 1, a.c_hi, a.c_lo);
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 140);
  const float amax = part_row_absmax(a, row, part, tmax, redf, tid, sync, wait_cycles, err);
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 141);
  const int bits = a.bits;
  const float qmaxf = (float)((1 << (bits - 1)) - 1), qminf = -(float)(1 << (bits - 1));
  const float s = __fdiv_rn(amax, qmaxf);
  const bool nz = amax > 0.f;
  const float rs = nz ? __frcp_rn(s) : 0.f;
  if (part == 0 && tid == 0 && a.scales != nullptr) a.scales[row] = nz ? s : 0.f;
  const int kout = (part / n) * a.B + ps * L + V * tid;   // first output position of this thread
#pragma unroll
  for (int g4 = 0; g4 < V / 4; ++g4) {
    const float yy[4] = {y[4 * g4], y[4 * g4 + 1], y[4 * g4 + 2], y[4 * g4 + 3]};
    float q[4] = {0.f, 0.f, 0.f, 0.f};
    if (nz) quant_code4(yy, s, rs, qminf, qmaxf, q);
    uint32_t w0 = 0u, w1 = 0u;
    if (bits == 4) {
#pragma unroll
      for (int j = 0; j < 4; ++j) w0 |= e4m3_byte(q[j]) << (8 * j);
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint32_t b0, b1;
        part_code_bytes(q[j], 8, b0, b1);
        w0 |= b0 << (8 * j);
        w1 |= b1 << (8 * j);
      }
    }
    part_store4(a, row, kout + 4 * g4, w0, w1, err);
  }
  if (tid == 0) DPTQ_TRACE_CLOCK(tr, 143);
}

}  // namespace dptq
