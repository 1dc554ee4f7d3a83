// qgemm.cu -- integer GEMM of packed int4 weights against 4/8-bit activation codes on
// the sm_103a tensor cores, with exact int32 results and the scale epilogue
// (Section 2: Y = X W^T with both operands dequantized as s * c, Eq. 2; Section 4.2:
// per-token activation scales, per-channel weight scales).
//
// sm_103a exposes no integer tcgen05 MMA, so the integers travel through FP8 E4M3,
// where they are exact:
//   * a weight code q in [-7, 7] is stored as a sign-magnitude nibble; the nibble
//     placed in the low bits of a byte (sign moved to bit 7) is the E4M3 subnormal
//     q * 2^-9, so widening is two mask-and-shift operations per four weights;
//   * a 4-bit activation code is an E4M3 normal number;
//   * an 8-bit activation code c is split into c = hi + lo with hi = sign*16*(|c|>>4)
//     and lo = sign*(|c|&15), both exact in E4M3, and both planes are multiplied into
//     the same accumulator.
// Every product and every partial sum is then an integer multiple of 2^-9; as long as
// the sum of |products| of one accumulator stays below 2^24 units the fp32 tensor-core
// accumulation is exact.  K is cut into segments of `seg_blocks` k-blocks with their
// own accumulators when a tile could exceed that bound (8-bit codes, K > 18688).
//
// Operand roles (swap-AB): A (MMA M = 128) = weight rows, B (MMA N = NT) = tokens.
// D[n][m] lives in TMEM with lane = output channel and column = token.
//
// Warp roles of the persistent CTA (one per SM):
//   warp 0      producer: bulk copies (TMA engine) of packed weight tiles and of the
//               pre-swizzled E4M3 activation tiles into a `stages`-deep ring
//   warp 1      TMEM allocator + single-thread tcgen05.mma issuer
//   warps 2-5   converters: packed int4 -> E4M3 in the 128-byte swizzle layout
//   warps 6-9   epilogue: tcgen05.ld -> int32 -> scales -> fp16, or int32 atomics into
//               the split-tile scratch, the last contributor finishing the tile
// Work: whole tiles round-robin first (`dp_tiles`), then the remaining tiles' k-blocks
// split evenly over the CTAs (stream-K), so every SM streams the same number of
// weight bytes.
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "dptq_device.cuh"
#include "dptq_internal.h"

namespace dptq {

constexpr int kGemmThreads = 320;
constexpr int kConvWarp0 = 2, kNumConvWarps = 4;
constexpr int kEpiWarp0 = 6, kNumEpiWarps = 4;
constexpr int kConvBytes = 128 * 128;   // one weight tile widened to E4M3
constexpr int kMaxStages = 8;
constexpr int kSmemLimit = 232448;      // 227 KB opt-in dynamic shared memory per CTA
constexpr int kBarrierBytes = 1024;

struct Unit {
  int tile;
  int kb0, kb1;
  int slot;          // split-tile scratch slot, -1 when this CTA owns the whole tile
  int contributors;  // CTAs that add into the slot
};

// Deterministic enumeration of one CTA's work; every warp role walks the same list.
struct UnitIter {
  int cta, G, KB, dp_tiles, dp_next;
  long long sk_iters, it, it_end;

  __device__ __forceinline__ long long sk_begin(int c) const { return ((long long)c * sk_iters) / G; }
  __device__ __forceinline__ int cta_of(long long i) const {
    return (int)(((i + 1) * (long long)G - 1) / sk_iters);
  }
  __device__ __forceinline__ void init(const GemmArgs& a) {
    cta = blockIdx.x;
    G = gridDim.x;
    KB = a.KB;
    dp_tiles = a.dp_tiles;
    dp_next = cta;
    sk_iters = a.sk_iters;
    it = sk_iters > 0 ? sk_begin(cta) : 0;
    it_end = sk_iters > 0 ? sk_begin(cta + 1) : 0;
  }
  __device__ __forceinline__ bool next(Unit& u) {
    if (dp_next < dp_tiles) {
      u.tile = dp_next;
      u.kb0 = 0;
      u.kb1 = KB;
      u.slot = -1;
      u.contributors = 1;
      dp_next += G;
      return true;
    }
    if (it >= it_end) return false;
    const long long t = it / KB;
    const int kb0 = (int)(it - t * KB);
    const long long left = it_end - it;
    const int kb1 = (int)((long long)(KB - kb0) < left ? KB : kb0 + left);
    const int c0 = cta_of(t * KB), c1 = cta_of(t * KB + KB - 1);
    u.tile = dp_tiles + (int)t;
    u.kb0 = kb0;
    u.kb1 = kb1;
    u.slot = (c0 == c1) ? -1 : c0;
    u.contributors = c1 - c0 + 1;
    it += kb1 - kb0;
    return true;
  }
};

// Widen four sign-magnitude nibbles (low halves of the bytes of w) to E4M3 subnormals.
__device__ __forceinline__ uint32_t widen_lo(uint32_t w) {
  return (w & 0x07070707u) | ((w << 4) & 0x80808080u);
}
// ... and the four high halves (whose sign bit already sits at bit 7).
__device__ __forceinline__ uint32_t widen_hi(uint32_t w) {
  return ((w >> 4) & 0x07070707u) | (w & 0x80808080u);
}

template <int NT>
struct Smem {
  static constexpr int kActBytes = NT * 128;  // one plane of the token tile
  uint8_t* base;
  int stages, planes;
  __device__ __forceinline__ int stage_bytes() const { return kConvBytes + planes * kActBytes + kWTileBytes; }
  __device__ __forceinline__ uint8_t* conv(int s) const { return base + s * stage_bytes(); }
  __device__ __forceinline__ uint8_t* act(int s, int p) const { return conv(s) + kConvBytes + p * kActBytes; }
  __device__ __forceinline__ uint8_t* wpack(int s) const { return conv(s) + kConvBytes + planes * kActBytes; }
};

template <int NT>
__global__ void __launch_bounds__(kGemmThreads, 1) qgemm_kernel(const GemmArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = a.stages;
  Smem<NT> sm{smem, S, a.planes};
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S * sm.stage_bytes());
  uint64_t* full = bars;
  uint64_t* convb = bars + kMaxStages;
  uint64_t* empty = bars + 2 * kMaxStages;
  uint64_t* tfull = bars + 3 * kMaxStages;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* esync = drain + 1;   // epilogue-group barrier (4 warps), bounded waits
  uint32_t* tmem_base_sh = reinterpret_cast<uint32_t*>(esync + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_base_sh + 1);
  volatile int* last_flag = reinterpret_cast<volatile int*>(tmem_base_sh + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&convb[s], kNumConvWarps);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kNumEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_init(esync, kNumEpiWarps);
    *abort_flag = 0;
    *last_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_base_sh, a.tmem_cols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_base_sh;
  pdl_launch_dependents();

  UnitIter iter;
  iter.init(a);
  Unit un;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol_w = l2_policy_evict_first();   // weights are streamed once
      const uint64_t pol_a = l2_policy_evict_last();    // activations are re-read per n-tile
      const uint32_t act_bytes = (uint32_t)NT * 128;
      const uint32_t tx = (uint32_t)kWTileBytes + (uint32_t)a.planes * act_bytes;
      const size_t plane_stride = (size_t)a.KB * a.M_pad * 128;
      // Weight tiles do not depend on the previous kernel; the first `S` stages are
      // requested before waiting for it (programmatic dependent launch) and their
      // activation halves are issued once the previous kernel has finished.
      bool waited = false;
      int npend = 0;
      int pend_s[kMaxStages];
      const uint8_t* pend_src[kMaxStages];
      int g = 0;
      while (iter.next(un)) {
        const int nt = un.tile / a.m_tiles;
        const int mt = un.tile - nt * a.m_tiles;
        for (int kb = un.kb0; kb < un.kb1; ++kb, ++g) {
          const int s = g % S;
          if (!mbar_wait(&empty[s], ((g / S) & 1) ^ 1, abort_flag, a.err, kDevTimeoutEmpty)) goto producer_done;
          mbar_arrive_expect_tx(&full[s], tx);
          bulk_g2s(sm.wpack(s), a.wt + ((size_t)nt * a.KB + kb) * kWTileBytes, kWTileBytes, &full[s], pol_w);
          const uint8_t* asrc = a.act + ((size_t)kb * a.M_pad + (size_t)mt * NT) * 128;
          if (waited) {
            for (int p = 0; p < a.planes; ++p)
              bulk_g2s(sm.act(s, p), asrc + p * plane_stride, act_bytes, &full[s], pol_a);
          } else {
            pend_s[npend] = s;
            pend_src[npend] = asrc;
            ++npend;
            if (npend == S) {
              pdl_wait();
              waited = true;
              for (int i = 0; i < npend; ++i)
                for (int p = 0; p < a.planes; ++p)
                  bulk_g2s(sm.act(pend_s[i], p), pend_src[i] + p * plane_stride, act_bytes, &full[pend_s[i]], pol_a);
              npend = 0;
            }
          }
        }
      }
      if (!waited) {
        pdl_wait();
        for (int i = 0; i < npend; ++i)
          for (int p = 0; p < a.planes; ++p)
            bulk_g2s(sm.act(pend_s[i], p), pend_src[i] + p * plane_stride, act_bytes, &full[pend_s[i]], pol_a);
      }
    producer_done:
      // Do not leave the CTA while copies into its shared memory may be in flight.
      if (*abort_flag) {
        volatile int no_abort = 0;
        for (int gg = (g > S ? g - S : 0); gg < g; ++gg)
          mbar_wait(&full[gg % S], (gg / S) & 1, &no_abort, a.err, kDevTimeoutDrain);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_e4m3_m128(NT);
      int g = 0, u = 0;
      while (iter.next(un)) {
        const int b = a.nbuf == 2 ? (u & 1) : 0;
        const uint32_t tpar = ((a.nbuf == 2 ? (u >> 1) : u) & 1) ^ 1;
        if (!mbar_wait(&tempty[b], tpar, abort_flag, a.err, kDevTimeoutTmemEmpty)) break;
        tc_fence_after();
        const uint32_t dbase = tmem_base + (uint32_t)(b * NT * a.segs);
        const int seg0 = un.kb0 / a.seg_blocks;
        bool ok = true;
        for (int kb = un.kb0; kb < un.kb1; ++kb, ++g) {
          const int s = g % S;
          if (!mbar_wait(&convb[s], (g / S) & 1, abort_flag, a.err, kDevTimeoutConv)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = dbase + (uint32_t)((kb / a.seg_blocks - seg0) * NT);
          const bool fresh = (kb == un.kb0) || (kb % a.seg_blocks == 0);
          const uint64_t ad = sdesc_sw128(smem_u32(sm.conv(s)));
          for (int p = 0; p < a.planes; ++p) {
            const uint64_t bd = sdesc_sw128(smem_u32(sm.act(s, p)));
#pragma unroll
            for (int ks = 0; ks < 4; ++ks)   // 4 x (K = 32 FP8 elements = 32 bytes)
              mma_f8(d, ad + 2 * ks, bd + 2 * ks, idesc, (fresh && p == 0 && ks == 0) ? 0u : 1u);
          }
          mma_commit(&empty[s]);
        }
        if (!ok) break;
        mma_commit(&tfull[b]);
        ++u;
      }
      // Every MMA this thread issued must be complete before TMEM is released.
      mma_commit(drain);
      volatile int no_abort = 0;
      mbar_wait(drain, 0, &no_abort, a.err, kDevTimeoutDrain);
    }
  } else if (warp < kEpiWarp0) {
    // ------------------------------------------------------------ converters
    const int ctid = threadIdx.x - kConvWarp0 * 32;   // 0..127
    int g = 0;
    while (iter.next(un)) {
      bool ok = true;
      for (int kb = un.kb0; kb < un.kb1; ++kb, ++g) {
        const int s = g % S;
        if (!mbar_wait(&full[s], (g / S) & 1, abort_flag, a.err, kDevTimeoutFull)) {
          ok = false;
          break;
        }
        const uint8_t* wp = sm.wpack(s);
        uint8_t* cv = sm.conv(s);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int unit = i * 128 + ctid;   // (row r, 16-weight chunk j)
          const int r = unit >> 3, j = unit & 7;
          const uint2 w = *reinterpret_cast<const uint2*>(wp + r * 64 + j * 8);
          const uint4 o = make_uint4(widen_lo(w.x), widen_hi(w.x), widen_lo(w.y), widen_hi(w.y));
          *reinterpret_cast<uint4*>(cv + r * 128 + ((j ^ (r & 7)) << 4)) = o;
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&convb[s]);
      }
      if (!ok) break;
    }
  } else {
    // ------------------------------------------------------------ epilogue
    pdl_wait();   // scales come from the previous kernel; `out` may still be read by it
    const int q = warp & 3;                    // TMEM lane quarter of this warp
    const int etid = threadIdx.x - kEpiWarp0 * 32;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    int esync_phase = 0;
    // All four epilogue warps meet here; waits are bounded, so an aborted pipeline can
    // never strand a warp.
    auto epi_sync = [&]() -> bool {
      __syncwarp();
      if (lane == 0) mbar_arrive(esync);
      const bool ok = mbar_wait(esync, (uint32_t)(esync_phase & 1), abort_flag, a.err, kDevTimeoutTmemFull);
      ++esync_phase;
      return ok;
    };
    int u = 0;
    while (iter.next(un)) {
      const int b = a.nbuf == 2 ? (u & 1) : 0;
      const uint32_t tpar = (a.nbuf == 2 ? (u >> 1) : u) & 1;
      if (!mbar_wait(&tfull[b], tpar, abort_flag, a.err, kDevTimeoutTmemFull)) break;
      tc_fence_after();
      const int nt = un.tile / a.m_tiles;
      const int mt = un.tile - nt * a.m_tiles;
      const int n = nt * 128 + q * 32 + lane;
      const int m0 = mt * NT;
      const int nseg = (un.kb1 - 1) / a.seg_blocks - un.kb0 / a.seg_blocks + 1;
      const uint32_t tb = tmem_base + lane_base + (uint32_t)(b * NT * a.segs);
      const float swn = n < a.N ? a.sw[n] : 0.f;
      int32_t* wsl = un.slot >= 0 ? a.ws + (size_t)un.slot * (NT * 128) : nullptr;
#pragma unroll 1
      for (int c0 = 0; c0 < NT; c0 += 16) {
        int acc[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) acc[i] = 0;
        for (int sg = 0; sg < nseg; ++sg) {
          uint32_t r[16];
          tmem_ld16(tb + (uint32_t)(sg * NT + c0), r);
          tmem_ld_wait();
#pragma unroll
          for (int i = 0; i < 16; ++i) acc[i] += __float2int_rn(__uint_as_float(r[i]) * 512.f);
        }
        if (wsl == nullptr) {
          if (n < a.N) {
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const int m = m0 + c0 + i;
              if (m < a.M) {
                const float t = __fmul_rn(__int2float_rn(acc[i]), a.sa[m]);
                a.out[(size_t)m * a.N + n] = __float2half_rn(__fmul_rn(t, swn));
                if (a.acc_out) a.acc_out[(size_t)m * a.N + n] = acc[i];
              }
            }
          }
        } else {
#pragma unroll
          for (int i = 0; i < 16; ++i) atomicAdd(wsl + (c0 + i) * 128 + q * 32 + lane, acc[i]);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[b]);
      ++u;
      if (wsl != nullptr) {
        // Split tile: publish this CTA's part, and let the last contributor finish.
        __threadfence();
        if (!epi_sync()) break;
        if (etid == 0) {
          const unsigned prev = atomicAdd(a.counters + un.slot, 1u);
          const int last = prev == (unsigned)(un.contributors - 1);
          if (last) a.counters[un.slot] = 0u;   // every contributor has arrived
          *last_flag = last;
        }
        if (!epi_sync()) break;
        if (*last_flag) {
          __threadfence();
          for (int c = 0; c < NT; ++c) {
            int32_t* p = wsl + c * 128 + q * 32 + lane;
            const int v = __ldcg(p);
            __stcg(p, 0);   // leave the scratch zeroed for the next launch
            const int m = m0 + c;
            if (n < a.N && m < a.M) {
              const float t = __fmul_rn(__int2float_rn(v), a.sa[m]);
              a.out[(size_t)m * a.N + n] = __float2half_rn(__fmul_rn(t, swn));
              if (a.acc_out) a.acc_out[(size_t)m * a.N + n] = v;
            }
          }
        }
        if (!epi_sync()) break;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, a.tmem_cols);
  }
}

// ------------------------------------------------------------------ host planning
int gemm_pick_nt(int M, int bits, int KB) {
  (void)KB;
  if (M <= 16) return 16;
  if (M <= 32) return 32;
  if (M <= 64) return 64;
  if (M <= 128 || bits == 8) return 128;
  return 256;
}

template <int NT>
static int gemm_smem_bytes(int stages, int planes) {
  return 1024 + stages * (kConvBytes + planes * NT * 128 + kWTileBytes) + kBarrierBytes;
}

static int smem_for(int nt, int stages, int planes) {
  switch (nt) {
    case 16: return gemm_smem_bytes<16>(stages, planes);
    case 32: return gemm_smem_bytes<32>(stages, planes);
    case 64: return gemm_smem_bytes<64>(stages, planes);
    case 128: return gemm_smem_bytes<128>(stages, planes);
    default: return gemm_smem_bytes<256>(stages, planes);
  }
}

bool plan_gemm(int M, int N, int K_pad, int bits, int num_sms, GemmPlan& plan) {
  GemmArgs& a = plan.args;
  const int KB = K_pad / kKBlock;
  const int planes = bits == 8 ? 2 : 1;
  // Largest |code| * |weight| per k-block, and the k-blocks one fp32 accumulator can
  // take before the exact-integer bound 2^24 could be crossed.
  const long long per_block = (long long)(bits == 8 ? 128 : 8) * 7 * kKBlock;
  int seg_blocks = (int)(((1LL << 24) - 1) / per_block);
  if (seg_blocks > KB) seg_blocks = KB;
  const int segs = ceil_div(KB, seg_blocks);
  int nt = gemm_pick_nt(M, bits, KB);
  while (nt > 16 && nt * segs > 512) nt >>= 1;
  if (nt * segs > 512) return false;
  int stages = kMaxStages;
  while (stages > 2 && smem_for(nt, stages, planes) > kSmemLimit) --stages;
  if (smem_for(nt, stages, planes) > kSmemLimit) return false;
  const int nbuf = 2 * nt * segs <= 512 ? 2 : 1;
  uint32_t cols = 32;
  while (cols < (uint32_t)(nbuf * nt * segs)) cols <<= 1;

  const int M_pad = round_up(M, nt);
  const int n_wtiles = ceil_div(N, 128);
  const int m_tiles = M_pad / nt;
  const long long tiles = (long long)n_wtiles * m_tiles;
  const long long iters = tiles * KB;
  int G = (int)(iters < num_sms ? iters : num_sms);
  if (G < 1) G = 1;
  long long dp = 0;
  if (tiles >= 2LL * G) dp = (tiles / G - 1) * G;

  plan.nt = nt;
  plan.M_pad = M_pad;
  plan.grid = G;
  plan.smem_bytes = smem_for(nt, stages, planes);
  a.M = M;
  a.N = N;
  a.M_pad = M_pad;
  a.KB = KB;
  a.planes = planes;
  a.n_wtiles = n_wtiles;
  a.m_tiles = m_tiles;
  a.seg_blocks = seg_blocks;
  a.segs = segs;
  a.nbuf = nbuf;
  a.stages = stages;
  a.dp_tiles = (int)dp;
  a.sk_iters = (tiles - dp) * KB;
  a.tmem_cols = cols;
  return true;
}

template <int NT>
static cudaError_t launch_nt(const GemmPlan& plan, cudaStream_t s, bool pdl) {
  cudaError_t e = cudaFuncSetAttribute(qgemm_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, plan.smem_bytes);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)plan.grid);
  cfg.blockDim = dim3(kGemmThreads);
  cfg.dynamicSmemBytes = (size_t)plan.smem_bytes;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, qgemm_kernel<NT>, plan.args);
}

cudaError_t launch_gemm(const GemmPlan& plan, cudaStream_t s, bool pdl) {
  switch (plan.nt) {
    case 16: return launch_nt<16>(plan, s, pdl);
    case 32: return launch_nt<32>(plan, s, pdl);
    case 64: return launch_nt<64>(plan, s, pdl);
    case 128: return launch_nt<128>(plan, s, pdl);
    case 256: return launch_nt<256>(plan, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace dptq
