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
//   warp 0      weight producer: bulk copies (TMA engine) of packed weight tiles into a
//               `stages`-deep ring (a stage holds KPS k-blocks of 128), from the start
//   warp 1      TMEM allocator + single-thread tcgen05.mma issuer
//   warps 2-9   converters: packed int4 -> E4M3 (into tensor memory, or shared memory
//               in the 128-byte swizzle layout); in a fused launch they first rotate and
//               quantize the token rows
//   warps 10-13 epilogue: tcgen05.ld -> int32 -> scales -> fp16, or partial sums into
//               the split-tile scratch, the last contributor finishing the tile
//   warp 14     activation producer: bulk copies of the pre-swizzled E4M3 activation
//               tiles into the same ring, once the previous kernel (and, fused, the row
//               quantization) is done
// Work: whole tiles round-robin first (`dp_tiles`), then the remaining tiles' k-blocks
// split evenly over the CTAs (stream-K), so every SM streams the same number of
// weight bytes.
#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "dptq_device.cuh"
#include "dptq_internal.h"
#include "rotate_row.cuh"

namespace dptq {

constexpr int kNumConvWarps = 8, kConvWarp0 = 2;
#ifndef DPTQ_TRACE_STAGES
#define DPTQ_TRACE_STAGES 16
#endif
// Trace builds record per-stage stamps for the first kTraceStages stages of each role.
constexpr int kTraceStages = DPTQ_TRACE_STAGES;
constexpr int kNumEpiWarps = 4, kEpiWarp0 = kConvWarp0 + kNumConvWarps;
constexpr int kActWarp = kEpiWarp0 + kNumEpiWarps;               // activation producer
constexpr int kGemmThreads = 32 * (kActWarp + 1);                // 480
constexpr int kConvThreads = 32 * kNumConvWarps;
constexpr int kConvBytes = 128 * 128;   // one weight tile widened to E4M3
constexpr int kMaxStages = 8;
constexpr int kMaxConvSlots = 4;
constexpr int kSmemLimit = 232448;      // 227 KB opt-in dynamic shared memory per CTA
constexpr int kBarrierBytes = 2048;   // barriers and flags, token scales (tiles <= 64), output transpose (1 KB)

struct Unit {
  int tile;
  int i0, i1;        // iteration range (stages of KPS k-blocks) within the tile
  int slot;          // split-tile scratch slot, -1 when this CTA owns the whole tile
  int contributors;  // CTAs that add into the slot
};

// Deterministic enumeration of one CTA's work; every warp role walks the same list.
// The stream-K part spans fewer than 2 * G * KI iterations (at most 2G tiles are left
// after the data-parallel rounds), so all products below fit in 32 bits (the planner
// checks this); 32-bit divisions keep the per-unit cost low.
struct UnitIter {
  uint32_t cta, G, KI, dp_tiles, dp_next;
  uint32_t sk_iters, it, it_end;

  __device__ __forceinline__ uint32_t sk_begin(uint32_t c) const { return (c * sk_iters) / G; }
  __device__ __forceinline__ uint32_t cta_of(uint32_t i) const { return ((i + 1) * G - 1) / sk_iters; }
  __device__ __forceinline__ void init(const GemmArgs& a) {
    cta = blockIdx.x;
    G = gridDim.x;
    KI = (uint32_t)a.KI;
    dp_tiles = (uint32_t)a.dp_tiles;
    dp_next = cta;
    sk_iters = (uint32_t)a.sk_iters;
    it = sk_iters > 0 ? sk_begin(cta) : 0;
    it_end = sk_iters > 0 ? sk_begin(cta + 1) : 0;
  }
  __device__ __forceinline__ bool next(Unit& u) {
    if (dp_next < dp_tiles) {
      u.tile = (int)dp_next;
      u.i0 = 0;
      u.i1 = (int)KI;
      u.slot = -1;
      u.contributors = 1;
      dp_next += G;
      return true;
    }
    if (it >= it_end) return false;
    const uint32_t t = it / KI;
    const uint32_t i0 = it - t * KI;
    const uint32_t left = it_end - it;
    const uint32_t i1 = KI - i0 < left ? KI : i0 + left;
    const uint32_t c0 = cta_of(t * KI), c1 = cta_of(t * KI + KI - 1);
    u.tile = (int)(dp_tiles + t);
    u.i0 = (int)i0;
    u.i1 = (int)i1;
    u.slot = (c0 == c1) ? -1 : (int)c0;
    u.contributors = (int)(c1 - c0 + 1);
    it += i1 - i0;
    return true;
  }
};

// Ring position (stage index and the parity of its current phase), advanced without
// divisions.
struct Ring {
  int s = 0;
  uint32_t ph = 0;
  int S;
  __device__ __forceinline__ explicit Ring(int stages) : S(stages) {}
  __device__ __forceinline__ void next() {
    if (++s == S) {
      s = 0;
      ph ^= 1u;
    }
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

// Where the widened weights (the MMA's A operand) live: tensor memory for two-block
// stages (decode) and for 192-token tiles, whose two accumulators (384 columns) leave
// 128 columns for four one-block slots; shared memory otherwise.  With the A operand in
// tensor memory a stage costs shared memory only its bulk copies and the MMA's B reads.
__host__ __device__ constexpr bool a_in_tmem(int nt, int kps) { return kps == 2 || nt == 192; }

// Shared-memory layout: a ring of `conv_slots` widened weight slots (KPS tiles of 16 KB
// each, 1024-aligned swizzle atoms; absent when the widened weights live in tensor
// memory) followed by the `stages`-deep ring of bulk-copy slots.  A bulk-copy slot holds
// KPS x planes token tiles and the KPS packed weight tiles of one stage.
template <int NT, int KPS>
struct Smem {
  static constexpr int kActBytes = NT * 128;  // one plane of one token tile
  uint8_t* base;
  int planes;
  int conv_slots;
  int slot_bytes;
  __device__ __forceinline__ Smem(uint8_t* b, int p, int cs) : base(b), planes(p), conv_slots(cs) {
    slot_bytes = KPS * (p * kActBytes + kWTileBytes);
  }
  __device__ __forceinline__ uint8_t* conv(int c, int h) const { return base + (c * KPS + h) * kConvBytes; }
  __device__ __forceinline__ uint8_t* slot(int s) const {
    return base + conv_slots * KPS * kConvBytes + s * slot_bytes;
  }
  // Plane-major within a stage, so that a plane's KPS k-blocks are adjacent (one bulk copy
  // when they are adjacent in global memory too).
  __device__ __forceinline__ uint8_t* act(int s, int h, int p) const { return slot(s) + (p * KPS + h) * kActBytes; }
  __device__ __forceinline__ uint8_t* wpack(int s) const { return slot(s) + KPS * planes * kActBytes; }
  __device__ __forceinline__ uint8_t* end(int S) const { return slot(S); }
};

// RQV != 0 (decode, two-block stages) makes the launch FUSED: it first rotates and
// quantizes the token rows itself.  Each row is split into rq_np parts, each part
// rotating only its own outputs (RQV = kPartBlocks: whole blocks per part;
// kPartSlice4 / kPartSlice8: slices of one block, 4 or 8 values per thread); the parts
// of a row exchange their maxima through global slots, and the converter warps publish
// the rows on a grid counter.  Every producer streams its first weight stages meanwhile
// and requests activation tiles once all rows are in; the epilogue reads the token
// scales after the same point, and the last CTA to get there resets the counters and
// the slots.
template <int NT, int KPS, int RQV>
__global__ void __launch_bounds__(kGemmThreads, 1) qgemm_kernel(const GemmArgs a) {
  constexpr bool FUSED = RQV != 0;
  // Two-block stages (token tiles of up to 64, weight streaming) and 192-token tiles
  // widen the weights straight into tensor memory and feed the MMA's A operand from
  // there; other one-block stages widen into shared memory.
  constexpr bool kATmem = a_in_tmem(NT, KPS);
  // Two-block stages with the widened weights in tensor memory: the converter warps form
  // two groups of four (one warp per TMEM lane quarter) that take alternate stages, each
  // warp widening both k-blocks of its quarter, so that two stages convert at once.
  constexpr bool kAltConv = kATmem && KPS == 2;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = a.stages;
  const int CS = a.conv_slots;
  const Smem<NT, KPS> sm(smem, a.planes, kATmem ? 0 : CS);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm.end(S));
  uint64_t* full = bars;                     // slot s: weight copies landed
  uint64_t* empty = bars + kMaxStages;       // slot s: MMA done with it
  uint64_t* afull = bars + 2 * kMaxStages;   // slot s: activation copies landed
  uint64_t* cfull = bars + 3 * kMaxStages;   // widened slot c: written
  uint64_t* tfull = cfull + 2 * kMaxConvSlots;
  uint64_t* tempty = tfull + 2;
  uint64_t* drain = tempty + 2;
  uint64_t* esync = drain + 1;   // epilogue-group barrier (4 warps), bounded waits
  uint64_t* aready = esync + 1;  // fused: all token rows are quantized (producer -> epilogue)
  uint32_t* tmem_base_sh = reinterpret_cast<uint32_t*>(aready + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_base_sh + 1);
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_base_sh + 2);   // epilogue: 2 units x 2
  float* sa_sh = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 512);   // token scales (NT <= 64)
  __half* xpose = reinterpret_cast<__half*>(reinterpret_cast<uint8_t*>(bars) + 1024);  // 4 x [4 tokens][32 ch]
  unsigned char* rot_smem = reinterpret_cast<unsigned char*>(bars) + kBarrierBytes;    // fused: one row's scratch

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  unsigned long long* const tr = DPTQ_TRACE_BUF();
  (void)tr;
  if (threadIdx.x == 0) DPTQ_TRACE_ENTRY(tr);

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
      mbar_init(&afull[s], 1);
    }
    for (int c = 0; c < CS; ++c) {
      mbar_init(&cfull[c], kAltConv ? kNumConvWarps / 2 : kNumConvWarps);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], kNumEpiWarps);
    }
    mbar_init(drain, 1);
    mbar_init(esync, kNumEpiWarps);
    mbar_init(aready, 1);
    *abort_flag = 0;
    for (int i = 0; i < 4; ++i) flags[i] = 0;
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
  if (threadIdx.x == 0) DPTQ_TRACE_POINT(tr, 1);
  pdl_launch_dependents();

  UnitIter iter;
  iter.init(a);
  Unit un;

  if (warp == 0 || warp == kActWarp) {
    // ------------------------------------------------------------ producers
    // Warp 0 streams the packed weight tiles, which do not depend on the previous kernel,
    // from the first moment; warp kActWarp requests the activation tiles, which do: it
    // waits for the previous kernel (programmatic dependent launch) and, in a fused
    // launch, for every token row to be published, then follows the ring.  Both walk the
    // same stages and wait for the same `empty` barriers; each arms its own barrier of a
    // stage (`full`: weights, `afull`: activations).  Whole warps, uniform control flow;
    // an elected leader issues the copies.
    const bool wprod = warp == 0;
    const bool leader = elect_one();
    if (leader && wprod) DPTQ_TRACE_POINT(tr, 117);
    const uint64_t pol_w = l2_policy_evict_first();   // weights are streamed once
    const uint64_t pol_a = l2_policy_evict_last();    // activations are re-read per n-tile
    const uint32_t act_bytes = (uint32_t)NT * 128;
    const uint32_t w_bytes = (uint32_t)KPS * kWTileBytes;
    const uint32_t a_tx = (uint32_t)(KPS * a.planes) * act_bytes;
    const size_t plane_stride = (size_t)a.KB * a.M_pad * 128;
    const size_t kb_stride = (size_t)a.M_pad * 128;
    // Decode launches: once the ring's first S stages are requested, the weight producer
    // requests the rest of its CTA's share (up to a cap) into L2, so that HBM streams the
    // weights while the ring is still full (the token rows are being rotated, or the
    // previous kernel finishes).  Units are visited in processing order; each unit's
    // weight range is contiguous (tile-major, k-blocks consecutive) and, with one token
    // tile, belongs to this CTA.
    auto prefetch_share = [&]() {
      if (!(wprod && leader && a.l2_prefetch > 0)) return;
      UnitIter pit;
      pit.init(a);
      Unit pu;
      long long skip = (long long)S * w_bytes;   // fetched by the ring directly
      long long budget = a.l2_prefetch;
      while (budget > 0 && pit.next(pu)) {
        const int tile_n = pu.tile / a.m_tiles;
        const uint8_t* base = a.wt + ((size_t)tile_n * a.KB + (size_t)pu.i0 * KPS) * kWTileBytes;
        long long len = (long long)(pu.i1 - pu.i0) * w_bytes;
        if (skip >= len) {
          skip -= len;
          continue;
        }
        base += skip;
        len -= skip;
        skip = 0;
        if (len > budget) len = budget;
        budget -= len;
        for (long long off = 0; off < len; off += 32768)
          bulk_prefetch_l2(base + off, (uint32_t)(len - off < 32768 ? len - off : 32768));
      }
    };
    // The activation producer starts once the previous kernel has finished and, in a fused
    // launch, every token row has been quantized.
    bool ok = true;
    if (!wprod) {
      pdl_wait();
      if constexpr (FUSED) {
        const long long t0 = clock64();
        while (true) {
          int st = 0;
          if (lane == 0) {
            if (ld_acquire_gpu(a.gsync) >= (uint32_t)(a.rq_items + a.rq_shortfall))
              st = 1;
            else if (*abort_flag)
              st = 2;
            else if (clock64() - t0 > a.wait_cycles) {
              *abort_flag = 1;
              atomicCAS(a.err, 0, (int)kDevTimeoutGrid);
              st = 2;
            }
          }
          st = __shfl_sync(0xffffffffu, st, 0);
          if (st == 1) break;
          if (st == 2) {
            ok = false;
            break;
          }
          __nanosleep(32);
        }
        if (ok) {
          fence_proxy_async_global();   // the bulk copies read what other CTAs stored
          if (leader) {
            DPTQ_TRACE_POINT(tr, 116);
            mbar_arrive(aready);
          }
        }
      }
    }
    Ring rg(S);
    int g = 0;
    while (ok && iter.next(un)) {
      const int nt = un.tile / a.m_tiles;
      const int mt = un.tile - nt * a.m_tiles;
      if (leader && wprod) DPTQ_TRACE_POINT(tr, 118);
      const uint8_t* wsrc = a.wt + ((size_t)nt * a.KB + (size_t)un.i0 * KPS) * kWTileBytes;
      const uint8_t* asrc = a.act + ((size_t)un.i0 * KPS * a.M_pad + (size_t)mt * NT) * 128;
      for (int it = un.i0; it < un.i1; ++it, ++g, rg.next(), wsrc += w_bytes, asrc += KPS * kb_stride) {
        const int s = rg.s;
        const bool tg = kTraceStages > 10 && wprod && leader && g >= 8 && g < 11;   // clocked stages (trace builds)
        (void)tg;
        if (FUSED && wprod && g == a.pre_stages &&
            !mbar_wait_warp(aready, 0, abort_flag, a.err, kDevTimeoutGrid, a.wait_cycles)) {
          ok = false;   // the rows never became ready
          break;
        }
        if (tg) DPTQ_TRACE_CLOCK(tr, 224 + 3 * (g - 8));
        if (!mbar_wait_warp(&empty[s], rg.ph ^ 1u, abort_flag, a.err, kDevTimeoutEmpty, a.wait_cycles)) {
          ok = false;
          break;
        }
        if (leader) {
          if (tg) DPTQ_TRACE_CLOCK(tr, 225 + 3 * (g - 8));
          if (wprod) {
            if (g < kTraceStages) DPTQ_TRACE_POINT(tr, 8 + g);
            mbar_arrive_expect_tx(&full[s], w_bytes);
            // debug builds: the stage's weight bytes lie inside the packed tiles (site 1)
            if (DPTQ_CHECK(nt < a.n_wtiles && (it + 1) * KPS <= a.KB, a.err, 1))
              bulk_g2s(sm.wpack(s), wsrc, w_bytes, &full[s], pol_w);
            if (g < kTraceStages) DPTQ_TRACE_POINT(tr, 24 + g);
            if (g == S - 1) prefetch_share();
          } else {
            mbar_arrive_expect_tx(&afull[s], a_tx);
            // debug builds: the stage's token tile lies inside the operand planes (site 2)
            if (!DPTQ_CHECK(mt < a.m_tiles && (it + 1) * KPS <= a.KB, a.err, 2)) {
              // skipped: the stage's barrier never completes, and the consumers' bounded
              // waits end the launch with the check's code already in the error word
            } else if (kb_stride == act_bytes) {
              // One token tile: a plane's KPS k-blocks are contiguous in global memory and in
              // the stage, so each plane is one copy (the bulk-copy engine's cost is largely
              // per copy).
              for (int pl = 0; pl < a.planes; ++pl)
                bulk_g2s(sm.act(s, 0, pl), asrc + pl * plane_stride, KPS * act_bytes, &afull[s], pol_a);
            } else {
#pragma unroll
              for (int h = 0; h < KPS; ++h)
                for (int pl = 0; pl < a.planes; ++pl)
                  bulk_g2s(sm.act(s, h, pl), asrc + h * kb_stride + pl * plane_stride, act_bytes, &afull[s], pol_a);
            }
          }
          if (tg) DPTQ_TRACE_CLOCK(tr, 226 + 3 * (g - 8));
        }
        __syncwarp();
      }
    }
    __syncwarp();
    // Do not leave the CTA while copies into its shared memory may be in flight: after an
    // abort, wait (bounded) for the copies this warp armed in the last S stages.
    if (*abort_flag) {
      volatile int no_abort = 0;
      for (int gg = (g > S ? g - S : 0); gg < g; ++gg)
        mbar_wait_warp(wprod ? &full[gg % S] : &afull[gg % S], (gg / S) & 1, &no_abort, a.err, kDevTimeoutDrain);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    // The whole warp runs the loop (uniform control flow, warp-wide waits) and one lane,
    // elected once, issues every MMA and commit: tcgen05 issue from a converged warp's
    // leader is about twice as fast as from a thread looping alone, and a commit tracks
    // the MMAs of the thread that issues it.  Descriptors and TMEM addresses advance by
    // additions, segment boundaries by a countdown.
    const bool leader = elect_one();
    const uint32_t idesc = idesc_e4m3_m128(NT);
    const int planes = a.planes;
    // Shared-memory descriptors hold address >> 4 in their low bits, so a byte offset
    // `o` into a region is `desc + (o >> 4)`.
    const uint64_t act_desc0 = sdesc_sw128(smem_u32(sm.act(0, 0, 0)));
    const uint64_t conv_desc0 = kATmem ? 0 : sdesc_sw128(smem_u32(sm.conv(0, 0)));
    const uint32_t slot_step = (uint32_t)(sm.slot_bytes >> 4);
    const uint32_t act_step = (uint32_t)(Smem<NT, KPS>::kActBytes >> 4);
    const uint32_t a_tmem0 = tmem_base + a.a_col0;
    Ring rg(S), rc(CS);
    int u = 0, mma_done = 0;
    while (iter.next(un)) {
      const int b = a.nbuf == 2 ? (u & 1) : 0;
      const uint32_t tpar = ((a.nbuf == 2 ? (u >> 1) : u) & 1) ^ 1;
      if (!mbar_wait_warp(&tempty[b], tpar, abort_flag, a.err, kDevTimeoutTmemEmpty, a.wait_cycles)) break;
      tc_fence_after();
      uint32_t d = tmem_base + (uint32_t)(b * NT * a.segs);
      int seg_left = a.seg_iters - un.i0 % a.seg_iters;   // iterations left in this segment
      uint32_t fresh = 1;
      bool ok = true;
      for (int it = un.i0; it < un.i1; ++it, rg.next(), rc.next()) {
        const int s = rg.s, c = rc.s;
        const int gm = it - un.i0 + mma_done;
        const bool tgm = kTraceStages > 10 && leader && gm >= 8 && gm < 11;   // stages whose steps are clocked (trace builds)
        (void)tgm;
        if (tgm) DPTQ_TRACE_CLOCK(tr, 200 + 8 * (gm - 8));
        if (!mbar_wait_warp(&afull[s], rg.ph, abort_flag, a.err, kDevTimeoutFull, a.wait_cycles)) {
          ok = false;
          break;
        }
        if (tgm) DPTQ_TRACE_CLOCK(tr, 201 + 8 * (gm - 8));
        if (!mbar_wait_warp(&cfull[c], rc.ph, abort_flag, a.err, kDevTimeoutConv, a.wait_cycles)) {
          ok = false;
          break;
        }
        if (tgm) DPTQ_TRACE_CLOCK(tr, 202 + 8 * (gm - 8));
        if (leader && gm < kTraceStages) DPTQ_TRACE_POINT(tr, 72 + gm);
        tc_fence_after();
        if (seg_left == 0) {   // next exact-accumulation segment: next accumulator
          d += NT;
          fresh = 1;
          seg_left = a.seg_iters;
        }
        const uint64_t bd_slot = act_desc0 + (uint64_t)(s * slot_step);
        if (leader) {
#pragma unroll
          for (int h = 0; h < KPS; ++h) {
            const uint64_t ad = conv_desc0 + (uint64_t)((c * KPS + h) * (kConvBytes >> 4));
            const uint32_t at = a_tmem0 + (uint32_t)((c * KPS + h) * 32);   // 32 columns per k-block
#pragma unroll
            for (int p = 0; p < 2; ++p) {
              if (p < planes) {
                const uint64_t bd = bd_slot + (uint64_t)((p * KPS + h) * act_step);
#pragma unroll
                for (int ks = 0; ks < 4; ++ks) {   // 4 x (K = 32 FP8 elements = 32 bytes = 8 columns)
                  const uint32_t accumulate = (h | p | ks) ? 1u : (fresh ^ 1u);
                  if (kATmem)
                    mma_f8_ts(d, at + (uint32_t)(8 * ks), bd + 2 * ks, idesc, accumulate);
                  else
                    mma_f8(d, ad + 2 * ks, bd + 2 * ks, idesc, accumulate);
                }
              }
            }
          }
          if (tgm) DPTQ_TRACE_CLOCK(tr, 203 + 8 * (gm - 8));
          // One commit per stage: it frees the bulk-copy slot (producer) and tells the
          // converters that widened slot c may be overwritten (they wait on the same
          // barrier, one ring position CS stages back).
          mma_commit(&empty[s]);
          if (tgm) DPTQ_TRACE_CLOCK(tr, 205 + 8 * (gm - 8));
          if (gm < kTraceStages) DPTQ_TRACE_POINT(tr, 88 + gm);
        }
        __syncwarp();
        if (tgm) DPTQ_TRACE_CLOCK(tr, 206 + 8 * (gm - 8));
        fresh = 0;
        --seg_left;
      }
      if (!ok) break;
      if (leader) mma_commit(&tfull[b]);
      __syncwarp();
      mma_done += un.i1 - un.i0;
      ++u;
    }
    if (leader) DPTQ_TRACE_POINT(tr, 124);   // last MMA issued
    // Every MMA the leader issued must be complete before TMEM is released.
    if (leader) mma_commit(drain);
    __syncwarp();
    volatile int no_abort = 0;
    mbar_wait_warp(drain, 0, &no_abort, a.err, kDevTimeoutDrain);
  } else if (warp < kEpiWarp0) {
    // ------------------------------------------------------------ converters
    const int ctid = threadIdx.x - kConvWarp0 * 32;   // 0..255
    if constexpr (FUSED) {
      // Rotate + quantize this CTA's (row, part) items into the activation planes and
      // scales, then publish them.  The 8 converter warps meet at named barrier 1.
      pdl_wait();   // the rows come from the previous kernel
      if (ctid == 0) {
        DPTQ_TRACE_POINT(tr, 125);
        DPTQ_TRACE_CLOCK(tr, 160);
      }
      const auto csync = [] { asm volatile("bar.sync 1, %0;" ::"n"(kConvThreads) : "memory"); };
      // Rows go out in rounds of G / np rows, CTA c taking part c % np of rows
      // c / np, c / np + G / np, ...: the parts of a row, which wait for one another's
      // maxima, always run in the same round.
      const int np = a.rq.np;
      const int rpr = (int)gridDim.x / np;
      int nitems = 0;
      if ((int)blockIdx.x < rpr * np) {
        const int part = (int)blockIdx.x % np;
        for (int row = (int)blockIdx.x / np; row < a.rq.rows_out; row += rpr) {
          if (nitems) csync();   // the previous row's readers are done with the scratch
          if constexpr (RQV == kPartBlocks)
            rotate_quant_part_blocks(a.rq, row, part, rot_smem, ctid, csync, a.wait_cycles, a.err);
          else
            rotate_quant_part_slice<RQV>(a.rq, row, part, rot_smem, ctid, csync, a.wait_cycles, a.err);
          ++nitems;
        }
      }
      if (ctid == 0) {
        DPTQ_TRACE_POINT(tr, 126);
        DPTQ_TRACE_CLOCK(tr, 161);
      }
      if (nitems) {
        csync();   // every converter thread's code and scale stores precede the release
        if (ctid == 0) release_add_gpu(a.gsync, (uint32_t)nitems);
      }
      if (ctid == 0) DPTQ_TRACE_POINT(tr, 127);
    }
    // rl trails rg by CS stages: the MMA of stage gc - CS was the last to read widened
    // slot c, and its commit completes that stage's `empty` barrier.
    Ring rg(S), rc(CS), rl(S);
    const int grp = (warp - kConvWarp0) >> 2;   // converter group (alternate stages)
    const int tid_grp = (warp - kConvWarp0 - 4 * grp) * 32 + lane;
    (void)tid_grp;
    int gc = 0;
    while (iter.next(un)) {
      bool ok = true;
      for (int it = un.i0; it < un.i1; ++it, ++gc, rg.next(), rc.next()) {
        const int s = rg.s, c = rc.s;
        if (gc > CS) rl.next();   // rl = ring position of stage gc - CS (from gc = CS on)
        if (kAltConv && (gc & 1) != grp) continue;   // the other group's stage
        const bool tgc = kTraceStages > 10 && (kAltConv ? tid_grp == 0 : ctid == 0) && gc >= 8 && gc < 11;   // clocked (trace builds)
        (void)tgc;
        if (tgc) DPTQ_TRACE_CLOCK(tr, 180 + 6 * (gc - 8));
        // First the MMA of stage gc - CS (widened slot c free).  It also orders the wait
        // on full[s]: a parity wait cannot tell a phase from the one two phases later,
        // and a group that skips stages could otherwise look at slot s while its previous
        // copy (stage gc - S, converted by the other group) is still in flight.  With
        // S >= CS, that copy has landed and been consumed once the MMA of stage gc - CS
        // is done.
        if (gc >= CS && !mbar_wait(&empty[rl.s], rl.ph, abort_flag, a.err, kDevTimeoutConv, a.wait_cycles)) {
          ok = false;
          break;
        }
        if (tgc) DPTQ_TRACE_CLOCK(tr, 181 + 6 * (gc - 8));
        if (!mbar_wait(&full[s], rg.ph, abort_flag, a.err, kDevTimeoutFull, a.wait_cycles)) {
          ok = false;
          break;
        }
        if (tgc) DPTQ_TRACE_CLOCK(tr, 182 + 6 * (gc - 8));
        if ((kAltConv ? tid_grp == 0 : ctid == 0) && gc < kTraceStages) DPTQ_TRACE_POINT(tr, 40 + gc);
        const uint8_t* __restrict__ wp = sm.wpack(s);
        if constexpr (kAltConv) {
          // Warp of lane quarter q widens both k-blocks of rows 32q..32q+31: each thread
          // reads its row's 2 x 64 packed bytes (4 chunks of 32 k per block) and stores
          // 2 x 32 columns of its TMEM lane.
          tc_fence_after();
          const int q = warp & 3;
          const uint8_t* src = wp + (q * 32 + lane) * 16;
          uint4 w[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) w[j] = *reinterpret_cast<const uint4*>(src + (j >> 2) * kWTileBytes + (j & 3) * 2048);
#ifdef DPTQ_TRACE
          if (tgc) {
            volatile uint32_t sink = w[0].x ^ w[7].w;
            (void)sink;
            DPTQ_TRACE_CLOCK(tr, 183 + 6 * (gc - 8));
          }
#endif
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            uint32_t v[32];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const uint4 ww = w[4 * h + j];
              v[8 * j + 0] = widen_lo(ww.x);
              v[8 * j + 1] = widen_hi(ww.x);
              v[8 * j + 2] = widen_lo(ww.y);
              v[8 * j + 3] = widen_hi(ww.y);
              v[8 * j + 4] = widen_lo(ww.z);
              v[8 * j + 5] = widen_hi(ww.z);
              v[8 * j + 6] = widen_lo(ww.w);
              v[8 * j + 7] = widen_hi(ww.w);
            }
            tmem_st32(tmem_base + ((uint32_t)(q * 32) << 16) + a.a_col0 + (uint32_t)((c * KPS + h) * 32), v);
          }
          tmem_st_wait();
          tc_fence_before();
          if (tgc) DPTQ_TRACE_CLOCK(tr, 184 + 6 * (gc - 8));
        } else if constexpr (kATmem && KPS == 1) {
          // Warp (lane quarter q, half hs) widens k columns 64 hs .. 64 hs + 63 of rows
          // 32q..32q+31: each thread reads its row's 32 packed bytes (chunks 2 hs and
          // 2 hs + 1 of 32 k) and stores 16 columns of its TMEM lane.
          tc_fence_after();
          const int q = warp & 3;
          const int hs = (warp - kConvWarp0) >> 2;
          const uint8_t* src = wp + (2 * hs) * 2048 + (q * 32 + lane) * 16;
          uint4 w[2];
#pragma unroll
          for (int j = 0; j < 2; ++j) w[j] = *reinterpret_cast<const uint4*>(src + j * 2048);
          uint32_t v[16];
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            v[8 * j + 0] = widen_lo(w[j].x);
            v[8 * j + 1] = widen_hi(w[j].x);
            v[8 * j + 2] = widen_lo(w[j].y);
            v[8 * j + 3] = widen_hi(w[j].y);
            v[8 * j + 4] = widen_lo(w[j].z);
            v[8 * j + 5] = widen_hi(w[j].z);
            v[8 * j + 6] = widen_lo(w[j].w);
            v[8 * j + 7] = widen_hi(w[j].w);
          }
          tmem_st16(tmem_base + ((uint32_t)(q * 32) << 16) + a.a_col0 + (uint32_t)(c * 32 + hs * 16), v);
          tmem_st_wait();
          tc_fence_before();
        } else {
          // Each thread widens 2 * KPS x 16 packed bytes: (tile h, row r, 16-byte chunk jj
          // = 32 weights) into swizzled chunks 2jj and 2jj + 1 of row r.  All loads are
          // issued before any store.
          uint4 w[2 * KPS];
          if (ctid == 0 && gc == 8) DPTQ_TRACE_CLOCK(tr, 230);
#pragma unroll
          for (int i = 0; i < 2 * KPS; ++i) {
            const int p = i * kConvThreads + ctid;   // 16-byte unit: tile p >> 9
            const int qq = p & 511;
            w[i] = *reinterpret_cast<const uint4*>(wp + (p >> 9) * kWTileBytes + (qq & 3) * 2048 + (qq >> 2) * 16);
          }
#ifdef DPTQ_TRACE
          if (ctid == 0 && gc == 8) {
            volatile uint32_t sink = w[0].x ^ w[2 * KPS - 1].w;
            (void)sink;
            DPTQ_TRACE_CLOCK(tr, 231);
          }
#endif
#pragma unroll
          for (int i = 0; i < 2 * KPS; ++i) {
            const int p = i * kConvThreads + ctid;
            const int qq = p & 511;
            const int r = qq >> 2, j0 = (qq & 3) * 2;
            uint8_t* row = sm.conv(c, p >> 9) + r * 128;
            *reinterpret_cast<uint4*>(row + ((j0 ^ (r & 7)) << 4)) =
                make_uint4(widen_lo(w[i].x), widen_hi(w[i].x), widen_lo(w[i].y), widen_hi(w[i].y));
            *reinterpret_cast<uint4*>(row + (((j0 + 1) ^ (r & 7)) << 4)) =
                make_uint4(widen_lo(w[i].z), widen_hi(w[i].z), widen_lo(w[i].w), widen_hi(w[i].w));
          }
          if (ctid == 0 && gc == 8) DPTQ_TRACE_CLOCK(tr, 232);
          fence_proxy_async_smem();
          if (ctid == 0 && gc == 8) DPTQ_TRACE_CLOCK(tr, 233);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&cfull[c]);
        if (tgc) DPTQ_TRACE_CLOCK(tr, 185 + 6 * (gc - 8));
        if ((kAltConv ? tid_grp == 0 : ctid == 0) && gc < kTraceStages) DPTQ_TRACE_POINT(tr, 56 + gc);
      }
      if (!ok) break;
    }
  } else {
    // ------------------------------------------------------------ epilogue
    pdl_wait();   // scales come from the previous kernel; `out` may still be read by it
    bool epi_ok = true;
    if constexpr (FUSED) {
      epi_ok = mbar_wait(aready, 0, abort_flag, a.err, kDevTimeoutGrid, a.wait_cycles);
      // This CTA's producer has passed its wait on the row counter (or gave up): the last
      // CTA to get here resets both grid counters for the next launch, which touches them
      // only after this grid ends.  Done here, while the weights still stream, the atomic's
      // round trip stays off the kernel's exit.
      if (threadIdx.x == kEpiWarp0 * 32) {
        const uint32_t prev = atom_add_acq_rel_gpu(a.gsync + 1, 1u);
        if (prev == gridDim.x - 1) {   // every part has also read its row's maxima
          a.gsync[0] = 0u;
          a.gsync[1] = 0u;
          for (int r = 0; r < a.rq.rows_out; ++r)
            *reinterpret_cast<uint4*>(a.rq.pmax + kRowMaxStride * r) = make_uint4(0u, 0u, 0u, 0u);
        }
      }
    }
    const float* __restrict__ sa_g = a.sa;
    const float* __restrict__ sw_g = a.sw;
    __half* __restrict__ out_g = a.out;
    int32_t* __restrict__ acc_g = a.acc_out;
    int32_t* __restrict__ ws_g = a.ws;
    const int q = warp & 3;                    // TMEM lane quarter of this warp
    const int etid = threadIdx.x - kEpiWarp0 * 32;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    int esync_phase = 0;
    // All four epilogue warps meet here; waits are bounded, so an aborted pipeline can
    // never strand a warp.
    auto epi_sync = [&]() -> bool {
      __syncwarp();
      if (lane == 0) mbar_arrive(esync);
      const bool ok = mbar_wait(esync, (uint32_t)(esync_phase & 1), abort_flag, a.err, kDevTimeoutTmemFull, a.wait_cycles);
      ++esync_phase;
      return ok;
    };
    int sa_mt = -1;   // token tile whose activation scales sit in sa_sh
    int u = 0;
    while (epi_ok && iter.next(un)) {
      const int b = a.nbuf == 2 ? (u & 1) : 0;
      const uint32_t tpar = (a.nbuf == 2 ? (u >> 1) : u) & 1;
      const int nt = un.tile / a.m_tiles;
      const int mt = un.tile - nt * a.m_tiles;
      const int n = nt * 128 + q * 32 + lane;
      const int m0 = mt * NT;
      // Scales are fetched while the MMAs of this unit still run.  Tiles of more than 64
      // tokens take their token scales 32 at a time, one per lane (coalesced), and hand
      // them out by shuffles.
      const float swn = n < a.N ? sw_g[n] : 0.f;
      auto sa_group = [&](int c) { return m0 + c + lane < a.M ? __ldg(sa_g + m0 + c + lane) : 0.f; };
      float sa_nxt = NT > 64 ? sa_group(0) : 0.f;
      float sa_grp = 0.f;
      if (NT <= 64 && mt != sa_mt) {
        if (!epi_sync()) break;   // every warp is done with the previous token tile's scales
        for (int i = etid; i < NT; i += kNumEpiWarps * 32) sa_sh[i] = m0 + i < a.M ? sa_g[m0 + i] : 0.f;
        if (!epi_sync()) break;
        sa_mt = mt;
      }
      if (!mbar_wait(&tfull[b], tpar, abort_flag, a.err, kDevTimeoutTmemFull, a.wait_cycles)) break;
      if (etid == 0 && u < 4) DPTQ_TRACE_POINT(tr, 104 + u);
      tc_fence_after();
      const int nseg = (un.i1 - 1) / a.seg_iters - un.i0 / a.seg_iters + 1;
      const uint32_t tb = tmem_base + lane_base + (uint32_t)(b * NT * a.segs);
      // debug builds: a split tile's slot is one of the grid's (site 3)
      int32_t* __restrict__ wsl =
          un.slot >= 0 && DPTQ_CHECK(un.slot < (int)gridDim.x, a.err, 3) ? ws_g + (size_t)un.slot * (NT * 128) : nullptr;
      // Split tile.  If every other contributor has already added its part to the slot,
      // this CTA finishes the tile straight from its accumulators (slot + own part);
      // otherwise it adds its part and the last contributor to arrive finishes.
      volatile int* const flag = flags + 2 * (u & 1);   // [0]: all others in, [1]: last
      bool finish = wsl == nullptr;
      if (wsl != nullptr) {
        if (etid == 0) *flag = ld_acquire_gpu(a.counters + un.slot) == (uint32_t)(un.contributors - 1);
        if (!epi_sync()) break;
        finish = *flag != 0;
        if (etid == 0) DPTQ_TRACE_POINT(tr, 3);
      }
      // Output of 16 tokens of this thread's channel.  With a 16-byte aligned `out`, each
      // warp transposes 4 tokens x 32 channels at a time through shared memory and every
      // lane stores 4 consecutive channels of one token (8 bytes instead of four 2-byte
      // stores).  Token scales come from shared memory for tiles of up to 64 tokens, else
      // from the (cached) global array.
      // vf[i] = fp32(acc) of token c0 + i (the caller's exact conversion); v, if given,
      // the int32 accumulators for the optional dump.
      auto write_out = [&](int c0, const float (&vf)[16], const int* v) {
        __half hv[16];
#pragma unroll
        for (int i = 0; i < 16; i += 2) {
          const float sa0 = NT <= 64 ? sa_sh[c0 + i] : __shfl_sync(0xffffffffu, sa_grp, (c0 & 31) + i);
          const float sa1 = NT <= 64 ? sa_sh[c0 + i + 1] : __shfl_sync(0xffffffffu, sa_grp, (c0 & 31) + i + 1);
          const __half2 h2 = __floats2half2_rn(__fmul_rn(__fmul_rn(vf[i], sa0), swn),
                                               __fmul_rn(__fmul_rn(vf[i + 1], sa1), swn));
          hv[i] = __low2half(h2);
          hv[i + 1] = __high2half(h2);
        }
        if (acc_g != nullptr && n < a.N) {
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (m0 + c0 + i < a.M) acc_g[(size_t)(m0 + c0 + i) * a.N + n] = v != nullptr ? v[i] : __float2int_rn(vf[i]);
        }
        if (a.out_vec) {
          __half* xw = xpose + q * 128;
          const int c = lane >> 3;                 // token of this lane's 8-byte store
          const int nn = nt * 128 + q * 32 + (lane & 7) * 4;
#pragma unroll
          for (int g4 = 0; g4 < 4; ++g4) {
#pragma unroll
            for (int i = 0; i < 4; ++i) xw[i * 32 + lane] = hv[4 * g4 + i];
            __syncwarp();
            const uint2 val = *reinterpret_cast<const uint2*>(xw + c * 32 + (lane & 7) * 4);
            __syncwarp();
            const int m = m0 + c0 + 4 * g4 + c;
            if (m < a.M && nn < a.N) *reinterpret_cast<uint2*>(out_g + (size_t)m * a.N + nn) = val;
          }
        } else if (n < a.N) {
#pragma unroll
          for (int i = 0; i < 16; ++i)
            if (m0 + c0 + i < a.M) out_g[(size_t)(m0 + c0 + i) * a.N + n] = hv[i];
        }
      };
      // Split-tile partial sums.  With one exact-accumulation segment (every partial
      // sum and every sum of partial sums is an integer multiple of 2^-9 below 2^24
      // units, so exact in fp32) the raw fp32 accumulators are added with vector
      // reductions into a slot laid out [token / 4][channel][token % 4] (a warp's vector
      // access covers 512 contiguous bytes); otherwise int32 atomics, token-major.
      const bool f32 = a.segs == 1;
      float* const wslf = wsl != nullptr ? reinterpret_cast<float*>(wsl) + (size_t)(q * 32 + lane) * 4 : nullptr;
      if (f32) {
        // Chunks of 16 tokens, two per iteration.  When this CTA finishes a split tile, the
        // slot reads of the next chunk are issued before the current chunk is processed,
        // so their L2 latency overlaps that work.
        const bool rd = finish && wsl != nullptr;
        float4 s0[4], s1[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) s0[j] = s1[j] = make_float4(0.f, 0.f, 0.f, 0.f);
        auto load_slot = [&](int c, float4 (&d)[4]) {
#pragma unroll
          for (int j = 0; j < 4; ++j) d[j] = __ldcg(reinterpret_cast<const float4*>(wslf + (c / 4 + j) * 512));
        };
        auto chunk = [&](int c, const float4 (&sv)[4]) {
          uint32_t r[16];
          tmem_ld16(tb + (uint32_t)c, r);
          tmem_ld_wait();
          if (etid == 0 && c == 0) DPTQ_TRACE_POINT(tr, 2);
          float f[16];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            f[4 * j] = __fadd_rn(sv[j].x, __uint_as_float(r[4 * j]));
            f[4 * j + 1] = __fadd_rn(sv[j].y, __uint_as_float(r[4 * j + 1]));
            f[4 * j + 2] = __fadd_rn(sv[j].z, __uint_as_float(r[4 * j + 2]));
            f[4 * j + 3] = __fadd_rn(sv[j].w, __uint_as_float(r[4 * j + 3]));
          }
          if (rd) {
#pragma unroll
            for (int j = 0; j < 4; ++j)   // zero for the next launch
              __stcg(reinterpret_cast<float4*>(wslf + (c / 4 + j) * 512), make_float4(0.f, 0.f, 0.f, 0.f));
          }
          if (etid == 0) DPTQ_TRACE_POINT(tr, c == 0 ? 4 : 119);
          if (finish) {
            // f * 2^9 is the exact integer accumulator (below 2^24 in one segment), so it
            // is already fp32(acc).
            float vf[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) vf[i] = f[i] * 512.f;
            write_out(c, vf, nullptr);
          } else {
#pragma unroll
            for (int j = 0; j < 4; ++j)
              red_add_v4_f32(wslf + (c / 4 + j) * 512, f[4 * j], f[4 * j + 1], f[4 * j + 2], f[4 * j + 3]);
          }
          if (etid == 0) DPTQ_TRACE_POINT(tr, c == 0 ? 6 : 123);
        };
        if (rd) load_slot(0, s0);
#pragma unroll 1
        for (int c0 = 0; c0 < NT; c0 += 32) {
          if (NT > 64) {
            sa_grp = sa_nxt;
            if (c0 + 32 < NT) sa_nxt = sa_group(c0 + 32);
          }
          const bool two = c0 + 16 < NT;
          if (rd && two) load_slot(c0 + 16, s1);
          chunk(c0, s0);
          if (two) {
            if (rd && c0 + 32 < NT) load_slot(c0 + 32, s0);
            chunk(c0 + 16, s1);
          }
        }
      } else {
#pragma unroll 1
        for (int c0 = 0; c0 < NT; c0 += 16) {
          int acc[16];
          if (NT > 64 && (c0 & 31) == 0) sa_grp = sa_group(c0);
          if (finish && wsl != nullptr) {
#pragma unroll
            for (int i = 0; i < 16; ++i) acc[i] = __ldcg(wsl + (c0 + i) * 128 + q * 32 + lane);
#pragma unroll
            for (int i = 0; i < 16; ++i) __stcg(wsl + (c0 + i) * 128 + q * 32 + lane, 0);   // zero for the next launch
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) acc[i] = 0;
          }
          for (int sg = 0; sg < nseg; ++sg) {
            uint32_t r[16];
            tmem_ld16(tb + (uint32_t)(sg * NT + c0), r);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) acc[i] += __float2int_rn(__uint_as_float(r[i]) * 512.f);
          }
          if (finish) {
            float vf[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) vf[i] = __int2float_rn(acc[i]);
            write_out(c0, vf, acc);
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) atomicAdd(wsl + (c0 + i) * 128 + q * 32 + lane, acc[i]);
          }
          if (etid == 0) DPTQ_TRACE_POINT(tr, c0 == 0 ? 6 : 123);
        }
      }
      if (etid == 0 && u < 4) DPTQ_TRACE_POINT(tr, 112 + u);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[b]);
      ++u;
      if (wsl != nullptr && finish) {
        if (etid == 0) a.counters[un.slot] = 0u;   // every other contributor has arrived
      } else if (wsl != nullptr) {
        // Publish this CTA's part; the contributor that arrives last finishes the tile.
        __threadfence();
        if (!epi_sync()) break;
        if (etid == 0) {
          const uint32_t prev = atom_add_acq_rel_gpu(a.counters + un.slot, 1u);
          const int last = prev == (uint32_t)(un.contributors - 1);
          if (last) a.counters[un.slot] = 0u;
          flag[1] = last;
          DPTQ_TRACE_POINT(tr, 5);
        }
        if (!epi_sync()) break;
        if (flag[1] && f32) {
          // The slot holds the whole tile.  Chunks of 16 tokens, the next chunk's reads
          // issued before the current chunk is written, so that one L2 round trip covers
          // two chunks.
          float4 p0[4], p1[4];
          auto load_slot = [&](int c, float4 (&d)[4]) {
#pragma unroll
            for (int j = 0; j < 4; ++j) d[j] = __ldcg(reinterpret_cast<const float4*>(wslf + (c / 4 + j) * 512));
          };
          auto emit = [&](int c, const float4 (&d)[4]) {
            float vf[16];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              vf[4 * j] = d[j].x * 512.f;   // exact: one segment's sums are below 2^24 units
              vf[4 * j + 1] = d[j].y * 512.f;
              vf[4 * j + 2] = d[j].z * 512.f;
              vf[4 * j + 3] = d[j].w * 512.f;
            }
#pragma unroll
            for (int j = 0; j < 4; ++j)   // zero for the next launch
              __stcg(reinterpret_cast<float4*>(wslf + (c / 4 + j) * 512), make_float4(0.f, 0.f, 0.f, 0.f));
            write_out(c, vf, nullptr);
          };
          load_slot(0, p0);
#pragma unroll 1
          for (int c0 = 0; c0 < NT; c0 += 32) {
            if (NT > 64) sa_grp = sa_group(c0);
            const bool two = c0 + 16 < NT;
            if (two) load_slot(c0 + 16, p1);
            emit(c0, p0);
            if (two) {
              if (c0 + 32 < NT) load_slot(c0 + 32, p0);
              emit(c0 + 16, p1);
            }
          }
        } else if (flag[1]) {
#pragma unroll 1
          for (int c0 = 0; c0 < NT; c0 += 16) {
            if (NT > 64 && (c0 & 31) == 0) sa_grp = sa_group(c0);
            float vf[16];
            int v[16];
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = __ldcg(wsl + (c0 + i) * 128 + q * 32 + lane);
#pragma unroll
            for (int i = 0; i < 16; ++i) __stcg(wsl + (c0 + i) * 128 + q * 32 + lane, 0);
#pragma unroll
            for (int i = 0; i < 16; ++i) vf[i] = __int2float_rn(v[i]);
            write_out(c0, vf, v);
          }
        }
        if (etid == 0) {
          DPTQ_TRACE_POINT(tr, 7);
          DPTQ_TRACE_VALUE(tr, 121, flag[1] + 2);
        }
      }
      if (wsl != nullptr && finish && etid == 0) DPTQ_TRACE_VALUE(tr, 121, 1);
      if (etid == 0 && u <= 4) DPTQ_TRACE_POINT(tr, 108 + u - 1);
    }
    if (etid == 0) DPTQ_TRACE_VALUE(tr, 122, u);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, a.tmem_cols);
  }
  if (threadIdx.x == 0) DPTQ_TRACE_POINT(tr, 120);
}

// ------------------------------------------------------------------ host planning
int gemm_pick_nt(int M, int bits, int KB) {
  (void)KB;
  if (M <= 16) return 16;
  if (M <= 32) return 32;
  if (M <= 64) return 64;
  if (M <= 128 || (bits == 8 && a8_tile128())) return 128;
  return 192;
}

// Token tiles of up to 64 columns stream weights (decode): two k-blocks per stage to
// halve the per-byte barrier and conversion overhead.  192-token tiles (weights in
// tensor memory) take two as well: their MMA warp would otherwise spend more time per
// k-block on barrier waits and commits than the tensor pipe spends on the MMAs.  Other
// wide tiles keep one k-block per stage for a deeper ring.
static int kps_for(int nt) { return nt <= 64 || nt == 192 ? 2 : 1; }

static int smem_for(int nt, int kps, int stages, int planes, int conv_slots) {
  return 1024 + conv_slots * kps * kConvBytes + stages * kps * (planes * nt * 128 + kWTileBytes) + kBarrierBytes;
}

bool plan_gemm(int M, int N, int K_pad, int bits, int num_sms, GemmPlan& plan, int rot_smem) {
  GemmArgs& a = plan.args;
  const int KB = K_pad / kKBlock;
  const int planes = bits == 8 ? 2 : 1;
  int nt = gemm_pick_nt(M, bits, KB);
  int kps = kps_for(nt);
  // A8 192-token tiles take one k-block per stage: a stage holds two 24 KB activation
  // planes, so two-block stages would leave room for only two of them.
  if (nt == 192 && planes == 2) kps = 1;
  if (KB % kps != 0) kps = 1;
  // Largest |code| * |weight| sum per stage, and the stages one fp32 accumulator can
  // take before the exact-integer bound 2^24 could be crossed.
  auto seg_plan = [&](int kps_, int& seg_iters, int& segs) {
    const int KI = KB / kps_;
    const long long per_iter = (long long)(bits == 8 ? 128 : 8) * 7 * kKBlock * kps_;
    seg_iters = (int)(((1LL << 24) - 1) / per_iter);
    if (seg_iters > KI) seg_iters = KI;
    segs = (KI + seg_iters - 1) / seg_iters;
  };
  int seg_iters, segs;
  seg_plan(kps, seg_iters, segs);
  while (nt > 16 && nt * segs > 512) {
    nt = nt == 192 ? 128 : nt >> 1;
    const int k2 = (nt == 192 && planes == 2) ? 1 : kps_for(nt);
    if (k2 != kps && KB % k2 == 0) {
      kps = k2;
      seg_plan(kps, seg_iters, segs);
    }
  }
  if (nt * segs > 512) return false;
  // Widened weights live in TMEM for two-block stages and 192-token tiles (A operand
  // read from TMEM; 4 slots of 32 columns per k-block after the accumulators), else in
  // shared memory: as many slots as fit next to at least 4 bulk-copy stages (the
  // converters may run that far ahead of MMA completion).
  const bool a_tmem = a_in_tmem(nt, kps);
  int conv_slots = kMaxConvSlots;
  if (!a_tmem)
    while (conv_slots > 2 && smem_for(nt, kps, 4, planes, conv_slots) > kSmemLimit) --conv_slots;
  else   // room for two accumulators next to the slots
    while (conv_slots > 2 && 2 * nt * segs + conv_slots * kps * 32 > 512) --conv_slots;
  const int smem_conv = a_tmem ? 0 : conv_slots;
  // A fused launch needs two-block stages (weights widened into TMEM) and room for one
  // row's rotation scratch next to at least 3 stages.
  const bool fused = rot_smem > 0;
  if (fused && kps != 2) return false;
  auto smem_total = [&](int st) { return smem_for(nt, kps, st, planes, smem_conv) + (fused ? rot_smem : 0); };
  int stages = kMaxStages;
  while (stages > 2 && smem_total(stages) > kSmemLimit) --stages;
  if (smem_total(stages) > kSmemLimit || (fused && stages < 3)) return false;
  // The converters learn that a widened slot is free from the `empty` barrier of the
  // stage that last read it, CS stages back; with CS <= stages that barrier cannot
  // complete a further phase before they look.
  if (conv_slots > stages) conv_slots = stages;
  const int a_cols = a_tmem ? conv_slots * kps * 32 : 0;
  const int nbuf = 2 * nt * segs + a_cols <= 512 ? 2 : 1;
  if (nbuf * nt * segs + a_cols > 512) return false;
  const int acc_cols = nbuf * nt * segs;
  uint32_t cols = 32;
  while (cols < (uint32_t)(acc_cols + a_cols)) cols <<= 1;

  const int KI = KB / kps;
  const int M_pad = round_up(M, nt);
  const int n_wtiles = ceil_div(N, 128);
  const int m_tiles = M_pad / nt;
  const long long tiles = (long long)n_wtiles * m_tiles;
  const long long iters = tiles * KI;
  int G = (int)(iters < num_sms ? iters : num_sms);
  if (G < 1) G = 1;
  if (nt <= 64 && m_tiles == 1) {
    // Decode (one token tile, weights streamed once).  A tile split over several CTAs costs
    // its contributors fp32 reductions through L2 and a fence, and the tile's finisher an
    // extra round trip at the end of the launch; measured on GB300 that outweighs a
    // longer stream per CTA.  So: whole tiles, one per CTA, when they fit on the SMs and a
    // tile is at most twice a CTA's fair share of the stages; otherwise stream-K with at
    // most four CTAs per tile.  A fused launch keeps whole tiles only while they leave a
    // CTA for each of four parts of every token row: with fewer, its rows would be split
    // in two (slower rotation, measured: LLaMA-2-7B q|k|v at M = 32 is faster on all SMs).
    const bool rows_fit = !fused || (long long)M_pad * 4 <= tiles;
    if (decode_whole_tiles() && rows_fit && tiles <= num_sms && (long long)KI * num_sms <= 2 * iters)
      G = (int)tiles;
    else if (4 * tiles < G)
      G = (int)(4 * tiles);
  }
  long long dp = 0;
  if (tiles >= 2LL * G) dp = (tiles / G - 1) * G;

  plan.fused = fused;
  plan.a_tmem = a_tmem;
  plan.nt = nt;
  plan.kps = kps;
  plan.M_pad = M_pad;
  plan.grid = G;
  plan.smem_bytes = smem_total(stages);
  a.M = M;
  a.N = N;
  a.M_pad = M_pad;
  a.KB = KB;
  a.KI = KI;
  a.planes = planes;
  a.n_wtiles = n_wtiles;
  a.m_tiles = m_tiles;
  a.seg_iters = seg_iters;
  a.segs = segs;
  a.nbuf = nbuf;
  a.a_col0 = (uint32_t)acc_cols;
  a.stages = stages;
  a.conv_slots = conv_slots;
  a.dp_tiles = (int)dp;
  a.sk_iters = (tiles - dp) * KI;
  // 32-bit work enumeration on the device (UnitIter).
  if ((long long)a.sk_iters * G + G >= (1LL << 32) || tiles >= (1LL << 31)) return false;
  a.tmem_cols = cols;
  a.out_vec = 0;
  // Decode plans (one token tile of at most 64, weights streamed once): each CTA may
  // request up to 512 KB of its share into L2 ahead of the ring (76 MB over 152 SMs,
  // within the 129 MB L2).
  a.l2_prefetch = (nt <= 64 && m_tiles == 1 && l2_prefetch_allowed()) ? 512LL * 1024 : 0;
  a.rq = RQArgs{};
  a.gsync = nullptr;
  // Fused: every token row is split into 4 parts (each rotates and quantizes its share
  // of the row) when each part gets a CTA of its own; else into 2 parts with a CTA each,
  // for rows of at most 8192 elements (at most 4096 per part); else into 4 parts in two
  // rounds of rows.  A launch whose grid is smaller than that leaves the rows to the
  // separate rotate-quantize launch (no fused plan).
  int np = 1;
  if (fused) {
    if ((long long)M_pad * 4 <= G)
      np = 4;
    else if ((long long)M_pad * 2 <= G && K_pad <= 2 * 4096)
      np = 2;
    else if ((long long)M_pad * 4 <= 2LL * G)
      np = 4;
    else
      return false;
  }
  a.rq_np = np;
  a.rq_items = fused ? M_pad * np : 0;
  a.rq_shortfall = 0;
  a.pre_stages = 2;
  a.wait_cycles = kWaitTimeoutCycles;
  return true;
}

// How the fused launch splits a row over its np parts (two or four): slices of one
// block when the row has fewer blocks than parts (K a multiple of B, n = np B / K >= 2
// parts per block, slices of 1024 or 2048 elements), else whole blocks (every part at
// most 4096 elements: K <= 4096 np).  -1: neither applies.
int fused_rotation_variant(int K, int B, int tail, int np) {
  if (np != 2 && np != 4) return -1;
  if (tail == 0 && K % B == 0 && (np * B) % K == 0) {
    const int n = np * B / K;
    if (n >= 2 && B / n == 1024) return kPartSlice4;
    if (n >= 2 && B / n == 2048) return kPartSlice8;
  }
  const int gr = B > 128 ? B : 128;
  const int ng = (K + gr - 1) / gr;
  return (ng + np - 1) / np * gr <= 4096 ? kPartBlocks : -1;
}

template <int NT, int KPS, int RQV = 0>
static cudaError_t launch_nt(const GemmPlan& plan, cudaStream_t s, bool pdl) {
  cudaError_t e = ensure_max_dyn_smem(qgemm_kernel<NT, KPS, RQV>);
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
  cfg.numAttrs = (pdl && pdl_allowed()) ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, qgemm_kernel<NT, KPS, RQV>, plan.args);
}

cudaError_t launch_gemm(const GemmPlan& plan, cudaStream_t s, bool pdl) {
  if (plan.fused) {
    const int v = fused_rotation_variant(plan.args.rq.K, plan.args.rq.B, plan.args.rq.tail, plan.args.rq_np);
    if (v < 0 || plan.args.rq.np != plan.args.rq_np) return cudaErrorInvalidValue;
#define DPTQ_FUSED_NT(nt)                                                      \
  case nt:                                                                     \
    return v == kPartSlice4   ? launch_nt<nt, 2, kPartSlice4>(plan, s, pdl)    \
           : v == kPartSlice8 ? launch_nt<nt, 2, kPartSlice8>(plan, s, pdl)    \
                              : launch_nt<nt, 2, kPartBlocks>(plan, s, pdl);
    switch (plan.nt) {
      DPTQ_FUSED_NT(16)
      DPTQ_FUSED_NT(32)
      DPTQ_FUSED_NT(64)
      default: return cudaErrorInvalidValue;
    }
#undef DPTQ_FUSED_NT
  }
  if (plan.kps == 2) {
    switch (plan.nt) {
      case 16: return launch_nt<16, 2>(plan, s, pdl);
      case 32: return launch_nt<32, 2>(plan, s, pdl);
      case 64: return launch_nt<64, 2>(plan, s, pdl);
      case 192: return launch_nt<192, 2>(plan, s, pdl);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (plan.nt) {
    case 16: return launch_nt<16, 1>(plan, s, pdl);
    case 32: return launch_nt<32, 1>(plan, s, pdl);
    case 64: return launch_nt<64, 1>(plan, s, pdl);
    case 128: return launch_nt<128, 1>(plan, s, pdl);
    case 192: return launch_nt<192, 1>(plan, s, pdl);
    case 256: return launch_nt<256, 1>(plan, s, pdl);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace dptq

#ifdef DPTQ_TRACE
// Trace builds only: set (or clear with NULL) the device buffer of 256 stamps per CTA.
extern "C" int dptq_trace_set(void* dev_buffer) {
  return (int)cudaMemcpyToSymbol(dptq::g_dptq_trace, &dev_buffer, sizeof(dev_buffer));
}
#endif
