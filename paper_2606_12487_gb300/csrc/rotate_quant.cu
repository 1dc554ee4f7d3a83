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
