// dptq_internal.h -- host-side declarations shared by the CUDA translation units of
// libdptq (kernel argument blocks and launchers).  Not part of the public ABI.
#pragma once
#include <cstdint>
#include <string>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

// The layer handle behind dptq_handle.
struct dptq_linear {
  int device;
  int N, K, K_pad, KB, N_pad;
  int had_block;
  uint8_t* wt;  // [N_pad/128][KB][4 chunks of 32 k][128 rows][16 B] sign-magnitude nibbles
  float* sw;    // [N_pad]
  int8_t* signs;  // randomized Hadamard diagonal [K] on the device, or null (plain block Hadamard)
};

namespace dptq {

// K is processed in blocks of 128 elements: one 128-byte row of the MMA's swizzled
// FP8 operand tile.  Packed weights and activation operands pad K to a multiple of
// kKPad so that a pipeline stage may hold two blocks.
constexpr int kKBlock = 128;
constexpr int kKPad = 256;
// One (128 output channels) x (128 k) tile of packed 4-bit weights.
constexpr int kWTileBytes = 128 * 64;

inline int ceil_div(long long a, long long b) { return (int)((a + b - 1) / b); }
inline int round_up(int a, int b) { return ceil_div(a, b) * b; }

// ------------------------------------------------------------------ rotate + quantize
enum RQMode : int {
  kRQPublic = 0,   // codes in the public format (A4 packed nibbles / A8 int8) + scales
  kRQAct = 1,      // codes as E4M3 planes in the GEMM's swizzled tile layout + scales
  kRQY = 2,        // rotated fp32 activations (test hook)
  kRQWeights = 3,  // packed sign-magnitude int4 weight tiles + per-channel scales
};

constexpr int kRowMaxStride = 32;   // words per row of the fused launch's row-maximum slots

struct RQArgs {
  const __half* x;   // [rows_in][K] binary16, row-major
  const int8_t* signs;  // randomized Hadamard diagonal [K] (+1 / -1, 16-byte aligned) or null
  int rows_in;       // rows that carry data (M tokens or N channels)
  int rows_out;      // rows written (padded; rows >= rows_in are zero)
  int K;             // logical K
  int KB;            // K_pad / 128
  int B;             // Hadamard block size (power of two)
  int log2B;
  int nfull;         // number of whole blocks of size B
  int tail;          // tail block size (power of two) or 0
  int log2T;         // log2(tail) (0 when there is no tail)
  int chunk;         // elements rotated per shared-memory pass (a multiple of B)
  float c_hi, c_lo;  // 1/sqrt(2) as an fp32 pair (c_hi + c_lo to ~2^-48)
  // Non-power-of-two tail block r = tail_p 2^log2T (tail_p > 1): H_p (x) H_(2^log2T), H_p
  // from Paley's first construction with the prime tail_p - 1; y = S 2^-(24 + tail_j)
  // (t_hi + t_lo), t the fp32 pair of 1/sqrt(tail_p 2^(log2T & 1)).  tail_p = 1: a
  // power-of-two tail (or none).
  int tail_p;
  int tail_j;
  float t_hi, t_lo;
  int bits;          // 4 or 8
  // Fused decode launch: parts per row and the row-maximum slots, kRowMaxStride words
  // per row of which the first np are used (1 + the bits of each part's largest |y|;
  // 0 = not yet written; zero between launches).
  int np;
  uint32_t* pmax;
  float* scales;     // [rows_out] (rows >= rows_in get 0); may be null in kRQY
  void* out;         // mode-dependent destination
};

cudaError_t launch_rotate_quant(RQMode mode, const RQArgs& a, cudaStream_t s, bool pdl);
// Shared memory of one row part in the fused decode launch: the padded int64 transpose
// chunk (4096 + 256 values), two planes of staged codes (4096 bytes each) and 16 warp
// maxima.
constexpr int kRQPartSmemBytes = (4096 + 256) * 8 + 2 * 4096 + 16 * 8;
size_t rotate_quant_smem(int K, int chunk);
// Shared-memory budget of one CTA (227 KB opt-in).
constexpr size_t kSmemPerBlock = 232448;

// Public codes (A4 packed two's complement / A8 int8) -> E4M3 GEMM planes.
struct CodesArgs {
  const uint8_t* codes;
  int M, M_pad, K, KB, bits;
  uint8_t* act;
};
cudaError_t launch_codes_to_act(const CodesArgs& a, cudaStream_t s);

// ------------------------------------------------------------------ KV4 and policy
struct KvArgs {
  const __half* kv;   // [rows][cols]
  int rows, cols, group;
  uint8_t* codes;     // [rows][cols / 2]
  float* scales;      // [rows][cols / group]
};
cudaError_t launch_kv4(const KvArgs& a, int num_sms, cudaStream_t s);

struct PolicyArgs {
  const float* x;     // [L][T][d]
  const float* dx;    // [L][T][d]
  int L, T, d, bits;
  double eps, tau_jr, tau_snr;
  double* jr;         // [L]
  double* snr;        // [L]
  uint8_t* bits_out;  // [L]
  int* err;           // device error word (bounded waits that gave up)
};
cudaError_t launch_policy(const PolicyArgs& a, int num_sms, cudaStream_t s);

// ------------------------------------------------------------------ GEMM
struct GemmArgs {
  const uint8_t* wt;   // [NTw][KB][4][128][16] packed sign-magnitude nibbles (chunk-major tiles)
  const uint8_t* act;  // [planes][KB][M_pad][128] E4M3, rows pre-swizzled
  const float* sa;     // [>= M] per-token scales
  const float* sw;     // [>= N] per-channel scales
  __half* out;         // [M][N]
  int32_t* acc_out;    // optional [M][N]
  int32_t* ws;         // split-tile partial sums: [grid][NT * 128]
  uint32_t* counters;  // [grid] arrival counters (zero between launches)
  int* err;            // device error word
  int M, N, M_pad, KB, planes;
  int KI;              // pipeline iterations per tile (KB / k-blocks per stage)
  int n_wtiles;        // N_pad / 128
  int m_tiles;         // M_pad / NT
  int seg_iters;       // iterations per exact fp32 accumulation segment
  int segs;            // accumulator segments per tile
  int nbuf;            // TMEM accumulator buffers (1 or 2)
  int stages;          // bulk-copy ring depth
  int conv_slots;      // widened-weight ring depth
  uint32_t a_col0;     // first TMEM column of the widened-weight slots (A operand in TMEM)
  int dp_tiles;        // tiles processed whole, round-robin, before the stream-K part
  long long sk_iters;  // stream-K iterations (tiles after dp_tiles, times KI)
  uint32_t tmem_cols;
  int out_vec;         // `out` is 16-byte aligned: the epilogue stores 8 channels at a time
  long long l2_prefetch;  // weight bytes past the first ring stages each CTA requests into L2 up front (0: none)
  // Fused launch: weight stages the producer requests before the token rows are ready
  // (set from pre_stages_setting());
  // the rest of the ring and the L2 prefetch wait for the rows (while the rows are
  // rotated, the parts' exchanges of their maxima cross the memory system, and a full
  // ring fill in flight delays them by microseconds).
  int pre_stages;
  // Fused decode launches only: the rotation + quantization of the M_pad token rows
  // (written to `act` / `sa` by the converter warps of CTAs 0, 1, ...) and the two grid
  // counters [rows ready, CTAs done] that order it before the GEMM (zero between launches).
  RQArgs rq;
  int rq_np;           // parts per token row (1, 2 or 4): work item = row * rq_np + part
  int rq_items;        // M_pad * rq_np: the value the rows-ready counter reaches
  int rq_shortfall;    // test hook: extra items the activation producer waits for (0)
  uint32_t* gsync;
  long long wait_cycles;   // bound of every pipeline wait (SM cycles) before the kernel gives up
};

struct GemmPlan {
  bool fused;     // rotation + quantization inside the GEMM launch
  bool a_tmem;    // widened weights (MMA A operand) in tensor memory, else shared memory
  int nt;          // token tile (MMA N): 16, 32, 64, 128, 192 or 256
  int kps;         // k-blocks of 128 per pipeline stage (1 or 2)
  int M_pad;
  int grid;
  int smem_bytes;
  GemmArgs args;
};

// Fills everything in `plan.args` that depends only on shapes; the caller sets the
// pointers.  Returns false if the shape cannot be run.
// `rot_smem` > 0 plans the fused decode kernel: that many extra bytes of shared memory
// for the rotation of one row, two k-blocks per stage; false if it does not fit.
bool plan_gemm(int M, int N, int K_pad, int bits, int num_sms, GemmPlan& plan, int rot_smem = 0);
// Row split of the fused launch for K, B, the (power-of-two) tail and np parts per row:
// kPartBlocks, kPartSlice4 or kPartSlice8 (rotate_row.cuh), or -1 when none applies.
int fused_rotation_variant(int K, int B, int tail, int np);
cudaError_t launch_gemm(const GemmPlan& plan, cudaStream_t s, bool pdl);

// Programmatic dependent launch is on unless the environment sets DPTQ_PDL=0 (kernels
// then start only after their predecessor has finished, e.g. for profilers).
bool pdl_allowed();
// The fused decode kernel is used unless the environment sets DPTQ_FUSED=0.
bool fused_allowed();
// Bound of the GEMM kernels' pipeline waits in SM cycles: DPTQ_WAIT_CYCLES, else about
// one second.  Tests of the time-out path shorten it.
long long wait_cycles_setting();
// Test hook: DPTQ_TEST_ROWS_SHORTFALL=n makes the first fused launch of the process wait
// for n more published token rows than any CTA publishes, so that its bounded wait runs
// out (returns n once, then 0).
int take_rows_shortfall();
// Decode GEMM launches prefetch their weight share into L2 unless DPTQ_L2PF=0.
bool l2_prefetch_allowed();
int pre_stages_setting();
bool decode_whole_tiles();   // DPTQ_DECODE_WHOLE_TILES=0: decode grids never shrink to one CTA per tile
bool a8_tile128();   // DPTQ_A8_TILE128=1: A8 prefill on 128-token tiles (weights widened into shared memory)
// The GEMM operand rows are rotated and quantized by the whole-row kernel (sums kept in
// registers) unless DPTQ_ROWS_KERNEL=0 (the per-row kernel with an fp32 row in shared
// memory).
bool rows_kernel_allowed();

// The fixed scratch of dptq_qlinear_static on device `dev`: read its device error word
// into *word and, when it is non-zero, clear the word, the split-tile sums and the
// arrival counters (synchronous; no allocation).  *word = 0 when the scratch was never
// set up on that device.
cudaError_t static_scratch_check_reset(int dev, int* word);

// Raise a kernel's ceiling for dynamic shared memory to the most the device allows it, once
// per device.
// Every launch of a kernel then fits its ceiling whatever size was launched last: a CUDA
// graph that captured launches of one kernel with different shared-memory sizes (4- and
// 8-bit plans) replays them, and a profiler that re-launches one of its nodes on its own
// finds a ceiling that node fits.  (Setting the ceiling to each launch's own size made the
// value left by the last captured launch govern such re-launches.)
cudaError_t ensure_max_dyn_smem_impl(const void* fn);
template <class Kernel>
cudaError_t ensure_max_dyn_smem(Kernel* fn) {
  return ensure_max_dyn_smem_impl(reinterpret_cast<const void*>(fn));
}

// Message returned by dptq_last_error_message() on the calling thread.
void set_error_message(const std::string& m);
int gemm_pick_nt(int M, int bits, int KB);

}  // namespace dptq
