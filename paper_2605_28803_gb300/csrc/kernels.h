// Host-side interface between the C ABI (api.cu) and the kernels.  Internal to libqvla.
#pragma once

#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace qvla {

// ---- rotate + quantise (rotate_quant.cu) ----
struct RotQuantArgs {
  const void* x;           // device [M][K], dtype xdt
  int xdt;                 // 0 f16, 1 bf16, 2 f32
  int M, K;
  int log_b;               // log2 of the Hadamard block, 0 = none
  float inv_sqrt_b;        // float32(1 / sqrt(b))
  int mode;                // 0 per-token, 1 per-step (step_scale), 2 absmax only
  const float* step_scale; // device, one float (mode 1)
  uint8_t* xq;             // device output, by out_mode:
  int out_mode;            // 4-bit codes: 0 packed nibbles [M][K/2]; 1 one E4M3 operand byte per
                           //   code [M][K] (the GEMM's internal encoding);
                           // 8-bit codes: 2 int8 rows [M][K]; 3 the GEMM's two operand planes
                           //   [M][2K] (per 128 codes: high nibbles, then low nibbles)
  float* xscale;           // device [M]
  int32_t* xsum;           // device [M] or null
  float* absmax;           // device, one float (mode 2), or one per scale group
  int gshift = 30;         // scale groups of 2^gshift channels (>= 30: one group; else a group
                           //   holds whole Hadamard blocks and >= 128 channels): step_scale
                           //   then points at the step's [K >> gshift] entries, absmax too
  int32_t* xgsum = nullptr;  // device [M][K >> gshift] per-group code sums, or null
  int32_t* zero = nullptr;   // device ints set to 0 once x has been waited for (the next GEMM's
  int zero_n = 0;            //   work-unit counters), or null
  cudaStream_t stream;
};
bool rotate_quant_supported(int log_b);
// The rotate-quantise kernel in passes (rotate_quant_pass.cu): up to 64 rows of 16-bit
// activations into operand bytes (out_mode 1) with one scale per row, per token or per step,
// Hadamard block <= 2048 and at most 8 passes of 2048 (or fewer, smaller) channels per row.
// *launched is false (nothing enqueued) outside that range; the outputs are those of the
// row-per-warp kernel, bit for bit.  launch_rotate_quant takes it first.
cudaError_t launch_rotate_quant_pass(const RotQuantArgs& a, bool* launched);
cudaError_t read_and_clear_error_word_rqp(unsigned int* out, cudaStream_t stream);
cudaError_t set_debug_hooks_rqp(unsigned long long wait_limit_ns, int hold);
cudaError_t launch_rotate_quant(const RotQuantArgs& a);

// ---- int8 codes to the W4A8 GEMM's operand planes (a8_planes.cu) ----
// xq: device [M][K] int8 codes (16-byte aligned rows); planes: device [M][2K]; xsum: device [M]
// or null (cleared, then the codes' row sums added).
cudaError_t launch_a8_planes(const int8_t* xq, int M, int K, uint8_t* planes, int32_t* xsum, cudaStream_t stream);

// ---- online x . P . BlockDiag(U_b) (block_rotate.cu) ----
// x, out: device [M][K] of activation dtype xdt (0 f16, 1 bf16, 2 f32); perm: device int32 [K]
// (identity when the layer has none); rot: device float32 [K/block][block][block], 16-byte
// aligned; block in {16, 32, 64} dividing K.
cudaError_t launch_block_rotate(const void* x, int xdt, int M, int K, const int32_t* perm, const float* rot, int block,
                                void* out, cudaStream_t stream);

// ---- W4A4 GEMM + epilogue (gemm.cu) ----
struct GemmArgs {
  const uint8_t* xq;       // device activations, by x_bytes:
  int x_bytes;             // 0: packed int4 codes [M][K/2]; 1: the rotate-quantise kernel's
                           //   operand bytes of int4 codes [M][K]; 2: its two operand planes of
                           //   int8 codes [M][2K] (the W4A8 variant, K <= 4096)
  const float* xscale;     // device [M]
  const int32_t* xsum;     // device [M]
  const uint8_t* wq;       // device weight codes, tiled: 8 KB chunks of 128 rows x 128 codes,
                           // [groups][K/128][128][64 B], groups even (rows past N are zero)
  const float* wscale;     // device [N]
  const float* wcorr;      // device [N]: 8 * sum_k wq[n,k] as float (128 * sum for x_bytes 2)
  const float* bias;       // device [N] (zeros when the layer has no bias)
  void* y;                 // device [M][N], dtype ydt
  int ydt;                 // 0 f16, 1 bf16
  int32_t* acc;            // device [M][N] or null
  int M, N, K;             // N = weight rows (2H for a gated layer)
  int gated;               // 1: rows interleave gate/up in 128-row groups; y is [M][N/2] = h
  // per-step, per-group activation scales (x_bytes 1, not gated; acc unused): gscale device
  // [K/group] the step's scales, xgsum device [M][K/group] the activations' group code sums,
  // wgcorr device [N][K/group] 8 x the weights' group code sums; group = channels per scale
  const float* gscale = nullptr;
  const int32_t* xgsum = nullptr;
  const float* wgcorr = nullptr;
  int group = 0;
  // the fused one-launch linear (launch_gemm_fused): raw activations x [M][K] of dtype xdt
  // (0 f16, 1 bf16) with Hadamard block 2^log_b; xscale then points at the step's one scale
  const void* x = nullptr;
  int xdt = 0;
  int log_b = 0;
  float inv_sqrt_b = 1.0f;
  // token-major tiles of a non-gated layer may split their k-blocks into `parts` work units
  // when the tiles leave SMs idle: the units' FP32 partials go to part_ws (part_ws_floats
  // floats) and part_cnt (part_cnt_n ints, zero at launch; the GEMM leaves them zero) counts
  // each tile's finished units.  Null: no split.  `parts` is set by the tile-shape choice.
  int parts = 1;
  float* part_ws = nullptr;
  size_t part_ws_floats = 0;
  int* part_cnt = nullptr;
  int part_cnt_n = 0;
  int num_sms;
  cudaStream_t stream;
};
cudaError_t launch_gemm_w4a4(const GemmArgs& a);
// The token-major launch plan of launch_gemm_w4a4 for int4 operand-byte activations and M > 128
// (host logic only; a's device pointers are not read): the tile shape (0 single CTAs 128 x 128,
// 1 single CTAs 128 x 256, 2 CTA pairs 256 x 128, 3 CTA pairs 256 x 256) and *parts, the work
// units per tile (1 = whole tiles).
int token_major_plan(const GemmArgs& a, int* parts);

// The one-launch linear for a small batch with a per-step scale (gemm_fused.cu): the weight-major
// split-K GEMM whose CTAs rotate and quantise the activations themselves.  *launched is false
// (and nothing was enqueued) when the shape is outside what it takes: M > 128, gated or grouped
// layers, K beyond 4096, or no split of K that fits its shared-memory tiles.
cudaError_t launch_gemm_fused(const GemmArgs& a, bool* launched);

// Decode-sized batches (gemv.cu): the integer product and epilogue on the CUDA cores for
// M <= kGemvMaxM tokens, with activations as operand bytes (x_bytes 1) or packed codes (0), gated
// or not, one scale per token or per step (no per-group tables).  *launched is false (nothing
// enqueued) outside that range.  The outputs are those of launch_gemm_w4a4, bit for bit.
// x_bytes 3 (M = 1): the raw activations x (dtype xdt == ydt, Hadamard block 2^log_b <= 2048
// dividing the rotation pass) are rotated and quantised in the same launch; xscale is the step's
// one scale or null for a per-token scale, xq and xsum are unused.  Taken where each CTA's
// k-range touches at most two rotation passes.  The outputs are those of the rotate-quantise
// kernel followed by launch_gemm_w4a4, bit for bit.
constexpr int kGemvMaxM = 4;
cudaError_t launch_gemv_w4a4(const GemmArgs& a, bool* launched);

// Read and clear the device-side error words of the kernels that wait (gemm.cu, gemm_fused.cu).
cudaError_t read_and_clear_error_word(unsigned int* out, cudaStream_t stream);
cudaError_t read_and_clear_error_word_fused(unsigned int* out, cudaStream_t stream);

// Test hooks (qvla_debug.h): the wait limit of the bounded waits and whether GEMM load warps hold
// back every copy, for the kernels of gemm.cu and of gemm_fused.cu.  Synchronise the device first.
cudaError_t set_debug_hooks_gemm(unsigned long long wait_limit_ns, int hold_loads);
cudaError_t set_debug_hooks_fused(unsigned long long wait_limit_ns, int hold_loads);
cudaError_t set_debug_hooks_gemv(unsigned long long wait_limit_ns, int hold_loads);
cudaError_t read_and_clear_error_word_gemv(unsigned int* out, cudaStream_t stream);

}  // namespace qvla
