// Dispatch of the W4A4 GEMM (the kernel template lives in gemm_kernel.cuh): tile shapes and
// orientations for each launch, and the device error word of the kernels instantiated here.
#include "gemm_kernel.cuh"

namespace qvla {
namespace {

// Per-group step scales: int4 operand bytes, 128-wide tiles at most (the running sum takes a
// third TMEM region).
template <typename OutT>
cudaError_t launch_grouped(const GemmArgs& a) {
  if (a.gated || a.x_bytes != 1) return cudaErrorInvalidValue;
  if (a.M > 128) return launch_cfg<128, false, false, 1, OutT, true>(a);
  const int mpad = (a.M + 15) / 16 * 16;
  if (mpad <= 16) return launch_cfg<16, true, false, 1, OutT, true>(a);
  if (mpad <= 32) return launch_cfg<32, true, false, 1, OutT, true>(a);
  if (mpad <= 64) return launch_cfg<64, true, false, 1, OutT, true>(a);
  return launch_cfg<128, true, false, 1, OutT, true>(a);
}

// Token-major tile shapes and their estimated launch times (ns): a fixed cost plus, per wave of
// persistent CTAs (or CTA pairs), a per-tile cost and a cost per k-block, fitted to GB300
// measurements (M 256-8192, K 1024-16384; pairs only from K = 1024): single CTAs with 128- / 256-wide tiles 2300 + waves x
// (2000 + 344 / k-block) and 2000 + waves x (2500 + 560 / k-block); CTA pairs (256 tokens over two
// SMs, half the weight rows staged per SM) 3900 + waves x (1000 + 351 / k-block) and 3800 + waves
// x (2900 + 375 / k-block).  A pair wave holds half as many tiles, each of twice the tokens.
// A non-gated layer whose tiles leave SMs (or pairs) idle may split each tile's k-blocks into 2
// or 4 work units of at least 16 k-blocks (their partials in the caller's workspace, the tile's
// last unit finishing it): a wave of units then costs per_tile + split + k-blocks per unit x
// per_kb, with split fitted on 816 x 16384 -> 2048: 4900 ns for single CTAs (128-wide tiles in 4
// parts, 56.0 us against 53.9 whole) and 14500 for pairs (256-wide tiles in 2 parts, 45.2 us).
enum class TileShape { kSingle128, kSingle256, kPair128, kPair256 };

TileShape token_major_shape(const GemmArgs& a, int* parts) {
  const long nkb = a.K / kBK, sms = a.num_sms, npairs = a.num_sms / 2;
  const long t1 = (a.M + kBM - 1) / kBM, t2 = (a.M + 2 * kBM - 1) / (2 * kBM);
  const long n128 = a.gated ? 0 : (a.N + 127) / 128, n256 = (a.N + 255) / 256;
  const bool can_split = !a.gated && a.part_ws != nullptr && a.part_cnt != nullptr;
  // estimated time of a shape (tiles of bn weight rows, `halves` CTAs each) at its best split
  auto est = [&](long tiles, long units, long fixed, long per_tile, long per_kb, long bn, long halves, int* q_out) {
    const long split = halves == 2 ? 14500 : 4900;
    const long whole = fixed + (tiles + units - 1) / units * (per_tile + nkb * per_kb);
    long best = whole;
    *q_out = 1;
    if (!can_split || tiles >= units) return best;
    for (int q = 2; q <= 4; q *= 2) {
      if (nkb / q < 16 || static_cast<size_t>(tiles * halves * q * kBM * bn) > a.part_ws_floats ||
          tiles * halves > a.part_cnt_n)
        continue;
      const long t = fixed + (tiles * q + units - 1) / units * (per_tile + split + (nkb + q - 1) / q * per_kb);
      if (t < best && 10 * t < 9 * whole) {  // a split only where it is estimated 10% faster
        best = t;
        *q_out = q;
      }
    }
    return best;
  };
  int q = 1;
  TileShape best = TileShape::kSingle256;
  long t = est(t1 * n256, sms, 2000, 2500, 560, 256, 1, &q);
  *parts = q;
  auto consider = [&](TileShape s, long v) {
    if (v < t) {
      t = v;
      best = s;
      *parts = q;
    }
  };
  if (n128) consider(TileShape::kSingle128, est(t1 * n128, sms, 2300, 2000, 344, 128, 1, &q));
  // pairs need a few k-blocks per tile to hide their larger per-tile hand-over (measured at
  // K = 256: 12% slower than single CTAs where this estimate favoured the pair)
  if (a.M > kBM && npairs > 0 && nkb >= 8) {
    consider(TileShape::kPair256, est(t2 * n256, npairs, 3800, 2900, 375, 256, 2, &q));
    if (n128) consider(TileShape::kPair128, est(t2 * n128, npairs, 3900, 1000, 351, 128, 2, &q));
  }
  return best;
}

template <int kX, typename OutT>
cudaError_t launch_out(const GemmArgs& a) {
  if (a.gated || a.M > 128) {
    if constexpr (kX == 2) {
      // 8-bit activation planes: single CTAs; tile width by waves x tile width
      if (a.gated) return launch_cfg<256, false, true, kX, OutT>(a);  // gate/up pairs share a 256-row tile
      const long tm = (a.M + kBM - 1) / kBM;
      const long w256 = (tm * ((a.N + 255) / 256) + a.num_sms - 1) / a.num_sms;
      const long w128 = (tm * ((a.N + 127) / 128) + a.num_sms - 1) / a.num_sms;
      if (w128 * 128 < w256 * 256) return launch_cfg<128, false, false, kX, OutT>(a);
      return launch_cfg<256, false, false, kX, OutT>(a);
    } else {
      // gated layers always take 256-wide tiles: a tile's gate and up rows meet in one epilogue
      GemmArgs b = a;
      switch (token_major_shape(a, &b.parts)) {
        case TileShape::kPair256:
          return b.gated ? launch_cfg<256, false, true, kX, OutT, false, true>(b)
                         : launch_cfg<256, false, false, kX, OutT, false, true>(b);
        case TileShape::kPair128:
          return launch_cfg<128, false, false, kX, OutT, false, true>(b);
        case TileShape::kSingle128:
          return launch_cfg<128, false, false, kX, OutT>(b);
        default:
          return b.gated ? launch_cfg<256, false, true, kX, OutT>(b) : launch_cfg<256, false, false, kX, OutT>(b);
      }
    }
  }
  const int mpad = (a.M + 15) / 16 * 16;
  if (mpad <= 16) return launch_cfg<16, true, false, kX, OutT>(a);
  if (mpad <= 32) return launch_cfg<32, true, false, kX, OutT>(a);
  if (mpad <= 64) return launch_cfg<64, true, false, kX, OutT>(a);
  return launch_cfg<128, true, false, kX, OutT>(a);
}

}  // namespace

int token_major_plan(const GemmArgs& a, int* parts) { return static_cast<int>(token_major_shape(a, parts)); }

cudaError_t launch_gemm_w4a4(const GemmArgs& a) {
  if (a.M == 0) return cudaSuccess;
  {  // one to four tokens: the weight stream decides, so the CUDA-core GEMV takes it
    bool launched = false;
    const cudaError_t e = launch_gemv_w4a4(a, &launched);
    if (e != cudaSuccess || launched) return e;
  }
  if (a.gscale) return a.ydt == 0 ? launch_grouped<__half>(a) : launch_grouped<__nv_bfloat16>(a);
  if (a.x_bytes == 2) return a.ydt == 0 ? launch_out<2, __half>(a) : launch_out<2, __nv_bfloat16>(a);
  if (a.x_bytes == 1) return a.ydt == 0 ? launch_out<1, __half>(a) : launch_out<1, __nv_bfloat16>(a);
  return a.ydt == 0 ? launch_out<0, __half>(a) : launch_out<0, __nv_bfloat16>(a);
}

cudaError_t set_debug_hooks_gemm(unsigned long long wait_limit_ns, int hold_loads) {
  return set_debug_hooks(wait_limit_ns, hold_loads);
}

cudaError_t read_and_clear_error_word(unsigned int* out, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(out, g_error_word, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_error_word, &zero, sizeof(unsigned int));
}

}  // namespace qvla
