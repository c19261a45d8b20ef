// The one-launch small-batch linear: the weight-major split-K GEMM of gemm_kernel.cuh with its
// fused rotate + quantise prologue (kX == 3), instantiated here by the 16-bit activation type (the
// output type is the same), token-tile width and channels per lane.
#include "gemm_kernel.cuh"

namespace qvla {
namespace {

template <typename OutT, int kE, typename XT>
cudaError_t launch_fused_bn(const GemmArgs& a) {
  if (a.M <= 16) return launch_fused_cfg<16, OutT, kE, XT>(a);
  if (a.M <= 32) return launch_fused_cfg<32, OutT, kE, XT>(a);
  if (a.M <= 64) return launch_fused_cfg<64, OutT, kE, XT>(a);
  return launch_fused_cfg<128, OutT, kE, XT>(a);
}

template <typename T>
cudaError_t launch_fused_e(const GemmArgs& a) {
  // a warp task takes a row chunk of 512 channels up to K = 512, 1024 up to K = 1024, 2048 beyond
  if (a.K <= 512) return launch_fused_bn<T, 16, T>(a);
  return a.K <= 1024 ? launch_fused_bn<T, 32, T>(a) : launch_fused_bn<T, 64, T>(a);
}

}  // namespace

cudaError_t launch_gemm_fused(const GemmArgs& a, bool* launched) {
  *launched = false;
  // activations and outputs of one 16-bit type (f16 -> f16, bf16 -> bf16)
  if (a.M < 1 || a.M > 128 || a.gated || a.gscale || a.K > 4096 || a.K < 512 || a.xdt != a.ydt ||
      (a.xdt != 0 && a.xdt != 1) || a.log_b > 12)
    return cudaSuccess;
  const cudaError_t e = a.xdt == 0 ? launch_fused_e<__half>(a) : launch_fused_e<__nv_bfloat16>(a);
  if (e == kNotApplicable) return cudaSuccess;
  *launched = e == cudaSuccess;
  return e;
}

cudaError_t set_debug_hooks_fused(unsigned long long wait_limit_ns, int hold_loads) {
  return set_debug_hooks(wait_limit_ns, hold_loads);
}

cudaError_t read_and_clear_error_word_fused(unsigned int* out, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(out, g_error_word, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_error_word, &zero, sizeof(unsigned int));
}

}  // namespace qvla
