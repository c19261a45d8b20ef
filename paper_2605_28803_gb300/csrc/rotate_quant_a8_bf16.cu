// Rotate + quantise kernels with 8-bit codes for bf16 activations (the template lives in
// rotate_quant.cuh).
#include "rotate_quant.cuh"

namespace qvla {
cudaError_t launch_rotate_quant_a8_bf16(const RotQuantArgs& a) { return rq::launch_dtype<__nv_bfloat16, true>(a); }
}  // namespace qvla
