// Rotate + quantise kernels with 8-bit codes for f16 activations (the template lives in
// rotate_quant.cuh).
#include "rotate_quant.cuh"

namespace qvla {
cudaError_t launch_rotate_quant_a8_f16(const RotQuantArgs& a) { return rq::launch_dtype<__half, true>(a); }
}  // namespace qvla
