// Rotate + quantise kernels for f32 activations (the template lives in rotate_quant.cuh).
#include "rotate_quant.cuh"

namespace qvla {
cudaError_t launch_rotate_quant_f32(const RotQuantArgs& a) { return rq::launch_dtype<float, false>(a); }
}  // namespace qvla
