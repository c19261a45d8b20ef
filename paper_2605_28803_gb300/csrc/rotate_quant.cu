// Dispatch of the rotate + quantise kernels by activation dtype.
#include "kernels.h"

namespace qvla {

cudaError_t launch_rotate_quant_f16(const RotQuantArgs& a);
cudaError_t launch_rotate_quant_bf16(const RotQuantArgs& a);
cudaError_t launch_rotate_quant_f32(const RotQuantArgs& a);
cudaError_t launch_rotate_quant_a8_f16(const RotQuantArgs& a);
cudaError_t launch_rotate_quant_a8_bf16(const RotQuantArgs& a);
cudaError_t launch_rotate_quant_a8_f32(const RotQuantArgs& a);

bool rotate_quant_supported(int log_b) { return log_b >= 0 && log_b <= 12; }

cudaError_t launch_rotate_quant(const RotQuantArgs& a) {
  {  // operand bytes of 16-bit activations, one scale per row: one CTA per 2048-channel pass
    bool launched = false;
    const cudaError_t e = launch_rotate_quant_pass(a, &launched);
    if (e != cudaSuccess || launched) return e;
  }
  if (a.out_mode >= 2) {
    switch (a.xdt) {
      case 0: return launch_rotate_quant_a8_f16(a);
      case 1: return launch_rotate_quant_a8_bf16(a);
      case 2: return launch_rotate_quant_a8_f32(a);
      default: return cudaErrorInvalidValue;
    }
  }
  switch (a.xdt) {
    case 0: return launch_rotate_quant_f16(a);
    case 1: return launch_rotate_quant_bf16(a);
    case 2: return launch_rotate_quant_f32(a);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace qvla
