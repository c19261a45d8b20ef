// Host-only weight packing (no CUDA).  Internal to libqvla.
#pragma once

#include <cstdint>

namespace qvla {

// Arguments are validated by the caller (api.cu).  wdt: 0 f16, 1 bf16, 2 f32.
void pack_weights_host_impl(const void* W, int wdt, int N, int K, const double* rot, int rot_block,
                            const int32_t* perm, int had_block, uint8_t* wq, float* wscale, int32_t* wsum);

// The zigzag channel permutation by weight energy and the block SVD factors (Sec. 4.1).
void zigzag_permutation_host(const void* W, int wdt, int N, int K, int block, int32_t* perm);
void block_svd_rotation_host(const void* W, int wdt, int N, int K, int block, const int32_t* perm, double* rot);

// GPTQ-style codes of the folded weights against n_cal calibration rows X (dtype xdt, [n_cal][K],
// folded the same way); false if the damped Hessian is not positive definite.
bool gptq_pack_host(const void* W, int wdt, int N, int K, const void* X, int xdt, int n_cal, const double* rot,
                    int rot_block, const int32_t* perm, int had_block, int block, double damp, uint8_t* wq,
                    float* wscale, int32_t* wsum);

// wsum[n] = sum of the int4 codes of packed row n.
void code_sums_host(const uint8_t* wq, int N, int K, int32_t* wsum);

}  // namespace qvla
