// Host-only weight packing (no CUDA).  Internal to libqvla.
#pragma once

#include <cstdint>

namespace qvla {

// Arguments are validated by the caller (api.cu).  wdt: 0 f16, 1 bf16, 2 f32.
void pack_weights_host_impl(const void* W, int wdt, int N, int K, const double* rot, int rot_block,
                            const int32_t* perm, int had_block, uint8_t* wq, float* wscale, int32_t* wsum);

// wsum[n] = sum of the int4 codes of packed row n.
void code_sums_host(const uint8_t* wq, int N, int K, int32_t* wsum);

}  // namespace qvla
