// int8 activation codes [M][K] (natural k order) to the W4A8 GEMM's two operand planes
// [M][2K]: per k-block of 128 codes, 128 bytes of high-nibble E4M3 then 128 of low-nibble
// E4M3, each group of 8 codes in the order k0 k2 k4 k6 k1 k3 k5 k7 (the order in which the GEMM
// expands the weights), and the row's code sum.  Serves the GEMM entry point that takes codes
// quantised elsewhere; the fused rotate + quantise kernel writes the planes directly.
#include <cuda_runtime.h>

#include "a8_codes.cuh"
#include "kernels.h"

namespace qvla {
namespace {

// One thread per 8 codes; a row's K / 8 threads are consecutive, so loads and stores coalesce.
__global__ void __launch_bounds__(256) a8_planes_kernel(const int8_t* __restrict__ xq, int M, int K,
                                                       uint8_t* __restrict__ planes, int32_t* __restrict__ xsum) {
  const int per_row = K / 8;
  const long long g = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (g >= static_cast<long long>(M) * per_row) return;
  const int m = static_cast<int>(g / per_row);
  const int c = static_cast<int>(g - static_cast<long long>(m) * per_row);  // group of 8 within the row
  const uint2 v = __ldg(reinterpret_cast<const uint2*>(xq + static_cast<size_t>(m) * K) + c);
  const uint32_t e = __byte_perm(v.x, v.y, 0x6420), o = __byte_perm(v.x, v.y, 0x7531);
  uint32_t he, ho, le, lo;
  a8_planes(e, o, he, ho, le, lo);
  const int k0 = 8 * c;
  uint8_t* hp = planes + static_cast<size_t>(m) * (2 * K) + 2 * (k0 & ~127) + (k0 & 127);
  *reinterpret_cast<uint2*>(hp) = make_uint2(he, ho);
  *reinterpret_cast<uint2*>(hp + 128) = make_uint2(le, lo);
  if (xsum != nullptr) {
    int s = __dp4a(static_cast<int>(v.x), 0x01010101, 0);
    s = __dp4a(static_cast<int>(v.y), 0x01010101, s);
    atomicAdd(xsum + m, s);
  }
}

}  // namespace

cudaError_t launch_a8_planes(const int8_t* xq, int M, int K, uint8_t* planes, int32_t* xsum, cudaStream_t stream) {
  if (M == 0) return cudaSuccess;
  if (xsum != nullptr) {
    cudaError_t e = cudaMemsetAsync(xsum, 0, static_cast<size_t>(M) * sizeof(int32_t), stream);
    if (e != cudaSuccess) return e;
  }
  const long long threads = static_cast<long long>(M) * (K / 8);
  const unsigned grid = static_cast<unsigned>((threads + 255) / 256);
  a8_planes_kernel<<<grid, 256, 0, stream>>>(xq, M, K, planes, xsum);
  return cudaGetLastError();
}

}  // namespace qvla
