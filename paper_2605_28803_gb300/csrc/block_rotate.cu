// Online data-dependent rotation x' = x . P . BlockDiag(U_1, ..., U_nb) (Sec. 4.1, Eq. 4-5) for a
// layer whose activations cannot take it upstream (layers that share an input but fold different
// U_b, such as Q, K and V).  Float32 products and sums, one rounding to the activation dtype; the
// Hadamard factor and the quantiser then run on x' as for any other layer.
//
// One CTA takes 64 rows of one channel block b: it stages U_b (row-major [i][c]) and the 64
// gathered input rows x[m][perm[b*kB + i]] in shared memory, and each thread accumulates a 4-row
// x (kB/16)-column patch of x'[m][b*kB + c] = sum_i x[m][perm[b*kB + i]] U_b[i][c] in the order
// i = 0, 1, ..., kB - 1.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "kernels.h"

namespace qvla {
namespace {

constexpr int kRows = 64;  // rows per CTA
constexpr int kBrThreads = 256;

template <typename T>
__device__ __forceinline__ float load_f(const T* p);
template <>
__device__ __forceinline__ float load_f<__half>(const __half* p) {
  return __half2float(*p);
}
template <>
__device__ __forceinline__ float load_f<__nv_bfloat16>(const __nv_bfloat16* p) {
  return __bfloat162float(*p);
}
template <>
__device__ __forceinline__ float load_f<float>(const float* p) {
  return *p;
}

template <typename T>
__device__ __forceinline__ T round_to(float v);
template <>
__device__ __forceinline__ __half round_to<__half>(float v) {
  return __float2half_rn(v);
}
template <>
__device__ __forceinline__ __nv_bfloat16 round_to<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}
template <>
__device__ __forceinline__ float round_to<float>(float v) {
  return v;
}

template <typename T, int kB>
__global__ void __launch_bounds__(kBrThreads) block_rotate_kernel(const T* __restrict__ x, int M, int K,
                                                                   const int32_t* __restrict__ perm,
                                                                   const float* __restrict__ rot, T* __restrict__ out) {
  static_assert(kB % 16 == 0 && kB <= 64, "blocks of 16, 32 or 64 channels");
  constexpr int kC = kB / 16;  // output columns per thread, 16 apart
  __shared__ __align__(16) float su[kB * kB];
  __shared__ float sz[kRows][kB + 1];  // padded: the two row groups of a warp read distinct banks
  const int b = blockIdx.x;
  const int m0 = blockIdx.y * kRows;
  const int t = threadIdx.x;

  // every load is issued before any is used: thread t gathers channel perm[b kB + t % kB] of rows
  // t / kB, t / kB + kRStep, ..., and copies float4 t, t + kBrThreads, ... of U_b
  static_assert(kBrThreads % kB == 0, "a thread's gathered channel is fixed");
  constexpr int kRStep = kBrThreads / kB;
  constexpr int kPer = kRows / kRStep;                     // gathered values per thread
  constexpr int kU4 = kB * kB / 4;                         // float4 of U_b
  constexpr int kUPer = (kU4 + kBrThreads - 1) / kBrThreads;
  const float4* usrc = reinterpret_cast<const float4*>(rot + static_cast<size_t>(b) * kB * kB);
  float4 uv[kUPer];
#pragma unroll
  for (int j = 0; j < kUPer; ++j)
    if (kU4 % kBrThreads == 0 || t + j * kBrThreads < kU4) uv[j] = __ldg(usrc + t + j * kBrThreads);
  const int gi = t % kB, gr = t / kB;
  const int col = __ldg(perm + b * kB + gi);
  float gv[kPer];
#pragma unroll
  for (int j = 0; j < kPer; ++j) {
    const int m = m0 + gr + j * kRStep;
    gv[j] = m < M ? load_f(x + static_cast<size_t>(m) * K + col) : 0.0f;
  }
#pragma unroll
  for (int j = 0; j < kUPer; ++j)
    if (kU4 % kBrThreads == 0 || t + j * kBrThreads < kU4) reinterpret_cast<float4*>(su)[t + j * kBrThreads] = uv[j];
#pragma unroll
  for (int j = 0; j < kPer; ++j) sz[gr + j * kRStep][gi] = gv[j];
  __syncthreads();

  const int rg = t >> 4, cg = t & 15;  // rows 4 rg .. 4 rg + 3, columns cg + 16 j
  float acc[4][kC];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int j = 0; j < kC; ++j) acc[a][j] = 0.0f;
#pragma unroll 4
  for (int i = 0; i < kB; ++i) {
    float z[4], u[kC];
#pragma unroll
    for (int a = 0; a < 4; ++a) z[a] = sz[4 * rg + a][i];
#pragma unroll
    for (int j = 0; j < kC; ++j) u[j] = su[i * kB + cg + 16 * j];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int j = 0; j < kC; ++j) acc[a][j] = fmaf(z[a], u[j], acc[a][j]);
  }
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const int m = m0 + 4 * rg + a;
    if (m >= M) continue;
    T* dst = out + static_cast<size_t>(m) * K + b * kB + cg;
#pragma unroll
    for (int j = 0; j < kC; ++j) dst[16 * j] = round_to<T>(acc[a][j]);
  }
}

template <typename T>
cudaError_t launch_t(const void* x, int M, int K, const int32_t* perm, const float* rot, int block, void* out,
                     cudaStream_t stream) {
  const dim3 grid(K / block, (M + kRows - 1) / kRows);
  const T* xt = static_cast<const T*>(x);
  T* ot = static_cast<T*>(out);
  switch (block) {
    case 16: block_rotate_kernel<T, 16><<<grid, kBrThreads, 0, stream>>>(xt, M, K, perm, rot, ot); break;
    case 32: block_rotate_kernel<T, 32><<<grid, kBrThreads, 0, stream>>>(xt, M, K, perm, rot, ot); break;
    case 64: block_rotate_kernel<T, 64><<<grid, kBrThreads, 0, stream>>>(xt, M, K, perm, rot, ot); break;
    default: return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_block_rotate(const void* x, int xdt, int M, int K, const int32_t* perm, const float* rot, int block,
                                void* out, cudaStream_t stream) {
  if (M == 0) return cudaSuccess;
  if (block <= 0 || K % block != 0) return cudaErrorInvalidValue;
  switch (xdt) {
    case 0: return launch_t<__half>(x, M, K, perm, rot, block, out, stream);
    case 1: return launch_t<__nv_bfloat16>(x, M, K, perm, rot, block, out, stream);
    case 2: return launch_t<float>(x, M, K, perm, rot, block, out, stream);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace qvla
