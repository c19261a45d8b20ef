// Fused online rotation + symmetric int4 activation quantisation (Sec. 4.1 Eq. 3-5, the online
// block-Hadamard factor; Sec. 4.2 Eq. 5-6 with per-token or per-step scales).
//
// One row of x is spread over K/EPT threads, EPT consecutive elements each (16-byte loads).
// The fast Walsh-Hadamard transform of a block of b = 2^LOGB elements runs its butterfly
// stages on the low log2(EPT) index bits in registers, then transposes once through shared
// memory so that each thread holds the elements that differ in the remaining bits, and runs
// those stages in registers too.  The row's scale (per token: max |y| / 7), the int4 codes and
// the code sum follow from registers; codes leave as packed nibbles.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"

namespace qvla {
namespace {

constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23: adding it rounds a |t| < 2^22 to an integer (half to even)

template <typename T>
struct Loader;

template <>
struct Loader<__half> {
  static constexpr int kPer16B = 8;
  __device__ __forceinline__ static void load(const void* p, float* v) {
    uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
    const __half2* h = reinterpret_cast<const __half2*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 f = __half22float2(h[i]);
      v[2 * i] = f.x;
      v[2 * i + 1] = f.y;
    }
  }
};

template <>
struct Loader<__nv_bfloat16> {
  static constexpr int kPer16B = 8;
  __device__ __forceinline__ static void load(const void* p, float* v) {
    uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {  // bf16 -> f32 is a 16-bit shift
      v[2 * i] = __uint_as_float(w[i] << 16);
      v[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
};

template <>
struct Loader<float> {
  static constexpr int kPer16B = 4;
  __device__ __forceinline__ static void load(const void* p, float* v) {
    float4 f = __ldg(reinterpret_cast<const float4*>(p));
    v[0] = f.x;
    v[1] = f.y;
    v[2] = f.z;
    v[3] = f.w;
  }
};

// Butterfly stages on register-index bits [lo_bit, hi_bit): (a, c) -> (a + c, a - c).
template <int kN, int kLoBit, int kHiBit>
__device__ __forceinline__ void fwht_regs(float (&v)[kN]) {
#pragma unroll
  for (int bit = kLoBit; bit < kHiBit; ++bit) {
    const int h = 1 << bit;
#pragma unroll
    for (int i = 0; i < kN; ++i) {
      if ((i & h) == 0) {
        const float a = v[i], c = v[i + h];
        v[i] = a + c;
        v[i + h] = a - c;
      }
    }
  }
}

// Exact symmetric int4 decision for one value: clamp(round(z / delta), -7, 7), half to even,
// on the exact quotient.  The fast path t = z * rcp is within 2^-20 of z / delta, so unless
// t lies within 2^-17 of a half-integer its nearest integer is the answer; otherwise the sign
// of fma(-h, delta, z) -- exact sign of z - h*delta for the half-integer h -- decides.
// Returns the code as the float kMagic + q (its low nibble is the two's-complement code).
__device__ __forceinline__ float quantize_one(float z, float delta, float rcp) {
  float t = fminf(fmaxf(z * rcp, -7.0f), 7.0f);
  float u = t + kMagic;
  const float n = u - kMagic;
  if (fabsf(t - n) >= 0.5f - 7.62939453125e-6f) {  // within 2^-17 of a tie: decide exactly
    const float fl = floorf(t);
    const float d = fmaf(-(fl + 0.5f), delta, z);
    float q = d > 0.0f ? fl + 1.0f : fl;
    if (d == 0.0f) q = (fmodf(fl, 2.0f) == 0.0f) ? fl : fl + 1.0f;  // exact tie: even neighbour
    q = fminf(fmaxf(q, -7.0f), 7.0f);
    u = q + kMagic;
  }
  return u;
}

__device__ __forceinline__ uint32_t nib(float u) { return __float_as_uint(u) & 0xFu; }

// kLogB: log2 of the Hadamard block (0 = no rotation).  kEpt: elements per thread.
template <typename T, int kLogB, int kEpt>
__global__ void __launch_bounds__(256) rotate_quant_kernel(const T* __restrict__ x, int M, int K, float inv_sqrt_b,
                                                             int mode, const float* __restrict__ step_scale,
                                                             uint8_t* __restrict__ xq, float* __restrict__ xscale,
                                                             int32_t* __restrict__ xsum, float* __restrict__ absmax_out) {
  constexpr int kP = (kEpt == 128) ? 7 : 6;  // log2(kEpt)
  static_assert((1 << kP) == kEpt, "EPT");
  constexpr bool kPhase2 = kLogB > kP;
  constexpr int kR = kPhase2 ? kLogB - kP : 0;  // bits handled after the transpose
  constexpr int kL = kP - kR;                  // contiguous low bits per run after the transpose
  static_assert(!kPhase2 || kL >= 1, "every run must hold whole nibble pairs");
  constexpr int kRun = kPhase2 ? (1 << kL) : kEpt;  // contiguous elements per run
  constexpr int kNV = kEpt / 4;                     // float4 per shared-memory line

  extern __shared__ float4 smem4[];
  __shared__ unsigned int s_max[32];
  __shared__ int s_sum[32];

  const int tpr = K / kEpt;           // threads per row
  const int rpc = blockDim.x / tpr;   // rows per CTA
  const int tid = threadIdx.x;
  const int rloc = tid / tpr;         // row within the CTA
  const int j = tid - rloc * tpr;     // thread within the row
  const int m = blockIdx.x * rpc + rloc;
  const bool active = (rloc < rpc) && (m < M);

  if (tid < 32) {
    s_max[tid] = 0u;
    s_sum[tid] = 0;
  }
  __syncthreads();

  float v[kEpt];
  // ---- load (phase-1 layout: elements j*kEpt .. j*kEpt + kEpt - 1 of the row) ----
  if (active) {
    const T* src = x + static_cast<size_t>(m) * K + static_cast<size_t>(j) * kEpt;
#pragma unroll
    for (int c = 0; c < kEpt / Loader<T>::kPer16B; ++c) Loader<T>::load(src + c * Loader<T>::kPer16B, v + c * Loader<T>::kPer16B);
  } else {
#pragma unroll
    for (int i = 0; i < kEpt; ++i) v[i] = 0.0f;
  }

  // ---- butterflies on the low bits ----
  constexpr int kLowBits = kLogB < kP ? kLogB : kP;
  fwht_regs<kEpt, 0, kLowBits>(v);

  // ---- transpose through shared memory, butterflies on the high bits ----
  if constexpr (kPhase2) {
    float* s = reinterpret_cast<float*>(smem4) + static_cast<size_t>(rloc) * K;
    float4* s4 = reinterpret_cast<float4*>(s);
#pragma unroll
    for (int c = 0; c < kNV; ++c) {
      const int line = j;
      s4[line * kNV + (c ^ (line & (kNV - 1)))] = make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
    }
    __syncthreads();
    const int jlo = j & ((1 << kR) - 1);
    const int jhi = j >> kR;
#pragma unroll
    for (int ih = 0; ih < (1 << kR); ++ih) {
      const int line = (jhi << kR) | ih;
      const int col = jlo << kL;
      if constexpr (kL >= 2) {
#pragma unroll
        for (int c = 0; c < (1 << (kL - 2)); ++c) {
          const int vv = (col >> 2) + c;
          const float4 f = s4[line * kNV + (vv ^ (line & (kNV - 1)))];
          const int r = (ih << kL) + 4 * c;
          v[r] = f.x;
          v[r + 1] = f.y;
          v[r + 2] = f.z;
          v[r + 3] = f.w;
        }
      } else {  // kL == 1: a float pair
        const int vv = col >> 2;
        const float2 f = *reinterpret_cast<const float2*>(
            reinterpret_cast<const float*>(s4 + line * kNV + (vv ^ (line & (kNV - 1)))) + (col & 3));
        v[ih << 1] = f.x;
        v[(ih << 1) + 1] = f.y;
      }
    }
    fwht_regs<kEpt, kL, kP>(v);
  }

  // ---- scale ----
  float local_max = 0.0f;
  if (mode != 1) {
#pragma unroll
    for (int i = 0; i < kEpt; ++i) local_max = fmaxf(local_max, fabsf(v[i]));
  }
  if (mode == 2) {  // calibration: CTA max, one atomic per CTA
    float w = local_max;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) w = fmaxf(w, __shfl_xor_sync(0xffffffffu, w, o));
    __syncthreads();
    if ((tid & 31) == 0) atomicMax(&s_max[0], __float_as_uint(w));
    __syncthreads();
    if (tid == 0) atomicMax(reinterpret_cast<unsigned int*>(absmax_out), __float_as_uint(__uint_as_float(s_max[0]) * inv_sqrt_b));
    return;
  }

  float delta;
  if (mode == 1) {
    delta = __ldg(step_scale);
  } else {
    // per-token: reduce |y| over the row (the row's threads are tpr consecutive threads)
    float w = local_max;
    if ((tpr & 31) == 0) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) w = fmaxf(w, __shfl_xor_sync(0xffffffffu, w, o));
      __syncthreads();
      if ((tid & 31) == 0) atomicMax(&s_max[rloc], __float_as_uint(w));
    } else if ((tpr & (tpr - 1)) == 0) {
      for (int o = tpr >> 1; o > 0; o >>= 1) w = fmaxf(w, __shfl_xor_sync(0xffffffffu, w, o));
      __syncthreads();
      if (j == 0) atomicMax(&s_max[rloc], __float_as_uint(w));
    } else {
      __syncthreads();
      atomicMax(&s_max[rloc], __float_as_uint(w));
    }
    __syncthreads();
    // max |Z| of the normalised rotation: rounding is monotone, so round(max * c) = max round(y * c)
    const float zmax = (kLogB == 0) ? __uint_as_float(s_max[rloc]) : __uint_as_float(s_max[rloc]) * inv_sqrt_b;
    delta = __fdiv_rn(zmax, 7.0f);
  }
  if (active && j == 0) xscale[m] = delta;

  // ---- codes ----
  float rcp = (delta > 0.0f) ? __fdiv_rn(1.0f, delta) : 0.0f;
  const bool zero_scale = !(delta > 0.0f);
  // A scale so small that 1/delta overflows: decide by plain division (no tie refinement).
  const bool tiny_scale = !zero_scale && isinf(rcp);
  float codesum = 0.0f;
  uint8_t* dst = xq + static_cast<size_t>(m) * (K / 2);
#pragma unroll
  for (int run = 0; run < kEpt / kRun; ++run) {
    int e0;  // first element of this run within the row
    if constexpr (kPhase2) {
      e0 = ((j >> kR) << kLogB) | (run << kP) | ((j & ((1 << kR) - 1)) << kL);
    } else {
      e0 = j * kEpt;
    }
    uint32_t packed[(kRun + 7) / 8];
#pragma unroll
    for (int w = 0; w < (kRun + 7) / 8; ++w) packed[w] = 0u;
#pragma unroll
    for (int i = 0; i < kRun; ++i) {
      float z = v[run * kRun + i];
      if (kLogB != 0) z *= inv_sqrt_b;
      float u;
      if (zero_scale) {
        u = kMagic;
      } else if (tiny_scale) {
        u = fminf(fmaxf(__fdiv_rn(z, delta), -7.0f), 7.0f) + kMagic;
      } else {
        u = quantize_one(z, delta, rcp);
      }
      codesum += u - kMagic;
      packed[i / 8] |= nib(u) << (4 * (i % 8));
    }
    if (active) {
      uint8_t* p = dst + (e0 >> 1);
      if constexpr (kRun == 2) {
        *p = static_cast<uint8_t>(packed[0]);
      } else if constexpr (kRun == 4) {
        *reinterpret_cast<uint16_t*>(p) = static_cast<uint16_t>(packed[0]);
      } else if constexpr (kRun == 8) {
        *reinterpret_cast<uint32_t*>(p) = packed[0];
      } else if constexpr (kRun == 16) {
        *reinterpret_cast<uint2*>(p) = make_uint2(packed[0], packed[1]);
      } else {
#pragma unroll
        for (int w = 0; w < kRun / 8; w += 4)
          *reinterpret_cast<uint4*>(p + 4 * w) = make_uint4(packed[w], packed[w + 1], packed[w + 2], packed[w + 3]);
      }
    }
  }
  if (xsum != nullptr) {
    int cs = static_cast<int>(codesum);
    if ((tpr & 31) == 0) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cs += __shfl_xor_sync(0xffffffffu, cs, o);
      if ((tid & 31) == 0) atomicAdd(&s_sum[rloc], cs);
    } else if ((tpr & (tpr - 1)) == 0) {
      for (int o = tpr >> 1; o > 0; o >>= 1) cs += __shfl_xor_sync(0xffffffffu, cs, o);
      if (j == 0) atomicAdd(&s_sum[rloc], cs);
    } else {
      atomicAdd(&s_sum[rloc], cs);
    }
    __syncthreads();
    if (active && j == 0) xsum[m] = s_sum[rloc];
  }
}

template <typename T, int kLogB>
cudaError_t launch_t(const RotQuantArgs& a) {
  constexpr int kEpt = kLogB >= 12 ? 128 : 64;
  const int tpr = a.K / kEpt;
  int tpb = tpr >= 128 ? tpr : (128 / tpr) * tpr;
  const int rpc = tpb / tpr;
  if (rpc > 32) {  // the per-row reduction slots hold 32 rows
    tpb = 32 * tpr;
  }
  const int rows = tpb / tpr;
  const int grid = (a.M + rows - 1) / rows;
  if (grid == 0) return cudaSuccess;
  const size_t smem = (kLogB > ((kEpt == 128) ? 7 : 6)) ? static_cast<size_t>(tpb) * kEpt * sizeof(float) : 0;
  auto kern = rotate_quant_kernel<T, kLogB, kEpt>;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  kern<<<grid, tpb, smem, a.stream>>>(reinterpret_cast<const T*>(a.x), a.M, a.K, a.inv_sqrt_b, a.mode, a.step_scale,
                                      a.xq, a.xscale, a.xsum, a.absmax);
  return cudaGetLastError();
}

template <typename T>
cudaError_t launch_dtype(const RotQuantArgs& a) {
  switch (a.log_b) {
    case 0: return launch_t<T, 0>(a);
    case 1: return launch_t<T, 1>(a);
    case 2: return launch_t<T, 2>(a);
    case 3: return launch_t<T, 3>(a);
    case 4: return launch_t<T, 4>(a);
    case 5: return launch_t<T, 5>(a);
    case 6: return launch_t<T, 6>(a);
    case 7: return launch_t<T, 7>(a);
    case 8: return launch_t<T, 8>(a);
    case 9: return launch_t<T, 9>(a);
    case 10: return launch_t<T, 10>(a);
    case 11: return launch_t<T, 11>(a);
    case 12: return launch_t<T, 12>(a);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

bool rotate_quant_supported(int log_b) { return log_b >= 0 && log_b <= 12; }

cudaError_t launch_rotate_quant(const RotQuantArgs& a) {
  switch (a.xdt) {
    case 0: return launch_dtype<__half>(a);
    case 1: return launch_dtype<__nv_bfloat16>(a);
    case 2: return launch_dtype<float>(a);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace qvla
