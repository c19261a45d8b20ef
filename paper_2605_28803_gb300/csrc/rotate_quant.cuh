// Fused online rotation + symmetric int4 activation quantisation (Sec. 4.1 Eq. 3-5, the online
// block-Hadamard factor; Sec. 4.2 Eq. 5-6 with per-token or per-step scales).
//
// One row of x is spread over K/EPT threads, EPT consecutive elements each (16-byte loads),
// held as float2 pairs.  The fast Walsh-Hadamard transform of a block of b = 2^LOGB elements
// runs its butterfly stages on the low log2(EPT) index bits in registers (stages of distance
// >= 2 as packed f32x2 adds/subs), then transposes once through shared memory so that each
// thread holds the elements that differ in the remaining bits, and runs those in registers
// too.  The scale (per token: max |y| / q_max; or the step's table entry), the codes, their
// packing and the row's code sum follow from registers.  Codes are int4 (q_max 7) or, for the
// W4A8 variant, int8 (q_max 127).  Instantiated per input dtype and code width in
// rotate_quant_{f16,bf16,f32}.cu (4-bit) and rotate_quant_a8_{f16,bf16,f32}.cu (8-bit).
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>

#include "a8_codes.cuh"
#include "griddep.cuh"
#include "kernels.h"

namespace qvla {
namespace rq {

constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23: t + kMagic rounds |t| < 2^22 to an integer, half to even
// The fast path t = y * (c / delta) is within 2^-20 of the exact z / delta (|t| <= 8); a value
// closer than this to a half-integer is decided exactly instead.
constexpr float kTieBand = 0.5f - 7.62939453125e-6f;  // 0.5 - 2^-17
// With 8-bit codes |t| <= 128, so the fast path is within 2^-15: a wider band, 2^-12.
constexpr float kTieBand8 = 0.5f - 2.44140625e-4f;

template <typename T>
struct Loader;

template <>
struct Loader<__half> {
  static constexpr int kPer16B = 8;
  __device__ __forceinline__ static void load(const void* p, float2* v) {
    uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
    const __half2* h = reinterpret_cast<const __half2*>(&u);
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = __half22float2(h[i]);
  }
};

template <>
struct Loader<__nv_bfloat16> {
  static constexpr int kPer16B = 8;
  __device__ __forceinline__ static void load(const void* p, float2* v) {
    uint4 u = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xFFFF0000u));
  }
};

template <>
struct Loader<float> {
  static constexpr int kPer16B = 4;
  __device__ __forceinline__ static void load(const void* p, float2* v) {
    float4 f = __ldg(reinterpret_cast<const float4*>(p));
    v[0] = make_float2(f.x, f.y);
    v[1] = make_float2(f.z, f.w);
  }
};

// (a, c) -> (a + c, a - c), two lanes at once; a - c as one rounding of c * (-1) + a, the same
// value a subtraction gives.
__device__ __forceinline__ void bfly2(float2& a, float2& c) {
  const float2 s = __fadd2_rn(a, c);
  c = __ffma2_rn(c, make_float2(-1.0f, -1.0f), a);
  a = s;
}

// Butterflies on element-index bits [lo, hi) of v (kN float2 = 2 kN elements; bit 0 is the
// pair's own lane).
template <int kN, int kLo, int kHi>
__device__ __forceinline__ void fwht_regs(float2 (&v)[kN]) {
  if constexpr (kLo == 0 && kHi > 0) {
#pragma unroll
    for (int i = 0; i < kN; ++i) {
      const float a = v[i].x, c = v[i].y;
      v[i] = make_float2(a + c, a - c);
    }
  }
#pragma unroll
  for (int bit = (kLo > 1 ? kLo : 1); bit < kHi; ++bit) {
    const int h = 1 << (bit - 1);  // distance in float2 units
#pragma unroll
    for (int i = 0; i < kN; ++i)
      if ((i & h) == 0) bfly2(v[i], v[i + h]);
  }
}

// The exact decision for one value (rare: only near a tie, or when 1/delta overflows): round
// half to even of the exact quotient z / delta for z = float32(y * c), by the sign of
// z - h delta (one FMA is exact in sign) at the half-integer h next to t, then the clamp to
// [-qmax, qmax].  Returns kMagic + q.
static __device__ __noinline__ float exact_code(float y, float c, float delta, float cr, float qmax, float band) {
  const float z = y * c;
  if (isinf(cr)) return fminf(fmaxf(__fdiv_rn(z, delta), -qmax), qmax) + kMagic;  // tiny delta
  const float t = fminf(fmaxf(y * cr, -qmax), qmax);
  if (fabsf(t - ((t + kMagic) - kMagic)) < band) return t + kMagic;  // not near a tie
  const float fl = floorf(t);
  const float d = fmaf(-(fl + 0.5f), delta, z);
  float q = d > 0.0f ? fl + 1.0f : fl;
  if (d == 0.0f) q = (static_cast<int>(fl) & 1) ? fl + 1.0f : fl;
  q = fminf(fmaxf(q, -qmax), qmax);
  return q + kMagic;
}

// The low bytes of four words, in order, as one word.  A code held as the float kMagic + q has
// q's two's-complement low byte as the low byte of its bits.
__device__ __forceinline__ uint32_t low_bytes(float a, float b, float c, float d) {
  return __byte_perm(__byte_perm(__float_as_uint(a), __float_as_uint(b), 0x0040),
                     __byte_perm(__float_as_uint(c), __float_as_uint(d), 0x0040), 0x5410);
}

// Sum of the 8 two's-complement codes of a packed word, plus 64 (each code offset by 8).
__device__ __forceinline__ uint32_t sum8_offset(uint32_t w, uint32_t acc) {
  const uint32_t o = w ^ 0x88888888u;
  const uint32_t s = (o & 0x0F0F0F0Fu) + ((o >> 4) & 0x0F0F0F0Fu);
  return __dp4a(s, 0x01010101u, acc);
}

// kLogB: log2 of the Hadamard block (0 = no rotation).  kEpt: elements per thread.
// kStep: the scale is the step table entry (else per token; per-token mode also serves the
// calibration max when absmax_out is set).  Scale groups: channel k belongs to group
// k >> gshift (gshift >= 30: one group).  A group holds whole Hadamard blocks and at least 128
// channels, so all of a thread's elements share one group: with a per-group step table
// (step_scale[g]) the thread takes its group's entry, xgsum (when set) receives each group's
// code sum [M][K >> gshift], and calibration (absmax_out) raises one maximum per group.
// kA8: 8-bit codes (q_max 127; out_mode int8 rows or the GEMM's two operand planes), else
// 4-bit (q_max 7; packed nibbles or operand bytes).
template <typename T, int kLogB, int kEpt, bool kStep, bool kA8>
__global__ void __launch_bounds__(256) rotate_quant_kernel(const T* __restrict__ x, int M, int K, float inv_sqrt_b,
                                                             const float* __restrict__ step_scale,
                                                             uint8_t* __restrict__ xq, float* __restrict__ xscale,
                                                             int32_t* __restrict__ xsum, float* __restrict__ absmax_out,
                                                             int out_mode, int gshift, int32_t* __restrict__ xgsum,
                                                             int32_t* __restrict__ zero, int zero_n) {
  constexpr float kQ = kA8 ? 127.0f : 7.0f;
  constexpr float kBand = kA8 ? kTieBand8 : kTieBand;
  constexpr int kP = (kEpt == 128) ? 7 : 6;  // log2(kEpt)
  static_assert((1 << kP) == kEpt, "EPT");
  constexpr int kN = kEpt / 2;                // float2 per thread
  constexpr bool kPhase2 = kLogB > kP;
  constexpr int kR = kPhase2 ? kLogB - kP : 0;  // bits handled after the transpose
  constexpr int kL = kP - kR;                  // contiguous low bits per run after the transpose
  static_assert(!kPhase2 || kL >= 1, "every run must hold whole nibble pairs");
  constexpr int kRun = kPhase2 ? (1 << kL) : kEpt;  // contiguous elements per run
  constexpr int kNV = kEpt / 4;                     // float4 per shared-memory line

  extern __shared__ float4 smem4[];
  __shared__ unsigned int s_max[32];
  __shared__ unsigned int s_sum[32];

  const int tpr = K / kEpt;           // threads per row
  const int rpc = blockDim.x / tpr;   // rows per CTA
  const int tid = threadIdx.x;
  const int rloc = tid / tpr;         // row within the CTA
  const int j = tid - rloc * tpr;     // thread within the row
  const int m = blockIdx.x * rpc + rloc;
  const bool active = (rloc < rpc) && (m < M);
  // the channel of this thread's first element, and so its scale group
  int e_first;
  if constexpr (kPhase2) {
    e_first = ((j >> kR) << kLogB) | ((j & ((1 << kR) - 1)) << kL);
  } else {
    e_first = j * kEpt;
  }
  const int grp = gshift >= 30 ? 0 : e_first >> gshift;

  if (tid < 32) {
    s_max[tid] = 0u;
    s_sum[tid] = 0u;
  }

  griddep_wait();  // x comes from the previous kernel, which may still read xq / xscale / xsum
  griddep_launch_dependents();
  if (zero != nullptr && blockIdx.x == 0)  // the next GEMM's work-unit counters (its previous use is over)
    for (int i = tid; i < zero_n; i += blockDim.x) zero[i] = 0;
  float2 v[kN];
  if (active) {
    const T* src = x + static_cast<size_t>(m) * K + static_cast<size_t>(j) * kEpt;
#pragma unroll
    for (int c = 0; c < kEpt / Loader<T>::kPer16B; ++c)
      Loader<T>::load(src + c * Loader<T>::kPer16B, v + c * (Loader<T>::kPer16B / 2));
  } else {
#pragma unroll
    for (int i = 0; i < kN; ++i) v[i] = make_float2(0.0f, 0.0f);
  }
  __syncthreads();  // the reduction slots are cleared before any thread adds to them

  constexpr int kLowBits = kLogB < kP ? kLogB : kP;
  fwht_regs<kN, 0, kLowBits>(v);

  if constexpr (kPhase2) {
    float4* s4 = reinterpret_cast<float4*>(reinterpret_cast<float*>(smem4) + static_cast<size_t>(rloc) * K);
#pragma unroll
    for (int c = 0; c < kNV; ++c) {
      const int line = j;
      s4[line * kNV + (c ^ (line & (kNV - 1)))] = make_float4(v[2 * c].x, v[2 * c].y, v[2 * c + 1].x, v[2 * c + 1].y);
    }
    // A Hadamard block's 2^kR threads (at most 32, starting at a multiple of 2^kR) lie in one
    // warp, and each reads back only its block's lines: the warp alone must have stored them.
    static_assert(kR <= 5, "a Hadamard block's threads fit in one warp");
    __syncwarp();
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
          const int r = ((ih << kL) + 4 * c) >> 1;
          v[r] = make_float2(f.x, f.y);
          v[r + 1] = make_float2(f.z, f.w);
        }
      } else {  // kL == 1: one pair
        const int vv = col >> 2;
        v[ih] = *reinterpret_cast<const float2*>(
            reinterpret_cast<const float*>(s4 + line * kNV + (vv ^ (line & (kNV - 1)))) + (col & 3));
      }
    }
    fwht_regs<kN, kL, kP>(v);
  }

  // ---- scale ----
  float delta;
  if constexpr (kStep) {
    delta = __ldg(step_scale + grp);
  } else {
    float w = 0.0f;
#pragma unroll
    for (int i = 0; i < kN; ++i) w = fmaxf(w, fmaxf(fabsf(v[i].x), fabsf(v[i].y)));
    if (absmax_out != nullptr && gshift < 30) {
      // per-group calibration: the group's threads are consecutive lanes, tg of them (tg | 32)
      const int tg = (1 << gshift) / kEpt;
      for (int o = tg >> 1; o > 0; o >>= 1) w = fmaxf(w, __shfl_xor_sync(0xffffffffu, w, o));
      if (active && (j & (tg - 1)) == 0)
        atomicMax(reinterpret_cast<unsigned int*>(absmax_out + grp), __float_as_uint(w * inv_sqrt_b));
      return;
    }
    if ((tpr & 31) == 0) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) w = fmaxf(w, __shfl_xor_sync(0xffffffffu, w, o));
      if ((tid & 31) == 0) atomicMax(&s_max[rloc], __float_as_uint(w));
    } else if ((tpr & (tpr - 1)) == 0) {
      for (int o = tpr >> 1; o > 0; o >>= 1) w = fmaxf(w, __shfl_xor_sync(0xffffffffu, w, o));
      if (j == 0) atomicMax(&s_max[rloc], __float_as_uint(w));
    } else {
      atomicMax(&s_max[rloc], __float_as_uint(w));
    }
    __syncthreads();
    // max |Z| of the normalised rotation: rounding is monotone, so round(max * c) = max round(y * c)
    const float zmax = __uint_as_float(s_max[rloc]) * inv_sqrt_b;
    if (absmax_out != nullptr) {  // calibration: one atomic per row
      if (active && j == 0) atomicMax(reinterpret_cast<unsigned int*>(absmax_out), __float_as_uint(zmax));
      return;
    }
    delta = __fdiv_rn(zmax, kQ);
  }
  if (active && j == 0) xscale[m] = delta;

  // ---- codes ----
  const bool zero_scale = !(delta > 0.0f);
  const float rcp = zero_scale ? 0.0f : __fdiv_rn(1.0f, delta);
  const bool tiny_scale = !zero_scale && isinf(rcp);  // 1/delta overflows: plain division
  const float cr = inv_sqrt_b * rcp;                  // y * cr ~ z / delta (0 when delta = 0: codes 0)
  // codes in register order, 8 per word (register element r = 8 g + i)
  // 4-bit: pk = packed nibbles; 8-bit: ev / od = the two's-complement code bytes of the even /
  // odd elements of each group of 8
  uint32_t pk[kA8 ? 1 : kEpt / 8], ev[kA8 ? kEpt / 8 : 1], od[kA8 ? kEpt / 8 : 1];
  uint32_t sum_acc = 0;
  const float2 cr2 = make_float2(cr, cr);
  const float2 magic2 = make_float2(kMagic, kMagic), nmagic2 = make_float2(-kMagic, -kMagic);
  const float2 neg2 = make_float2(-1.0f, -1.0f);
#pragma unroll
  for (int g = 0; g < kEpt / 8; ++g) {
    // elements 8 g + 2 i (.x) and 8 g + 2 i + 1 (.y), as kMagic + code, two at a time
    float2 u[4];
    float dev = 0.0f;  // the largest distance |t - round(t)| of the 8
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float2 t = __fmul2_rn(v[4 * g + i], cr2);
      if constexpr (kStep) {
        t.x = fminf(fmaxf(t.x, -kQ), kQ);
        t.y = fminf(fmaxf(t.y, -kQ), kQ);
      }
      u[i] = __fadd2_rn(t, magic2);
      const float2 d = __ffma2_rn(__fadd2_rn(u[i], nmagic2), neg2, t);  // t - round(t)
      dev = fmaxf(dev, fmaxf(fabsf(d.x), fabsf(d.y)));
    }
    if (dev >= kBand || tiny_scale) {  // rare: decide these values exactly
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        u[i].x = exact_code(v[4 * g + i].x, inv_sqrt_b, delta, cr, kQ, kBand);
        u[i].y = exact_code(v[4 * g + i].y, inv_sqrt_b, delta, cr, kQ, kBand);
      }
    }
    // byte j of the packed word: code 8 g + 2 j (low nibble) and 8 g + 2 j + 1 (high nibble)
    const uint32_t even = low_bytes(u[0].x, u[1].x, u[2].x, u[3].x);
    const uint32_t odd = low_bytes(u[0].y, u[1].y, u[2].y, u[3].y);
    if constexpr (kA8) {
      ev[g] = even;
      od[g] = odd;
      sum_acc = __dp4a(even ^ 0x80808080u, 0x01010101u, sum_acc);  // sum of q + 128
      sum_acc = __dp4a(odd ^ 0x80808080u, 0x01010101u, sum_acc);
    } else {
      pk[g] = (even & 0x0F0F0F0Fu) | ((odd << 4) & 0xF0F0F0F0u);
      sum_acc = sum8_offset(pk[g], sum_acc);
    }
  }

  // ---- store: run r holds register elements [r kRun, (r + 1) kRun), contiguous in the row ----
  if constexpr (!kA8) {
  if (active && out_mode == 0) {  // packed nibbles [M][K/2]
    uint8_t* dst = xq + static_cast<size_t>(m) * (K / 2);
#pragma unroll
    for (int run = 0; run < kEpt / kRun; ++run) {
      int e0;  // first element of this run within the row
      if constexpr (kPhase2) {
        e0 = ((j >> kR) << kLogB) | (run << kP) | ((j & ((1 << kR) - 1)) << kL);
      } else {
        e0 = j * kEpt;
      }
      uint8_t* p = dst + (e0 >> 1);
      constexpr int kBytes = kRun / 2;
      const int b0 = run * kBytes;  // first byte of the run in pk
      if constexpr (kBytes == 1) {
        *p = static_cast<uint8_t>(pk[b0 >> 2] >> (8 * (b0 & 3)));
      } else if constexpr (kBytes == 2) {
        *reinterpret_cast<uint16_t*>(p) = static_cast<uint16_t>(pk[b0 >> 2] >> (8 * (b0 & 3)));
      } else if constexpr (kBytes == 4) {
        *reinterpret_cast<uint32_t*>(p) = pk[b0 >> 2];
      } else if constexpr (kBytes == 8) {
        *reinterpret_cast<uint2*>(p) = make_uint2(pk[b0 >> 2], pk[(b0 >> 2) + 1]);
      } else {
#pragma unroll
        for (int w = 0; w < kBytes / 4; w += 4)
          *reinterpret_cast<uint4*>(p + 4 * w) =
              make_uint4(pk[(b0 >> 2) + w], pk[(b0 >> 2) + w + 1], pk[(b0 >> 2) + w + 2], pk[(b0 >> 2) + w + 3]);
      }
    }
  } else if (active) {
    // One byte per code, the GEMM's tensor-core operand encoding: code q as the E4M3 byte
    // q + 8 (= q XOR 8).  Within each group of 8 consecutive k the bytes are stored in the order
    // k0 k2 k4 k6 k1 k3 k5 k7 -- the order the GEMM gives the packed operand it expands -- so
    // both operands of the dot product agree.
    uint8_t* dst = xq + static_cast<size_t>(m) * K;
    uint32_t lo[kEpt / 8], hi[kEpt / 8];
#pragma unroll
    for (int g = 0; g < kEpt / 8; ++g) {
      lo[g] = (pk[g] ^ 0x88888888u) & 0x0F0F0F0Fu;          // even elements of the 8
      hi[g] = ((pk[g] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;   // odd elements
    }
#pragma unroll
    for (int run = 0; run < kEpt / kRun; ++run) {
      int e0;
      if constexpr (kPhase2) {
        e0 = ((j >> kR) << kLogB) | (run << kP) | ((j & ((1 << kR) - 1)) << kL);
      } else {
        e0 = j * kEpt;
      }
      uint8_t* gb = dst + (e0 & ~7);  // the 8-byte group this run starts in
      const int o = e0 & 7;
      if constexpr (kRun >= 8) {
#pragma unroll
        for (int t = 0; t < kRun / 8; ++t) {
          const int w = run * (kRun / 8) + t;
          *reinterpret_cast<uint2*>(dst + e0 + 8 * t) = make_uint2(lo[w], hi[w]);
        }
      } else if constexpr (kRun == 4) {  // elements o..o+3 (o = 0 or 4) of a group
        const int w = run >> 1, h = run & 1;
        *reinterpret_cast<uint16_t*>(gb + (o >> 1)) = static_cast<uint16_t>(lo[w] >> (16 * h));
        *reinterpret_cast<uint16_t*>(gb + 4 + (o >> 1)) = static_cast<uint16_t>(hi[w] >> (16 * h));
      } else {  // kRun == 2: elements o, o+1
        const int w = run >> 2, q = run & 3;
        gb[o >> 1] = static_cast<uint8_t>(lo[w] >> (8 * q));
        gb[4 + (o >> 1)] = static_cast<uint8_t>(hi[w] >> (8 * q));
      }
    }
  }
  }  // 4-bit
  if constexpr (kA8) {
    if (active) {
#pragma unroll
      for (int run = 0; run < kEpt / kRun; ++run) {
        int e0;  // first element of this run within the row
        if constexpr (kPhase2) {
          e0 = ((j >> kR) << kLogB) | (run << kP) | ((j & ((1 << kR) - 1)) << kL);
        } else {
          e0 = j * kEpt;
        }
        if (out_mode == 2) {
          // int8 codes [M][K], natural order
          int8_t* dst = reinterpret_cast<int8_t*>(xq) + static_cast<size_t>(m) * K + e0;
          if constexpr (kRun >= 8) {
#pragma unroll
            for (int t = 0; t < kRun / 8; ++t) {
              const int w = run * (kRun / 8) + t;
              *reinterpret_cast<uint2*>(dst + 8 * t) =
                  make_uint2(__byte_perm(ev[w], od[w], 0x5140), __byte_perm(ev[w], od[w], 0x7362));
            }
          } else if constexpr (kRun == 4) {  // elements 4 h .. 4 h + 3 of group w
            const int w = run >> 1, h = run & 1;
            *reinterpret_cast<uint32_t*>(dst) = h ? __byte_perm(ev[w], od[w], 0x7362) : __byte_perm(ev[w], od[w], 0x5140);
          } else {  // kRun == 2: elements 2 q, 2 q + 1 of group w
            const int w = run >> 2, q = run & 3;
            *reinterpret_cast<uint16_t*>(dst) =
                static_cast<uint16_t>(((ev[w] >> (8 * q)) & 0xFFu) | (((od[w] >> (8 * q)) & 0xFFu) << 8));
          }
        } else {
          // the GEMM's two operand planes [M][2K]: per k-block of 128 codes, 128 bytes of the
          // high nibbles (E4M3 of v 2^-5) then 128 of the low nibbles (E4M3 of v 2^-9), each
          // group of 8 in the order k0 k2 k4 k6 k1 k3 k5 k7; nibbles of q + 128
          uint8_t* hp = xq + static_cast<size_t>(m) * (2 * K) + 2 * (e0 & ~127) + ((e0 & 127) & ~7);
          uint8_t* lp = hp + 128;
          auto planes = [&](int w, uint32_t& he, uint32_t& ho, uint32_t& le, uint32_t& lo) {
            a8_planes(ev[w], od[w], he, ho, le, lo);
          };
          if constexpr (kRun >= 8) {
#pragma unroll
            for (int t = 0; t < kRun / 8; ++t) {
              uint32_t he, ho, le, lo;
              planes(run * (kRun / 8) + t, he, ho, le, lo);
              *reinterpret_cast<uint2*>(hp + 8 * t) = make_uint2(he, ho);
              *reinterpret_cast<uint2*>(lp + 8 * t) = make_uint2(le, lo);
            }
          } else if constexpr (kRun == 4) {  // elements o .. o + 3 (o = 4 h) of a group
            const int w = run >> 1, h = run & 1, o = e0 & 7;
            uint32_t he, ho, le, lo;
            planes(w, he, ho, le, lo);
            *reinterpret_cast<uint16_t*>(hp + (o >> 1)) = static_cast<uint16_t>(he >> (16 * h));
            *reinterpret_cast<uint16_t*>(hp + 4 + (o >> 1)) = static_cast<uint16_t>(ho >> (16 * h));
            *reinterpret_cast<uint16_t*>(lp + (o >> 1)) = static_cast<uint16_t>(le >> (16 * h));
            *reinterpret_cast<uint16_t*>(lp + 4 + (o >> 1)) = static_cast<uint16_t>(lo >> (16 * h));
          } else {  // kRun == 2: elements o, o + 1 (o = 2 q)
            const int w = run >> 2, q = run & 3, o = e0 & 7;
            uint32_t he, ho, le, lo;
            planes(w, he, ho, le, lo);
            hp[o >> 1] = static_cast<uint8_t>(he >> (8 * q));
            hp[4 + (o >> 1)] = static_cast<uint8_t>(ho >> (8 * q));
            lp[o >> 1] = static_cast<uint8_t>(le >> (8 * q));
            lp[4 + (o >> 1)] = static_cast<uint8_t>(lo >> (8 * q));
          }
        }
      }
    }
  }
  if (xgsum != nullptr) {  // the code sum of each scale group of the row (tg consecutive lanes)
    int gs = static_cast<int>(sum_acc) - (kA8 ? 128 : 8) * kEpt;
    const int tg = (1 << gshift) / kEpt;
    for (int o = tg >> 1; o > 0; o >>= 1) gs += __shfl_xor_sync(0xffffffffu, gs, o);
    if (active && (j & (tg - 1)) == 0) xgsum[static_cast<size_t>(m) * (K >> gshift) + grp] = gs;
  }
  if (xsum != nullptr) {
    int cs = static_cast<int>(sum_acc) - (kA8 ? 128 : 8) * kEpt;  // every code carried an offset
    if ((tpr & 31) == 0) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) cs += __shfl_xor_sync(0xffffffffu, cs, o);
      if ((tid & 31) == 0) atomicAdd(&s_sum[rloc], static_cast<unsigned int>(cs));
    } else if ((tpr & (tpr - 1)) == 0) {
      for (int o = tpr >> 1; o > 0; o >>= 1) cs += __shfl_xor_sync(0xffffffffu, cs, o);
      if (j == 0) atomicAdd(&s_sum[rloc], static_cast<unsigned int>(cs));
    } else {
      atomicAdd(&s_sum[rloc], static_cast<unsigned int>(cs));
    }
    __syncthreads();
    if (active && j == 0) xsum[m] = static_cast<int32_t>(s_sum[rloc]);
  }
}

template <typename T, int kLogB, bool kStep, bool kA8>
cudaError_t launch_t(const RotQuantArgs& a) {
  constexpr int kEpt = kLogB >= 12 ? 128 : 64;
  const int tpr = a.K / kEpt;
  int tpb = tpr >= 128 ? tpr : (128 / tpr) * tpr;
  if (tpb / tpr > 32) tpb = 32 * tpr;  // the per-row reduction slots hold 32 rows
  const int rows = tpb / tpr;
  const int grid = (a.M + rows - 1) / rows;
  if (grid == 0) return cudaSuccess;
  const size_t smem = (kLogB > ((kEpt == 128) ? 7 : 6)) ? static_cast<size_t>(tpb) * kEpt * sizeof(float) : 0;
  auto kern = rotate_quant_kernel<T, kLogB, kEpt, kStep, kA8>;
  if (smem > 48 * 1024) {
    // raise the kernel's limit once per device to the most any K asks of it (one kernel serves
    // several K, so several sizes: at most 256 threads x 128 float32 = 128 KB)
    constexpr int kMaxSmem = 128 * 1024;
    if (smem > static_cast<size_t>(kMaxSmem)) return cudaErrorInvalidValue;
    static std::atomic<unsigned long long> raised{0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(raised.load() & bit)) {
      e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kMaxSmem);
      if (e != cudaSuccess) return e;
      raised.fetch_or(bit);
    }
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(tpb);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // may overlap the previous kernel
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, reinterpret_cast<const T*>(a.x), a.M, a.K, a.inv_sqrt_b, a.step_scale,
                                     a.xq, a.xscale, a.xsum, a.mode == 2 ? a.absmax : nullptr, a.out_mode,
                                     a.gshift, a.xgsum, a.zero, a.zero_n);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <typename T, bool kStep, bool kA8>
cudaError_t launch_mode(const RotQuantArgs& a) {
  switch (a.log_b) {
    case 0: return launch_t<T, 0, kStep, kA8>(a);
    case 1: return launch_t<T, 1, kStep, kA8>(a);
    case 2: return launch_t<T, 2, kStep, kA8>(a);
    case 3: return launch_t<T, 3, kStep, kA8>(a);
    case 4: return launch_t<T, 4, kStep, kA8>(a);
    case 5: return launch_t<T, 5, kStep, kA8>(a);
    case 6: return launch_t<T, 6, kStep, kA8>(a);
    case 7: return launch_t<T, 7, kStep, kA8>(a);
    case 8: return launch_t<T, 8, kStep, kA8>(a);
    case 9: return launch_t<T, 9, kStep, kA8>(a);
    case 10: return launch_t<T, 10, kStep, kA8>(a);
    case 11: return launch_t<T, 11, kStep, kA8>(a);
    case 12: return launch_t<T, 12, kStep, kA8>(a);
    default: return cudaErrorInvalidValue;
  }
}

// kA8: the 8-bit instantiations (out_mode 2 or 3), compiled in translation units of their own.
template <typename T, bool kA8>
cudaError_t launch_dtype(const RotQuantArgs& a) {
  return a.mode == 1 ? launch_mode<T, true, kA8>(a) : launch_mode<T, false, kA8>(a);
}

}  // namespace rq
}  // namespace qvla
