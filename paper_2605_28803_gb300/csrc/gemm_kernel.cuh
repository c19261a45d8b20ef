// W4A4 GEMM with the dequantisation epilogue (Sec. 4.2, Eq. 7) on the 5th-generation tensor cores.
//
// acc[m,n] = sum_k qx[m,k] qw[n,k] is an exact integer product.  sm_103a has no integer
// tcgen05 kind, so the codes travel as E4M3: a code q becomes the byte q + 8 (offset binary),
// worth (q + 8) 2^-9 exactly, and tcgen05.mma.kind::f8f6f4 accumulates the products
// (qx + 8)(qw + 8) 2^-18 in FP32 in TMEM.  Every partial sum is an integer multiple of 2^-18
// below 2^6 (K <= 16384), so the FP32 accumulation is exact.  The epilogue removes the offset
// with the code sums:
//   acc = S 2^18 - 8 sum_k qx[m,k] - 8 sum_k qw[n,k] - 64 K
// then y = fma(acc, xscale[m] * wscale[n], bias[n]) rounded once to fp16/bf16.
//
// One persistent CTA per SM.  Warp roles:
//   warps 0-3   epilogue: TMEM -> registers -> dequantise -> global (one accumulator row per thread)
//   warp  4     TMEM allocation; lane 0 issues the MMAs and the commits
//   warp  5     lane 0 issues TMA tensor loads of packed int4 tiles into a staging ring
//   warps 6-13  converters: staged nibbles -> E4M3 bytes in the 128-byte-swizzled K-major
//               layout the MMA descriptors expect
// Shared memory holds kStages staged (packed) and kStages expanded k-blocks of 128 codes; TMEM
// holds two accumulators so the epilogue of one tile overlaps the main loop of the next.  The epilogue stages each tile's
// per-column parameters (weight scale, weight-code correction, bias) in shared memory.
//
// Two orientations: for M > 128 the MMA's M side is the activations (tile 128 tokens x 256
// weight rows); for M <= 128 ("swap") it is the weights (128 weight rows x Mpad tokens),
// so that a small batch does not waste the 128-row MMA.  A small batch has few tiles, so in
// the weight-major orientation a cluster of up to 8 CTAs shares each tile, splitting K: every
// CTA computes an FP32 partial (exact, like the whole sum) and pushes each slice of its rows,
// with asynchronous stores that complete on the receiver's mbarrier, to the CTA owning those
// rows, which sums the slices in its own shared memory and applies the epilogue.  No CTA reads
// another's shared memory, so the cluster needs no barrier around the reduction.
//
// Both kernels of the linear are launched with programmatic stream serialization, so each may
// start (allocate TMEM, initialise barriers, request weights) while the previous kernel of the
// stream finishes; everything that touches the previous kernel's data waits for it first.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstdint>
#include <map>
#include <mutex>
#include <set>
#include <tuple>

#include "griddep.cuh"
#include "kernels.h"
#include "ptx.cuh"
#include "rotate_quant.cuh"

namespace qvla {
namespace {

// Test hook (qvla_debug_hold_gemm_loads): while set, the load warp of a GEMM issues no copy at all,
// so every wait on those copies runs out (see qvla_debug.h).  Per translation unit.
static __device__ int g_debug_hold_loads;

constexpr int kBM = 128;        // MMA M (rows of the MMA A operand)
constexpr int kBK = 128;        // codes per k-block (one 128-byte swizzle row of E4M3)
constexpr int kEpiWarps = 4;
constexpr int kEpiThreads = kEpiWarps * 32;
constexpr int kMmaWarp = 4;
constexpr int kTmaWarp = 5;
constexpr int kConvWarps = 8;
constexpr int kConvThreads = kConvWarps * 32;
constexpr int kThreads = (kEpiWarps + 2 + kConvWarps) * 32;
constexpr uint32_t kEpiBarrier = 1;  // named barrier of the epilogue warps

// kStageA / kStageB: whether operand A / B of the MMA arrives packed (staged, then expanded by
// the converters); otherwise it arrives as operand bytes straight from a swizzled TMA load.
// kPlanes: operand-byte planes per k-block of the activations (2 for 8-bit codes: the high and
// the low nibbles, each one 128-byte tile against the same weight tile).
// kRecv: bytes after the rings where the weight-major split-K reduction receives the partials
// of the cluster's CTAs.
// kExtra: bytes after the receive area (the fused prologue's staging and operand tile);
// kBInStage: operand B lives in the stages (false: the fused prologue's tile holds it).
template <int kBN, bool kStageA = true, bool kStageB = true, int kPlanes = 1, int kRecv = 0, int kExtra = 0,
          bool kBInStage = true>
struct Cfg {
  static constexpr int kTileA1 = kBM * kBK;   // bytes of E4M3 of one plane
  static constexpr int kTileB1 = kBN * kBK;
  static constexpr int kTileA = kTileA1 * (kStageA ? 1 : kPlanes);
  static constexpr int kTileB = kBInStage ? kTileB1 * (kStageB ? 1 : kPlanes) : 0;
  static constexpr int kStage = kTileA + kTileB;             // expanded k-block
  static constexpr int kRawA = kStageA ? kBM * kBK / 2 : 0;  // packed k-block (64-byte rows)
  static constexpr int kRawB = kStageB ? kBN * kBK / 2 : 0;
  static constexpr int kRaw = kRawA + kRawB;
  static constexpr int kStagesRaw = (216 * 1024 - kRecv - kExtra) / (kStage + kRaw);
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kRecvOff = kStages * (kStage + kRaw);
  static constexpr int kExtraOff = kRecvOff + kRecv;
  static constexpr int kSmem = kExtraOff + kExtra + 1024;  // + alignment slack
  static constexpr uint32_t kTmemCols = (2 * kBN) <= 32 ? 32 : (2 * kBN) <= 64 ? 64 : (2 * kBN) <= 128 ? 128 : (2 * kBN) <= 256 ? 256 : 512;
  static_assert(kStages >= 2, "stages");
  static_assert(kRaw % 1024 == 0 && kStage % 1024 == 0, "1024-byte aligned stages");
};

struct Params {
  // The MMA operands: the weights (A when swapped, else B) in the layer's tiled layout, one
  // contiguous 8 KB chunk per 128 rows x k-block ([rows/128][K/128][128][64 B]); the
  // activations through a tensor map.
  const uint8_t* a;
  const uint8_t* b;
  int rows_a, rows_b, K;
  const float* xscale;
  const int32_t* xsum;
  const float* wscale;  // [N]
  const float* wcorr;   // [N] 8 * sum_k qw[n,k]
  const float* bias;    // [N] (zeros when the layer has none)
  void* y;
  int32_t* acc;
  int M, N;      // N = weight rows of the layer (2H for a gated layer)
  int ldy;       // row length of y (N, or H for a gated layer)
  int splits;    // weight-major orientation: CTAs of a cluster splitting K (1 = no split)
  // token-major, non-gated: each tile's k-blocks in `parts` work units (1 = whole tiles), each
  // unit's FP32 partial in part_ws [tile][part][CTA of the pair][kBN / 4][kBM] (float4 elements);
  // part_cnt [tile][CTA of the pair] counts the finished units (zero at launch; the tile's last
  // unit adds the partials to its own, applies the epilogue and resets the count)
  int parts;
  float* part_ws;
  int* part_cnt;
  float kconst;  // the zero-point constant of the accumulator: 64 K (int4 codes), 1024 K (int8)
  // per-group step scales (kGroup): the step's scales [ngroups], each group's code sums of the
  // activations [M][ngroups] and 8 x of the weights [N][ngroups], k-blocks per group, 64 x
  // the group's channels
  const float* gscale;
  const int32_t* xgsum;
  const float* wgcorr;
  int gkb, ngroups;
  float gconst;
  // fused prologue (kX == 3): the raw activations [M][K], the Hadamard block and its scale;
  // xscale then points at the step's scale (one float)
  const void* x;
  int log_b;
  float inv_sqrt_b;
};

__device__ __forceinline__ void epi_sync() {
  asm volatile("bar.sync %0, %1;" ::"n"(kEpiBarrier), "n"(kEpiThreads) : "memory");
}

// Expand one 16-byte chunk (32 codes) into 32 E4M3 bytes at row + the two swizzled 16-byte
// columns o0 and o1 of a 128-byte-swizzled tile row.  The byte order inside each group of 8
// codes becomes (0,2,4,6,1,3,5,7); both operands get the same order, so the dot product over
// k is unchanged.
__device__ __forceinline__ void store_chunk(uint8_t* row, int o0, int o1, uint4 v) {
  uint32_t o[8];
  int4x8_to_e4m3_offset(v.x, o[0], o[1]);
  int4x8_to_e4m3_offset(v.y, o[2], o[3]);
  int4x8_to_e4m3_offset(v.z, o[4], o[5]);
  int4x8_to_e4m3_offset(v.w, o[6], o[7]);
  *reinterpret_cast<uint4*>(row + o0) = make_uint4(o[0], o[1], o[2], o[3]);
  *reinterpret_cast<uint4*>(row + o1) = make_uint4(o[4], o[5], o[6], o[7]);
}

// GELU, tanh form, written as g * sigmoid(2u) = g / (1 + exp(-2u)), u = sqrt(2/pi) (g + 0.044715 g^3):
// the same function as 0.5 g (1 + tanh(u)) without the cancellation of 1 + tanh near u -> -inf.
__device__ __forceinline__ float gelu_tanh(float g) {
  const float u = 0.7978845608028654f * g * fmaf(0.044715f, g * g, 1.0f);
  return __fdividef(g, 1.0f + __expf(-2.0f * u));
}

// Two floats rounded to the output dtype (one pair conversion), as raw bits.
template <typename OutT>
__device__ __forceinline__ uint32_t pack2(float a, float b);
template <>
__device__ __forceinline__ uint32_t pack2<__half>(float a, float b) {
  __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
template <>
__device__ __forceinline__ uint32_t pack2<__nv_bfloat16>(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
// The two values of a pair, back to float.
template <typename OutT>
__device__ __forceinline__ float2 unpack2(uint32_t v);
template <>
__device__ __forceinline__ float2 unpack2<__half>(uint32_t v) {
  return __half22float2(*reinterpret_cast<__half2*>(&v));
}
template <>
__device__ __forceinline__ float2 unpack2<__nv_bfloat16>(uint32_t v) {
  return make_float2(__uint_as_float(v << 16), __uint_as_float(v & 0xFFFF0000u));
}
template <typename OutT>
__device__ __forceinline__ OutT to_out(float v);
template <>
__device__ __forceinline__ __half to_out<__half>(float v) { return __float2half_rn(v); }
template <>
__device__ __forceinline__ __nv_bfloat16 to_out<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

// 32 outputs (16 packed pairs) of one row: 4 x 16-byte stores, or element stores at a ragged edge.
template <typename OutT>
__device__ __forceinline__ void store_row32(OutT* dst, const uint32_t (&pk)[16], int nvalid) {
  if (nvalid == 32) {
    uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
  } else {
    uint16_t* d = reinterpret_cast<uint16_t*>(dst);
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (i < nvalid) d[i] = static_cast<uint16_t>(pk[i >> 1] >> (16 * (i & 1)));
  }
}

// Epilogue parameters of 4 consecutive weight rows n .. n + 3 and one token m (split-K reduction);
// indices past the end are clamped so the loads can be issued unconditionally.
struct SplitParams {
  float cm, xs;       // kconst + 8 xsum[m], xscale[m]
  float4 wc, ws, bs;  // wcorr, wscale, bias of rows n .. n + 3
  template <bool kGroup, bool kFused = false>
  __device__ __forceinline__ void load(const Params& p, int n, int m) {
    n = min(n, p.N - 4);
    m = min(m, p.M - 1);
    if constexpr (kFused) {  // the activation code sums are already out of the partials
      cm = p.kconst;
      xs = __ldg(p.xscale);
      wc = __ldg(reinterpret_cast<const float4*>(p.wcorr + n));
    } else if constexpr (!kGroup) {  // grouped partials arrive scaled and corrected
      cm = p.kconst + 8.0f * static_cast<float>(__ldg(p.xsum + m));
      xs = __ldg(p.xscale + m);
      wc = __ldg(reinterpret_cast<const float4*>(p.wcorr + n));
    } else {
      cm = xs = 0.0f;
      wc = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
    }
    ws = __ldg(reinterpret_cast<const float4*>(p.wscale + n));
    bs = __ldg(reinterpret_cast<const float4*>(p.bias + n));
  }
};

// ---- fused rotate + quantise prologue (kX == 3: the weight-major GEMM reads raw activations) ----
// For a small batch with a per-step scale (no reduction along the row), every CTA of a split-K
// cluster rotates and quantises its own share of the token rows, over whole rows, and hands each
// CTA of the cluster the operand bytes of that CTA's k-range.  A warp task is one row and one
// chunk of C = 32 kE output channels, kE consecutive ones per lane:
//   b <= C: the chunk holds whole Hadamard blocks of the input chunk;
//   b >  C: chunk c of its block B is (sum_a (-1)^popcount(a & j) x_a) . H_C, x_a the a-th C-wide
//           piece of block B and j the chunk's index in it (Sylvester H_b = H_{b/C} (x) H_C).
// Butterflies run on the lane's own bits in registers, then across lanes by shuffles; the codes
// are those of the separate rotate + quantise kernel (fast path, exact decision near a tie).
constexpr int kFuseStagingMax = 48 * 1024;  // staged operand bytes of this CTA's rows (rows x K)
constexpr int kFuseXBMax = 32 * 1024;       // the operand tile of this CTA's k-range (k-blocks x BN x 128)
constexpr int kFuseExtra = kFuseStagingMax + kFuseXBMax;
constexpr int kProWarps = kEpiWarps + kConvWarps;  // warps that run the prologue
constexpr int kProThreads = kProWarps * 32;
constexpr uint32_t kProBarrier = 2;                // named barrier of the prologue warps

__device__ __forceinline__ void pro_sync() {
  asm volatile("bar.sync %0, %1;" ::"n"(kProBarrier), "n"(kProThreads) : "memory");
}

// One warp task.  x: [M][K] activations; row m; output chunk c (channels [c C, c C + C));
// cr = (1/sqrt(b)) / delta and delta the step scale; staging: this CTA's staged bytes, laid out
// [destination CTA][its k-block][row - m0][128 B, 128-byte swizzled by row & 7] for CTA k-ranges
// of w channels and `rows` staged rows.
template <typename XT, int kE>
__device__ __forceinline__ void fuse_task(const XT* __restrict__ x, int K, int log_b, float inv_sqrt_b, float delta,
                                          float cr, int m, int c, int lane, uint8_t* staging, int m0, int rows, int w) {
  constexpr int kN = kE / 2;         // float2 per lane
  constexpr int kLogE = kE == 64 ? 6 : kE == 32 ? 5 : 4;
  constexpr int kC = 32 * kE;        // channels per task
  constexpr int kPer16 = 16 / static_cast<int>(sizeof(XT));
  static_assert((1 << kLogE) == kE, "elements per lane");
  const int b = 1 << log_b;
  float2 v[kN];
  const XT* row = x + static_cast<size_t>(m) * K;
  if (b <= kC) {
    const XT* src = row + c * kC + lane * kE;
#pragma unroll
    for (int q = 0; q < kE / kPer16; ++q) rq::Loader<XT>::load(src + q * kPer16, v + q * (kPer16 / 2));
  } else {
    // the signed sum of the b / C pieces of the block (the Hadamard stages on the high bits)
    const int blk0 = (c * kC) & ~(b - 1);
    const int jc = (c * kC - blk0) / kC;
#pragma unroll
    for (int i = 0; i < kN; ++i) v[i] = make_float2(0.0f, 0.0f);
    for (int a = 0; a < b / kC; ++a) {
      const float sg = (__popc(a & jc) & 1) ? -1.0f : 1.0f;
      const float2 sg2 = make_float2(sg, sg);
      const XT* src = row + blk0 + a * kC + lane * kE;
#pragma unroll
      for (int q = 0; q < kE / kPer16; ++q) {
        float2 t[kPer16 / 2];
        rq::Loader<XT>::load(src + q * kPer16, t);
#pragma unroll
        for (int i = 0; i < kPer16 / 2; ++i) v[q * (kPer16 / 2) + i] = __ffma2_rn(t[i], sg2, v[q * (kPer16 / 2) + i]);
      }
    }
  }
  // butterflies on the lane's own index bits (bit 0 is the pair's own lane)
  const int nreg = log_b < kLogE ? log_b : kLogE;
  if (nreg > 0) {
#pragma unroll
    for (int i = 0; i < kN; ++i) {
      const float a0 = v[i].x, c0 = v[i].y;
      v[i] = make_float2(a0 + c0, a0 - c0);
    }
  }
#pragma unroll
  for (int bit = 1; bit < kLogE; ++bit) {
    if (bit < nreg) {
      const int h = 1 << (bit - 1);
#pragma unroll
      for (int i = 0; i < kN; ++i)
        if ((i & h) == 0) rq::bfly2(v[i], v[i + h]);
    }
  }
  // butterflies across lanes: the lower lane of a pair keeps a + c, the upper one a - c
  const int nlane = (log_b < kLogE + 5 ? log_b : kLogE + 5) - kLogE;
  for (int lb = 0; lb < nlane; ++lb) {
    const int mask = 1 << lb;
    const float sgn = (lane & mask) ? -1.0f : 1.0f;
    const float2 sg2 = make_float2(sgn, sgn);
#pragma unroll
    for (int i = 0; i < kN; ++i) {
      float2 pv;
      pv.x = __shfl_xor_sync(0xffffffffu, v[i].x, mask);
      pv.y = __shfl_xor_sync(0xffffffffu, v[i].y, mask);
      v[i] = __ffma2_rn(v[i], sg2, pv);
    }
  }
  // codes, as in the separate kernel's per-step path
  const bool zero_scale = !(delta > 0.0f);
  const float rcp = zero_scale ? 0.0f : __fdiv_rn(1.0f, delta);
  const bool tiny_scale = !zero_scale && isinf(rcp);
  const float2 cr2 = make_float2(cr, cr);
  const float2 magic2 = make_float2(rq::kMagic, rq::kMagic), nmagic2 = make_float2(-rq::kMagic, -rq::kMagic);
  const float2 neg2 = make_float2(-1.0f, -1.0f);
  const int ch0 = c * kC + lane * kE;  // this lane's first output channel
  const int r = m - m0;
#pragma unroll
  for (int g2 = 0; g2 < kE / 16; ++g2) {  // 16 channels = one 16-byte operand chunk
    uint32_t o[4];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int g = 2 * g2 + h;  // group of 8 channels
      float2 u[4];
      float dev = 0.0f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float2 t = __fmul2_rn(v[4 * g + i], cr2);
        t.x = fminf(fmaxf(t.x, -7.0f), 7.0f);
        t.y = fminf(fmaxf(t.y, -7.0f), 7.0f);
        u[i] = __fadd2_rn(t, magic2);
        const float2 d = __ffma2_rn(__fadd2_rn(u[i], nmagic2), neg2, t);
        dev = fmaxf(dev, fmaxf(fabsf(d.x), fabsf(d.y)));
      }
      if (dev >= rq::kTieBand || tiny_scale) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          u[i].x = rq::exact_code(v[4 * g + i].x, inv_sqrt_b, delta, cr, 7.0f, rq::kTieBand);
          u[i].y = rq::exact_code(v[4 * g + i].y, inv_sqrt_b, delta, cr, 7.0f, rq::kTieBand);
        }
      }
      // operand bytes q + 8 in the order k0 k2 k4 k6 k1 k3 k5 k7 of the group
      o[2 * h] = (rq::low_bytes(u[0].x, u[1].x, u[2].x, u[3].x) & 0x0F0F0F0Fu) ^ 0x08080808u;
      o[2 * h + 1] = (rq::low_bytes(u[0].y, u[1].y, u[2].y, u[3].y) & 0x0F0F0F0Fu) ^ 0x08080808u;
    }
    const int ch = ch0 + 16 * g2;
    const int d = ch / w, kb = (ch % w) / kBK, q16 = (ch % kBK) >> 4;
    uint8_t* dst = staging + ((d * (w / kBK) + kb) * rows + r) * 128 + ((q16 ^ (m & 7)) << 4);
    *reinterpret_cast<uint4*>(dst) = make_uint4(o[0], o[1], o[2], o[3]);
  }
}

// kX: how the activations arrive.  0: packed int4, staged and expanded like the weights.
// 1: operand bytes ([rows][K], written by the rotate-quantise kernel), TMA-loaded with the
// 128-byte swizzle straight into the MMA operand tile; only the weights are staged and
// expanded.  2: the two operand planes of 8-bit codes ([rows][2K]: per k-block the high then
// the low nibbles), both loaded per k-block and multiplied with the same expanded weight tile.
// kGroup: per-step, per-group activation scales.  Each group's k-blocks accumulate into a fresh
// TMEM buffer; the epilogue removes that group's zero point exactly, scales by the group's
// Delta and adds the result into a running FP32 sum held in TMEM beside the two buffers.
// kPair: token-major on a CTA pair (cluster of 2): one 2-SM MMA (cta_group::2, M = 256) per
// step covers 256 tokens x kBN weight rows; each CTA stages its 128 token rows and half of the
// weight rows and receives its 128 rows of the accumulator in its own TMEM.  The leader (rank 0)
// issues the MMAs; operand-byte activation tiles of both CTAs complete on the leader's barrier
// directly, and one peer thread forwards the completion of each stage by the peer's converters
// (its half of the weight rows, and with packed activations its token rows too).
// kX 3 (fused): weight-major only; the activations arrive raw ([M][K] of XT) and the CTAs of the
// split-K cluster rotate and quantise them in a prologue (fuse_task), kFuseE channels per lane.
template <int kBN, bool kSwap, bool kGated, int kX, typename OutT, bool kGroup = false, bool kPair = false,
          int kFuseE = 32, typename XT = __half>
__global__ void __launch_bounds__(kThreads, 1) gemm_w4a4_kernel(const __grid_constant__ CUtensorMap tmap_a,
                                                                 const __grid_constant__ CUtensorMap tmap_b, Params p) {
  constexpr bool kFused = kX == 3;
  constexpr bool kXBytes = kX == 1 || kX == 2;
  constexpr int kPlanes = kX == 2 ? 2 : 1;
  constexpr bool kStageA = !(kXBytes && !kSwap);  // operand A is the activations unless swapped
  constexpr bool kStageB = !(kXBytes && kSwap) && !kFused;
  static_assert(!kPair || (!kSwap && !kGroup && kX <= 1), "pairs: token-major, int4 activations");
  static_assert(!kFused || (kSwap && !kGated && !kGroup), "the fused prologue: weight-major, per-step scale");
  constexpr int kBS = kPair ? kBN / 2 : kBN;  // weight rows this CTA stages
  using C = Cfg<kBS, kStageA, kStageB, kPlanes, kSwap ? kBM * kBN * 4 : 0, kFused ? kFuseExtra : 0, !kFused>;
  static_assert(kSwap || kBN % 128 == 0, "a weight tile is whole 128-row chunks");
  static_assert(!kGroup || (kBN <= 128 && !kGated && kX == 1), "grouped scales: int4 operand bytes, BN <= 128");
  // TMEM columns: two accumulators, plus the running sum of the grouped mode
  constexpr uint32_t kTmemCols = kPair ? (2 * kBN <= 256 ? 256 : 512)
                                       : !kGroup ? C::kTmemCols : (3 * kBN <= 64 ? 64 : 3 * kBN <= 128 ? 128 : 3 * kBN <= 256 ? 256 : 512);
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~uintptr_t(1023));

  __shared__ __align__(8) uint64_t bar_raw_full[C::kStages];   // TMA bytes landed
  __shared__ __align__(8) uint64_t bar_raw_empty[C::kStages];  // converters done with the staged k-block
  __shared__ __align__(8) uint64_t bar_full[C::kStages];       // expanded k-block ready for the MMA
  __shared__ __align__(8) uint64_t bar_empty[C::kStages];      // MMAs done reading it
  __shared__ __align__(8) uint64_t bar_tfull[2];
  __shared__ __align__(8) uint64_t bar_tempty[2];
  __shared__ __align__(8) uint64_t bar_done;
  __shared__ __align__(8) uint64_t bar_recv;  // split-K: every CTA's slice of this CTA's rows has landed
  __shared__ __align__(8) uint64_t bar_xready;  // fused: this CTA's operand tile is complete
  __shared__ int s_xs[kFused ? kBN : 1];        // fused: code sums of each token over this CTA's k-range
  __shared__ uint32_t s_tmem_base;
  __shared__ int s_epi_abort;  // set by an epilogue thread whose wait timed out
  __shared__ int s_last;       // split of K: this unit was its tile's last to finish
  // per-column parameters of the current tile (non-swap): weight scale, code correction, bias
  __shared__ __align__(16) float s_ws[kSwap ? 1 : kBN];
  __shared__ __align__(16) float s_wc[kSwap ? 1 : kBN];
  __shared__ __align__(16) float s_bs[kSwap ? 1 : kBN];

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  const int tiles_a = (p.rows_a + (kPair ? 2 : 1) * kBM - 1) / ((kPair ? 2 : 1) * kBM);
  const int tiles_b = (p.rows_b + kBN - 1) / kBN;
  const int ntiles = tiles_a * tiles_b;
  const int nkb_all = p.K / kBK;
  const int parts = p.parts;
  const int nunits = ntiles * parts;
  // split-K (weight-major orientation): the `splits` CTAs of a cluster share one tile, CTA r
  // taking k-blocks [kb0, kb1); without a split every CTA runs whole tiles persistently
  const int splits = kSwap ? p.splits : 1;
  const uint32_t krank = (kSwap && splits > 1) ? cluster_ctarank() : 0u;
  const uint32_t prank = kPair ? cluster_ctarank() : 0u;  // 0: the pair's leader, which issues the MMAs
  const int udiv = kPair ? 2 : splits;                      // CTAs per work unit
  // (grouped scales: the split falls on group boundaries, so each group's partial is whole)
  const int kb0 = kGroup ? ((p.ngroups * static_cast<int>(krank)) / splits) * p.gkb
                         : (nkb_all * static_cast<int>(krank)) / splits;
  const int kb1 = kGroup ? ((p.ngroups * (static_cast<int>(krank) + 1)) / splits) * p.gkb
                         : (nkb_all * (static_cast<int>(krank) + 1)) / splits;
  // this CTA's first tile and the tile stride, read where they are used (held in registers
  // across the role loops they would cost a register in every role)
#define QVLA_UNIT0 (blockIdx.x / static_cast<unsigned>(udiv))
#define QVLA_NUNITS (gridDim.x / static_cast<unsigned>(udiv))
  // work unit u: tile u / parts, k-blocks [ka, kz) of this CTA's range (all of it when parts = 1)
  auto unit_range = [&](int u, int& tile, int& ka, int& kz) {
    tile = u / parts;
    const int part = u - tile * parts;
    ka = kb0 + (kb1 - kb0) * part / parts;
    kz = kb0 + (kb1 - kb0) * (part + 1) / parts;
  };
  uint8_t* const raw = smem + C::kStages * C::kStage;  // staging ring after the expanded stages

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&bar_raw_full[s]), 1);
      mbar_init(smem_u32(&bar_raw_empty[s]), kConvThreads);
      // + the TMA thread's byte count; a pair's leader also counts the peer's forwarder, while the
      // peer's own barrier counts its converters only
      mbar_init(smem_u32(&bar_full[s]), kPair && prank != 0 ? kConvThreads
                                                            : kConvThreads + (kXBytes ? 1 : 0) + (kPair ? 1 : 0));
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&bar_tfull[i]), 1);
      mbar_init(smem_u32(&bar_tempty[i]), kEpiThreads + (kPair ? kEpiWarps : 0));
    }
    mbar_init(smem_u32(&bar_done), 1);
    mbar_init(smem_u32(&bar_recv), 1);
    // fused: the expected operand bytes (thread 0), and every prologue thread once its own
    // stores to the tile are done
    mbar_init(smem_u32(&bar_xready), 1 + (kFused ? kProThreads : 0));
    mbar_init_fence();
    s_epi_abort = 0;
  }
  if (warp == kMmaWarp) {
    if constexpr (kPair) {
      tmem_alloc_pair<kTmemCols>(smem_u32(&s_tmem_base));
    } else {
      tmem_alloc<kTmemCols>(smem_u32(&s_tmem_base));
    }
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (kPair) cluster_sync();  // both CTAs' barriers exist before any arrival crosses the pair
  tc_fence_after();
  const uint32_t tmem_base = s_tmem_base;
  if constexpr (kFused) {
    // every CTA of the cluster sends this one its k-range of every token row
    if (threadIdx.x == 0)
      mbar_arrive_expect_tx(smem_u32(&bar_xready), static_cast<uint32_t>(p.M * (kb1 - kb0) * kBK));
  }
  // split-K: the token columns of this cluster's tile that hold tokens (only those are exchanged)
  const int split_cols = kSwap ? max(0, min(kBN, p.rows_b - static_cast<int>(QVLA_UNIT0 / static_cast<unsigned>(tiles_a)) * kBN))
                               : kBN;
  if (kSwap && splits > 1) {
    // split-K: this CTA receives one slice of its rows from every CTA of the cluster; the
    // cluster barrier completed before the first send guarantees every receiver's barrier exists
    if (threadIdx.x == 0) mbar_arrive_expect_tx(smem_u32(&bar_recv), static_cast<uint32_t>(kBM * split_cols * 4));
    if constexpr (kFused) {
      cluster_sync();  // the prologue sends early: every barrier of the cluster exists from here on
    } else {
      cluster_arrive_relaxed();
    }
  }
  if (threadIdx.x == 0) griddep_launch_dependents();

  // fused (kX 3): the prologue of prologue warp pw (the epilogue warps, then the converters once
  // their k-blocks are expanded).  This CTA rotates and quantises token rows [m0, m0 + rows),
  // stages their operand bytes, and copies to each CTA of the cluster its k-range of them.
  uint8_t* const fuse_staging = smem + C::kExtraOff;
  uint8_t* const fuse_xb = fuse_staging + kFuseStagingMax;  // this CTA's operand tile [k-block][BN][128]
  auto fused_prologue = [&](int pw) {
    if constexpr (kFused) {
      griddep_wait();  // the activations come from the previous kernel
      const int rows_per = (p.M + splits - 1) / splits;
      const int m0 = min(p.M, static_cast<int>(krank) * rows_per);
      const int rows = min(p.M, m0 + rows_per) - m0;
      const int nkbw = kb1 - kb0;
      const int w = nkbw * kBK;
      const float delta = __ldg(p.xscale);
      const float cr = p.inv_sqrt_b * (delta > 0.0f ? __fdiv_rn(1.0f, delta) : 0.0f);
      constexpr int kCh = 32 * kFuseE;
      const int chunks = p.K / kCh;
      const XT* xin = static_cast<const XT*>(p.x);
      for (int t = pw; t < rows * chunks; t += kProWarps)
        fuse_task<XT, kFuseE>(xin, p.K, p.log_b, p.inv_sqrt_b, delta, cr, m0 + t / chunks, t % chunks, lane, fuse_staging,
                              m0, rows, w);
      // padding rows M .. BN - 1 of this CTA's tile: zero bytes (their outputs are never stored)
      const int pad16 = (kBN - p.M) * (kBK / 16);
      for (int i = pw * 32 + lane; i < pad16 * nkbw; i += kProThreads)
        *reinterpret_cast<uint4*>(fuse_xb + (i / pad16) * (kBN * kBK) + p.M * kBK + (i % pad16) * 16) =
            make_uint4(0u, 0u, 0u, 0u);
      fence_proxy_async_smem();  // the staged bytes are read, and the tile is multiplied, by the async proxy
      mbar_arrive(smem_u32(&bar_xready));
      pro_sync();
      if (pw == 0 && rows > 0 && lane < splits * nkbw) {
        const int d = lane / nkbw, kb = lane % nkbw;
        const uint32_t dst = smem_u32(fuse_xb + kb * (kBN * kBK) + m0 * kBK);
        const uint32_t bar = smem_u32(&bar_xready);
        bulk_copy_s2c(splits > 1 ? mapa_shared(dst, static_cast<uint32_t>(d)) : dst,
                      smem_u32(fuse_staging + (d * nkbw + kb) * rows * kBK), static_cast<uint32_t>(rows * kBK),
                      splits > 1 ? mapa_shared(bar, static_cast<uint32_t>(d)) : bar);
        bulk_commit();
      }
    }
  };

  if (warp == kTmaWarp) {
    // ------------------------------------------------------------------ TMA loads of packed tiles
    if (lane == 0) {
      if constexpr (!kFused) tma_prefetch_desc(kSwap ? &tmap_b : &tmap_a);  // the activations' map (the weights need none)
      // Weight-major orientation with operand-byte activations: the staging ring holds weights
      // only, which no earlier kernel writes, so the first stages are requested before waiting
      // for the previous kernel (a small batch's GEMM is mostly this latency).
      int pre = 0;
      const bool hold = *const_cast<volatile int*>(&g_debug_hold_loads) != 0;  // test hook: issue nothing
      if constexpr ((kXBytes || kFused) && kSwap) {
        const int unit0 = static_cast<int>(QVLA_UNIT0);
        if (unit0 < ntiles && !hold) {
          const int ta = unit0 % tiles_a;
          pre = min(C::kStages, kb1 - kb0);
          for (int i = 0; i < pre; ++i) {
            const uint32_t bar = smem_u32(&bar_raw_full[i]);
            mbar_arrive_expect_tx(bar, C::kRaw);
            bulk_load(smem_u32(raw + i * C::kRaw), p.a + (static_cast<size_t>(ta) * nkb_all + kb0 + i) * 8192, 8192, bar);
          }
        }
      }
      griddep_wait();
      int it = 0;
      bool ok = !hold;
      for (int u = QVLA_UNIT0; u < nunits && ok; u += QVLA_NUNITS) {
        int tile, ka, kz;
        unit_range(u, tile, ka, kz);
        const int ta = tile % tiles_a, tb = tile / tiles_a;
        for (int kb = ka; kb < kz; ++kb, ++it) {
          const int s = it % C::kStages;
          const uint32_t ph = static_cast<uint32_t>(it / C::kStages) & 1u;
          if (it >= pre) {
            if (!mbar_wait(smem_u32(&bar_raw_empty[s]), ph ^ 1u)) { ok = false; break; }
            const uint32_t bar = smem_u32(&bar_raw_full[s]);
            mbar_arrive_expect_tx(bar, C::kRaw);
            const uint32_t dst = smem_u32(raw + s * C::kRaw);
            if constexpr (kStageA) {
              if constexpr (kSwap) {
                bulk_load(dst, p.a + (static_cast<size_t>(ta) * nkb_all + kb) * 8192, 8192, bar);
              } else {
                tma_load_2d(dst, &tmap_a, kb * (kBK / 2), kPair ? ta * 2 * kBM + static_cast<int>(prank) * kBM : ta * kBM, bar);
              }
            }
            if constexpr (kStageB) {
              if constexpr (kPair) {
                // this CTA's half of the weight tile: chunk 2 tb + rank (kBN 256), or half of chunk tb
                if constexpr (kBN == 256) {
                  bulk_load(dst + C::kRawA, p.b + (static_cast<size_t>(tb * 2 + prank) * nkb_all + kb) * 8192, 8192, bar);
                } else {
                  bulk_load(dst + C::kRawA, p.b + (static_cast<size_t>(tb) * nkb_all + kb) * 8192 + prank * 4096, 4096, bar);
                }
              } else if constexpr (!kSwap) {
#pragma unroll
                for (int c = 0; c < kBN / 128; ++c)
                  bulk_load(dst + C::kRawA + c * 8192,
                            p.b + (static_cast<size_t>(tb * (kBN / 128) + c) * nkb_all + kb) * 8192, 8192, bar);
              } else {
                tma_load_2d(dst + C::kRawA, &tmap_b, kb * (kBK / 2), tb * kBN, bar);
              }
            }
          }
          if constexpr (kXBytes) {
            // the activation operand goes straight into the expanded stage once the MMAs are done with it
            if (!mbar_wait(smem_u32(&bar_empty[s]), ph ^ 1u)) { ok = false; break; }
            const uint32_t fb = smem_u32(&bar_full[s]);
            const uint32_t e = smem_u32(smem + s * C::kStage);
            if constexpr (kPair) {
              // both CTAs' activation rows complete on the leader's barrier
              if (prank == 0) mbar_arrive_expect_tx(fb, 2 * C::kTileA);
              tma_load_2d_pair(e, &tmap_a, kb * kBK, ta * 2 * kBM + static_cast<int>(prank) * kBM, mapa_shared(fb, 0));
            } else if constexpr (!kSwap) {
              mbar_arrive_expect_tx(fb, C::kTileA);
#pragma unroll
              for (int pl = 0; pl < kPlanes; ++pl)
                tma_load_2d(e + pl * C::kTileA1, &tmap_a, (kb * kPlanes + pl) * kBK, ta * kBM, fb);
            } else {
              mbar_arrive_expect_tx(fb, C::kTileB);
#pragma unroll
              for (int pl = 0; pl < kPlanes; ++pl)
                tma_load_2d(e + C::kTileA + pl * C::kTileB1, &tmap_b, (kb * kPlanes + pl) * kBK, tb * kBN, fb);
            }
          }
        }
      }
      // before leaving, let every load issued above land (a no-op unless a wait timed out)
      for (int k = 0; k < C::kStages && k < it; ++k) {
        const int j = it - 1 - k;
        mbar_wait(smem_u32(&bar_raw_full[j % C::kStages]), static_cast<uint32_t>(j / C::kStages) & 1u);
      }
    }
    __syncwarp();
  } else if (warp > kTmaWarp) {
    // ------------------------------------------------------------------ converters
    const int ct = threadIdx.x - (kTmaWarp + 1) * 32;  // 0 .. kConvThreads-1
    constexpr int kChunksA = kStageA ? kBM * 4 : 0;     // 16-byte packed chunks per k-block
    constexpr int kChunks = kChunksA + (kStageB ? kBS * 4 : 0);
    constexpr int kPer = (kChunks + kConvThreads - 1) / kConvThreads;
    // destination of each of this thread's chunks: tile byte offset of the row and the two
    // swizzled 16-byte columns; the staged chunk c sits at byte 16 c of the staging k-block
    int d_row[kPer], d_o0[kPer], d_o1[kPer];
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int c = ct + i * kConvThreads;
      const int cc = c < kChunksA ? c : c - kChunksA;
      const int r = cc >> 2, q = cc & 3;
      d_row[i] = (c < kChunksA ? 0 : C::kTileA) + r * 128;
      d_o0[i] = ((2 * q) ^ (r & 7)) << 4;
      d_o1[i] = ((2 * q + 1) ^ (r & 7)) << 4;
    }
    int it = 0;
    bool ok = true;
    for (int u = QVLA_UNIT0; u < nunits && ok; u += QVLA_NUNITS) {
      int tile, ka, kz;
      unit_range(u, tile, ka, kz);
      for (int kb = ka; kb < kz; ++kb, ++it) {
        const int s = it % C::kStages;
        const uint32_t ph = static_cast<uint32_t>(it / C::kStages) & 1u;
        if (!mbar_wait(smem_u32(&bar_raw_full[s]), ph)) { ok = false; break; }
        if (!mbar_wait(smem_u32(&bar_empty[s]), ph ^ 1u)) { ok = false; break; }
        const uint8_t* src = raw + s * C::kRaw;
        uint8_t* dst = smem + s * C::kStage;
        uint4 v[kPer];
#pragma unroll
        for (int i = 0; i < kPer; ++i)
          if (kChunks % kConvThreads == 0 || ct + i * kConvThreads < kChunks)
            v[i] = *reinterpret_cast<const uint4*>(src + 16 * (ct + i * kConvThreads));
#pragma unroll
        for (int i = 0; i < kPer; ++i)
          if (kChunks % kConvThreads == 0 || ct + i * kConvThreads < kChunks)
            store_chunk(dst + d_row[i], d_o0[i], d_o1[i], v[i]);
        // The staged k-block is released only now: the conversions above consumed every loaded
        // value, so the loads have completed, and the proxy fence orders them (and the stores)
        // before the async proxy's next accesses, the TMA's refill of the staging stage and the
        // MMAs' reads of the expanded one.  Releasing it straight after issuing the loads let
        // a refill overwrite the stage under loads still in flight (measured: the MMA of k-block
        // j then used some rows of k-block j + kStages).
        fence_proxy_async_smem();
        mbar_arrive(smem_u32(&bar_raw_empty[s]));
        mbar_arrive(smem_u32(&bar_full[s]));
      }
    }
    if constexpr (kFused) fused_prologue(kEpiWarps + (warp - kTmaWarp - 1));
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------------ MMA issuer
    if (kPair && lane == 0 && prank == 0) {
      constexpr uint32_t kIdesc = idesc_e4m3_f32(2 * kBM, kBN);
      int it = 0, tile_iter = 0;
      bool ok = true;
      for (int u = QVLA_UNIT0; u < nunits && ok; u += QVLA_NUNITS, ++tile_iter) {
        int tile, ka, kz;
        unit_range(u, tile, ka, kz);
        (void)tile;
        const int buf = tile_iter & 1;
        const uint32_t aph = static_cast<uint32_t>(tile_iter >> 1) & 1u;
        if (!mbar_wait(smem_u32(&bar_tempty[buf]), aph ^ 1u)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(buf * kBN);
        for (int kb = ka; kb < kz; ++kb, ++it) {
          const int s = it % C::kStages;
          const uint32_t ph = static_cast<uint32_t>(it / C::kStages) & 1u;
          if (!mbar_wait(smem_u32(&bar_full[s]), ph)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + s * C::kStage);
          const uint32_t sb = sa + C::kTileA;
#pragma unroll
          for (int kk = 0; kk < kBK / 32; ++kk)
            mma_e4m3_pair(d, smem_desc_sw128(sa + kk * 32), smem_desc_sw128(sb + kk * 32), kIdesc,
                          (kb != ka || kk != 0) ? 1u : 0u);
          mma_commit_pair(smem_u32(&bar_empty[s]), 3);  // both CTAs' stage s is free
        }
        if (!ok) break;
        mma_commit_pair(smem_u32(&bar_tfull[buf]), 3);
      }
      mma_commit_pair(smem_u32(&bar_done), 1);
      mbar_wait(smem_u32(&bar_done), 0);
    } else if (kPair && lane == 0) {
      // the peer's forwarder: once this CTA's converters have filled stage s, one arrival tells
      // the leader (the converters themselves arrive locally)
      int it = 0;
      bool ok = true;
      for (int u = QVLA_UNIT0; u < nunits && ok; u += QVLA_NUNITS) {
        int tile, ka, kz;
        unit_range(u, tile, ka, kz);
        (void)tile;
        for (int kb = ka; kb < kz; ++kb, ++it) {
          const int s = it % C::kStages;
          if (!mbar_wait(smem_u32(&bar_full[s]), static_cast<uint32_t>(it / C::kStages) & 1u)) { ok = false; break; }
          mbar_arrive_peer(mapa_shared(smem_u32(&bar_full[s]), 0));
        }
      }
    } else if (kPair) {
      // the other lanes of a pair's MMA warp have no role
    } else if (lane == 0 && kGroup) {
      // one accumulator per scale group, alternating between the two buffers group by group
      constexpr uint32_t kIdesc = idesc_e4m3_f32(kBM, kBN);
      int it = 0, gi = 0;
      bool ok = true;
      const int gkb = p.gkb;
      for (int tile = QVLA_UNIT0; tile < ntiles && ok; tile += QVLA_NUNITS) {
        for (int kg = kb0; kg < kb1; kg += gkb, ++gi) {
          const int buf = gi & 1;
          if (!mbar_wait(smem_u32(&bar_tempty[buf]), (static_cast<uint32_t>(gi >> 1) & 1u) ^ 1u)) { ok = false; break; }
          tc_fence_after();
          const uint32_t d = tmem_base + static_cast<uint32_t>(buf * kBN);
          for (int q = 0; q < gkb; ++q, ++it) {
            const int s = it % C::kStages;
            const uint32_t ph = static_cast<uint32_t>(it / C::kStages) & 1u;
            if (!mbar_wait(smem_u32(&bar_full[s]), ph)) { ok = false; break; }
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + s * C::kStage);
            const uint32_t sb = sa + C::kTileA;
#pragma unroll
            for (int kk = 0; kk < kBK / 32; ++kk)
              mma_e4m3(d, smem_desc_sw128(sa + kk * 32), smem_desc_sw128(sb + kk * 32), kIdesc, (q != 0 || kk != 0) ? 1u : 0u);
            mma_commit(smem_u32(&bar_empty[s]));
          }
          if (!ok) break;
          mma_commit(smem_u32(&bar_tfull[buf]));
        }
      }
      mma_commit(smem_u32(&bar_done));
      mbar_wait(smem_u32(&bar_done), 0);
    } else if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_e4m3_f32(kBM, kBN);
      int it = 0, tile_iter = 0;
      bool ok = true;
      for (int u = QVLA_UNIT0; u < nunits && ok; u += QVLA_NUNITS, ++tile_iter) {
        int tile, ka, kz;
        unit_range(u, tile, ka, kz);
        (void)tile;
        const int buf = tile_iter & 1;
        const uint32_t aph = static_cast<uint32_t>(tile_iter >> 1) & 1u;
        if (!mbar_wait(smem_u32(&bar_tempty[buf]), aph ^ 1u)) { ok = false; break; }
        tc_fence_after();
        if constexpr (kFused) {  // the operand tile, from every CTA of the cluster
          if (!mbar_wait_cluster(smem_u32(&bar_xready), 0)) { ok = false; break; }
        }
        const uint32_t d = tmem_base + static_cast<uint32_t>(buf * kBN);
        for (int kb = ka; kb < kz; ++kb, ++it) {
          const int s = it % C::kStages;
          const uint32_t ph = static_cast<uint32_t>(it / C::kStages) & 1u;
          if (!mbar_wait(smem_u32(&bar_full[s]), ph)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + s * C::kStage);
          const uint32_t sb = kFused ? smem_u32(fuse_xb + (kb - kb0) * (kBN * kBK)) : sa + C::kTileA;
#pragma unroll
          for (int pl = 0; pl < kPlanes; ++pl) {
            // plane pl of the activations against the same weight tile
            const uint32_t pa = sa + (kStageA ? 0 : pl * C::kTileA1);
            const uint32_t pb = sb + (kStageB ? 0 : pl * C::kTileB1);
#pragma unroll
            for (int kk = 0; kk < kBK / 32; ++kk) {
              mma_e4m3(d, smem_desc_sw128(pa + kk * 32), smem_desc_sw128(pb + kk * 32), kIdesc,
                       (kb != ka || pl != 0 || kk != 0) ? 1u : 0u);
            }
          }
          mma_commit(smem_u32(&bar_empty[s]));
        }
        if (!ok) break;
        mma_commit(smem_u32(&bar_tfull[buf]));
      }
      // every MMA issued above has completed once this barrier flips
      mma_commit(smem_u32(&bar_done));
      mbar_wait(smem_u32(&bar_done), 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ epilogue
    const int et = threadIdx.x;  // 0..127 = TMEM lane
    int tile_iter = 0;
    const float k64 = p.kconst;
    griddep_wait();  // xscale / xsum come from the previous kernel, and y may still be read by it
    if constexpr (kFused) {
      fused_prologue(warp);
      // each token's code sum over this CTA's k-range, from the operand bytes (q + 8 each)
      const bool landed = mbar_wait_cluster(smem_u32(&bar_xready), 0);
      if (et < kBN) {
        unsigned int sum = 0;
        if (landed && et < p.M) {
          for (int kb = 0; kb < kb1 - kb0; ++kb) {
            const uint4* rowp = reinterpret_cast<const uint4*>(fuse_xb + kb * (kBN * kBK) + et * kBK);
#pragma unroll
            for (int q = 0; q < kBK / 16; ++q) {
              const uint4 v = rowp[q];
              sum = __dp4a(v.x, 0x01010101u, sum);
              sum = __dp4a(v.y, 0x01010101u, sum);
              sum = __dp4a(v.z, 0x01010101u, sum);
              sum = __dp4a(v.w, 0x01010101u, sum);
            }
          }
        }
        s_xs[et] = (landed && et < p.M) ? static_cast<int>(sum) - 8 * (kb1 - kb0) * kBK : 0;
      }
      if (!landed) s_epi_abort = 1;
      epi_sync();
    }
    if constexpr (kGroup) {
      // ---- grouped scales: promote each group's exact partial into the running sum ----
      constexpr int kChunk = kBN < 32 ? kBN : 32;
      const int G = p.ngroups, gkb = p.gkb;
      const int g0 = kb0 / gkb, g1 = kb1 / gkb;
      const float gconst = p.gconst;
      int gi = 0;
      for (int tile = QVLA_UNIT0; tile < ntiles; tile += QVLA_NUNITS) {
        const int ta = tile % tiles_a, tb = tile / tiles_a;
        epi_sync();
        if (s_epi_abort) break;
        if constexpr (!kSwap) {
          for (int c = et; c < kBN; c += kEpiThreads) {
            const int n = min(tb * kBN + c, p.N - 1);
            s_ws[c] = __ldg(p.wscale + n);
            s_bs[c] = __ldg(p.bias + n);
          }
          epi_sync();
        }
        const uint32_t lane_base = tmem_base + (static_cast<uint32_t>(warp * 32) << 16);
        const uint32_t run = lane_base + static_cast<uint32_t>(2 * kBN);  // the running sum's columns
        const int ra = ta * kBM + et;  // this thread's MMA-A row
        bool ok = true;
        for (int g = g0; g < g1; ++g, ++gi) {
          const int buf = gi & 1;
          if (!mbar_wait(smem_u32(&bar_tfull[buf]), static_cast<uint32_t>(gi >> 1) & 1u)) {
            s_epi_abort = 1;
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t part = lane_base + static_cast<uint32_t>(buf * kBN);
          const float dg = __ldg(p.gscale + g);
          const bool first = g == g0, last = g == g1 - 1;
          // the fixed part of this row's correction: 8 x its code sum over the group + 64 x size
          const bool rok = ra < (kSwap ? p.N : p.M);
          const int rc = rok ? ra : 0;
          const float rcorr = kSwap ? __ldg(p.wgcorr + static_cast<size_t>(rc) * G + g) + gconst
                                    : 8.0f * static_cast<float>(__ldg(p.xgsum + static_cast<size_t>(rc) * G + g)) + gconst;
#pragma unroll 1
          for (int c0 = 0; c0 < kBN; c0 += kChunk) {
            uint32_t r[32], R[32];
            __syncwarp();
            if constexpr (kChunk == 32) {
              tmem_ld32(part + c0, r);
              if (!first) tmem_ld32(run + c0, R);
            } else {
              tmem_ld16(part + c0, r);
              if (!first) tmem_ld16(run + c0, R);
            }
            tmem_ld_wait();
            const int col0 = tb * kBN + c0;  // first column (token when swapped, weight row else)
#pragma unroll
            for (int i = 0; i < kChunk; ++i) {
              const int col = min(col0 + i, (kSwap ? p.M : p.N) - 1);
              const float ccorr = kSwap ? 8.0f * static_cast<float>(__ldg(p.xgsum + static_cast<size_t>(col) * G + g))
                                        : __ldg(p.wgcorr + static_cast<size_t>(col) * G + g);
              // exact: the group's integer accumulator, below 2^24
              const float acc = fmaf(__uint_as_float(r[i]), 262144.0f, -(rcorr + ccorr));
              R[i] = __float_as_uint(fmaf(dg, acc, first ? 0.0f : __uint_as_float(R[i])));
            }
            if (!last) {
              if constexpr (kChunk == 32) {
                tmem_st32(run + c0, R);
              } else {
                tmem_st16(run + c0, R);
              }
              continue;
            }
            // the last group: y = Delta_W[n] x (sum over groups) + bias
            if constexpr (kSwap) {
              const int n = ra;
              if (splits > 1) {  // the cluster reduction below applies the epilogue
                float* partial = reinterpret_cast<float*>(smem);
#pragma unroll
                for (int i = 0; i < kChunk; ++i) partial[(c0 + i) * kBM + et] = __uint_as_float(R[i]);
              } else if (rok) {
                const float ws = __ldg(p.wscale + n), b = __ldg(p.bias + n);
#pragma unroll
                for (int i = 0; i < kChunk; ++i) {
                  const int m = col0 + i;
                  if (m < p.M)
                    reinterpret_cast<OutT*>(p.y)[static_cast<size_t>(m) * p.ldy + n] =
                        to_out<OutT>(fmaf(__uint_as_float(R[i]), ws, b));
                }
              }
            } else if (rok && col0 < p.N) {
              uint32_t pk[16];
#pragma unroll
              for (int i = 0; i < 16; ++i)
                pk[i] = pack2<OutT>(fmaf(__uint_as_float(R[2 * i]), s_ws[c0 + 2 * i], s_bs[c0 + 2 * i]),
                                    fmaf(__uint_as_float(R[2 * i + 1]), s_ws[c0 + 2 * i + 1], s_bs[c0 + 2 * i + 1]));
              store_row32(reinterpret_cast<OutT*>(p.y) + static_cast<size_t>(ra) * p.ldy + col0, pk, min(32, p.N - col0));
            }
          }
          tmem_st_wait();
          tc_fence_before();
          mbar_arrive(smem_u32(&bar_tempty[buf]));
        }
        if (!ok) continue;
      }
    } else
    for (int u = QVLA_UNIT0; u < nunits; u += QVLA_NUNITS, ++tile_iter) {
      int tile, ka, kz;
      unit_range(u, tile, ka, kz);
      (void)ka;
      (void)kz;
      const int part = u - tile * parts;
      const int ta = tile % tiles_a, tb = tile / tiles_a;
      const int buf = tile_iter & 1;
      const uint32_t aph = static_cast<uint32_t>(tile_iter >> 1) & 1u;
      // All epilogue threads pass this barrier every tile, so the abort decision below is
      // uniform and no thread is left waiting at a named barrier.  It also tells the writers
      // of the column parameters that the previous tile's readers are done.
      epi_sync();
      if (s_epi_abort) break;
      if constexpr (!kSwap) {
        // stage this tile's column parameters while the accumulator is still being computed
        for (int c = et; c < kBN; c += kEpiThreads) {
          const int n = min(tb * kBN + c, p.N - 1);
          s_ws[c] = __ldg(p.wscale + n);
          s_wc[c] = __ldg(p.wcorr + n);
          s_bs[c] = __ldg(p.bias + n);
        }
        epi_sync();
      }
      if (!mbar_wait(smem_u32(&bar_tfull[buf]), aph)) {
        s_epi_abort = 1;
        continue;
      }
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(warp * 32) << 16) + static_cast<uint32_t>(buf * kBN);
      const int ra = kPair ? ta * 2 * kBM + static_cast<int>(prank) * kBM + et : ta * kBM + et;  // this thread's MMA-A row
      if constexpr (!kSwap && !kGated) {
        // rows = tokens m, columns = weight rows n
        const int m = ra;
        const bool mok = m < p.M;
        const float xs = mok ? p.xscale[m] : 0.0f;
        const float cm = mok ? 8.0f * static_cast<float>(p.xsum[m]) + k64 : 0.0f;
        OutT* yrow = reinterpret_cast<OutT*>(p.y) + static_cast<size_t>(mok ? m : 0) * p.ldy;
        // split of K (parts > 1): this unit's partial goes to its slot, and the tile's last unit
        // to finish adds the other units' slots to its own accumulator (exact: every partial is a
        // non-negative integer multiple of the same power of two, and so is their sum, below 2^24
        // of them).  A slot holds float4 (row r, columns 4j .. 4j+3) at j * kBM + r, so the 32
        // rows of a warp move 512 contiguous bytes per access.  On a CTA pair each CTA has slots
        // and a count of its own 128 rows: slot (tile, part, CTA rank), count (tile, CTA rank).
        constexpr int kHalves = kPair ? 2 : 1;
        constexpr int kSlot4 = kBM * kBN / 4;
        const int half = static_cast<int>(prank);
        float4* const slot4 = parts > 1 ? reinterpret_cast<float4*>(p.part_ws) + static_cast<size_t>((tile * parts + part) * kHalves + half) * kSlot4 + et : nullptr;
        bool last = parts == 1;
        if (parts > 1) {
#pragma unroll 1
          for (int c0 = 0; c0 < kBN; c0 += 32) {
            uint32_t r[32];
            __syncwarp();
            tmem_ld32(taddr + c0, r);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 32; i += 4)
              __stcg(slot4 + ((c0 + i) / 4) * kBM, make_float4(__uint_as_float(r[i]), __uint_as_float(r[i + 1]),
                                                                __uint_as_float(r[i + 2]), __uint_as_float(r[i + 3])));
          }
          // the slot is written (every row: the barrier, then the counting thread's fence) before
          // the unit is counted, and the last unit reads the slots after its fence
          epi_sync();
          if (et == 0) {
            __threadfence();
            s_last = atomicAdd(p.part_cnt + tile * kHalves + half, 1) == parts - 1;
          }
          epi_sync();
          last = s_last != 0;
          if (last) __threadfence();
        }
#pragma unroll 1
        for (int c0 = 0; c0 < kBN && last; c0 += 32) {
          uint32_t r[32];
          __syncwarp();
          tmem_ld32(taddr + c0, r);
          tmem_ld_wait();
#pragma unroll 1
          for (int q = 0; q < parts; ++q) {
            if (q == part) continue;
            const float4* const o4 = slot4 + static_cast<ptrdiff_t>(q - part) * kHalves * kSlot4 + (c0 / 4) * kBM;
            float4 v[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = __ldcg(o4 + j * kBM);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              r[4 * j] = __float_as_uint(__uint_as_float(r[4 * j]) + v[j].x);
              r[4 * j + 1] = __float_as_uint(__uint_as_float(r[4 * j + 1]) + v[j].y);
              r[4 * j + 2] = __float_as_uint(__uint_as_float(r[4 * j + 2]) + v[j].z);
              r[4 * j + 3] = __float_as_uint(__uint_as_float(r[4 * j + 3]) + v[j].w);
            }
          }
          const int n0 = tb * kBN + c0;
          if (mok && n0 < p.N) {
            const int nvalid = min(32, p.N - n0);
            float acc[32];
            uint32_t pk[16];
#pragma unroll
            for (int i4 = 0; i4 < 8; ++i4) {
              const float4 ws = *reinterpret_cast<const float4*>(s_ws + c0 + 4 * i4);
              const float4 wc = *reinterpret_cast<const float4*>(s_wc + c0 + 4 * i4);
              const float4 bs = *reinterpret_cast<const float4*>(s_bs + c0 + 4 * i4);
              const float wsv[4] = {ws.x, ws.y, ws.z, ws.w}, wcv[4] = {wc.x, wc.y, wc.z, wc.w};
              const float bsv[4] = {bs.x, bs.y, bs.z, bs.w};
              float yv[4];
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const int i = 4 * i4 + k;
                acc[i] = fmaf(__uint_as_float(r[i]), 262144.0f, -(cm + wcv[k]));
                yv[k] = fmaf(acc[i], xs * wsv[k], bsv[k]);
              }
              pk[2 * i4] = pack2<OutT>(yv[0], yv[1]);
              pk[2 * i4 + 1] = pack2<OutT>(yv[2], yv[3]);
            }
            store_row32(yrow + n0, pk, nvalid);
            if (p.acc) {
              int32_t* arow = p.acc + static_cast<size_t>(m) * p.N + n0;
#pragma unroll
              for (int i = 0; i < 32; ++i)
                if (i < nvalid) arow[i] = static_cast<int32_t>(acc[i]);
            }
          }
        }
        if (parts > 1 && last && et == 0) p.part_cnt[tile * kHalves + half] = 0;  // ready for the next launch
      } else if constexpr (!kSwap && kGated) {
        // Gated MLP: tile columns [0, kBN/2) are the gate rows of hidden units
        // j0 .. j0 + kBN/2 - 1 and columns [kBN/2, kBN) the up rows of the same units.
        // gate and up are rounded to the output dtype like a stand-alone linear's outputs,
        // then h = gelu_tanh(gate) * up is rounded once more and stored [M][H].
        constexpr int kHalf = kBN / 2;
        const int m = ra;
        const bool mok = m < p.M;
        const float xs = mok ? p.xscale[m] : 0.0f;
        const float cm = mok ? 8.0f * static_cast<float>(p.xsum[m]) + k64 : 0.0f;
        const int j0 = tb * kHalf;
        const int H = p.N / 2;
        OutT* yrow = reinterpret_cast<OutT*>(p.y) + static_cast<size_t>(mok ? m : 0) * p.ldy;
#pragma unroll 1
        for (int c0 = 0; c0 < kHalf; c0 += 16) {
          uint32_t rg[16], ru[16];
          __syncwarp();
          tmem_ld16(taddr + c0, rg);
          tmem_ld16(taddr + kHalf + c0, ru);
          tmem_ld_wait();
          if (mok) {
            uint32_t pk[8];
#pragma unroll
            for (int i4 = 0; i4 < 4; ++i4) {
              const int cg = c0 + 4 * i4, cu = cg + kHalf;
              const float4 wsg = *reinterpret_cast<const float4*>(s_ws + cg);
              const float4 wcg = *reinterpret_cast<const float4*>(s_wc + cg);
              const float4 bsg = *reinterpret_cast<const float4*>(s_bs + cg);
              const float4 wsu = *reinterpret_cast<const float4*>(s_ws + cu);
              const float4 wcu = *reinterpret_cast<const float4*>(s_wc + cu);
              const float4 bsu = *reinterpret_cast<const float4*>(s_bs + cu);
              const float wsgv[4] = {wsg.x, wsg.y, wsg.z, wsg.w}, wcgv[4] = {wcg.x, wcg.y, wcg.z, wcg.w};
              const float bsgv[4] = {bsg.x, bsg.y, bsg.z, bsg.w}, wsuv[4] = {wsu.x, wsu.y, wsu.z, wsu.w};
              const float wcuv[4] = {wcu.x, wcu.y, wcu.z, wcu.w}, bsuv[4] = {bsu.x, bsu.y, bsu.z, bsu.w};
              float hv[4];
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const int i = 4 * i4 + k;
                const float ag = fmaf(__uint_as_float(rg[i]), 262144.0f, -(cm + wcgv[k]));
                const float au = fmaf(__uint_as_float(ru[i]), 262144.0f, -(cm + wcuv[k]));
                // gate and up rounded to the output dtype (one pair conversion), then h
                const float2 gu = unpack2<OutT>(pack2<OutT>(fmaf(ag, xs * wsgv[k], bsgv[k]), fmaf(au, xs * wsuv[k], bsuv[k])));
                hv[k] = gelu_tanh(gu.x) * gu.y;
                if (p.acc) {  // debug view in natural order: [gate units | up units]
                  int32_t* arow = p.acc + static_cast<size_t>(m) * p.N;
                  arow[j0 + c0 + i] = static_cast<int32_t>(ag);
                  arow[H + j0 + c0 + i] = static_cast<int32_t>(au);
                }
              }
              pk[2 * i4] = pack2<OutT>(hv[0], hv[1]);
              pk[2 * i4 + 1] = pack2<OutT>(hv[2], hv[3]);
            }
            uint4* d = reinterpret_cast<uint4*>(yrow + j0 + c0);
            d[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            d[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
          }
        }
      } else {
        // rows = weight rows n, columns = tokens m
        const int n = ra;
        const bool nok = n < p.N;
        const float ws = nok ? __ldg(p.wscale + n) : 0.0f;
        const float cn = nok ? __ldg(p.wcorr + n) + k64 : 0.0f;
        const float b = nok ? __ldg(p.bias + n) : 0.0f;
        constexpr int kChunk = kBN < 32 ? kBN : 32;
        float* part = reinterpret_cast<float*>(smem);  // split-K partial [kBN][128]; the stages are idle now
#pragma unroll 1
        for (int c0 = 0; c0 < kBN; c0 += kChunk) {
          uint32_t r[32];
          __syncwarp();
          if constexpr (kChunk == 32) {
            tmem_ld32(taddr + c0, r);
          } else {
            tmem_ld16(taddr + c0, r);
          }
          tmem_ld_wait();
          if (splits > 1) {  // leave the partial sums for the cluster reduction below
#pragma unroll
            for (int i = 0; i < kChunk; ++i) {
              // fused: this range's activation code sums leave the partial here (exact: both are
              // integer multiples of 2^-18 below 2^6)
              part[(c0 + i) * kBM + et] =
                  kFused ? fmaf(static_cast<float>(s_xs[c0 + i]), -3.0517578125e-05f, __uint_as_float(r[i]))
                         : __uint_as_float(r[i]);
            }
            continue;
          }
          const int m0 = tb * kBN + c0;
          if (nok) {
#pragma unroll
            for (int i = 0; i < kChunk; ++i) {
              const int m = m0 + i;
              if (m < p.M) {
                const float corr = cn + 8.0f * static_cast<float>(kFused ? s_xs[m] : __ldg(p.xsum + m));
                const float acc = fmaf(__uint_as_float(r[i]), 262144.0f, -corr);
                reinterpret_cast<OutT*>(p.y)[static_cast<size_t>(m) * p.ldy + n] =
                    to_out<OutT>(fmaf(acc, __ldg(p.xscale + (kFused ? 0 : m)) * ws, b));
                if (p.acc) p.acc[static_cast<size_t>(m) * p.N + n] = static_cast<int32_t>(acc);
              }
            }
          }
        }
      }
      tc_fence_before();
      if (kPair && prank != 0) {  // the peer's epilogue warps report to the leader
        __syncwarp();
        if (lane == 0) mbar_arrive_peer(mapa_shared(smem_u32(&bar_tempty[buf]), 0));
      } else {
        mbar_arrive(smem_u32(&bar_tempty[buf]));
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if constexpr (kPair) cluster_sync();  // the leader's MMAs into this CTA's TMEM are complete
  if constexpr (kSwap) {
    if (splits > 1) {
      // split-K: every CTA's partial [kBN columns][128 rows] is in its shared memory.  CTA r
      // owns rows [r R, (r + 1) R) of the tile (R = 128 / splits): each CTA pushes its slice of
      // those rows into CTA r's receive area ([source CTA][column][R rows]) with asynchronous
      // stores that complete on CTA r's barrier; CTA r then sums the slices from its own shared
      // memory and applies the epilogue.  An element is 4 consecutive weight rows of one token
      // column; its epilogue parameters are fetched one element ahead (the first while the
      // partials are in flight).  No CTA reads another's shared memory, so none waits for the
      // others before leaving.
      if constexpr (!kFused) cluster_wait();  // pairs with the arrive after set-up: every receive barrier is initialised
      const int R = kBM / splits;
      const float* part = reinterpret_cast<const float*>(smem);
      const uint32_t recv0 = smem_u32(smem + C::kRecvOff);
      // kThreads is a multiple of kBM / 4, so a thread's row (and owner) is the same at every step
      static_assert(kThreads % (kBM / 4) == 0, "fixed row per thread");
      {
        const int row = (static_cast<int>(threadIdx.x) % (kBM / 4)) * 4;
        const int owner = row / R;
        const uint32_t rbar = mapa_shared(smem_u32(&bar_recv), static_cast<uint32_t>(owner));
        const uint32_t rdst = mapa_shared(recv0, static_cast<uint32_t>(owner)) +
                              static_cast<uint32_t>((static_cast<int>(krank) * kBN * R + (row - owner * R)) * 4);
        for (int col = static_cast<int>(threadIdx.x) / (kBM / 4); col < split_cols; col += kThreads / (kBM / 4))
          st_async_v4(rdst + static_cast<uint32_t>(col * R * 4), *reinterpret_cast<const float4*>(part + col * kBM + row), rbar);
      }
      const int R4 = R / 4;
      const int unit0 = static_cast<int>(QVLA_UNIT0);
      const int total = unit0 < ntiles && !s_epi_abort ? R4 * split_cols : 0;
      const int ta = unit0 % tiles_a, tb = unit0 / tiles_a;
      auto coords = [&](int e, int& n, int& m, int& row, int& col) {
        row = (e % R4) * 4;  // within this CTA's R rows
        col = e / R4;
        n = ta * kBM + static_cast<int>(krank) * R + row;
        m = tb * kBN + col;
      };
      griddep_wait();
      SplitParams nxt;
      int e = threadIdx.x;
      if (e < total) {
        int n, m, row, col;
        coords(e, n, m, row, col);
        nxt.template load<kGroup, kFused>(p, n, m);
      }
      // acquire at cluster scope: the asynchronous stores release their bytes at cluster scope
      const bool landed = mbar_wait_cluster(smem_u32(&bar_recv), 0);
      const float* recv = reinterpret_cast<const float*>(smem + C::kRecvOff);
      for (; landed && e < total; e += kThreads) {
        int n, m, row, col;
        coords(e, n, m, row, col);
        const SplitParams cur = nxt;
        if (e + kThreads < total) {
          int n2, m2, r2, c2;
          coords(e + kThreads, n2, m2, r2, c2);
          nxt.template load<kGroup, kFused>(p, n2, m2);
        }
        // exact: the partials add up to the tile's accumulator, an integer below 2^24 times 2^-18
        float4 sum = *reinterpret_cast<const float4*>(recv + col * R + row);
#pragma unroll
        for (int q = 1; q < 8; ++q)
          if (q < splits) {
            const float4 v = *reinterpret_cast<const float4*>(recv + (q * kBN + col) * R + row);
            sum.x += v.x;
            sum.y += v.y;
            sum.z += v.z;
            sum.w += v.w;
          }
        if (kGroup && n < p.N && m < p.M) {  // grouped: the partials are scaled and corrected sums
          const uint32_t lo = pack2<OutT>(fmaf(sum.x, cur.ws.x, cur.bs.x), fmaf(sum.y, cur.ws.y, cur.bs.y));
          const uint32_t hi = pack2<OutT>(fmaf(sum.z, cur.ws.z, cur.bs.z), fmaf(sum.w, cur.ws.w, cur.bs.w));
          *reinterpret_cast<uint2*>(reinterpret_cast<OutT*>(p.y) + static_cast<size_t>(m) * p.ldy + n) =
              make_uint2(lo, hi);
        } else if (n < p.N && m < p.M) {  // N % 16 == 0, so rows n .. n + 3 all exist
          const float a0 = fmaf(sum.x, 262144.0f, -(cur.wc.x + cur.cm));
          const float a1 = fmaf(sum.y, 262144.0f, -(cur.wc.y + cur.cm));
          const float a2 = fmaf(sum.z, 262144.0f, -(cur.wc.z + cur.cm));
          const float a3 = fmaf(sum.w, 262144.0f, -(cur.wc.w + cur.cm));
          const float xs = cur.xs;
          const uint32_t lo = pack2<OutT>(fmaf(a0, xs * cur.ws.x, cur.bs.x), fmaf(a1, xs * cur.ws.y, cur.bs.y));
          const uint32_t hi = pack2<OutT>(fmaf(a2, xs * cur.ws.z, cur.bs.z), fmaf(a3, xs * cur.ws.w, cur.bs.w));
          *reinterpret_cast<uint2*>(reinterpret_cast<OutT*>(p.y) + static_cast<size_t>(m) * p.ldy + n) =
              make_uint2(lo, hi);
          if (p.acc)
            *reinterpret_cast<int4*>(p.acc + static_cast<size_t>(m) * p.N + n) =
                make_int4(static_cast<int32_t>(a0), static_cast<int32_t>(a1), static_cast<int32_t>(a2),
                          static_cast<int32_t>(a3));
        }
      }
    }
  }
  if constexpr (kFused) {
    if (warp == 0) bulk_wait_read();  // the staged bytes this CTA sent are read
  }
  tc_fence_after();
  if (warp == kMmaWarp) {
    if constexpr (kPair) {
      tmem_dealloc_pair<kTmemCols>(tmem_base);
    } else {
      tmem_dealloc<kTmemCols>(tmem_base);
    }
  }
#undef QVLA_UNIT0
#undef QVLA_NUNITS
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// A [rows][row_bytes] byte matrix read in boxes of 64 bytes (one k-block of packed codes) x
// box_rows rows; rows past the end read as zero.
cudaError_t make_tmap(CUtensorMap* m, const void* base, int rows, int row_bytes, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(row_bytes), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(row_bytes)};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK / 2), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// An operand for the swizzled direct load: [rows][K] operand bytes in boxes of 128 bytes (one
// k-block) x box_rows, written into shared memory with the 128-byte swizzle of the MMA layout.
cudaError_t make_tmap_bytes(CUtensorMap* m, const void* base, int rows, int K, int box_rows) {
  PFN_cuTensorMapEncodeTiled_v12000 enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  const cuuint64_t dims[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(rows)};
  const cuuint64_t strides[1] = {static_cast<cuuint64_t>(K)};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Raise a kernel's dynamic shared-memory limit, once per kernel and device.
cudaError_t prepare_kernel(const void* kern, int smem) {
  static std::mutex mu;
  static std::set<std::pair<const void*, int>> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  if (done.count({kern, dev})) return cudaSuccess;
  e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess) done.insert({kern, dev});
  return e;
}

// How many clusters of cfg's shape (its only attribute: the cluster dimension) can be resident
// at once, cached per kernel, cluster size and device; 0 if the query fails.
int max_active_clusters(const void* kern, const cudaLaunchConfig_t& cfg) {
  static std::mutex mu;
  static std::map<std::tuple<const void*, unsigned, int>, int> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  const unsigned cs = cfg.attrs[0].val.clusterDim.x;
  std::lock_guard<std::mutex> lock(mu);
  auto it = cache.find({kern, cs, dev});
  if (it != cache.end()) return it->second;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  cache[{kern, cs, dev}] = n;
  return n;
}

// Returned by launch_fused_cfg when the shape does not fit the fused kernel (nothing launched).
constexpr cudaError_t kNotApplicable = cudaErrorNotSupported;

// The fused one-launch linear on BN-token tiles with kE channels per lane: picks the largest
// split of K (1, 2, 4, 8 CTAs per weight tile) for which one tile per CTA fits the SMs, the
// k-range fits the stages and the operand tile, the staged rows fit, every (CTA, k-block) copy
// has a lane to issue it, and every cluster is resident.  kNotApplicable if none does.
template <int kBN, typename OutT, int kE, typename XT>
cudaError_t launch_fused_cfg(const GemmArgs& a) {
  using C = Cfg<kBN, true, false, 1, kBM * kBN * 4, kFuseExtra, false>;
  if (a.M > kBN || a.K % (32 * kE) != 0 || a.K % kBK != 0) return kNotApplicable;
  const int nkb = a.K / kBK;
  const int tiles = (a.N + kBM - 1) / kBM;
  auto kern = gemm_w4a4_kernel<kBN, true, false, 3, OutT, false, false, kE, XT>;
  cudaError_t e = prepare_kernel(reinterpret_cast<const void*>(kern), C::kSmem);
  if (e != cudaSuccess) return e == kNotApplicable ? cudaErrorUnknown : e;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::kSmem;
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  int splits = 0;
  for (int s = 8; s >= 1; s /= 2) {
    const int range = nkb / s;
    if (nkb % s != 0 || range > C::kStages || range * kBN * kBK > kFuseXBMax || s * range > 32) continue;
    if ((a.M + s - 1) / s * a.K > kFuseStagingMax || tiles * s > a.num_sms) continue;
    if (s > 1) {
      attr[0].val.clusterDim.x = static_cast<unsigned>(s);
      cfg.gridDim = dim3(tiles * s);
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      if (max_active_clusters(reinterpret_cast<const void*>(kern), cfg) < tiles) continue;
    }
    splits = s;
    break;
  }
  if (splits == 0) return kNotApplicable;
  Params p = {};
  p.a = a.wq;
  p.rows_a = a.N;
  p.b = nullptr;
  p.rows_b = a.M;
  p.K = a.K;
  p.kconst = 64.0f * static_cast<float>(a.K);
  p.xscale = a.xscale;
  p.xsum = nullptr;
  p.wscale = a.wscale;
  p.wcorr = a.wcorr;
  p.bias = a.bias;
  p.y = a.y;
  p.acc = nullptr;
  p.M = a.M;
  p.N = a.N;
  p.ldy = a.N;
  p.splits = splits;
  p.parts = 1;
  p.part_ws = nullptr;
  p.part_cnt = nullptr;
  p.x = a.x;
  p.log_b = a.log_b;
  p.inv_sqrt_b = a.inv_sqrt_b;
  attr[0].val.clusterDim.x = static_cast<unsigned>(splits);
  cfg.gridDim = dim3(tiles * splits);
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  CUtensorMap none = {};
  e = cudaLaunchKernelEx(&cfg, kern, none, none, p);
  if (e == cudaSuccess) e = cudaGetLastError();
  return e == kNotApplicable ? cudaErrorUnknown : e;  // a real failure is never read as "not applicable"
}

template <int kBN, bool kSwap, bool kGated, int kX, typename OutT, bool kGroup = false, bool kPair = false>
cudaError_t launch_cfg(const GemmArgs& a) {
  constexpr bool kXBytes = kX >= 1;
  constexpr int kPlanes = kX == 2 ? 2 : 1;
  constexpr bool kStageA = !(kXBytes && !kSwap);
  constexpr bool kStageB = !(kXBytes && kSwap);
  using C = Cfg<kPair ? kBN / 2 : kBN, kStageA, kStageB, kPlanes, kSwap ? kBM * kBN * 4 : 0>;
  Params p;
  if (kSwap) {
    p.a = a.wq;
    p.rows_a = a.N;
    p.b = a.xq;
    p.rows_b = a.M;
  } else {
    p.a = a.xq;
    p.rows_a = a.M;
    p.b = a.wq;
    p.rows_b = a.N;
  }
  p.K = a.K;
  p.kconst = (kX == 2 ? 1024.0f : 64.0f) * static_cast<float>(a.K);
  p.gscale = a.gscale;
  p.xgsum = a.xgsum;
  p.wgcorr = a.wgcorr;
  p.gkb = a.group / kBK;
  p.ngroups = a.group > 0 ? a.K / a.group : 0;
  p.gconst = 64.0f * static_cast<float>(a.group);
  p.xscale = a.xscale;
  p.xsum = a.xsum;
  p.wscale = a.wscale;
  p.wcorr = a.wcorr;
  p.bias = a.bias;
  p.y = a.y;
  p.acc = a.acc;
  p.M = a.M;
  p.N = a.N;
  p.ldy = a.gated ? a.N / 2 : a.N;
  const int tm = kPair ? (p.rows_a + 2 * kBM - 1) / (2 * kBM) : (p.rows_a + kBM - 1) / kBM;
  const int tiles = tm * ((p.rows_b + kBN - 1) / kBN);
  if (tiles == 0) return cudaSuccess;
  auto kern = gemm_w4a4_kernel<kBN, kSwap, kGated, kX, OutT, kGroup, kPair>;
  cudaError_t e = prepare_kernel(reinterpret_cast<const void*>(kern), C::kSmem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::kSmem;
  cfg.stream = a.stream;
  // attr[0]: may start while the previous kernel of the stream finishes; attr[1]: cluster shape
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr + 1;
  cfg.numAttrs = 1;
  // weight-major orientation: while the tiles alone leave SMs idle, split K over a cluster of
  // up to 8 CTAs, as long as every cluster of the grid can be resident at once
  int splits = 1;
  if (kSwap) {
    const int nkb = kGroup ? p.ngroups : p.K / kBK;  // grouped scales split whole groups
    while (splits < 8 && 2 * splits <= nkb && tiles * 2 * splits <= a.num_sms) {
      attr[1].val.clusterDim.x = static_cast<unsigned>(2 * splits);
      cfg.gridDim = dim3(tiles * 2 * splits);
      if (max_active_clusters(reinterpret_cast<const void*>(kern), cfg) < tiles) break;
      splits *= 2;
    }
  }
  p.splits = splits;
  // token-major tiles of a non-gated layer: each tile's k-blocks in a.parts work units over the
  // persistent CTAs (or pairs), partials in the caller's workspace, when it has room for them
  p.parts = 1;
  p.part_ws = nullptr;
  p.part_cnt = nullptr;
  if constexpr (!kSwap && !kGated && !kGroup && kX <= 1) {
    const long halves = kPair ? 2 : 1;
    if (a.parts > 1 && a.part_ws != nullptr && a.part_cnt != nullptr && p.K / kBK >= a.parts &&
        static_cast<size_t>(tiles) * halves * a.parts * kBM * kBN <= a.part_ws_floats && tiles * halves <= a.part_cnt_n) {
      p.parts = a.parts;
      p.part_ws = a.part_ws;
      p.part_cnt = a.part_cnt;
    }
  }
  attr[1].val.clusterDim.x = static_cast<unsigned>(kPair ? 2 : splits);
  if (kPair) {
    const int pairs = a.num_sms / 2, units = tiles * p.parts;
    cfg.gridDim = dim3(2 * (units < pairs ? units : pairs));
  } else {
    const int units = tiles * p.parts;
    cfg.gridDim = dim3(splits > 1 ? tiles * splits : (units < a.num_sms ? units : a.num_sms));
  }
  cfg.attrs = attr;
  cfg.numAttrs = (kPair || splits > 1) ? 2 : 1;  // a cluster launch for pairs and when K is split
  // a tensor map for the activations only (the weights arrive as contiguous chunks)
  CUtensorMap ta = {}, tb = {};
  if constexpr (kSwap) {
    e = kStageB ? make_tmap(&tb, p.b, p.rows_b, p.K / 2, kBN)
                : make_tmap_bytes(&tb, p.b, p.rows_b, kPlanes * p.K, kBN);
  } else {
    e = kStageA ? make_tmap(&ta, p.a, p.rows_a, p.K / 2, kBM)
                : make_tmap_bytes(&ta, p.a, p.rows_a, kPlanes * p.K, kBM);
  }
  if (e != cudaSuccess) return e;
  e = cudaLaunchKernelEx(&cfg, kern, ta, tb, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// Test hooks of the kernels instantiated in the including translation unit.
inline cudaError_t set_debug_hooks(unsigned long long wait_limit_ns, int hold_loads) {
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyToSymbol(g_wait_limit_ns, &wait_limit_ns, sizeof(wait_limit_ns));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_debug_hold_loads, &hold_loads, sizeof(hold_loads));
}

}  // namespace
}  // namespace qvla
