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
//   warps 5-12  two producer groups of four warps, taking alternate k-blocks: they load packed
//               nibbles from global memory, expand them to E4M3 bytes and store them in the
//               128-byte-swizzled K-major layout the MMA descriptors expect.
// Shared memory holds kStages k-blocks of 128 codes; TMEM holds two accumulators so the
// epilogue of one tile overlaps the main loop of the next.
//
// Two orientations: for M > 128 the MMA's M side is the activations (tile 128 tokens x 256
// weight rows); for M <= 128 ("swap") it is the weights (128 weight rows x Mpad tokens),
// so that a small batch does not waste the 128-row MMA.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "kernels.h"
#include "ptx.cuh"

namespace qvla {
namespace {

constexpr int kBM = 128;        // MMA M (rows of the MMA A operand)
constexpr int kBK = 128;        // codes per k-block (one 128-byte swizzle row of E4M3)
constexpr int kEpiWarps = 4;
constexpr int kMmaWarp = 4;
constexpr int kProdWarpsPerGroup = 4;
constexpr int kProdGroups = 2;
constexpr int kProdThreadsPerGroup = kProdWarpsPerGroup * 32;
constexpr int kThreads = (kEpiWarps + 1 + kProdGroups * kProdWarpsPerGroup) * 32;

template <int kBN>
struct Cfg {
  static constexpr int kTileA = kBM * kBK;    // bytes of E4M3
  static constexpr int kTileB = kBN * kBK;
  static constexpr int kStage = kTileA + kTileB;
  static constexpr int kStagesRaw = (200 * 1024) / kStage;
  static constexpr int kStages = kStagesRaw > 8 ? 8 : kStagesRaw;
  static constexpr int kSmem = kStages * kStage + 1024;  // + alignment slack
  static constexpr uint32_t kTmemCols = (2 * kBN) <= 32 ? 32 : (2 * kBN) <= 64 ? 64 : (2 * kBN) <= 128 ? 128 : (2 * kBN) <= 256 ? 256 : 512;
  static_assert(kStages >= 2, "stages");
};

struct Params {
  const uint8_t* a;   // MMA A operand rows [rows_a][K/2]
  const uint8_t* b;   // MMA B operand rows [rows_b][K/2]
  int rows_a, rows_b, K;
  const float* xscale;
  const int32_t* xsum;
  const float* wscale;
  const int32_t* wsum;
  const float* bias;
  void* y;
  int32_t* acc;
  int M, N;      // N = weight rows of the layer (2H for a gated layer)
  int ldy;       // row length of y (N, or H for a gated layer)
};

__device__ __forceinline__ uint4 ldg_nc(const uint8_t* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// Expand one 16-byte chunk (32 codes) into 32 E4M3 bytes and store them as the two 16-byte
// columns 2q and 2q+1 of row r of a 128-byte-swizzled tile.
__device__ __forceinline__ void store_chunk(uint8_t* tile, int r, int q, uint4 v) {
  uint32_t o[8];
  int4x8_to_e4m3_offset(v.x, o[0], o[1]);
  int4x8_to_e4m3_offset(v.y, o[2], o[3]);
  int4x8_to_e4m3_offset(v.z, o[4], o[5]);
  int4x8_to_e4m3_offset(v.w, o[6], o[7]);
  uint8_t* row = tile + r * 128;
  const int sw = r & 7;
  *reinterpret_cast<uint4*>(row + (((2 * q) ^ sw) << 4)) = make_uint4(o[0], o[1], o[2], o[3]);
  *reinterpret_cast<uint4*>(row + (((2 * q + 1) ^ sw) << 4)) = make_uint4(o[4], o[5], o[6], o[7]);
}

// GELU, tanh form, written as g * sigmoid(2u) = g / (1 + exp(-2u)), u = sqrt(2/pi) (g + 0.044715 g^3):
// the same function as 0.5 g (1 + tanh(u)) without the cancellation of 1 + tanh near u -> -inf.
__device__ __forceinline__ float gelu_tanh(float g) {
  const float u = 0.7978845608028654f * g * fmaf(0.044715f, g * g, 1.0f);
  return __fdividef(g, 1.0f + __expf(-2.0f * u));
}

template <typename OutT>
__device__ __forceinline__ OutT to_out(float v);
template <>
__device__ __forceinline__ __half to_out<__half>(float v) { return __float2half_rn(v); }
template <>
__device__ __forceinline__ __nv_bfloat16 to_out<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }
__device__ __forceinline__ float from_out(__half v) { return __half2float(v); }
__device__ __forceinline__ float from_out(__nv_bfloat16 v) { return __bfloat162float(v); }

// 32 outputs of one row as 4 x 16-byte stores (or element stores at a ragged edge).
template <typename OutT>
__device__ __forceinline__ void store_row32(OutT* dst, const OutT (&out)[32], int nvalid) {
  if (nvalid == 32) {
    const uint4* src = reinterpret_cast<const uint4*>(out);
    uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i] = src[i];
  } else {
    for (int i = 0; i < nvalid; ++i) dst[i] = out[i];
  }
}

template <int kBN, bool kSwap, bool kGated, typename OutT>
__global__ void __launch_bounds__(kThreads, 1) gemm_w4a4_kernel(Params p) {
  using C = Cfg<kBN>;
  extern __shared__ uint8_t dyn_smem[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_smem) + 1023) & ~uintptr_t(1023));

  __shared__ __align__(8) uint64_t bar_full[C::kStages];
  __shared__ __align__(8) uint64_t bar_empty[C::kStages];
  __shared__ __align__(8) uint64_t bar_tfull[2];
  __shared__ __align__(8) uint64_t bar_tempty[2];
  __shared__ __align__(8) uint64_t bar_done;
  __shared__ uint32_t s_tmem_base;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  const int tiles_a = (p.rows_a + kBM - 1) / kBM;
  const int tiles_b = (p.rows_b + kBN - 1) / kBN;
  const int ntiles = tiles_a * tiles_b;
  const int nkb = p.K / kBK;
  const int kbytes = p.K / 2;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(smem_u32(&bar_full[s]), kProdThreadsPerGroup);
      mbar_init(smem_u32(&bar_empty[s]), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(smem_u32(&bar_tfull[i]), 1);
      mbar_init(smem_u32(&bar_tempty[i]), kEpiWarps * 32);
    }
    mbar_init(smem_u32(&bar_done), 1);
    mbar_init_fence();
  }
  if (warp == kMmaWarp) tmem_alloc<C::kTmemCols>(smem_u32(&s_tmem_base));
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = s_tmem_base;

  if (warp >= kMmaWarp + 1) {
    // ------------------------------------------------------------------ producers
    const int g = (warp - (kMmaWarp + 1)) / kProdWarpsPerGroup;
    const int pt = threadIdx.x - (kMmaWarp + 1) * 32 - g * kProdThreadsPerGroup;
    constexpr int kChunksA = kBM * 4;   // 16-byte packed chunks per A tile
    constexpr int kChunksB = kBN * 4;
    constexpr int kPerThreadA = kChunksA / kProdThreadsPerGroup;
    constexpr int kPerThreadB = (kChunksB + kProdThreadsPerGroup - 1) / kProdThreadsPerGroup;
    int it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x) {
      const int ta = tile % tiles_a, tb = tile / tiles_a;
      for (int kb = 0; kb < nkb; ++kb, ++it) {
        if ((it & 1) != g) continue;
        const int s = it % C::kStages;
        const uint32_t ph = static_cast<uint32_t>(it / C::kStages) & 1u;
        uint4 va[kPerThreadA], vb[kPerThreadB];
#pragma unroll
        for (int i = 0; i < kPerThreadA; ++i) {
          const int c = pt + i * kProdThreadsPerGroup;
          const int row = ta * kBM + (c >> 2);
          va[i] = row < p.rows_a ? ldg_nc(p.a + static_cast<size_t>(row) * kbytes + kb * 64 + (c & 3) * 16)
                                 : make_uint4(0x88888888u, 0x88888888u, 0x88888888u, 0x88888888u);
        }
#pragma unroll
        for (int i = 0; i < kPerThreadB; ++i) {
          const int c = pt + i * kProdThreadsPerGroup;
          const int row = tb * kBN + (c >> 2);
          vb[i] = (c < kChunksB && row < p.rows_b)
                      ? ldg_nc(p.b + static_cast<size_t>(row) * kbytes + kb * 64 + (c & 3) * 16)
                      : make_uint4(0x88888888u, 0x88888888u, 0x88888888u, 0x88888888u);
        }
        if (!mbar_wait(smem_u32(&bar_empty[s]), ph ^ 1u)) { ok = false; break; }
        uint8_t* sa = smem + s * C::kStage;
        uint8_t* sb = sa + C::kTileA;
#pragma unroll
        for (int i = 0; i < kPerThreadA; ++i) {
          const int c = pt + i * kProdThreadsPerGroup;
          store_chunk(sa, c >> 2, c & 3, va[i]);
        }
#pragma unroll
        for (int i = 0; i < kPerThreadB; ++i) {
          const int c = pt + i * kProdThreadsPerGroup;
          if (c < kChunksB) store_chunk(sb, c >> 2, c & 3, vb[i]);
        }
        fence_proxy_async_smem();
        mbar_arrive(smem_u32(&bar_full[s]));
      }
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_e4m3_f32(kBM, kBN);
      int it = 0, tile_iter = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < ntiles && ok; tile += gridDim.x, ++tile_iter) {
        const int buf = tile_iter & 1;
        const uint32_t aph = static_cast<uint32_t>(tile_iter >> 1) & 1u;
        if (!mbar_wait(smem_u32(&bar_tempty[buf]), aph ^ 1u)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d = tmem_base + static_cast<uint32_t>(buf * kBN);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = it % C::kStages;
          const uint32_t ph = static_cast<uint32_t>(it / C::kStages) & 1u;
          if (!mbar_wait(smem_u32(&bar_full[s]), ph)) { ok = false; break; }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + s * C::kStage);
          const uint32_t sb = sa + C::kTileA;
#pragma unroll
          for (int kk = 0; kk < kBK / 32; ++kk) {
            mma_e4m3(d, smem_desc_sw128(sa + kk * 32), smem_desc_sw128(sb + kk * 32), kIdesc,
                     (kb | kk) != 0 ? 1u : 0u);
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
    const float k64 = 64.0f * static_cast<float>(p.K);
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++tile_iter) {
      const int ta = tile % tiles_a, tb = tile / tiles_a;
      const int buf = tile_iter & 1;
      const uint32_t aph = static_cast<uint32_t>(tile_iter >> 1) & 1u;
      if (!mbar_wait(smem_u32(&bar_tfull[buf]), aph)) break;
      tc_fence_after();
      const uint32_t taddr = tmem_base + (static_cast<uint32_t>(warp * 32) << 16) + static_cast<uint32_t>(buf * kBN);
      const int ra = ta * kBM + et;  // this thread's MMA-A row
      if constexpr (!kSwap && !kGated) {
        // rows = tokens m, columns = weight rows n
        const int m = ra;
        const bool mok = m < p.M;
        const float xs = mok ? p.xscale[m] : 0.0f;
        const float cm = mok ? 8.0f * static_cast<float>(p.xsum[m]) + k64 : 0.0f;
        OutT* yrow = reinterpret_cast<OutT*>(p.y) + static_cast<size_t>(mok ? m : 0) * p.ldy;
#pragma unroll 1
        for (int c0 = 0; c0 < kBN; c0 += 32) {
          uint32_t r[32];
          __syncwarp();
          tmem_ld32(taddr + c0, r);
          tmem_ld_wait();
          const int n0 = tb * kBN + c0;
          if (mok && n0 < p.N) {
            const int nvalid = min(32, p.N - n0);
            alignas(16) OutT out[32];
            int32_t ai[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int n = min(n0 + i, p.N - 1);
              const float corr = cm + 8.0f * static_cast<float>(__ldg(p.wsum + n));
              const float acc = fmaf(__uint_as_float(r[i]), 262144.0f, -corr);
              const float b = p.bias ? __ldg(p.bias + n) : 0.0f;
              out[i] = to_out<OutT>(fmaf(acc, xs * __ldg(p.wscale + n), b));
              ai[i] = static_cast<int32_t>(acc);
            }
            store_row32(yrow + n0, out, nvalid);
            if (p.acc) {
              int32_t* arow = p.acc + static_cast<size_t>(m) * p.N + n0;
              for (int i = 0; i < nvalid; ++i) arow[i] = ai[i];
            }
          }
        }
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
        for (int c0 = 0; c0 < kHalf; c0 += 32) {
          uint32_t rg[32], ru[32];
          __syncwarp();
          tmem_ld32(taddr + c0, rg);
          tmem_ld32(taddr + kHalf + c0, ru);
          tmem_ld_wait();
          if (mok) {
            alignas(16) OutT out[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int ng = tb * kBN + c0 + i, nu = ng + kHalf;
              const float ag = fmaf(__uint_as_float(rg[i]), 262144.0f, -(cm + 8.0f * static_cast<float>(__ldg(p.wsum + ng))));
              const float au = fmaf(__uint_as_float(ru[i]), 262144.0f, -(cm + 8.0f * static_cast<float>(__ldg(p.wsum + nu))));
              const float g = from_out(to_out<OutT>(fmaf(ag, xs * __ldg(p.wscale + ng), p.bias ? __ldg(p.bias + ng) : 0.0f)));
              const float u = from_out(to_out<OutT>(fmaf(au, xs * __ldg(p.wscale + nu), p.bias ? __ldg(p.bias + nu) : 0.0f)));
              out[i] = to_out<OutT>(gelu_tanh(g) * u);
              if (p.acc) {  // debug view in natural order: [gate units | up units]
                int32_t* arow = p.acc + static_cast<size_t>(m) * p.N;
                arow[j0 + c0 + i] = static_cast<int32_t>(ag);
                arow[H + j0 + c0 + i] = static_cast<int32_t>(au);
              }
            }
            store_row32(yrow + j0 + c0, out, 32);
          }
        }
      } else {
        // rows = weight rows n, columns = tokens m
        const int n = ra;
        const bool nok = n < p.N;
        const float ws = nok ? __ldg(p.wscale + n) : 0.0f;
        const float cn = nok ? 8.0f * static_cast<float>(__ldg(p.wsum + n)) + k64 : 0.0f;
        const float b = (nok && p.bias) ? __ldg(p.bias + n) : 0.0f;
        constexpr int kChunk = kBN < 32 ? kBN : 32;
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
          const int m0 = tb * kBN + c0;
          if (nok) {
#pragma unroll
            for (int i = 0; i < kChunk; ++i) {
              const int m = m0 + i;
              if (m < p.M) {
                const float corr = cn + 8.0f * static_cast<float>(__ldg(p.xsum + m));
                const float acc = fmaf(__uint_as_float(r[i]), 262144.0f, -corr);
                reinterpret_cast<OutT*>(p.y)[static_cast<size_t>(m) * p.ldy + n] =
                    to_out<OutT>(fmaf(acc, __ldg(p.xscale + m) * ws, b));
                if (p.acc) p.acc[static_cast<size_t>(m) * p.N + n] = static_cast<int32_t>(acc);
              }
            }
          }
        }
      }
      tc_fence_before();
      mbar_arrive(smem_u32(&bar_tempty[buf]));
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc<C::kTmemCols>(tmem_base);
}

template <int kBN, bool kSwap, bool kGated, typename OutT>
cudaError_t launch_cfg(const GemmArgs& a) {
  using C = Cfg<kBN>;
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
  p.xscale = a.xscale;
  p.xsum = a.xsum;
  p.wscale = a.wscale;
  p.wsum = a.wsum;
  p.bias = a.bias;
  p.y = a.y;
  p.acc = a.acc;
  p.M = a.M;
  p.N = a.N;
  p.ldy = a.gated ? a.N / 2 : a.N;
  const int tiles = ((p.rows_a + kBM - 1) / kBM) * ((p.rows_b + kBN - 1) / kBN);
  const int grid = tiles < a.num_sms ? tiles : a.num_sms;
  if (grid == 0) return cudaSuccess;
  auto kern = gemm_w4a4_kernel<kBN, kSwap, kGated, OutT>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess) return e;
  kern<<<grid, kThreads, C::kSmem, a.stream>>>(p);
  return cudaGetLastError();
}

template <typename OutT>
cudaError_t launch_out(const GemmArgs& a) {
  if (a.gated) return launch_cfg<256, false, true, OutT>(a);  // gate/up pairs share a 256-row tile
  if (a.M > 128) return launch_cfg<256, false, false, OutT>(a);
  const int mpad = (a.M + 15) / 16 * 16;
  if (mpad <= 16) return launch_cfg<16, true, false, OutT>(a);
  if (mpad <= 32) return launch_cfg<32, true, false, OutT>(a);
  if (mpad <= 64) return launch_cfg<64, true, false, OutT>(a);
  return launch_cfg<128, true, false, OutT>(a);
}

}  // namespace

cudaError_t launch_gemm_w4a4(const GemmArgs& a) {
  if (a.M == 0) return cudaSuccess;
  return a.ydt == 0 ? launch_out<__half>(a) : launch_out<__nv_bfloat16>(a);
}

cudaError_t read_and_clear_error_word(unsigned int* out, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(out, g_error_word, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_error_word, &zero, sizeof(unsigned int));
}

}  // namespace qvla
