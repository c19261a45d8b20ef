// Rotate + quantise in passes: the online rotation and activation quantisation (Sec. 4.1 Eq. 3-5,
// Sec. 4.2 Eq. 5-6) of a few rows of 16-bit activations into the GEMM's operand bytes, one CTA per
// 2048-channel pass of a row.
//
// The row-per-warp kernel of rotate_quant.cuh gives each thread 64 channels, so a thread's chain
// of dependent work is long; with a few rows that chain is the whole kernel.  Here a pass of
// C channels (C the largest power of two up to 2048 dividing K, holding whole Hadamard blocks) is
// spread over 256 threads, 8 channels each: the butterflies on index bits 0-2 run in registers,
// on bits 3-7 across the lanes, and after one transpose through shared memory thread t holds the
// channels t + 256 w (w < 8) and runs bits 8-10.  The stage order and every rounding are those of
// the row-per-warp kernel (stages in increasing index-bit order, each sum and difference rounded
// once), and so are the scale and the codes (its fast path, tie band and exact rule, value by
// value), so the outputs are the same bits.  The P = K / C passes of a row form a cluster: with
// per-token scales each CTA sends its pass's largest |value| to every CTA of the cluster
// (st.async completing on an mbarrier, a bounded wait) and all take the row's maximum; each
// sends its code sum to the first CTA, which writes the row's scale and sum.  The operand bytes
// (code q as the byte q + 8, each group of 8 channels stored k0 k2 k4 k6 k1 k3 k5 k7) are staged
// in shared memory and leave in 16-byte stores.
#include "rotate_quant.cuh"
#include "ptx.cuh"

namespace qvla {
namespace {

constexpr int kRqpThreads = 256;
// test hook (qvla_debug.h): nonzero, the CTAs of a cluster send each other nothing, so every
// receiving wait runs out
static __device__ int g_rqp_hold;
constexpr int kRqpMaxPasses = 8;  // a cluster of at most 8 CTAs (K <= 16384)
constexpr int kRqpMaxRows = 64;   // the rows it takes (more rows go to the row-per-warp kernel)

struct RqpParams {
  const void* x;            // [M][K] activations
  uint8_t* xq;              // [M][K] operand bytes
  float* xscale;            // [M]
  int32_t* xsum;            // [M] or null
  const float* step_scale;  // per-step mode: the step's scale
  int32_t* zero;            // ints set to 0 once x has been waited for, or null
  int zero_n;
  int M, K, C, P, log_b;
  float inv_sqrt_b;
};

template <typename XT, bool kStep>
__global__ void __launch_bounds__(kRqpThreads) rotate_quant_pass_kernel(RqpParams p) {
  extern __shared__ __align__(16) uint8_t smem[];
  __shared__ uint32_t s_wmax[kRqpThreads / 32], s_wsum[kRqpThreads / 32];
  __shared__ uint32_t s_maxes[kRqpMaxPasses], s_sums[kRqpMaxPasses];  // received from the cluster
  __shared__ __align__(8) uint64_t bar_max, bar_sum;
  const int C = p.C, P = p.P, lb = p.log_b;
  float* const s_rot = reinterpret_cast<float*>(smem);  // [C] the pass, for the transpose
  uint8_t* const s_out = smem + 4 * C;                  // [C] its operand bytes
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int m = static_cast<int>(blockIdx.x) / P, rank = static_cast<int>(blockIdx.x) % P;
  const bool exch_max = !kStep && P > 1;
  const bool hold = P > 1 && *const_cast<volatile int*>(&g_rqp_hold) != 0;
  if (P > 1) {
    // the cluster barrier completed before the first send guarantees every receiver's barrier
    if (t == 0) {
      mbar_init(smem_u32(&bar_max), 1);
      mbar_init(smem_u32(&bar_sum), 1);
      mbar_init_fence();
      if (exch_max) mbar_arrive_expect_tx(smem_u32(&bar_max), static_cast<uint32_t>(4 * P));
      if (rank == 0) mbar_arrive_expect_tx(smem_u32(&bar_sum), static_cast<uint32_t>(4 * P));
    }
    cluster_arrive_relaxed();
  }
  griddep_wait();  // x comes from the previous kernel, which may still read xq / xscale / xsum
  griddep_launch_dependents();
  if (p.zero != nullptr && blockIdx.x == 0)  // the next GEMM's work-unit counters
    for (int i = threadIdx.x; i < p.zero_n; i += kRqpThreads) p.zero[i] = 0;

  float2 v[4];
  const bool holds = 8 * t < C;  // the thread holds channels 8 t .. 8 t + 7 of the pass
  if (holds) {
    rq::Loader<XT>::load(static_cast<const XT*>(p.x) + static_cast<size_t>(m) * p.K + static_cast<size_t>(rank) * C + 8 * t,
                         v);
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = make_float2(0.0f, 0.0f);
  }
  if (lb > 0) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float a = v[i].x, d = v[i].y;
      v[i] = make_float2(a + d, a - d);
    }
  }
  if (lb > 1) {
    rq::bfly2(v[0], v[1]);
    rq::bfly2(v[2], v[3]);
  }
  if (lb > 2) {
    rq::bfly2(v[0], v[2]);
    rq::bfly2(v[1], v[3]);
  }
#pragma unroll
  for (int bit = 3; bit < 8; ++bit) {
    if (bit < lb) {  // the lower lane of a pair keeps a + d, the upper one a - d
      const int mask = 1 << (bit - 3);
      const float sg = (lane & mask) ? -1.0f : 1.0f;
      const float2 sg2 = make_float2(sg, sg);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float2 pv;
        pv.x = __shfl_xor_sync(0xffffffffu, v[i].x, mask);
        pv.y = __shfl_xor_sync(0xffffffffu, v[i].y, mask);
        v[i] = __ffma2_rn(v[i], sg2, pv);
      }
    }
  }
  if (holds) {
    reinterpret_cast<float4*>(s_rot)[2 * t] = make_float4(v[0].x, v[0].y, v[1].x, v[1].y);
    reinterpret_cast<float4*>(s_rot)[2 * t + 1] = make_float4(v[2].x, v[2].y, v[3].x, v[3].y);
  }
  __syncthreads();
  float yv[8];
#pragma unroll
  for (int w = 0; w < 8; ++w) yv[w] = t + 256 * w < C ? s_rot[t + 256 * w] : 0.0f;
#pragma unroll
  for (int bit = 8; bit < 11; ++bit) {
    if (bit < lb) {
      const int h = 1 << (bit - 8);
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        if ((w & h) == 0) {
          const float a = yv[w], d = yv[w + h];
          yv[w] = a + d;
          yv[w + h] = a - d;
        }
      }
    }
  }

  // the pass's largest |value| (non-negative floats order as their bit patterns), then the row's
  const float mx = fmaxf(fmaxf(fmaxf(fabsf(yv[0]), fabsf(yv[1])), fmaxf(fabsf(yv[2]), fabsf(yv[3]))),
                         fmaxf(fmaxf(fabsf(yv[4]), fabsf(yv[5])), fmaxf(fabsf(yv[6]), fabsf(yv[7]))));
  const uint32_t wmax = __reduce_max_sync(0xffffffffu, __float_as_uint(mx));
  if (lane == 0) s_wmax[warp] = wmax;
  __syncthreads();
  uint32_t cmax = 0u;
#pragma unroll
  for (int i = 0; i < kRqpThreads / 32; ++i) cmax = max(cmax, s_wmax[i]);
  bool ok = true;
  if (P > 1) cluster_wait();  // pairs with the arrive at set-up
  if (exch_max) {
    if (t < P && !hold)
      st_async_u32(mapa_shared(smem_u32(&s_maxes[rank]), static_cast<uint32_t>(t)), cmax,
                   mapa_shared(smem_u32(&bar_max), static_cast<uint32_t>(t)));
    ok = mbar_wait_cluster(smem_u32(&bar_max), 0);
    cmax = 0u;
    for (int src = 0; src < P; ++src) cmax = max(cmax, s_maxes[src]);
  }
  // the scale: the step's, or max |Z| of the normalised rotation over the row over q_max = 7
  const float delta = kStep ? __ldg(p.step_scale) : __fdiv_rn(__uint_as_float(cmax) * p.inv_sqrt_b, 7.0f);
  const float cr = p.inv_sqrt_b * (delta > 0.0f ? __fdiv_rn(1.0f, delta) : 0.0f);  // infinite iff 1 / delta overflows

  // codes: operand byte q + 8 of channel e at byte 8 (e / 8) + j, j = i / 2 for the even i = e % 8
  // and 4 + i / 2 for the odd
  uint32_t qs = 0u;
#pragma unroll
  for (int w = 0; w < 8; ++w) {
    const int e = t + 256 * w;
    if (e < C) {
      const float y = yv[w];
      float tt = __fmul_rn(y, cr);  // rounded on its own, as the row-per-warp kernel's packed multiply
      if (kStep) tt = fminf(fmaxf(tt, -7.0f), 7.0f);
      float u = __fadd_rn(tt, rq::kMagic);
      const float d = __fmaf_rn(__fadd_rn(u, -rq::kMagic), -1.0f, tt);
      if (fabsf(d) >= rq::kTieBand || isinf(cr)) u = rq::exact_code(y, p.inv_sqrt_b, delta, cr, 7.0f, rq::kTieBand);
      const uint32_t q8 = (__float_as_uint(u) & 0xFu) ^ 0x8u;
      const int i = e & 7;
      s_out[(e & ~7) + ((i & 1) ? 4 + (i >> 1) : (i >> 1))] = static_cast<uint8_t>(q8);
      qs += q8;
    }
  }
  const uint32_t wsum = __reduce_add_sync(0xffffffffu, qs);
  if (lane == 0) s_wsum[warp] = wsum;
  __syncthreads();
  uint8_t* const dst = p.xq + static_cast<size_t>(m) * p.K + static_cast<size_t>(rank) * C;
  for (int i = t; i < C / 16; i += kRqpThreads) reinterpret_cast<uint4*>(dst)[i] = reinterpret_cast<const uint4*>(s_out)[i];

  // the row's code sum (of q + 8 over K channels) at the first CTA of the cluster
  uint32_t csum = 0u;
#pragma unroll
  for (int i = 0; i < kRqpThreads / 32; ++i) csum += s_wsum[i];
  if (P > 1) {
    if (t == 0 && !hold)
      st_async_u32(mapa_shared(smem_u32(&s_sums[rank]), 0u), csum, mapa_shared(smem_u32(&bar_sum), 0u));
    if (rank == 0) {
      ok = mbar_wait_cluster(smem_u32(&bar_sum), 0) && ok;
      csum = 0u;
      for (int src = 0; src < P; ++src) csum += s_sums[src];
    }
  }
  (void)ok;  // a wait that ran out has recorded QVLA_ERR_TIMEOUT; the outputs are then not defined
  if (rank == 0 && t == 0) {
    p.xscale[m] = delta;
    if (p.xsum) p.xsum[m] = static_cast<int32_t>(csum - 8u * static_cast<uint32_t>(p.K));
  }
}

template <typename XT, bool kStep>
cudaError_t launch_rqp(const RotQuantArgs& a, const RqpParams& p) {
  auto kern = rotate_quant_pass_kernel<XT, kStep>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(p.M) * static_cast<unsigned>(p.P));
  cfg.blockDim = dim3(kRqpThreads);
  cfg.dynamicSmemBytes = 5 * static_cast<size_t>(p.C);
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // may overlap the previous kernel
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = static_cast<unsigned>(p.P);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.P > 1 ? 2 : 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_rotate_quant_pass(const RotQuantArgs& a, bool* launched) {
  *launched = false;
  // 16-bit activations into 4-bit operand bytes, one scale per row (per token or per step), for
  // up to 64 rows: there the latency of one row decides, and a pass's 256 threads cut it
  // (measured, one call: 1 x 2048 6.8 against 8.8 us, 4 x 16384 8.8 against 10.9 us; the DiT
  // step at 50 tokens 691 -> 647 us).  At hundreds of rows the row-per-warp kernel's cheaper
  // stages per element win (816 x 16384: 27.3 against 41.6 us).
  if (a.out_mode != 1 || (a.mode != 0 && a.mode != 1) || (a.xdt != 0 && a.xdt != 1) || a.gshift < 30 ||
      a.xgsum != nullptr || a.M < 1 || a.M > kRqpMaxRows)
    return cudaSuccess;
  int C = 2048;
  while (a.K % C != 0) C /= 2;
  const int P = a.K / C;
  if (a.log_b < 0 || (1 << a.log_b) > C || P > kRqpMaxPasses || C < 128) return cudaSuccess;
  RqpParams p;
  p.x = a.x;
  p.xq = a.xq;
  p.xscale = a.xscale;
  p.xsum = a.xsum;
  p.step_scale = a.step_scale;
  p.zero = a.zero;
  p.zero_n = a.zero_n;
  p.M = a.M;
  p.K = a.K;
  p.C = C;
  p.P = P;
  p.log_b = a.log_b;
  p.inv_sqrt_b = a.inv_sqrt_b;
  cudaError_t e;
  if (a.xdt == 0)
    e = a.mode == 1 ? launch_rqp<__half, true>(a, p) : launch_rqp<__half, false>(a, p);
  else
    e = a.mode == 1 ? launch_rqp<__nv_bfloat16, true>(a, p) : launch_rqp<__nv_bfloat16, false>(a, p);
  *launched = e == cudaSuccess;
  return e;
}

cudaError_t read_and_clear_error_word_rqp(unsigned int* out, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(out, g_error_word, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_error_word, &zero, sizeof(unsigned int));
}

cudaError_t set_debug_hooks_rqp(unsigned long long wait_limit_ns, int hold) {
  const unsigned long long v = wait_limit_ns ? wait_limit_ns : kWaitLimitNs;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return e;
  e = cudaMemcpyToSymbol(g_wait_limit_ns, &v, sizeof(v));
  if (e != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_rqp_hold, &hold, sizeof(hold));
}

}  // namespace qvla
