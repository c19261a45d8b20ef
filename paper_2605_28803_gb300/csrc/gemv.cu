// Decode-sized batches (M <= 4 tokens): the W4A4 linear's integer product and dequantisation
// (Sec. 4.2, Eq. 7) as a GEMV on the CUDA cores.
//
// At one to four tokens the linear reads about two integer operations' worth of work per packed
// weight byte, so it is bound by the weight stream alone.  The tensor-core GEMM stages its
// weights through the bulk-copy engine, whose DRAM-side rate per SM stays near 25 GB/s however
// many copies are in flight; vector loads from many threads with more bytes in flight stream
// faster.  Here every SM streams its share of the weights with coalesced 16-byte loads (the first
// ones issued before waiting for the previous kernel), unpacks the codes to offset-binary bytes
// q + 8 and multiplies them with the activations' operand bytes (or packed codes) by dp4a:
//   S[n, m] = sum_k (q_w[n,k] + 8)(q_x[m,k] + 8)             (exact, unsigned 32-bit)
//   acc     = S - 8 sum_k q_x[m,k] - 8 sum_k q_w[n,k] - 64 K  (as the tensor-core path)
// and the epilogue is the tensor-core path's, operation for operation, so the outputs are the
// same bits.  K is split over a cluster of up to 8 CTAs; the partial sums meet in shared memory
// across the cluster (distributed shared memory) and each CTA finishes a slice of the rows.
//
// Work of a CTA: one 128-row weight group (a gated layer: the gate group and the up group of
// 128 hidden units) over its k-range.  Warp w takes the 32-row slice w % 4 and every other
// k-block (w / 4 picks which); lane l loads the 16-byte quarter l % 4 of rows 8 t + l / 4
// (t = 0..3) of the slice, so each load instruction reads 512 contiguous bytes of the layer's
// tiled weights.  The four lanes that share a row add their sums by shuffles at the end.
#include "gemm_kernel.cuh"

namespace qvla {
namespace {

constexpr int kGvThreads = 256;  // 8 warps: 4 row slices x 2 k-block phases
constexpr int kGemvActMax = 96 * 1024;  // shared memory for a CTA's activation bytes
constexpr int kGvPhases = kGvThreads / 32 / 4;

// k-blocks of weight loads a warp keeps in flight: 64 KB per CTA at one token, 32 KB where the
// accumulators of more tokens (or of a gated layer's two groups) need the registers
template <int kM, bool kGated>
__host__ __device__ constexpr int gv_ring() {
  return kM == 1 ? (kGated ? 2 : 4) : 2;
}

// Four bytes into the shared memory of a CTA of the cluster, completing 4 bytes of the
// transaction count of that CTA's mbarrier (addresses from mapa_shared).
__device__ __forceinline__ void st_async_u32(uint32_t cluster_addr, uint32_t v, uint32_t cluster_bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(cluster_addr), "r"(v),
               "r"(cluster_bar)
               : "memory");
}

struct GvParams {
  const uint8_t* wq;      // tiled weights [groups][K/128][128][64 B]
  const uint8_t* xq;      // activations: operand bytes [M][K] (kXB 1) or packed nibbles [M][K/2] (kXB 0)
  const float* xscale;    // [M]
  const int32_t* xsum;    // [M]
  const float* wscale;    // [N]
  const float* wcorr;     // [N] 8 * sum_k q_w
  const float* bias;      // [N]
  void* y;
  int32_t* acc;           // [M][N] or null
  int M, N, K, ldy, nkb, splits;
  float kconst;           // 64 K
};

// The offset-binary bytes q + 8 of a packed word's 8 codes: lo = codes 0, 2, 4, 6, hi = 1, 3, 5, 7
// (the order in which the rotate-quantise kernel writes its operand bytes).
__device__ __forceinline__ void unpack8(uint32_t w, uint32_t& lo, uint32_t& hi) { int4x8_to_e4m3_offset(w, lo, hi); }

template <int kM, bool kGated, int kXB, typename OutT>
__global__ void __launch_bounds__(kGvThreads) gemv_w4a4_kernel(GvParams p) {
  constexpr int kParts = kGated ? 2 : 1;  // 128-row weight groups per CTA
  constexpr int kGvRing = gv_ring<kM, kGated>();
  constexpr int kActKb = kXB == 1 ? kBK : kBK / 2;  // activation bytes per token and k-block
  __shared__ uint32_t s_part[kParts][128][kM];
  // split K: the slices of this CTA's rows from every CTA of the cluster, [source][row][part][m]
  __shared__ uint32_t s_recv[128 * kParts * kM];
  __shared__ __align__(8) uint64_t bar_recv;
  extern __shared__ __align__(16) uint8_t s_act[];  // [kM][k-range] activation bytes of this CTA

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = p.splits;
  const int unit = static_cast<int>(blockIdx.x) / S;
  const int rank = static_cast<int>(blockIdx.x) % S;  // the CTA's rank in its cluster of S
  const int kb0 = p.nkb * rank / S, kb1 = p.nkb * (rank + 1) / S;
  const int slice = warp & 3, kpar = warp >> 2;  // kpar in [0, kGvPhases)
  const int q = lane & 3;
  const int R = 128 / S;  // rows this CTA finishes: [rank R, (rank + 1) R)

  for (int i = threadIdx.x; i < kParts * 128 * kM; i += kGvThreads) (&s_part[0][0][0])[i] = 0u;
  if (S > 1) {
    // every CTA of the cluster sends this one its partials of these rows; the cluster barrier
    // completed before the first send guarantees every receiver's barrier exists
    if (threadIdx.x == 0) {
      mbar_init(smem_u32(&bar_recv), 1);
      mbar_init_fence();
      mbar_arrive_expect_tx(smem_u32(&bar_recv), static_cast<uint32_t>(S * R * kParts * kM * 4));
    }
    cluster_arrive_relaxed();
  }

  // weights of one k-block for this lane: kParts x 4 rows x one 16-byte quarter
  auto load_w = [&](int kb, uint4 (&w)[kParts][4]) {
#pragma unroll
    for (int part = 0; part < kParts; ++part) {
      const int g = kGated ? 2 * unit + part : unit;
      const uint4* chunk = reinterpret_cast<const uint4*>(p.wq + (static_cast<size_t>(g) * p.nkb + kb) * 8192);
#pragma unroll
      for (int t = 0; t < 4; ++t) w[part][t] = __ldg(chunk + slice * 128 + t * 32 + lane);
    }
  };

  uint4 ring[kGvRing][kParts][4];
#pragma unroll
  for (int i = 0; i < kGvRing; ++i) {
    const int kb = kb0 + kpar + kGvPhases * i;
    if (kb < kb1) load_w(kb, ring[i]);  // the weights no earlier kernel writes: before the wait
  }
  griddep_wait();  // the activations, their scales and sums come from the previous kernel
  if (threadIdx.x == 0) griddep_launch_dependents();
  // the epilogue's parameters of this thread's (row, token) entries, fetched while the weights stream
  constexpr int kEnt = (128 * kM + kGvThreads - 1) / kGvThreads;
  float e_cm[kEnt], e_xs[kEnt], e_wc[kEnt][kParts], e_ws[kEnt][kParts], e_bs[kEnt][kParts];
#pragma unroll
  for (int u = 0; u < kEnt; ++u) {
    const int e = threadIdx.x + u * kGvThreads;
    const int row = rank * R + min(e, R * kM - 1) / kM, m = min(e % kM, p.M - 1);
    e_cm[u] = 8.0f * static_cast<float>(p.xsum[m]) + p.kconst;
    e_xs[u] = p.xscale[m];
#pragma unroll
    for (int part = 0; part < kParts; ++part) {
      const int n = kGated ? 2 * unit * 128 + part * 128 + row : min(unit * 128 + row, p.N - 1);
      e_wc[u][part] = __ldg(p.wcorr + n);
      e_ws[u][part] = __ldg(p.wscale + n);
      e_bs[u][part] = __ldg(p.bias + n);
    }
  }
  {  // this CTA's k-range of every token's activation bytes, once, into shared memory
    const int row16 = (kb1 - kb0) * kActKb / 16;  // 16-byte pieces per token
    for (int i = threadIdx.x; i < p.M * row16; i += kGvThreads) {
      const int m = i / row16, c = i % row16;
      reinterpret_cast<uint4*>(s_act)[m * row16 + c] = __ldg(reinterpret_cast<const uint4*>(
          p.xq + static_cast<size_t>(m) * (p.K / (kBK / kActKb)) + kb0 * kActKb) + c);
    }
  }
  __syncthreads();

  uint32_t acc[kParts][4][kM];
#pragma unroll
  for (int part = 0; part < kParts; ++part)
#pragma unroll
    for (int t = 0; t < 4; ++t)
#pragma unroll
      for (int m = 0; m < kM; ++m) acc[part][t][m] = 0u;

  for (int base = 0;; base += kGvRing) {
#pragma unroll
    for (int i = 0; i < kGvRing; ++i) {
      const int kb = kb0 + kpar + kGvPhases * (base + i);
      if (kb < kb1) {
        // the activation bytes of this quarter of the k-block, every token: lo / hi per 8 codes
        uint32_t alo[kM][4], ahi[kM][4];
#pragma unroll
        for (int m = 0; m < kM; ++m) {
          if (m < p.M) {
            const uint8_t* arow = s_act + (static_cast<size_t>(m) * (kb1 - kb0) + (kb - kb0)) * kActKb;
            if constexpr (kXB == 1) {
              const uint4* src = reinterpret_cast<const uint4*>(arow + q * 32);
              const uint4 v0 = src[0], v1 = src[1];
              alo[m][0] = v0.x; ahi[m][0] = v0.y; alo[m][1] = v0.z; ahi[m][1] = v0.w;
              alo[m][2] = v1.x; ahi[m][2] = v1.y; alo[m][3] = v1.z; ahi[m][3] = v1.w;
            } else {
              const uint4 v = *reinterpret_cast<const uint4*>(arow + q * 16);
              unpack8(v.x, alo[m][0], ahi[m][0]);
              unpack8(v.y, alo[m][1], ahi[m][1]);
              unpack8(v.z, alo[m][2], ahi[m][2]);
              unpack8(v.w, alo[m][3], ahi[m][3]);
            }
          } else {
#pragma unroll
            for (int j = 0; j < 4; ++j) alo[m][j] = ahi[m][j] = 0u;
          }
        }
#pragma unroll
        for (int part = 0; part < kParts; ++part) {
#pragma unroll
          for (int t = 0; t < 4; ++t) {
            const uint32_t wv[4] = {ring[i][part][t].x, ring[i][part][t].y, ring[i][part][t].z, ring[i][part][t].w};
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              uint32_t lo, hi;
              unpack8(wv[j], lo, hi);
#pragma unroll
              for (int m = 0; m < kM; ++m) acc[part][t][m] = __dp4a(hi, ahi[m][j], __dp4a(lo, alo[m][j], acc[part][t][m]));
            }
          }
        }
        const int kbn = kb + kGvPhases * kGvRing;
        if (kbn < kb1) load_w(kbn, ring[i]);
      }
    }
    if (kb0 + kpar + kGvPhases * (base + kGvRing) >= kb1) break;
  }

  // the four lanes of a row add up, then the warps of a slice meet in shared memory
#pragma unroll
  for (int part = 0; part < kParts; ++part)
#pragma unroll
    for (int t = 0; t < 4; ++t)
#pragma unroll
      for (int m = 0; m < kM; ++m) {
        uint32_t v = acc[part][t][m];
        v += __shfl_xor_sync(0xffffffffu, v, 1);
        v += __shfl_xor_sync(0xffffffffu, v, 2);
        acc[part][t][m] = v;
      }
  if (q == 0) {
#pragma unroll
    for (int part = 0; part < kParts; ++part)
#pragma unroll
      for (int t = 0; t < 4; ++t)
#pragma unroll
        for (int m = 0; m < kM; ++m) atomicAdd(&s_part[part][slice * 32 + 8 * t + lane / 4][m], acc[part][t][m]);
  }
  __syncthreads();
  bool landed = true;
  if (S > 1) {
    cluster_wait();  // pairs with the arrive at set-up: every receive barrier is initialised
    // each partial goes to the CTA that finishes its row, as an asynchronous store completing on
    // that CTA's barrier; no CTA reads another's shared memory, so none waits for the others to leave
    for (int i = threadIdx.x; i < 128 * kParts * kM; i += kGvThreads) {
      const int row = i / (kParts * kM), part = (i / kM) % kParts, m = i % kM;
      const int d = row / R;
      const uint32_t dst = smem_u32(&s_recv[((rank * R + (row - d * R)) * kParts + part) * kM + m]);
      st_async_u32(mapa_shared(dst, static_cast<uint32_t>(d)), s_part[part][row][m],
                   mapa_shared(smem_u32(&bar_recv), static_cast<uint32_t>(d)));
    }
    landed = mbar_wait_cluster(smem_u32(&bar_recv), 0);
  }

  // rank r finishes rows [r R, (r + 1) R) of the group(s), adding every rank's partial
#pragma unroll
  for (int u = 0; u < kEnt; ++u) {
    const int e = threadIdx.x + u * kGvThreads;
    if (!landed || e >= R * kM) continue;
    const int rr = e / kM, row = rank * R + rr, m = e % kM;
    if (m >= p.M) continue;
    uint32_t sum[kParts];
#pragma unroll
    for (int part = 0; part < kParts; ++part) {
      if (S > 1) {
        sum[part] = 0u;
        for (int src = 0; src < S; ++src) sum[part] += s_recv[((src * R + rr) * kParts + part) * kM + m];
      } else {
        sum[part] = s_part[part][row][m];
      }
    }
    // the epilogue of the tensor-core path: exact accumulator, one float32 scale product, fma, one rounding
    if constexpr (!kGated) {
      const int n = unit * 128 + row;
      if (n < p.N) {
        const float a = static_cast<float>(sum[0]) - (e_cm[u] + e_wc[u][0]);
        reinterpret_cast<OutT*>(p.y)[static_cast<size_t>(m) * p.ldy + n] = to_out<OutT>(fmaf(a, e_xs[u] * e_ws[u][0], e_bs[u][0]));
        if (p.acc) p.acc[static_cast<size_t>(m) * p.N + n] = static_cast<int32_t>(a);
      }
    } else {
      // weight rows 256 unit + row (gate) and + 128 (up) of hidden unit j; h = gelu(gate) * up
      const int H = p.N / 2, j = unit * 128 + row;
      if (j < H) {
        const float ag = static_cast<float>(sum[0]) - (e_cm[u] + e_wc[u][0]);
        const float au = static_cast<float>(sum[1]) - (e_cm[u] + e_wc[u][1]);
        const float2 gu = unpack2<OutT>(pack2<OutT>(fmaf(ag, e_xs[u] * e_ws[u][0], e_bs[u][0]),
                                                    fmaf(au, e_xs[u] * e_ws[u][1], e_bs[u][1])));
        reinterpret_cast<OutT*>(p.y)[static_cast<size_t>(m) * p.ldy + j] = to_out<OutT>(gelu_tanh(gu.x) * gu.y);
        if (p.acc) {
          p.acc[static_cast<size_t>(m) * p.N + j] = static_cast<int32_t>(ag);
          p.acc[static_cast<size_t>(m) * p.N + H + j] = static_cast<int32_t>(au);
        }
      }
    }
  }
}

template <int kM, bool kGated, int kXB, typename OutT>
cudaError_t launch_gv(const GemmArgs& a, GvParams p, int units) {
  auto kern = gemv_w4a4_kernel<kM, kGated, kXB, OutT>;
  // the largest k-range of a CTA, for every token
  const size_t act = static_cast<size_t>(kM) * ((p.nkb + p.splits - 1) / p.splits) * (kXB == 1 ? kBK : kBK / 2);
  if (act > static_cast<size_t>(kGemvActMax)) return kNotApplicable;
  if (act > 48 * 1024) {
    cudaError_t e = prepare_kernel(reinterpret_cast<const void*>(kern), kGemvActMax);
    if (e != cudaSuccess) return e == kNotApplicable ? cudaErrorUnknown : e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(kGvThreads);
  cfg.gridDim = dim3(units * p.splits);
  cfg.dynamicSmemBytes = act;
  cfg.stream = a.stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = static_cast<unsigned>(p.splits);
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = p.splits > 1 ? 2 : 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, kern, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <bool kGated, int kXB, typename OutT>
cudaError_t launch_gv_m(const GemmArgs& a, const GvParams& p, int units) {
  if (a.M == 1) return launch_gv<1, kGated, kXB, OutT>(a, p, units);
  if (a.M == 2) return launch_gv<2, kGated, kXB, OutT>(a, p, units);
  return launch_gv<4, kGated, kXB, OutT>(a, p, units);
}

template <int kXB, typename OutT>
cudaError_t launch_gv_g(const GemmArgs& a, const GvParams& p, int units) {
  return a.gated ? launch_gv_m<true, kXB, OutT>(a, p, units) : launch_gv_m<false, kXB, OutT>(a, p, units);
}

}  // namespace

cudaError_t read_and_clear_error_word_gemv(unsigned int* out, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(out, g_error_word, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_error_word, &zero, sizeof(unsigned int));
}

cudaError_t set_debug_hooks_gemv(unsigned long long wait_limit_ns, int hold_loads) {
  return set_debug_hooks(wait_limit_ns, hold_loads);
}

cudaError_t launch_gemv_w4a4(const GemmArgs& a, bool* launched) {
  *launched = false;
  if (a.M < 1 || a.M > kGemvMaxM || a.gscale || (a.x_bytes != 0 && a.x_bytes != 1)) return cudaSuccess;
  GvParams p;
  p.wq = a.wq;
  p.xq = a.xq;
  p.xscale = a.xscale;
  p.xsum = a.xsum;
  p.wscale = a.wscale;
  p.wcorr = a.wcorr;
  p.bias = a.bias;
  p.y = a.y;
  p.acc = a.acc;
  p.M = a.M;
  p.N = a.N;
  p.K = a.K;
  p.ldy = a.gated ? a.N / 2 : a.N;
  p.nkb = a.K / kBK;
  p.kconst = 64.0f * static_cast<float>(a.K);
  // one CTA per 128-row group (gated: per 128 hidden units, gate and up), K split over a cluster
  // of up to 8 until the grid holds about two CTAs per SM
  const int units = a.gated ? a.N / 256 : (a.N + 127) / 128;
  int splits = 1;
  while (splits < 8 && 2 * splits <= p.nkb && units * splits < 2 * a.num_sms) splits *= 2;
  p.splits = splits;
  cudaError_t e = a.x_bytes == 1 ? (a.ydt == 0 ? launch_gv_g<1, __half>(a, p, units) : launch_gv_g<1, __nv_bfloat16>(a, p, units))
                                 : (a.ydt == 0 ? launch_gv_g<0, __half>(a, p, units) : launch_gv_g<0, __nv_bfloat16>(a, p, units));
  if (e == kNotApplicable) return cudaSuccess;  // the activations of a CTA would not fit
  *launched = e == cudaSuccess;
  return e;
}

}  // namespace qvla
