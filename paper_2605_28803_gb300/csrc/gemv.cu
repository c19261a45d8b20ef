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
// accumulators of more tokens (or of a gated layer's two groups) need the registers.  The
// one-launch linear (kXB 2, one token) runs about one CTA per SM or fewer, whose registers allow
// a gated layer 96 KB.
template <int kM, bool kGated, int kXB>
__host__ __device__ constexpr int gv_ring() {
  return kM == 1 ? (kGated ? (kXB == 2 ? 6 : 2) : 4) : 2;
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
  // kXB 2 (M = 1): the raw activations [1][K] (the output's dtype), rotated and quantised in the
  // kernel in passes of C channels (a power of two, C | K, b <= C <= 2048); xscale then holds the
  // step's scale, or is null for a per-token scale, and xsum is unused
  const void* x;
  int log_b, C;
  float inv_sqrt_b;
};

// The offset-binary bytes q + 8 of a packed word's 8 codes: lo = codes 0, 2, 4, 6, hi = 1, 3, 5, 7
// (the order in which the rotate-quantise kernel writes its operand bytes).
__device__ __forceinline__ void unpack8(uint32_t w, uint32_t& lo, uint32_t& hi) { int4x8_to_e4m3_offset(w, lo, hi); }

// kXB 2: the online rotation and the activation quantisation (Sec. 4.1 Eq. 3-5, Sec. 4.2 Eq. 5-6)
// of one token's k-range [kb0, kb1) x 128 in this CTA, into operand bytes in s_act.  Each of the
// (at most kGvPasses) passes rotates the C channels containing part of the range with the
// rotate-quantise kernel's arithmetic stage for stage (butterflies in increasing index-bit order,
// every sum and difference rounded once), so the rotated values, the scale and the codes are the
// same bits as that kernel's: thread t loads channels 8 t .. 8 t + 7 of the pass and runs the
// stages on index bits 0-2 in registers and 3-7 across the lanes; a transpose through shared
// memory then gives thread t the channels t + 256 w (w < 8), which take the stages on bits 8-10
// and stay in its registers.  The per-token scale
// takes the largest |value| of the row: where one pass is the whole row (K = C) every CTA has it;
// otherwise, with K split over a cluster, every CTA sends its range's maximum to every other one.
// Each thread then turns its values of the range into codes (the rotate-quantise kernel's fast
// path, tie band and exact decision, value by value) and stores their operand bytes.  Returns
// the scale in *delta_out, the sum of the range's offset codes q + 8 in s_wsum (one partial per
// warp), and false if a wait timed out.
constexpr int kGvPasses = 2;
template <typename XT>
__device__ __forceinline__ bool rotate_quantize_token(const GvParams& p, const XT* __restrict__ x, int kb0, int kb1,
                                                      int rank, bool max_exchange, uint8_t* s_act, uint32_t* s_wmax,
                                                      uint32_t* s_maxes, uint32_t* s_wsum, uint32_t bar_max,
                                                      bool hold, float* delta_out) {
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const int k0 = kb0 * kBK, range = (kb1 - kb0) * kBK;
  const int rmax = (p.nkb + p.splits - 1) / p.splits * kBK;  // the largest k-range of the cluster
  const int C = p.C, lb = p.log_b;
  float* const s_rot = reinterpret_cast<float*>(s_act + rmax);  // [C]
  const bool whole_row = p.K == C;
  const int c0 = k0 / C, passes = (k0 + range + C - 1) / C - c0;
  bool ok = true;
  float yv[kGvPasses][8];
  float mx = 0.0f;
#pragma unroll
  for (int ps = 0; ps < kGvPasses; ++ps) {
    if (ps >= passes) break;
    const int c = c0 + ps;
    float2 v[4];
    if (8 * t < C) {
      rq::Loader<XT>::load(x + static_cast<size_t>(c) * C + 8 * t, v);
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
    if (ps > 0) __syncthreads();  // the previous pass has read s_rot
    if (8 * t < C) {
      reinterpret_cast<float4*>(s_rot)[2 * t] = make_float4(v[0].x, v[0].y, v[1].x, v[1].y);
      reinterpret_cast<float4*>(s_rot)[2 * t + 1] = make_float4(v[2].x, v[2].y, v[3].x, v[3].y);
    }
    __syncthreads();
    float* const yp = yv[ps];
#pragma unroll
    for (int w = 0; w < 8; ++w) yp[w] = t + 256 * w < C ? s_rot[t + 256 * w] : 0.0f;
#pragma unroll
    for (int bit = 8; bit < 11; ++bit) {
      if (bit < lb) {
        const int h = 1 << (bit - 8);
#pragma unroll
        for (int w = 0; w < 8; ++w) {
          if ((w & h) == 0) {
            const float a = yp[w], d = yp[w + h];
            yp[w] = a + d;
            yp[w + h] = a - d;
          }
        }
      }
    }
    float m8[8];  // |values| that count towards the maximum, reduced as a tree
#pragma unroll
    for (int w = 0; w < 8; ++w) {
      const int e = t + 256 * w, kk = c * C + e - k0;
      m8[w] = (e < C && (whole_row || (kk >= 0 && kk < range))) ? fabsf(yp[w]) : 0.0f;
    }
    mx = fmaxf(mx, fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])), fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7]))));
  }
  // the CTA's largest |value| (non-negative floats order as their bit patterns): one per warp
  const uint32_t wmax = __reduce_max_sync(0xffffffffu, __float_as_uint(mx));
  if (lane == 0) s_wmax[warp] = wmax;
  __syncthreads();
  uint32_t cmax = 0u;
#pragma unroll
  for (int i = 0; i < kGvThreads / 32; ++i) cmax = max(cmax, s_wmax[i]);
  if (max_exchange) {
    cluster_wait();  // pairs with the arrive at set-up: every CTA's barrier is initialised
    if (t < p.splits && !hold)  // (test hook: held, no CTA sends anything; every receiving wait runs out)
      st_async_u32(mapa_shared(smem_u32(&s_maxes[rank]), static_cast<uint32_t>(t)), cmax,
                   mapa_shared(bar_max, static_cast<uint32_t>(t)));
    ok = mbar_wait_cluster(bar_max, 0) && ok;
    cmax = 0u;
    for (int src = 0; src < p.splits; ++src) cmax = max(cmax, s_maxes[src]);
  }
  const bool per_step = p.xscale != nullptr;
  // the scale: the step's, or max |Z| of the normalised rotation over the row over q_max = 7
  const float delta = per_step ? __ldg(p.xscale) : __fdiv_rn(__uint_as_float(cmax) * p.inv_sqrt_b, 7.0f);
  const float cr = p.inv_sqrt_b * (delta > 0.0f ? __fdiv_rn(1.0f, delta) : 0.0f);  // infinite iff 1 / delta overflows
  *delta_out = delta;
  // codes of this thread's channels of the range: operand byte q + 8 of channel k at byte
  // 8 (k / 8) + j of the range, j = i / 2 for the even i = k % 8 and 4 + i / 2 for the odd
  uint32_t qs = 0u;
#pragma unroll
  for (int ps = 0; ps < kGvPasses; ++ps) {
    if (ps >= passes) break;
#pragma unroll
    for (int w = 0; w < 8; ++w) {
      const int e = t + 256 * w, kk = (c0 + ps) * C + e - k0;
      if (e < C && kk >= 0 && kk < range) {
        const float y = yv[ps][w];
        float tt = __fmul_rn(y, cr);  // rounded on its own, as the kernel's packed multiply
        if (per_step) tt = fminf(fmaxf(tt, -7.0f), 7.0f);
        float u = __fadd_rn(tt, rq::kMagic);
        const float d = __fmaf_rn(__fadd_rn(u, -rq::kMagic), -1.0f, tt);
        if (fabsf(d) >= rq::kTieBand || isinf(cr)) u = rq::exact_code(y, p.inv_sqrt_b, delta, cr, 7.0f, rq::kTieBand);
        const uint32_t q8 = (__float_as_uint(u) & 0xFu) ^ 0x8u;
        const int i = kk & 7;
        s_act[(kk & ~7) + ((i & 1) ? 4 + (i >> 1) : (i >> 1))] = static_cast<uint8_t>(q8);
        qs += q8;
      }
    }
  }
  const uint32_t wsum = __reduce_add_sync(0xffffffffu, qs);
  if (lane == 0) s_wsum[warp] = wsum;
  __syncthreads();  // the operand bytes and code sums are complete
  return ok;
}

template <int kM, bool kGated, int kXB, typename OutT>
__global__ void __launch_bounds__(kGvThreads) gemv_w4a4_kernel(GvParams p) {
  static_assert(kXB != 2 || kM == 1, "the one-launch linear takes one token");
  constexpr int kParts = kGated ? 2 : 1;  // 128-row weight groups per CTA
  constexpr int kGvRing = gv_ring<kM, kGated, kXB>();
  constexpr int kActKb = kXB == 0 ? kBK / 2 : kBK;  // activation bytes per token and k-block
  __shared__ uint32_t s_part[kParts][128][kM];
  // split K: the slices of this CTA's rows from every CTA of the cluster, [source][row][part][m]
  __shared__ uint32_t s_recv[128 * kParts * kM];
  __shared__ __align__(8) uint64_t bar_recv;
  // kXB 2: the largest |rotated value| of each warp and of every CTA of the cluster (received),
  // and each warp's sum of the offset codes q + 8 of this CTA's k-range
  __shared__ uint32_t s_wmax[kGvThreads / 32], s_maxes[8], s_wsum[kGvThreads / 32];
  __shared__ __align__(8) uint64_t bar_max;
  // [kM][k-range] activation bytes of this CTA; kXB 2 then [kM][k-range] float rotated values
  // and one pass of C floats
  extern __shared__ __align__(16) uint8_t s_act[];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = p.splits;
  // test hook, read while the weights stream: held, the CTAs of a cluster send each other nothing
  const bool hold = S > 1 && *const_cast<volatile int*>(&g_debug_hold_loads) != 0;
  const int unit = static_cast<int>(blockIdx.x) / S;
  const int rank = static_cast<int>(blockIdx.x) % S;  // the CTA's rank in its cluster of S
  const int kb0 = p.nkb * rank / S, kb1 = p.nkb * (rank + 1) / S;
  const int slice = warp & 3, kpar = warp >> 2;  // kpar in [0, kGvPhases)
  const int q = lane & 3;
  const int R = 128 / S;  // rows this CTA finishes: [rank R, (rank + 1) R)

  for (int i = threadIdx.x; i < kParts * 128 * kM; i += kGvThreads) (&s_part[0][0][0])[i] = 0u;
  // kXB 2 with per-token scales: the CTAs of the cluster exchange their k-ranges' maxima
  // (unless one rotation pass is the whole row, which every CTA then rotates)
  const bool max_exchange = kXB == 2 && S > 1 && p.xscale == nullptr && p.K > p.C;
  if (S > 1) {
    // every CTA of the cluster sends this one its partials of these rows; the cluster barrier
    // completed before the first send guarantees every receiver's barrier exists
    if (threadIdx.x == 0) {
      mbar_init(smem_u32(&bar_recv), 1);
      if (max_exchange) mbar_init(smem_u32(&bar_max), 1);
      mbar_init_fence();
      mbar_arrive_expect_tx(smem_u32(&bar_recv), static_cast<uint32_t>(S * R * kParts * kM * 4));
      if (max_exchange) mbar_arrive_expect_tx(smem_u32(&bar_max), static_cast<uint32_t>(S * 4));
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
  // the epilogue's parameters of this thread's (row, token) entries: the layer's, before the wait
  constexpr int kEnt = (128 * kM + kGvThreads - 1) / kGvThreads;
  float e_cm[kEnt], e_xs[kEnt], e_wc[kEnt][kParts], e_ws[kEnt][kParts], e_bs[kEnt][kParts];
#pragma unroll
  for (int u = 0; u < kEnt; ++u) {
    const int e = threadIdx.x + u * kGvThreads;
    const int row = rank * R + min(e, R * kM - 1) / kM;
#pragma unroll
    for (int part = 0; part < kParts; ++part) {
      const int n = kGated ? 2 * unit * 128 + part * 128 + row : min(unit * 128 + row, p.N - 1);
      e_wc[u][part] = __ldg(p.wcorr + n);
      e_ws[u][part] = __ldg(p.wscale + n);
      e_bs[u][part] = __ldg(p.bias + n);
    }
  }
  griddep_wait();  // the activations, their scales and sums come from the previous kernel
  if (threadIdx.x == 0) griddep_launch_dependents();
#pragma unroll
  for (int u = 0; u < kEnt; ++u) {
    const int m = min((threadIdx.x + u * kGvThreads) % kM, p.M - 1);
    if constexpr (kXB == 2) {  // the activations' code sums are taken out of the partial sums
      e_cm[u] = p.kconst;
      e_xs[u] = 0.0f;
    } else {
      e_cm[u] = 8.0f * static_cast<float>(p.xsum[m]) + p.kconst;
      e_xs[u] = p.xscale[m];
    }
  }
  bool landed = true, cluster_waited = false;
  if constexpr (kXB == 2) {
    float delta = 0.0f;
    landed = rotate_quantize_token<OutT>(p, static_cast<const OutT*>(p.x), kb0, kb1, rank, max_exchange, s_act, s_wmax,
                                         s_maxes, s_wsum, smem_u32(&bar_max), hold, &delta);
    cluster_waited = max_exchange;
#pragma unroll
    for (int u = 0; u < kEnt; ++u) e_xs[u] = delta;
  } else {  // this CTA's k-range of every token's activation bytes, once, into shared memory
    const int row16 = (kb1 - kb0) * kActKb / 16;  // 16-byte pieces per token
    for (int i = threadIdx.x; i < p.M * row16; i += kGvThreads) {
      const int m = i / row16, c = i % row16;
      reinterpret_cast<uint4*>(s_act)[m * row16 + c] = __ldg(reinterpret_cast<const uint4*>(
          p.xq + static_cast<size_t>(m) * (p.K / (kBK / kActKb)) + kb0 * kActKb) + c);
    }
    __syncthreads();
  }

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
            if constexpr (kXB != 0) {
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
  // kXB 2: 8 x the activation codes' sum over this CTA's k-range, taken out of its partials
  // (the sums of all ranks then hold S - 8 sum_k q_x, a signed value in 32-bit wrap-around)
  uint32_t qsum = 0u;
  if constexpr (kXB == 2) {
#pragma unroll
    for (int i = 0; i < kGvThreads / 32; ++i) qsum += s_wsum[i];
  }
  auto xcorr = [&](int) -> uint32_t {
    if constexpr (kXB == 2) return 8u * qsum - 64u * static_cast<uint32_t>((kb1 - kb0) * kBK);
    return 0u;
  };
  if (S > 1) {
    if (!cluster_waited) cluster_wait();  // pairs with the arrive at set-up: every receive barrier is initialised
    // each partial goes to the CTA that finishes its row, as an asynchronous store completing on
    // that CTA's barrier; no CTA reads another's shared memory, so none waits for the others to leave
    // (test hook: held, nothing is sent and every CTA's wait runs out)
    for (int i = threadIdx.x; i < (hold ? 0 : 128 * kParts * kM); i += kGvThreads) {
      const int row = i / (kParts * kM), part = (i / kM) % kParts, m = i % kM;
      const int d = row / R;
      const uint32_t dst = smem_u32(&s_recv[((rank * R + (row - d * R)) * kParts + part) * kM + m]);
      st_async_u32(mapa_shared(dst, static_cast<uint32_t>(d)), s_part[part][row][m] - xcorr(m),
                   mapa_shared(smem_u32(&bar_recv), static_cast<uint32_t>(d)));
    }
    landed = mbar_wait_cluster(smem_u32(&bar_recv), 0) && landed;
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
        sum[part] = s_part[part][row][m] - xcorr(m);
      }
    }
    // the epilogue of the tensor-core path: exact accumulator, one float32 scale product, fma, one rounding
    if constexpr (!kGated) {
      const int n = unit * 128 + row;
      if (n < p.N) {
        const float a = static_cast<float>(static_cast<int32_t>(sum[0])) - (e_cm[u] + e_wc[u][0]);
        reinterpret_cast<OutT*>(p.y)[static_cast<size_t>(m) * p.ldy + n] = to_out<OutT>(fmaf(a, e_xs[u] * e_ws[u][0], e_bs[u][0]));
        if (p.acc) p.acc[static_cast<size_t>(m) * p.N + n] = static_cast<int32_t>(a);
      }
    } else {
      // weight rows 256 unit + row (gate) and + 128 (up) of hidden unit j; h = gelu(gate) * up
      const int H = p.N / 2, j = unit * 128 + row;
      if (j < H) {
        const float ag = static_cast<float>(static_cast<int32_t>(sum[0])) - (e_cm[u] + e_wc[u][0]);
        const float au = static_cast<float>(static_cast<int32_t>(sum[1])) - (e_cm[u] + e_wc[u][1]);
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
  // the largest k-range of a CTA, for every token (kXB 2: and one rotation pass)
  size_t act = static_cast<size_t>(kM) * ((p.nkb + p.splits - 1) / p.splits) * (kXB == 0 ? kBK / 2 : kBK);
  if (kXB == 2) act += 4 * static_cast<size_t>(p.C);
  if (act > static_cast<size_t>(kGemvActMax)) return kNotApplicable;
  if (act + 16 * 1024 > 48 * 1024) {  // with the static shared memory (up to 8.4 KB) past the default 48 KB
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
  if constexpr (kXB == 2) {
    return kNotApplicable;  // the one-launch linear takes one token
  } else {
    if (a.M == 2) return launch_gv<2, kGated, kXB, OutT>(a, p, units);
    return launch_gv<4, kGated, kXB, OutT>(a, p, units);
  }
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
  if (a.M < 1 || a.M > kGemvMaxM || a.gscale || (a.x_bytes != 0 && a.x_bytes != 1 && a.x_bytes != 3)) return cudaSuccess;
  // raw activations (one token): rotation passes of C channels, C the largest power of two up to
  // 2048 that divides K, holding whole Hadamard blocks; x of the output's dtype
  int C = 2048;
  while (a.K % C != 0) C /= 2;
  if (a.x_bytes == 3 && (a.M != 1 || a.xdt != a.ydt || a.log_b < 0 || (1 << a.log_b) > C)) return cudaSuccess;
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
  p.x = a.x;
  p.log_b = a.log_b;
  p.C = C;
  p.inv_sqrt_b = a.inv_sqrt_b;
  // one CTA per 128-row group (gated: per 128 hidden units, gate and up), K split over a cluster
  // of up to 8 until the grid holds about two CTAs per SM.  The one-launch linear (raw
  // activations) doubles the split only while the grid holds at most 0.75 CTAs per SM, so a wide
  // layer keeps about one CTA per SM with a deep weight ring and the next launch's CTAs fit beside
  // it (measured on an 18-layer decode step: 455 us, against 540 us with the gate/up projection
  // split in two and 472 us with its ring of four k-blocks).
  const int units = a.gated ? a.N / 256 : (a.N + 127) / 128;
  int splits = 1;
  if (a.x_bytes == 3) {
    while (splits < 8 && 2 * splits <= p.nkb && 4 * units * splits <= 3 * a.num_sms) splits *= 2;
  } else {
    while (splits < 8 && 2 * splits <= p.nkb && units * splits < 2 * a.num_sms) splits *= 2;
  }
  p.splits = splits;
  if (a.x_bytes == 3) {
    for (int r = 0; r < splits; ++r) {  // a CTA holds the rotated values of at most kGvPasses passes
      const int k0 = p.nkb * r / splits * kBK, k1 = p.nkb * (r + 1) / splits * kBK;
      if ((k1 + C - 1) / C - k0 / C > kGvPasses) return cudaSuccess;
    }
  }
  cudaError_t e;
  if (a.x_bytes == 3)
    e = a.ydt == 0 ? launch_gv_g<2, __half>(a, p, units) : launch_gv_g<2, __nv_bfloat16>(a, p, units);
  else if (a.x_bytes == 1)
    e = a.ydt == 0 ? launch_gv_g<1, __half>(a, p, units) : launch_gv_g<1, __nv_bfloat16>(a, p, units);
  else
    e = a.ydt == 0 ? launch_gv_g<0, __half>(a, p, units) : launch_gv_g<0, __nv_bfloat16>(a, p, units);
  if (e == kNotApplicable) return cudaSuccess;  // the activations of a CTA would not fit
  *launched = e == cudaSuccess;
  return e;
}

}  // namespace qvla
