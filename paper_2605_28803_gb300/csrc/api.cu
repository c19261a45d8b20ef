// The C ABI of libqvla (include/qvla.h): argument validation, layer objects and kernel dispatch.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "../../include/qvla.h"
#include "../../include/qvla_debug.h"
#include "kernels.h"
#include "pack.h"

struct qvla_layer {
  int N = 0, K = 0, had_block = 1, log_b = 0;  // N = weight rows (2H when gated)
  int gated = 0;
  int xdt = 0, ydt = 0;
  int device = 0;
  uint8_t* wq = nullptr;      // device, tiled: [groups][K/128][128 rows][64 B] (see upload_layer)
  float* wscale = nullptr;    // device [N]
  float* wcorr = nullptr;     // device [N]: 8 * (sum of the codes of row n), the GEMM's offset correction
  float* wcorr8 = nullptr;    // device [N]: 128 * (sum of the codes of row n), the same for 8-bit activations
  float* bias = nullptr;      // device [N] (zeros when the layer was given none)
  float* table = nullptr;     // device [table_cap]: T step scales, or T x G group scales
  int T = 0, table_cap = 0;
  int grouped = 0;            // the table holds one scale per (step, channel group)
  int group = 128, G = 1;     // channels per scale group (max(128, had_block)) and groups per row
  float* wgcorr = nullptr;    // device [N][G]: 8 * (sum of row n's codes over group g), non-gated layers
  int32_t* rperm = nullptr;   // device [K]: online permutation (identity when only U is given)
  float* rrot = nullptr;      // device [K/rblock][rblock][rblock]: online U_b blocks, float32
  int rblock = 0;             // 0: the activations arrive in the P.U basis (no online rotation)
};

namespace {

thread_local std::string g_last_error;

qvla_status fail(qvla_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_last_error = buf;
  return s;
}

qvla_status cuda_fail(cudaError_t e, const char* what) {
  return fail(e == cudaErrorMemoryAllocation ? QVLA_ERR_OOM : QVLA_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define QVLA_CUDA(call, what)                        \
  do {                                               \
    cudaError_t e_ = (call);                         \
    if (e_ != cudaSuccess) return cuda_fail(e_, what); \
  } while (0)

int ilog2_exact(int v) {
  if (v < 1 || (v & (v - 1))) return -1;
  int l = 0;
  while ((1 << l) < v) ++l;
  return l;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

qvla_status check_shape(int N, int K, int had_block) {
  if (K <= 0 || K % 128 != 0) return fail(QVLA_ERR_INVALID_ARG, "K=%d must be a positive multiple of 128", K);
  if (K > 16384) return fail(QVLA_ERR_UNSUPPORTED, "K=%d exceeds 16384 (exact float32 accumulation bound)", K);
  if (N <= 0 || N % 16 != 0) return fail(QVLA_ERR_INVALID_ARG, "N=%d must be a positive multiple of 16", N);
  const int lb = ilog2_exact(had_block);
  if (lb < 0) return fail(QVLA_ERR_INVALID_ARG, "had_block=%d is not a power of two", had_block);
  if (had_block > 4096) return fail(QVLA_ERR_UNSUPPORTED, "had_block=%d exceeds 4096", had_block);
  if (K % had_block != 0) return fail(QVLA_ERR_INVALID_ARG, "K=%d is not a multiple of had_block=%d", K, had_block);
  return QVLA_OK;
}

int num_sms(int device) {
  static std::mutex mu;
  static std::vector<int> cache;
  std::lock_guard<std::mutex> lk(mu);
  if (device >= static_cast<int>(cache.size())) cache.resize(device + 1, 0);
  if (cache[device] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, device) != cudaSuccess || v <= 0) v = 148;
    cache[device] = v;
  }
  return cache[device];
}

size_t round256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }

// bytes of an [M][K] activation tensor of the layer's input dtype
size_t rotated_bytes(const qvla_layer* L, int M) {
  return static_cast<size_t>(M) * L->K * (L->xdt == QVLA_F32 ? 4 : 2);
}

qvla_status check_rows(int M) {
  if (M < 0 || M > (1 << 20)) return fail(QVLA_ERR_INVALID_ARG, "M=%d outside [0, 2^20]", M);
  return QVLA_OK;
}

qvla_status launch_rq(const void* x, int xdt, int M, int K, int had_block, int mode, const float* step_scale,
                      uint8_t* xq, float* xscale, int32_t* xsum, float* absmax, void* stream, int out_mode = 0,
                      int group = 0, int32_t* xgsum = nullptr, int32_t* zero = nullptr, int zero_n = 0) {
  qvla::RotQuantArgs a;
  a.x = x;
  a.xdt = xdt;
  a.M = M;
  a.K = K;
  a.log_b = ilog2_exact(had_block);
  a.inv_sqrt_b = static_cast<float>(1.0 / std::sqrt(static_cast<double>(had_block)));
  a.mode = mode;
  a.step_scale = step_scale;
  a.xq = xq;
  a.xscale = xscale;
  a.xsum = xsum;
  a.absmax = absmax;
  a.out_mode = out_mode;
  a.gshift = group > 0 ? ilog2_exact(group) : 30;
  a.xgsum = xgsum;
  a.zero = zero;
  a.zero_n = zero_n;
  a.stream = static_cast<cudaStream_t>(stream);
  QVLA_CUDA(qvla::launch_rotate_quant(a), "rotate_quantize launch");
  return QVLA_OK;
}

// A layer's buffers live on the device that was current when it was created; its kernels must be
// launched with that device current.
qvla_status check_layer_device(const qvla_layer* L) {
  int dev = 0;
  QVLA_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  if (dev != L->device)
    return fail(QVLA_ERR_INVALID_ARG, "the current device is %d but the layer lives on device %d", dev, L->device);
  return QVLA_OK;
}

qvla_status resolve_step(const qvla_layer* layer, int step, const float** step_scale) {
  if (step == -1) {
    *step_scale = nullptr;
    return QVLA_OK;
  }
  if (step < 0 || step >= layer->T)
    return fail(QVLA_ERR_STEP_RANGE, "step %d outside the layer's table of %d steps", step, layer->T);
  *step_scale = layer->table + static_cast<size_t>(step) * (layer->grouped ? layer->G : 1);
  return QVLA_OK;
}

}  // namespace

extern "C" {

const char* qvla_last_error(void) { return g_last_error.c_str(); }

int qvla_abi_version(void) { return 1; }

qvla_status qvla_pack_weights_host(const void* W, qvla_dtype wdt, int N, int K, const double* rot, int rot_block,
                                   const int32_t* perm, int had_block, uint8_t* wq, float* wscale, int32_t* wsum) {
  g_last_error.clear();
  if (!W || !wq || !wscale) return fail(QVLA_ERR_INVALID_ARG, "W, wq and wscale must not be NULL");
  if (wdt != QVLA_F16 && wdt != QVLA_BF16 && wdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad weight dtype %d", wdt);
  if (qvla_status s = check_shape(N, K, had_block)) return s;
  if (rot) {
    if (rot_block <= 0 || K % rot_block != 0)
      return fail(QVLA_ERR_INVALID_ARG, "rot_block=%d must divide K=%d", rot_block, K);
  }
  if (perm) {
    std::vector<char> seen(K, 0);
    for (int k = 0; k < K; ++k) {
      if (perm[k] < 0 || perm[k] >= K || seen[perm[k]]) return fail(QVLA_ERR_INVALID_ARG, "perm is not a permutation of [0, K)");
      seen[perm[k]] = 1;
    }
  }
  qvla::pack_weights_host_impl(W, static_cast<int>(wdt), N, K, rot, rot_block, perm, had_block, wq, wscale, wsum);
  return QVLA_OK;
}

qvla_status qvla_gptq_pack_host(const void* W, qvla_dtype wdt, int N, int K, const void* X, qvla_dtype xdt,
                                int n_cal, const double* rot, int rot_block, const int32_t* perm, int had_block,
                                int block, double damp, uint8_t* wq, float* wscale, int32_t* wsum) {
  g_last_error.clear();
  if (!W || !X || !wq || !wscale) return fail(QVLA_ERR_INVALID_ARG, "W, X, wq and wscale must not be NULL");
  if (wdt != QVLA_F16 && wdt != QVLA_BF16 && wdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad weight dtype %d", wdt);
  if (xdt != QVLA_F16 && xdt != QVLA_BF16 && xdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad calibration dtype %d", xdt);
  if (qvla_status s = check_shape(N, K, had_block)) return s;
  if (K > 16384) return fail(QVLA_ERR_INVALID_ARG, "K=%d: GPTQ supports K <= 16384", K);
  if (n_cal < 1) return fail(QVLA_ERR_INVALID_ARG, "n_cal=%d must be >= 1", n_cal);
  if (block < 1) return fail(QVLA_ERR_INVALID_ARG, "block=%d must be >= 1", block);
  if (!(damp >= 0.0) || std::isinf(damp)) return fail(QVLA_ERR_INVALID_ARG, "damp must be finite and >= 0");
  if (rot && (rot_block <= 0 || K % rot_block != 0))
    return fail(QVLA_ERR_INVALID_ARG, "rot_block=%d must divide K=%d", rot_block, K);
  if (perm) {
    std::vector<char> seen(K, 0);
    for (int k = 0; k < K; ++k) {
      if (perm[k] < 0 || perm[k] >= K || seen[perm[k]]) return fail(QVLA_ERR_INVALID_ARG, "perm is not a permutation of [0, K)");
      seen[perm[k]] = 1;
    }
  }
  try {
    if (!qvla::gptq_pack_host(W, static_cast<int>(wdt), N, K, X, static_cast<int>(xdt), n_cal, rot, rot_block, perm,
                              had_block, block, damp, wq, wscale, wsum))
      return fail(QVLA_ERR_INVALID_ARG, "the damped Hessian is not positive definite (raise damp)");
  } catch (const std::bad_alloc&) {
    return fail(QVLA_ERR_OOM, "host allocation failed");
  }
  return QVLA_OK;
}

qvla_status qvla_block_svd_rotation(const void* W, qvla_dtype wdt, int N, int K, int block, int32_t* perm,
                                    double* rot) {
  g_last_error.clear();
  if (!W || !perm || !rot) return fail(QVLA_ERR_INVALID_ARG, "W, perm and rot must not be NULL");
  if (wdt != QVLA_F16 && wdt != QVLA_BF16 && wdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad weight dtype %d", wdt);
  if (N <= 0 || K <= 0) return fail(QVLA_ERR_INVALID_ARG, "N=%d and K=%d must be positive", N, K);
  if (block < 1 || block > 512 || K % block != 0)
    return fail(QVLA_ERR_INVALID_ARG, "block=%d must be in [1, 512] and divide K=%d", block, K);
  qvla::zigzag_permutation_host(W, static_cast<int>(wdt), N, K, block, perm);
  qvla::block_svd_rotation_host(W, static_cast<int>(wdt), N, K, block, perm, rot);
  return QVLA_OK;
}

static qvla_status upload_layer(int N, int K, int had_block, qvla_dtype xdt, qvla_dtype ydt, int gated,
                                const uint8_t* wq, const float* wscale, const float* bias, qvla_layer** out) {
  if (xdt != QVLA_F16 && xdt != QVLA_BF16 && xdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad activation dtype %d", xdt);
  if (ydt != QVLA_F16 && ydt != QVLA_BF16) return fail(QVLA_ERR_INVALID_ARG, "output dtype must be F16 or BF16");
  for (int n = 0; n < N; ++n)
    if (!(wscale[n] >= 0.0f) || std::isinf(wscale[n])) return fail(QVLA_ERR_INVALID_ARG, "wscale[%d] is not a finite non-negative float", n);
  std::vector<int32_t> wsum(N);
  qvla::code_sums_host(wq, N, K, wsum.data());
  std::vector<float> wcorr(N), wcorr8(N), zero_bias;
  for (int n = 0; n < N; ++n) {
    wcorr[n] = 8.0f * static_cast<float>(wsum[n]);      // exact: |8 wsum| <= 2^20
    wcorr8[n] = 128.0f * static_cast<float>(wsum[n]);   // exact: |128 wsum| <= 2^24
  }
  if (!bias) {
    zero_bias.assign(N, 0.0f);
    bias = zero_bias.data();
  }
  auto* L = new (std::nothrow) qvla_layer();
  if (!L) return fail(QVLA_ERR_OOM, "host allocation failed");
  L->gated = gated;
  L->N = N;
  L->K = K;
  L->had_block = had_block;
  L->log_b = ilog2_exact(had_block);
  L->xdt = xdt;
  L->ydt = ydt;
  L->group = std::max(128, had_block);
  L->G = K / L->group;
  cudaGetDevice(&L->device);
  // Weights are stored tiled: each group of 128 rows x one k-block of 128 codes (64 bytes per
  // row) is one contiguous 8 KB chunk, chunks ordered by row group, then k-block; rows past N
  // are zero, and the number of groups is even (a 256-row GEMM tile reads groups in pairs).
  // The GEMM fetches a chunk with one bulk copy instead of 128 separate 64-byte rows.
  const int groups = ((N + 255) / 256) * 2, kblocks = K / 128;
  const size_t rb = static_cast<size_t>(K / 2);
  const size_t wbytes = static_cast<size_t>(groups) * kblocks * 8192;
  std::vector<uint8_t> tiled;
  try {
    tiled.assign(wbytes, 0);
  } catch (...) {
    delete L;
    return fail(QVLA_ERR_OOM, "host allocation failed");
  }
  for (int n = 0; n < N; ++n)
    for (int kb = 0; kb < kblocks; ++kb)
      std::memcpy(tiled.data() + ((static_cast<size_t>(n / 128) * kblocks + kb) * 128 + n % 128) * 64,
                  wq + n * rb + static_cast<size_t>(kb) * 64, 64);
  cudaError_t e = cudaMalloc(&L->wq, wbytes);
  if (e == cudaSuccess) e = cudaMalloc(&L->wscale, N * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&L->wcorr, N * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&L->wcorr8, N * sizeof(float));
  if (e == cudaSuccess) e = cudaMalloc(&L->bias, N * sizeof(float));
  if (e == cudaSuccess) e = cudaMemcpy(L->wq, tiled.data(), wbytes, cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(L->wscale, wscale, N * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(L->wcorr, wcorr.data(), N * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(L->wcorr8, wcorr8.data(), N * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess) e = cudaMemcpy(L->bias, bias, N * sizeof(float), cudaMemcpyHostToDevice);
  if (e == cudaSuccess && !gated) {  // per-group code sums for per-group step scales
    std::vector<float> wg(static_cast<size_t>(N) * L->G, 0.0f);
    for (int n = 0; n < N; ++n)
      for (int k = 0; k < K; ++k) {
        const int b = wq[static_cast<size_t>(n) * rb + k / 2];
        int q = (k & 1) ? (b >> 4) : (b & 0xF);
        q = q >= 8 ? q - 16 : q;
        wg[static_cast<size_t>(n) * L->G + k / L->group] += 8.0f * static_cast<float>(q);  // exact integers
      }
    e = cudaMalloc(&L->wgcorr, wg.size() * sizeof(float));
    if (e == cudaSuccess) e = cudaMemcpy(L->wgcorr, wg.data(), wg.size() * sizeof(float), cudaMemcpyHostToDevice);
  }
  if (e != cudaSuccess) {
    qvla_layer_destroy(L);
    return cuda_fail(e, "layer upload");
  }
  *out = L;
  return QVLA_OK;
}

qvla_status qvla_layer_create(int N, int K, int had_block, qvla_dtype xdt, qvla_dtype ydt, const uint8_t* wq,
                              const float* wscale, const float* bias, qvla_layer** out) {
  g_last_error.clear();
  if (!wq || !wscale || !out) return fail(QVLA_ERR_INVALID_ARG, "wq, wscale and out must not be NULL");
  if (qvla_status s = check_shape(N, K, had_block)) return s;
  return upload_layer(N, K, had_block, xdt, ydt, 0, wq, wscale, bias, out);
}

qvla_status qvla_layer_create_gated(int H, int K, int had_block, qvla_dtype xdt, qvla_dtype ydt, const uint8_t* wq_gate,
                                    const float* wscale_gate, const uint8_t* wq_up, const float* wscale_up,
                                    const float* bias_gate, const float* bias_up, qvla_layer** out) {
  g_last_error.clear();
  if (!wq_gate || !wscale_gate || !wq_up || !wscale_up || !out)
    return fail(QVLA_ERR_INVALID_ARG, "weights, scales and out must not be NULL");
  if ((bias_gate == nullptr) != (bias_up == nullptr))
    return fail(QVLA_ERR_INVALID_ARG, "give both biases or neither");
  if (H <= 0 || H % 128 != 0) return fail(QVLA_ERR_INVALID_ARG, "H=%d must be a positive multiple of 128", H);
  if (qvla_status s = check_shape(2 * H, K, had_block)) return s;
  // interleave: weight rows [256 t, 256 t + 128) = gate rows [128 t, 128 t + 128),
  //             rows [256 t + 128, 256 t + 256) = up rows of the same hidden units
  const size_t rb = static_cast<size_t>(K / 2);
  std::vector<uint8_t> wq(static_cast<size_t>(2) * H * rb);
  std::vector<float> ws(2 * H), bs(bias_gate ? 2 * H : 0);
  for (int t = 0; t < H / 128; ++t)
    for (int i = 0; i < 128; ++i) {
      const int j = 128 * t + i;
      const int rg = 256 * t + i, ru = rg + 128;
      std::memcpy(wq.data() + rg * rb, wq_gate + j * rb, rb);
      std::memcpy(wq.data() + ru * rb, wq_up + j * rb, rb);
      ws[rg] = wscale_gate[j];
      ws[ru] = wscale_up[j];
      if (bias_gate) {
        bs[rg] = bias_gate[j];
        bs[ru] = bias_up[j];
      }
    }
  return upload_layer(2 * H, K, had_block, xdt, ydt, 1, wq.data(), ws.data(), bias_gate ? bs.data() : nullptr, out);
}

qvla_status qvla_pack_weights(const void* W, qvla_dtype wdt, int N, int K, const double* rot, int rot_block,
                              const int32_t* perm, int had_block, const float* bias, qvla_dtype xdt, qvla_dtype ydt,
                              qvla_layer** out) {
  g_last_error.clear();
  if (qvla_status s = check_shape(N, K, had_block)) return s;
  std::vector<uint8_t> wq;
  std::vector<float> ws;
  try {
    wq.resize(static_cast<size_t>(N) * (K / 2));
    ws.resize(N);
  } catch (...) {
    return fail(QVLA_ERR_OOM, "host allocation failed");
  }
  if (qvla_status s = qvla_pack_weights_host(W, wdt, N, K, rot, rot_block, perm, had_block, wq.data(), ws.data(), nullptr))
    return s;
  return qvla_layer_create(N, K, had_block, xdt, ydt, wq.data(), ws.data(), bias, out);
}

qvla_status qvla_layer_destroy(qvla_layer* L) {
  g_last_error.clear();
  if (!L) return QVLA_OK;
  cudaDeviceSynchronize();
  cudaFree(L->wq);
  cudaFree(L->wscale);
  cudaFree(L->wcorr);
  cudaFree(L->wcorr8);
  cudaFree(L->wgcorr);
  cudaFree(L->bias);
  cudaFree(L->table);
  cudaFree(L->rperm);
  cudaFree(L->rrot);
  delete L;
  return QVLA_OK;
}

namespace {
qvla_status check_scales(const float* scales, size_t n) {
  for (size_t i = 0; i < n; ++i)
    if (!(scales[i] > 0.0f) || std::isinf(scales[i])) return fail(QVLA_ERR_INVALID_ARG, "scales[%zu] must be finite and > 0", i);
  return QVLA_OK;
}

// Upload a table of T x per_step floats (already checked), growing the allocation only when it
// is too small (a smaller or equal table is written in place: captured graphs keep the address).
qvla_status upload_table(qvla_layer* L, const float* scales, int T, int per_step) {
  const size_t n = static_cast<size_t>(T) * per_step;
  L->T = 0;
  if (n > static_cast<size_t>(L->table_cap)) {
    QVLA_CUDA(cudaDeviceSynchronize(), "synchronise before table reallocation");
    cudaFree(L->table);
    L->table = nullptr;
    L->table_cap = 0;
    QVLA_CUDA(cudaMalloc(&L->table, n * sizeof(float)), "step table allocation");
    L->table_cap = static_cast<int>(n);
  }
  QVLA_CUDA(cudaMemcpy(L->table, scales, n * sizeof(float), cudaMemcpyHostToDevice), "step table upload");
  L->T = T;
  return QVLA_OK;
}
}  // namespace

qvla_status qvla_set_step_scales(qvla_layer* L, const float* scales, int T) {
  g_last_error.clear();
  if (!L || !scales) return fail(QVLA_ERR_INVALID_ARG, "layer and scales must not be NULL");
  if (T < 1 || T > (1 << 20)) return fail(QVLA_ERR_INVALID_ARG, "T=%d must be in [1, 2^20]", T);
  if (qvla_status s = check_scales(scales, static_cast<size_t>(T))) return s;
  L->grouped = 0;
  return upload_table(L, scales, T, 1);
}

qvla_status qvla_set_step_group_scales(qvla_layer* L, const float* scales, int T, int G) {
  g_last_error.clear();
  if (!L || !scales) return fail(QVLA_ERR_INVALID_ARG, "layer and scales must not be NULL");
  if (L->gated) return fail(QVLA_ERR_UNSUPPORTED, "per-group step scales are not available for gated layers");
  if (T < 1 || T > (1 << 16)) return fail(QVLA_ERR_INVALID_ARG, "T=%d must be in [1, 2^16]", T);
  if (G != L->G)
    return fail(QVLA_ERR_INVALID_ARG, "G=%d: this layer has %d groups of %d channels", G, L->G, L->group);
  if (qvla_status s = check_scales(scales, static_cast<size_t>(T) * G)) return s;
  L->grouped = 1;
  return upload_table(L, scales, T, G);
}

qvla_status qvla_layer_scale_groups(const qvla_layer* L, int* G, int* group) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (G) *G = L->G;
  if (group) *group = L->group;
  return QVLA_OK;
}

qvla_status qvla_layer_set_online_rotation(qvla_layer* L, const int32_t* perm, const double* rot, int rot_block) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_layer_device(L)) return s;
  const int K = L->K;
  if (!perm && !rot) {  // back to activations that arrive in the P.U basis
    QVLA_CUDA(cudaDeviceSynchronize(), "synchronise before freeing the online rotation");
    cudaFree(L->rperm);
    cudaFree(L->rrot);
    L->rperm = nullptr;
    L->rrot = nullptr;
    L->rblock = 0;
    return QVLA_OK;
  }
  if (!rot) rot_block = 16;  // a permutation alone: identity blocks
  if (rot_block != 16 && rot_block != 32 && rot_block != 64)
    return fail(QVLA_ERR_UNSUPPORTED, "rot_block=%d: the online rotation takes blocks of 16, 32 or 64 channels", rot_block);
  if (K % rot_block != 0) return fail(QVLA_ERR_INVALID_ARG, "rot_block=%d does not divide K=%d", rot_block, K);
  std::vector<int32_t> hp(K);
  if (perm) {
    std::vector<char> seen(K, 0);
    for (int k = 0; k < K; ++k) {
      const int32_t v = perm[k];
      if (v < 0 || v >= K || seen[v]) return fail(QVLA_ERR_INVALID_ARG, "perm is not a permutation of [0, K)");
      seen[v] = 1;
      hp[k] = v;
    }
  } else {
    for (int k = 0; k < K; ++k) hp[k] = k;
  }
  const size_t nrot = static_cast<size_t>(K) * rot_block;  // (K / rot_block) blocks of rot_block^2
  std::vector<float> hr(nrot, 0.0f);
  for (size_t i = 0; i < nrot; ++i) {
    if (rot) {
      if (!std::isfinite(rot[i])) return fail(QVLA_ERR_INVALID_ARG, "rot holds a non-finite entry");
      hr[i] = static_cast<float>(rot[i]);
    } else {
      const size_t e = i % (static_cast<size_t>(rot_block) * rot_block);
      hr[i] = (e / rot_block == e % rot_block) ? 1.0f : 0.0f;
    }
  }
  QVLA_CUDA(cudaDeviceSynchronize(), "synchronise before replacing the online rotation");
  cudaFree(L->rperm);
  cudaFree(L->rrot);
  L->rperm = nullptr;
  L->rrot = nullptr;
  L->rblock = 0;
  QVLA_CUDA(cudaMalloc(&L->rperm, hp.size() * sizeof(int32_t)), "online permutation allocation");
  QVLA_CUDA(cudaMalloc(&L->rrot, hr.size() * sizeof(float)), "online rotation allocation");
  QVLA_CUDA(cudaMemcpy(L->rperm, hp.data(), hp.size() * sizeof(int32_t), cudaMemcpyHostToDevice), "online permutation upload");
  QVLA_CUDA(cudaMemcpy(L->rrot, hr.data(), hr.size() * sizeof(float), cudaMemcpyHostToDevice), "online rotation upload");
  L->rblock = rot_block;
  return QVLA_OK;
}

qvla_status qvla_online_rotate(const qvla_layer* L, const void* x, int M, void* out, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_rows(M)) return s;
  if (!L->rblock) return fail(QVLA_ERR_INVALID_ARG, "the layer has no online rotation");
  if (M == 0) return QVLA_OK;
  if (!x || !out) return fail(QVLA_ERR_INVALID_ARG, "x and out must not be NULL");
  QVLA_CUDA(qvla::launch_block_rotate(x, L->xdt, M, L->K, L->rperm, L->rrot, L->rblock, out,
                                      static_cast<cudaStream_t>(stream)),
            "online rotation launch");
  return QVLA_OK;
}

qvla_status qvla_layer_info(const qvla_layer* L, int* N, int* K, int* had_block, int* T) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (N) *N = L->gated ? L->N / 2 : L->N;
  if (K) *K = L->K;
  if (had_block) *had_block = L->had_block;
  if (T) *T = L->T;
  return QVLA_OK;
}

qvla_status qvla_rotate_quantize_rows(const void* x, qvla_dtype xdt, int M, int K, int had_block, const float* step_scale,
                                      uint8_t* xq, float* xscale, int32_t* xsum, void* stream) {
  g_last_error.clear();
  if (qvla_status s = check_rows(M)) return s;
  if (qvla_status s = check_shape(16, K, had_block)) return s;
  if (xdt != QVLA_F16 && xdt != QVLA_BF16 && xdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad activation dtype %d", xdt);
  if (M == 0) return QVLA_OK;
  if (!x || !xq || !xscale) return fail(QVLA_ERR_INVALID_ARG, "x, xq and xscale must not be NULL");
  if (!aligned16(x) || !aligned16(xq)) return fail(QVLA_ERR_INVALID_ARG, "x and xq must be 16-byte aligned");
  return launch_rq(x, xdt, M, K, had_block, step_scale ? 1 : 0, step_scale, xq, xscale, xsum, nullptr, stream);
}

qvla_status qvla_rotate_quantize(const qvla_layer* L, const void* x, int M, int step, uint8_t* xq, float* xscale,
                                 int32_t* xsum, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_rows(M)) return s;
  const float* ss = nullptr;
  if (qvla_status s = resolve_step(L, step, &ss)) return s;
  if (ss && L->grouped)
    return fail(QVLA_ERR_UNSUPPORTED, "per-group step scales run through qvla_w4a4_linear only (codes alone have no single scale)");
  if (L->rblock)
    return fail(QVLA_ERR_UNSUPPORTED, "the layer's online rotation runs in qvla_w4a4_linear / qvla_linear_quantize");
  if (M == 0) return QVLA_OK;
  if (!x || !xq || !xscale) return fail(QVLA_ERR_INVALID_ARG, "x, xq and xscale must not be NULL");
  if (!aligned16(x) || !aligned16(xq)) return fail(QVLA_ERR_INVALID_ARG, "x and xq must be 16-byte aligned");
  return launch_rq(x, L->xdt, M, L->K, L->had_block, ss ? 1 : 0, ss, xq, xscale, xsum, nullptr, stream);
}

qvla_status qvla_rotated_absmax(const void* x, qvla_dtype xdt, int M, int K, int had_block, float* absmax, void* stream) {
  g_last_error.clear();
  if (qvla_status s = check_rows(M)) return s;
  if (qvla_status s = check_shape(16, K, had_block)) return s;
  if (xdt != QVLA_F16 && xdt != QVLA_BF16 && xdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad activation dtype %d", xdt);
  if (M == 0) return QVLA_OK;
  if (!x || !absmax) return fail(QVLA_ERR_INVALID_ARG, "x and absmax must not be NULL");
  if (!aligned16(x)) return fail(QVLA_ERR_INVALID_ARG, "x must be 16-byte aligned");
  return launch_rq(x, xdt, M, K, had_block, 2, nullptr, nullptr, nullptr, nullptr, absmax, stream);
}

qvla_status qvla_rotated_absmax_groups(const void* x, qvla_dtype xdt, int M, int K, int had_block, float* absmax,
                                       void* stream) {
  g_last_error.clear();
  if (qvla_status s = check_rows(M)) return s;
  if (qvla_status s = check_shape(16, K, had_block)) return s;
  if (xdt != QVLA_F16 && xdt != QVLA_BF16 && xdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad activation dtype %d", xdt);
  const int group = std::max(128, had_block);
  if (K % group != 0) return fail(QVLA_ERR_INVALID_ARG, "K=%d is not a multiple of the group size %d", K, group);
  if (M == 0) return QVLA_OK;
  if (!x || !absmax) return fail(QVLA_ERR_INVALID_ARG, "x and absmax must not be NULL");
  if (!aligned16(x)) return fail(QVLA_ERR_INVALID_ARG, "x must be 16-byte aligned");
  return launch_rq(x, xdt, M, K, had_block, 2, nullptr, nullptr, nullptr, nullptr, absmax, stream, 0, group);
}

qvla_status qvla_rotate_quantize_rows_a8(const void* x, qvla_dtype xdt, int M, int K, int had_block,
                                         const float* step_scale, int8_t* xq, float* xscale, int32_t* xsum,
                                         void* stream) {
  g_last_error.clear();
  if (qvla_status s = check_rows(M)) return s;
  if (qvla_status s = check_shape(16, K, had_block)) return s;
  if (xdt != QVLA_F16 && xdt != QVLA_BF16 && xdt != QVLA_F32) return fail(QVLA_ERR_INVALID_ARG, "bad activation dtype %d", xdt);
  if (M == 0) return QVLA_OK;
  if (!x || !xq || !xscale) return fail(QVLA_ERR_INVALID_ARG, "x, xq and xscale must not be NULL");
  if (!aligned16(x) || !aligned16(xq)) return fail(QVLA_ERR_INVALID_ARG, "x and xq must be 16-byte aligned");
  return launch_rq(x, xdt, M, K, had_block, step_scale ? 1 : 0, step_scale, reinterpret_cast<uint8_t*>(xq), xscale,
                   xsum, nullptr, stream, 2);
}

}  // extern "C"

namespace {
// The workspace's room for the GEMM's split of K: the work units' partials and the tiles' counters.
struct PartWorkspace {
  float* ws = nullptr;
  size_t floats = 0;
  int32_t* cnt = nullptr;
  int n = 0;
};

qvla_status launch_gemm(const qvla_layer* L, const uint8_t* xq, int x_bytes, const float* xscale, const int32_t* xsum,
                        int M, void* y, int32_t* acc, void* stream, const float* gscale = nullptr,
                        const int32_t* xgsum = nullptr, const PartWorkspace* pw = nullptr) {
  qvla::GemmArgs a;
  a.xq = xq;
  a.x_bytes = x_bytes;
  a.xscale = xscale;
  a.xsum = xsum;
  a.wq = L->wq;
  a.wscale = L->wscale;
  a.wcorr = x_bytes == 2 ? L->wcorr8 : L->wcorr;
  a.bias = L->bias;
  a.y = y;
  a.ydt = L->ydt;
  a.acc = acc;
  a.M = M;
  a.N = L->N;
  a.K = L->K;
  a.gated = L->gated;
  if (gscale) {
    a.gscale = gscale;
    a.xgsum = xgsum;
    a.wgcorr = L->wgcorr;
    a.group = L->group;
  }
  if (pw != nullptr && pw->ws != nullptr) {
    a.part_ws = pw->ws;
    a.part_ws_floats = pw->floats;
    a.part_cnt = pw->cnt;
    a.part_cnt_n = pw->n;
  }
  a.num_sms = num_sms(L->device);
  a.stream = static_cast<cudaStream_t>(stream);
  QVLA_CUDA(qvla::launch_gemm_w4a4(a), "gemm launch");
  return QVLA_OK;
}
}  // namespace

extern "C" {

qvla_status qvla_gemm_w4a4(const qvla_layer* L, const uint8_t* xq, const float* xscale, const int32_t* xsum, int M, void* y,
                           int32_t* acc, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_rows(M)) return s;
  if (M == 0) return QVLA_OK;
  if (!xq || !xscale || !xsum || !y) return fail(QVLA_ERR_INVALID_ARG, "xq, xscale, xsum and y must not be NULL");
  if (!aligned16(xq) || !aligned16(y) || !aligned16(acc))
    return fail(QVLA_ERR_INVALID_ARG, "xq, y and acc must be 16-byte aligned");
  return launch_gemm(L, xq, 0, xscale, xsum, M, y, acc, stream);
}

namespace {
// The linear's workspace: what it needs, and the optional room for the GEMM's split of K.
size_t workspace_min(const qvla_layer* L, int M) {
  // the codes travel between the two kernels as one operand byte each; then the scales, the
  // code sums and the per-group code sums (used with per-group step scales)
  return round256(static_cast<size_t>(M) * L->K) + round256(static_cast<size_t>(M) * 4) * 2 +
         round256(static_cast<size_t>(M) * L->G * 4) + (L->rblock ? round256(rotated_bytes(L, M)) : 0);
}
constexpr int kMaxParts = 4;  // work units per tile of the GEMM's split of K
// The GEMM's split of K: a non-gated token-major layer (M > 128) whose 128 x 256 tiles leave SMs
// idle may split; room for kMaxParts FP32 partials of every output (rows and weight rows padded to
// 256) and a count for each 128 x 128 tile covers every tile shape it can take.
bool may_split_mn(int M, int N, bool gated, int sms) {
  if (M <= 128 || gated) return false;
  return static_cast<long>((M + 127) / 128) * ((N + 255) / 256) < sms;
}
size_t split_floats_mn(int M, int N) {
  return static_cast<size_t>((M + 255) / 256) * 256 * ((N + 255) / 256) * 256 * kMaxParts;
}
int split_counts_mn(int M, int N) { return ((M + 127) / 128) * ((N + 127) / 128); }
bool may_split(const qvla_layer* L, int M) { return may_split_mn(M, L->N, L->gated != 0, num_sms(L->device)); }
size_t split_floats(const qvla_layer* L, int M) { return split_floats_mn(M, L->N); }
int split_counts(const qvla_layer* L, int M) { return split_counts_mn(M, L->N); }
size_t workspace_parts(const qvla_layer* L, int M) {
  if (!may_split(L, M)) return 0;
  return round256(split_floats(L, M) * 4) + round256(static_cast<size_t>(split_counts(L, M)) * 4);
}
}  // namespace

size_t qvla_linear_workspace_bytes(const qvla_layer* L, int M) {
  if (!L || M <= 0) return 0;
  return workspace_min(L, M) + workspace_parts(L, M);
}

namespace {
struct LinearWorkspace {
  uint8_t* xb;       // [M][K] operand bytes
  float* xscale;     // [M]
  int32_t* xsum;     // [M]
  int32_t* xgsum;    // [M][G]
  void* xrot;        // [M][K] x . P . BlockDiag(U_b) in the activation dtype (layers with an online rotation)
  PartWorkspace parts;  // the GEMM's split of K (empty when the workspace has no room for it)
};

qvla_status carve_workspace(const qvla_layer* L, int M, void* workspace, size_t workspace_bytes, LinearWorkspace* w) {
  if (!workspace) return fail(QVLA_ERR_INVALID_ARG, "workspace must not be NULL");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return fail(QVLA_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const size_t need = workspace_min(L, M);
  if (workspace_bytes < need)
    return fail(QVLA_ERR_INVALID_ARG, "workspace of %zu bytes is smaller than the %zu needed", workspace_bytes, need);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  w->xb = ws;
  w->xscale = reinterpret_cast<float*>(ws + round256(static_cast<size_t>(M) * L->K));
  w->xsum = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(w->xscale) + round256(static_cast<size_t>(M) * 4));
  w->xgsum = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(w->xsum) + round256(static_cast<size_t>(M) * 4));
  w->xrot = reinterpret_cast<uint8_t*>(w->xgsum) + round256(static_cast<size_t>(M) * L->G * 4);
  const size_t parts = workspace_parts(L, M);
  if (parts > 0 && workspace_bytes >= need + parts) {  // room for the GEMM's split of K
    w->parts.ws = reinterpret_cast<float*>(ws + need);
    w->parts.floats = split_floats(L, M);
    w->parts.cnt = reinterpret_cast<int32_t*>(ws + need + round256(w->parts.floats * 4));
    w->parts.n = split_counts(L, M);
  }
  return QVLA_OK;
}

// The activations the quantiser sees: x itself, or x . P . BlockDiag(U_b) formed in the workspace
// when the layer carries an online rotation.
qvla_status online_input(const qvla_layer* L, const void* x, int M, const LinearWorkspace& w, void* stream,
                         const void** xin) {
  *xin = x;
  if (!L->rblock) return QVLA_OK;
  QVLA_CUDA(qvla::launch_block_rotate(x, L->xdt, M, L->K, L->rperm, L->rrot, L->rblock, w.xrot,
                                      static_cast<cudaStream_t>(stream)),
            "online rotation launch");
  *xin = w.xrot;
  return QVLA_OK;
}
}  // namespace

qvla_status qvla_linear_quantize(const qvla_layer* L, const void* x, int M, int step, void* workspace,
                                 size_t workspace_bytes, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_rows(M)) return s;
  const float* ss = nullptr;
  if (qvla_status s = resolve_step(L, step, &ss)) return s;
  if (ss && L->grouped)
    return fail(QVLA_ERR_UNSUPPORTED, "per-group step scales run through qvla_w4a4_linear (the halves carry no step)");
  if (M == 0) return QVLA_OK;
  if (!x) return fail(QVLA_ERR_INVALID_ARG, "x must not be NULL");
  if (!aligned16(x)) return fail(QVLA_ERR_INVALID_ARG, "x must be 16-byte aligned");
  LinearWorkspace w;
  if (qvla_status s = carve_workspace(L, M, workspace, workspace_bytes, &w)) return s;
  const void* xin = nullptr;
  if (qvla_status s = online_input(L, x, M, w, stream, &xin)) return s;
  // (the rotate-quantise kernel also clears the GEMM's counters of the split of K)
  return launch_rq(xin, L->xdt, M, L->K, L->had_block, ss ? 1 : 0, ss, w.xb, w.xscale, w.xsum, nullptr, stream, 1, 0,
                   nullptr, w.parts.cnt, w.parts.n);
}

qvla_status qvla_linear_gemm(const qvla_layer* L, void* workspace, size_t workspace_bytes, int M, void* y,
                             void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_rows(M)) return s;
  if (M == 0) return QVLA_OK;
  if (!y) return fail(QVLA_ERR_INVALID_ARG, "y must not be NULL");
  if (!aligned16(y)) return fail(QVLA_ERR_INVALID_ARG, "y must be 16-byte aligned");
  LinearWorkspace w;
  if (qvla_status s = carve_workspace(L, M, workspace, workspace_bytes, &w)) return s;
  return launch_gemm(L, w.xb, 1, w.xscale, w.xsum, M, y, nullptr, stream, nullptr, nullptr, &w.parts);
}

namespace {
// The one-launch linear (fused rotate + quantise prologue in the GEMM) where the layer and batch
// allow it: a per-step scale (one per tensor), no online P.U, not gated, f16/bf16 activations,
// M <= 128.  *launched tells whether it was enqueued.
qvla_status try_fused(const qvla_layer* L, const void* x, int M, const float* step_scale, void* y, void* stream,
                      bool* launched) {
  *launched = false;
  if (!step_scale || L->grouped || L->rblock || L->gated || M > 128 || (L->xdt != QVLA_F16 && L->xdt != QVLA_BF16))
    return QVLA_OK;
  qvla::GemmArgs a;
  a.xq = nullptr;
  a.x_bytes = 3;
  a.xscale = step_scale;
  a.xsum = nullptr;
  a.wq = L->wq;
  a.wscale = L->wscale;
  a.wcorr = L->wcorr;
  a.bias = L->bias;
  a.y = y;
  a.ydt = L->ydt;
  a.acc = nullptr;
  a.M = M;
  a.N = L->N;
  a.K = L->K;
  a.gated = 0;
  a.x = x;
  a.xdt = L->xdt;
  a.log_b = L->log_b;
  a.inv_sqrt_b = static_cast<float>(1.0 / std::sqrt(static_cast<double>(L->had_block)));
  a.num_sms = num_sms(L->device);
  a.stream = static_cast<cudaStream_t>(stream);
  QVLA_CUDA(qvla::launch_gemm_fused(a, launched), "fused linear launch");
  return QVLA_OK;
}

// Decode-sized batches (M <= 4): one launch of the CUDA-core GEMV that rotates and quantises the
// activations itself, where the layer allows it (f16/bf16 input and output of one dtype,
// Hadamard block <= 2048, no per-group step tables, the CTA's working set within its shared
// memory).  The outputs are those of the rotate-quantise kernel followed by the GEMM, bit for bit.
qvla_status try_gemv_fused(const qvla_layer* L, const void* x, int M, const float* step_scale, void* y, void* stream,
                           bool* launched) {
  *launched = false;
  if (M > qvla::kGemvMaxM || (step_scale && L->grouped) || L->xdt != L->ydt ||
      (L->xdt != QVLA_F16 && L->xdt != QVLA_BF16))
    return QVLA_OK;
  qvla::GemmArgs a;
  a.xq = nullptr;
  a.x_bytes = 3;
  a.xscale = step_scale;
  a.xsum = nullptr;
  a.wq = L->wq;
  a.wscale = L->wscale;
  a.wcorr = L->wcorr;
  a.bias = L->bias;
  a.y = y;
  a.ydt = L->ydt;
  a.acc = nullptr;
  a.M = M;
  a.N = L->N;
  a.K = L->K;
  a.gated = L->gated;
  a.x = x;
  a.xdt = L->xdt;
  a.log_b = L->log_b;
  a.inv_sqrt_b = static_cast<float>(1.0 / std::sqrt(static_cast<double>(L->had_block)));
  a.num_sms = num_sms(L->device);
  a.stream = static_cast<cudaStream_t>(stream);
  QVLA_CUDA(qvla::launch_gemv_w4a4(a, launched), "decode linear launch");
  return QVLA_OK;
}
}  // namespace

qvla_status qvla_w4a4_linear_fused(const qvla_layer* L, const void* x, int M, int step, void* y, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_rows(M)) return s;
  if (step < 0) return fail(QVLA_ERR_UNSUPPORTED, "the one-launch linear takes a per-step scale (step >= 0)");
  const float* ss = nullptr;
  if (qvla_status s = resolve_step(L, step, &ss)) return s;
  if (M == 0) return QVLA_OK;
  if (!x || !y) return fail(QVLA_ERR_INVALID_ARG, "x and y must not be NULL");
  if (!aligned16(x) || !aligned16(y)) return fail(QVLA_ERR_INVALID_ARG, "x and y must be 16-byte aligned");
  if (qvla_status s = check_layer_device(L)) return s;
  bool launched = false;
  if (qvla_status s = try_fused(L, x, M, ss, y, stream, &launched)) return s;
  if (!launched)
    return fail(QVLA_ERR_UNSUPPORTED,
                "the one-launch linear does not take this layer or batch (M=%d, K=%d, N=%d): use qvla_w4a4_linear", M,
                L->K, L->N);
  return QVLA_OK;
}

qvla_status qvla_w4a4_linear(const qvla_layer* L, const void* x, int M, int step, void* y, void* workspace,
                             size_t workspace_bytes, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_rows(M)) return s;
  const float* ss = nullptr;
  if (qvla_status s = resolve_step(L, step, &ss)) return s;
  if (M == 0) return QVLA_OK;
  if (!x || !y) return fail(QVLA_ERR_INVALID_ARG, "x and y must not be NULL");
  if (!aligned16(x) || !aligned16(y)) return fail(QVLA_ERR_INVALID_ARG, "x and y must be 16-byte aligned");
  LinearWorkspace w;
  if (qvla_status s = carve_workspace(L, M, workspace, workspace_bytes, &w)) return s;
  const void* xin = nullptr;
  if (qvla_status s = online_input(L, x, M, w, stream, &xin)) return s;
  bool launched = false;  // one to four tokens: a single launch where the layer allows it
  if (qvla_status s = try_gemv_fused(L, xin, M, ss, y, stream, &launched)) return s;
  if (launched) return QVLA_OK;
  if (ss && L->grouped) {  // per-group step scales: per-group codes and sums, promoted per group
    if (qvla_status s = launch_rq(xin, L->xdt, M, L->K, L->had_block, 1, ss, w.xb, w.xscale, nullptr, nullptr, stream, 1,
                                  L->group, w.xgsum))
      return s;
    return launch_gemm(L, w.xb, 1, w.xscale, w.xsum, M, y, nullptr, stream, ss, w.xgsum);
  }
  if (qvla_status s = launch_rq(xin, L->xdt, M, L->K, L->had_block, ss ? 1 : 0, ss, w.xb, w.xscale, w.xsum, nullptr,
                                stream, 1, 0, nullptr, w.parts.cnt, w.parts.n))
    return s;
  return launch_gemm(L, w.xb, 1, w.xscale, w.xsum, M, y, nullptr, stream, nullptr, nullptr, &w.parts);
}

}  // extern "C"

// ---- W4A8: 8-bit activation codes against the same int4 weights ----
namespace {
constexpr int kMaxKA8 = 4096;  // the FP32 accumulator is exact while 255 x 15 x K < 2^24

qvla_status check_a8(const qvla_layer* L) {
  if (L->K > kMaxKA8)
    return fail(QVLA_ERR_UNSUPPORTED, "K=%d: 8-bit activations need K <= %d (exact accumulation)", L->K, kMaxKA8);
  return QVLA_OK;
}

struct A8Workspace {
  uint8_t* planes;   // [M][2K] operand planes
  float* xscale;     // [M]
  int32_t* xsum;     // [M]
};

qvla_status carve_a8(const qvla_layer* L, int M, void* workspace, size_t workspace_bytes, A8Workspace* w) {
  if (!workspace) return fail(QVLA_ERR_INVALID_ARG, "workspace must not be NULL");
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return fail(QVLA_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  const size_t need = qvla_w4a8_workspace_bytes(L, M);
  if (workspace_bytes < need)
    return fail(QVLA_ERR_INVALID_ARG, "workspace of %zu bytes is smaller than the %zu needed", workspace_bytes, need);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  w->planes = ws;
  w->xscale = reinterpret_cast<float*>(ws + round256(static_cast<size_t>(M) * 2 * L->K));
  w->xsum = reinterpret_cast<int32_t*>(reinterpret_cast<uint8_t*>(w->xscale) + round256(static_cast<size_t>(M) * 4));
  return QVLA_OK;
}
}  // namespace

extern "C" {

size_t qvla_w4a8_workspace_bytes(const qvla_layer* L, int M) {
  if (!L || M <= 0) return 0;
  return round256(static_cast<size_t>(M) * 2 * L->K) + round256(static_cast<size_t>(M) * 4) * 2;
}

qvla_status qvla_w4a8_linear(const qvla_layer* L, const void* x, int M, int step, void* y, void* workspace,
                             size_t workspace_bytes, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_a8(L)) return s;
  if (qvla_status s = check_rows(M)) return s;
  const float* ss = nullptr;
  if (qvla_status s = resolve_step(L, step, &ss)) return s;
  if (ss && L->grouped) return fail(QVLA_ERR_UNSUPPORTED, "per-group step scales are for int4 activation codes");
  if (L->rblock)
    return fail(QVLA_ERR_UNSUPPORTED, "the layer's online rotation runs in qvla_w4a4_linear / qvla_linear_quantize");
  if (M == 0) return QVLA_OK;
  if (!x || !y) return fail(QVLA_ERR_INVALID_ARG, "x and y must not be NULL");
  if (!aligned16(x) || !aligned16(y)) return fail(QVLA_ERR_INVALID_ARG, "x and y must be 16-byte aligned");
  A8Workspace w;
  if (qvla_status s = carve_a8(L, M, workspace, workspace_bytes, &w)) return s;
  if (qvla_status s = launch_rq(x, L->xdt, M, L->K, L->had_block, ss ? 1 : 0, ss, w.planes, w.xscale, w.xsum, nullptr,
                                stream, 3))
    return s;
  return launch_gemm(L, w.planes, 2, w.xscale, w.xsum, M, y, nullptr, stream);
}

qvla_status qvla_gemm_w4a8(const qvla_layer* L, const int8_t* xq, const float* xscale, int M, void* y, int32_t* acc,
                           void* workspace, size_t workspace_bytes, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_a8(L)) return s;
  if (qvla_status s = check_rows(M)) return s;
  if (M == 0) return QVLA_OK;
  if (!xq || !xscale || !y) return fail(QVLA_ERR_INVALID_ARG, "xq, xscale and y must not be NULL");
  if (!aligned16(xq) || !aligned16(y) || !aligned16(acc))
    return fail(QVLA_ERR_INVALID_ARG, "xq, y and acc must be 16-byte aligned");
  A8Workspace w;
  if (qvla_status s = carve_a8(L, M, workspace, workspace_bytes, &w)) return s;
  QVLA_CUDA(qvla::launch_a8_planes(xq, M, L->K, w.planes, w.xsum, static_cast<cudaStream_t>(stream)), "a8 planes launch");
  return launch_gemm(L, w.planes, 2, xscale, w.xsum, M, y, acc, stream);
}

}  // extern "C"

// ---- allocation-free linear: a fixed scratch area in this translation unit ----
namespace {
static __device__ __align__(256) uint8_t g_noalloc_scratch[QVLA_NOALLOC_SCRATCH_BYTES];
std::mutex g_noalloc_mu;
std::vector<void*> g_noalloc_addr;  // device address of g_noalloc_scratch, per device

// The array's name in host code is only a host-side stand-in; its device address comes from
// cudaGetSymbolAddress, looked up once per device with that device current.
qvla_status noalloc_scratch(void** out) {
  int dev = 0;
  QVLA_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (dev >= static_cast<int>(g_noalloc_addr.size())) g_noalloc_addr.resize(dev + 1, nullptr);
  if (g_noalloc_addr[dev] == nullptr) {
    void* p = nullptr;
    QVLA_CUDA(cudaGetSymbolAddress(&p, g_noalloc_scratch), "cudaGetSymbolAddress of the no-alloc scratch");
    g_noalloc_addr[dev] = p;
  }
  *out = g_noalloc_addr[dev];
  return QVLA_OK;
}
}  // namespace

extern "C" {

qvla_status qvla_w4a4_linear_noalloc(const qvla_layer* L, const void* x, int M, int step, void* y, void* stream) {
  g_last_error.clear();
  if (!L) return fail(QVLA_ERR_INVALID_ARG, "layer must not be NULL");
  if (qvla_status s = check_layer_device(L)) return s;  // the scratch looked up is the current device's
  if (qvla_status s = check_rows(M)) return s;
  // the scratch holds what the linear needs; the GEMM's split of K runs only where it fits as well
  const size_t need = workspace_min(L, M);
  if (need > QVLA_NOALLOC_SCRATCH_BYTES)
    return fail(QVLA_ERR_UNSUPPORTED, "M=%d, K=%d needs %zu bytes of scratch; the allocation-free linear holds %zu", M, L->K,
                need, static_cast<size_t>(QVLA_NOALLOC_SCRATCH_BYTES));
  if (M == 0) return qvla_w4a4_linear(L, x, M, step, y, nullptr, 0, stream);
  void* scratch = nullptr;
  if (qvla_status s = noalloc_scratch(&scratch)) return s;
  return qvla_w4a4_linear(L, x, M, step, y, scratch, QVLA_NOALLOC_SCRATCH_BYTES, stream);
}

qvla_status qvla_debug_set_hooks(unsigned long long wait_limit_ns, int hold_gemm_loads) {
  g_last_error.clear();
  const unsigned long long limit = wait_limit_ns ? wait_limit_ns : 2000000000ull;
  const int hold = hold_gemm_loads ? 1 : 0;
  QVLA_CUDA(qvla::set_debug_hooks_gemm(limit, hold), "test hooks (gemm)");
  QVLA_CUDA(qvla::set_debug_hooks_fused(limit, hold), "test hooks (fused)");
  QVLA_CUDA(qvla::set_debug_hooks_gemv(limit, hold), "test hooks (gemv)");
  QVLA_CUDA(qvla::set_debug_hooks_rqp(limit, hold), "test hooks (rotate-quantise)");
  return QVLA_OK;
}

qvla_status qvla_debug_gemm_plan(int M, int K, int N, int gated, int sms, int split_room, int* shape, int* parts) {
  g_last_error.clear();
  if (!shape || !parts) return fail(QVLA_ERR_INVALID_ARG, "shape and parts must not be NULL");
  if (M <= 128) return fail(QVLA_ERR_INVALID_ARG, "M=%d: up to 128 rows run weight-major, not token-major", M);
  if (K <= 0 || K % 128 != 0) return fail(QVLA_ERR_INVALID_ARG, "K=%d must be a positive multiple of 128", K);
  if (N <= 0 || N % 16 != 0 || (gated && N % 256 != 0))
    return fail(QVLA_ERR_INVALID_ARG, "N=%d must be a positive multiple of 16 (of 256 when gated)", N);
  if (sms < 2) return fail(QVLA_ERR_INVALID_ARG, "num_sms=%d must be at least 2", sms);
  qvla::GemmArgs a = {};
  a.x_bytes = 1;
  a.M = M;
  a.N = N;
  a.K = K;
  a.gated = gated ? 1 : 0;
  a.num_sms = sms;
  static float no_floats;  // stand-ins for the workspace: the plan reads only whether it is there
  static int no_counts;
  if (split_room && may_split_mn(M, N, gated != 0, sms)) {
    a.part_ws = &no_floats;
    a.part_ws_floats = split_floats_mn(M, N);
    a.part_cnt = &no_counts;
    a.part_cnt_n = split_counts_mn(M, N);
  }
  *shape = qvla::token_major_plan(a, parts);
  return QVLA_OK;
}

qvla_status qvla_check_device(void* stream) {
  g_last_error.clear();
  unsigned int word = 0, word_fused = 0, word_gemv = 0, word_rqp = 0;
  QVLA_CUDA(qvla::read_and_clear_error_word(&word, static_cast<cudaStream_t>(stream)), "device check");
  QVLA_CUDA(qvla::read_and_clear_error_word_fused(&word_fused, static_cast<cudaStream_t>(stream)), "device check");
  QVLA_CUDA(qvla::read_and_clear_error_word_gemv(&word_gemv, static_cast<cudaStream_t>(stream)), "device check");
  QVLA_CUDA(qvla::read_and_clear_error_word_rqp(&word_rqp, static_cast<cudaStream_t>(stream)), "device check");
  if ((word | word_fused | word_gemv | word_rqp) & 1u)
    return fail(QVLA_ERR_TIMEOUT, "a kernel wait ran out of its time limit");
  return QVLA_OK;
}

}  // extern "C"
