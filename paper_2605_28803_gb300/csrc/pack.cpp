// Offline weight preparation on the host (Sec. 4.1 Eq. 4-5 fold; Sec. 4.2 Eq. 5-6 per output
// channel): W'_n = W_n . P . BlockDiag(U_b) . BlockDiag(H_b / sqrt(b)) in float64, rounded once
// to float32, then Delta_W[n] = max |W'_n| / 7 (float32) and int4 codes
// clamp(round(W'/Delta_W), -7, 7) rounded half to even on the exact quotient, nibble-packed.
// The Hadamard factor is applied with an in-place radix-2 fast transform.
//
// Also the offline choice of P and U_b (Sec. 4.1, after Eq. 4): the zigzag channel permutation
// by weight energy, and per block of input channels the left singular vectors of the block's
// row partition, found as the eigenvectors of its Gram matrix by cyclic Jacobi rotations.
//
// And the LLM side's GPTQ-style codes (Sec. 5.1: block size 128, damping ratio 0.01), from the
// published GPTQ algorithm: the RTN scale per output row, then the columns in order, each
// column's rounding error fed forward through the upper Cholesky factor of the damped inverse
// Hessian of calibration activations in the folded basis.
#include "pack.h"

#include <algorithm>
#include <atomic>
#include <cfenv>
#include <cmath>
#include <cstring>
#include <thread>
#include <vector>

namespace qvla {
namespace {

float half_to_float(uint16_t h) {
  const uint32_t sign = static_cast<uint32_t>(h & 0x8000u) << 16;
  const uint32_t exp = (h >> 10) & 0x1Fu;
  const uint32_t man = h & 0x3FFu;
  uint32_t bits;
  if (exp == 0) {
    if (man == 0) {
      bits = sign;
    } else {  // subnormal: man * 2^-24
      float f = std::ldexp(static_cast<float>(man), -24);
      std::memcpy(&bits, &f, 4);
      bits |= sign;
    }
  } else if (exp == 31) {
    bits = sign | 0x7F800000u | (man << 13);
  } else {
    bits = sign | ((exp + 112u) << 23) | (man << 13);
  }
  float f;
  std::memcpy(&f, &bits, 4);
  return f;
}

float bf16_to_float(uint16_t b) {
  const uint32_t bits = static_cast<uint32_t>(b) << 16;
  float f;
  std::memcpy(&f, &bits, 4);
  return f;
}

double load_elem(const void* W, int wdt, size_t i) {
  switch (wdt) {
    case 0: return half_to_float(static_cast<const uint16_t*>(W)[i]);
    case 1: return bf16_to_float(static_cast<const uint16_t*>(W)[i]);
    default: return static_cast<const float*>(W)[i];
  }
}

// In-place fast Walsh-Hadamard transform of n = 2^k doubles (Sylvester order), unnormalised.
void fwht(double* v, int n) {
  for (int h = 1; h < n; h <<= 1)
    for (int i = 0; i < n; i += 2 * h)
      for (int j = i; j < i + h; ++j) {
        const double a = v[j], c = v[j + h];
        v[j] = a + c;
        v[j + h] = a - c;
      }
}

// Round half to even of the exact quotient z / d for float32 z and d > 0: the float64 quotient
// lies at least 2^-25 (relative) from any half-integer it is not equal to, so the float64
// nearest-even rounding takes the exact decision.
int quantize_code(float z, float d) {
  if (!(d > 0.0f)) return 0;
  const double t = static_cast<double>(z) / static_cast<double>(d);
  if (std::isnan(t)) return 0;
  double r = std::nearbyint(t);  // default rounding mode: to nearest, ties to even
  r = std::min(7.0, std::max(-7.0, r));
  return static_cast<int>(r);
}

// Row n of a [rows][K] matrix times P . BlockDiag(U_b) . BlockDiag(H_b / sqrt(b)) into a (float64);
// b is scratch.  The same product folds a weight row (Eq. 5) and rotates an activation row.
void fold_row(const void* W, int wdt, int K, int n, const double* rot, int rot_block, const int32_t* perm,
              int had_block, std::vector<double>& a, std::vector<double>& b) {
  const size_t base = static_cast<size_t>(n) * K;
  for (int k = 0; k < K; ++k) a[k] = load_elem(W, wdt, base + (perm ? perm[k] : k));
  if (rot) {
    std::fill(b.begin(), b.end(), 0.0);
    for (int blk = 0; blk < K / rot_block; ++blk) {
      const double* u = rot + static_cast<size_t>(blk) * rot_block * rot_block;
      const double* x = a.data() + static_cast<size_t>(blk) * rot_block;
      double* o = b.data() + static_cast<size_t>(blk) * rot_block;
      for (int i = 0; i < rot_block; ++i) {
        const double xi = x[i];
        if (xi == 0.0) continue;
        const double* urow = u + static_cast<size_t>(i) * rot_block;
        for (int j = 0; j < rot_block; ++j) o[j] += xi * urow[j];
      }
    }
    a.swap(b);
  }
  if (had_block > 1) {
    const double s = 1.0 / std::sqrt(static_cast<double>(had_block));
    for (int blk = 0; blk < K / had_block; ++blk) {
      double* v = a.data() + static_cast<size_t>(blk) * had_block;
      fwht(v, had_block);
      for (int i = 0; i < had_block; ++i) v[i] *= s;
    }
  }
}

void pack_row(const void* W, int wdt, int K, int n, const double* rot, int rot_block, const int32_t* perm,
              int had_block, std::vector<double>& a, std::vector<double>& b, std::vector<float>& f, uint8_t* wq,
              float* wscale, int32_t* wsum) {
  fold_row(W, wdt, K, n, rot, rot_block, perm, had_block, a, b);
  float amax = 0.0f;
  for (int k = 0; k < K; ++k) {
    f[k] = static_cast<float>(a[k]);
    amax = std::max(amax, std::fabs(f[k]));
  }
  const float d = amax / 7.0f;
  wscale[n] = d;
  int32_t sum = 0;
  uint8_t* row = wq + static_cast<size_t>(n) * (K / 2);
  for (int k = 0; k < K; k += 2) {
    const int q0 = quantize_code(f[k], d), q1 = quantize_code(f[k + 1], d);
    sum += q0 + q1;
    row[k / 2] = static_cast<uint8_t>((q0 & 0xF) | ((q1 & 0xF) << 4));
  }
  if (wsum) wsum[n] = sum;
}

}  // namespace

void pack_weights_host_impl(const void* W, int wdt, int N, int K, const double* rot, int rot_block,
                            const int32_t* perm, int had_block, uint8_t* wq, float* wscale, int32_t* wsum) {
  std::fesetround(FE_TONEAREST);
  unsigned nt = std::max(1u, std::min(32u, std::thread::hardware_concurrency()));
  nt = std::min<unsigned>(nt, static_cast<unsigned>(std::max(1, N)));
  std::atomic<int> next{0};
  auto worker = [&]() {
    std::fesetround(FE_TONEAREST);
    std::vector<double> a(K), b(K);
    std::vector<float> f(K);
    for (;;) {
      const int n = next.fetch_add(1);
      if (n >= N) break;
      pack_row(W, wdt, K, n, rot, rot_block, perm, had_block, a, b, f, wq, wscale, wsum);
    }
  };
  std::vector<std::thread> pool;
  for (unsigned i = 1; i < nt; ++i) pool.emplace_back(worker);
  worker();
  for (auto& t : pool) t.join();
}

namespace {

// Eigen-decomposition of a symmetric c x c matrix a (row-major, destroyed) by cyclic Jacobi
// rotations: on return the eigenvalues are on a's diagonal and v's column j is the unit
// eigenvector of eigenvalue a[j][j].  Each rotation zeroes one off-diagonal pair exactly in
// exact arithmetic; sweeps repeat until the off-diagonal mass is negligible.
void jacobi_eigen(std::vector<double>& a, std::vector<double>& v, int c) {
  v.assign(static_cast<size_t>(c) * c, 0.0);
  for (int i = 0; i < c; ++i) v[static_cast<size_t>(i) * c + i] = 1.0;
  auto A = [&](int i, int j) -> double& { return a[static_cast<size_t>(i) * c + j]; };
  auto V = [&](int i, int j) -> double& { return v[static_cast<size_t>(i) * c + j]; };
  double total = 0.0;
  for (int i = 0; i < c; ++i)
    for (int j = 0; j < c; ++j) total += A(i, j) * A(i, j);
  for (int sweep = 0; sweep < 100; ++sweep) {
    double off = 0.0;
    for (int p = 0; p < c; ++p)
      for (int q = p + 1; q < c; ++q) off += A(p, q) * A(p, q);
    if (off <= 1e-32 * total) break;
    for (int p = 0; p < c - 1; ++p)
      for (int q = p + 1; q < c; ++q) {
        const double apq = A(p, q);
        if (apq == 0.0) continue;
        // the rotation angle that zeroes A(p, q): t = tan(phi), the smaller root
        const double theta = (A(q, q) - A(p, p)) / (2.0 * apq);
        const double t = (theta >= 0.0 ? 1.0 : -1.0) / (std::fabs(theta) + std::sqrt(theta * theta + 1.0));
        const double cs = 1.0 / std::sqrt(t * t + 1.0), sn = t * cs;
        for (int k = 0; k < c; ++k) {  // columns p and q
          const double akp = A(k, p), akq = A(k, q);
          A(k, p) = cs * akp - sn * akq;
          A(k, q) = sn * akp + cs * akq;
        }
        for (int k = 0; k < c; ++k) {  // rows p and q
          const double apk = A(p, k), aqk = A(q, k);
          A(p, k) = cs * apk - sn * aqk;
          A(q, k) = sn * apk + cs * aqk;
        }
        for (int k = 0; k < c; ++k) {
          const double vkp = V(k, p), vkq = V(k, q);
          V(k, p) = cs * vkp - sn * vkq;
          V(k, q) = sn * vkp + cs * vkq;
        }
      }
  }
}

}  // namespace

void zigzag_permutation_host(const void* W, int wdt, int N, int K, int block, int32_t* perm) {
  std::vector<double> energy(K, 0.0);
  for (int n = 0; n < N; ++n)
    for (int k = 0; k < K; ++k) {
      const double w = load_elem(W, wdt, static_cast<size_t>(n) * K + k);
      energy[k] += w * w;
    }
  std::vector<int> order(K);
  for (int k = 0; k < K; ++k) order[k] = k;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return energy[a] > energy[b]; });
  const int nb = K / block;
  for (int i = 0; i < K; ++i) {
    const int r = i / nb, pos = i % nb;
    const int b = (r % 2 == 0) ? pos : nb - 1 - pos;
    perm[b * block + r] = order[i];
  }
}

void block_svd_rotation_host(const void* W, int wdt, int N, int K, int block, const int32_t* perm, double* rot) {
  const int nb = K / block;
  unsigned nt = std::max(1u, std::min(32u, std::thread::hardware_concurrency()));
  nt = std::min<unsigned>(nt, static_cast<unsigned>(std::max(1, nb)));
  std::atomic<int> next{0};
  auto worker = [&]() {
    std::vector<double> wb(static_cast<size_t>(N) * block), g(static_cast<size_t>(block) * block), v;
    std::vector<int> idx(block);
    for (;;) {
      const int b = next.fetch_add(1);
      if (b >= nb) break;
      // the block's input channels (after P) for every output row
      for (int n = 0; n < N; ++n)
        for (int i = 0; i < block; ++i) {
          const int k = b * block + i;
          wb[static_cast<size_t>(n) * block + i] = load_elem(W, wdt, static_cast<size_t>(n) * K + (perm ? perm[k] : k));
        }
      // Gram matrix of the paper's row partition W_b (block x N): G = W_b W_b^T
      std::fill(g.begin(), g.end(), 0.0);
      for (int n = 0; n < N; ++n) {
        const double* row = wb.data() + static_cast<size_t>(n) * block;
        for (int i = 0; i < block; ++i) {
          const double ri = row[i];
          for (int j = i; j < block; ++j) g[static_cast<size_t>(i) * block + j] += ri * row[j];
        }
      }
      for (int i = 0; i < block; ++i)
        for (int j = 0; j < i; ++j) g[static_cast<size_t>(i) * block + j] = g[static_cast<size_t>(j) * block + i];
      jacobi_eigen(g, v, block);
      // columns by descending eigenvalue (= sigma^2), each with its largest entry positive
      for (int i = 0; i < block; ++i) idx[i] = i;
      std::stable_sort(idx.begin(), idx.end(), [&](int a, int c) {
        return g[static_cast<size_t>(a) * block + a] > g[static_cast<size_t>(c) * block + c];
      });
      double* u = rot + static_cast<size_t>(b) * block * block;
      for (int j = 0; j < block; ++j) {
        const int src = idx[j];
        int arg = 0;
        for (int i = 1; i < block; ++i)
          if (std::fabs(v[static_cast<size_t>(i) * block + src]) > std::fabs(v[static_cast<size_t>(arg) * block + src])) arg = i;
        const double sgn = v[static_cast<size_t>(arg) * block + src] < 0.0 ? -1.0 : 1.0;
        for (int i = 0; i < block; ++i) u[static_cast<size_t>(i) * block + j] = sgn * v[static_cast<size_t>(i) * block + src];
      }
    }
  };
  std::vector<std::thread> pool;
  for (unsigned i = 1; i < nt; ++i) pool.emplace_back(worker);
  worker();
  for (auto& t : pool) t.join();
}

namespace {

// Runs fn(i) for i in [0, n) on up to 32 threads (contiguous chunks).
template <typename F>
void parallel_for(int n, F fn) {
  if (n <= 0) return;
  unsigned nt = std::max(1u, std::min(32u, std::thread::hardware_concurrency()));
  nt = std::min<unsigned>(nt, static_cast<unsigned>(n));
  if (nt == 1 || n < 64) {
    for (int i = 0; i < n; ++i) fn(i);
    return;
  }
  std::atomic<int> next{0};
  auto worker = [&]() {
    std::fesetround(FE_TONEAREST);
    for (;;) {
      const int i0 = next.fetch_add(16);
      if (i0 >= n) break;
      for (int i = i0; i < std::min(n, i0 + 16); ++i) fn(i);
    }
  };
  std::vector<std::thread> pool;
  for (unsigned t = 1; t < nt; ++t) pool.emplace_back(worker);
  worker();
  for (auto& t : pool) t.join();
}

}  // namespace

bool gptq_pack_host(const void* W, int wdt, int N, int K, const void* X, int xdt, int n_cal, const double* rot,
                    int rot_block, const int32_t* perm, int had_block, int block, double damp, uint8_t* wq,
                    float* wscale, int32_t* wsum) {
  std::fesetround(FE_TONEAREST);
  const size_t KK = static_cast<size_t>(K) * K;
  // calibration rows in the folded basis, stored transposed [K][n_cal] for the Hessian's dot products
  std::vector<double> xt(static_cast<size_t>(K) * n_cal);
  {
    std::vector<double> a(K), b(K);
    for (int r = 0; r < n_cal; ++r) {
      fold_row(X, xdt, K, r, rot, rot_block, perm, had_block, a, b);
      for (int k = 0; k < K; ++k) xt[static_cast<size_t>(k) * n_cal + r] = a[k];
    }
  }
  // H = 2/n X'^T X' (both triangles)
  std::vector<double> h(KK);
  const double c2 = 2.0 / n_cal;
  parallel_for(K, [&](int i) {
    const double* xi = xt.data() + static_cast<size_t>(i) * n_cal;
    for (int j = i; j < K; ++j) {
      const double* xj = xt.data() + static_cast<size_t>(j) * n_cal;
      double acc = 0.0;
      for (int r = 0; r < n_cal; ++r) acc += xi[r] * xj[r];
      h[static_cast<size_t>(i) * K + j] = c2 * acc;
    }
  });
  for (int i = 0; i < K; ++i)
    for (int j = 0; j < i; ++j) h[static_cast<size_t>(i) * K + j] = h[static_cast<size_t>(j) * K + i];
  xt.clear();
  xt.shrink_to_fit();
  // dead columns and damping
  std::vector<char> dead(K, 0);
  double mean_diag = 0.0;
  for (int k = 0; k < K; ++k) {
    double& d = h[static_cast<size_t>(k) * K + k];
    if (d == 0.0) {
      dead[k] = 1;
      d = 1.0;
    }
    mean_diag += d;
  }
  mean_diag /= K;
  for (int k = 0; k < K; ++k) h[static_cast<size_t>(k) * K + k] += damp * mean_diag;
  // H = T T^T with T upper triangular (Cholesky in reversed index order), in place in H's
  // upper triangle; then U = T^-1 is upper triangular with H^-1 = U^T U, the factor GPTQ uses.
  for (int j = K - 1; j >= 0; --j) {
    double* hj = h.data() + static_cast<size_t>(j) * K;
    double djj = hj[j];
    for (int k = j + 1; k < K; ++k) djj -= hj[k] * hj[k];
    if (!(djj > 0.0)) return false;
    const double tjj = std::sqrt(djj);
    hj[j] = tjj;
    parallel_for(j, [&](int i) {
      double* hi = h.data() + static_cast<size_t>(i) * K;
      double v = hi[j];
      for (int k = j + 1; k < K; ++k) v -= hi[k] * hj[k];
      hi[j] = v / tjj;
    });
  }
  std::vector<double> u(KK, 0.0);  // U = T^-1, column by column: T U[:, c] = e_c
  parallel_for(K, [&](int c) {
    u[static_cast<size_t>(c) * K + c] = 1.0 / h[static_cast<size_t>(c) * K + c];
    for (int i = c - 1; i >= 0; --i) {
      const double* hi = h.data() + static_cast<size_t>(i) * K;
      double v = 0.0;
      for (int k = i + 1; k <= c; ++k) v += hi[k] * u[static_cast<size_t>(k) * K + c];
      u[static_cast<size_t>(i) * K + c] = -v / hi[i];
    }
  });
  h.clear();
  h.shrink_to_fit();
  // each output row: the folded weights rounded to float32, the RTN scale, then the columns in
  // order with error feedback; updates past the current block of columns are batched per block
  parallel_for(N, [&](int n) {
    std::vector<double> a(K), b(K), err(block);
    fold_row(W, wdt, K, n, rot, rot_block, perm, had_block, a, b);
    float amax = 0.0f;
    for (int k = 0; k < K; ++k) {
      const float f = static_cast<float>(a[k]);
      a[k] = dead[k] ? 0.0 : static_cast<double>(f);
      amax = std::max(amax, std::fabs(f));
    }
    const float d32 = amax / 7.0f;
    const double d = d32;
    wscale[n] = d32;
    int32_t sum = 0;
    uint8_t* row = wq + static_cast<size_t>(n) * (K / 2);
    for (int i1 = 0; i1 < K; i1 += block) {
      const int i2 = std::min(K, i1 + block);
      for (int i = i1; i < i2; ++i) {
        const double* ui = u.data() + static_cast<size_t>(i) * K;
        double q = 0.0;
        if (d > 0.0) q = std::min(7.0, std::max(-7.0, std::nearbyint(a[i] / d)));
        const int qi = static_cast<int>(q);
        sum += qi;
        if (i & 1) {
          row[i / 2] = static_cast<uint8_t>(row[i / 2] | ((qi & 0xF) << 4));
        } else {
          row[i / 2] = static_cast<uint8_t>(qi & 0xF);
        }
        const double e = (a[i] - d * q) / ui[i];
        err[i - i1] = e;
        for (int j = i; j < i2; ++j) a[j] -= e * ui[j];
      }
      for (int i = i1; i < i2; ++i) {
        const double e = err[i - i1];
        const double* ui = u.data() + static_cast<size_t>(i) * K;
        for (int j = i2; j < K; ++j) a[j] -= e * ui[j];
      }
    }
    if (wsum) wsum[n] = sum;
  });
  return true;
}

void code_sums_host(const uint8_t* wq, int N, int K, int32_t* wsum) {
  for (int n = 0; n < N; ++n) {
    const uint8_t* row = wq + static_cast<size_t>(n) * (K / 2);
    int32_t s = 0;
    for (int j = 0; j < K / 2; ++j) {
      int lo = row[j] & 0xF, hi = row[j] >> 4;
      s += (lo >= 8 ? lo - 16 : lo) + (hi >= 8 ? hi - 16 : hi);
    }
    wsum[n] = s;
  }
}

}  // namespace qvla
