// Host-side AATC planner: calibration statistics, eigenbasis, attention-aware weights,
// integer reverse water-filling and per-channel scales (Sec. 5 Steps 1-2; Algorithm 1,
// calibration half).  Plain C++17, fp64, no LAPACK: the eigenbasis comes from a cyclic
// Jacobi iteration on the 128x128 second-moment matrix.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <numeric>
#include <queue>
#include <thread>
#include <vector>

#include "aatc.h"
#include "aatc_internal.h"

namespace aatc {
namespace {

constexpr int kD = 128;

// C = (1/N) sum_n x_n x_n^T over fp32 rows of width d, accumulated in fp64 (Sec. 5 Step 1:
// Sigma = X^T X / T).
void second_moment(const float* x, int n, std::vector<double>& c, int d = kD) {
  c.assign(static_cast<size_t>(d) * d, 0.0);
  std::vector<double> row(d);
  for (int t = 0; t < n; ++t) {
    const float* xt = x + static_cast<size_t>(t) * d;
    for (int i = 0; i < d; ++i) row[i] = xt[i];
    for (int i = 0; i < d; ++i) {
      const double xi = row[i];
      double* ci = c.data() + static_cast<size_t>(i) * d;
      for (int j = i; j < d; ++j) ci[j] += xi * row[j];
    }
  }
  const double inv = 1.0 / n;
  for (int i = 0; i < d; ++i)
    for (int j = i; j < d; ++j) {
      c[static_cast<size_t>(i) * d + j] *= inv;
      c[static_cast<size_t>(j) * d + i] = c[static_cast<size_t>(i) * d + j];
    }
}

// Cyclic Jacobi: rotate away each off-diagonal element in turn until the off-diagonal mass is
// negligible.  a is overwritten (its diagonal converges to the eigenvalues); v accumulates the
// rotations, so columns of v are the eigenvectors.
void jacobi_eigen(std::vector<double>& a, std::vector<double>& v, int n = kD) {
  const size_t kD = static_cast<size_t>(n);   // the matrix width (128, or 128 G_h for a head group)
  v.assign(kD * kD, 0.0);
  for (size_t i = 0; i < kD; ++i) v[i * kD + i] = 1.0;
  double frob = 0.0;
  for (double e : a) frob += e * e;
  const double tiny = 1e-300;
  for (int sweep = 0; sweep < 100; ++sweep) {
    double off = 0.0;
    for (size_t p = 0; p < kD; ++p)
      for (size_t q = p + 1; q < kD; ++q) off += a[p * kD + q] * a[p * kD + q];
    if (off <= 1e-30 * frob || off < tiny) break;
    for (size_t p = 0; p + 1 < kD; ++p) {
      for (size_t q = p + 1; q < kD; ++q) {
        const double apq = a[p * kD + q];
        if (std::fabs(apq) < tiny) continue;
        const double app = a[p * kD + p], aqq = a[q * kD + q];
        // Choose the rotation angle that zeroes a_pq: tan(2 phi) = 2 a_pq / (a_qq - a_pp),
        // taking the smaller root t = tan(phi) for stability.
        const double theta = (aqq - app) / (2.0 * apq);
        const double t = (theta >= 0 ? 1.0 : -1.0) / (std::fabs(theta) + std::sqrt(theta * theta + 1.0));
        const double c = 1.0 / std::sqrt(t * t + 1.0);
        const double s = t * c;
        for (size_t k = 0; k < kD; ++k) {       // A <- A J (columns p, q)
          const double akp = a[k * kD + p], akq = a[k * kD + q];
          a[k * kD + p] = c * akp - s * akq;
          a[k * kD + q] = s * akp + c * akq;
        }
        for (size_t k = 0; k < kD; ++k) {       // A <- J^T A (rows p, q)
          const double apk = a[p * kD + k], aqk = a[q * kD + k];
          a[p * kD + k] = c * apk - s * aqk;
          a[q * kD + k] = s * apk + c * aqk;
        }
        a[p * kD + q] = a[q * kD + p] = 0.0;
        for (size_t k = 0; k < kD; ++k) {       // V <- V J
          const double vkp = v[k * kD + p], vkq = v[k * kD + q];
          v[k * kD + p] = c * vkp - s * vkq;
          v[k * kD + q] = s * vkp + c * vkq;
        }
      }
    }
  }
}

double percentile99(std::vector<double>& vals) {
  std::sort(vals.begin(), vals.end());
  const double pos = 0.99 * static_cast<double>(vals.size() - 1);
  const size_t lo = static_cast<size_t>(std::floor(pos));
  const size_t hi = std::min(lo + 1, vals.size() - 1);
  return vals[lo] + (pos - static_cast<double>(lo)) * (vals[hi] - vals[lo]);
}

struct StreamJob {
  const float* x;              // calibration vectors [n][128]
  int n;
  const float* const* q_heads; // query heads of the group (keys only) or nullptr
  int n_q_heads_in_group;
  int n_q;
  int budget;
  int b_max;
  bool var_only;
  float* basis_out;            // [128][128]
  uint8_t* bits_out;           // [128]
  float* scales_out;           // [128]
  double* sigma2_out;          // [128] or null
  double* weights_out;         // [128] or null
};

void plan_one_stream(const StreamJob& job) {
  std::vector<double> c, v;
  second_moment(job.x, job.n, c);
  jacobi_eigen(c, v);
  // eigenvalues descending (stable on the Jacobi index order), canonical signs
  std::vector<int> ord(kD);
  std::iota(ord.begin(), ord.end(), 0);
  std::stable_sort(ord.begin(), ord.end(), [&](int i, int j) { return c[i * kD + i] > c[j * kD + j]; });
  std::vector<double> lam(kD), u(kD * kD);   // u[d][k]
  for (int k = 0; k < kD; ++k) {
    const int src = ord[k];
    lam[k] = c[src * kD + src];
    int imax = 0;
    double amax = -1.0;
    for (int d = 0; d < kD; ++d) {
      const double a = std::fabs(v[d * kD + src]);
      if (a > amax) { amax = a; imax = d; }
    }
    const double sgn = v[imax * kD + src] < 0 ? -1.0 : 1.0;
    for (int d = 0; d < kD; ++d) u[d * kD + k] = sgn * v[d * kD + src];
  }
  // weights: w^K_c = sum_heads u_c^T M_j u_c with M_j = mean_i q_i q_i^T; w^V_c = 1
  std::vector<double> w(kD, 1.0);
  if (!job.var_only && job.q_heads != nullptr) {
    std::vector<double> m(kD * kD, 0.0), mj;
    for (int j = 0; j < job.n_q_heads_in_group; ++j) {
      second_moment(job.q_heads[j], job.n_q, mj);
      for (int i = 0; i < kD * kD; ++i) m[i] += mj[i];
    }
    for (int k = 0; k < kD; ++k) {
      double acc = 0.0;
      for (int i = 0; i < kD; ++i) {
        double row = 0.0;
        for (int j2 = 0; j2 < kD; ++j2) row += m[i * kD + j2] * u[j2 * kD + k];
        acc += u[i * kD + k] * row;
      }
      w[k] = acc;
    }
  }
  // storage order: g = w * sigma^2 descending, stable
  std::vector<double> g(kD);
  for (int k = 0; k < kD; ++k) g[k] = w[k] * lam[k];
  std::vector<int> so(kD);
  std::iota(so.begin(), so.end(), 0);
  std::stable_sort(so.begin(), so.end(), [&](int i, int j) { return g[i] > g[j]; });
  std::vector<double> gs(kD);
  for (int c2 = 0; c2 < kD; ++c2) gs[c2] = g[so[c2]];
  // exact integer reverse water-filling by marginal gains (gain of one more bit on channel c at
  // b_c bits is (3/4) g_c 4^-b_c; the 3/4 is common), ties to the lower storage index
  std::vector<int> bits(kD, 0);
  for (int it = 0; it < job.budget; ++it) {
    int best = -1;
    double bg = -1.0;
    for (int c2 = 0; c2 < kD; ++c2) {
      if (bits[c2] >= job.b_max) continue;
      const double gain = std::ldexp(gs[c2], -2 * bits[c2]);
      if (best < 0 || gain > bg) { best = c2; bg = gain; }
    }
    if (best < 0) break;
    ++bits[best];
  }
  // scales: 99th percentile of |u_c . x| over the calibration vectors
  std::vector<double> h(static_cast<size_t>(job.n) * kD, 0.0);
  for (int t = 0; t < job.n; ++t) {
    const float* xt = job.x + static_cast<size_t>(t) * kD;
    double* ht = h.data() + static_cast<size_t>(t) * kD;
    for (int d = 0; d < kD; ++d) {
      const double xd = xt[d];
      const double* ud = u.data() + d * kD;
      for (int k = 0; k < kD; ++k) ht[k] += xd * ud[k];
    }
  }
  std::vector<double> col(job.n);
  for (int c2 = 0; c2 < kD; ++c2) {
    const int k = so[c2];
    for (int t = 0; t < job.n; ++t) col[t] = std::fabs(h[static_cast<size_t>(t) * kD + k]);
    job.scales_out[c2] = static_cast<float>(percentile99(col));
    job.bits_out[c2] = static_cast<uint8_t>(bits[c2]);
    for (int d = 0; d < kD; ++d) job.basis_out[d * kD + c2] = static_cast<float>(u[d * kD + k]);
    if (job.sigma2_out) job.sigma2_out[c2] = lam[k];
    if (job.weights_out) job.weights_out[c2] = w[k];
  }
}

// Linear-interpolation percentile (rank p (N-1), the NumPy default) of a copy of `vals`.
double percentile_linear(std::vector<double> vals, double p) {
  std::sort(vals.begin(), vals.end());
  const double r = p * (static_cast<double>(vals.size()) - 1.0);
  const size_t lo = static_cast<size_t>(std::floor(r));
  const size_t hi = std::min(lo + 1, vals.size() - 1);
  return vals[lo] + (r - static_cast<double>(lo)) * (vals[hi] - vals[lo]);
}

// Exact integer reverse water-filling over a pool of channels: the budget goes, one bit at a
// time, to the largest marginal gain g_c 4^-b_c (b_c < b_max); ties to the lower pool index.
void greedy_pool(const std::vector<double>& g, int budget, int b_max, std::vector<int>& bits) {
  bits.assign(g.size(), 0);
  using Item = std::pair<double, long>;                       // (gain, -index): max-heap order
  std::priority_queue<Item> heap;
  for (size_t i = 0; i < g.size(); ++i)
    if (b_max > 0) heap.emplace(g[i], -static_cast<long>(i));
  for (int it = 0; it < budget && !heap.empty(); ++it) {
    const Item top = heap.top();
    heap.pop();
    const size_t i = static_cast<size_t>(-top.second);
    if (++bits[i] < b_max) heap.emplace(std::ldexp(g[i], -2 * bits[i]), top.second);
  }
}

bool budget_from_avg(double avg, int b_max, int* budget) {
  const double b = avg * kD;
  const double r = std::nearbyint(b);
  if (!std::isfinite(b) || std::fabs(b - r) > 1e-9 || r < 0 || r > static_cast<double>(b_max) * kD) return false;
  *budget = static_cast<int>(r);
  return true;
}

}  // namespace
}  // namespace aatc

extern "C" aatc_status_t aatc_calibrate(const aatc_dims_t* dims, const float* calib_k,
                                        const float* calib_v, int32_t n_calib, const float* calib_q,
                                        int32_t n_calib_q, double avg_bits_k, double avg_bits_v,
                                        int32_t weights_mode, float* basis_out, uint8_t* bits_out,
                                        float* scales_out, double* sigma2_out, double* weights_out,
                                        int32_t n_threads) {
  using namespace aatc;
  if (!valid_dims(dims) || !calib_k || !calib_v || !basis_out || !bits_out || !scales_out)
    return AATC_ERR_INVALID_ARG;
  if (n_calib < 2 || (calib_q && n_calib_q < 1) || (weights_mode != 0 && weights_mode != 1))
    return AATC_ERR_INVALID_ARG;
  int bk = 0, bv = 0;
  if (!budget_from_avg(avg_bits_k, dims->b_max, &bk) || !budget_from_avg(avg_bits_v, dims->b_max, &bv))
    return AATC_ERR_BUDGET;
  const int L = dims->n_layers, H = dims->n_kv_heads, HQ = dims->n_q_heads, G = HQ / H;
  const size_t cal = static_cast<size_t>(n_calib) * kD;
  const size_t qsz = static_cast<size_t>(n_calib_q) * kD;
  std::vector<const float*> qptr(static_cast<size_t>(L) * HQ, nullptr);
  if (calib_q)
    for (int l = 0; l < L; ++l)
      for (int j = 0; j < HQ; ++j) qptr[static_cast<size_t>(l) * HQ + j] = calib_q + (static_cast<size_t>(l) * HQ + j) * qsz;
  std::vector<StreamJob> jobs;
  for (int l = 0; l < L; ++l)
    for (int h = 0; h < H; ++h)
      for (int kind = 0; kind < 2; ++kind) {
        const size_t s = (static_cast<size_t>(l) * H + h) * 2 + kind;
        const size_t lh = static_cast<size_t>(l) * H + h;
        StreamJob j;
        j.x = (kind == 0 ? calib_k : calib_v) + lh * cal;
        j.n = n_calib;
        j.q_heads = (kind == 0 && calib_q) ? qptr.data() + static_cast<size_t>(l) * HQ + static_cast<size_t>(h) * G : nullptr;
        j.n_q_heads_in_group = G;
        j.n_q = n_calib_q;
        j.budget = kind == 0 ? bk : bv;
        j.b_max = dims->b_max;
        j.var_only = weights_mode == 1;
        j.basis_out = basis_out + s * kD * kD;
        j.bits_out = bits_out + s * kD;
        j.scales_out = scales_out + s * kD;
        j.sigma2_out = sigma2_out ? sigma2_out + s * kD : nullptr;
        j.weights_out = weights_out ? weights_out + s * kD : nullptr;
        jobs.push_back(j);
      }
  int nt = n_threads > 0 ? n_threads : static_cast<int>(std::thread::hardware_concurrency());
  nt = std::max(1, std::min<int>(nt, static_cast<int>(jobs.size())));
  std::atomic<size_t> next{0};
  auto worker = [&]() {
    for (size_t i = next++; i < jobs.size(); i = next++) plan_one_stream(jobs[i]);
  };
  std::vector<std::thread> pool;
  for (int t = 1; t < nt; ++t) pool.emplace_back(worker);
  worker();
  for (auto& th : pool) th.join();
  return AATC_OK;
}

// Head-group stream (Sec. 5 Step 1, remark on multi-head attention): the g_h kv-heads of a group
// concatenated into vectors of width d = 128 g_h get one PCA basis, one weighted reverse
// water-filling over the d channels (budget avg_bits * d) and one P99 scale per channel.  Query
// head j of the group belongs to kv-head j / group; its score q . k_block sees only that block, so
// its key weight is u_c[block]^T M_j u_c[block] with M_j the second moment of its calibration
// queries (Eq. waterfilling-keys with the query embedded at its block).
extern "C" aatc_status_t aatc_calibrate_head_group(int32_t g_h, int32_t group, const float* calib, int32_t n_calib,
                                                   const float* calib_q, int32_t n_calib_q, double avg_bits,
                                                   int32_t b_max, int32_t weights_mode, float* basis_out,
                                                   uint8_t* bits_out, float* scales_out, double* sigma2_out,
                                                   double* weights_out) {
  using namespace aatc;
  if (g_h < 1 || g_h > 8 || group < 1 || !calib || n_calib < 2 || !basis_out || !bits_out || !scales_out ||
      (calib_q && n_calib_q < 1) || (weights_mode != 0 && weights_mode != 1) || b_max < 1 ||
      b_max > AATC_MAX_PLAN_BITS)
    return AATC_ERR_INVALID_ARG;
  const int d = kD * g_h;
  const double bd = avg_bits * d, br = std::nearbyint(bd);
  if (!std::isfinite(bd) || std::fabs(bd - br) > 1e-9 || br < 0 || br > static_cast<double>(b_max) * d)
    return AATC_ERR_BUDGET;
  const int budget = static_cast<int>(br);
  const size_t n = static_cast<size_t>(n_calib);
  std::vector<float> x(n * d);                             // concatenated group vectors [n][d]
  for (int m = 0; m < g_h; ++m)
    for (size_t t = 0; t < n; ++t)
      for (int i = 0; i < kD; ++i) x[t * d + m * kD + i] = calib[(m * n + t) * kD + i];
  std::vector<double> c, v;
  second_moment(x.data(), n_calib, c, d);
  jacobi_eigen(c, v, d);
  // eigenvalues descending (stable on the Jacobi index order), canonical signs
  std::vector<int> ord(d);
  std::iota(ord.begin(), ord.end(), 0);
  std::stable_sort(ord.begin(), ord.end(),
                   [&](int i, int j) { return c[static_cast<size_t>(i) * d + i] > c[static_cast<size_t>(j) * d + j]; });
  std::vector<double> lam(d), u(static_cast<size_t>(d) * d);   // u[dim][k]
  for (int k = 0; k < d; ++k) {
    const int src = ord[k];
    lam[k] = c[static_cast<size_t>(src) * d + src];
    int imax = 0;
    double amax = -1.0;
    for (int r = 0; r < d; ++r) {
      const double a = std::fabs(v[static_cast<size_t>(r) * d + src]);
      if (a > amax) { amax = a; imax = r; }
    }
    const double sgn = v[static_cast<size_t>(imax) * d + src] < 0 ? -1.0 : 1.0;
    for (int r = 0; r < d; ++r) u[static_cast<size_t>(r) * d + k] = sgn * v[static_cast<size_t>(r) * d + src];
  }
  std::vector<double> w(d, 1.0);
  if (weights_mode == 0 && calib_q) {
    std::fill(w.begin(), w.end(), 0.0);
    std::vector<double> mj;
    for (int j = 0; j < g_h * group; ++j) {
      second_moment(calib_q + static_cast<size_t>(j) * n_calib_q * kD, n_calib_q, mj);
      const int b0 = (j / group) * kD;                     // the query's kv-head block
      for (int k = 0; k < d; ++k) {
        double acc = 0.0;
        for (int i = 0; i < kD; ++i) {
          double row = 0.0;
          for (int i2 = 0; i2 < kD; ++i2) row += mj[i * kD + i2] * u[static_cast<size_t>(b0 + i2) * d + k];
          acc += u[static_cast<size_t>(b0 + i) * d + k] * row;
        }
        w[k] += acc;
      }
    }
  }
  std::vector<double> g(d);
  for (int k = 0; k < d; ++k) g[k] = w[k] * lam[k];
  std::vector<int> so(d);
  std::iota(so.begin(), so.end(), 0);
  std::stable_sort(so.begin(), so.end(), [&](int i, int j) { return g[i] > g[j]; });
  std::vector<double> gs(d);
  for (int c2 = 0; c2 < d; ++c2) gs[c2] = g[so[c2]];
  std::vector<int> bits;
  greedy_pool(gs, budget, b_max, bits);
  std::vector<double> col(n);
  for (int c2 = 0; c2 < d; ++c2) {
    const int k = so[c2];
    for (size_t t = 0; t < n; ++t) {
      double h = 0.0;
      for (int r = 0; r < d; ++r) h += static_cast<double>(x[t * d + r]) * u[static_cast<size_t>(r) * d + k];
      col[t] = std::fabs(h);
    }
    scales_out[c2] = static_cast<float>(percentile99(col));
    bits_out[c2] = static_cast<uint8_t>(bits[c2]);
    for (int r = 0; r < d; ++r) basis_out[static_cast<size_t>(r) * d + c2] = static_cast<float>(u[static_cast<size_t>(r) * d + k]);
    if (sigma2_out) sigma2_out[c2] = lam[k];
    if (weights_out) weights_out[c2] = w[k];
  }
  return AATC_OK;
}

extern "C" aatc_status_t aatc_allocate_global(const aatc_dims_t* dims, const double* sigma2,
                                              const double* weights, double avg_bits_k, double avg_bits_v,
                                              int32_t n_protect, uint8_t* bits_out) {
  using namespace aatc;
  if (!valid_dims(dims) || !sigma2 || !weights || !bits_out || n_protect < 0) return AATC_ERR_INVALID_ARG;
  const int L = dims->n_layers, H = dims->n_kv_heads, b_max = dims->b_max;
  const int np = std::min(n_protect, L);
  for (size_t i = 0; i < static_cast<size_t>(L) * H * 2 * kD; ++i)
    if (!std::isfinite(sigma2[i]) || !std::isfinite(weights[i]) || sigma2[i] < 0.0 || weights[i] < 0.0)
      return AATC_ERR_INVALID_ARG;
  for (int kind = 0; kind < 2; ++kind) {
    const double avg = kind == 0 ? avg_bits_k : avg_bits_v;
    int per_stream = 0;
    if (!budget_from_avg(avg, b_max, &per_stream)) return AATC_ERR_BUDGET;
    // protected layers: per-stream allocation, the average budget for values and one bit per
    // channel more for keys (capped at b_max)
    const int prot = std::min(per_stream + (kind == 0 ? kD : 0), b_max * kD);
    const long total = static_cast<long>(per_stream) * L * H;
    const long rest = total - static_cast<long>(prot) * np * H;
    const long pool_cap = static_cast<long>(b_max) * kD * (L - np) * H;
    if (rest < 0 || rest > pool_cap) return AATC_ERR_BUDGET;
    auto at = [&](int l, int h, int c) { return ((static_cast<size_t>(l) * H + h) * 2 + kind) * kD + c; };
    std::vector<int> bits;
    for (int l = 0; l < np; ++l)
      for (int h = 0; h < H; ++h) {
        std::vector<double> g(kD);
        for (int c = 0; c < kD; ++c) g[c] = weights[at(l, h, c)] * sigma2[at(l, h, c)];
        greedy_pool(g, prot, b_max, bits);
        for (int c = 0; c < kD; ++c) bits_out[at(l, h, c)] = static_cast<uint8_t>(bits[c]);
      }
    if (np == L) continue;
    // the pool: g = (sigma^2 / P95_l(sigma^2)) (w / P95_l(w)), percentiles over the layer's
    // channels of every kv-head
    std::vector<double> g;
    g.reserve(static_cast<size_t>(L - np) * H * kD);
    for (int l = np; l < L; ++l) {
      std::vector<double> sv, wv;
      for (int h = 0; h < H; ++h)
        for (int c = 0; c < kD; ++c) {
          sv.push_back(sigma2[at(l, h, c)]);
          wv.push_back(weights[at(l, h, c)]);
        }
      double ps = percentile_linear(sv, 0.95), pw = percentile_linear(wv, 0.95);
      if (!(ps > 0.0)) ps = 1.0;
      if (!(pw > 0.0)) pw = 1.0;
      for (int h = 0; h < H; ++h)
        for (int c = 0; c < kD; ++c) g.push_back((sigma2[at(l, h, c)] / ps) * (weights[at(l, h, c)] / pw));
    }
    greedy_pool(g, static_cast<int>(rest), b_max, bits);
    size_t i = 0;
    for (int l = np; l < L; ++l)
      for (int h = 0; h < H; ++h)
        for (int c = 0; c < kD; ++c) bits_out[at(l, h, c)] = static_cast<uint8_t>(bits[i++]);
  }
  return AATC_OK;
}

// ------------------------------------------------------------------ transform from model weights

namespace aatc {
namespace {

// Round an fp32 value to bf16 bits, round to nearest even (finite inputs).
uint16_t bf16_bits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  const uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return static_cast<uint16_t>(u >> 16);
}

}  // namespace
}  // namespace aatc

extern "C" aatc_status_t aatc_whitening_transform(int32_t d_model, int32_t n, const float* x, const float* w,
                                                  float* a_out, float* b_out, double* s_out, float* p_out,
                                                  float* ahat_out) {
  using namespace aatc;
  if (d_model < 1 || n < 1 || !x || !w) return AATC_ERR_INVALID_ARG;
  const size_t dm = static_cast<size_t>(d_model);
  for (size_t i = 0; i < dm * kD; ++i)
    if (!std::isfinite(w[i])) return AATC_ERR_INVALID_ARG;
  // C = K^T K / n with K = X W (= W^T Sigma_X W = W~^T W~ for W~ = L^T W, any L L^T = Sigma_X)
  std::vector<double> c(kD * kD, 0.0), k(kD), wd(dm * kD);
  for (size_t i = 0; i < dm * kD; ++i) wd[i] = w[i];
  for (int t = 0; t < n; ++t) {
    const float* xt = x + static_cast<size_t>(t) * dm;
    std::fill(k.begin(), k.end(), 0.0);
    for (size_t i = 0; i < dm; ++i) {
      const double xi = xt[i];
      if (!std::isfinite(xi)) return AATC_ERR_INVALID_ARG;
      if (xi == 0.0) continue;
      const double* wi = wd.data() + i * kD;
      for (int j = 0; j < kD; ++j) k[j] += xi * wi[j];
    }
    for (int i = 0; i < kD; ++i) {
      double* ci = c.data() + i * kD;
      const double ki = k[i];
      for (int j = i; j < kD; ++j) ci[j] += ki * k[j];
    }
  }
  for (int i = 0; i < kD; ++i)
    for (int j = i; j < kD; ++j) {
      c[i * kD + j] /= n;
      c[j * kD + i] = c[i * kD + j];
    }
  // C = P diag(S^2) P^T: eigenvalues descending (stable), sign-canonical columns
  std::vector<double> v;
  jacobi_eigen(c, v);
  std::vector<int> ord(kD);
  std::iota(ord.begin(), ord.end(), 0);
  std::stable_sort(ord.begin(), ord.end(), [&](int i, int j) { return c[i * kD + i] > c[j * kD + j]; });
  std::vector<double> s(kD), p(kD * kD);                      // p[d][k]
  for (int kk = 0; kk < kD; ++kk) {
    const int src = ord[kk];
    const double lam = c[src * kD + src];
    if (!(lam > 0.0)) return AATC_ERR_INVALID_ARG;             // W~ must have full column rank
    s[kk] = std::sqrt(lam);
    int imax = 0;
    double amax = -1.0;
    for (int d = 0; d < kD; ++d) {
      const double a = std::fabs(v[d * kD + src]);
      if (a > amax) { amax = a; imax = d; }
    }
    const double sgn = v[imax * kD + src] < 0 ? -1.0 : 1.0;
    for (int d = 0; d < kD; ++d) p[d * kD + kk] = sgn * v[d * kD + src];
  }
  // A_hat = W P;  A = A_hat S^-1/2;  B = S^1/2 P^T
  for (size_t i = 0; i < dm; ++i) {
    const double* wi = wd.data() + i * kD;
    for (int kk = 0; kk < kD; ++kk) {
      double acc = 0.0;
      for (int d = 0; d < kD; ++d) acc += wi[d] * p[d * kD + kk];
      if (ahat_out) ahat_out[i * kD + kk] = static_cast<float>(acc);
      if (a_out) a_out[i * kD + kk] = static_cast<float>(acc / std::sqrt(s[kk]));
    }
  }
  for (int kk = 0; kk < kD; ++kk) {
    if (s_out) s_out[kk] = s[kk];
    for (int d = 0; d < kD; ++d) {
      if (b_out) b_out[kk * kD + d] = static_cast<float>(std::sqrt(s[kk]) * p[d * kD + kk]);
      if (p_out) p_out[d * kD + kk] = static_cast<float>(p[d * kD + kk]);
    }
  }
  return AATC_OK;
}

extern "C" aatc_status_t aatc_hidden_operand(const aatc_dims_t* dims, int32_t d_model, const float* w_k,
                                             const float* w_v, const float* basis, uint16_t* out) {
  using namespace aatc;
  if (!valid_dims(dims) || d_model < 64 || d_model % 64 != 0 || !w_k || !w_v || !basis || !out)
    return AATC_ERR_INVALID_ARG;
  const int L = dims->n_layers, H = dims->n_kv_heads;
  const size_t dm = static_cast<size_t>(d_model), ld = static_cast<size_t>(H) * kD;
  for (int l = 0; l < L; ++l)
    for (int h = 0; h < H; ++h)
      for (int kind = 0; kind < 2; ++kind) {
        const float* wl = (kind == 0 ? w_k : w_v) + static_cast<size_t>(l) * dm * ld + static_cast<size_t>(h) * kD;
        const float* u = basis + ((static_cast<size_t>(l) * H + h) * 2 + kind) * kD * kD;   // [dim][channel]
        uint16_t* o = out + ((static_cast<size_t>(l) * H + h) * 2 + kind) * kD * dm;        // [channel][d_model]
        for (size_t i = 0; i < dm; ++i) {
          const float* wi = wl + i * ld;
          for (int c2 = 0; c2 < kD; ++c2) {
            double acc = 0.0;
            for (int d = 0; d < kD; ++d) acc += static_cast<double>(wi[d]) * u[d * kD + c2];
            if (!std::isfinite(acc)) return AATC_ERR_INVALID_ARG;
            o[static_cast<size_t>(c2) * dm + i] = bf16_bits(static_cast<float>(acc));
          }
        }
      }
  return AATC_OK;
}
