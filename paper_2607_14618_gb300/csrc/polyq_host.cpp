// Host side of the PolyQ library: error proxies (Section 3.1), width
// allocation (Section 3.2), quanta matching (Section 3.3), bit-specific
// activation-aware scaling (Section 3.4), clustering permutation and bit
// blocks (Sections 4.1, 4.2), group quantisation and packing, and the
// permutation merge rule (Section 4.3).
//
// Build with -ffp-contract=off: every floating-point step below is a single
// IEEE double operation in the order written, so the result is the same on
// any host.
#include <algorithm>
#include <atomic>
#include <cfenv>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <functional>
#include <new>
#include <queue>
#include <string>
#include <thread>
#include <vector>

#include "polyq.h"
#include "polyq_internal.h"

struct polyq_layer {
  int64_t N = 0, K = 0, S = 0, G = 0;
  double budget = 0.0;
  std::vector<uint8_t> bits;      // [K] original order
  std::vector<int32_t> perm;      // [K] clustered -> original
  std::vector<polyq_block> blocks;
  std::vector<uint8_t> packed;    // [N][S]
  std::vector<uint32_t> meta;     // [N][G] scale | zero << 16
  std::vector<int32_t> out_perm;  // [N]
  std::vector<float> xscale;      // [K] clustered order; empty = not scaled
  double alpha[5] = {-1, -1, -1, -1, -1};
};

namespace {

thread_local std::string g_err;

const int kPalette[5] = {2, 3, 4, 8, 16};

int width_index(int b) {
  for (int i = 0; i < 5; ++i)
    if (kPalette[i] == b) return i;
  return -1;
}

// Error proxy of Section 3.1 instantiated from saliency: (sal/(2^b-1))^2,
// with E_16 = 0.
double proxy_error(double sal, int b) {
  if (b == 16) return 0.0;
  double e = sal / (double)((1 << b) - 1);
  return e * e;
}


struct Cand {
  double g;
  int32_t k;
  int32_t bn;
};
struct CandLess {  // max-heap on gain, then lower channel index first
  bool operator()(const Cand& a, const Cand& b) const {
    if (a.g != b.g) return a.g < b.g;
    return a.k > b.k;
  }
};

int run_threads(int64_t n, int want, const std::function<void(int64_t, int64_t)>& fn);

}  // namespace

extern "C" const char* polyq_last_error(void) { return g_err.c_str(); }

int polyq_set_error(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

void polyq_clear_error() { g_err.clear(); }

extern "C" uint16_t polyq_f64_to_f16(double x) {
  // Round-to-nearest-even into fp16 directly from double: scale by a power
  // of two so that one fp16 quantum is 1, round with nearbyint (the default
  // rounding mode is to-nearest-even), then encode.
  uint16_t sign = std::signbit(x) ? 0x8000 : 0;
  double ax = std::fabs(x);
  if (std::isnan(x)) return 0x7E00;
  if (ax == 0.0) return sign;
  if (ax >= 65520.0) return sign | 0x7C00;
  int e;
  std::frexp(ax, &e);       // ax in [2^(e-1), 2^e)
  int E = e - 1;
  if (E < -14) E = -14;     // subnormal quantum 2^-24
  double r = std::nearbyint(std::ldexp(ax, 10 - E));  // value / 2^(E-10)
  double v = std::ldexp(r, E - 10);
  if (v == 0.0) return sign;
  if (v < 6.103515625e-05) return sign | (uint16_t)std::ldexp(v, 24);
  int e2;
  std::frexp(v, &e2);
  int E2 = e2 - 1;
  if (E2 > 15) return sign | 0x7C00;
  uint32_t frac = (uint32_t)std::ldexp(v, 10 - E2) - 1024u;
  return (uint16_t)(sign | ((uint32_t)(E2 + 15) << 10) | frac);
}

static double f16_to_f64(uint16_t h) {
  int s = h >> 15, e = (h >> 10) & 31, f = h & 1023;
  double v;
  if (e == 0) v = std::ldexp((double)f, -24);
  else if (e == 31) v = f ? NAN : INFINITY;
  else v = std::ldexp((double)(1024 + f), e - 25);
  return s ? -v : v;
}

namespace {

int run_threads(int64_t n, int want, const std::function<void(int64_t, int64_t)>& fn) {
  int nt = want > 0 ? want : (int)std::max(1u, std::thread::hardware_concurrency());
  if (nt > 64) nt = 64;
  if (n < 2 * nt) nt = 1;
  if (nt == 1) {
    fn(0, n);
    return 0;
  }
  std::vector<std::thread> th;
  for (int t = 0; t < nt; ++t) {
    int64_t a = n * t / nt, b = n * (t + 1) / nt;
    th.emplace_back(fn, a, b);
  }
  for (auto& x : th) x.join();
  return 0;
}

// sal_k = a_k * sqrt(sum_n W[n,k]^2); for each k the sum runs over n in
// order, in fp64 (products of fp32 values are exact in fp64).
void saliency(const float* W, int64_t N, int64_t K, const float* a, std::vector<double>& sal,
              int nthreads) {
  sal.assign(K, 0.0);
  run_threads(K, nthreads, [&](int64_t k0, int64_t k1) {
    std::vector<double> acc(k1 - k0, 0.0);
    for (int64_t n = 0; n < N; ++n) {
      const float* row = W + n * K;
      for (int64_t k = k0; k < k1; ++k) {
        double w = (double)row[k];
        double sq = w * w;
        acc[k - k0] = acc[k - k0] + sq;
      }
    }
    for (int64_t k = k0; k < k1; ++k) sal[k] = (double)a[k] * std::sqrt(acc[k - k0]);
  });
}

// Per-width error table E[width index][k] (Section 3.1).
struct ErrTable {
  std::vector<double> e[5];
  double at(int b, int64_t k) const { return e[width_index(b)][k]; }
  // gain per extra bit of the step b -> bn (Section 3.2)
  double gain(int64_t k, int b, int bn) const {
    return (at(b, k) - at(bn, k)) / (double)(bn - b);
  }
};

void saliency_table(const std::vector<double>& sal, const std::vector<int>& pal, ErrTable& E) {
  for (int b : pal) {
    std::vector<double>& v = E.e[width_index(b)];
    v.resize(sal.size());
    for (size_t k = 0; k < sal.size(); ++k) v[k] = proxy_error(sal[k], b);
  }
}

// Section 3.2 greedy allocation under budget B.
void allocate(const std::vector<double>& sal, const ErrTable& E, double B,
              const std::vector<int>& pal, int rule, std::vector<uint8_t>& bits) {
  const int64_t K = (int64_t)sal.size();
  const int bmin = pal[0];
  bits.assign(K, (uint8_t)bmin);
  int64_t delta = (int64_t)std::floor(B * (double)K + 0.5) - (int64_t)bmin * K;
  if (delta <= 0 || pal.size() == 1) return;
  auto next_w = [&](int b) -> int {
    for (size_t i = 0; i + 1 < pal.size(); ++i)
      if (pal[i] == b) return pal[i + 1];
    return 0;
  };
  if (rule == POLYQ_ALLOC_LADDER) {
    std::vector<int32_t> order(K);
    for (int64_t k = 0; k < K; ++k) order[k] = (int32_t)k;
    std::stable_sort(order.begin(), order.end(),
                     [&](int32_t x, int32_t y) { return sal[x] > sal[y]; });
    for (int32_t k : order) {
      if (delta == 0) break;
      int b = bits[k];
      for (int bn = next_w(b); bn && bn - b <= delta; bn = next_w(b)) {
        delta -= bn - b;
        b = bn;
      }
      bits[k] = (uint8_t)b;
    }
    return;
  }
  std::vector<Cand> init;
  init.reserve(K);
  const int b1 = next_w(bmin);
  for (int64_t k = 0; k < K; ++k) init.push_back({E.gain(k, bmin, b1), (int32_t)k, b1});
  std::priority_queue<Cand, std::vector<Cand>, CandLess> heap(CandLess(), std::move(init));
  while (delta > 0 && !heap.empty()) {
    Cand c = heap.top();
    heap.pop();
    int cost = c.bn - bits[c.k];
    if (cost > delta) continue;  // Delta only shrinks: this step never fits
    bits[c.k] = (uint8_t)c.bn;
    delta -= cost;
    int bn2 = next_w(c.bn);
    if (bn2) heap.push({E.gain(c.k, c.bn, bn2), c.k, bn2});
  }
}

int64_t seg_bytes_for(int b, int64_t kb) {
  int64_t raw = b == 16 ? kb * 2 : (kb * b + 7) / 8;
  return (raw + 15) / 16 * 16;
}

// The group quantiser: scale and zero (fp16 values) and codes of the cn
// weights w[0..cn) at width b < 16.
void quant_group(const double* w, int cn, int b, double* s_out, double* z_out, uint32_t* q) {
  const double qmax = (double)((1 << b) - 1);
  double lo = INFINITY, hi = -INFINITY;
  for (int i = 0; i < cn; ++i) {
    lo = std::min(lo, w[i]);
    hi = std::max(hi, w[i]);
  }
  double s = f16_to_f64(polyq_f64_to_f16((hi - lo) / qmax));
  if (s == 0.0) {
    double alt = std::max(std::max(std::fabs(lo), std::fabs(hi)), 6.103515625e-05);
    s = f16_to_f64(polyq_f64_to_f16(alt));
  }
  double z = std::nearbyint((-lo) / s);
  z = std::min(std::max(z, 0.0), qmax);
  for (int i = 0; i < cn; ++i) {
    double v = std::nearbyint(w[i] / s) + z;
    v = std::min(std::max(v, 0.0), qmax);
    q[i] = (uint32_t)v;
  }
  *s_out = s;
  *z_out = z;
}

// Quantise and pack rows [r0, r1) of the layer.  With activation factors t
// (original channel order) the packed weight is W / t.
void pack_rows(const float* W, int64_t K, const double* t, polyq_layer& L, int64_t r0,
               int64_t r1) {
  std::vector<double> w(POLYQ_GROUP);
  std::vector<uint32_t> q(POLYQ_GROUP);
  for (int64_t n = r0; n < r1; ++n) {
    const float* row = W + n * K;
    uint8_t* prow = L.packed.data() + n * L.S;
    uint32_t* mrow = L.meta.data() + n * L.G;
    auto wv = [&](int32_t k) { return t ? (double)row[k] / t[k] : (double)row[k]; };
    for (const polyq_block& blk : L.blocks) {
      uint8_t* seg = prow + blk.seg_off;
      const int32_t* pp = L.perm.data() + blk.pos0;
      const int b = blk.bits;
      if (b == 16) {
        for (int32_t i = 0; i < blk.n_ch; ++i) {
          uint16_t h = polyq_f64_to_f16(wv(pp[i]));
          seg[2 * i] = (uint8_t)(h & 0xFF);
          seg[2 * i + 1] = (uint8_t)(h >> 8);
        }
        continue;
      }
      uint64_t acc = 0;  // LSB-first bit writer
      int nacc = 0;
      int64_t wb = 0;
      for (int32_t g = 0; g < blk.n_grp; ++g) {
        int32_t c0 = g * POLYQ_GROUP;
        int32_t cn = std::min<int32_t>(POLYQ_GROUP, blk.n_ch - c0);
        for (int32_t i = 0; i < cn; ++i) w[i] = wv(pp[c0 + i]);
        double s, z;
        quant_group(w.data(), cn, b, &s, &z, q.data());
        mrow[blk.grp_off + g] =
            (uint32_t)polyq_f64_to_f16(s) | ((uint32_t)polyq_f64_to_f16(z) << 16);
        for (int32_t i = 0; i < cn; ++i) {
          acc |= (uint64_t)q[i] << nacc;
          nacc += b;
          while (nacc >= 8) {
            seg[wb++] = (uint8_t)(acc & 0xFF);
            acc >>= 8;
            nacc -= 8;
          }
        }
      }
      if (nacc > 0) seg[wb++] = (uint8_t)(acc & 0xFF);
      // remaining padding bytes are already zero (buffer zero-initialised)
    }
  }
}

// Quantiser-in-the-loop proxy (Section 3.1): for each palette width b < 16
// the whole layer is quantised at b with groups of 64 consecutive original
// channels, and E_b[k] = sum_n (w'[n][k] - W[n][k])^2 * x2[k], rows added in
// order; E_16 = 0.  Threads split the groups.
void quant_table(const float* W, int64_t N, int64_t K, const std::vector<double>& x2,
                 const std::vector<int>& pal, int nthreads, ErrTable& E) {
  const int64_t ng = (K + POLYQ_GROUP - 1) / POLYQ_GROUP;
  for (int b : pal) {
    std::vector<double>& e = E.e[width_index(b)];
    e.assign(K, 0.0);
    if (b == 16) continue;
    run_threads(ng, nthreads, [&](int64_t g0, int64_t g1) {
      double w[POLYQ_GROUP];
      uint32_t q[POLYQ_GROUP];
      for (int64_t n = 0; n < N; ++n) {
        const float* row = W + n * K;
        for (int64_t g = g0; g < g1; ++g) {
          const int64_t c0 = g * POLYQ_GROUP;
          const int cn = (int)std::min<int64_t>(POLYQ_GROUP, K - c0);
          for (int i = 0; i < cn; ++i) w[i] = (double)row[c0 + i];
          double sc, z;
          quant_group(w, cn, b, &sc, &z, q);
          for (int i = 0; i < cn; ++i) {
            double d = ((double)q[i] - z) * sc - w[i];
            e[c0 + i] = e[c0 + i] + d * d;
          }
        }
      }
    });
    for (int64_t k = 0; k < K; ++k) e[k] = e[k] * x2[k];
  }
}

// Section 3.3, step 1: target block sizes, multiples of the quanta near the
// allocation's counts, summing to K, with the realised budget closest to
// round(B*K) (the rule is spelled out at polyq_pack_opts).
std::vector<int64_t> quanta_targets(const std::vector<int>& pal, const std::vector<int64_t>& cnt,
                                    const int32_t* quanta, double B, int64_t K) {
  const int m = (int)pal.size();
  const int64_t T = (int64_t)std::floor(B * (double)K + 0.5);
  std::vector<std::vector<int64_t>> cand(m);
  for (int i = 0; i < m; ++i) {
    const int64_t q = quanta[width_index(pal[i])];
    const int64_t base = cnt[i] / q;
    for (int d = -1; d <= 2; ++d) {
      const int64_t v = q * (base + d);
      if (v >= 0 && v <= K && (cand[i].empty() || cand[i].back() != v)) cand[i].push_back(v);
    }
  }
  // key: (|bits - T|, sum |c^ - c|, counts lexicographic)
  bool have = false;
  int64_t best_mis = 0, best_mv = 0;
  std::vector<int64_t> best(m), cur(m);
  auto consider = [&]() {
    int64_t tb = 0, mv = 0;
    for (int i = 0; i < m; ++i) {
      tb += (int64_t)pal[i] * cur[i];
      mv += std::llabs(cur[i] - cnt[i]);
    }
    const int64_t mis = std::llabs(tb - T);
    if (!have || mis < best_mis || (mis == best_mis && (mv < best_mv || (mv == best_mv && cur < best)))) {
      have = true;
      best_mis = mis;
      best_mv = mv;
      best = cur;
    }
  };
  // exact: every width a multiple of its quantum
  std::vector<size_t> ix(m, 0);
  for (;;) {
    int64_t sum = 0;
    for (int i = 0; i < m; ++i) sum += (cur[i] = cand[i][ix[i]]);
    if (sum == K) consider();
    int i = m - 1;
    while (i >= 0 && ++ix[i] == cand[i].size()) ix[i--] = 0;
    if (i < 0) break;
  }
  if (!have && m > 1) {
    // the narrowest width takes the remainder
    std::fill(ix.begin(), ix.end(), 0);
    for (;;) {
      int64_t rest = 0;
      for (int i = 1; i < m; ++i) rest += (cur[i] = cand[i][ix[i]]);
      cur[0] = K - rest;
      if (cur[0] >= 0) consider();
      int i = m - 1;
      while (i >= 1 && ++ix[i] == cand[i].size()) ix[i--] = 0;
      if (i < 1) break;
    }
  }
  if (!have) best.assign(1, K);  // a one-width palette keeps every channel
  return best;
}

// Section 3.3, step 2: move channels between neighbouring widths until the
// per-width counts are the targets; promotions by largest gain per bit
// (lower channel first), demotions by smallest gain (higher channel first).
void reassign(const std::vector<int>& pal, const std::vector<int64_t>& target, const ErrTable& E,
              std::vector<uint8_t>& bits) {
  const int m = (int)pal.size();
  const int64_t K = (int64_t)bits.size();
  std::vector<int64_t> flow(m > 1 ? m - 1 : 0);
  int64_t acc = 0;
  for (int i = 0; i + 1 < m; ++i) {
    int64_t c = 0;
    for (int64_t k = 0; k < K; ++k) c += bits[k] == pal[i];
    acc += c - target[i];
    flow[i] = acc;
  }
  std::vector<int32_t> mem;
  for (int i = 0; i + 1 < m; ++i) {
    if (flow[i] <= 0) continue;
    const int b = pal[i], bn = pal[i + 1];
    mem.clear();
    for (int64_t k = 0; k < K; ++k)
      if (bits[k] == b) mem.push_back((int32_t)k);
    std::stable_sort(mem.begin(), mem.end(), [&](int32_t x, int32_t y) {
      const double gx = E.gain(x, b, bn), gy = E.gain(y, b, bn);
      if (gx != gy) return gx > gy;
      return x < y;
    });
    for (int64_t j = 0; j < flow[i]; ++j) bits[mem[j]] = (uint8_t)bn;
  }
  for (int i = m - 2; i >= 0; --i) {
    if (flow[i] >= 0) continue;
    const int b = pal[i], bn = pal[i + 1];
    mem.clear();
    for (int64_t k = 0; k < K; ++k)
      if (bits[k] == bn) mem.push_back((int32_t)k);
    std::stable_sort(mem.begin(), mem.end(), [&](int32_t x, int32_t y) {
      const double gx = E.gain(x, b, bn), gy = E.gain(y, b, bn);
      if (gx != gy) return gx < gy;
      return x > y;
    });
    for (int64_t j = 0; j < -flow[i]; ++j) bits[mem[j]] = (uint8_t)b;
  }
}

// Section 3.4: for each width present the exponent alpha (grid j/10) whose
// activation factors t_k = fp32_rn(m_k^-alpha) give the smallest mean of
// ||Q_b(W/t)[:,k]*t_k - W[:,k]||^2 * x2[k] over the block, with the block's
// own groups.  Fills t (original order) and alpha per width index.
void choose_alphas(const float* W, int64_t N, int64_t K, const std::vector<uint8_t>& bits,
                   const float* a, const std::vector<double>& x2, int nthreads,
                   std::vector<double>& t, double* alpha) {
  std::vector<double> m(K);
  double tot = 0.0;
  for (int64_t k = 0; k < K; ++k) tot = tot + (double)a[k];
  const double mean = tot / (double)K;
  for (int64_t k = 0; k < K; ++k) m[k] = (double)a[k] / mean;
  t.assign(K, 1.0);
  for (int wi = 0; wi < 5; ++wi) alpha[wi] = -1.0;
  for (int b : kPalette) {
    std::vector<int32_t> idx;
    for (int64_t k = 0; k < K; ++k)
      if (bits[k] == b) idx.push_back((int32_t)k);
    if (idx.empty()) continue;
    if (b == 16) {  // E_16 = 0 for every alpha
      alpha[width_index(b)] = 0.0;
      continue;
    }
    const int64_t kb = (int64_t)idx.size();
    const int64_t ng = (kb + POLYQ_GROUP - 1) / POLYQ_GROUP;
    bool have = false;
    double best_e = 0.0, best_a = 0.0;
    std::vector<double> best_t, tb(kb), err(kb);
    for (int j = 0; j <= 10; ++j) {
      const double al = j / 10.0;
      bool ok = true;
      for (int64_t i = 0; i < kb; ++i) {
        tb[i] = (double)(float)std::pow(m[idx[i]], -al);
        if (!(std::isfinite(tb[i]) && tb[i] > 0.0)) ok = false;
      }
      if (!ok) continue;
      std::atomic<bool> range_ok(true);
      std::fill(err.begin(), err.end(), 0.0);
      run_threads(ng, nthreads, [&](int64_t g0, int64_t g1) {
        double w[POLYQ_GROUP];
        uint32_t q[POLYQ_GROUP];
        for (int64_t n = 0; n < N; ++n) {
          const float* row = W + n * K;
          for (int64_t g = g0; g < g1; ++g) {
            const int64_t c0 = g * POLYQ_GROUP;
            const int cn = (int)std::min<int64_t>(POLYQ_GROUP, kb - c0);
            for (int i = 0; i < cn; ++i) {
              w[i] = (double)row[idx[c0 + i]] / tb[c0 + i];
              if (!(std::fabs(w[i]) <= 65504.0)) range_ok = false;
            }
            double sc, z;
            quant_group(w, cn, b, &sc, &z, q);
            for (int i = 0; i < cn; ++i) {
              double d = ((double)q[i] - z) * sc * tb[c0 + i] - (double)row[idx[c0 + i]];
              err[c0 + i] = err[c0 + i] + d * d;
            }
          }
        }
      });
      if (!range_ok.load()) continue;
      double s = 0.0;
      for (int64_t i = 0; i < kb; ++i) s = s + err[i] * x2[idx[i]];
      const double e = s / (double)kb;
      if (!have || e < best_e) {
        have = true;
        best_e = e;
        best_a = al;
        best_t = tb;
      }
    }
    alpha[width_index(b)] = best_a;  // alpha = 0 is always usable
    for (int64_t i = 0; i < kb; ++i) t[idx[i]] = best_t[i];
  }
}

bool is_perm(const int32_t* p, int64_t n) {
  std::vector<uint8_t> seen(n, 0);
  for (int64_t i = 0; i < n; ++i) {
    if (p[i] < 0 || p[i] >= n || seen[p[i]]) return false;
    seen[p[i]] = 1;
  }
  return true;
}

}  // namespace

extern "C" void polyq_pack_opts_default(polyq_pack_opts* o) {
  if (!o) return;
  std::memset(o, 0, sizeof *o);
  o->group_size = POLYQ_GROUP;
  o->palette_mask = (1u << 2) | (1u << 3) | (1u << 4) | (1u << 8) | (1u << 16);
  o->alloc_rule = POLYQ_ALLOC_WATERFILL;
}

extern "C" int polyq_pack(const float* W, int64_t N, int64_t K, const float* act_absmean,
                          double budget_bits, const polyq_pack_opts* opts, polyq_layer** out) {
  polyq_clear_error();
  if (!out) return polyq_set_error(POLYQ_EINVAL, "polyq_pack: out is NULL");
  *out = nullptr;
  polyq_pack_opts o;
  if (opts) o = *opts;
  else polyq_pack_opts_default(&o);
  if (!W) return polyq_set_error(POLYQ_EINVAL, "polyq_pack: W is NULL");
  if (N <= 0 || K <= 0 || N > (1ll << 31) - 1 || K > (1ll << 31) - 1)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: bad shape N=%lld K=%lld", (long long)N,
                           (long long)K);
  if (o.group_size != POLYQ_GROUP)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_pack: group_size must be 64");
  if (o.alloc_rule != POLYQ_ALLOC_WATERFILL && o.alloc_rule != POLYQ_ALLOC_LADDER)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: unknown alloc_rule %d", o.alloc_rule);
  if (o.proxy != POLYQ_PROXY_SALIENCY && o.proxy != POLYQ_PROXY_QUANT)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: unknown proxy %d", o.proxy);
  if (o.proxy == POLYQ_PROXY_QUANT && o.alloc_rule == POLYQ_ALLOC_LADDER)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: the ladder rule needs the saliency proxy");
  if (o.snap_quanta != 0 && o.snap_quanta != 1)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: snap_quanta must be 0 or 1");
  if (o.act_scaling != 0 && o.act_scaling != 1)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: act_scaling must be 0 or 1");
  if (o.snap_quanta && o.forced_bits)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: forced_bits cannot be snapped to quanta");
  int32_t quanta[5] = POLYQ_GPU_QUANTA;
  {
    int nz = 0;
    for (int i = 0; i < 5; ++i) nz += o.quanta[i] != 0;
    if (nz == 5) {
      for (int i = 0; i < 5; ++i) {
        if (o.quanta[i] < 1 || o.quanta[i] > (1 << 24))
          return polyq_set_error(POLYQ_EINVAL, "polyq_pack: quanta[%d] = %d", i, o.quanta[i]);
        quanta[i] = o.quanta[i];
      }
    } else if (nz != 0) {
      return polyq_set_error(POLYQ_EINVAL, "polyq_pack: set all five quanta or none");
    }
  }
  uint32_t mask = o.palette_mask ? o.palette_mask
                                 : ((1u << 2) | (1u << 3) | (1u << 4) | (1u << 8) | (1u << 16));
  std::vector<int> pal;
  for (int b : kPalette)
    if (mask & (1u << b)) pal.push_back(b);
  if (pal.empty() || (mask & ~((1u << 2) | (1u << 3) | (1u << 4) | (1u << 8) | (1u << 16))))
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: bad palette mask 0x%x", mask);
  if ((!o.forced_bits || o.act_scaling) && !act_absmean)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: act_absmean is NULL");
  if (!o.forced_bits) {
    if (!(budget_bits >= 2.0 && budget_bits <= 16.0))
      return polyq_set_error(POLYQ_EINVAL, "polyq_pack: budget %g outside [2,16]", budget_bits);
  }
  // weights: finite and inside fp16 range
  {
    std::atomic<bool> bad(false);
    run_threads(N, o.n_threads, [&](int64_t a, int64_t b) {
      for (int64_t i = a * K; i < b * K; ++i) {
        float v = W[i];
        if (!(std::fabs(v) <= 65504.0f)) {
          bad = true;
          return;
        }
      }
    });
    if (bad.load()) return polyq_set_error(POLYQ_EINVAL, "polyq_pack: W must be finite, |W| <= 65504");
  }
  if (std::fegetround() != FE_TONEAREST)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: host rounding mode must be to-nearest");

  polyq_layer* L = new (std::nothrow) polyq_layer;
  if (!L) return polyq_set_error(POLYQ_ENOMEM, "polyq_pack: out of host memory");
  try {
    L->N = N;
    L->K = K;
    L->budget = budget_bits;
    if (o.forced_bits) {
      L->bits.assign(o.forced_bits, o.forced_bits + K);
      for (int64_t k = 0; k < K; ++k)
        if (width_index(L->bits[k]) < 0) {
          delete L;
          return polyq_set_error(POLYQ_EINVAL, "polyq_pack: forced width %d at %lld",
                                 (int)L->bits[k], (long long)k);
        }
    }
    // E[x^2] of the quantiser proxy and the scaling search
    std::vector<double> x2;
    if (o.proxy == POLYQ_PROXY_QUANT || o.act_scaling) {
      x2.resize(K);
      for (int64_t k = 0; k < K; ++k) {
        const double v = o.act_sqmean ? (double)o.act_sqmean[k] : (double)act_absmean[k];
        x2[k] = o.act_sqmean ? v : v * v;
        if (!(x2[k] >= 0.0 && std::isfinite(x2[k]))) {
          delete L;
          return polyq_set_error(POLYQ_EINVAL, "polyq_pack: E[x^2] of channel %lld is not finite "
                                 "and >= 0", (long long)k);
        }
      }
    }
    if (!o.forced_bits) {
      std::vector<double> sal;
      ErrTable E;
      if (o.proxy == POLYQ_PROXY_QUANT) {
        sal.assign(K, 0.0);  // unused by the waterfilling rule
        quant_table(W, N, K, x2, pal, o.n_threads, E);
      } else {
        saliency(W, N, K, act_absmean, sal, o.n_threads);
        saliency_table(sal, pal, E);
      }
      allocate(sal, E, budget_bits, pal, o.alloc_rule, L->bits);
      if (o.snap_quanta) {
        std::vector<int64_t> cnt(pal.size(), 0);
        for (size_t i = 0; i < pal.size(); ++i)
          for (int64_t k = 0; k < K; ++k) cnt[i] += L->bits[k] == pal[i];
        const std::vector<int64_t> tgt = quanta_targets(pal, cnt, quanta, budget_bits, K);
        reassign(pal, tgt, E, L->bits);
      }
    }
    std::vector<double> tfac;
    if (o.act_scaling)
      choose_alphas(W, N, K, L->bits, act_absmean, x2, o.n_threads, tfac, L->alpha);
    // Section 4.1: stable clustering by width
    L->perm.reserve(K);
    for (int b : kPalette)
      for (int64_t k = 0; k < K; ++k)
        if (L->bits[k] == b) L->perm.push_back((int32_t)k);
    // Section 4.2: blocks
    int32_t pos = 0, off = 0, goff = 0;
    for (int b : kPalette) {
      int32_t kb = 0;
      for (int64_t k = 0; k < K; ++k) kb += L->bits[k] == b;
      if (!kb) continue;
      polyq_block blk;
      blk.bits = b;
      blk.n_ch = kb;
      blk.pos0 = pos;
      blk.seg_off = off;
      blk.seg_bytes = (int32_t)seg_bytes_for(b, kb);
      blk.grp_off = goff;
      blk.n_grp = b == 16 ? 0 : (kb + POLYQ_GROUP - 1) / POLYQ_GROUP;
      L->blocks.push_back(blk);
      pos += kb;
      off += blk.seg_bytes;
      goff += blk.n_grp;
    }
    L->S = off;
    L->G = goff;
    L->packed.assign((size_t)(N * L->S), 0);
    L->meta.assign((size_t)(N * L->G), 0);
    L->out_perm.resize(N);
    for (int64_t n = 0; n < N; ++n) L->out_perm[n] = (int32_t)n;
    const double* tp = o.act_scaling ? tfac.data() : nullptr;
    run_threads(N, o.n_threads, [&](int64_t a, int64_t b) { pack_rows(W, K, tp, *L, a, b); });
    if (o.act_scaling) {
      L->xscale.resize(K);
      for (int64_t p = 0; p < K; ++p) L->xscale[p] = (float)tfac[L->perm[p]];
    }
  } catch (const std::bad_alloc&) {
    delete L;
    return polyq_set_error(POLYQ_ENOMEM, "polyq_pack: out of host memory");
  }
  *out = L;
  return POLYQ_OK;
}

extern "C" void polyq_free(polyq_layer* L) { delete L; }

extern "C" int polyq_layer_info(const polyq_layer* L, polyq_info* out) {
  polyq_clear_error();
  if (!L || !out) return polyq_set_error(POLYQ_EINVAL, "polyq_layer_info: NULL argument");
  std::memset(out, 0, sizeof *out);
  out->N = L->N;
  out->K = L->K;
  out->row_stride = L->S;
  out->n_groups = L->G;
  out->n_blocks = (int32_t)L->blocks.size();
  for (size_t i = 0; i < L->blocks.size(); ++i) out->blocks[i] = L->blocks[i];
  out->budget = L->budget;
  int64_t sum = 0;
  for (uint8_t b : L->bits) sum += b;
  out->b_real = (double)sum / (double)L->K;
  out->packed_bytes = L->N * L->S;
  out->meta_bytes = L->N * L->G * 4;
  out->meta_stride = (L->G + 3) / 4 * 4;
  int64_t pad = 0;
  for (const polyq_block& b : L->blocks) {
    const int64_t raw = b.bits == 16 ? 2 * (int64_t)b.n_ch : ((int64_t)b.n_ch * b.bits + 7) / 8;
    pad += b.seg_bytes - raw;
  }
  out->pad_bytes = pad;
  for (int i = 0; i < 5; ++i) out->alpha[i] = L->alpha[i];
  out->has_xscale = L->xscale.empty() ? 0 : 1;
  return POLYQ_OK;
}

extern "C" int polyq_layer_xscale(const polyq_layer* L, float* xscale) {
  polyq_clear_error();
  if (!L || !xscale) return polyq_set_error(POLYQ_EINVAL, "polyq_layer_xscale: NULL argument");
  for (int64_t p = 0; p < L->K; ++p) xscale[p] = L->xscale.empty() ? 1.0f : L->xscale[p];
  return POLYQ_OK;
}

extern "C" int polyq_layer_export(const polyq_layer* L, uint8_t* packed, uint32_t* meta,
                                  int64_t meta_stride, int32_t* perm, uint8_t* bits,
                                  int32_t* out_perm) {
  polyq_clear_error();
  if (!L) return polyq_set_error(POLYQ_EINVAL, "polyq_layer_export: NULL layer");
  if (meta && meta_stride < L->G)
    return polyq_set_error(POLYQ_EINVAL, "polyq_layer_export: meta_stride %lld < n_groups %lld",
                           (long long)meta_stride, (long long)L->G);
  if (packed) std::memcpy(packed, L->packed.data(), L->packed.size());
  if (meta) {
    for (int64_t n = 0; n < L->N; ++n) {
      uint32_t* dst = meta + n * meta_stride;
      if (L->G) std::memcpy(dst, L->meta.data() + n * L->G, L->G * 4);
      for (int64_t g = L->G; g < meta_stride; ++g) dst[g] = 0u;
    }
  }
  if (perm) std::memcpy(perm, L->perm.data(), L->perm.size() * 4);
  if (bits) std::memcpy(bits, L->bits.data(), L->bits.size());
  if (out_perm) std::memcpy(out_perm, L->out_perm.data(), L->out_perm.size() * 4);
  return POLYQ_OK;
}

extern "C" int polyq_layer_permute_rows(polyq_layer* L, const int32_t* rp) {
  polyq_clear_error();
  if (!L || !rp) return polyq_set_error(POLYQ_EINVAL, "polyq_layer_permute_rows: NULL argument");
  if (!is_perm(rp, L->N))
    return polyq_set_error(POLYQ_EINVAL, "polyq_layer_permute_rows: not a permutation of 0..N-1");
  std::vector<uint8_t> np(L->packed.size());
  std::vector<uint32_t> nm(L->meta.size());
  std::vector<int32_t> no(L->N);
  for (int64_t i = 0; i < L->N; ++i) {
    int64_t s = rp[i];
    std::memcpy(np.data() + i * L->S, L->packed.data() + s * L->S, L->S);
    if (L->G) std::memcpy(nm.data() + i * L->G, L->meta.data() + s * L->G, L->G * 4);
    no[i] = L->out_perm[s];
  }
  L->packed.swap(np);
  L->meta.swap(nm);
  L->out_perm.swap(no);
  return POLYQ_OK;
}

extern "C" int polyq_permute_merge(const int32_t* beta, const int32_t* pc, int64_t n,
                                   int32_t* gather_out) {
  polyq_clear_error();
  if (!beta || !pc || !gather_out || n <= 0)
    return polyq_set_error(POLYQ_EINVAL, "polyq_permute_merge: bad argument");
  if (!is_perm(beta, n) || !is_perm(pc, n))
    return polyq_set_error(POLYQ_EINVAL, "polyq_permute_merge: inputs must be permutations");
  std::vector<int32_t> inv(n);
  for (int64_t i = 0; i < n; ++i) inv[beta[i]] = (int32_t)i;
  for (int64_t p = 0; p < n; ++p) gather_out[p] = inv[pc[p]];
  return POLYQ_OK;
}

extern "C" int polyq_dev_layer_fill(const polyq_layer* L, const uint8_t* packed_dev,
                                    const uint32_t* meta_dev, const int32_t* gather_dev,
                                    polyq_dev_layer* out) {
  polyq_clear_error();
  if (!L || !out || !packed_dev || (!meta_dev && L->G))
    return polyq_set_error(POLYQ_EINVAL, "polyq_dev_layer_fill: NULL argument");
  std::memset(out, 0, sizeof *out);
  out->packed = packed_dev;
  out->meta = meta_dev;
  out->gather = gather_dev;
  out->N = L->N;
  out->K = L->K;
  out->row_stride = L->S;
  out->n_groups = L->G;
  out->meta_stride = (L->G + 3) / 4 * 4;
  out->n_blocks = (int32_t)L->blocks.size();
  for (size_t i = 0; i < L->blocks.size(); ++i) out->blocks[i] = L->blocks[i];
  return POLYQ_OK;
}

// Structural checks on a device-layer descriptor (host only, no device reads).
int polyq_check_dev_layer(const polyq_dev_layer* L, const char* who) {
  if (!L) return polyq_set_error(POLYQ_EINVAL, "%s: NULL layer", who);
  if (!L->packed) return polyq_set_error(POLYQ_EINVAL, "%s: packed is NULL", who);
  if (L->N <= 0 || L->K <= 0 || L->N > (1ll << 31) - 1 || L->K > (1ll << 31) - 1)
    return polyq_set_error(POLYQ_EINVAL, "%s: bad shape", who);
  if (L->row_stride <= 0 || L->row_stride % 16)
    return polyq_set_error(POLYQ_EINVAL, "%s: row_stride must be a positive multiple of 16", who);
  if (((uintptr_t)L->packed) % 16 || ((uintptr_t)L->meta) % 16 || ((uintptr_t)L->xscale) % 16)
    return polyq_set_error(POLYQ_EINVAL, "%s: packed/meta/xscale must be 16-byte aligned", who);
  if (L->n_blocks < 1 || L->n_blocks > POLYQ_MAX_BLOCKS)
    return polyq_set_error(POLYQ_EINVAL, "%s: bad block count", who);
  int32_t pos = 0, off = 0, goff = 0, prev = 0;
  for (int i = 0; i < L->n_blocks; ++i) {
    const polyq_block& b = L->blocks[i];
    if (width_index(b.bits) < 0 || b.bits <= prev || b.n_ch <= 0 || b.pos0 != pos ||
        b.seg_off != off || b.seg_bytes != seg_bytes_for(b.bits, b.n_ch) || b.grp_off != goff ||
        b.n_grp != (b.bits == 16 ? 0 : (b.n_ch + POLYQ_GROUP - 1) / POLYQ_GROUP))
      return polyq_set_error(POLYQ_EINVAL, "%s: corrupt block table entry %d", who, i);
    prev = b.bits;
    pos += b.n_ch;
    off += b.seg_bytes;
    goff += b.n_grp;
  }
  if (pos != L->K || off != L->row_stride || goff != L->n_groups)
    return polyq_set_error(POLYQ_EINVAL, "%s: block table does not cover the layer", who);
  if (L->n_groups > 0 && !L->meta) return polyq_set_error(POLYQ_EINVAL, "%s: meta is NULL", who);
  if (L->meta_stride < L->n_groups || L->meta_stride % 4)
    return polyq_set_error(POLYQ_EINVAL, "%s: meta_stride must be a multiple of 4 >= n_groups",
                           who);
  return POLYQ_OK;
}
