// Host side of the PolyQ library: width allocation (Section 3.2), clustering
// permutation and bit blocks (Sections 4.1, 4.2), group quantisation and
// packing, and the permutation merge rule (Section 4.3).
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

// Gain per extra bit, Section 3.2.
double step_gain(double sal, int b, int bn) {
  return (proxy_error(sal, b) - proxy_error(sal, bn)) / (double)(bn - b);
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

// Section 3.2 greedy allocation under budget B.
void allocate(const std::vector<double>& sal, double B, const std::vector<int>& pal, int rule,
              std::vector<uint8_t>& bits) {
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
  for (int64_t k = 0; k < K; ++k) init.push_back({step_gain(sal[k], bmin, b1), (int32_t)k, b1});
  std::priority_queue<Cand, std::vector<Cand>, CandLess> heap(CandLess(), std::move(init));
  while (delta > 0 && !heap.empty()) {
    Cand c = heap.top();
    heap.pop();
    int cost = c.bn - bits[c.k];
    if (cost > delta) continue;  // Delta only shrinks: this step never fits
    bits[c.k] = (uint8_t)c.bn;
    delta -= cost;
    int bn2 = next_w(c.bn);
    if (bn2) heap.push({step_gain(sal[c.k], c.bn, bn2), c.k, bn2});
  }
}

int64_t seg_bytes_for(int b, int64_t kb) {
  int64_t raw = b == 16 ? kb * 2 : (kb * b + 7) / 8;
  return (raw + 15) / 16 * 16;
}

// Quantise and pack rows [r0, r1) of the layer.
void pack_rows(const float* W, int64_t K, polyq_layer& L, int64_t r0, int64_t r1) {
  std::vector<double> w(POLYQ_GROUP);
  std::vector<uint32_t> q(POLYQ_GROUP);
  for (int64_t n = r0; n < r1; ++n) {
    const float* row = W + n * K;
    uint8_t* prow = L.packed.data() + n * L.S;
    uint32_t* mrow = L.meta.data() + n * L.G;
    for (const polyq_block& blk : L.blocks) {
      uint8_t* seg = prow + blk.seg_off;
      const int32_t* pp = L.perm.data() + blk.pos0;
      const int b = blk.bits;
      if (b == 16) {
        for (int32_t i = 0; i < blk.n_ch; ++i) {
          uint16_t h = polyq_f64_to_f16((double)row[pp[i]]);
          seg[2 * i] = (uint8_t)(h & 0xFF);
          seg[2 * i + 1] = (uint8_t)(h >> 8);
        }
        continue;
      }
      const double qmax = (double)((1 << b) - 1);
      uint64_t acc = 0;  // LSB-first bit writer
      int nacc = 0;
      int64_t wb = 0;
      for (int32_t g = 0; g < blk.n_grp; ++g) {
        int32_t c0 = g * POLYQ_GROUP;
        int32_t cn = std::min<int32_t>(POLYQ_GROUP, blk.n_ch - c0);
        double lo = INFINITY, hi = -INFINITY;
        for (int32_t i = 0; i < cn; ++i) {
          w[i] = (double)row[pp[c0 + i]];
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
        for (int32_t i = 0; i < cn; ++i) {
          double v = std::nearbyint(w[i] / s) + z;
          v = std::min(std::max(v, 0.0), qmax);
          q[i] = (uint32_t)v;
        }
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
  if (o.snap_quanta != 0)
    return polyq_set_error(POLYQ_EUNSUPPORTED, "polyq_pack: quanta matching is not built");
  if (o.alloc_rule != POLYQ_ALLOC_WATERFILL && o.alloc_rule != POLYQ_ALLOC_LADDER)
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: unknown alloc_rule %d", o.alloc_rule);
  uint32_t mask = o.palette_mask ? o.palette_mask
                                 : ((1u << 2) | (1u << 3) | (1u << 4) | (1u << 8) | (1u << 16));
  std::vector<int> pal;
  for (int b : kPalette)
    if (mask & (1u << b)) pal.push_back(b);
  if (pal.empty() || (mask & ~((1u << 2) | (1u << 3) | (1u << 4) | (1u << 8) | (1u << 16))))
    return polyq_set_error(POLYQ_EINVAL, "polyq_pack: bad palette mask 0x%x", mask);
  if (!o.forced_bits) {
    if (!act_absmean) return polyq_set_error(POLYQ_EINVAL, "polyq_pack: act_absmean is NULL");
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
    } else {
      std::vector<double> sal;
      saliency(W, N, K, act_absmean, sal, o.n_threads);
      allocate(sal, budget_bits, pal, o.alloc_rule, L->bits);
    }
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
    run_threads(N, o.n_threads, [&](int64_t a, int64_t b) { pack_rows(W, K, *L, a, b); });
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
  if (((uintptr_t)L->packed) % 16 || ((uintptr_t)L->meta) % 16)
    return polyq_set_error(POLYQ_EINVAL, "%s: packed/meta must be 16-byte aligned", who);
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
