// Section 4.4 graph-based permutation planning on the host: channel orders
// ("bases") for the activation edges of a static operator DAG, chosen so
// that the explicit activation shuffles cost the least modelled traffic
// (Section 5.4: A16 read + write, 4 bytes per channel per shuffle).
//
// Edges joined by order-keeping nodes form regions; every edge of a region
// carries the same order.  A region's cost for a candidate order is one
// shuffle per distinct (edge, order wanted by a consumer) that differs from
// it, plus one per fixed-order producer that differs, each of the edge's
// width.  The candidates are the natural order and the permutations of the
// linears reading the region; regions are independent, so taking the
// cheapest candidate of each gives the plan.
#include <algorithm>
#include <cstring>
#include <map>
#include <new>
#include <set>
#include <utility>
#include <vector>

#include "polyq.h"
#include "polyq_internal.h"

namespace {

constexpr int32_t kNatural = -1;

struct Dsu {
  std::vector<int32_t> p;
  explicit Dsu(int32_t n) : p(n) {
    for (int32_t i = 0; i < n; ++i) p[i] = i;
  }
  int32_t find(int32_t i) {
    while (p[i] != i) i = p[i] = p[p[i]];
    return i;
  }
  void join(int32_t a, int32_t b) {
    a = find(a);
    b = find(b);
    if (a != b) p[std::max(a, b)] = std::min(a, b);
  }
};

int check_nodes(const polyq_plan_node* nodes, int32_t n_nodes, const int64_t* dims,
                int32_t n_edges, const int64_t* perm_lens, int32_t n_perms) {
  const char* who = "polyq_plan_graph";
  std::vector<uint8_t> produced(n_edges, 0);
  auto edge_ok = [&](int32_t e) { return e >= 0 && e < n_edges; };
  for (int32_t i = 0; i < n_nodes; ++i) {
    const polyq_plan_node& nd = nodes[i];
    if (nd.n_in < 0 || nd.n_in > 3)
      return polyq_set_error(POLYQ_EINVAL, "%s: node %d has %d inputs", who, i, nd.n_in);
    for (int j = 0; j < nd.n_in; ++j)
      if (!edge_ok(nd.in[j]))
        return polyq_set_error(POLYQ_EINVAL, "%s: node %d input %d is not an edge", who, i, j);
    if (nd.out != -1 && !edge_ok(nd.out))
      return polyq_set_error(POLYQ_EINVAL, "%s: node %d output is not an edge", who, i);
    if (nd.out >= 0) {
      if (produced[nd.out])
        return polyq_set_error(POLYQ_EINVAL, "%s: edge %d has two producers", who, nd.out);
      produced[nd.out] = 1;
    }
    bool ok = true;
    switch (nd.kind) {
      case POLYQ_NODE_SOURCE_FIXED:
      case POLYQ_NODE_SOURCE_FREE:
        ok = nd.n_in == 0 && nd.out >= 0;
        break;
      case POLYQ_NODE_LINEAR:
        ok = nd.n_in == 1 && nd.out >= 0 && nd.perm >= 0 && nd.perm < n_perms &&
             perm_lens[nd.perm] == dims[nd.in[0]];
        break;
      case POLYQ_NODE_ELEMENTWISE:
        ok = nd.n_in >= 1 && nd.out >= 0;
        for (int j = 0; ok && j < nd.n_in; ++j) ok = dims[nd.in[j]] == dims[nd.out];
        break;
      case POLYQ_NODE_BOUNDARY:
        ok = nd.n_in >= 1;
        break;
      case POLYQ_NODE_ATTENTION:
        ok = nd.n_in == 3;
        break;
      default:
        return polyq_set_error(POLYQ_EINVAL, "%s: node %d has unknown kind %d", who, i, nd.kind);
    }
    if (!ok)
      return polyq_set_error(POLYQ_EINVAL, "%s: node %d (kind %d) has wrong inputs, output, "
                             "widths or permutation", who, i, nd.kind);
  }
  return POLYQ_OK;
}

}  // namespace

extern "C" int polyq_plan_graph(const polyq_plan_node* nodes, int32_t n_nodes,
                                const int64_t* dims, int32_t n_edges,
                                const int32_t* const* perms, const int64_t* perm_lens,
                                int32_t n_perms, int32_t* labels, int64_t* bytes_per_token) {
  polyq_clear_error();
  const char* who = "polyq_plan_graph";
  if (!nodes || n_nodes < 1 || !dims || n_edges < 1 || !labels || n_perms < 0 ||
      (n_perms > 0 && (!perms || !perm_lens)))
    return polyq_set_error(POLYQ_EINVAL, "%s: bad argument", who);
  for (int32_t e = 0; e < n_edges; ++e)
    if (dims[e] < 1 || dims[e] > (1ll << 31) - 1)
      return polyq_set_error(POLYQ_EINVAL, "%s: edge %d has width %lld", who, e,
                             (long long)dims[e]);
  try {
    // permutations: validity, identity -> natural, equal contents -> one key
    std::vector<int32_t> key(n_perms);
    std::map<std::vector<int32_t>, int32_t> seen;
    for (int32_t i = 0; i < n_perms; ++i) {
      const int64_t n = perm_lens[i];
      if (!perms[i] || n < 1 || n > (1ll << 31) - 1)
        return polyq_set_error(POLYQ_EINVAL, "%s: permutation %d is empty", who, i);
      std::vector<uint8_t> hit(n, 0);
      bool ident = true;
      for (int64_t j = 0; j < n; ++j) {
        const int32_t v = perms[i][j];
        if (v < 0 || v >= n || hit[v])
          return polyq_set_error(POLYQ_EINVAL, "%s: perms[%d] is not a permutation", who, i);
        hit[v] = 1;
        ident = ident && v == j;
      }
      if (ident) {
        key[i] = kNatural;
        continue;
      }
      key[i] = seen.emplace(std::vector<int32_t>(perms[i], perms[i] + n), i).first->second;
    }
    int rc = check_nodes(nodes, n_nodes, dims, n_edges, perm_lens, n_perms);
    if (rc) return rc;

    // regions
    Dsu dsu(n_edges);
    for (int32_t i = 0; i < n_nodes; ++i) {
      const polyq_plan_node& nd = nodes[i];
      if (nd.kind == POLYQ_NODE_ELEMENTWISE)
        for (int j = 0; j < nd.n_in; ++j) dsu.join(nd.in[j], nd.out);
      else if (nd.kind == POLYQ_NODE_ATTENTION && nd.out >= 0 && dims[nd.in[2]] == dims[nd.out])
        dsu.join(nd.in[2], nd.out);
    }
    // requests: (edge, order) wanted by consumers, fixed by producers
    std::set<std::pair<int32_t, int32_t>> want;
    std::vector<std::pair<int32_t, int32_t>> fixed;
    for (int32_t i = 0; i < n_nodes; ++i) {
      const polyq_plan_node& nd = nodes[i];
      switch (nd.kind) {
        case POLYQ_NODE_LINEAR:
          want.insert({nd.in[0], key[nd.perm]});
          break;
        case POLYQ_NODE_BOUNDARY:
          for (int j = 0; j < nd.n_in; ++j) want.insert({nd.in[j], kNatural});
          if (nd.out >= 0) fixed.push_back({nd.out, kNatural});
          break;
        case POLYQ_NODE_ATTENTION:
          want.insert({nd.in[0], kNatural});
          want.insert({nd.in[1], kNatural});
          if (nd.out >= 0 && dims[nd.in[2]] != dims[nd.out]) {
            want.insert({nd.in[2], kNatural});
            fixed.push_back({nd.out, kNatural});
          }
          break;
        case POLYQ_NODE_SOURCE_FIXED:
          fixed.push_back({nd.out, kNatural});
          break;
        default:
          break;
      }
    }
    // per region: total width of requests, and what each order saves
    struct Region {
      int64_t total = 0;
      std::map<int32_t, int64_t> saved;  // order -> width it satisfies
    };
    std::map<int32_t, Region> reg;
    for (int32_t e = 0; e < n_edges; ++e) reg[dsu.find(e)];
    for (const auto& w : want) {
      Region& r = reg[dsu.find(w.first)];
      r.total += dims[w.first];
      r.saved[w.second] += dims[w.first];
    }
    for (const auto& f : fixed) {
      Region& r = reg[dsu.find(f.first)];
      r.total += dims[f.first];
      r.saved[f.second] += dims[f.first];
    }
    int64_t cost = 0;
    std::map<int32_t, int32_t> choice;
    for (auto& kv : reg) {
      Region& r = kv.second;
      // candidates: natural first, then orders wanted here in ascending id
      // (fixed producers only ever want the natural order)
      int32_t best = kNatural;
      int64_t best_saved = r.saved.count(kNatural) ? r.saved[kNatural] : 0;
      for (const auto& s : r.saved)
        if (s.first != kNatural && s.second > best_saved) {
          best = s.first;
          best_saved = s.second;
        }
      choice[kv.first] = best;
      cost += r.total - best_saved;
    }
    for (int32_t e = 0; e < n_edges; ++e) labels[e] = choice[dsu.find(e)];
    if (bytes_per_token) *bytes_per_token = 4 * cost;
  } catch (const std::bad_alloc&) {
    return polyq_set_error(POLYQ_ENOMEM, "%s: out of host memory", who);
  }
  return POLYQ_OK;
}
