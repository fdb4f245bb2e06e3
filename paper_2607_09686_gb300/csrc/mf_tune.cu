// Cache-size tuner (host code): predicts, for candidate cache percentages, the misses a route
// trace incurs and the resulting decode time, and picks the accepted candidate with the highest
// predicted rate.
//
// Throughput model (section "Throughput Model"):
//   T(p) = tokens / (compute_time + materialization_time(p) + pressure_penalty(F))
// with compute_time = tokens * t_token (measured, every expert resident), materialization_time
// = misses(p) * t_miss (measured per payload) and no pressure term inside the static budget (the
// slot pool is dedicated HBM).  The Discussion ("Cache Hit Rate Is an Incomplete Objective")
// asks for the cache point of least latency under the budget rather than the highest hit rate;
// mf_plan supplies the budget decision for each candidate.
//
// misses(p) follows the library's cache semantics: each layer has its own least-recently-used
// cache of S slots; a step of T tokens presents its distinct experts once each, in
// first-occurrence order or resident-first order, and the kernels decide them one at a time in
// that order (their waves of S only group the accesses for the compute: no access evicts an
// expert accessed earlier in its own wave), so the replay is serial.
//   First-occurrence order: LRU is a stack algorithm (Mattson et al., 1970): a cache of S slots
//   holds the S most recently used experts, so an access hits exactly when its stack distance
//   (1 + the number of distinct experts used since its previous access) is at most S.  One pass
//   over the trace gives the distance histogram, and hits(S) for every S.
//   Resident-first order (steps of more than one token; a one-token step keeps first-occurrence
//   order, as mf_access_order specifies): the order depends on what is resident, so each
//   distinct S is replayed on its own.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

#include "mawforge.h"

namespace {

// Distinct experts of tokens [t0, t1) of layer l, in (token, rank) first-occurrence order.
void step_experts(const int32_t* routes, int n_tokens, int k, int l, int t0, int t1, std::vector<int>& seen_at,
                  int stamp, std::vector<int>& out) {
  out.clear();
  const int32_t* r = routes + ((size_t)l * n_tokens + t0) * k;
  for (int i = 0; i < (t1 - t0) * k; ++i) {
    const int e = r[i];
    if (seen_at[e] != stamp) {
      seen_at[e] = stamp;
      out.push_back(e);
    }
  }
}

// hist[d] = accesses with stack distance d (1..E); cold = first accesses; per layer, summed.
void stack_distances(const int32_t* routes, int L, int n_tokens, int k, int E, int T, std::vector<uint64_t>& hist,
                     uint64_t& cold, uint64_t& accesses) {
  hist.assign((size_t)E + 1, 0);
  cold = accesses = 0;
  std::vector<int> seen_at(E, -1), uniq, stack;  // stack: most recent last
  int stamp = 0;
  for (int l = 0; l < L; ++l) {
    stack.clear();
    for (int t0 = 0; t0 < n_tokens; t0 += T) {
      step_experts(routes, n_tokens, k, l, t0, std::min(n_tokens, t0 + T), seen_at, stamp++, uniq);
      for (int e : uniq) {
        ++accesses;
        auto it = std::find(stack.rbegin(), stack.rend(), e);
        if (it == stack.rend()) {
          ++cold;
        } else {
          ++hist[(size_t)(it - stack.rbegin()) + 1];
          stack.erase(std::next(it).base());
        }
        stack.push_back(e);
      }
    }
  }
}

// Misses of a serial replay with S slots per layer, resident-first order within each step of
// more than one token.
uint64_t replay_resident_first(const int32_t* routes, int L, int n_tokens, int k, int E, int T, int S,
                               uint64_t& accesses) {
  uint64_t misses = 0;
  accesses = 0;
  std::vector<int> seen_at(E, -1), uniq, order, lru;  // lru: most recent last, size <= S
  std::vector<char> resident(E, 0);
  int stamp = 0;
  for (int l = 0; l < L; ++l) {
    lru.clear();
    std::fill(resident.begin(), resident.end(), 0);
    for (int t0 = 0; t0 < n_tokens; t0 += T) {
      const int t1 = std::min(n_tokens, t0 + T);
      step_experts(routes, n_tokens, k, l, t0, t1, seen_at, stamp++, uniq);
      order.clear();
      if (t1 - t0 > 1) {
        for (int e : uniq)
          if (resident[e]) order.push_back(e);
        for (int e : uniq)
          if (!resident[e]) order.push_back(e);
      } else {
        order = uniq;
      }
      for (int e : order) {
        ++accesses;
        if (resident[e]) {
          lru.erase(std::find(lru.begin(), lru.end(), e));
        } else {
          ++misses;
          if ((int)lru.size() == S) {
            resident[lru.front()] = 0;
            lru.erase(lru.begin());
          }
          resident[e] = 1;
        }
        lru.push_back(e);
      }
    }
  }
  return misses;
}

}  // namespace

extern "C" int mf_tune_cache(const mf_model_t* m, const mf_plan_req_t* req, const int32_t* routes, int n_tokens,
                             int T, int order, double t_token_s, double t_miss_s, const double* pcts, int n,
                             mf_tune_point_t* out, int* best) {
  if (!m || !req || !routes || !pcts || !out || !best || n < 1 || n_tokens < 1 || T < 1) return MF_E_INVAL;
  if (order != MF_ORDER_FIRST_OCCURRENCE && order != MF_ORDER_RESIDENT_FIRST) return MF_E_INVAL;
  if (!(t_token_s >= 0.0) || !(t_miss_s >= 0.0) || !std::isfinite(t_token_s) || !std::isfinite(t_miss_s))
    return MF_E_INVAL;
  // every candidate's plan first: the model and the requests are validated before any work
  std::vector<mf_plan_t> plans((size_t)n);
  for (int i = 0; i < n; ++i) {
    mf_plan_req_t r = *req;
    r.cache_pct = pcts[i];
    const int rc = mf_plan(m, &r, &plans[(size_t)i]);
    if (rc != MF_OK && rc != MF_E_BUDGET) return rc;
  }
  const int L = m->n_layers, E = m->n_experts, k = m->top_k;
  const size_t n_routes = (size_t)L * n_tokens * k;
  for (size_t i = 0; i < n_routes; ++i)
    if (routes[i] < 0 || routes[i] >= E) return MF_E_INVAL;

  std::vector<uint64_t> hist;
  uint64_t cold = 0, accesses = 0;
  if (order == MF_ORDER_FIRST_OCCURRENCE) stack_distances(routes, L, n_tokens, k, E, T, hist, cold, accesses);
  std::vector<mf_tune_point_t> res((size_t)n);
  for (int i = 0; i < n; ++i) {
    const mf_plan_t& p = plans[(size_t)i];
    mf_tune_point_t& o = res[(size_t)i];
    std::memset(&o, 0, sizeof(o));
    o.cache_pct = pcts[i];
    o.accepted = p.accepted;
    o.slots_per_layer = p.slots_per_layer;
    o.pool_bytes = p.pool_bytes;
    o.footprint_bytes = p.footprint_bytes;
    const int S = p.slots_per_layer;
    if (order == MF_ORDER_FIRST_OCCURRENCE) {
      uint64_t hits = 0;
      for (int d = 1; d <= std::min(S, E); ++d) hits += hist[(size_t)d];
      o.accesses = accesses;
      o.hits = hits;
      o.misses = accesses - hits;
    } else {
      int same = -1;  // candidates with the same S replay identically
      for (int j = 0; j < i && same < 0; ++j)
        if (res[(size_t)j].slots_per_layer == S) same = j;
      if (same >= 0) {
        o.accesses = res[(size_t)same].accesses;
        o.misses = res[(size_t)same].misses;
      } else {
        o.misses = replay_resident_first(routes, L, n_tokens, k, E, T, S, o.accesses);
      }
      o.hits = o.accesses - o.misses;
    }
    o.bytes_materialized = o.misses * p.payload_bytes;
    o.predicted_s = (double)n_tokens * t_token_s + (double)o.misses * t_miss_s;
    o.predicted_tokens_per_s = o.predicted_s > 0.0 ? (double)n_tokens / o.predicted_s : 0.0;
  }
  int b = -1;
  for (int i = 0; i < n; ++i) {
    const mf_tune_point_t& o = res[(size_t)i];
    if (!o.accepted) continue;
    if (b < 0 || o.predicted_tokens_per_s > res[(size_t)b].predicted_tokens_per_s ||
        (o.predicted_tokens_per_s == res[(size_t)b].predicted_tokens_per_s && o.pool_bytes < res[(size_t)b].pool_bytes))
      b = i;
  }
  std::memcpy(out, res.data(), sizeof(mf_tune_point_t) * (size_t)n);
  *best = b;
  return b >= 0 ? MF_OK : MF_E_BUDGET;
}
