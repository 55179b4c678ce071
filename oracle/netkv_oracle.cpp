// NetKV CPU oracle: a plain, slow, double-precision statement of what the
// decode-instance scoring path computes (arXiv 2606.03910, "NetKV").
//
// TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
// load this file; only the tests, the package's smoke check and the benchmark's
// CPU-baseline leg use it.  It shares no code with the CUDA library: it knows
// the instance tree only through the documented link-numbering convention and
// computes everything by the definitions below, in double precision.
//
// What it states, with the paper's passage for each part:
//   * KV size, Eq. 1 (Sec. III-B): s = 2 * n_layers * n_kv_heads * d_head * l * b_elem.
//   * Locality tier tau(p,d) in {0,1,2,3} (Sec. III-A): same node / leaf / pod / other,
//     found here by climbing the tree from both instances until their ancestors meet.
//   * Effective bandwidth, Eq. 4 (Sec. III-D), generalised per link: the bottleneck
//     of B_level(e) * (1 - u_e) over every link e on the up and down path, with the
//     self-contention count n_inflight = 0 (the paper allows n_inflight == 0 when
//     telemetry already covers the scheduler's flows).  With one utilisation per tier
//     this is exactly B_tau * (1 - c_tau) (Sec. III-D, per-tier collapse).
//   * Paper-literal per-tier mode (Sec. III-E): B_eff = B_tau * (1 - c_tau) from four
//     per-tier congestion values, no minimum over a path's lower levels.
//   * Directed links (optional): one utilisation per link and direction; a transfer
//     climbs the source's links at their upward utilisation and descends the
//     destination's at their downward one.
//   * Transfer time, Eq. 3: T = s / B_eff + L_tau.
//   * Block-level prefix hit (Sec. III-B): lambda = 16 * |LCP_block(h_r, K_d)|, the number
//     of leading blocks of the request's hash chain that are all in decode d's cache.
//   * Effective transfer size, Eq. 2: s_eff = s * (1 - lambda / l).
//   * Algorithm 1 (Sec. V-A) as a weighted score: filter by capacity (line 1), reject
//     when nothing is feasible (line 2), score every candidate (lines 3-11), take the
//     argmin with the lowest index among equal scores (line 13), then update load.
//   * Evolving caches (the simulator's LRU-managed block cache, Sec. VI-B), in
//     oracle_schedule_stream_evolving: a dispatch makes the request's blocks the most
//     recently used ones of its decode's cache (block 0 last, so the most recent), the
//     least recently used blocks beyond the decode's capacity are evicted, and later
//     arrivals match against the caches of their moment.
//   * The compute-load model (Sec. III-C, IV-B, the feasible set of Sec. IV-A), in
//     oracle_schedule_stream_load: T_queue + T_decode from each decode's request count
//     and t_iter(beta) = a + b beta, memory feasibility m_d >= s_eff + m_min.
//   * Self-contention (Eq. 4's n_inflight, Algorithm 1 lines 5 and 14, Sec. V-C), in
//     oracle_schedule_stream_inflight: a per-(prefill, tier) counter divides the
//     effective bandwidth by 1 + n; a dispatch raises the counter of its tier (saturating
//     at the cap) and its transfer completes, lowering it again (never below zero), at
//     the arrival time plus the chosen candidate's transfer time rounded to whole
//     microseconds.  Completions due at or before an arrival are applied before it.
//
// Parity: pinned by the not-gpu tests (worked example of Sec. III-D, closed forms of
// Eq. 1, the per-tier special case of Eq. 4, brute force on tiny instances,
// Propositions 1 and 2, first-miss LCP semantics).
#include <omp.h>

#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <list>
#include <queue>
#include <unordered_map>
#include <unordered_set>
#include <vector>

namespace {

struct Tree {
  uint32_t f[4];  // instances per node, nodes per leaf, leaves per pod, pods
  uint64_t n;     // instances
  uint64_t n_node, n_leaf, n_pod;
};

Tree make_tree(const uint32_t* fanout) {
  Tree t;
  for (int k = 0; k < 4; ++k) t.f[k] = fanout[k];
  t.n_pod = t.f[3];
  t.n_leaf = t.n_pod * t.f[2];
  t.n_node = t.n_leaf * t.f[1];
  t.n = t.n_node * t.f[0];
  return t;
}

// Ancestor of instance i at height h: h=0 the instance, 1 its node, 2 its leaf,
// 3 its pod, 4 the spine (index 0).
uint64_t ancestor(const Tree& t, uint64_t i, int h) {
  uint64_t a = i;
  for (int k = 0; k < h && k < 4; ++k) a /= t.f[k];
  return h >= 4 ? 0 : a;
}

// Link from the height-h ancestor of i up to its parent.  Links are numbered in
// consecutive blocks per level: instance-node links [0, N), node-leaf links
// [N, N + n_node), leaf-pod links next, pod-spine links last.
uint64_t uplink(const Tree& t, uint64_t i, int h) {
  uint64_t base = 0;
  const uint64_t block[4] = {t.n, t.n_node, t.n_leaf, t.n_pod};
  for (int k = 0; k < h; ++k) base += block[k];
  return base + ancestor(t, i, h);
}

// Locality tier: the lowest height h such that i and j share their height-(h+1) ancestor.
int tier(const Tree& t, uint64_t i, uint64_t j) {
  for (int h = 0; h < 4; ++h)
    if (ancestor(t, i, h + 1) == ancestor(t, j, h + 1)) return h;
  return 3;
}

// Bottleneck residual bandwidth over the unique tree path between i and j.
double path_bottleneck(const Tree& t, const double* bw, const float* u_row,
                       uint64_t i, uint64_t j, int* tau_out) {
  const int tau = tier(t, i, j);
  double b = std::numeric_limits<double>::infinity();
  for (int h = 0; h <= tau; ++h) {
    const uint64_t ei = uplink(t, i, h), ej = uplink(t, j, h);
    const double ri = bw[h] * (1.0 - (double)u_row[ei]);
    const double rj = bw[h] * (1.0 - (double)u_row[ej]);
    if (ri < b) b = ri;
    if (rj < b) b = rj;
  }
  if (tau_out) *tau_out = tau;
  return b;
}

// Directed links (one utilisation per link and direction): a transfer from instance i to
// instance j climbs i's links (their upward utilisation) and descends j's links (their
// downward utilisation).  With u_up == u_down this is path_bottleneck.
double path_bottleneck_dir(const Tree& t, const double* bw, const float* u_up,
                           const float* u_down, uint64_t i, uint64_t j, int* tau_out) {
  const int tau = tier(t, i, j);
  double b = std::numeric_limits<double>::infinity();
  for (int h = 0; h <= tau; ++h) {
    const double ri = bw[h] * (1.0 - (double)u_up[uplink(t, i, h)]);
    const double rj = bw[h] * (1.0 - (double)u_down[uplink(t, j, h)]);
    if (ri < b) b = ri;
    if (rj < b) b = rj;
  }
  if (tau_out) *tau_out = tau;
  return b;
}

void ranks(const uint8_t* role, uint64_t n, std::vector<uint64_t>& pre, std::vector<uint64_t>& dec) {
  pre.clear();
  dec.clear();
  for (uint64_t i = 0; i < n; ++i) (role[i] ? dec : pre).push_back(i);
}

// One decode's block cache as the simulator keeps it (Sec. VI-B: an LRU-managed KV-block
// cache): block hashes in recency order, most recent first, at most `cap` of them.
struct LruCache {
  std::list<uint64_t> order;  // most recent first
  std::unordered_map<uint64_t, std::list<uint64_t>::iterator> where;
  uint64_t cap = 0;

  bool contains(uint64_t h) const { return where.count(h) != 0; }
  // h becomes the most recently used block
  void touch(uint64_t h) {
    auto it = where.find(h);
    if (it != where.end()) {
      order.splice(order.begin(), order, it->second);
    } else {
      order.push_front(h);
      where[h] = order.begin();
    }
  }
  // drop least recently used blocks until at most cap remain
  void evict() {
    while (order.size() > cap) {
      where.erase(order.back());
      order.pop_back();
    }
  }
  // a request's chain enters the cache: its blocks are used from the last to the first,
  // so that block 0 ends up the most recent and a cached prefix loses its tail first
  void use_chain(const uint64_t* h, uint64_t n) {
    for (uint64_t j = n; j-- > 0;) touch(h[j]);
    evict();
  }
};

}  // namespace

extern "C" {

// OpenMP threads of the calling thread's later parallel regions (timing only: results do
// not depend on it).
void oracle_set_threads(int n) { omp_set_num_threads(n > 0 ? n : 1); }

// ---------------------------------------------------------------- closed forms
// Eq. 1: bytes of KV cache per token, s_r / l_r.
double oracle_kv_bytes_per_token(uint32_t n_layers, uint32_t n_kv_heads, uint32_t d_head,
                                 uint32_t b_elem) {
  return 2.0 * n_layers * n_kv_heads * d_head * (double)b_elem;
}

// Eq. 4: per-tier effective bandwidth with the self-contention count.
double oracle_beff_tier(double B_tau, double c_tau, double n_inflight) {
  return B_tau * (1.0 - c_tau) / (1.0 + n_inflight);
}

// Eq. 3: transfer time of s bytes.
double oracle_transfer_time(double s, double B_eff, double L_tau) { return s / B_eff + L_tau; }

// Eq. 2: effective transfer size after a lambda-token prefix hit.
double oracle_s_eff(double s_r, double lambda, double l_r) { return s_r * (1.0 - lambda / l_r); }

// ---------------------------------------------------------------- topology
int oracle_tier(const uint32_t* fanout, uint64_t i, uint64_t j) {
  return tier(make_tree(fanout), i, j);
}

// Links on the path between instances i and j (at most 8); returns the count.
int oracle_path_links(const uint32_t* fanout, uint64_t i, uint64_t j, uint64_t* links, int* levels) {
  const Tree t = make_tree(fanout);
  const int tau = tier(t, i, j);
  int n = 0;
  for (int h = 0; h <= tau; ++h) {
    links[n] = uplink(t, i, h); levels[n++] = h;
    links[n] = uplink(t, j, h); levels[n++] = h;
  }
  return n;
}

uint64_t oracle_used_links(const uint32_t* fanout) {
  const Tree t = make_tree(fanout);
  return t.n + t.n_node + t.n_leaf + t.n_pod;
}

// ---------------------------------------------------------------- oracle matrix
// C[s][p][d] = kv / Bbot(s,p,d) + L_tau(p,d), p over prefill ranks, d over decode
// ranks (ranks = role order), util [n_snap][n_links].
void oracle_cost_matrix(const uint32_t* fanout, const uint8_t* role, const double* bw,
                        const double* lat, const float* util, uint64_t n_links,
                        uint64_t n_snap, double kv_bytes, double* C) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, dec;
  ranks(role, t.n, pre, dec);
  const uint64_t P = pre.size(), D = dec.size();
#pragma omp parallel for collapse(2) schedule(static)
  for (uint64_t s = 0; s < n_snap; ++s)
    for (uint64_t p = 0; p < P; ++p)
      for (uint64_t d = 0; d < D; ++d) {
        int tau = 0;
        const double b = path_bottleneck(t, bw, util + s * n_links, pre[p], dec[d], &tau);
        C[(s * P + p) * D + d] = kv_bytes / b + lat[tau];
      }
}

// Selected entries (s[k], p[k], d[k]) of the same matrix; util rows indexed by s[k].
void oracle_cost_entries(const uint32_t* fanout, const uint8_t* role, const double* bw,
                         const double* lat, const float* util, uint64_t n_links,
                         const uint64_t* s, const uint64_t* p, const uint64_t* d, uint64_t n,
                         double kv_bytes, double* out) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, dec;
  ranks(role, t.n, pre, dec);
#pragma omp parallel for schedule(static)
  for (uint64_t k = 0; k < n; ++k) {
    int tau = 0;
    const double b = path_bottleneck(t, bw, util + s[k] * n_links, pre[p[k]], dec[d[k]], &tau);
    out[k] = kv_bytes / b + lat[tau];
  }
}

// Bottleneck of the up path from instance i to its height-(k+1) ancestor, for every
// instance and k = 0..3: UB[s][i][k] = min over h <= k of bw[h] * (1 - u[s][uplink(i,h)]).
void oracle_up_bottleneck(const uint32_t* fanout, const double* bw, const float* util,
                          uint64_t n_links, uint64_t n_snap, double* UB) {
  const Tree t = make_tree(fanout);
#pragma omp parallel for collapse(2) schedule(static)
  for (uint64_t s = 0; s < n_snap; ++s)
    for (uint64_t i = 0; i < t.n; ++i) {
      double b = std::numeric_limits<double>::infinity();
      for (int k = 0; k < 4; ++k) {
        const double r = bw[k] * (1.0 - (double)util[s * n_links + uplink(t, i, k)]);
        if (r < b) b = r;
        UB[(s * t.n + i) * 4 + k] = b;
      }
    }
}

// Directed links: the same matrix with transfers climbing the prefill's links at their
// upward utilisation util_up and descending the decode's at their downward utilisation
// util_down (both [n_snap][n_links]).
void oracle_cost_matrix_directed(const uint32_t* fanout, const uint8_t* role, const double* bw,
                                 const double* lat, const float* util_up, const float* util_down,
                                 uint64_t n_links, uint64_t n_snap, double kv_bytes, double* C) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, dec;
  ranks(role, t.n, pre, dec);
  const uint64_t P = pre.size(), D = dec.size();
#pragma omp parallel for collapse(2) schedule(static)
  for (uint64_t s = 0; s < n_snap; ++s)
    for (uint64_t p = 0; p < P; ++p)
      for (uint64_t d = 0; d < D; ++d) {
        int tau = 0;
        const double b = path_bottleneck_dir(t, bw, util_up + s * n_links, util_down + s * n_links,
                                             pre[p], dec[d], &tau);
        C[(s * P + p) * D + d] = kv_bytes / b + lat[tau];
      }
}

// Level bottlenecks with directed links: for a prefill instance the climb at upward
// utilisation, for a decode instance at downward utilisation (the direction a transfer
// crosses its links): UB[s][i][k] = min over h <= k of bw[h] * (1 - u_dir(i)[s][uplink(i,h)]).
void oracle_level_bottleneck_directed(const uint32_t* fanout, const uint8_t* role,
                                      const double* bw, const float* util_up,
                                      const float* util_down, uint64_t n_links, uint64_t n_snap,
                                      double* UB) {
  const Tree t = make_tree(fanout);
#pragma omp parallel for collapse(2) schedule(static)
  for (uint64_t s = 0; s < n_snap; ++s)
    for (uint64_t i = 0; i < t.n; ++i) {
      const float* u = (role[i] ? util_down : util_up) + s * n_links;
      double b = std::numeric_limits<double>::infinity();
      for (int k = 0; k < 4; ++k) {
        const double r = bw[k] * (1.0 - (double)u[uplink(t, i, k)]);
        if (r < b) b = r;
        UB[(s * t.n + i) * 4 + k] = b;
      }
    }
}

// Paper-literal per-tier oracle (Sec. III-E, Eq. 4 with n_inflight = 0): the four maps
// tier tau(p,d), bandwidth B_tau, congestion c_tau and latency L_tau, so that a pair's
// bandwidth is B_tau * (1 - c_tau) with no minimum over the lower levels of its path.
// c: [n_snap][4] per-tier congestion.
void oracle_cost_matrix_tiers(const uint32_t* fanout, const uint8_t* role, const double* bw,
                              const double* lat, const float* c, uint64_t n_snap,
                              double kv_bytes, double* C) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, dec;
  ranks(role, t.n, pre, dec);
  const uint64_t P = pre.size(), D = dec.size();
#pragma omp parallel for collapse(2) schedule(static)
  for (uint64_t s = 0; s < n_snap; ++s)
    for (uint64_t p = 0; p < P; ++p)
      for (uint64_t d = 0; d < D; ++d) {
        const int tau = tier(t, pre[p], dec[d]);
        const double b = bw[tau] * (1.0 - (double)c[s * 4 + tau]);
        C[(s * P + p) * D + d] = kv_bytes / b + lat[tau];
      }
}

// ---------------------------------------------------------------- prefix match
// M[r][d] = number of leading blocks of chain r found in cache K_{g(r),d}, where the
// cache of (set g, decode d) is the key list keys[key_off[g*D+d] .. key_off[g*D+d+1]),
// and set g serves requests [set_off[g], set_off[g+1]).  The scan stops at the first
// block that is not cached.
void oracle_prefix_match(const uint64_t* keys, const uint64_t* key_off, uint32_t D,
                         const uint64_t* chains, const uint64_t* chain_off, uint32_t R,
                         const uint32_t* set_off, uint32_t n_sets, uint16_t* M) {
  for (uint32_t g = 0; g < n_sets; ++g) {
    std::vector<std::unordered_set<uint64_t>> K(D);
    for (uint32_t d = 0; d < D; ++d) {
      const uint64_t t = (uint64_t)g * D + d;
      K[d].reserve(key_off[t + 1] - key_off[t]);
      for (uint64_t j = key_off[t]; j < key_off[t + 1]; ++j) K[d].insert(keys[j]);
    }
#pragma omp parallel for schedule(dynamic, 16)
    for (int64_t r = set_off[g]; r < (int64_t)set_off[g + 1]; ++r) {
      for (uint32_t d = 0; d < D; ++d) {
        uint64_t m = 0;
        for (uint64_t j = chain_off[r]; j < chain_off[r + 1]; ++j) {
          if (K[d].count(chains[j]) == 0) break;
          ++m;
        }
        M[(uint64_t)r * D + d] = (uint16_t)m;
      }
    }
  }
  (void)R;
}

// Prefix match of selected requests against ONE cache (key list), for sampled checks:
// out[k] = leading blocks of chain k (chains[chain_off[k]..chain_off[k+1])) found in keys.
void oracle_prefix_match_one(const uint64_t* keys, uint64_t n_keys, const uint64_t* chains,
                             const uint64_t* chain_off, uint64_t n, uint16_t* out) {
  std::unordered_set<uint64_t> K(keys, keys + n_keys);
  for (uint64_t k = 0; k < n; ++k) {
    uint64_t m = 0;
    for (uint64_t j = chain_off[k]; j < chain_off[k + 1]; ++j) {
      if (K.count(chains[j]) == 0) break;
      ++m;
    }
    out[k] = (uint16_t)m;
  }
}

// ---------------------------------------------------------------- greedy
// One stream of Algorithm 1 with the weighted score
//   score(d) = w_net * T_xfer(d) + w_prefix * miss(d) + w_load * theta * load[d],
//   T_xfer(d) = s_eff(d) / Bbot(k_r, p_r, d) + L_tau,  s_eff(d) = (l - 16 M[r][d]) * bpt,
//   miss(d)   = (l - 16 M[r][d]) / l,
// feasible iff load[d] + l <= cap.  Events are processed in order: a departure of a
// dispatched request releases its tokens; an arrival picks the feasible candidate of
// minimum score (lowest index among equal scores) or is rejected (-1), then adds its
// tokens to the chosen decode.
//
// hint (nullable): decisions of another implementation.  Where hint[r] differs from the
// oracle's choice, the step is a near-tie when hint[r] is feasible and its score is
// within rel_tol * best of the best score, and a mismatch otherwise; in both cases the
// oracle continues from hint[r] so that later steps are compared from the same state.
// counts[0] += near-ties, counts[1] += mismatches, counts[2] += rejects.
//
// best/second: the minimum score and the minimum over the other feasible candidates
// (+inf when absent), both from the oracle's own scores.
// util_down: NULL for undirected links, else the downward utilisation rows (util then
// holds the upward ones).  tier_mode: util holds per-tier congestion rows c[4] (n_links
// = 4) and a pair's bandwidth is B_tau * (1 - c_tau), the paper-literal oracle.
void oracle_schedule_stream(const uint32_t* fanout, const uint8_t* role, const double* bw,
                            const double* lat, const float* util, const float* util_down,
                            int tier_mode, uint64_t n_links,
                            const uint32_t* len, const uint32_t* prefill, const uint32_t* snap,
                            const uint16_t* M, const uint32_t* events, uint64_t n_events,
                            double w_net, double w_prefix, double w_load, double theta,
                            int64_t cap, uint64_t bytes_per_token, const int64_t* load_init,
                            const int32_t* hint, double rel_tol, int32_t* dec, double* best,
                            double* second, int64_t* load_out, int64_t* counts) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, decs;
  ranks(role, t.n, pre, decs);
  const uint64_t D = decs.size();
  std::vector<int64_t> load(D, 0);
  if (load_init)
    for (uint64_t d = 0; d < D; ++d) load[d] = load_init[d];
  std::vector<double> score(D);
  const double inf = std::numeric_limits<double>::infinity();

  for (uint64_t e = 0; e < n_events; ++e) {
    const uint32_t code = events[e];
    const uint32_t r = code & 0x7fffffffu;
    const int64_t l = len[r];
    if (code >> 31) {  // departure
      if (dec[r] >= 0) load[dec[r]] -= l;
      continue;
    }
    const float* u_row = util + (uint64_t)snap[r] * n_links;
    const float* d_row = util_down ? util_down + (uint64_t)snap[r] * n_links : u_row;
    const uint64_t p = pre[prefill[r]];
    int32_t arg = -1;
    for (uint64_t d = 0; d < D; ++d) {
      if (load[d] + l > cap) { score[d] = inf; continue; }
      int tau = 0;
      double b;
      if (tier_mode) {
        tau = tier(t, p, decs[d]);
        b = bw[tau] * (1.0 - (double)u_row[tau]);
      } else {
        b = path_bottleneck_dir(t, bw, u_row, d_row, p, decs[d], &tau);
      }
      const int64_t lam = 16 * (int64_t)M[(uint64_t)r * D + d];
      const double s_eff = (double)((l - lam) * (int64_t)bytes_per_token);
      const double T = s_eff / b + lat[tau];
      const double miss = (double)(l - lam) / (double)l;
      score[d] = w_net * T + w_prefix * miss + w_load * (theta * (double)load[d]);
      if (arg < 0 || score[d] < score[arg]) arg = (int32_t)d;
    }
    double b1 = inf, b2 = inf;
    if (arg >= 0) {
      b1 = score[arg];
      for (uint64_t d = 0; d < D; ++d)
        if ((int32_t)d != arg && score[d] < b2) b2 = score[d];
    }
    int32_t chosen = arg;
    if (hint && hint[r] != arg) {
      const int32_t h = hint[r];
      const bool near = (arg >= 0 && h >= 0 && (uint64_t)h < D && score[h] != inf &&
                         score[h] - b1 <= rel_tol * std::fabs(b1));
      counts[near ? 0 : 1] += 1;
      chosen = (h >= 0 && (uint64_t)h < D) ? h : -1;
    }
    if (chosen < 0) counts[2] += 1;
    dec[r] = chosen;
    best[r] = b1;
    second[r] = b2;
    if (chosen >= 0) load[chosen] += l;
  }
  for (uint64_t d = 0; d < D; ++d) load_out[d] = load[d];
}

// Algorithm 1 with self-contention.  As oracle_schedule_stream, plus:
//   arrival_us[r]  arrival time of request r in microseconds (events are in time order);
//   inflight_cap   the counter's maximum (0 turns self-contention off);
//   xfer_hint[r]   (nullable) another implementation's transfer time of r in whole
//                  microseconds: when it differs from this one's by at most one (the same
//                  transfer time rounded from a different precision), it is adopted so
//                  that both continue from the same completion time (counted);
//   xfer_us[r]     out: the chosen candidate's transfer time in whole microseconds,
//                  -1 when r is rejected.
// counts: near-ties, unexplained decisions, rejects, adopted transfer times, unexplained
// transfer times.
void oracle_schedule_stream_inflight(
    const uint32_t* fanout, const uint8_t* role, const double* bw, const double* lat,
    const float* util, uint64_t n_links, const uint32_t* len, const uint32_t* prefill,
    const uint32_t* snap, const int64_t* arrival_us, const uint16_t* M, const uint32_t* events,
    uint64_t n_events, double w_net, double w_prefix, double w_load, double theta, int64_t cap,
    uint64_t bytes_per_token, uint32_t inflight_cap, const int64_t* load_init,
    const int32_t* hint, const int32_t* xfer_hint, double rel_tol, int32_t* dec, double* best,
    double* second, int32_t* xfer_us, int64_t* load_out, int64_t* counts) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, decs;
  ranks(role, t.n, pre, decs);
  const uint64_t D = decs.size(), P = pre.size();
  std::vector<int64_t> load(D, 0);
  if (load_init)
    for (uint64_t d = 0; d < D; ++d) load[d] = load_init[d];
  std::vector<uint32_t> inflight(P * 4, 0);  // [prefill rank][tier]
  // pending completions: (time, prefill rank * 4 + tier), earliest first
  typedef std::pair<int64_t, uint64_t> Done;
  std::priority_queue<Done, std::vector<Done>, std::greater<Done>> pending;
  std::vector<double> score(D), xfer(D);
  const double inf = std::numeric_limits<double>::infinity();

  for (uint64_t e = 0; e < n_events; ++e) {
    const uint32_t code = events[e];
    const uint32_t r = code & 0x7fffffffu;
    const int64_t l = len[r];
    if (code >> 31) {  // departure
      if (dec[r] >= 0) load[dec[r]] -= l;
      continue;
    }
    const int64_t now = arrival_us[r];
    while (!pending.empty() && pending.top().first <= now) {  // transfers done by now
      uint32_t& n = inflight[pending.top().second];
      if (n > 0) n -= 1;
      pending.pop();
    }
    const float* u_row = util + (uint64_t)snap[r] * n_links;
    const uint64_t pr = prefill[r];
    const uint64_t p = pre[pr];
    int32_t arg = -1;
    for (uint64_t d = 0; d < D; ++d) {
      int tau = 0;
      const double b = path_bottleneck(t, bw, u_row, p, decs[d], &tau);
      const double b_eff = b / (1.0 + (double)inflight[pr * 4 + tau]);  // Eq. 4
      const int64_t lam = 16 * (int64_t)M[(uint64_t)r * D + d];
      const double s_eff = (double)((l - lam) * (int64_t)bytes_per_token);
      xfer[d] = s_eff / b_eff + lat[tau];
      if (load[d] + l > cap) { score[d] = inf; continue; }
      const double miss = (double)(l - lam) / (double)l;
      score[d] = w_net * xfer[d] + w_prefix * miss + w_load * (theta * (double)load[d]);
      if (arg < 0 || score[d] < score[arg]) arg = (int32_t)d;
    }
    double b1 = inf, b2 = inf;
    if (arg >= 0) {
      b1 = score[arg];
      for (uint64_t d = 0; d < D; ++d)
        if ((int32_t)d != arg && score[d] < b2) b2 = score[d];
    }
    int32_t chosen = arg;
    if (hint && hint[r] != arg) {
      const int32_t h = hint[r];
      const bool near = (arg >= 0 && h >= 0 && (uint64_t)h < D && score[h] != inf &&
                         score[h] - b1 <= rel_tol * std::fabs(b1));
      counts[near ? 0 : 1] += 1;
      chosen = (h >= 0 && (uint64_t)h < D) ? h : -1;
    }
    dec[r] = chosen;
    best[r] = b1;
    second[r] = b2;
    if (chosen < 0) {
      counts[2] += 1;
      xfer_us[r] = -1;
      continue;
    }
    load[chosen] += l;
    int64_t dt = std::llround(xfer[chosen] * 1e6);  // whole microseconds, half up
    if (xfer_hint && xfer_hint[r] != dt) {
      const int64_t diff = (int64_t)xfer_hint[r] - dt;
      const bool close = xfer_hint[r] >= 0 && diff >= -1 && diff <= 1;
      counts[close ? 3 : 4] += 1;
      if (close) dt = xfer_hint[r];
    }
    xfer_us[r] = (int32_t)dt;
    int tau = 0;
    path_bottleneck(t, bw, u_row, p, decs[chosen], &tau);
    uint32_t& n = inflight[pr * 4 + tau];  // Algorithm 1 line 14
    if (n < inflight_cap) n += 1;
    pending.push(Done(now + dt, pr * 4 + tau));
  }
  for (uint64_t d = 0; d < D; ++d) load_out[d] = load[d];
}

// Algorithm 1 with the paper's compute-load model (Sec. III-C decode state, Sec. IV-B
// component models, the feasible set of the objective in Sec. IV-A).  Decode d holds n[d]
// requests (dispatched, not departed) and m[d] bytes of free memory; with the batch
// beta = min(n, beta_max) and the queue q = n - beta,
//     T_queue  = max(0, q - (beta_max - beta)) * t_iter(beta),  T_decode = t_iter(beta + 1),
//     t_iter(beta) = t_a + t_b * beta,
//     score = w_net * T_xfer + w_prefix * miss + w_load * (T_queue + T_decode)
// over the feasible set m[d] >= s_eff(d) + m_min.  A dispatch to d* adds one request and
// takes s_eff(d*) bytes; its departure returns both.  m_init [D] (nullable: m0 each),
// n_init [D] (nullable: 0).  Outputs n_out, m_out [D].
void oracle_schedule_stream_load(
    const uint32_t* fanout, const uint8_t* role, const double* bw, const double* lat,
    const float* util, uint64_t n_links, const uint32_t* len, const uint32_t* prefill,
    const uint32_t* snap, const uint16_t* M, const uint32_t* events, uint64_t n_events,
    double w_net, double w_prefix, double w_load, uint64_t bytes_per_token, double t_a,
    double t_b, int64_t beta_max, int64_t m_min, int64_t m0, const int64_t* m_init,
    const int32_t* n_init, const int32_t* hint, double rel_tol, int32_t* dec, double* best,
    double* second, int32_t* n_out, int64_t* m_out, int64_t* counts) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, decs;
  ranks(role, t.n, pre, decs);
  const uint64_t D = decs.size();
  std::vector<int64_t> n(D, 0), m(D, m0);
  for (uint64_t d = 0; d < D; ++d) {
    if (n_init) n[d] = n_init[d];
    if (m_init) m[d] = m_init[d];
  }
  std::vector<double> score(D);
  const double inf = std::numeric_limits<double>::infinity();
  auto s_eff_of = [&](uint32_t r, uint64_t d) {
    const int64_t l = len[r];
    return (l - 16 * (int64_t)M[(uint64_t)r * D + d]) * (int64_t)bytes_per_token;
  };
  for (uint64_t e = 0; e < n_events; ++e) {
    const uint32_t code = events[e];
    const uint32_t r = code & 0x7fffffffu;
    if (code >> 31) {  // departure: the request leaves its decode and frees its bytes
      if (dec[r] >= 0) {
        n[dec[r]] -= 1;
        m[dec[r]] += s_eff_of(r, (uint64_t)dec[r]);
      }
      continue;
    }
    const int64_t l = len[r];
    const float* u_row = util + (uint64_t)snap[r] * n_links;
    const uint64_t p = pre[prefill[r]];
    int32_t arg = -1;
    for (uint64_t d = 0; d < D; ++d) {
      const int64_t s_eff = s_eff_of(r, d);
      if (m[d] < s_eff + m_min) { score[d] = inf; continue; }
      int tau = 0;
      const double b = path_bottleneck(t, bw, u_row, p, decs[d], &tau);
      const double T = (double)s_eff / b + lat[tau];
      const double miss = (double)(l - 16 * (int64_t)M[(uint64_t)r * D + d]) / (double)l;
      const int64_t beta = n[d] < beta_max ? n[d] : beta_max;
      const int64_t q = n[d] - beta;
      const int64_t blocked = q - (beta_max - beta);
      const double t_iter = t_a + t_b * (double)beta;
      const double t_queue = (blocked > 0 ? (double)blocked : 0.0) * t_iter;
      const double t_decode = t_a + t_b * (double)(beta + 1);
      score[d] = w_net * T + w_prefix * miss + w_load * (t_queue + t_decode);
      if (arg < 0 || score[d] < score[arg]) arg = (int32_t)d;
    }
    double b1 = inf, b2 = inf;
    if (arg >= 0) {
      b1 = score[arg];
      for (uint64_t d = 0; d < D; ++d)
        if ((int32_t)d != arg && score[d] < b2) b2 = score[d];
    }
    int32_t chosen = arg;
    if (hint && hint[r] != arg) {
      const int32_t h = hint[r];
      const bool near = (arg >= 0 && h >= 0 && (uint64_t)h < D && score[h] != inf &&
                         score[h] - b1 <= rel_tol * std::fabs(b1));
      counts[near ? 0 : 1] += 1;
      chosen = (h >= 0 && (uint64_t)h < D) ? h : -1;
    }
    if (chosen < 0) counts[2] += 1;
    dec[r] = chosen;
    best[r] = b1;
    second[r] = b2;
    if (chosen >= 0) {
      n[chosen] += 1;
      m[chosen] -= s_eff_of(r, (uint64_t)chosen);
    }
  }
  for (uint64_t d = 0; d < D; ++d) {
    n_out[d] = (int32_t)n[d];
    m_out[d] = m[d];
  }
}

// Algorithm 1 with evolving caches: the simulator's LRU-managed block cache of Sec. VI-B.
// A stream starts from its decodes' caches, given as key lists keys, key_off [D+1], each
// list from the most to the least recently used block.  Every arrival's prefix hits are
// taken against the caches as they are at that arrival (first-miss scan, Sec. III-B).  A
// dispatch to d* uses every block of the request's chain (chains, chain_off [R+1]) on
// K_{d*}: the blocks from the last to the first become the most recently used ones
// (present blocks are refreshed, absent ones inserted), then least recently used blocks
// are evicted until at most cap_blocks remain.  A list longer than cap_blocks is cut to
// its cap_blocks most recent blocks at the start.  Departures leave the caches as they
// are.  Scores, feasibility and load as oracle_schedule_stream.
//   M_out [R][D]: the hits each arrival was scored with.
//   cache_out (nullable) [D][cache_stride], cache_len [D]: each decode's cache after the
//   last event, most recent first (cache_stride >= cap_blocks when cache_out is given).
void oracle_schedule_stream_evolving(
    const uint32_t* fanout, const uint8_t* role, const double* bw, const double* lat,
    const float* util, uint64_t n_links, const uint32_t* len, const uint32_t* prefill,
    const uint32_t* snap, const uint64_t* keys, const uint64_t* key_off, uint64_t cap_blocks,
    const uint64_t* chains, const uint64_t* chain_off, const uint32_t* events,
    uint64_t n_events, double w_net, double w_prefix, double w_load, double theta, int64_t cap,
    uint64_t bytes_per_token, const int32_t* hint, double rel_tol, int32_t* dec, double* best,
    double* second, uint16_t* M_out, int64_t* load_out, int64_t* counts, uint64_t* cache_out,
    uint64_t cache_stride, uint64_t* cache_len) {
  const Tree t = make_tree(fanout);
  std::vector<uint64_t> pre, decs;
  ranks(role, t.n, pre, decs);
  const uint64_t D = decs.size();
  std::vector<LruCache> K(D);
  for (uint64_t d = 0; d < D; ++d) {
    K[d].cap = cap_blocks;
    K[d].use_chain(keys + key_off[d], key_off[d + 1] - key_off[d]);
  }
  std::vector<int64_t> load(D, 0);
  std::vector<double> score(D);
  const double inf = std::numeric_limits<double>::infinity();
  for (uint64_t e = 0; e < n_events; ++e) {
    const uint32_t code = events[e];
    const uint32_t r = code & 0x7fffffffu;
    const int64_t l = len[r];
    if (code >> 31) {
      if (dec[r] >= 0) load[dec[r]] -= l;
      continue;
    }
    for (uint64_t d = 0; d < D; ++d) {  // hits against the caches as they are now
      uint64_t m = 0;
      for (uint64_t j = chain_off[r]; j < chain_off[r + 1]; ++j) {
        if (!K[d].contains(chains[j])) break;
        ++m;
      }
      M_out[(uint64_t)r * D + d] = (uint16_t)m;
    }
    const float* u_row = util + (uint64_t)snap[r] * n_links;
    const uint64_t p = pre[prefill[r]];
    int32_t arg = -1;
    for (uint64_t d = 0; d < D; ++d) {
      if (load[d] + l > cap) { score[d] = inf; continue; }
      int tau = 0;
      const double b = path_bottleneck(t, bw, u_row, p, decs[d], &tau);
      const int64_t lam = 16 * (int64_t)M_out[(uint64_t)r * D + d];
      const double s_eff = (double)((l - lam) * (int64_t)bytes_per_token);
      const double T = s_eff / b + lat[tau];
      const double miss = (double)(l - lam) / (double)l;
      score[d] = w_net * T + w_prefix * miss + w_load * (theta * (double)load[d]);
      if (arg < 0 || score[d] < score[arg]) arg = (int32_t)d;
    }
    double b1 = inf, b2 = inf;
    if (arg >= 0) {
      b1 = score[arg];
      for (uint64_t d = 0; d < D; ++d)
        if ((int32_t)d != arg && score[d] < b2) b2 = score[d];
    }
    int32_t chosen = arg;
    if (hint && hint[r] != arg) {
      const int32_t h = hint[r];
      const bool near = (arg >= 0 && h >= 0 && (uint64_t)h < D && score[h] != inf &&
                         score[h] - b1 <= rel_tol * std::fabs(b1));
      counts[near ? 0 : 1] += 1;
      chosen = (h >= 0 && (uint64_t)h < D) ? h : -1;
    }
    if (chosen < 0) counts[2] += 1;
    dec[r] = chosen;
    best[r] = b1;
    second[r] = b2;
    if (chosen >= 0) {
      load[chosen] += l;
      K[chosen].use_chain(chains + chain_off[r], chain_off[r + 1] - chain_off[r]);
    }
  }
  for (uint64_t d = 0; d < D; ++d) {
    load_out[d] = load[d];
    if (cache_len) cache_len[d] = K[d].order.size();
    if (cache_out) {
      uint64_t i = 0;
      for (uint64_t h : K[d].order) cache_out[d * cache_stride + i++] = h;
    }
  }
}

}  // extern "C"
