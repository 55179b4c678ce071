// The greedy of Algorithm 1 (Sec. V-A) over independent scheduling streams.
//
// One CTA per stream walks that stream's events in order.  Each thread owns NPT
// consecutive decode ranks and keeps their load (active tokens) and instance links in
// registers, so the state of a stream never leaves the SM.  An arrival scores every
// candidate in parallel (the per-candidate work is the tier test, the bottleneck min of
// two level bottlenecks, one division for T_xfer and one for the missed fraction), then
// a (score, index) argmin that also carries the second-best score: a shuffle butterfly
// inside each warp and, for CTAs of several warps, one barrier and a second butterfly
// over the per-warp partials (double-buffered so one barrier per arrival suffices).
// Ties go to the lowest decode rank (line 13).  The decision is written by lane 0 of
// every warp, so a later departure event is resolved by the same lanes that wrote it.
// Events are software-pipelined (up to five events ahead) so that no global load sits
// on the per-event critical path (see the loop below).
// Without a workspace the network, prefix and load terms are combined on the fly from
// the level bottlenecks UB and the prefix hits M.  With a workspace, base_kernel first
// computes the decision-independent network + prefix term of every (arrival, decode)
// in parallel, and the greedy only adds the load term: the sequential part of a step
// shrinks to a load, a capacity test, one multiply-add and the argmin per candidate.
#include <math.h>

#include <type_traits>

#include "score.cuh"

namespace {

constexpr uint32_t kNone = 0xffffffffu;

__device__ __forceinline__ void combine(float& b, uint32_t& i, float& s, float b2, uint32_t i2,
                                        float s2) {
  const bool other = (b2 < b) || (b2 == b && i2 < i);
  if (other) {
    s = fminf(s2, b);
    b = b2;
    i = i2;
  } else {
    s = fminf(s, b2);
  }
}

// (score, index, second) argmin over the lanes of one segment of LPS lanes.
template <int LPS>
__device__ __forceinline__ void seg_argmin(float& b, uint32_t& i, float& s, uint32_t mask) {
#pragma unroll
  for (int o = LPS / 2; o; o >>= 1) {
    const float b2 = __shfl_xor_sync(mask, b, o, LPS);
    const uint32_t i2 = __shfl_xor_sync(mask, i, o, LPS);
    const float s2 = __shfl_xor_sync(mask, s, o, LPS);
    combine(b, i, s, b2, i2, s2);
  }
}

// Order-preserving 32-bit keys of fp32 scores, so that warp-wide redux minima give the
// (score, rank) argmin; kNoKey (above every float's key) stands for "no candidate".
constexpr uint32_t kNoKey = 0xffffffffu;
__device__ __forceinline__ uint32_t score_key(float x) {
  const uint32_t u = __float_as_uint(__fadd_rn(x, 0.0f));  // -0 and +0 tie, as compared
  return u ^ ((uint32_t)((int32_t)u >> 31) | 0x80000000u);
}
__device__ __forceinline__ float key_score(uint32_t k) {
  if (k == kNoKey) return __int_as_float(0x7f800000);
  return __uint_as_float(k ^ ((k >> 31) ? 0x80000000u : 0xffffffffu));
}
// Block-free argmin over the 32 lanes of a warp: (best key, its lowest rank, second key),
// where a lane offers (key, rank, key of its own runner-up).
__device__ __forceinline__ void warp_argmin_keys(uint32_t& key, uint32_t& rank, uint32_t& key2) {
  const uint32_t bk = __reduce_min_sync(0xffffffffu, key);
  const uint32_t br = __reduce_min_sync(0xffffffffu, key == bk ? rank : kNone);
  // the winning lane offers its runner-up; every other lane its best
  const uint32_t sk = __reduce_min_sync(0xffffffffu, (key == bk && rank == br) ? key2 : key);
  key = bk;
  rank = br;
  key2 = sk;
}

// The paper's compute-load model (Sec. III-C, IV-B) as kernel parameters.
struct LoadModel {
  float t_a, t_b;      // t_iter(beta) = t_a + t_b * beta
  int32_t beta_max;
  int64_t m_min, m0;
};

// Self-contention (Eq. 4's n_inflight, Algorithm 1 lines 5 and 14, Sec. V-C): the
// candidate's bandwidth is divided by 1 + n; T is returned for the completion time.
__device__ __forceinline__ float contended_score(const netkv_weights& w, uint32_t l, uint32_t m,
                                                 float ub_p, float ub_d, float lat_tau,
                                                 uint32_t n, float& T, int* status) {
  uint32_t lam = 16u * m;
  if (m > l / 16u) {
    flag_status(status, NETKV_DEV_EDOMAIN);
    lam = lam < l ? lam : l;
  }
  const uint32_t miss_tok = l - lam;
  const float bb = fminf(ub_p, ub_d);
  const float b_eff = n ? bb / (float)(1u + n) : bb;
  const float s_eff = (float)((int64_t)miss_tok * (int64_t)w.bytes_per_token);
  T = s_eff / b_eff + lat_tau;
  const float miss = (float)miss_tok / (float)l;
  return w.w_net * T + w.w_prefix * miss;
}

// combine() carrying the winner's transfer time along
__device__ __forceinline__ void combine_t(float& b, uint32_t& i, float& s, float& tt, float b2,
                                          uint32_t i2, float s2, float t2) {
  const bool other = (b2 < b) || (b2 == b && i2 < i);
  if (other) {
    s = fminf(s2, b);
    b = b2;
    i = i2;
    tt = t2;
  } else {
    s = fminf(s, b2);
  }
}
template <int LPS>
__device__ __forceinline__ void seg_argmin_t(float& b, uint32_t& i, float& s, float& tt,
                                             uint32_t mask) {
#pragma unroll
  for (int o = LPS / 2; o; o >>= 1) {
    const float b2 = __shfl_xor_sync(mask, b, o, LPS);
    const uint32_t i2 = __shfl_xor_sync(mask, i, o, LPS);
    const float s2 = __shfl_xor_sync(mask, s, o, LPS);
    const float t2 = __shfl_xor_sync(mask, tt, o, LPS);
    combine_t(b, i, s, tt, b2, i2, s2, t2);
  }
}

// Pending transfer completions of one stream: a binary min-heap in shared memory kept by
// the stream's lead thread, keys (completion time in us << 16) | (prefill rank << 2) | tier.
struct DoneHeap {
  unsigned long long* a;
  uint32_t n, cap;
  __device__ bool push(unsigned long long k) {
    if (n == cap) return false;
    uint32_t i = n++;
    while (i > 0) {
      const uint32_t p = (i - 1) >> 1;
      if (a[p] <= k) break;
      a[i] = a[p];
      i = p;
    }
    a[i] = k;
    return true;
  }
  __device__ void pop() {
    const unsigned long long k = a[--n];
    if (n == 0) return;
    uint32_t i = 0;
    for (;;) {
      uint32_t c = 2 * i + 1;
      if (c >= n) break;
      if (c + 1 < n && a[c + 1] < a[c]) ++c;
      if (a[c] >= k) break;
      a[i] = a[c];
      i = c;
    }
    a[i] = k;
  }
};

// s_eff / Bbot, the factor self-contention multiplies by 1 + n (Eq. 4): written beside
// the base scores when the greedy runs with self-contention.
__device__ __forceinline__ float xfer_factor(const netkv_weights& w, uint32_t l, uint32_t m,
                                             float ub_p, float ub_d) {
  const uint32_t lam = min(16u * m, l);
  const float s_eff = (float)((int64_t)(l - lam) * (int64_t)w.bytes_per_token);
  return s_eff / fminf(ub_p, ub_d);
}

// Base scores of every arrival (pools of at most 32 decodes): the events of a stream are
// split into contiguous ranges over the segments (LPS lanes each) of grid.y blocks, and
// lane sl of a segment owns decode sl.  As in base_wide_kernel, a lane keeps its decode's
// quotients bytes_per_token / UB_d[k] for the current snapshot and each arrival divides
// once per level for its prefill and once for 1 / l:
//     base = w_net * (miss_tok * max(qp[tau], qd[tau]) + L_tau) + w_prefix * miss_tok * (1/l)
// Departures and invalid events are skipped (the greedy reports them).  kUtil: `UB` holds
// the utilisation rows [n_snap][n_links] instead of the level bottlenecks, and the
// bottlenecks are taken from the links' entries.  X (self-contention) gets s_eff / Bbot.
template <int LPS, bool kUtil = false>
__global__ void __launch_bounds__(256, 6) base_kernel(
    TopoArgs t, uint32_t n_streams, const netkv_weights* __restrict__ W, uint32_t R,
    const uint32_t* __restrict__ len, const uint32_t* __restrict__ prefill,
    const uint32_t* __restrict__ snap, const uint16_t* __restrict__ M,
    const float* __restrict__ UB, uint32_t n_snap, const uint32_t* __restrict__ events,
    const uint64_t* __restrict__ event_off, float* __restrict__ base, int* status,
    float* __restrict__ X = nullptr) {
  constexpr uint32_t kSegs = 256 / LPS;
  constexpr uint32_t kNone = 0xffffffffu;  // no event (a departure code: skipped)
  const uint32_t seg = threadIdx.x / LPS, sl = threadIdx.x % LPS;
  const uint32_t D = t.D, N = t.N;
  const bool mine = sl < D;  // D <= LPS: lane sl owns decode sl
  const float4 lat = make_float4(t.lat[0], t.lat[1], t.lat[2], t.lat[3]);
  const uint32_t inst = mine ? __ldg(t.dec + sl) : 0u;
  const uint4 ld = __ldg(t.links + inst);
  // an arrival's length, prefill rank, snapshot and this lane's prefix hit
  auto fields = [&](uint32_t code, uint32_t& l, uint32_t& pr, uint32_t& k, uint32_t& m) {
    const uint32_t r = code & 0x7fffffffu;
    l = pr = k = m = 0u;
    if (!(code >> 31) && r < R) {
      l = __ldg(len + r);
      pr = __ldg(prefill + r);
      k = __ldg(snap + r);
      if (mine) m = __ldg(M + (uint64_t)r * D + sl);
    }
  };
  for (uint32_t stream = blockIdx.x; stream < n_streams; stream += gridDim.x) {
    const float w_net = W[stream].w_net, w_prefix = W[stream].w_prefix;
    const float bpt = (float)W[stream].bytes_per_token;
    // each segment takes a contiguous range of the stream's events, so consecutive
    // arrivals share their snapshot
    const uint64_t e0 = event_off[stream], e1 = event_off[stream + 1];
    const uint64_t n_seg = (uint64_t)gridDim.y * kSegs;
    const uint64_t span = (e1 - e0 + n_seg - 1) / n_seg;
    const uint64_t eb = e0 + ((uint64_t)blockIdx.y * kSegs + seg) * span;
    const uint64_t ee = min(e1, eb + span);
    uint32_t cur_k = 0xffffffffu;
    float4 qd = make_float4(0.f, 0.f, 0.f, 0.f);
    // software pipeline: the next event's fields and the code after it are loaded while
    // the current arrival is scored, so an arrival waits for one round trip (its
    // utilisation entries) instead of three
    uint32_t c_next = eb + 1 < ee ? __ldg(events + eb + 1) : kNone;
    uint32_t code_n = eb < ee ? __ldg(events + eb) : kNone;
    uint32_t l_n, pr_n, k_n, m_n;
    fields(code_n, l_n, pr_n, k_n, m_n);
    for (uint64_t e = eb; e < ee; ++e) {
      const uint32_t code = code_n, l = l_n, pr = pr_n, k = k_n, m = m_n;
      code_n = c_next;
      c_next = e + 2 < ee ? __ldg(events + e + 2) : kNone;
      fields(code_n, l_n, pr_n, k_n, m_n);
      const uint32_t r = code & 0x7fffffffu;
      if ((code >> 31) || r >= R) continue;
      if (pr >= t.P || k >= n_snap || l == 0 || !mine) continue;
      if (k != cur_k) {  // the decode's level bottlenecks of a new snapshot
        cur_k = k;
        const float4 ub = kUtil ? level_bottlenecks_of(t, UB + (uint64_t)k * t.n_links, ld, status)
                                : __ldg(reinterpret_cast<const float4*>(UB) + (uint64_t)k * N + inst);
        qd = make_float4(bpt / ub.x, bpt / ub.y, bpt / ub.z, bpt / ub.w);
      }
      const uint32_t pinst = __ldg(t.pre + pr);
      const uint4 lp = __ldg(t.links + pinst);
      const int tau = tier_of(lp, ld);
      const float ubp = kUtil ? pick4(level_bottlenecks_of(t, UB + (uint64_t)k * t.n_links, lp,
                                                           status), tau)
                              : __ldg(UB + ((uint64_t)k * N + pinst) * 4 + tau);
      uint32_t lam = 16u * m;
      if (m > l / 16u) {
        flag_status(status, NETKV_DEV_EDOMAIN);
        lam = lam < l ? lam : l;
      }
      const float miss_tok = (float)(l - lam);
      const float q = fmaxf(bpt / ubp, pick4(qd, tau));
      const float T = __fmaf_rn(miss_tok, q, pick4(lat, tau));
      base[(uint64_t)r * D + sl] = __fmaf_rn(w_net, T, w_prefix * (miss_tok * (1.0f / (float)l)));
      if (X) X[(uint64_t)r * D + sl] = miss_tok * q;
    }
  }
}

// ---- candidate lists: a bound on every decode a walk need not rescore ----------------
// The load term of a score is w_load * theta * load >= 0, so a decode's score is never below
// its base score, and the fp32 score fma(w_load, theta * load, base) is monotone in both the
// load and the base.  For each arrival the base pass lists the pool's kListLen smallest
// (base, rank) pairs in that order and a bound (tau, tau_rank): every decode not listed has
// (base, rank) >= (tau, tau_rank).  A walk that knows a lower bound
// L on every decode's current load then has, for every unlisted decode d,
//     score(d) >= fma(w_load, theta * L, base(d)) >= fma(w_load, theta * L, tau) =: LB,
// so the best listed (score, rank) is the argmin of all decodes when its score is below LB, or
// equal to tau with a rank below tau_rank (with L >= 0, an unlisted decode scores at least its
// base); the second-best listed score is the second-best of all when it is <= LB.  Otherwise
// the walk rescans the arrival's full row.  The result is the full argmin in every case.
//
// Bound keys: score_key(tau), or kNoKey when every decode of the pool is listed, or
// kBoundInvalid (below every float's key) when the list cannot bound anything (a NaN score).
constexpr int kListLen = 32;             // (rank, base) pairs listed per arrival: one a lane
constexpr uint32_t kListChunk = 1024;    // decodes per base-pass block (256 threads, 4 each)
constexpr uint32_t kListMinD = 1025;     // listed pools: 1,025 .. 4,096 decodes, whose
constexpr uint32_t kListMaxD = 4096;     // 2 .. 4 chunk lists are merged into the pool's
// The list arrays of a workspace (all null: the staged walk runs).
struct ListWs {
  uint2 *chunk_lists = nullptr, *chunk_bounds = nullptr, *lists = nullptr, *bounds = nullptr;
};
constexpr int kListLevels = 8;           // distinct base scores a block walks up per arrival
constexpr uint32_t kBoundInvalid = 0u;

// Per-level exchange of a block's NW <= 32 warps, double-buffered by barrier phase.
template <int NW>
struct ListShared {
  uint32_t cnt[2][NW];  // pairs of the warp at the current key
  uint32_t nxt[2][NW];  // the warp's smallest key above it
};

// The pool's list and bound for one arrival, by the whole block: walking up the distinct
// keys of the pool (at most kListLevels of them), the pairs of each key are listed in rank
// order until kListLen are listed; the next pair is the bound.  Every warp first finds its
// smallest key and how many of its pairs hold it, so that after one block barrier the
// pool's smallest key and its pairs are placed: when there are more than kListLen of them
// (ties, the common case) that barrier is the only one.  Each further level costs one
// barrier: every warp counts its pairs at the key and finds its smallest key above it, and
// after the barrier each thread places its own pairs by the counts of the warps before it.
// When the levels run out first, the bound is (next key, rank 0) or, with no key left, the
// pool is listed entirely (kNoKey).  k: the thread's NPT = 4 keys (kNoKey past D) of
// decodes d0 .. d0 + 3 (lane-major within a warp, warps in rank order).  `phase` counts the
// block's barrier phases (uniform).  NaN scores make the bound kBoundInvalid.
template <int NW>
__device__ __forceinline__ void block_levels(ListShared<NW>& S, uint32_t& phase, const uint32_t (&k)[4],
                                             bool nan, uint32_t d0, uint2* __restrict__ out,
                                             uint2* __restrict__ bound) {
  const uint32_t tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const uint32_t below = (1u << lane) - 1u;
  // pairs of this thread at key v placed from position base_pos (in rank order)
  auto place = [&](uint32_t v, uint32_t base_pos) {
    uint32_t pos = base_pos;
#pragma unroll
    for (int j = 0; j < 4; ++j) pos += __popc(__ballot_sync(0xffffffffu, k[j] == v) & below);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      if (k[j] == v) {
        if (pos < (uint32_t)kListLen)
          out[pos] = make_uint2(d0 + j, __float_as_uint(key_score(v)));
        else if (pos == (uint32_t)kListLen)
          *bound = make_uint2(d0 + j, v);
        ++pos;
      }
    }
  };
  // level 0: each warp's smallest key, its pairs at that key, and whether a score is NaN
  {
    const uint32_t m = __reduce_min_sync(0xffffffffu, min(min(k[0], k[1]), min(k[2], k[3])));
    uint32_t c = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) c += __popc(__ballot_sync(0xffffffffu, k[j] == m));
    const bool bad = __any_sync(0xffffffffu, nan);
    if (lane == 0) {
      S.nxt[phase & 1][wid] = m;
      S.cnt[phase & 1][wid] = c | (bad ? 0x80000000u : 0u);
    }
  }
  __syncthreads();
  uint32_t v, cum;
  {
    const uint32_t b = phase & 1;
    const uint32_t mw = lane < (uint32_t)NW ? S.nxt[b][lane] : kNoKey;
    const uint32_t cw = lane < (uint32_t)NW ? S.cnt[b][lane] : 0u;
    ++phase;
    if (__reduce_or_sync(0xffffffffu, cw & 0x80000000u)) {
      if (tid < (uint32_t)kListLen) out[tid] = make_uint2(kNone, 0x7f800000u);
      if (tid == 0) *bound = make_uint2(0u, kBoundInvalid);
      return;
    }
    v = __reduce_min_sync(0xffffffffu, mw);
    if (v == kNoKey) {  // no decode at all
      if (tid < (uint32_t)kListLen) out[tid] = make_uint2(kNone, 0x7f800000u);
      if (tid == 0) *bound = make_uint2(kNone, kNoKey);
      return;
    }
    const uint32_t c = mw == v ? cw : 0u;  // a warp whose smallest key is above v has none at v
    const uint32_t off = __reduce_add_sync(0xffffffffu, lane < wid ? c : 0u);
    cum = __reduce_add_sync(0xffffffffu, c);
    place(v, off);
  }
  for (int lev = 1; lev < kListLevels && cum <= (uint32_t)kListLen; ++lev) {
    // each warp's smallest key above v and its pairs at that key, as at level 0
    const uint32_t b = phase & 1;
    uint32_t m = kNoKey;
#pragma unroll
    for (int j = 0; j < 4; ++j) m = min(m, k[j] > v ? k[j] : kNoKey);
    m = __reduce_min_sync(0xffffffffu, m);
    uint32_t c = 0;
#pragma unroll
    for (int j = 0; j < 4; ++j) c += __popc(__ballot_sync(0xffffffffu, k[j] == m));
    if (lane == 0) {
      S.nxt[b][wid] = m;
      S.cnt[b][wid] = c;
    }
    __syncthreads();
    const uint32_t mw = lane < (uint32_t)NW ? S.nxt[b][lane] : kNoKey;
    const uint32_t cw = lane < (uint32_t)NW ? S.cnt[b][lane] : 0u;
    ++phase;
    v = __reduce_min_sync(0xffffffffu, mw);
    if (v == kNoKey) break;  // every pair is listed
    const uint32_t cv = mw == v ? cw : 0u;
    const uint32_t off = __reduce_add_sync(0xffffffffu, lane < wid ? cv : 0u);
    const uint32_t total = __reduce_add_sync(0xffffffffu, cv);
    place(v, cum + off);
    cum += total;
  }
  if (cum <= (uint32_t)kListLen) {  // as many pairs as the list holds, or fewer
    if (tid >= cum && tid < (uint32_t)kListLen) out[tid] = make_uint2(kNone, 0x7f800000u);
    if (tid == 0) {
      if (v == kNoKey) {
        *bound = make_uint2(kNone, kNoKey);
      } else {  // the levels ran out: every pair not listed has a key above v
        *bound = make_uint2(0u, v + 1u);
      }
    }
  }
}

// The pool's list and bound from its chunks' (one warp per request).  Every chunk list is
// sorted by (key, rank); in 64-bit form (key << 32 | rank) a chunk's list is its real pairs,
// then all ones.  With B the smallest chunk bound, a pair x < B is the pool's
// p-th smallest, p = the number of pairs below x in every chunk list (its own position in its
// own list, a binary search by shuffles in the others'), and is listed when p < kListLen;
// the pool's bound is the pair with p == kListLen if there is one, else B.  Requests whose
// arrival the base pass skipped merge whatever their slots hold; the walk never reads them.
__device__ __forceinline__ unsigned long long list_pair(uint2 e) {  // (rank, base bits)
  return e.x == kNone ? ~0ull
                      : ((unsigned long long)score_key(__uint_as_float(e.y)) << 32) | e.x;
}
__global__ void __launch_bounds__(256) merge_lists_kernel(
    const uint2* __restrict__ chunk_lists, const uint2* __restrict__ chunk_bounds, uint32_t n_ch,
    uint32_t R, uint2* __restrict__ lists, uint2* __restrict__ bounds) {
  constexpr uint32_t kMaxCh = kListMaxD / kListChunk;
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  for (uint64_t r = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; r < R; r += n_warps) {
    unsigned long long x[kMaxCh], bd[kMaxCh];
    uint32_t xb[kMaxCh];
    unsigned long long B = ~0ull;
#pragma unroll
    for (uint32_t c = 0; c < kMaxCh; ++c) {
      x[c] = bd[c] = ~0ull;
      xb[c] = 0x7f800000u;
      if (c < n_ch) {
        const uint2 e = __ldcs(chunk_lists + ((r * n_ch + c) * kListLen + lane));
        const uint2 b = chunk_bounds[r * n_ch + c];
        x[c] = list_pair(e);
        xb[c] = e.y;
        bd[c] = ((unsigned long long)b.y << 32) | b.x;
        B = min(B, bd[c]);
      }
    }
    uint2 mine = make_uint2(kNone, 0x7f800000u);
    bool has_bound = false;  // some pair is the (kListLen + 1)-th below B
    unsigned long long pb = 0;
#pragma unroll
    for (uint32_t c = 0; c < kMaxCh; ++c) {
      const unsigned long long v = x[c];
      uint32_t p = lane;  // pairs below v in its own list
#pragma unroll
      for (uint32_t o = 0; o < kMaxCh; ++o) {
        if (o == c || o >= n_ch) continue;
        uint32_t lo = 0;  // pairs of list o below v, by binary search over its 32 lanes
#pragma unroll
        for (uint32_t step = 16; step; step >>= 1) {
          const unsigned long long u = __shfl_sync(0xffffffffu, x[o], lo + step - 1);
          if (u < v) lo += step;
        }
        const unsigned long long u31 = __shfl_sync(0xffffffffu, x[o], 31);
        if (lo == 31 && u31 < v) lo = 32;  // every pair of list o is below v
        p += lo;
      }
      const bool real = c < n_ch && v < B && (uint32_t)(v & 0xffffffffu) != kNone;
      // the real pair at lane `lane` sits at pool position p: list it or make it the bound
      if (real && p < (uint32_t)kListLen) {
        lists[r * kListLen + p] = make_uint2((uint32_t)v, xb[c]);
      }
      const bool is_b = real && p == (uint32_t)kListLen;
      if (__any_sync(0xffffffffu, is_b)) {
        const uint32_t src = __ffs(__ballot_sync(0xffffffffu, is_b)) - 1;
        pb = __shfl_sync(0xffffffffu, v, src);
        has_bound = true;
      }
    }
    // how many pairs were listed: positions beyond them are empty
    uint32_t n_listed = 0;
#pragma unroll
    for (uint32_t c = 0; c < kMaxCh; ++c)
      n_listed += __popc(__ballot_sync(0xffffffffu, c < n_ch && x[c] < B &&
                                                         (uint32_t)(x[c] & 0xffffffffu) != kNone));
    if (lane >= n_listed) lists[r * kListLen + lane] = mine;
    if (lane == 0) {
      const unsigned long long b = has_bound ? pb : B;
      bounds[r] = make_uint2((uint32_t)b, (uint32_t)(b >> 32));
    }
  }
}

// Base scores for pools of more than 32 decodes.  A block takes one chunk of 256 * NPT
// decodes of one stream and a contiguous range of its events; each thread owns NPT
// consecutive decodes.  Arrivals in a range mostly share their telemetry snapshot, so a
// thread keeps, for its decodes and the current snapshot, the quotients
// qd[k] = bytes_per_token / UB_d[k] of every level k, and recomputes them only when the
// snapshot changes; per arrival it divides once per level for the prefill,
// qp[k] = bytes_per_token / UB_p[k], and once for 1 / l.  Division of positive operands is
// monotone, so bytes_per_token / min(UB_p, UB_d) = max(qp, qd) exactly, and a candidate
// costs a tier test, a max and three multiply-adds:
//     base = w_net * (miss_tok * max(qp[tau], qd[tau]) + L_tau) + w_prefix * miss_tok * (1/l)
// (two roundings more than dividing per candidate: a relative difference below 3e-7).
// The next arrival's request fields and prefix hits are loaded one arrival ahead; hits are
// read 8 bytes and scores written 16 bytes at a time when the rows allow it.
// kUtil: as for base_kernel (UB holds the utilisation rows).  X (self-contention) keeps
// the per-candidate division s_eff / Bbot.
// kList: the block also writes each arrival's candidate list and bound for its chunk of
// decodes (lists[r][chunk][kListLen], bounds[r][chunk]) with block_levels; merge_lists_kernel
// then merges the chunks' lists into the pool's.
template <int NPT, bool kUtil = false, bool kList = false, int BT = 256>
__global__ void __launch_bounds__(BT, 1024 / BT) base_wide_kernel(
    TopoArgs t, uint32_t n_streams, const netkv_weights* __restrict__ W, uint32_t R,
    const uint32_t* __restrict__ len, const uint32_t* __restrict__ prefill,
    const uint32_t* __restrict__ snap, const uint16_t* __restrict__ M,
    const float* __restrict__ UB, uint32_t n_snap, const uint32_t* __restrict__ events,
    const uint64_t* __restrict__ event_off, float* __restrict__ base, int* status,
    float* __restrict__ X = nullptr, uint2* __restrict__ lists = nullptr,
    uint2* __restrict__ bounds = nullptr) {
  static_assert(!kList || NPT == 4, "lists take 4 decodes a thread");
  static_assert(BT % 32 == 0 && BT <= 1024, "block of whole warps");
  __shared__ std::conditional_t<kList, ListShared<BT / 32>, char> S;
  uint32_t phase = 0;  // block barrier phases of the list selection (buffer parity)
  constexpr uint32_t kChunk = (uint32_t)BT * NPT;
  constexpr uint32_t kBad = 0xffffffffu;
  const uint32_t D = t.D, N = t.N;
  const uint32_t n_chunks = (D + kChunk - 1) / kChunk;
  const bool vec = NPT == 4 && (D % 4u == 0) && ((reinterpret_cast<uintptr_t>(M) & 7u) == 0) &&
                   ((reinterpret_cast<uintptr_t>(base) & 15u) == 0);
  const float4 lat = make_float4(t.lat[0], t.lat[1], t.lat[2], t.lat[3]);
  for (uint64_t sc = blockIdx.x; sc < (uint64_t)n_streams * n_chunks; sc += gridDim.x) {
    const uint32_t stream = (uint32_t)(sc / n_chunks);
    const uint32_t d0 = (uint32_t)(sc % n_chunks) * kChunk + threadIdx.x * NPT;
    uint3 lt[NPT];     // level-1..3 links of each decode: its tier against a prefill
    uint32_t inst[NPT];
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      inst[j] = d0 + j < D ? __ldg(t.dec + d0 + j) : 0u;
      const uint4 l = __ldg(t.links + inst[j]);
      lt[j] = make_uint3(l.y, l.z, l.w);
    }
    const netkv_weights w = W[stream];
    const float bpt = (float)w.bytes_per_token;
    // a contiguous range of the stream's events
    const uint64_t e0 = event_off[stream], e1 = event_off[stream + 1];
    const uint64_t span = (e1 - e0 + gridDim.y - 1) / gridDim.y;
    const uint64_t eb = e0 + blockIdx.y * span;
    const uint64_t ee = min(e1, eb + span);

    // request fields of an event: kBad r for departures and events to skip
    auto fields = [&](uint64_t e, uint32_t& r, uint32_t& l, uint32_t& pr, uint32_t& k,
                      uint32_t* m) {
      r = kBad;
      if (e >= ee) return;
      const uint32_t code = __ldg(events + e);
      const uint32_t rr = code & 0x7fffffffu;
      if ((code >> 31) || rr >= R) return;
      l = __ldg(len + rr);
      pr = __ldg(prefill + rr);
      k = __ldg(snap + rr);
      if (pr >= t.P || k >= n_snap || l == 0) return;
      r = rr;
      const uint16_t* mrow = M + (uint64_t)rr * D + d0;
      if (vec) {
        if (d0 < D) {
          const uint2 v = __ldcs(reinterpret_cast<const uint2*>(mrow));
          m[0] = v.x & 0xffffu;
          m[1] = v.x >> 16;
          m[2] = v.y & 0xffffu;
          m[3] = v.y >> 16;
        }
      } else {
#pragma unroll
        for (int j = 0; j < NPT; ++j) m[j] = d0 + j < D ? (uint32_t)__ldcs(mrow + j) : 0u;
      }
    };

    float4 qd[NPT];  // bytes_per_token / UB_d[k] of the current snapshot
    uint32_t cur_k = kBad;
    uint32_t nr, nl = 0, npr = 0, nk = 0, nm[NPT];
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      nm[j] = 0;
      qd[j] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    uint64_t e = eb;
    fields(e, nr, nl, npr, nk, nm);
    for (; e < ee; ++e) {
      const uint32_t r = nr, l = nl, pr = npr, k = nk;
      uint32_t m[NPT];
#pragma unroll
      for (int j = 0; j < NPT; ++j) m[j] = nm[j];
      fields(e + 1, nr, nl, npr, nk, nm);
      if (r == kBad) continue;
      if (k != cur_k) {  // the decodes' level bottlenecks of a new snapshot
        cur_k = k;
        const float* urow = UB + (uint64_t)k * t.n_links;
#pragma unroll
        for (int j = 0; j < NPT; ++j) {
          if (d0 + j < D) {
            const float4 ub = kUtil
                ? level_bottlenecks_of(t, urow, __ldg(t.links + inst[j]), status)
                : __ldg(reinterpret_cast<const float4*>(UB) + (uint64_t)k * N + inst[j]);
            qd[j] = make_float4(bpt / ub.x, bpt / ub.y, bpt / ub.z, bpt / ub.w);
          }
        }
      }
      const uint32_t pinst = __ldg(t.pre + pr);
      const uint4 lp = __ldg(t.links + pinst);
      const float4 ubp = kUtil
          ? level_bottlenecks_of(t, UB + (uint64_t)k * t.n_links, lp, status)
          : __ldg(reinterpret_cast<const float4*>(UB) + (uint64_t)k * N + pinst);
      const float4 qp = make_float4(bpt / ubp.x, bpt / ubp.y, bpt / ubp.z, bpt / ubp.w);
      const float rl = 1.0f / (float)l;
      float out[NPT];
#pragma unroll
      for (int j = 0; j < NPT; ++j) {
        const int tau = (lp.y == lt[j].x) ? 0 : (lp.z == lt[j].y) ? 1 : (lp.w == lt[j].z) ? 2 : 3;
        uint32_t lam = 16u * m[j];
        if (m[j] > l / 16u) {
          flag_status(status, NETKV_DEV_EDOMAIN);
          lam = lam < l ? lam : l;
        }
        const float miss_tok = (float)(l - lam);
        const float q = fmaxf(pick4(qp, tau), pick4(qd[j], tau));
        const float T = __fmaf_rn(miss_tok, q, pick4(lat, tau));
        out[j] = __fmaf_rn(w.w_net, T, w.w_prefix * (miss_tok * rl));
        if (X && d0 + j < D) X[(uint64_t)r * D + d0 + j] = miss_tok * q;
      }
      float* brow = base + (uint64_t)r * D + d0;
      if (vec) {
        if (d0 < D) __stcs(reinterpret_cast<float4*>(brow), make_float4(out[0], out[1], out[2], out[3]));
      } else {
#pragma unroll
        for (int j = 0; j < NPT; ++j)
          if (d0 + j < D) __stcs(brow + j, out[j]);
      }
      if constexpr (kList) {
        uint32_t key[4];
        bool nan = false;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const bool present = d0 + j < D;
          key[j] = present ? score_key(out[j]) : kNoKey;
          nan |= present && !(out[j] == out[j]);
        }
        const uint64_t slot = (uint64_t)r * n_chunks + (uint32_t)(sc % n_chunks);
        block_levels(S, phase, key, nan, d0, lists + slot * kListLen, bounds + slot);
      }
    }
  }
}

// LPS = lanes per stream.  LPS == 32: one stream per CTA of BLOCK threads.  LPS < 32
// (BLOCK == 32, NPT == 1, D <= LPS): a warp runs 32 / LPS streams side by side, one per
// segment of LPS lanes, so that small decode pools still use every lane.
// Self-contention (kInfl): each stream keeps n_inflight[prefill][tier] as four 8-bit
// counters per prefill rank and its pending completions in a heap, both in dynamic
// shared memory (`infl_bytes` per stream: counters, then `heap_cap` heap keys).  The
// lead thread applies the completions due by an arrival's time before it is scored
// (one extra stream barrier per arrival), and after the decision raises the chosen
// tier's counter (saturating at `inflight_cap`), records the transfer time and pushes
// its completion.  The argmin carries the winner's transfer time along.
// Compute-load model (kLoad): load[j] holds decode j's free bytes and held[j] its request
// count; a candidate is feasible iff free >= s_eff + m_min, its load term is
// T_queue + T_decode from the count (beta = min(n, beta_max), q = n - beta), a dispatch
// takes s_eff bytes and one count and the departure returns them (its prefix hits come
// through the same pipeline as an arrival's).
template <int NPT, int BLOCK, int LPS, bool kBase, bool kInfl = false, bool kLoad = false>
__global__ void __launch_bounds__(BLOCK) schedule_kernel(
    TopoArgs t, uint32_t n_streams, const netkv_weights* __restrict__ W, uint32_t R,
    const float* __restrict__ base, const uint32_t* __restrict__ len,
    const uint32_t* __restrict__ prefill, const uint32_t* __restrict__ snap,
    const uint16_t* __restrict__ M, const float* __restrict__ UB, uint32_t n_snap,
    const uint32_t* __restrict__ events, const uint64_t* __restrict__ event_off,
    const int64_t* __restrict__ load_init, int32_t* dec, float* __restrict__ best,
    float* __restrict__ second, int64_t* __restrict__ load_final, int* status,
    const int64_t* __restrict__ arrival_us = nullptr, uint32_t inflight_cap = 0,
    int32_t* __restrict__ xfer_us = nullptr, uint32_t infl_bytes = 0, uint32_t heap_cap = 0,
    LoadModel lm = LoadModel{0.f, 0.f, 0, 0, 0}, const int32_t* __restrict__ n_init = nullptr,
    int32_t* __restrict__ n_final = nullptr, const float* __restrict__ xf = nullptr) {
  static_assert(LPS == 32 || (BLOCK == 32 && NPT == 1), "packed streams use one warp");
  static_assert(!(kLoad && (kBase || kInfl)), "the load model scores from UB and M alone");
  constexpr int NW = BLOCK / 32;
  __shared__ float s_b[2][NW];
  __shared__ uint32_t s_i[2][NW];
  __shared__ float s_s[2][NW];
  __shared__ float s_t[2][NW];
  const uint32_t lane_w = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const uint32_t seg = LPS == 32 ? 0u : lane_w / LPS;
  const uint32_t stream = LPS == 32 ? blockIdx.x : blockIdx.x * (32 / LPS) + seg;
  if (stream >= n_streams) return;  // whole segments only: never inside a CTA of LPS == 32
  const uint32_t smask = LPS == 32 ? 0xffffffffu : (((1u << LPS) - 1u) << (seg * LPS));
  const uint32_t tid = LPS == 32 ? threadIdx.x : lane_w % LPS;  // thread within the stream
  const uint32_t lane = LPS == 32 ? lane_w : tid;                // lane within the segment
  const bool lead_thread = tid == 0;
  const uint32_t D = t.D, N = t.N;
  const netkv_weights w = W[stream];
  const float4 lat = make_float4(t.lat[0], t.lat[1], t.lat[2], t.lat[3]);
  const float inf = __int_as_float(0x7f800000);

  int64_t load[NPT];
  int32_t held[NPT];  // compute-load model: requests held by the decode
  uint4 ld[NPT];  // links of the decode instance; .x is the instance index itself
#pragma unroll
  for (int j = 0; j < NPT; ++j) {
    const uint32_t d = tid * NPT + j;
    load[j] = kLoad ? lm.m0 : 0;
    held[j] = 0;
    ld[j] = make_uint4(0, 0, 0, 0);
    if (d < D) {
      ld[j] = __ldg(t.links + __ldg(t.dec + d));
      if (load_init) load[j] = load_init[(uint64_t)stream * D + d];
      if (kLoad && n_init) held[j] = n_init[(uint64_t)stream * D + d];
    }
  }

  const uint64_t e0 = event_off[stream], e1 = event_off[stream + 1];
  uint32_t parity = 0;

  uint32_t* cnt = nullptr;  // n_inflight: byte `tier` of cnt[prefill rank]
  DoneHeap heap = {nullptr, 0u, 0u};
  if constexpr (kInfl) {
    extern __shared__ __align__(16) unsigned char infl_smem[];
    unsigned char* mine = infl_smem + (size_t)(LPS == 32 ? 0u : seg) * infl_bytes;
    cnt = reinterpret_cast<uint32_t*>(mine);
    heap.a = reinterpret_cast<unsigned long long*>(mine + (size_t)((t.P * 4u + 15u) & ~15u));
    heap.cap = heap_cap;
    for (uint32_t i = tid; i < t.P; i += (LPS == 32 ? BLOCK : LPS)) cnt[i] = 0u;
    if (LPS == 32) __syncthreads(); else __syncwarp(smask);
  }

  // Software pipeline over events.  When event e is processed, its operands were
  // requested PD iterations earlier: event e+PD+1 gets its level bottlenecks (and, for a
  // departure, its decision) requested, event e+FD+1 its request fields and prefix hits,
  // event e+CD+1 its code; every global load is consumed at least one iteration after
  // it is issued, PD iterations for the level-bottleneck rows that come from DRAM.  The
  // topology tables read on the way (prefill instance and links) are L1-resident.  A
  // prefetched decision is superseded when the request's arrival was processed after
  // the prefetch was issued (the last PD+1 arrivals are kept in registers).
  constexpr int PD = 1;
  constexpr int FD = PD + 1;
  constexpr int CD = PD + 2;
  const uint32_t kBad = 0xffffffffu;
  uint32_t cq[CD + 1];                        // event codes, index i = event e+i
  uint32_t lq[FD + 1], pq[FD + 1], kq[FD + 1], mq[FD + 1][NPT];
  float xq[FD + 1][NPT];  // s_eff / Bbot with self-contention over base scores
  int64_t tq[FD + 1];                         // arrival times (self-contention only)
  float4 ubpq[PD + 1];
  float ubdq[PD + 1][NPT];
  int tauq[PD + 1][NPT];
  int32_t decq[PD + 1];
  uint32_t arr_r[PD + 1];                     // last arrivals processed, newest first
  int32_t arr_d[PD + 1];
#pragma unroll
  for (int i = 0; i <= PD; ++i) {
    arr_r[i] = kBad;
    arr_d[i] = -1;
  }

  // fields of an event (len, prefill, snap, prefix hits); kBad code or bad r gives zeros
  auto fields = [&](uint32_t code, uint32_t& l, uint32_t& pr, uint32_t& k, uint32_t* m) {
    l = pr = k = 0;
#pragma unroll
    for (int j = 0; j < NPT; ++j) m[j] = 0;
    if (code == kBad) return;
    const uint32_t r = code & 0x7fffffffu;
    if (r >= R) return;
    l = __ldg(len + r);
    if (code >> 31) {
      if (kLoad) {  // the departure returns the bytes its dispatch took
        const uint16_t* m_row = M + (uint64_t)r * D;
#pragma unroll
        for (int j = 0; j < NPT; ++j) {
          const uint32_t d = tid * NPT + j;
          if (d < D) m[j] = __ldg(m_row + d);
        }
      }
      return;
    }
    pr = __ldg(prefill + r);
    k = __ldg(snap + r);
    if (kBase) {  // precomputed network + prefix terms, carried as raw bits
      const float* b_row = base + (uint64_t)r * D;
#pragma unroll
      for (int j = 0; j < NPT; ++j) {
        const uint32_t d = tid * NPT + j;
        if (d < D) m[j] = __float_as_uint(__ldg(b_row + d));
      }
    } else {
      const uint16_t* m_row = M + (uint64_t)r * D;
#pragma unroll
      for (int j = 0; j < NPT; ++j) {
        const uint32_t d = tid * NPT + j;
        if (d < D) m[j] = __ldg(m_row + d);
      }
    }
  };
  // level bottlenecks (arrival) or decision (departure) of an event whose fields are known
  auto operands = [&](uint32_t code, uint32_t pr, uint32_t k, float4& ubp, float* ubd, int* tau,
                      int32_t& dec_pref) {
    dec_pref = -1;
    ubp = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      ubd[j] = 0.0f;
      tau[j] = 0;
    }
    if (code == kBad) return;
    const uint32_t r = code & 0x7fffffffu;
    if (r >= R) return;
    if (code >> 31) {
      if (lane == 0) dec_pref = *((volatile int32_t*)(dec + r));
      return;
    }
    if ((kBase && !kInfl) || pr >= t.P || k >= n_snap) return;
    const uint32_t pinst = __ldg(t.pre + pr);
    const uint4 lp = __ldg(t.links + pinst);
    if (!kBase) ubp = __ldg(reinterpret_cast<const float4*>(UB) + (uint64_t)k * N + pinst);
    const float* ub_row = UB + (uint64_t)k * N * 4;
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      tau[j] = tier_of(lp, ld[j]);
      if (!kBase && tid * NPT + j < D) ubd[j] = __ldg(ub_row + (uint64_t)ld[j].x * 4 + tau[j]);
    }
  };
  // with self-contention over base scores: the arrival's s_eff / Bbot row
  auto xrow = [&](uint32_t code, float* x) {
#pragma unroll
    for (int j = 0; j < NPT; ++j) x[j] = 0.0f;
    if (!(kBase && kInfl) || code == kBad || (code >> 31)) return;
    const uint32_t r = code & 0x7fffffffu;
    if (r >= R) return;
    const float* x_row = xf + (uint64_t)r * D;
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      const uint32_t d = tid * NPT + j;
      if (d < D) x[j] = __ldg(x_row + d);
    }
  };

#pragma unroll
  for (int i = 0; i <= CD; ++i) cq[i] = (e0 + i < e1) ? __ldg(events + e0 + i) : kBad;
  auto time_of = [&](uint32_t code) -> int64_t {
    if (!kInfl || code == kBad || (code >> 31) || (code & 0x7fffffffu) >= R) return 0;
    return __ldg(arrival_us + (code & 0x7fffffffu));
  };
#pragma unroll
  for (int i = 0; i <= FD; ++i) {
    fields(cq[i], lq[i], pq[i], kq[i], mq[i]);
    xrow(cq[i], xq[i]);
    tq[i] = time_of(cq[i]);
  }
#pragma unroll
  for (int i = 0; i <= PD; ++i) operands(cq[i], pq[i], kq[i], ubpq[i], ubdq[i], tauq[i], decq[i]);

  for (uint64_t e = e0; e < e1; ++e) {
    // take event e's operands, then advance the pipeline by one event
    const uint32_t code = cq[0], l = lq[0], pr = pq[0], k = kq[0];
    const int64_t now = tq[0];
    const float4 ubp = ubpq[0];
    float ubd[NPT];
    int tau[NPT];
    uint32_t m[NPT];
    float xv[NPT];
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      ubd[j] = ubdq[0][j];
      tau[j] = tauq[0][j];
      m[j] = mq[0][j];
      xv[j] = xq[0][j];
    }
    const int32_t dec_pref = decq[0];
#pragma unroll
    for (int i = 0; i < CD; ++i) cq[i] = cq[i + 1];
#pragma unroll
    for (int i = 0; i < FD; ++i) {
      lq[i] = lq[i + 1];
      pq[i] = pq[i + 1];
      kq[i] = kq[i + 1];
      tq[i] = tq[i + 1];
#pragma unroll
      for (int j = 0; j < NPT; ++j) {
        mq[i][j] = mq[i + 1][j];
        xq[i][j] = xq[i + 1][j];
      }
    }
#pragma unroll
    for (int i = 0; i < PD; ++i) {
      ubpq[i] = ubpq[i + 1];
      decq[i] = decq[i + 1];
#pragma unroll
      for (int j = 0; j < NPT; ++j) {
        ubdq[i][j] = ubdq[i + 1][j];
        tauq[i][j] = tauq[i + 1][j];
      }
    }
    cq[CD] = (e + 1 + CD < e1) ? __ldg(events + e + 1 + CD) : kBad;
    fields(cq[FD], lq[FD], pq[FD], kq[FD], mq[FD]);
    xrow(cq[FD], xq[FD]);
    tq[FD] = time_of(cq[FD]);
    operands(cq[PD], pq[PD], kq[PD], ubpq[PD], ubdq[PD], tauq[PD], decq[PD]);

    const uint32_t r = code & 0x7fffffffu;
    if (r >= R) {
      if (lead_thread) flag_status(status, NETKV_DEV_ERANGE);
      continue;
    }
    if (code >> 31) {  // departure: release the tokens of a dispatched request
      int32_t dd = __shfl_sync(smask, dec_pref, 0, LPS);
#pragma unroll
      for (int i = PD; i >= 0; --i)  // decided after the prefetch was issued
        if (r == arr_r[i]) dd = arr_d[i];
      if (dd >= 0 && (uint32_t)dd < D) {
#pragma unroll
        for (int j = 0; j < NPT; ++j)
          if (tid * NPT + j == (uint32_t)dd) {
            if (kLoad) {
              const uint32_t lam = min(16u * m[j], l);
              load[j] += (int64_t)(l - lam) * (int64_t)w.bytes_per_token;
              held[j] -= 1;
            } else {
              load[j] -= l;
            }
          }
      }
      continue;
    }
    if (pr >= t.P || k >= n_snap || l == 0) {
      if (lead_thread) {
        flag_status(status, l == 0 ? NETKV_DEV_EDOMAIN : NETKV_DEV_ERANGE);
        best[r] = inf;
        second[r] = inf;
        if (kInfl) xfer_us[r] = -1;
      }
      if (lane == 0) *((volatile int32_t*)(dec + r)) = -1;
#pragma unroll
      for (int i = PD; i > 0; --i) {
        arr_r[i] = arr_r[i - 1];
        arr_d[i] = arr_d[i - 1];
      }
      arr_r[0] = r;
      arr_d[0] = -1;
      continue;
    }

    uint32_t cw = 0;  // self-contention counters of the request's prefill, a byte per tier
    if constexpr (kInfl) {
      if (lead_thread) {  // transfers completed by now (Algorithm 1 line 14's callback)
        while (heap.n > 0 && (int64_t)(heap.a[0] >> 16) <= now) {
          const uint32_t pt = (uint32_t)(heap.a[0] & 0xffffu);
          heap.pop();
          uint32_t* c = cnt + (pt >> 2);
          const uint32_t sh = 8u * (pt & 3u);
          if ((*c >> sh) & 0xffu) *c -= 1u << sh;
        }
      }
      if (LPS == 32) __syncthreads(); else __syncwarp(smask);
      cw = cnt[pr];
    }
    float b = inf, s2 = inf, bt = 0.0f;
    uint32_t bi = kNone;
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      const uint32_t d = tid * NPT + j;
      if (d < D) {
        bool feasible = load[j] + (int64_t)l <= w.cap_tokens;
        float sc, tj = 0.0f;
        if (kLoad) {  // Sec. IV-B: T_queue + T_decode; Sec. IV-A: m_d >= s_eff + m_min
          const uint32_t lam = min(16u * m[j], l);
          feasible = load[j] >= (int64_t)(l - lam) * (int64_t)w.bytes_per_token + lm.m_min;
          const int32_t beta = min(held[j], lm.beta_max);
          const int32_t blocked = (held[j] - beta) - (lm.beta_max - beta);
          const float t_queue = (blocked > 0 ? (float)blocked : 0.0f) * (lm.t_a + lm.t_b * (float)beta);
          const float t_decode = lm.t_a + lm.t_b * (float)(beta + 1);
          sc = base_score(w, l, m[j], pick4(ubp, tau[j]), ubd[j], pick4(lat, tau[j]), status) +
               w.w_load * (t_queue + t_decode);
        } else if (kBase && kInfl) {  // base + w_net (s_eff / Bbot) n: Eq. 4's 1 + n
          const uint32_t n = (cw >> (8 * tau[j])) & 0xffu;
          sc = (__uint_as_float(m[j]) + w.w_net * (xv[j] * (float)n)) +
               w.w_load * (w.theta_s_per_token * (float)load[j]);
          tj = xv[j] * (float)(1u + n) + pick4(lat, tau[j]);
        } else if (kBase) {
          sc = __uint_as_float(m[j]) + w.w_load * (w.theta_s_per_token * (float)load[j]);
        } else if (kInfl) {
          const float net_prefix =
              contended_score(w, l, m[j], pick4(ubp, tau[j]), ubd[j], pick4(lat, tau[j]),
                              (cw >> (8 * tau[j])) & 0xffu, tj, status);
          sc = net_prefix + w.w_load * (w.theta_s_per_token * (float)load[j]);
        } else {
          const float net_prefix = base_score(w, l, m[j], pick4(ubp, tau[j]), ubd[j],
                                              pick4(lat, tau[j]), status);
          sc = net_prefix + w.w_load * (w.theta_s_per_token * (float)load[j]);
        }
        if (feasible) {
          if (bi == kNone || sc < b) {
            s2 = b;
            b = sc;
            bi = d;
            bt = tj;
          } else if (sc < s2) {
            s2 = sc;
          }
        }
      }
    }
    if constexpr (kInfl) seg_argmin_t<LPS>(b, bi, s2, bt, smask);
    else seg_argmin<LPS>(b, bi, s2, smask);
    if (NW > 1) {
      if (lane == 0) {
        s_b[parity][wid] = b;
        s_i[parity][wid] = bi;
        s_s[parity][wid] = s2;
        if (kInfl) s_t[parity][wid] = bt;
      }
      __syncthreads();
      b = inf;
      s2 = inf;
      bi = kNone;
      if (lane < (uint32_t)NW) {
        b = s_b[parity][lane];
        bi = s_i[parity][lane];
        s2 = s_s[parity][lane];
        if (kInfl) bt = s_t[parity][lane];
      }
      if constexpr (kInfl) seg_argmin_t<32>(b, bi, s2, bt, 0xffffffffu);
      else seg_argmin<32>(b, bi, s2, 0xffffffffu);
      parity ^= 1u;
    }
    const int32_t dstar = bi == kNone ? -1 : (int32_t)bi;
    if constexpr (kLoad) {
      if (dstar >= 0) {
#pragma unroll
        for (int j = 0; j < NPT; ++j)
          if (tid * NPT + j == (uint32_t)dstar) {
            const uint32_t lam = min(16u * m[j], l);
            load[j] -= (int64_t)(l - lam) * (int64_t)w.bytes_per_token;
            held[j] += 1;
          }
      }
    }
    if constexpr (kInfl) {
      // the winner's tier: packed streams own one decode a lane, so its lane has it
      uint32_t ts_lane = 0;
      if (LPS < 32) ts_lane = (uint32_t)__shfl_sync(smask, tau[0], dstar < 0 ? 0 : dstar, LPS);
      if (lead_thread) {
        if (dstar < 0) {
          xfer_us[r] = -1;
        } else {  // the dispatch's tier counter (Algorithm 1 line 14) and its completion
          const float us = bt * 1.0e6f;
          const int64_t dt = us < 2147483520.0f ? __float2ll_rn(us) : 2147483647ll;
          xfer_us[r] = (int32_t)dt;
          uint32_t ts = ts_lane;
          if (LPS == 32) {
            const uint4 lp = __ldg(t.links + __ldg(t.pre + pr));
            const uint4 lo = __ldg(t.links + __ldg(t.dec + (uint32_t)dstar));
            ts = (uint32_t)tier_of(lp, lo);
          }
          uint32_t* c = cnt + pr;
          const uint32_t sh = 8u * ts;
          if (((*c >> sh) & 0xffu) < inflight_cap) *c += 1u << sh;
          if (!heap.push(((unsigned long long)(now + dt) << 16) | ((unsigned long long)pr << 2) | ts))
            flag_status(status, NETKV_DEV_EFULL);
        }
      }
    }
    if (!kLoad && dstar >= 0) {
#pragma unroll
      for (int j = 0; j < NPT; ++j)
        if (tid * NPT + j == (uint32_t)dstar) load[j] += l;
    }
    if (lane == 0) *((volatile int32_t*)(dec + r)) = dstar;
    if (lead_thread) {
      best[r] = b;
      second[r] = s2;
    }
#pragma unroll
    for (int i = PD; i > 0; --i) {
      arr_r[i] = arr_r[i - 1];
      arr_d[i] = arr_d[i - 1];
    }
    arr_r[0] = r;
    arr_d[0] = dstar;
  }
#pragma unroll
  for (int j = 0; j < NPT; ++j) {
    const uint32_t d = tid * NPT + j;
    if (d < D) {
      load_final[(uint64_t)stream * D + d] = load[j];
      if (kLoad) n_final[(uint64_t)stream * D + d] = held[j];
    }
  }
}

// ---- staged greedy: one CTA per stream with precomputed base scores ----------------
// Everything an event needs is copied into shared memory with cp.async STAGES events
// before the event is processed: each thread copies its own NPT base scores of an
// arrival's row, and lane 0 of each warp copies the event's request fields (length,
// prefill rank, snapshot and, for a departure, the decision recorded so far) into a
// record slot private to its warp.  A thread waits only for its own copies, and a warp
// reads its record after a warp barrier, so the ring needs no block barrier; the one
// block barrier per arrival is the argmin's.  A departure's decision may have been made
// after its record was copied: each warp keeps the last kRing arrivals' decisions.
// Event codes come from a shared two-chunk circular buffer (a chunk is BLOCK events,
// one per thread), refilled a chunk ahead with two block barriers per chunk.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async8(void* smem, const void* gmem) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;\n" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;\n" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

constexpr int kRing = 16;  // arrivals remembered per warp (>= STAGES + 1)

template <int NPT, int BLOCK, int STAGES>
__global__ void __launch_bounds__(BLOCK) schedule_staged_kernel(
    TopoArgs t, uint32_t n_streams, const netkv_weights* __restrict__ W, uint32_t R,
    const float* __restrict__ base, const uint32_t* __restrict__ len,
    const uint32_t* __restrict__ prefill, const uint32_t* __restrict__ snap, uint32_t n_snap,
    const uint32_t* __restrict__ events, const uint64_t* __restrict__ event_off,
    const int64_t* __restrict__ load_init, int32_t* dec, float* __restrict__ best,
    float* __restrict__ second, int64_t* __restrict__ load_final, int* status) {
  static_assert(kRing >= STAGES + 1 && kRing <= 32, "ring covers the staging distance");
  static_assert((BLOCK & (BLOCK - 1)) == 0 && STAGES < BLOCK, "code chunks");
  constexpr int NW = BLOCK / 32;
  constexpr uint32_t kBad = 0xffffffffu;
  extern __shared__ __align__(16) float ring[];  // [STAGES][BLOCK * NPT]
  __shared__ __align__(16) uint32_t rec[NW][STAGES][4];  // length, prefill, snapshot, decision
  __shared__ uint32_t aring_r[NW][kRing];
  __shared__ int32_t aring_d[NW][kRing];
  __shared__ uint32_t s_k[2][NW];
  __shared__ uint32_t s_i[2][NW];
  __shared__ uint32_t s_k2[2][NW];
  __shared__ uint32_t codes[2 * BLOCK];  // event e at (e - e0) mod 2 * BLOCK
  const uint32_t tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const uint32_t stream = blockIdx.x;
  if (stream >= n_streams) return;
  const uint32_t D = t.D;
  const bool vec = NPT % 4 == 0 && (D % 4u == 0) && ((reinterpret_cast<uintptr_t>(base) & 15u) == 0);
  const netkv_weights w = W[stream];
  const float inf = __int_as_float(0x7f800000);

  // per owned decode: load (active tokens), headroom cap - load clamped to 32 bits (0
  // for ranks past D) and theta * load, the last two redone only when the load changes
  int64_t load[NPT];
  uint32_t hr[NPT];
  float lt[NPT];
#pragma unroll
  for (int j = 0; j < NPT; ++j) {
    const uint32_t d = tid * NPT + j;
    load[j] = (load_init && d < D) ? load_init[(uint64_t)stream * D + d] : 0;
  }
  auto refresh = [&](int j) {
    const int64_t h = w.cap_tokens - load[j];
    hr[j] = tid * NPT + j >= D ? 0u : h <= 0 ? 0u : h >= 0xffffffffll ? 0xffffffffu : (uint32_t)h;
    lt[j] = w.theta_s_per_token * (float)load[j];
  };
#pragma unroll
  for (int j = 0; j < NPT; ++j) refresh(j);
  // add `delta` tokens to decode dd: only its owner thread does any work
  auto adjust = [&](uint32_t dd, int64_t delta) {
    const uint32_t jj = dd - tid * NPT;
    if (jj < (uint32_t)NPT) {
#pragma unroll
      for (int j = 0; j < NPT; ++j)
        if (jj == (uint32_t)j) {
          load[j] += delta;
          refresh(j);
        }
    }
  };
  if (lane < (uint32_t)kRing) {
    aring_r[wid][lane] = kBad;
    aring_d[wid][lane] = -1;
  }
  __syncwarp();
  const uint64_t e0 = event_off[stream], e1 = event_off[stream + 1];

  auto code_at = [&](uint64_t e) -> uint32_t { return e < e1 ? __ldg(events + e) : kBad; };
  // copies for one event into slot `slot` (one commit group per event, possibly empty)
  auto stage = [&](uint32_t code, uint32_t slot) {
    const uint32_t r = code & 0x7fffffffu;
    if (code != kBad && r < R) {
      if (lane == 0) {
        uint32_t* rc = rec[wid][slot];
        cp_async4(rc + 0, len + r);
        if (code >> 31) {
          cp_async4(rc + 3, dec + r);
        } else {
          cp_async4(rc + 1, prefill + r);
          cp_async4(rc + 2, snap + r);
        }
      }
      if (!(code >> 31)) {
        const float* src = base + (uint64_t)r * D + tid * NPT;
        float* dst = ring + (size_t)slot * (BLOCK * NPT) + tid * NPT;
        if (vec) {
#pragma unroll
          for (int j = 0; j < NPT; j += 4)
            if (tid * NPT + j < D) cp_async16(dst + j, src + j);
        } else {
#pragma unroll
          for (int j = 0; j < NPT; ++j)
            if (tid * NPT + j < D) cp_async4(dst + j, src + j);
        }
      }
    }
    cp_async_commit();
  };

  codes[tid] = code_at(e0 + tid);
  codes[BLOCK + tid] = code_at(e0 + BLOCK + tid);
  uint32_t next_code = code_at(e0 + 2 * BLOCK + tid);  // chunk 2, stored when chunk 1 starts
  __syncthreads();
  auto code_of = [&](uint64_t e) -> uint32_t {
    return codes[(uint32_t)((e - e0) & (2 * BLOCK - 1))];
  };
#pragma unroll
  for (int i = 0; i < STAGES; ++i) stage(code_of(e0 + i), (uint32_t)i);

  uint32_t slot = 0, parity = 0, n_arr = 0;
  for (uint64_t e = e0; e < e1; ++e) {
    const uint64_t off = e - e0;
    if (off != 0 && (off & (BLOCK - 1)) == 0) {
      // chunk k = off / BLOCK starts: chunk k - 1 is done everywhere; chunk k + 1 goes
      // into its place
      __syncthreads();
      codes[(uint32_t)((off - BLOCK) & (2 * BLOCK - 1)) + tid] = next_code;
      __syncthreads();
      next_code = code_at(e + 2 * BLOCK + tid);
    }
    const uint32_t code = code_of(e);
    const uint32_t ahead = code_of(e + STAGES);  // its copies go to the slot read here
    const uint32_t cur = slot;
    slot = slot + 1 == STAGES ? 0 : slot + 1;
    cp_async_wait<STAGES - 1>();  // this thread's copies for event e have landed
    __syncwarp();                  // and lane 0's record is visible to the warp

    const uint32_t r = code & 0x7fffffffu;
    if (r >= R) {
      if (tid == 0) flag_status(status, NETKV_DEV_ERANGE);
      __syncwarp();
      stage(ahead, cur);
      continue;
    }
    const uint4 f = *reinterpret_cast<const uint4*>(rec[wid][cur]);
    const uint32_t l = f.x;
    if (code >> 31) {  // departure: release the tokens of a dispatched request
      int32_t dd = (int32_t)f.w;
      const uint32_t hit = __ballot_sync(0xffffffffu, lane < (uint32_t)kRing &&
                                                          aring_r[wid][lane] == r);
      if (hit) dd = aring_d[wid][__ffs(hit) - 1];  // decided after the record was copied
      __syncwarp();
      stage(ahead, cur);
      if (dd >= 0 && (uint32_t)dd < D) adjust((uint32_t)dd, -(int64_t)l);
      continue;
    }
    const bool ok = f.y < t.P && f.z < n_snap && l != 0;
    const uint32_t ra = n_arr;
    n_arr = n_arr + 1 == (uint32_t)kRing ? 0 : n_arr + 1;
    if (!ok) {
      __syncwarp();
      stage(ahead, cur);
      if (tid == 0) {
        flag_status(status, l == 0 ? NETKV_DEV_EDOMAIN : NETKV_DEV_ERANGE);
        best[r] = inf;
        second[r] = inf;
      }
      if (lane == 0) {
        *((volatile int32_t*)(dec + r)) = -1;
        aring_r[wid][ra] = r;
        aring_d[wid][ra] = -1;
      }
      continue;
    }

    float bs[NPT];
    const float* src = ring + (size_t)cur * (BLOCK * NPT) + tid * NPT;
    if (vec) {
#pragma unroll
      for (int j = 0; j < NPT; j += 4) {
        const float4 v = *reinterpret_cast<const float4*>(src + j);
        bs[j] = v.x;
        bs[j + 1] = v.y;
        bs[j + 2] = v.z;
        bs[j + 3] = v.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < NPT; ++j) bs[j] = src[j];
    }
    // (score, rank) argmin with the second-best score, in two independent chains (even
    // and odd j) merged at the end; candidates are met in rank order within a chain
    float b = inf, s2 = inf, bo = inf, so = inf;
    uint32_t bi = kNone, bio = kNone;
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      const uint32_t d = tid * NPT + j;
      const bool feasible = l <= hr[j];  // load + l <= cap (l >= 1 here)
      const float sc = __fmaf_rn(w.w_load, lt[j], bs[j]);
      float& cb = (j & 1) ? bo : b;
      float& cs = (j & 1) ? so : s2;
      uint32_t& ci = (j & 1) ? bio : bi;
      const bool take = feasible && (ci == kNone || sc < cb);
      cs = take ? cb : (feasible ? fminf(cs, sc) : cs);
      cb = take ? sc : cb;
      ci = take ? d : ci;
    }
    if (NPT > 1) combine(b, bi, s2, bo, bio, so);
    __syncwarp();                // every lane has read the record and its scores
    stage(ahead, cur);  // before the slot is refilled
    uint32_t kb = bi == kNone ? kNoKey : score_key(b);
    uint32_t ks = score_key(s2);
    warp_argmin_keys(kb, bi, ks);
    if (NW > 1) {
      if (lane == 0) {
        s_k[parity][wid] = kb;
        s_i[parity][wid] = bi;
        s_k2[parity][wid] = ks;
      }
      __syncthreads();
      const uint32_t q = lane % NW;  // every lane holds some warp's partial
      kb = s_k[parity][q];
      bi = s_i[parity][q];
      ks = s_k2[parity][q];
      warp_argmin_keys(kb, bi, ks);
      parity ^= 1u;
    }
    b = key_score(kb);
    s2 = key_score(ks);
    const int32_t dstar = kb == kNoKey ? -1 : (int32_t)bi;
    if (dstar >= 0) adjust((uint32_t)dstar, (int64_t)l);
    if (lane == 0) {
      *((volatile int32_t*)(dec + r)) = dstar;
      aring_r[wid][ra] = r;
      aring_d[wid][ra] = dstar;
    }
    if (tid == 0) {
      best[r] = b;
      second[r] = s2;
    }
  }
  cp_async_wait<0>();
#pragma unroll
  for (int j = 0; j < NPT; ++j) {
    const uint32_t d = tid * NPT + j;
    if (d < D) load_final[(uint64_t)stream * D + d] = load[j];
  }
}

// ---- listed greedy: one warp per stream, candidate lists from the base pass ---------
// The stream's per-decode state lives in shared memory: load[d] (active tokens) and
// hl[d] = (headroom cap - load clamped to 32 bits, theta * load) for one 8-byte gather per
// candidate.  An arrival rescores only its listed candidates (lane i takes entry i) and
// checks the list's bound against lmin, a lower
// bound on every decode's load: exact at the start and after every full scan, lowered by
// departures and left unchanged by dispatches (which only raise a load).  An arrival the
// bounds do not certify is scanned in full from its base-score row, which also makes lmin
// exact again.  Certification needs w_load >= 0 and theta >= 0; a stream with other
// weights scans every arrival.
// Events go in windows of 32, double-buffered.  A window's records (code, length, prefill
// and snapshot, or for a departure the decision in global memory) and its arrivals' lists
// are copied with cp.async one window ahead, the copies of a departure's decision after the
// decisions of the window before were written back.  Before a window is walked, lane i
// prepares its event i: an arrival's validity and its certification threshold; a
// departure's decision, taken from the window before when its arrival is there, or marked
// as the slot of its arrival when that is earlier in the same window.  The arrival's
// certification threshold LB is prepared too, from lmin as the window starts; should a
// departure lower lmin during the window, the rest of the window computes it afresh.
// Decisions and scores are kept in the window buffer and written back when the window
// after starts.
struct __align__(16) ListWindow {
  uint4 rec[32];                                  // code, length, prefill | decision, snapshot
  uint2 bnd[32];                                  // (tau rank, tau key) of each arrival
  uint2 ent[32][kListLen];                        // (rank, base bits): each arrival's list
  int32_t wd[32];                                 // decisions of the window's arrivals
  uint32_t wbk[32], wsk[32];                      // their best and second-best keys
  uint32_t lb[32];                                // an arrival's LB key from the prepared lmin
};
constexpr uint32_t kInWindow = 0x40000000u;  // departure decision: the slot of its arrival

// The full argmin of one arrival from its base-score row (the listed walk's fallback), and
// the exact minimum load.  Kept out of line: the walk's fast path stays small.
__device__ __noinline__ float wide_to_float(int64_t x) { return (float)x; }

struct ScanResult {
  uint32_t kb, bi, ks;  // best key, its rank, second-best key
  int64_t lmin;         // the exact minimum load
};
__device__ __noinline__ ScanResult listed_full_scan(const float* __restrict__ row, uint32_t D,
                                                    bool vec, uint32_t l, float w_load,
                                                    const uint2* s_hl, const int64_t* s_load,
                                                    uint32_t lane) {
  float b = __int_as_float(0x7f800000), s2 = b;
  uint32_t ci = kNone;
  int64_t lm = INT64_MAX;
  auto visit = [&](uint32_t d, float bs) {
    const uint2 hl = s_hl[d];
    const int64_t ld = s_load[d];
    lm = ld < lm ? ld : lm;
    if (l <= hl.x) {
      const float sc = __fmaf_rn(w_load, __uint_as_float(hl.y), bs);
      const bool take = ci == kNone || sc < b;
      s2 = take ? b : fminf(s2, sc);
      b = take ? sc : b;
      ci = take ? d : ci;
    }
  };
  if (vec) {
#pragma unroll 4
    for (uint32_t d = 4 * lane; d < D; d += 128) {
      const float4 v = __ldcs(reinterpret_cast<const float4*>(row + d));
      visit(d, v.x);
      visit(d + 1, v.y);
      visit(d + 2, v.z);
      visit(d + 3, v.w);
    }
  } else {
#pragma unroll 4
    for (uint32_t d = lane; d < D; d += 32) visit(d, __ldcs(row + d));
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const int64_t x = __shfl_xor_sync(0xffffffffu, lm, o);
    lm = x < lm ? x : lm;
  }
  uint32_t kb = ci == kNone ? kNoKey : score_key(b), bi = ci, ks = score_key(s2);
  warp_argmin_keys(kb, bi, ks);
  return ScanResult{kb, bi, ks, lm};
}

__global__ void __launch_bounds__(32) schedule_listed_kernel(
    TopoArgs t, uint32_t n_streams, const netkv_weights* __restrict__ W, uint32_t R,
    const float* __restrict__ base, const uint2* __restrict__ lists,
    const uint2* __restrict__ bounds, const uint32_t* __restrict__ len,
    const uint32_t* __restrict__ prefill, const uint32_t* __restrict__ snap, uint32_t n_snap,
    const uint32_t* __restrict__ events, const uint64_t* __restrict__ event_off,
    const int64_t* __restrict__ load_init, int32_t* dec, float* __restrict__ best,
    float* __restrict__ second, int64_t* __restrict__ load_final, int* status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  constexpr uint32_t kBad = 0xffffffffu;
  const uint32_t lane = threadIdx.x;
  const uint32_t stream = blockIdx.x;
  if (stream >= n_streams) return;
  const uint32_t D = t.D;
  ListWindow* win = reinterpret_cast<ListWindow*>(smem_raw);  // [2]
  int64_t* s_load = reinterpret_cast<int64_t*>(win + 2);
  uint2* s_hl = reinterpret_cast<uint2*>(s_load + D);  // [D + 1]: s_hl[D] fits no request
  const netkv_weights w = W[stream];
  const bool listed = w.w_load >= 0.0f && w.theta_s_per_token >= 0.0f;
  const bool vec = (D % 4u == 0) && ((reinterpret_cast<uintptr_t>(base) & 15u) == 0);

  // (float)x of a load: through int32 when it fits (the same value, without the slow 64-bit
  // conversion, which stays out of line so that it is not evaluated on the common path)
  auto to_f = [](int64_t x) -> float {
    if (__builtin_expect(x == (int64_t)(int32_t)x, 1)) return (float)(int32_t)x;
    return wide_to_float(x);
  };
  auto hl_of = [&](int64_t ld) -> uint2 {
    const int64_t h = w.cap_tokens - ld;
    const uint32_t hr = h <= 0 ? 0u : h >= 0xffffffffll ? 0xffffffffu : (uint32_t)h;
    return make_uint2(hr, __float_as_uint(w.theta_s_per_token * to_f(ld)));
  };
  int64_t lmin = INT64_MAX;
  for (uint32_t d = lane; d < D; d += 32) {
    const int64_t ld = load_init ? load_init[(uint64_t)stream * D + d] : 0;
    s_load[d] = ld;
    s_hl[d] = hl_of(ld);
    lmin = ld < lmin ? ld : lmin;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const int64_t x = __shfl_xor_sync(0xffffffffu, lmin, o);
    lmin = x < lmin ? x : lmin;
  }
  float lt_min = w.theta_s_per_token * to_f(lmin);
  if (lane == 0) s_hl[D] = make_uint2(0u, 0u);
  __syncwarp();

  const uint64_t e0 = event_off[stream], e1 = event_off[stream + 1];
  const uint64_t n_win = (e1 - e0 + 31) / 32;
  auto codes_of = [&](uint64_t k) -> uint32_t {  // lane i: code of event i of window k
    const uint64_t e = e0 + 32 * k + lane;
    return e < e1 ? __ldg(events + e) : kBad;
  };
  // copies of window k (codes c) into buffer k & 1, as one cp.async group
  auto issue = [&](uint64_t k, uint32_t c) {
    ListWindow& wb = win[k & 1];
    const uint32_t r = c & 0x7fffffffu;
    const bool valid = c != kBad && r < R;
    wb.rec[lane].x = c;
    if (valid) {
      cp_async4(&wb.rec[lane].y, len + r);
      if (c >> 31) {
        cp_async4(&wb.rec[lane].z, dec + r);
      } else {
        cp_async4(&wb.rec[lane].z, prefill + r);
        cp_async4(&wb.rec[lane].w, snap + r);
      }
    }
    if (valid && !(c >> 31)) {  // the lane's arrival: its list (16 x 16 B) and bound
      const uint2* src = lists + (uint64_t)r * kListLen;
#pragma unroll
      for (int q = 0; q < kListLen; q += 2) cp_async16(&wb.ent[lane][q], src + q);
      cp_async8(&wb.bnd[lane], bounds + r);
    }
    cp_async_commit();
  };
  // decisions and scores of window k's arrivals to global memory (lane i: event i)
  auto write_back = [&](const ListWindow& wb) {
    const uint32_t c = wb.rec[lane].x, r = c & 0x7fffffffu;
    if (c != kBad && !(c >> 31) && r < R) {
      dec[r] = wb.wd[lane];
      best[r] = key_score(wb.wbk[lane]);
      second[r] = key_score(wb.wsk[lane]);
    }
  };
  // add `delta` tokens to decode dd: every lane computes the new state (no divergence), lane
  // 0 stores it (dispatches never lower lmin)
  auto adjust = [&](uint32_t dd, int64_t delta) {
    const int64_t ld = s_load[dd] + delta;
    const uint2 h = hl_of(ld);
    if (lane == 0) {
      s_load[dd] = ld;
      s_hl[dd] = h;
    }
    __syncwarp();
  };

  // departures find their arrival in the window before (decision) or in their own window
  // (slot) through tables keyed by r mod 128; a window whose arrivals collide in a table
  // searches by shuffles instead
  __shared__ uint2 s_prev[128];  // (r, decision)
  __shared__ uint2 s_cur[128];   // (r, window << 5 | slot)
  for (uint32_t q = lane; q < 128; q += 32) s_prev[q] = s_cur[q] = make_uint2(kBad, 0u);
  __syncwarp();
  uint32_t cn = codes_of(0);
  if (n_win > 0) issue(0, cn);
  cn = codes_of(1);
  uint32_t prev_code = kBad;  // lane j: event j of the window before and its decision
  int32_t prev_dec = -1;
  for (uint64_t k = 0; k < n_win; ++k) {
    if (k > 0) {  // the window before: remember its arrivals, write its results back
      const ListWindow& pb = win[(k - 1) & 1];
      prev_code = pb.rec[lane].x;
      prev_dec = pb.wd[lane];
      write_back(pb);
    }
    __syncwarp();  // every lane is done with buffer (k + 1) & 1
    if (k + 1 < n_win) issue(k + 1, cn);
    else cp_async_commit();
    cn = codes_of(k + 2);
    cp_async_wait<1>();  // window k's copies have landed
    __syncwarp();
    ListWindow& wb = win[k & 1];
    bool my_dep = false;   // lane i: event i is a departure to apply: its length and decode
    uint32_t my_l = 0;
    int32_t my_dd = -1;
    bool my_arr = false;   // event i is an arrival to decide
    {  // lane i prepares event i
      uint4 f = wb.rec[lane];
      const uint32_t c = f.x, r = c & 0x7fffffffu;
      // a departure's arrival in the window before, or earlier in this one (a lane's r
      // matches only an arrival's code)
      int32_t dd = (int32_t)f.z;
      const uint32_t tag = (uint32_t)(k << 5);
      const bool prev_arr = prev_code != kBad && !(prev_code >> 31);
      const bool cur_arr = c != kBad && !(c >> 31);
      if (prev_arr) s_prev[prev_code & 127u] = make_uint2(prev_code, (uint32_t)prev_dec);
      if (cur_arr) s_cur[c & 127u] = make_uint2(c, tag | lane);
      __syncwarp();
      const bool clash = (prev_arr && s_prev[prev_code & 127u].x != prev_code) ||
                         (cur_arr && s_cur[c & 127u].x != c);
      if (__any_sync(0xffffffffu, clash)) {
        for (uint32_t j = 0; j < 32; ++j) {
          const uint32_t pc = __shfl_sync(0xffffffffu, prev_code, j);
          const int32_t pd = __shfl_sync(0xffffffffu, prev_dec, j);
          if (pc == r) dd = pd;
        }
        for (uint32_t j = 0; j < 32; ++j) {
          const uint32_t cc = __shfl_sync(0xffffffffu, c, j);
          if (j < lane && cc == r) dd = (int32_t)(kInWindow | j);
        }
      } else if (c != kBad && (c >> 31) && r < R) {
        const uint2 pe = s_prev[r & 127u];
        if (pe.x == r) dd = (int32_t)pe.y;
        const uint2 ce = s_cur[r & 127u];
        if (ce.x == r && (ce.y & ~31u) == tag && (ce.y & 31u) < lane)
          dd = (int32_t)(kInWindow | (ce.y & 31u));
      }
      if (c == kBad) {
      } else if (r >= R) {
        flag_status(status, NETKV_DEV_ERANGE);
      } else if (c >> 31) {
        my_dep = f.y != 0u;  // a zero-length request released nothing
        my_l = f.y;
        my_dd = dd;
      } else {
        const uint32_t l = f.y;
        if (f.z < t.P && f.w < n_snap && l != 0) {
          const uint2 b = wb.bnd[lane];
          f.z = b.y;
          f.w = b.x;
          wb.lb[lane] = b.y == kNoKey || b.y == kBoundInvalid
                            ? b.y
                            : score_key(__fmaf_rn(w.w_load, lt_min, key_score(b.y)));
          my_arr = true;
        } else {
          flag_status(status, l == 0 ? NETKV_DEV_EDOMAIN : NETKV_DEV_ERANGE);
          wb.wd[lane] = -1;
          wb.wbk[lane] = kNoKey;
          wb.wsk[lane] = kNoKey;
        }
      }
      wb.rec[lane] = f;
    }
    __syncwarp();
    bool moved = false;  // lmin fell below the value the thresholds were prepared with
    const bool tie_ok = lmin >= 0;
    const uint32_t dep_mask = __ballot_sync(0xffffffffu, my_dep);
    uint32_t arr_mask = __ballot_sync(0xffffffffu, my_arr);
    uint32_t done = 0;  // events before `done` are applied
    // the departures between the last arrival and event `upto`, all at once: they commute
    // (each lowers one load), and lmin only needs the loads they leave
    auto depart = [&](uint32_t upto) {
      const uint32_t lo = done >= 32 ? 0u : ~0u << done;
      const uint32_t hi = upto >= 32 ? ~0u : (1u << upto) - 1u;
      const uint32_t bm = dep_mask & lo & hi;
      done = upto;
      if (!bm) return;
      __syncwarp();  // lane 0's decisions of this window are visible
      uint32_t d = kNone;
      if ((bm >> lane) & 1u) {
        int32_t dd = my_dd;
        if (dd >= 0 && ((uint32_t)dd & kInWindow)) dd = wb.wd[(uint32_t)dd & 31u];
        if (dd >= 0 && (uint32_t)dd < D) d = (uint32_t)dd;
      }
      // each lane releases its own decode; two departures of one decode (rare) go one by one
      const uint32_t peers = __match_any_sync(0xffffffffu, d);
      int64_t ld = INT64_MAX;
      if (__any_sync(0xffffffffu, d != kNone && __popc(peers) > 1)) {
        uint32_t rest = __ballot_sync(0xffffffffu, d != kNone);
        while (rest) {
          const uint32_t src = __ffs(rest) - 1;
          rest &= rest - 1;
          const uint32_t ds = __shfl_sync(0xffffffffu, d, src);
          const uint32_t ls = __shfl_sync(0xffffffffu, my_l, src);
          if (lane == 0) {
            const int64_t x = s_load[ds] - (int64_t)ls;
            s_load[ds] = x;
            s_hl[ds] = hl_of(x);
          }
          __syncwarp();
        }
        if (d != kNone) ld = s_load[d];
      } else if (d != kNone) {
        ld = s_load[d] - (int64_t)my_l;
        s_load[d] = ld;
        s_hl[d] = hl_of(ld);
      }
      if (__any_sync(0xffffffffu, ld < lmin)) {
#pragma unroll
        for (int o = 16; o; o >>= 1) {
          const int64_t x = __shfl_xor_sync(0xffffffffu, ld, o);
          ld = x < ld ? x : ld;
        }
        lmin = ld < lmin ? ld : lmin;
        lt_min = w.theta_s_per_token * to_f(lmin);
        moved = true;
      }
      __syncwarp();
    };
    while (arr_mask) {
      const uint32_t i = __ffs(arr_mask) - 1;
      arr_mask &= arr_mask - 1;
      // the arrival's record, list entry and threshold do not change: read them first
      const uint4 f = wb.rec[i];
      const uint2 e = wb.ent[i][lane];
      const uint32_t lb_i = wb.lb[i];
      depart(i);
      done = i + 1;
      const uint32_t l = f.y;
      // the lane's listed candidate (s_hl[D]: a sentinel no request fits, for empty entries)
      const uint2 hl = s_hl[min(e.x, D)];
      const uint32_t lk = l <= hl.x
          ? score_key(__fmaf_rn(w.w_load, __uint_as_float(hl.y), __uint_as_float(e.y)))
          : kNoKey;
      // (key, rank) argmin and second key: the rank and the second depend only on the key
      const uint32_t kb = __reduce_min_sync(0xffffffffu, lk);
      const uint32_t bi = __reduce_min_sync(0xffffffffu, lk == kb ? e.x : kNone);
      const uint32_t ties = __popc(__ballot_sync(0xffffffffu, lk == kb));
      const uint32_t ks_one = __reduce_min_sync(0xffffffffu, lk == kb ? kNoKey : lk);
      const uint32_t ks = ties >= 2 ? kb : ks_one;
      // the listed decision is taken at once; an arrival the bounds did not certify (rare)
      // takes it back and is decided by the full scan.  The dispatch's load is read before
      // the certification test, whose arithmetic then covers its latency.
      int32_t dstar = kb == kNoKey ? -1 : (int32_t)bi;
      const int64_t ld_star = s_load[dstar >= 0 ? (uint32_t)dstar : 0u];
      const uint32_t tk = f.z, ti = f.w;
      bool cert = listed && tk != kBoundInvalid;
      if (cert && tk != kNoKey) {
        const uint32_t klb =
            moved ? score_key(__fmaf_rn(w.w_load, lt_min, key_score(tk))) : lb_i;
        const bool tie = moved ? lmin >= 0 : tie_ok;
        cert = (kb < klb || (kb == tk && tie && bi < ti)) && ks <= klb;
      }
      if (dstar >= 0) {
        const int64_t ld = ld_star + (int64_t)l;
        const uint2 h = hl_of(ld);
        if (lane == 0) {
          s_load[dstar] = ld;
          s_hl[dstar] = h;
        }
        __syncwarp();
      }
      if (lane == 0) {
        wb.wd[i] = dstar;
        wb.wbk[i] = kb;
        wb.wsk[i] = ks;
      }
      if (!cert) {
        if (dstar >= 0) adjust((uint32_t)dstar, -(int64_t)l);
        const ScanResult sr = listed_full_scan(base + (uint64_t)(f.x & 0x7fffffffu) * D, D, vec,
                                               l, w.w_load, s_hl, s_load, lane);
        lmin = sr.lmin;
        lt_min = w.theta_s_per_token * to_f(lmin);
        dstar = sr.kb == kNoKey ? -1 : (int32_t)sr.bi;
        if (dstar >= 0) adjust((uint32_t)dstar, (int64_t)l);
        if (lane == 0) {
          wb.wd[i] = dstar;
          wb.wbk[i] = sr.kb;
          wb.wsk[i] = sr.ks;
        }
      }
    }
    depart(32);  // departures after the window's last arrival
  }
  __syncwarp();
  if (n_win > 0) write_back(win[(n_win - 1) & 1]);
  cp_async_wait<0>();
  __syncwarp();
  for (uint32_t d = lane; d < D; d += 32) load_final[(uint64_t)stream * D + d] = s_load[d];
}

// ---- windowed greedy of small pools (D <= LPS <= 16) with precomputed base scores -----
// 32 / LPS streams per warp, one segment of LPS lanes each; lane sl owns decode sl's load
// (and theta * load) in registers.  A stream's events go in windows of 32, double-buffered
// in shared memory: each event's record (code, length, prefill | decision, snapshot) and an
// arrival's base-score row are copied with cp.async one window ahead by the lane that
// prepares the event (event j of a window: lane j % LPS).  Before a window is walked, each
// departure's decision is found: from the window before or as the slot of its arrival in
// this window, through tables keyed by request index mod 64 (a window whose arrivals collide
// there searches by shuffles), else the copy of the global decision (written back one window
// earlier).  The window is then walked arrival by arrival, the segments of a warp side by
// side: the departures since a segment's last arrival are applied one after another (a
// broadcast and the owner lane's update each), then every lane scores its decode exactly as
// schedule_kernel does, and a segment butterfly takes the (score, rank) argmin with the
// second score.  Decisions and scores go back to global memory when the next window starts.
template <int LPS>
struct WinSeg {              // one stream's window buffer
  uint4 rec[32];             // code, length, prefill | decision, snapshot
  float bs[32][LPS];         // base scores of an arrival's row
  int32_t wd[32];            // decisions
  float wb[32], ws[32];      // best and second scores
};
constexpr int kWinWarps = 4;  // warps per block (independent)

template <int LPS>
__global__ void __launch_bounds__(32 * kWinWarps) schedule_window_kernel(
    TopoArgs t, uint32_t n_streams, const netkv_weights* __restrict__ W, uint32_t R,
    const float* __restrict__ base, const uint32_t* __restrict__ len,
    const uint32_t* __restrict__ prefill, const uint32_t* __restrict__ snap, uint32_t n_snap,
    const uint32_t* __restrict__ events, const uint64_t* __restrict__ event_off,
    const int64_t* __restrict__ load_init, int32_t* dec, float* __restrict__ best,
    float* __restrict__ second, int64_t* __restrict__ load_final, int* status) {
  static_assert(LPS == 8 || LPS == 16, "segments of 8 or 16 lanes");
  constexpr int S = 32 / LPS;  // streams per warp
  constexpr int E = 32 / LPS;  // events a lane prepares per window
  constexpr uint32_t kBad = 0xffffffffu;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  const uint32_t lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  const uint32_t seg = lane / LPS, sl = lane % LPS, seg0 = seg * LPS;
  const uint32_t smask = ((1u << LPS) - 1u) << seg0;
  const uint32_t stream = ((uint32_t)blockIdx.x * kWinWarps + wib) * S + seg;
  const bool live = stream < n_streams;
  WinSeg<LPS>* wsb = reinterpret_cast<WinSeg<LPS>*>(smem_raw) + ((size_t)wib * S + seg) * 2;
  uint2* tabs = reinterpret_cast<uint2*>(reinterpret_cast<WinSeg<LPS>*>(smem_raw) +
                                         (size_t)kWinWarps * S * 2) +
                ((size_t)wib * S + seg) * 128;
  uint2* tab_prev = tabs;       // (r, decision) of the window before's arrivals
  uint2* tab_cur = tabs + 64;   // (r, window << 5 | slot) of this window's arrivals
  // tokens released before the segment's b-th arrival of the window, per decode: rel[b][d]
  uint32_t* rel = reinterpret_cast<uint32_t*>(reinterpret_cast<uint2*>(
                      reinterpret_cast<WinSeg<LPS>*>(smem_raw) + (size_t)kWinWarps * S * 2) +
                  (size_t)kWinWarps * S * 128) +
                  ((size_t)wib * S + seg) * 33 * LPS;
  const uint32_t D = t.D;
  const netkv_weights w = live ? W[stream] : W[0];
  const float inf = __int_as_float(0x7f800000);
  const bool mine = live && sl < D;
  const bool vec4 = (D % 4u == 0) && ((reinterpret_cast<uintptr_t>(base) & 15u) == 0);

  int64_t load = 0;
  if (mine && load_init) load = load_init[(uint64_t)stream * D + sl];
  float ltf = w.theta_s_per_token * (float)load;
  for (uint32_t q = sl; q < 128; q += LPS) tabs[q] = make_uint2(kBad, 0u);
  for (uint32_t q = sl; q < 33u * LPS; q += LPS) rel[q] = 0u;

  const uint64_t e0 = live ? event_off[stream] : 0, e1 = live ? event_off[stream + 1] : 0;
  const uint32_t my_win = (uint32_t)((e1 - e0 + 31) / 32);
  const uint32_t n_win = __reduce_max_sync(0xffffffffu, my_win);
  auto codes_of = [&](uint32_t k, uint32_t* c) {
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint64_t e = e0 + 32ull * k + (uint32_t)q * LPS + sl;
      c[q] = e < e1 ? __ldg(events + e) : kBad;
    }
  };
  // window k's copies (codes c) into buffer k & 1, one cp.async group
  auto issue = [&](uint32_t k, const uint32_t* c) {
    WinSeg<LPS>& b = wsb[k & 1];
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t j = (uint32_t)q * LPS + sl, code = c[q], r = code & 0x7fffffffu;
      b.rec[j].x = code;
      if (code != kBad && r < R) {
        cp_async4(&b.rec[j].y, len + r);
        if (code >> 31) {
          cp_async4(&b.rec[j].z, dec + r);
        } else {
          cp_async4(&b.rec[j].z, prefill + r);
          cp_async4(&b.rec[j].w, snap + r);
          const float* row = base + (uint64_t)r * D;
          if (vec4) {  // 16-byte copies: D % 4 == 0 and an aligned base
            for (uint32_t d = 0; d < D; d += 4) cp_async16(&b.bs[j][d], row + d);
          } else {
            for (uint32_t d = 0; d < D; ++d) cp_async4(&b.bs[j][d], row + d);
          }
        }
      }
    }
    cp_async_commit();
  };

  uint32_t cn[E], cc[E], pc[E];  // codes of the next window, this one, the one before
  int32_t pd[E];                 // decisions of the window before (its arrivals)
#pragma unroll
  for (int q = 0; q < E; ++q) {
    pc[q] = kBad;
    pd[q] = -1;
  }
  codes_of(0, cc);
  if (n_win > 0) issue(0, cc);
  codes_of(1, cn);
  for (uint32_t k = 0; k < n_win; ++k) {
    if (k > 0) {  // the window before (codes pc): write its results back, remember them
      const WinSeg<LPS>& pb = wsb[(k - 1) & 1];
#pragma unroll
      for (int q = 0; q < E; ++q) {
        const uint32_t j = (uint32_t)q * LPS + sl, code = pc[q], r = code & 0x7fffffffu;
        pd[q] = -1;
        if (code != kBad && !(code >> 31) && r < R) {
          pd[q] = pb.wd[j];
          dec[r] = pb.wd[j];
          best[r] = pb.wb[j];
          second[r] = pb.ws[j];
          tab_prev[r & 63u] = make_uint2(r, (uint32_t)pd[q]);
        }
      }
    }
    __syncwarp();  // every lane is done with buffer (k + 1) & 1 and the tables
    if (k + 1 < n_win) issue(k + 1, cn);
    else cp_async_commit();
    uint32_t cn2[E];  // the window after next
    codes_of(k + 2, cn2);
    cp_async_wait<1>();
    __syncwarp();
    WinSeg<LPS>& b = wsb[k & 1];
    // prepare: this window's arrivals into the current table, then every departure's decision
    bool clash = false;
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t j = (uint32_t)q * LPS + sl, code = cc[q], r = code & 0x7fffffffu;
      if (code != kBad && !(code >> 31) && r < R) tab_cur[r & 63u] = make_uint2(r, (k << 5) | j);
      if (k > 0 && pc[q] != kBad && !(pc[q] >> 31) && (pc[q] & 0x7fffffffu) < R)
        clash |= tab_prev[pc[q] & 63u].x != pc[q];
    }
    __syncwarp();
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t j = (uint32_t)q * LPS + sl, code = cc[q], r = code & 0x7fffffffu;
      if (code != kBad && !(code >> 31) && r < R) clash |= tab_cur[r & 63u].y != ((k << 5) | j);
    }
    const bool seg_clash = (__ballot_sync(0xffffffffu, clash) & smask) != 0;
    uint32_t l_ev[E], dd_ev[E];  // per prepared event: length, departure's decode or marker
    uint32_t arr_bits = 0, dep_bits = 0;  // this lane's events, bit q
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t j = (uint32_t)q * LPS + sl, code = cc[q], r = code & 0x7fffffffu;
      const uint4 f = b.rec[j];
      l_ev[q] = f.y;
      dd_ev[q] = kBad;
      if (code == kBad) continue;
      if (r >= R) {
        flag_status(status, NETKV_DEV_ERANGE);
        continue;
      }
      if (code >> 31) {
        int32_t dd = (int32_t)f.z;
        if (!seg_clash) {
          const uint2 pe = tab_prev[r & 63u];
          if (pe.x == r) dd = (int32_t)pe.y;
          const uint2 ce = tab_cur[r & 63u];
          if (ce.x == r && (ce.y >> 5) == (k & 0x7ffffffu) && (ce.y & 31u) < j)
            dd = (int32_t)(kInWindow | (ce.y & 31u));
        }
        dd_ev[q] = (uint32_t)dd;
        if (f.y != 0u) dep_bits |= 1u << q;
      } else {
        if (f.z < t.P && f.w < n_snap && f.y != 0u) {
          arr_bits |= 1u << q;
        } else {
          flag_status(status, f.y == 0u ? NETKV_DEV_EDOMAIN : NETKV_DEV_ERANGE);
          b.wd[j] = -1;
          b.wb[j] = inf;
          b.ws[j] = inf;
        }
      }
    }
    if (__any_sync(0xffffffffu, seg_clash)) {  // collisions: search the windows by shuffles
#pragma unroll
      for (int q = 0; q < E; ++q) {
        const uint32_t j = (uint32_t)q * LPS + sl, r = cc[q] & 0x7fffffffu;
        const bool dep = cc[q] != kBad && (cc[q] >> 31) && r < R;
#pragma unroll
        for (int qq = 0; qq < E; ++qq) {
          for (uint32_t m = 0; m < (uint32_t)LPS; ++m) {
            const uint32_t pcs = __shfl_sync(0xffffffffu, pc[qq], seg0 + m);
            const int32_t pds = __shfl_sync(0xffffffffu, pd[qq], seg0 + m);
            const uint32_t ccs = __shfl_sync(0xffffffffu, cc[qq], seg0 + m);
            const uint32_t jj = (uint32_t)qq * LPS + m;
            if (seg_clash && dep) {
              if (pcs == r) dd_ev[q] = (uint32_t)pds;
              if (ccs == r && jj < j) dd_ev[q] = kInWindow | jj;
            }
          }
        }
      }
    }
    // the segment's arrival and departure slots (bit j of the window)
    uint32_t arr_mask = 0, dep_mask = 0;
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t ba = __ballot_sync(0xffffffffu, (arr_bits >> q) & 1u);
      const uint32_t bd = __ballot_sync(0xffffffffu, (dep_bits >> q) & 1u);
      arr_mask |= ((ba >> seg0) & ((1u << LPS) - 1u)) << (q * LPS);
      dep_mask |= ((bd >> seg0) & ((1u << LPS) - 1u)) << (q * LPS);
    }
    // a departure whose decode is known now (not an arrival of this window) adds its tokens
    // to rel[number of the segment's arrivals before it][decode]; the rest (and any of more
    // than 2^27 tokens, so that a sum of 32 fits in 32 bits) are released one by one
    uint32_t slow_bits = 0;
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t j = (uint32_t)q * LPS + sl;
      bool slow = false;
      if ((dep_bits >> q) & 1u) {
        const uint32_t dd = dd_ev[q];
        if ((dd & kInWindow) && (int32_t)dd >= 0) {
          slow = true;
        } else if (dd < D) {
          if (l_ev[q] < (1u << 27)) atomicAdd(&rel[__popc(arr_mask & ((1u << j) - 1u)) * LPS + dd], l_ev[q]);
          else slow = true;
        }
      }
      slow_bits |= (slow ? 1u : 0u) << q;
    }
    uint32_t slow_mask = 0;
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t bs_ = __ballot_sync(0xffffffffu, (slow_bits >> q) & 1u);
      slow_mask |= ((bs_ >> seg0) & ((1u << LPS) - 1u)) << (q * LPS);
    }
    __syncwarp();  // prepared results of invalid arrivals and the releases are visible
    // the segment's released tokens of batch `bi` (the departures before its bi-th arrival)
    auto release = [&](uint32_t bi) {
      if (mine) {
        const uint32_t x = rel[bi * LPS + sl];
        if (x != 0u) {
          rel[bi * LPS + sl] = 0u;
          load -= (int64_t)x;
          ltf = w.theta_s_per_token * (float)load;
        }
      }
    };
    // the departures of slots in `bits` (segment-uniform), in slot order
    auto apply = [&](uint32_t bits) {
      uint32_t n = __popc(bits);
      const uint32_t rounds = __reduce_max_sync(0xffffffffu, n);
      for (uint32_t it = 0; it < rounds; ++it) {
        const bool has = bits != 0;
        const uint32_t j = has ? __ffs(bits) - 1 : 0u;
        if (has) bits &= bits - 1;
        const uint32_t qj = j / LPS, holder = seg0 + j % LPS;
        uint32_t pv = 0, pl = 0;
#pragma unroll
        for (int q = 0; q < E; ++q)
          if ((uint32_t)q == qj) {
            pv = dd_ev[q];
            pl = l_ev[q];
          }
        uint32_t dd = __shfl_sync(0xffffffffu, pv, holder);
        const uint32_t l = __shfl_sync(0xffffffffu, pl, holder);
        if (has && dd != kBad && (dd & kInWindow) && (int32_t)dd >= 0) dd = (uint32_t)b.wd[dd & 31u];
        if (has && mine && dd == sl) {
          load -= (int64_t)l;
          ltf = w.theta_s_per_token * (float)load;
        }
      }
    };
    uint32_t done = 0;  // slots below `done` are applied or decided
    const uint32_t rounds = __reduce_max_sync(0xffffffffu, __popc(arr_mask));
    for (uint32_t it = 0; it < rounds; ++it) {
      __syncwarp();  // decisions stored by earlier rounds are visible
      const bool has = arr_mask != 0;
      const uint32_t a = has ? __ffs(arr_mask) - 1 : 0u;
      if (has) arr_mask &= arr_mask - 1;
      release(it);
      apply(has ? slow_mask & ((1u << a) - 1u) & ~((1u << done) - 1u) : 0u);
      if (has) done = a + 1;
      const uint4 f = b.rec[a];
      const uint32_t l = f.y;
      float bsc = inf, s2 = inf;
      uint32_t bi = kNone;
      if (has && mine && load + (int64_t)l <= w.cap_tokens) {
        bsc = __fmaf_rn(w.w_load, ltf, b.bs[a][sl]);
        bi = sl;
      }
      seg_argmin<LPS>(bsc, bi, s2, 0xffffffffu);
      const int32_t dstar = bi == kNone ? -1 : (int32_t)bi;
      if (has && mine && dstar == (int32_t)sl) {
        load += (int64_t)l;
        ltf = w.theta_s_per_token * (float)load;
      }
      if (has && sl == 0) {
        b.wd[a] = dstar;
        b.wb[a] = bsc;
        b.ws[a] = s2;
      }
    }
    __syncwarp();
    release(rounds);  // after the last arrival
    apply(slow_mask & ~((1u << done) - 1u) & (done >= 32 ? 0u : ~0u));
#pragma unroll
    for (int q = 0; q < E; ++q) {  // the codes move on by one window
      pc[q] = cc[q];
      cc[q] = cn[q];
      cn[q] = cn2[q];
    }
  }
  __syncwarp();
  if (n_win > 0) {  // the last window's results (its codes are pc now)
    const WinSeg<LPS>& pb = wsb[(n_win - 1) & 1];
#pragma unroll
    for (int q = 0; q < E; ++q) {
      const uint32_t j = (uint32_t)q * LPS + sl, code = pc[q], r = code & 0x7fffffffu;
      if (code != kBad && !(code >> 31) && r < R) {
        dec[r] = pb.wd[j];
        best[r] = pb.wb[j];
        second[r] = pb.ws[j];
      }
    }
  }
  cp_async_wait<0>();
  if (mine) load_final[(uint64_t)stream * D + sl] = load;
}

constexpr int kStages = 8;
constexpr uint32_t kHeapPerStream = 4096;       // pending completions, one stream per CTA
constexpr uint32_t kHeapPerPackedStream = 256;  // pending completions, packed streams
constexpr size_t kInflightSmemMax = 200u * 1024u;

template <int NPT, int BLOCK>
netkv_status launch_staged(const TopoArgs& t, uint32_t n_streams, const netkv_weights* d_w,
                           uint32_t R, const uint32_t* d_len, const uint32_t* d_prefill,
                           const uint32_t* d_snap, uint32_t n_snap, const uint32_t* d_events,
                           const uint64_t* d_event_off, const int64_t* d_load_init,
                           int32_t* d_dec, float* d_best, float* d_second,
                           int64_t* d_load_final, const float* d_base, int* d_status,
                           cudaStream_t s) {
  const size_t smem = sizeof(float) * (size_t)kStages * BLOCK * NPT;
  // the attribute is per device: set it before every launch that needs it (cheap)
  if (smem > 48u * 1024u)
    NETKV_CUDA_TRY(cudaFuncSetAttribute(schedule_staged_kernel<NPT, BLOCK, kStages>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  schedule_staged_kernel<NPT, BLOCK, kStages><<<n_streams, BLOCK, smem, s>>>(
      t, n_streams, d_w, R, d_base, d_len, d_prefill, d_snap, n_snap, d_events, d_event_off,
      d_load_init, d_dec, d_best, d_second, d_load_final, d_status);
  return netkv_launch_status();
}

// The windowed walk of pools of at most LPS decodes: 32 / LPS streams per warp.
template <int LPS>
netkv_status launch_window(const TopoArgs& t, uint32_t n_streams, const netkv_weights* d_w,
                           uint32_t R, const uint32_t* d_len, const uint32_t* d_prefill,
                           const uint32_t* d_snap, uint32_t n_snap, const uint32_t* d_events,
                           const uint64_t* d_event_off, const int64_t* d_load_init,
                           int32_t* d_dec, float* d_best, float* d_second,
                           int64_t* d_load_final, const float* d_base, int* d_status,
                           cudaStream_t s) {
  constexpr uint32_t S = 32 / LPS;
  const size_t smem = (size_t)kWinWarps * S *
                      (2 * sizeof(WinSeg<LPS>) + 128 * sizeof(uint2) + 33 * LPS * sizeof(uint32_t));
  if (smem > 48u * 1024u)  // per device: set before every launch that needs it
    NETKV_CUDA_TRY(cudaFuncSetAttribute(schedule_window_kernel<LPS>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  const uint64_t warps = ((uint64_t)n_streams + S - 1) / S;
  const unsigned grid = (unsigned)((warps + kWinWarps - 1) / kWinWarps);
  schedule_window_kernel<LPS><<<grid, 32 * kWinWarps, smem, s>>>(
      t, n_streams, d_w, R, d_base, d_len, d_prefill, d_snap, n_snap, d_events, d_event_off,
      d_load_init, d_dec, d_best, d_second, d_load_final, d_status);
  return netkv_launch_status();
}

// The listed walk: one warp per stream, its decode state in dynamic shared memory.
netkv_status launch_listed(const TopoArgs& t, uint32_t n_streams, const netkv_weights* d_w,
                           uint32_t R, const uint32_t* d_len, const uint32_t* d_prefill,
                           const uint32_t* d_snap, uint32_t n_snap, const uint32_t* d_events,
                           const uint64_t* d_event_off, const int64_t* d_load_init,
                           int32_t* d_dec, float* d_best, float* d_second,
                           int64_t* d_load_final, const float* d_base, const uint2* d_lists,
                           const uint2* d_bounds, int* d_status, cudaStream_t s) {
  const size_t smem = sizeof(ListWindow) * 2 + (size_t)t.D * (sizeof(int64_t) + sizeof(uint2)) +
                      sizeof(uint2);  // s_hl[D], the sentinel
  if (smem > 48u * 1024u)  // per device: set before every launch that needs it
    NETKV_CUDA_TRY(cudaFuncSetAttribute(schedule_listed_kernel,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
  schedule_listed_kernel<<<n_streams, 32, smem, s>>>(
      t, n_streams, d_w, R, d_base, d_lists, d_bounds, d_len, d_prefill, d_snap, n_snap,
      d_events, d_event_off, d_load_init, d_dec, d_best, d_second, d_load_final, d_status);
  return netkv_launch_status();
}

// The base-score pre-pass over every arrival (and, with d_X, the factor s_eff / Bbot that
// self-contention scales).
template <bool kUtil = false>
netkv_status launch_base(const TopoArgs& t, uint32_t n_streams, const netkv_weights* d_w,
                         uint32_t R, const uint32_t* d_len, const uint32_t* d_prefill,
                         const uint32_t* d_snap, const uint16_t* d_M, const float* d_UB,
                         uint32_t n_snap, const uint32_t* d_events, const uint64_t* d_event_off,
                         float* d_base, float* d_X, int* d_status, cudaStream_t s,
                         uint2* d_lists = nullptr, uint2* d_bounds = nullptr) {
    const uint32_t D = t.D;
    const unsigned gy = n_streams >= 1024u ? 1u : (1024u + n_streams - 1) / n_streams;
    const dim3 bgrid(n_streams < (1u << 20) ? n_streams : (1u << 20), gy);
    if (D <= 8)
      base_kernel<8, kUtil><<<bgrid, 256, 0, s>>>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M,
                                           d_UB, n_snap, d_events, d_event_off, d_base, d_status, d_X);
    else if (D <= 16)
      base_kernel<16, kUtil><<<bgrid, 256, 0, s>>>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M,
                                            d_UB, n_snap, d_events, d_event_off, d_base, d_status, d_X);
    else if (D <= 32)
      base_kernel<32, kUtil><<<bgrid, 256, 0, s>>>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M,
                                            d_UB, n_snap, d_events, d_event_off, d_base, d_status, d_X);
    else {
      // one block per (stream, chunk of decodes) and arrival segment, ~32 blocks per SM
      int dev = 0, sms = 0;
      cudaGetDevice(&dev);
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      const uint32_t chunk = D <= 256 ? 256u : 1024u;
      const uint64_t gx = (uint64_t)n_streams * ((D + chunk - 1) / chunk);
      const uint64_t want = (uint64_t)(sms > 0 ? sms : 1) * 32;
      const unsigned wx = (unsigned)(gx < (1u << 20) ? gx : (1u << 20));
      const unsigned wy = (unsigned)(gx >= want ? 1 : (want + gx - 1) / gx < 65535 ? (want + gx - 1) / gx : 65535);
      if (D <= 256)
        base_wide_kernel<1, kUtil><<<dim3(wx, wy), 256, 0, s>>>(t, n_streams, d_w, R, d_len, d_prefill,
                                                         d_snap, d_M, d_UB, n_snap, d_events,
                                                         d_event_off, d_base, d_status, d_X);
      else if (d_lists)
        base_wide_kernel<4, kUtil, true><<<dim3(wx, wy), 256, 0, s>>>(
            t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, d_events,
            d_event_off, d_base, d_status, d_X, d_lists, d_bounds);
      else
        base_wide_kernel<4, kUtil><<<dim3(wx, wy), 256, 0, s>>>(t, n_streams, d_w, R, d_len, d_prefill,
                                                         d_snap, d_M, d_UB, n_snap, d_events,
                                                         d_event_off, d_base, d_status, d_X);
    }
  return netkv_launch_status();
}

template <int NPT, int BLOCK, int LPS, bool kUtil = false>
netkv_status launch(const TopoArgs& t, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
                    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap,
                    const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
                    const uint32_t* d_events, const uint64_t* d_event_off,
                    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
                    int64_t* d_load_final, float* d_base, int* d_status, cudaStream_t s,
                    const ListWs* lw = nullptr) {
  const uint32_t per_cta = LPS == 32 ? 1u : 32u / LPS;
  const unsigned grid = (n_streams + per_cta - 1) / per_cta;
  if (d_base) {
    const bool lists = LPS == 32 && lw != nullptr && lw->lists != nullptr;
    if (launch_base<kUtil>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M, d_UB, n_snap,
                           d_events, d_event_off, d_base, nullptr, d_status, s,
                           lists ? lw->chunk_lists : nullptr,
                           lists ? lw->chunk_bounds : nullptr) != NETKV_OK)
      return NETKV_ECUDA;
    if (lists) {
      int dev = 0, sms = 0;
      cudaGetDevice(&dev);
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      const uint64_t blocks = ((uint64_t)R * 32 + 255) / 256;
      const uint64_t cap = (uint64_t)(sms > 0 ? sms : 1) * 64;
      merge_lists_kernel<<<(unsigned)(blocks < cap ? blocks : cap), 256, 0, s>>>(
          lw->chunk_lists, lw->chunk_bounds, (t.D + kListChunk - 1) / kListChunk, R, lw->lists,
          lw->bounds);
      if (netkv_launch_status() != NETKV_OK) return NETKV_ECUDA;
      return launch_listed(t, n_streams, d_w, R, d_len, d_prefill, d_snap, n_snap, d_events,
                           d_event_off, d_load_init, d_dec, d_best, d_second, d_load_final,
                           d_base, lw->lists, lw->bounds, d_status, s);
    }
    if (LPS == 32) {
      // one CTA per stream: the walk is bound by each warp's chain of dependent
      // instructions per event; 16 warps (4 per scheduler) measured best on 4,096 decodes
      const uint32_t D = t.D;
      if (D <= 32) return launch_staged<1, 32>(t, n_streams, d_w, R, d_len, d_prefill, d_snap,
                                               n_snap, d_events, d_event_off, d_load_init, d_dec,
                                               d_best, d_second, d_load_final, d_base, d_status, s);
      if (D <= 256) return launch_staged<1, 256>(t, n_streams, d_w, R, d_len, d_prefill, d_snap,
                                                 n_snap, d_events, d_event_off, d_load_init, d_dec,
                                                 d_best, d_second, d_load_final, d_base, d_status, s);
      if (D <= 1024) return launch_staged<2, 512>(t, n_streams, d_w, R, d_len, d_prefill, d_snap,
                                                  n_snap, d_events, d_event_off, d_load_init, d_dec,
                                                  d_best, d_second, d_load_final, d_base, d_status, s);
      if (D <= 2048) return launch_staged<4, 512>(t, n_streams, d_w, R, d_len, d_prefill, d_snap,
                                                  n_snap, d_events, d_event_off, d_load_init, d_dec,
                                                  d_best, d_second, d_load_final, d_base, d_status, s);
      return launch_staged<8, 512>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, n_snap,
                                   d_events, d_event_off, d_load_init, d_dec, d_best, d_second,
                                   d_load_final, d_base, d_status, s);
    } else if (LPS == 8 || LPS == 16) {
      return launch_window<(LPS == 16 ? 16 : 8)>(t, n_streams, d_w, R, d_len, d_prefill, d_snap,
                                                 n_snap, d_events, d_event_off, d_load_init,
                                                 d_dec, d_best, d_second, d_load_final, d_base,
                                                 d_status, s);
    } else {
      schedule_kernel<NPT, BLOCK, LPS, true><<<grid, BLOCK, 0, s>>>(
          t, n_streams, d_w, R, d_base, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, d_events,
          d_event_off, d_load_init, d_dec, d_best, d_second, d_load_final, d_status);
    }
  } else {
    schedule_kernel<NPT, BLOCK, LPS, false><<<grid, BLOCK, 0, s>>>(
        t, n_streams, d_w, R, nullptr, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, d_events,
        d_event_off, d_load_init, d_dec, d_best, d_second, d_load_final, d_status);
  }
  return netkv_launch_status();
}

// Self-contention launch: dynamic shared memory per stream holds the counters (four
// bytes per prefill rank) and a heap of pending completions.
template <int NPT, int BLOCK, int LPS>
netkv_status launch_inflight(const TopoArgs& t, uint32_t n_streams, const netkv_weights* d_w,
                             uint32_t R, const uint32_t* d_len, const uint32_t* d_prefill,
                             const uint32_t* d_snap, const int64_t* d_arrival_us,
                             const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
                             const uint32_t* d_events, const uint64_t* d_event_off,
                             uint32_t inflight_cap, const int64_t* d_load_init, int32_t* d_dec,
                             float* d_best, float* d_second, int32_t* d_xfer_us,
                             int64_t* d_load_final, float* d_base, float* d_X, int* d_status,
                             cudaStream_t s) {
  const uint32_t per_cta = LPS == 32 ? 1u : 32u / LPS;
  const unsigned grid = (n_streams + per_cta - 1) / per_cta;
  const uint32_t heap_cap = LPS == 32 ? kHeapPerStream : kHeapPerPackedStream;
  const uint32_t infl_bytes = ((t.P * 4u + 15u) & ~15u) + heap_cap * 8u;
  const size_t smem = (size_t)per_cta * infl_bytes;
  if (smem > kInflightSmemMax) return NETKV_EINVAL;
  if (d_base) {  // base scores and s_eff / Bbot of every arrival first, in parallel
    if (launch_base(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, d_events,
                    d_event_off, d_base, d_X, d_status, s) != NETKV_OK)
      return NETKV_ECUDA;
    if (smem > 48u * 1024u)  // per device: set before every launch that needs it
      NETKV_CUDA_TRY(cudaFuncSetAttribute(schedule_kernel<NPT, BLOCK, LPS, true, true>,
                                          cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          (int)kInflightSmemMax));
    schedule_kernel<NPT, BLOCK, LPS, true, true><<<grid, BLOCK, smem, s>>>(
        t, n_streams, d_w, R, d_base, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, d_events,
        d_event_off, d_load_init, d_dec, d_best, d_second, d_load_final, d_status, d_arrival_us,
        inflight_cap, d_xfer_us, infl_bytes, heap_cap, LoadModel{0.f, 0.f, 0, 0, 0}, nullptr,
        nullptr, d_X);
    return netkv_launch_status();
  }
  if (smem > 48u * 1024u)  // per device: set before every launch that needs it
    NETKV_CUDA_TRY(cudaFuncSetAttribute(schedule_kernel<NPT, BLOCK, LPS, false, true>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        (int)kInflightSmemMax));
  schedule_kernel<NPT, BLOCK, LPS, false, true><<<grid, BLOCK, smem, s>>>(
      t, n_streams, d_w, R, nullptr, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, d_events,
      d_event_off, d_load_init, d_dec, d_best, d_second, d_load_final, d_status, d_arrival_us,
      inflight_cap, d_xfer_us, infl_bytes, heap_cap);
  return netkv_launch_status();
}

}  // namespace

namespace {
size_t round256(size_t b) { return (b + 255) / 256 * 256; }
// the base-score rows [R][D], always part of a workspace
size_t base_ws_bytes(uint32_t R, uint32_t D) { return round256((size_t)R * D * sizeof(float)); }
// pools of 1,025 .. 4,096 decodes: the chunks' candidate lists [R][n_ch][kListLen] and bounds
// [R][n_ch], then the pool's [R][kListLen] and [R] (listed walk)
bool listed_pool(uint32_t D) { return D >= kListMinD && D <= kListMaxD; }
uint32_t list_chunks(uint32_t D) { return (D + kListChunk - 1) / kListChunk; }
size_t list_ws_bytes(uint32_t R, uint32_t D) {
  if (!listed_pool(D)) return 0;
  const size_t nc = list_chunks(D);
  return round256((size_t)R * nc * kListLen * sizeof(uint2)) + round256((size_t)R * nc * sizeof(uint2)) +
         round256((size_t)R * kListLen * sizeof(uint2)) + round256((size_t)R * sizeof(uint2));
}
// the list arrays inside a workspace of `bytes` bytes, or nulls (the staged walk)
ListWs list_ws(void* ws, size_t bytes, uint32_t R, uint32_t D) {
  ListWs l;
  if (!ws || R == 0 || list_ws_bytes(R, D) == 0 || bytes < base_ws_bytes(R, D) + list_ws_bytes(R, D))
    return l;
  const size_t nc = list_chunks(D);
  char* p = reinterpret_cast<char*>(ws) + base_ws_bytes(R, D);
  l.chunk_lists = reinterpret_cast<uint2*>(p);
  p += round256((size_t)R * nc * kListLen * sizeof(uint2));
  l.chunk_bounds = reinterpret_cast<uint2*>(p);
  p += round256((size_t)R * nc * sizeof(uint2));
  l.lists = reinterpret_cast<uint2*>(p);
  p += round256((size_t)R * kListLen * sizeof(uint2));
  l.bounds = reinterpret_cast<uint2*>(p);
  return l;
}
}  // namespace

extern "C" size_t netkv_schedule_workspace_size(uint32_t R, uint32_t D) {
  return base_ws_bytes(R, D) + list_ws_bytes(R, D);
}

extern "C" netkv_status netkv_schedule_streams(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap, const uint16_t* d_M,
    const float* d_UB, uint32_t n_snap, const uint32_t* d_events, const uint64_t* d_event_off,
    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
    int64_t* d_load_final, void* d_workspace, size_t workspace_bytes, int* d_status,
    netkv_stream_t stream) {
  if (!topo || !d_w || !d_event_off || !d_load_final) return NETKV_EINVAL;
  if (n_streams == 0) return NETKV_OK;
  if (n_streams > 0x7fffffffu) return NETKV_EINVAL;
  if (R > 0 && (!d_len || !d_prefill || !d_snap || !d_M || !d_UB || !d_dec || !d_best ||
                !d_second || !d_events))
    return NETKV_EINVAL;
  if (!aligned_to(d_w, 8) || !aligned_to(d_UB, 16) || !aligned_to(d_event_off, 8) ||
      !aligned_to(d_load_final, 8) || (d_load_init && !aligned_to(d_load_init, 8)))
    return NETKV_EINVAL;
  const TopoArgs t = topo_args(topo);
  const uint32_t D = t.D;
  cudaStream_t s = (cudaStream_t)stream;
  if (d_workspace && (!aligned_to(d_workspace, 256) || workspace_bytes < base_ws_bytes(R, D)))
    return NETKV_EINVAL;
  float* d_base = (d_workspace && R > 0) ? reinterpret_cast<float*>(d_workspace) : nullptr;
  const ListWs lw = list_ws(d_base ? d_workspace : nullptr, workspace_bytes, R, D);
#define NETKV_SCHED(NPT, BLOCK, LPS)                                                             \
  return launch<NPT, BLOCK, LPS>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, \
                            d_events, d_event_off, d_load_init, d_dec, d_best, d_second,       \
                            d_load_final, d_base, d_status, s, &lw)
  if (D <= 8) NETKV_SCHED(1, 32, 8);
  if (D <= 16) NETKV_SCHED(1, 32, 16);
  if (D <= 32) NETKV_SCHED(1, 32, 32);
  if (D <= 256) NETKV_SCHED(1, 256, 32);
  if (D <= 1024) NETKV_SCHED(4, 256, 32);
  if (D <= 4096) NETKV_SCHED(4, 1024, 32);
#undef NETKV_SCHED
  return NETKV_EINVAL;
}

// The same greedy with the level bottlenecks taken from the utilisation rows inside the
// base-score pass (see include/netkv.h): the workspace is required, and every launch is
// the workspace form of netkv_schedule_streams, whose walks never read UB.
extern "C" netkv_status netkv_schedule_streams_util(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap, const uint16_t* d_M,
    const float* d_util, uint32_t n_snap, const uint32_t* d_events, const uint64_t* d_event_off,
    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
    int64_t* d_load_final, void* d_workspace, size_t workspace_bytes, int* d_status,
    netkv_stream_t stream) {
  if (!topo || !d_w || !d_event_off || !d_load_final) return NETKV_EINVAL;
  if (n_streams == 0) return NETKV_OK;
  if (n_streams > 0x7fffffffu) return NETKV_EINVAL;
  if (R > 0 && (!d_len || !d_prefill || !d_snap || !d_M || !d_util || !d_dec || !d_best ||
                !d_second || !d_events))
    return NETKV_EINVAL;
  if (!aligned_to(d_w, 8) || !aligned_to(d_event_off, 8) || !aligned_to(d_load_final, 8) ||
      (d_util && !aligned_to(d_util, 4)) || (d_load_init && !aligned_to(d_load_init, 8)))
    return NETKV_EINVAL;
  const TopoArgs t = topo_args(topo);
  const uint32_t D = t.D;
  cudaStream_t s = (cudaStream_t)stream;
  if (!d_workspace || !aligned_to(d_workspace, 256) || workspace_bytes < base_ws_bytes(R, D))
    return NETKV_EINVAL;
  if (R == 0)  // no request: the walk only reports out-of-range events and copies the loads
    return netkv_schedule_streams(topo, n_streams, d_w, 0, d_len, d_prefill, d_snap, d_M,
                                  nullptr, n_snap, d_events, d_event_off, d_load_init, d_dec,
                                  d_best, d_second, d_load_final, nullptr, 0, d_status, stream);
  float* d_base = reinterpret_cast<float*>(d_workspace);
  const ListWs lw = list_ws(d_workspace, workspace_bytes, R, D);
#define NETKV_SCHED_U(NPT, BLOCK, LPS)                                                           \
  return launch<NPT, BLOCK, LPS, true>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M,     \
                                       d_util, n_snap, d_events, d_event_off, d_load_init,      \
                                       d_dec, d_best, d_second, d_load_final, d_base, d_status, \
                                       s, &lw)
  if (D <= 8) NETKV_SCHED_U(1, 32, 8);
  if (D <= 16) NETKV_SCHED_U(1, 32, 16);
  if (D <= 32) NETKV_SCHED_U(1, 32, 32);
  if (D <= 256) NETKV_SCHED_U(1, 256, 32);
  if (D <= 1024) NETKV_SCHED_U(4, 256, 32);
  if (D <= 4096) NETKV_SCHED_U(4, 1024, 32);
#undef NETKV_SCHED_U
  return NETKV_EINVAL;
}

extern "C" size_t netkv_schedule_inflight_workspace_size(uint32_t R, uint32_t D) {
  return 2 * netkv_schedule_workspace_size(R, D);
}

extern "C" netkv_status netkv_schedule_streams_inflight(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap,
    const int64_t* d_arrival_us, const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
    const uint32_t* d_events, const uint64_t* d_event_off, uint32_t inflight_cap,
    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
    int32_t* d_xfer_us, int64_t* d_load_final, void* d_workspace, size_t workspace_bytes,
    int* d_status, netkv_stream_t stream) {
  if (!topo || !d_w || !d_event_off || !d_load_final) return NETKV_EINVAL;
  if (inflight_cap > 255) return NETKV_EINVAL;
  if (n_streams == 0) return NETKV_OK;
  if (n_streams > 0x7fffffffu) return NETKV_EINVAL;
  if (R > 0 && (!d_len || !d_prefill || !d_snap || !d_arrival_us || !d_M || !d_UB || !d_dec ||
                !d_best || !d_second || !d_xfer_us || !d_events))
    return NETKV_EINVAL;
  if (!aligned_to(d_w, 8) || !aligned_to(d_UB, 16) || !aligned_to(d_event_off, 8) ||
      !aligned_to(d_load_final, 8) || (d_load_init && !aligned_to(d_load_init, 8)) ||
      (d_arrival_us && !aligned_to(d_arrival_us, 8)))
    return NETKV_EINVAL;
  const TopoArgs t = topo_args(topo);
  if (t.P >= (1u << 14)) return NETKV_EINVAL;  // prefill rank in a completion key
  const uint32_t D = t.D;
  cudaStream_t s = (cudaStream_t)stream;
  if (d_workspace && (!aligned_to(d_workspace, 256) ||
                      workspace_bytes < netkv_schedule_inflight_workspace_size(R, D)))
    return NETKV_EINVAL;
  float* d_base = (d_workspace && R > 0) ? reinterpret_cast<float*>(d_workspace) : nullptr;
  float* d_X = d_base ? reinterpret_cast<float*>(reinterpret_cast<char*>(d_workspace) +
                                                 netkv_schedule_workspace_size(R, D))
                      : nullptr;
#define NETKV_INFL(NPT, BLOCK, LPS)                                                             \
  return launch_inflight<NPT, BLOCK, LPS>(t, n_streams, d_w, R, d_len, d_prefill, d_snap,      \
                                          d_arrival_us, d_M, d_UB, n_snap, d_events,           \
                                          d_event_off, inflight_cap, d_load_init, d_dec,       \
                                          d_best, d_second, d_xfer_us, d_load_final, d_base,   \
                                          d_X, d_status, s)
  if (D <= 8) NETKV_INFL(1, 32, 8);
  if (D <= 16) NETKV_INFL(1, 32, 16);
  if (D <= 32) NETKV_INFL(1, 32, 32);
  if (D <= 256) NETKV_INFL(1, 256, 32);
  if (D <= 1024) NETKV_INFL(4, 256, 32);
  if (D <= 4096) NETKV_INFL(4, 1024, 32);
#undef NETKV_INFL
  return NETKV_EINVAL;
}

extern "C" netkv_status netkv_schedule_streams_load(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w,
    const netkv_load_model* model, uint32_t R, const uint32_t* d_len, const uint32_t* d_prefill,
    const uint32_t* d_snap, const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
    const uint32_t* d_events, const uint64_t* d_event_off, const int64_t* d_m_init,
    const int32_t* d_n_init, int32_t* d_dec, float* d_best, float* d_second, int64_t* d_m_final,
    int32_t* d_n_final, int* d_status, netkv_stream_t stream) {
  if (!topo || !d_w || !model || !d_event_off || !d_m_final || !d_n_final) return NETKV_EINVAL;
  if (model->beta_max < 1 || !(model->t_a_s >= 0) || !(model->t_b_s >= 0) ||
      !isfinite(model->t_a_s) || !isfinite(model->t_b_s) || model->m_min_bytes < 0)
    return NETKV_EINVAL;
  if (n_streams == 0) return NETKV_OK;
  if (n_streams > 0x7fffffffu) return NETKV_EINVAL;
  if (R > 0 && (!d_len || !d_prefill || !d_snap || !d_M || !d_UB || !d_dec || !d_best ||
                !d_second || !d_events))
    return NETKV_EINVAL;
  if (!aligned_to(d_w, 8) || !aligned_to(d_UB, 16) || !aligned_to(d_event_off, 8) ||
      !aligned_to(d_m_final, 8) || !aligned_to(d_n_final, 4) ||
      (d_m_init && !aligned_to(d_m_init, 8)) || (d_n_init && !aligned_to(d_n_init, 4)))
    return NETKV_EINVAL;
  const TopoArgs t = topo_args(topo);
  const uint32_t D = t.D;
  cudaStream_t s = (cudaStream_t)stream;
  const LoadModel lm = {model->t_a_s, model->t_b_s, model->beta_max, model->m_min_bytes,
                        model->m0_bytes};
#define NETKV_LOAD(NPT, BLOCK, LPS)                                                             \
  do {                                                                                          \
    const uint32_t per_cta = LPS == 32 ? 1u : 32u / LPS;                                        \
    schedule_kernel<NPT, BLOCK, LPS, false, false, true>                                        \
        <<<(n_streams + per_cta - 1) / per_cta, BLOCK, 0, s>>>(                                 \
            t, n_streams, d_w, R, nullptr, d_len, d_prefill, d_snap, d_M, d_UB, n_snap,         \
            d_events, d_event_off, d_m_init, d_dec, d_best, d_second, d_m_final, d_status,      \
            nullptr, 0u, nullptr, 0u, 0u, lm, d_n_init, d_n_final);                             \
    return netkv_launch_status();                                                               \
  } while (0)
  if (D <= 8) NETKV_LOAD(1, 32, 8);
  if (D <= 16) NETKV_LOAD(1, 32, 16);
  if (D <= 32) NETKV_LOAD(1, 32, 32);
  if (D <= 256) NETKV_LOAD(1, 256, 32);
  if (D <= 1024) NETKV_LOAD(4, 256, 32);
  if (D <= 4096) NETKV_LOAD(4, 1024, 32);
#undef NETKV_LOAD
  return NETKV_EINVAL;
}
