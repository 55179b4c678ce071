// The greedy of Algorithm 1 (Sec. V-A) with evolving decode caches: the LRU-managed
// KV-block caches of the simulator of Sec. VI-B.  Each arrival's prefix hits are taken
// against the caches as they are at that arrival, and a dispatch brings the request's
// chain into the chosen decode's cache as its most recently used blocks (from the last
// block to the first, so that block 0 is the most recent), evicting the least recently
// used blocks beyond the cache's capacity.
//
// State of one cache (a decode of a stream), in caller-owned memory:
//   recency log   2^log2_ring block hashes; every use of a block appends it at the next
//                 position (positions only grow; entry p sits at p mod 2^log2_ring)
//   hash table    2^log2_slots slots {hash, latest position of the hash in the log}
//   header        head (the oldest position still in the cache), tail (the next
//                 position), live blocks, occupied slots
// A block is cached iff its latest position is at least head, and a use zeroes the log
// entry it supersedes, so the non-zero entries of the window [head, tail) are exactly the
// cached blocks at their latest uses:
//   lookup    one probe of the table and a comparison with head;
//   use       append at tail, raise the slot's position (atomicMax, so a hash that occurs
//             twice in a chain keeps its later use) and zero the superseded entry;
//   evict     advance head past as many non-zero entries as blocks to evict (a coalesced
//             scan of the log, no lookups).
// The table keeps evicted hashes (with old positions) until the log or the table fills;
// then the cache is rebuilt in place: the non-zero entries are packed in order from head
// and the table is rebuilt from them.
//
// One CTA per stream walks the stream's events in order:
//   departure  the lead thread returns the request's tokens to its decode's load;
//   arrival    warps take decodes and find the first miss of the chain by following the
//              runs the chain's blocks form in the log (32 blocks a step); threads
//              take decodes and score them exactly as netkv_schedule_streams does without
//              a workspace (base score + w_load * theta * load), then a block-wide
//              (score, index) argmin; every thread then uses its share of the chain's
//              blocks on the chosen cache, and the CTA evicts in chunks of 256 log
//              entries with a block scan over their liveness.
#include <math.h>

#include "score.cuh"

namespace {

constexpr int kEvoBlock = 256;
constexpr int kEvoWarps = kEvoBlock / 32;
constexpr int kLruBlock = 1024;
constexpr uint64_t kMaxChain = 65535;
constexpr uint64_t kHeaderBytes = 64;
constexpr uint32_t kNoDecode = 0xffffffffu;

struct __align__(16) LruSlot {
  unsigned long long key;  // block hash; 0 marks an empty slot
  unsigned long long pos;  // latest log position of the hash; 0 = none
};

struct LruHeader {
  unsigned long long head, tail, live, n_keys;
};

struct LruGeom {
  uint32_t log2_slots, log2_ring;
  unsigned long long cap_blocks;   // blocks a cache keeps
  unsigned long long max_keys;     // occupied slots allowed before a rebuild
  unsigned long long cache_bytes;  // bytes of one cache's state
};

__host__ __device__ inline unsigned long long lru_cache_bytes(uint32_t ls, uint32_t lr) {
  return kHeaderBytes + (16ull << ls) + (8ull << lr);
}

__device__ __forceinline__ char* lru_base(void* state, const LruGeom& g, uint64_t c) {
  return reinterpret_cast<char*>(state) + c * g.cache_bytes;
}
__device__ __forceinline__ LruHeader* lru_header(void* state, const LruGeom& g, uint64_t c) {
  return reinterpret_cast<LruHeader*>(lru_base(state, g, c));
}
__device__ __forceinline__ LruSlot* lru_slots(void* state, const LruGeom& g, uint64_t c) {
  return reinterpret_cast<LruSlot*>(lru_base(state, g, c) + kHeaderBytes);
}
__device__ __forceinline__ unsigned long long* lru_ring(void* state, const LruGeom& g,
                                                        uint64_t c) {
  return reinterpret_cast<unsigned long long*>(lru_base(state, g, c) + kHeaderBytes +
                                               (16ull << g.log2_slots));
}

// Table and log entries change during a kernel (atomics, in-place rebuilds), so they are
// read with volatile loads, never through the read-only path.
__device__ __forceinline__ unsigned long long vload(const unsigned long long* p) {
  return *reinterpret_cast<const volatile unsigned long long*>(p);
}

// Latest log position of `key` (non-zero) in a cache's table; 0 when the key is absent.
__device__ __forceinline__ unsigned long long lru_find(const LruSlot* T, uint32_t ls,
                                                       unsigned long long key, int* status) {
  const unsigned long long mask = (1ull << ls) - 1;
  unsigned long long s = home_slot(key, ls);
  for (unsigned long long i = 0; i <= mask; ++i) {
    const unsigned long long k = vload(&T[s].key);
    if (k == key) return vload(&T[s].pos);
    if (k == 0ull) return 0ull;
    s = (s + 1) & mask;
  }
  flag_status(status, NETKV_DEV_EFULL);
  return 0ull;
}

// The slot of `key` (non-zero), claimed when the key is absent (fresh: claimed here).
__device__ __forceinline__ LruSlot* lru_claim(LruSlot* T, uint32_t ls, unsigned long long key,
                                              bool& fresh, int* status) {
  fresh = false;
  const unsigned long long mask = (1ull << ls) - 1;
  unsigned long long s = home_slot(key, ls);
  for (unsigned long long i = 0; i <= mask; ++i) {
    const unsigned long long k = vload(&T[s].key);
    if (k == key) return &T[s];
    if (k == 0ull) {
      const unsigned long long prev = atomicCAS(&T[s].key, 0ull, key);
      if (prev == 0ull) {
        fresh = true;
        return &T[s];
      }
      if (prev == key) return &T[s];
    }
    s = (s + 1) & mask;
  }
  flag_status(status, NETKV_DEV_EFULL);
  return nullptr;
}

// Exclusive prefix count of one flag per thread over a CTA of BLOCK threads; the total
// goes to every thread.  Contains two block barriers.
template <int BLOCK>
__device__ __forceinline__ uint32_t block_count(bool flag, uint32_t* warp_buf, uint32_t& total) {
  constexpr int NW = BLOCK / 32;
  const uint32_t lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const uint32_t b = __ballot_sync(0xffffffffu, flag);
  const uint32_t in_warp = __popc(b & ((1u << lane) - 1));
  if (lane == 0) warp_buf[wid] = __popc(b);
  __syncthreads();
  uint32_t before = 0, sum = 0;
#pragma unroll
  for (int i = 0; i < NW; ++i) {
    const uint32_t v = warp_buf[i];
    before += (uint32_t)i < wid ? v : 0u;
    sum += v;
  }
  __syncthreads();
  total = sum;
  return before + in_warp;
}

// Record that log position p (already holding `key`) is the latest use of the key: raise
// the slot's position and zero the superseded log entry, which is p itself when a later
// use of the key in the same pass got there first, else the key's previous entry when it
// lies in the log window [head, tail).  So the non-zero entries of the window are exactly
// the cached blocks, each at its latest use.  Counts claimed slots and keys that were not
// cached before.
__device__ __forceinline__ void lru_use(LruSlot* T, unsigned long long* ring, const LruGeom& g,
                                        unsigned long long key, unsigned long long p,
                                        unsigned long long head, unsigned int* fresh_cnt,
                                        unsigned int* live_cnt, int* status) {
  const unsigned long long qmask = (1ull << g.log2_ring) - 1;
  bool fresh;
  LruSlot* slot = lru_claim(T, g.log2_slots, key, fresh, status);
  if (!slot) {  // not indexed (a full table, flagged): the entry does not count as cached
    ring[p & qmask] = 0ull;
    return;
  }
  const unsigned long long old = atomicMax(&slot->pos, p);
  if (fresh) atomicAdd(fresh_cnt, 1u);
  if (old > p) {
    ring[p & qmask] = 0ull;
  } else if (old >= head) {
    ring[old & qmask] = 0ull;
  } else {
    atomicAdd(live_cnt, 1u);
  }
}

// Leading chain blocks cached in one cache: the first miss among blocks [0, n), found by
// one warp.  The blocks of a chain that entered the cache together sit in the log as one
// run in reverse order (block j at the run's start position minus j), so the warp looks a
// block up in the table once and then compares 32 chain blocks with the 32 log entries
// below its position per step (coalesced), looking up again only where chain and log part.
// A log entry in the window that holds the block's hash is its latest use (the others
// are zero), so a match there is a cached block.
__device__ __forceinline__ uint32_t lru_match(const LruSlot* T, const unsigned long long* ring,
                                              const LruGeom& g, unsigned long long head,
                                              const uint64_t* __restrict__ chain, uint32_t n,
                                              uint32_t lane, int* status) {
  const unsigned long long qmask = (1ull << g.log2_ring) - 1;
  uint32_t p = 0;
  unsigned long long rp = 0;  // log position of block p within the current run
  bool in_run = false;
  while (p < n) {
    const bool looked_up = !in_run;
    if (!in_run) {  // look block p up in the table
      unsigned long long pos = 0ull;
      if (lane == 0) {
        const unsigned long long key = __ldg(chain + p);
        if (key != 0ull) pos = lru_find(T, g.log2_slots, key, status);
      }
      pos = __shfl_sync(0xffffffffu, pos, 0);
      if (pos == 0ull || pos < head) return p;  // absent or evicted
      rp = pos;
      in_run = true;
    }
    const uint32_t j = p + lane;
    bool same = false;
    if (j < n && rp >= head && (unsigned long long)lane <= rp - head) {
      const unsigned long long ck = __ldg(chain + j);
      same = ck != 0ull && vload(ring + ((rp - lane) & qmask)) == ck;
    }
    const uint32_t ok = __ballot_sync(0xffffffffu, same);
    const uint32_t lead = ~ok ? (uint32_t)(__ffs(~ok) - 1) : 32u;
    if (lead == 0) {
      if (looked_up) {  // the table's latest position does not hold the hash: inconsistent
        if (lane == 0) flag_status(status, NETKV_DEV_EFULL);
        return p;
      }
      in_run = false;  // the run ended with the last step: look block p up
      continue;
    }
    p += lead;
    rp -= lead;
    if (lead < 32) in_run = false;
  }
  return n;
}

// (score, index) order with the runner-up carried along: lower score first, then lower
// decode rank (Algorithm 1 line 13).
__device__ __forceinline__ void take(float& b, uint32_t& i, float& s, float b2, uint32_t i2,
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
__device__ __forceinline__ void warp_take(float& b, uint32_t& i, float& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float b2 = __shfl_xor_sync(0xffffffffu, b, o);
    const uint32_t i2 = __shfl_xor_sync(0xffffffffu, i, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    take(b, i, s, b2, i2, s2);
  }
}

// Evict the `excess` least recently used blocks of a cache: advance head past that many
// non-zero log entries (a coalesced scan of the log).  CTA-wide.
__device__ void lru_evict(const unsigned long long* ring, const LruGeom& g,
                          unsigned long long& head, unsigned long long tail,
                          unsigned long long excess, uint32_t* warp_buf,
                          unsigned long long* s_newhead, int* status) {
  const unsigned long long qmask = (1ull << g.log2_ring) - 1;
  unsigned long long p = head;
  while (excess > 0) {
    if (p >= tail) {  // fewer cached blocks than the header counts: an inconsistent state
      if (threadIdx.x == 0) flag_status(status, NETKV_DEV_EFULL);
      break;
    }
    const unsigned long long i = p + threadIdx.x;
    const bool live = i < tail && vload(ring + (i & qmask)) != 0ull;
    uint32_t total;
    const uint32_t before = block_count<kEvoBlock>(live, warp_buf, total);
    if ((unsigned long long)total >= excess) {
      if (live && before + 1 == excess) *s_newhead = i + 1;
      __syncthreads();
      p = *s_newhead;
      __syncthreads();
      excess = 0;
    } else {
      excess -= total;
      p += kEvoBlock;
    }
  }
  head = p;
}

// Rebuild a cache in place: pack the non-zero log entries of [head, tail) in order from
// head, then clear the table and insert them at their new positions.  Returns the number
// kept (the cached blocks).  CTA-wide.
template <int BLOCK>
__device__ unsigned long long lru_rebuild(LruSlot* T, unsigned long long* ring, const LruGeom& g,
                                          unsigned long long head, unsigned long long tail,
                                          uint32_t* warp_buf, int* status) {
  const unsigned long long qmask = (1ull << g.log2_ring) - 1;
  unsigned long long kept = 0;
  for (unsigned long long p = head; p < tail; p += BLOCK) {
    const unsigned long long i = p + threadIdx.x;
    const unsigned long long key = i < tail ? vload(ring + (i & qmask)) : 0ull;
    uint32_t total;
    const uint32_t before = block_count<BLOCK>(key != 0ull, warp_buf, total);  // reads done
    // the write position never passes the entry's own: entries are only moved down
    if (key != 0ull) ring[(head + kept + before) & qmask] = key;
    kept += total;
    __syncthreads();
  }
  const unsigned long long n_slots = 1ull << g.log2_slots;
  for (unsigned long long s = threadIdx.x; s < n_slots; s += BLOCK)
    reinterpret_cast<ulonglong2*>(T)[s] = make_ulonglong2(0ull, 0ull);
  __syncthreads();
  for (unsigned long long i = threadIdx.x; i < kept; i += BLOCK) {
    const unsigned long long key = vload(ring + ((head + i) & qmask));
    bool fresh;
    LruSlot* slot = lru_claim(T, g.log2_slots, key, fresh, status);
    if (slot) atomicMax(&slot->pos, head + i);
  }
  __syncthreads();
  return kept;
}

// Initial state of every cache from its key list (most recently used block first): entry
// j of a list of K blocks is used at position K - j, so the list's first block is the
// most recent.  One CTA per cache.
__global__ void __launch_bounds__(kLruBlock) lru_init_kernel(void* state, LruGeom g,
                                                            uint64_t n_caches,
                                                            const uint64_t* __restrict__ keys,
                                                            const uint64_t* __restrict__ key_off,
                                                            int* status) {
  __shared__ unsigned int s_fresh, s_live;
  const unsigned long long qmask = (1ull << g.log2_ring) - 1;
  const unsigned long long n_slots = 1ull << g.log2_slots;
  for (uint64_t c = blockIdx.x; c < n_caches; c += gridDim.x) {
    LruSlot* T = lru_slots(state, g, c);
    unsigned long long* ring = lru_ring(state, g, c);
    for (unsigned long long s = threadIdx.x; s < n_slots; s += kLruBlock)
      reinterpret_cast<ulonglong2*>(T)[s] = make_ulonglong2(0ull, 0ull);
    if (threadIdx.x == 0) {
      s_fresh = 0;
      s_live = 0;
    }
    __syncthreads();
    uint64_t beg = 0, K = 0;
    if (keys) {
      beg = __ldg(key_off + c);
      const uint64_t end = __ldg(key_off + c + 1);
      if (end < beg) {
        if (threadIdx.x == 0) flag_status(status, NETKV_DEV_ERANGE);
      } else {
        K = end - beg;
      }
      if (K > g.cap_blocks) {  // a list longer than the capacity: keep its first entries
        if (threadIdx.x == 0) flag_status(status, NETKV_DEV_ERANGE);
        K = g.cap_blocks;
      }
    }
    for (uint64_t j = threadIdx.x; j < K; j += kLruBlock) {
      const unsigned long long key = __ldg(keys + beg + j);
      ring[(K - j) & qmask] = key;
      if (key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
    }
    __syncthreads();  // every entry is written before any is zeroed as superseded
    for (uint64_t j = threadIdx.x; j < K; j += kLruBlock) {
      const unsigned long long key = __ldg(keys + beg + j);
      if (key != 0ull) lru_use(T, ring, g, key, K - j, 1ull, &s_fresh, &s_live, status);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      LruHeader* h = lru_header(state, g, c);
      h->head = 1;
      h->tail = K + 1;
      h->live = s_live;
      h->n_keys = s_fresh;
    }
    __syncthreads();
  }
}

// Every cache's blocks from the most to the least recently used: out[c][0 .. len[c]).
__global__ void __launch_bounds__(kLruBlock) lru_export_kernel(const void* state, LruGeom g,
                                                              uint64_t n_caches,
                                                              unsigned long long* out,
                                                              unsigned long long* out_len,
                                                              int* status) {
  __shared__ uint32_t warp_buf[kLruBlock / 32];
  const unsigned long long qmask = (1ull << g.log2_ring) - 1;
  void* st = const_cast<void*>(state);
  for (uint64_t c = blockIdx.x; c < n_caches; c += gridDim.x) {
    const LruHeader* h = lru_header(st, g, c);
    const unsigned long long head = vload(&h->head), tail = vload(&h->tail);
    const LruSlot* T = lru_slots(st, g, c);
    const unsigned long long* ring = lru_ring(st, g, c);
    unsigned long long* o = out + c * g.cap_blocks;
    unsigned long long w = 0;
    for (unsigned long long top = tail; top > head;) {
      const unsigned long long chunk = top - head < kLruBlock ? top - head : kLruBlock;
      bool live = false;
      unsigned long long key = 0ull;
      if (threadIdx.x < chunk) {
        const unsigned long long i = top - 1 - threadIdx.x;  // newest first
        key = vload(ring + (i & qmask));
        live = key != 0ull;  // the window's non-zero entries are the cached blocks
      }
      uint32_t total;
      const uint32_t before = block_count<kLruBlock>(live, warp_buf, total);
      if (live && w + before < g.cap_blocks) o[w + before] = key;
      w += total;
      top -= chunk;
    }
    if (threadIdx.x == 0) {
      if (w > g.cap_blocks) flag_status(status, NETKV_DEV_EFULL);
      out_len[c] = w < g.cap_blocks ? w : g.cap_blocks;
    }
    __syncthreads();
  }
}

__global__ void __launch_bounds__(kEvoBlock) evolving_kernel(
    TopoArgs t, uint32_t n_streams, const netkv_weights* __restrict__ W, uint32_t R,
    const uint32_t* __restrict__ len, const uint32_t* __restrict__ prefill,
    const uint32_t* __restrict__ snap, const float* __restrict__ UB, uint32_t n_snap,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off,
    const uint32_t* __restrict__ events, const uint64_t* __restrict__ event_off, void* state,
    LruGeom g, const int64_t* __restrict__ load_init, int32_t* dec, float* __restrict__ best,
    float* __restrict__ second, uint16_t* __restrict__ M, int64_t* __restrict__ load_final,
    int* status) {
  extern __shared__ __align__(16) unsigned char evo_smem[];
  __shared__ uint32_t warp_buf[kEvoWarps];
  __shared__ float s_b[kEvoWarps], s_s[kEvoWarps];
  __shared__ uint32_t s_i[kEvoWarps];
  __shared__ int32_t s_dstar;
  __shared__ unsigned int s_cnt[2];  // fresh slots, newly cached blocks
  __shared__ unsigned long long s_newhead;
  const uint32_t D = t.D, N = t.N;
  unsigned long long* s_head = reinterpret_cast<unsigned long long*>(evo_smem);
  unsigned long long* s_tail = s_head + D;
  unsigned long long* s_live = s_tail + D;
  unsigned long long* s_keys = s_live + D;
  long long* s_load = reinterpret_cast<long long*>(s_keys + D);
  uint32_t* s_m = reinterpret_cast<uint32_t*>(s_load + D);
  const uint32_t stream = blockIdx.x;
  if (stream >= n_streams) return;
  const uint32_t tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const unsigned long long qmask = (1ull << g.log2_ring) - 1;
  const unsigned long long Q = 1ull << g.log2_ring;
  const uint64_t c0_cache = (uint64_t)stream * D;
  for (uint32_t d = tid; d < D; d += kEvoBlock) {
    const LruHeader* h = lru_header(state, g, c0_cache + d);
    s_head[d] = vload(&h->head);
    s_tail[d] = vload(&h->tail);
    s_live[d] = vload(&h->live);
    s_keys[d] = vload(&h->n_keys);
    s_load[d] = load_init ? load_init[c0_cache + d] : 0;
  }
  __syncthreads();
  const netkv_weights w = W[stream];
  const float4 lat = make_float4(t.lat[0], t.lat[1], t.lat[2], t.lat[3]);
  const float inf = __int_as_float(0x7f800000);
  const uint64_t e0 = event_off[stream], e1 = event_off[stream + 1];

  for (uint64_t e = e0; e < e1; ++e) {
    const uint32_t code = __ldg(events + e);
    const uint32_t r = code & 0x7fffffffu;
    if (r >= R) {
      if (tid == 0) flag_status(status, NETKV_DEV_ERANGE);
      continue;
    }
    if (code >> 31) {  // departure: the lead thread returns the tokens
      if (tid == 0) {
        const int32_t dd = *reinterpret_cast<const volatile int32_t*>(dec + r);
        if (dd >= 0 && (uint32_t)dd < D) s_load[dd] -= (long long)__ldg(len + r);
      }
      continue;
    }
    const uint32_t l = __ldg(len + r), pr = __ldg(prefill + r), k = __ldg(snap + r);
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    if (pr >= t.P || k >= n_snap || l == 0 || c1 < c0) {
      if (tid == 0) {
        flag_status(status, l == 0 ? NETKV_DEV_EDOMAIN : NETKV_DEV_ERANGE);
        best[r] = inf;
        second[r] = inf;
        dec[r] = -1;
      }
      for (uint32_t d = tid; d < D; d += kEvoBlock) M[(uint64_t)r * D + d] = 0;
      __syncthreads();
      continue;
    }
    uint64_t n = c1 - c0;
    if (n > kMaxChain) {
      if (tid == 0) flag_status(status, NETKV_DEV_EDOMAIN);
      n = kMaxChain;
    }
    const uint64_t* chain = chains + c0;

    // hits against the caches as they are now (Sec. III-B first-miss scan)
    for (uint32_t d = wid; d < D; d += kEvoWarps) {
      const uint32_t m = lru_match(lru_slots(state, g, c0_cache + d), lru_ring(state, g, c0_cache + d),
                                   g, s_head[d], chain, (uint32_t)n, lane, status);
      if (lane == 0) {
        s_m[d] = m;
        M[(uint64_t)r * D + d] = (uint16_t)m;
      }
    }
    if (tid == 0) {
      s_cnt[0] = 0;
      s_cnt[1] = 0;
    }
    __syncthreads();

    // scores over the feasible decodes and the lowest-index argmin (lines 1-13)
    const uint32_t pinst = __ldg(t.pre + pr);
    const uint4 lp = __ldg(t.links + pinst);
    const float4 ubp = __ldg(reinterpret_cast<const float4*>(UB) + (uint64_t)k * N + pinst);
    const float* ub_row = UB + (uint64_t)k * N * 4;
    float b = inf, s2 = inf;
    uint32_t bi = kNoDecode;
    for (uint32_t d = tid; d < D; d += kEvoBlock) {
      const uint4 ld = __ldg(t.links + __ldg(t.dec + d));
      const int tau = tier_of(lp, ld);
      const float ubd = __ldg(ub_row + (uint64_t)ld.x * 4 + tau);
      const long long load = s_load[d];
      if (load + (long long)l <= w.cap_tokens) {
        const float sc = base_score(w, l, s_m[d], pick4(ubp, tau), ubd, pick4(lat, tau), status) +
                         w.w_load * (w.theta_s_per_token * (float)load);
        take(b, bi, s2, sc, d, inf);
      }
    }
    warp_take(b, bi, s2);
    if (lane == 0) {
      s_b[wid] = b;
      s_i[wid] = bi;
      s_s[wid] = s2;
    }
    __syncthreads();
    if (wid == 0) {
      b = lane < (uint32_t)kEvoWarps ? s_b[lane] : inf;
      bi = lane < (uint32_t)kEvoWarps ? s_i[lane] : kNoDecode;
      s2 = lane < (uint32_t)kEvoWarps ? s_s[lane] : inf;
      warp_take(b, bi, s2);
      if (lane == 0) {
        const int32_t dstar = bi == kNoDecode ? -1 : (int32_t)bi;
        dec[r] = dstar;
        best[r] = b;
        second[r] = s2;
        if (dstar >= 0) s_load[dstar] += (long long)l;
        s_dstar = dstar;
      }
    }
    __syncthreads();
    const int32_t dstar = s_dstar;
    if (dstar < 0) continue;

    // the chain enters the chosen cache as its most recently used blocks
    const uint64_t cc = c0_cache + (uint32_t)dstar;
    LruSlot* T = lru_slots(state, g, cc);
    unsigned long long* ring = lru_ring(state, g, cc);
    if (s_tail[dstar] - s_head[dstar] + n > Q || s_keys[dstar] + n > g.max_keys) {
      const unsigned long long kept = lru_rebuild<kEvoBlock>(T, ring, g, s_head[dstar],
                                                             s_tail[dstar], warp_buf, status);
      if (tid == 0) {
        s_tail[dstar] = s_head[dstar] + kept;
        s_keys[dstar] = kept;
        s_live[dstar] = kept;
      }
      __syncthreads();
    }
    const unsigned long long P0 = s_tail[dstar], head = s_head[dstar];
    for (uint64_t j = tid; j < n; j += kEvoBlock) {  // block j is used at P0 + n - 1 - j
      const unsigned long long key = __ldg(chain + j);
      ring[(P0 + (n - 1 - j)) & qmask] = key;
      if (key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
    }
    __syncthreads();  // every entry is written before any is zeroed as superseded
    for (uint64_t j = tid; j < n; j += kEvoBlock) {
      const unsigned long long key = __ldg(chain + j);
      if (key != 0ull) lru_use(T, ring, g, key, P0 + (n - 1 - j), head, &s_cnt[0], &s_cnt[1], status);
    }
    __syncthreads();
    const unsigned long long tail = P0 + n;
    const unsigned long long live = s_live[dstar] + s_cnt[1];
    if (live > g.cap_blocks) {
      unsigned long long hd = head;
      lru_evict(ring, g, hd, tail, live - g.cap_blocks, warp_buf, &s_newhead, status);
      __syncthreads();
      if (tid == 0) {
        s_head[dstar] = hd;
        s_live[dstar] = g.cap_blocks;
      }
    } else if (tid == 0) {
      s_live[dstar] = live;
    }
    if (tid == 0) {
      s_tail[dstar] = tail;
      s_keys[dstar] += s_cnt[0];
    }
    __syncthreads();
  }
  __syncthreads();  // the lead thread's last departures are in s_load
  for (uint32_t d = tid; d < D; d += kEvoBlock) {
    LruHeader* h = lru_header(state, g, c0_cache + d);
    h->head = s_head[d];
    h->tail = s_tail[d];
    h->live = s_live[d];
    h->n_keys = s_keys[d];
    load_final[c0_cache + d] = s_load[d];
  }
}

bool lru_geom(const netkv_lru_config* cfg, LruGeom& g) {
  if (!cfg || cfg->cap_blocks < 1 || cfg->log2_slots < 4 || cfg->log2_slots > 31 ||
      cfg->log2_ring < 4 || cfg->log2_ring > 40)
    return false;
  g.log2_slots = cfg->log2_slots;
  g.log2_ring = cfg->log2_ring;
  g.cap_blocks = cfg->cap_blocks;
  g.max_keys = (3ull << cfg->log2_slots) / 4;
  g.cache_bytes = lru_cache_bytes(cfg->log2_slots, cfg->log2_ring);
  // after a rebuild the cache holds at most cap_blocks entries, and one chain must fit
  if ((1ull << cfg->log2_ring) < cfg->cap_blocks + kMaxChain + 1) return false;
  if (g.max_keys < cfg->cap_blocks + kMaxChain) return false;
  return true;
}

unsigned cache_grid(uint64_t n_caches) {
  return (unsigned)(n_caches < (1u << 20) ? n_caches : (1u << 20));
}

}  // namespace

extern "C" size_t netkv_lru_state_bytes(uint64_t n_caches, const netkv_lru_config* cfg) {
  LruGeom g;
  if (!lru_geom(cfg, g)) return 0;
  return (size_t)(n_caches * g.cache_bytes);
}

extern "C" netkv_status netkv_lru_init(void* d_state, size_t state_bytes, uint64_t n_caches,
                                       const netkv_lru_config* cfg, const uint64_t* d_keys,
                                       const uint64_t* d_key_off, int* d_status,
                                       netkv_stream_t stream) {
  LruGeom g;
  if (!d_state || !lru_geom(cfg, g) || (d_keys && !d_key_off)) return NETKV_EINVAL;
  if (state_bytes / g.cache_bytes < n_caches) return NETKV_EINVAL;
  if (!aligned_to(d_state, 16) || (d_keys && !aligned_to(d_keys, 8)) ||
      (d_key_off && !aligned_to(d_key_off, 8)))
    return NETKV_EINVAL;
  if (n_caches == 0) return NETKV_OK;
  lru_init_kernel<<<cache_grid(n_caches), kLruBlock, 0, (cudaStream_t)stream>>>(
      d_state, g, n_caches, d_keys, d_key_off, d_status);
  return netkv_launch_status();
}

extern "C" netkv_status netkv_lru_export(const void* d_state, size_t state_bytes,
                                         uint64_t n_caches, const netkv_lru_config* cfg,
                                         uint64_t* d_keys_out, uint64_t* d_len_out, int* d_status,
                                         netkv_stream_t stream) {
  LruGeom g;
  if (!d_state || !d_keys_out || !d_len_out || !lru_geom(cfg, g)) return NETKV_EINVAL;
  if (state_bytes / g.cache_bytes < n_caches) return NETKV_EINVAL;
  if (!aligned_to(d_state, 16) || !aligned_to(d_keys_out, 8) || !aligned_to(d_len_out, 8))
    return NETKV_EINVAL;
  if (n_caches == 0) return NETKV_OK;
  lru_export_kernel<<<cache_grid(n_caches), kLruBlock, 0, (cudaStream_t)stream>>>(
      d_state, g, n_caches, reinterpret_cast<unsigned long long*>(d_keys_out),
      reinterpret_cast<unsigned long long*>(d_len_out), d_status);
  return netkv_launch_status();
}

extern "C" netkv_status netkv_schedule_streams_evolving(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap, const float* d_UB,
    uint32_t n_snap, const uint64_t* d_chains, const uint64_t* d_chain_off,
    const uint32_t* d_events, const uint64_t* d_event_off, void* d_state, size_t state_bytes,
    const netkv_lru_config* cfg, const int64_t* d_load_init, int32_t* d_dec, float* d_best,
    float* d_second, uint16_t* d_M, int64_t* d_load_final, int* d_status,
    netkv_stream_t stream) {
  LruGeom g;
  if (!topo || !d_w || !d_event_off || !d_load_final || !d_state || !lru_geom(cfg, g))
    return NETKV_EINVAL;
  if (n_streams == 0) return NETKV_OK;
  if (n_streams > 0x7fffffffu) return NETKV_EINVAL;
  if (R > 0 && (!d_len || !d_prefill || !d_snap || !d_UB || !d_chains || !d_chain_off ||
                !d_events || !d_dec || !d_best || !d_second || !d_M))
    return NETKV_EINVAL;
  if (!aligned_to(d_w, 8) || !aligned_to(d_UB, 16) || !aligned_to(d_event_off, 8) ||
      !aligned_to(d_load_final, 8) || !aligned_to(d_state, 16) ||
      (d_load_init && !aligned_to(d_load_init, 8)) || (d_chains && !aligned_to(d_chains, 8)) ||
      (d_chain_off && !aligned_to(d_chain_off, 8)) || (d_M && !aligned_to(d_M, 2)))
    return NETKV_EINVAL;
  const TopoArgs t = topo_args(topo);
  if (t.D > 1024) return NETKV_EINVAL;
  if (state_bytes / g.cache_bytes < (uint64_t)n_streams * t.D) return NETKV_EINVAL;
  const size_t smem = (size_t)t.D * (4 * 8 + 8 + 4);
  evolving_kernel<<<n_streams, kEvoBlock, smem, (cudaStream_t)stream>>>(
      t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_UB, n_snap, d_chains, d_chain_off,
      d_events, d_event_off, d_state, g, d_load_init, d_dec, d_best, d_second, d_M,
      d_load_final, d_status);
  return netkv_launch_status();
}
