// Decode caches K_d and the block-level prefix hit of Sec. III-B:
// M[r][d] = |LCP_block(h_r, K_d)|, the number of leading blocks of request r's hash chain
// that are all cached on decode d.
//
// Cache index.  The caches of a table set are indexed per group of up to 64 decodes:
//   run keys    the group's distinct cached hashes in the order the key lists give them
//               (decode by decode, first appearance);
//   run masks   beside each run key, the mask of the group's decodes that cache it, in
//               1, 2, 4 or 8 bytes by the pool's size;
//   hash table  open addressing, 16-byte slots {hash, position in the run array}.
// Caches are filled with whole prefixes of chains, so a cached prefix sits in the run
// array as a contiguous run in chain order.
//   cache_build_kernel: one CTA per index; it walks the lists in order in chunks of 1024
//   keys, claims new hashes with atomicCAS, numbers them with a block-wide scan and
//   appends them to the run array, and ORs each decode's bit into the hashes it lists.
//
// Match.  One warp per (request, decode group).  The warp looks up the block at the
// current position in the hash table (one random access), then compares the chain with
// the run keys from that position on, 32 blocks per step (coalesced loads of 256 chain
// bytes, 256 key bytes and 32 .. 256 mask bytes): every block that equals the next run key
// is cached exactly on the decodes of that position's mask, and one ballot per live decode
// finds its first missing block.  Where chain and run part, the next block is looked up
// in the hash table again; a block absent from the table is missing on every decode.
// The answer never depends on the run order (any key order is exact); the order only
// decides how many random lookups a chain needs.  A decode leaves once its first miss is
// known and the warp stops when every decode of the group has missed.
//
// Prefix sharing.  Requests that share leading blocks have the same membership answers
// on those blocks, so with a workspace the match runs in three steps:
//   group_insert_kernel / group_resolve_kernel: requests are grouped by (table set,
//     first block hash) in an open-addressing table; each group's leader is its
//     longest chain (lowest index among equals); leaders go to a compact list (chains of
//     2,048 blocks or more first), and each member gets a record of its own and its
//     leader's chain offsets and lengths.
//   match_leaders_kernel: leaders (and ungrouped requests) run the full match, one task
//     per (leader, decode group) taken in order from a counter.
//   match_members_kernel: a member r with leader L compares chains to get
//     lcp = |common prefix of h_r and h_L| (capped at max_d M_L[d] + 1).  For a decode
//     with M_L[d] < lcp the first missing block of L lies inside the common prefix, so
//     M_r[d] = M_L[d] exactly; otherwise blocks [0, lcp) are all cached and the walk
//     resumes at block lcp.  The result equals the full match whatever the grouping.
//   match_members_wide_kernel: the same for pools of more than one decode group, one
//     warp per member: the common prefix is read once, the member's row is
//     min(M_L, lcp) elementwise, and block lcp is probed only in the groups where a
//     leader hit reaches lcp, up to 32 groups at a time.
#include "cache_index.cuh"

namespace {

constexpr int kBuildBlock = 1024;
constexpr int kMatchBlock = 256;
// Exclusive scan of one flag per thread over a 1024-thread block; returns the prefix and
// writes the block total to *total (shared).
__device__ __forceinline__ uint32_t block_scan(uint32_t flag, uint32_t* warp_sums,
                                               uint32_t* total) {
  const uint32_t lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const uint32_t b = __ballot_sync(0xffffffffu, flag);
  const uint32_t in_warp = __popc(b & ((1u << lane) - 1));
  if (lane == 0) warp_sums[wid] = __popc(b);
  __syncthreads();
  if (wid == 0) {
    const uint32_t v = warp_sums[lane];
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= (uint32_t)o) x += y;
    }
    warp_sums[lane] = x - v;  // exclusive
    if (lane == 31) *total = x;
  }
  __syncthreads();
  return warp_sums[wid] + in_warp;
}

__global__ void __launch_bounds__(kBuildBlock) cache_build_kernel(
    void* __restrict__ index, uint32_t n_sets, uint32_t D, uint32_t log2_cap,
    const uint64_t* __restrict__ keys, const uint64_t* __restrict__ key_off, int* status) {
  __shared__ uint32_t warp_sums[32];
  __shared__ uint32_t chunk_new;
  const uint64_t cap = 1ull << log2_cap, mask = cap - 1;
  const uint32_t n_dgroups = (D + kGroup - 1) / kGroup;
  const uint32_t mb = mask_bytes_of(D);
  const uint64_t n_index = (uint64_t)n_sets * n_dgroups;
  for (uint64_t idx = blockIdx.x; idx < n_index; idx += gridDim.x) {
    const uint64_t g = idx / n_dgroups;
    const uint32_t q = (uint32_t)(idx - g * n_dgroups);
    const IndexView v = index_view(index, idx, log2_cap, mb);
    IndexSlot* hash = v.hash;
    uint32_t run_len = 0;  // same value in every thread
    for (uint32_t d = q * kGroup; d < min(D, (q + 1) * kGroup); ++d) {
      const uint64_t t = g * D + d;
      const uint64_t beg = __ldg(key_off + t), end = __ldg(key_off + t + 1);
      if (end < beg) {
        if (threadIdx.x == 0) flag_status(status, NETKV_DEV_ERANGE);
        continue;
      }
      const unsigned long long bit = 1ull << (d % kGroup);
      for (uint64_t c = beg; c < end; c += kBuildBlock) {
        const uint64_t j = c + threadIdx.x;
        unsigned long long key = j < end ? __ldg(keys + j) : 0ull;
        if (j < end && key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
        bool is_new = false;
        uint64_t slot = 0;
        bool placed = false;
        if (key != 0ull) {
          slot = home_slot(key, log2_cap);
          for (uint64_t step = 0; step < cap; ++step) {
            const unsigned long long prev = atomicCAS(&hash[slot].key, 0ull, key);
            if (prev == 0ull || prev == key) {
              is_new = prev == 0ull;
              placed = true;
              break;
            }
            slot = (slot + 1) & mask;
          }
          if (!placed) flag_status(status, NETKV_DEV_EFULL);
        }
        const uint32_t pos = run_len + block_scan(is_new ? 1u : 0u, warp_sums, &chunk_new);
        if (is_new) {
          hash[slot].pos = pos;
          v.keys[pos] = key;
          run_mask_or(v, pos, bit);  // masks share 32-bit words: set by atomics only
        }
        __syncthreads();
        if (placed && !is_new) {
          const uint64_t p = *((volatile unsigned long long*)&hash[slot].pos);
          run_mask_or(v, p, bit);
        }
        run_len += chunk_new;
        __syncthreads();
      }
    }
  }
}

__device__ __forceinline__ int32_t find_set(const uint32_t* __restrict__ set_off, uint32_t n_sets,
                                            uint32_t r) {
  if (!set_off) return 0;
  if (r < __ldg(set_off) || r >= __ldg(set_off + n_sets)) return -1;
  uint32_t lo = 0, hi = n_sets;  // invariant: set_off[lo] <= r < set_off[hi]
  while (hi - lo > 1) {
    const uint32_t mid = (lo + hi) >> 1;
    if (__ldg(set_off + mid) <= r) lo = mid; else hi = mid;
  }
  return (int32_t)lo;
}

// Per-lane results of one decode group: lane j holds decodes j and j + 32.
struct GroupHits {
  uint32_t lo, hi;
};

__device__ __forceinline__ void set_hit(GroupHits& h, uint32_t lane, uint32_t j, uint32_t v) {
  if (j == lane) h.lo = v;
  if (j == lane + 32) h.hi = v;
}

// Every decode in `alive` misses at position v.
__device__ __forceinline__ void miss_all(GroupHits& h, uint32_t lane, unsigned long long alive,
                                         uint32_t v) {
  if ((alive >> lane) & 1ull) h.lo = v;
  if ((alive >> (lane + 32)) & 1ull) h.hi = v;
}

// First-miss scan of blocks [start, n) of one chain for the `alive` decodes of a group.
// Decodes found missing at position p get p; decodes never missing keep their value.
// start_pos: the run position of block `start` when the caller has already looked it up.
// kMB: the run masks' width when known at compile time (see run_mask), else 0.
template <int kMB = 0>
__device__ __forceinline__ void scan_chain(const IndexView& ix, uint32_t log2_cap,
                                           const uint64_t* __restrict__ chain, uint64_t start,
                                           uint64_t n, unsigned long long alive, GroupHits& h,
                                           uint32_t lane, int* status,
                                           unsigned long long start_pos = kNotFound) {
  const uint64_t cap = 1ull << log2_cap;
  const IndexSlot* __restrict__ hash = ix.hash;
  const unsigned long long* __restrict__ run_keys = ix.keys;
  uint64_t p = start;
  uint64_t seg_run = 0, seg_p = 0;  // run position matched with chain position seg_p
  bool in_run = false, fresh = false;
  if (start_pos != kNotFound) {
    seg_run = start_pos;
    seg_p = start;
    in_run = fresh = true;
  }
  while (p < n && alive) {
    const bool looked_up = !in_run || fresh;
    fresh = false;
    if (!in_run) {  // locate block p in the hash table
      const uint64_t key = __ldg(chain + p);
      unsigned long long pos = kNotFound;
      if (lane == 0) {
        if (key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
        else pos = lookup(hash, key, log2_cap, status);
      }
      pos = __shfl_sync(0xffffffffu, pos, 0);
      if (pos == kNotFound) {  // absent from every cache of the group
        miss_all(h, lane, alive, (uint32_t)p);
        return;
      }
      seg_run = pos;
      seg_p = p;
      in_run = true;
    }
    // blocks p .. p+31 against the run from seg_run
    const uint64_t i = p + lane;
    const uint64_t rp = seg_run + (i - seg_p);
    const bool in = i < n;
    const uint64_t ck = in ? __ldcs(chain + i) : 0ull;
    unsigned long long rkey = 0ull, rmask = 0ull;
    if (in && rp < cap) {
      rkey = __ldg(run_keys + rp);
      rmask = run_mask<kMB>(ix, rp);
    }
    const bool same = in && ck != 0ull && rkey == ck;
    const uint32_t run_ok = __ballot_sync(0xffffffffu, same);
    const uint32_t lead = (~run_ok) ? (uint32_t)(__ffs(~run_ok) - 1) : 32u;  // leading matches
    const bool counted = lane < lead;
    // decodes missing at some counted position of this step (usually none)
    const unsigned long long nm = counted ? (alive & ~rmask) : 0ull;
    unsigned long long a = ((unsigned long long)__reduce_or_sync(0xffffffffu, (uint32_t)(nm >> 32))
                            << 32) |
                           __reduce_or_sync(0xffffffffu, (uint32_t)nm);
    while (a) {
      const uint32_t j = __ffsll((long long)a) - 1;
      a &= a - 1;
      const uint32_t miss = __ballot_sync(0xffffffffu, (nm >> j) & 1ull);
      set_hit(h, lane, j, (uint32_t)(p + (uint64_t)(__ffs(miss) - 1)));
      alive &= ~(1ull << j);
    }
    if (lead == 0 && looked_up) {
      // the run entry the table points to does not hold the key: a corrupted index.
      // Report it and count the block as missing, so the walk always advances.
      if (lane == 0) flag_status(status, NETKV_DEV_EFULL);
      miss_all(h, lane, alive, (uint32_t)p);
      return;
    }
    p += lead;
    if (lead < 32) in_run = false;  // the run parts here: look the next block up
  }
}


// Group key of a request: its table set and first block hash, never zero.
__device__ __forceinline__ uint64_t group_key(uint64_t h0, uint32_t set) {
  uint64_t z = h0 ^ ((uint64_t)(set + 1) * 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  z ^= z >> 31;
  return z ? z : 1ull;
}

struct GroupSlot {
  unsigned long long key;
  unsigned long long code;  // (chain length << 32) | (0xffffffff - r): max = longest, lowest r
};

// Work counters at the end of the workspace.
struct MatchCounters {
  unsigned long long n_long;       // leaders listed from the front of the leader list
  unsigned long long n_short;      // leaders listed from its back
  unsigned long long next_task;    // next (leader, decode group) task of the leader pass
  unsigned long long next_member;  // next chunk of requests of the member pass
};

// Leaders with chains of at least this many blocks are listed first, so that the leader
// pass, which takes its tasks in list order, ends on short chains instead of waiting for
// a long one started last.
constexpr uint64_t kLongLeader = 2048;

// One thread per request: its table set (set_of) and group key (in rec[r].x, for the
// resolve pass) are recorded, and the group's slot keeps the longest chain.
__global__ void group_insert_kernel(GroupSlot* __restrict__ tab, uint32_t log2_slots,
                                    const uint64_t* __restrict__ chains,
                                    const uint64_t* __restrict__ chain_off, uint32_t R,
                                    const uint32_t* __restrict__ set_off, uint32_t n_sets,
                                    int32_t* __restrict__ set_of, ulonglong2* __restrict__ rec) {
  const uint64_t mask = (1ull << log2_slots) - 1;
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    const int32_t set = find_set(set_off, n_sets, r);
    set_of[r] = set;
    if (c1 <= c0 || set < 0) continue;
    const uint64_t n = c1 - c0;
    const uint64_t key = group_key(__ldg(chains + c0), (uint32_t)set);
    rec[r].x = key;
    const unsigned long long code =
        ((unsigned long long)(n < 0xffffffffull ? n : 0xffffffffull) << 32) | (0xffffffffu - r);
    uint64_t slot = home_slot(key, log2_slots);
    for (uint64_t step = 0; step <= mask; ++step) {
      const unsigned long long prev = atomicCAS(&tab[slot].key, 0ull, key);
      if (prev == 0ull || prev == key) {
        atomicMax(&tab[slot].code, code);
        break;
      }
      slot = (slot + 1) & mask;
    }
  }
}

// A member's record: its chain offset and length (clamped to 65,535 blocks) and its
// leader's, 48 + 16 bits each, so that the member pass fetches both chains' first blocks
// and the leader's hits in its first round trip.
constexpr uint64_t kOff48 = (1ull << 48) - 1;

__global__ void group_resolve_kernel(const GroupSlot* __restrict__ tab, uint32_t log2_slots,
                                     const uint64_t* __restrict__ chain_off, uint32_t R,
                                     uint32_t* __restrict__ leader_of,
                                     const int32_t* __restrict__ set_of,
                                     uint32_t* __restrict__ leaders, ulonglong2* __restrict__ rec,
                                     MatchCounters* counters, int* status) {
  const uint64_t mask = (1ull << log2_slots) - 1;
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    const int32_t set = __ldg(set_of + r);
    uint32_t lead = r;
    if (c1 > c0 && set >= 0) {
      const uint64_t key = rec[r].x;  // written by the insert pass
      uint64_t slot = home_slot(key, log2_slots);
      for (uint64_t step = 0; step <= mask; ++step) {
        const unsigned long long k = tab[slot].key;
        if (k == key) {
          const uint32_t L = 0xffffffffu - (uint32_t)(tab[slot].code & 0xffffffffull);
          // a leader from another table set (64-bit key collision) is never used
          if (L < R && __ldg(set_of + L) == set) lead = L;
          break;
        }
        if (k == 0ull) break;
        slot = (slot + 1) & mask;
      }
    }
    if (lead != r) {
      const uint64_t l0 = __ldg(chain_off + lead), l1 = __ldg(chain_off + lead + 1);
      if (c1 <= kOff48 && l1 <= kOff48 && l1 > l0) {
        const uint64_t n = c1 - c0, nl = l1 - l0;
        if (n > 65535) flag_status(status, NETKV_DEV_EDOMAIN);  // counted up to 65,535 blocks
        rec[r] = make_ulonglong2(c0 | (min(n, (uint64_t)65535) << 48),
                                 l0 | (min(nl, (uint64_t)65535) << 48));
      } else {
        lead = r;  // offsets beyond 48 bits: matched in full by the leader pass
      }
    }
    leader_of[r] = lead;
    if (lead == r) {  // long chains from the front of the list, the rest from its back
      if (c1 > c0 && c1 - c0 >= kLongLeader)
        leaders[atomicAdd(&counters->n_long, 1ull)] = r;
      else
        leaders[R - 1 - atomicAdd(&counters->n_short, 1ull)] = r;
    }
  }
}

// Chain r's extent clamped to 65535 blocks; false on a bad request (flagged).
__device__ __forceinline__ bool chain_extent(const uint64_t* __restrict__ chain_off,
                                             const uint32_t* __restrict__ set_off,
                                             uint32_t n_sets, const int32_t* __restrict__ set_of,
                                             uint32_t r, uint32_t lane, int* status,
                                             int32_t& set, uint64_t& c0, uint64_t& n) {
  set = set_of ? __ldg(set_of + r) : find_set(set_off, n_sets, r);
  c0 = __ldg(chain_off + r);
  const uint64_t c1 = __ldg(chain_off + r + 1);
  if (set < 0 || c1 < c0) {
    if (lane == 0) flag_status(status, NETKV_DEV_ERANGE);
    return false;
  }
  n = c1 - c0;
  if (n > 65535) {
    if (lane == 0) flag_status(status, NETKV_DEV_EDOMAIN);
    n = 65535;
  }
  return true;
}

__device__ __forceinline__ void store_hits(uint16_t* __restrict__ M, uint64_t row, uint32_t q0,
                                           uint32_t ng, uint32_t lane, const GroupHits& h) {
  if (lane < ng) M[row + q0 + lane] = (uint16_t)h.lo;
  if (lane + 32 < ng) M[row + q0 + lane + 32] = (uint16_t)h.hi;
}

// Leader pass: one task per (leader, decode group), taken in order from a global counter
// by whole warps, so long and short chains balance across the GPU.
__global__ void __launch_bounds__(kMatchBlock, 8) match_leaders_kernel(
    const void* __restrict__ index, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off, uint32_t R,
    const uint32_t* __restrict__ set_off, const int32_t* __restrict__ set_of,
    const uint32_t* __restrict__ leaders, MatchCounters* counters, uint16_t* __restrict__ M,
    int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t n_dgroups = (D + kGroup - 1) / kGroup;
  const unsigned long long n_long = *((volatile unsigned long long*)&counters->n_long);
  const unsigned long long total =
      (n_long + *((volatile unsigned long long*)&counters->n_short)) * n_dgroups;
  for (;;) {
    unsigned long long t = 0;
    if (lane == 0) t = atomicAdd(&counters->next_task, 1ull);
    t = __shfl_sync(0xffffffffu, t, 0);
    if (t >= total) break;
    const uint64_t li = n_dgroups == 1 ? t : t / n_dgroups;
    const uint32_t r = __ldg(leaders + (li < n_long ? li : (uint64_t)R - 1 - (li - n_long)));
    const uint32_t q = (uint32_t)(t - li * n_dgroups);
    const uint32_t q0 = q * kGroup, ng = min(kGroup, D - q0);
    GroupHits h = {0u, 0u};
    int32_t set;
    uint64_t c0, n;
    if (chain_extent(chain_off, set_off, n_sets, set_of, r, lane, status, set, c0, n)) {
      h.lo = h.hi = (uint32_t)n;
      const unsigned long long alive = ng >= 64 ? ~0ull : ((1ull << ng) - 1);
      const IndexView ix = index_view(index, (uint64_t)set * n_dgroups + q, log2_cap,
                                      mask_bytes_of(D));
      scan_chain(ix, log2_cap, chains + c0, 0, n, alive, h, lane, status);
    }
    store_hits(M, (uint64_t)r * D, q0, ng, lane, h);
  }
}

// Full match without a workspace: one warp per (request, decode group).
__global__ void __launch_bounds__(kMatchBlock, 8) match_kernel(
    const void* __restrict__ index, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off, uint32_t R,
    const uint32_t* __restrict__ set_off, uint16_t* __restrict__ M, int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t n_dgroups = (D + kGroup - 1) / kGroup;
  const uint64_t total = (uint64_t)R * n_dgroups;

  for (uint64_t task = warp; task < total; task += n_warps) {
    const uint32_t r = (uint32_t)(n_dgroups == 1 ? task : task / n_dgroups);
    const uint32_t q = (uint32_t)(task - (uint64_t)r * n_dgroups);
    const uint32_t q0 = q * kGroup, ng = min(kGroup, D - q0);
    GroupHits h = {0u, 0u};
    int32_t set;
    uint64_t c0, n;
    if (chain_extent(chain_off, set_off, n_sets, nullptr, r, lane, status, set, c0, n)) {
      h.lo = h.hi = (uint32_t)n;
      const unsigned long long alive = ng >= 64 ? ~0ull : ((1ull << ng) - 1);
      const IndexView ix = index_view(index, (uint64_t)set * n_dgroups + q, log2_cap,
                                      mask_bytes_of(D));
      scan_chain(ix, log2_cap, chains + c0, 0, n, alive, h, lane, status);
    }
    store_hits(M, (uint64_t)r * D, q0, ng, lane, h);
  }
}

// Member pass of pools of one decode group (D <= 64), for member r with leader `lead`.
// The record written by the grouping gives both chains' offsets and lengths, so the
// leader's hits and the first 128 blocks of both chains are fetched in one round trip (the
// cap on the common prefix, min(n_r, n_L, max_d M_L[d] + 1), is known once the hits
// arrive).  Then as the leader pass: decodes whose leader missed inside the common prefix
// take the leader's answer, the rest walk on from the common prefix.
__device__ __forceinline__ void member_match(const void* __restrict__ index, uint32_t D,
                                             uint32_t log2_cap,
                                             const uint64_t* __restrict__ chains, uint32_t r,
                                             uint32_t lead, int32_t set, ulonglong2 rc,
                                             uint16_t* __restrict__ M, uint32_t lane,
                                             int* status) {
  const uint32_t ng = D;  // one group
  const uint64_t c0 = rc.x & kOff48, n = rc.x >> 48;
  const uint64_t l0 = rc.y & kOff48, nl = rc.y >> 48;
  const uint64_t capn = min(n, nl);
  const uint64_t lrow = (uint64_t)lead * D;
  const uint32_t mlo = lane < ng ? (uint32_t)__ldg(M + lrow + lane) : 0u;
  const uint32_t mhi = lane + 32 < ng ? (uint32_t)__ldg(M + lrow + lane + 32) : 0u;
  uint64_t a[4], b[4];
  const uint64_t first = min(capn, (uint64_t)128);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint64_t i = 32 * k + lane;
    a[k] = i < first ? __ldcs(chains + c0 + i) : 0ull;
    b[k] = i < first ? __ldg(chains + l0 + i) : 0ull;
  }
  uint32_t mmax = max(mlo, mhi);
#pragma unroll
  for (int o = 16; o; o >>= 1) mmax = max(mmax, __shfl_xor_sync(0xffffffffu, mmax, o));
  const uint64_t cap = min(capn, (uint64_t)mmax + 1);
  uint64_t lcp = cap;  // common prefix, 128 blocks per step
  for (uint64_t base = 0; base < cap;) {
    uint64_t found = cap;
#pragma unroll
    for (int k = 3; k >= 0; --k) {
      const uint64_t i = base + 32 * k + lane;
      const uint32_t diff = __ballot_sync(0xffffffffu, i < cap && a[k] != b[k]);
      if (diff) found = base + 32 * k + (uint64_t)(__ffs(diff) - 1);
    }
    if (found < cap) {
      lcp = found;
      break;
    }
    base += 128;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint64_t i = base + 32 * k + lane;
      a[k] = i < cap ? __ldcs(chains + c0 + i) : 0ull;
      b[k] = i < cap ? __ldg(chains + l0 + i) : 0ull;
    }
  }
  GroupHits h = {(uint32_t)n, (uint32_t)n};
  // decodes whose leader missed inside the common prefix copy the leader's answer
  const uint32_t clo = __ballot_sync(0xffffffffu, lane < ng && (uint64_t)mlo < lcp);
  const uint32_t chi = __ballot_sync(0xffffffffu, lane + 32 < ng && (uint64_t)mhi < lcp);
  if ((clo >> lane) & 1u) h.lo = mlo;
  if ((chi >> lane) & 1u) h.hi = mhi;
  unsigned long long alive = ng >= 64 ? ~0ull : ((1ull << ng) - 1);
  alive &= ~((unsigned long long)clo | ((unsigned long long)chi << 32));
  scan_chain(index_view(index, (uint64_t)set, log2_cap, mask_bytes_of(D)), log2_cap,
             chains + c0, lcp, n, alive, h, lane, status);
  store_hits(M, (uint64_t)r * D, 0, ng, lane, h);
}

constexpr uint32_t kMemberChunk = 8;  // consecutive requests a warp takes at a time

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async4(void* smem, const void* gmem) {
  const unsigned sa = (unsigned)__cvta_generic_to_shared(smem);
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(sa), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;\n" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_group 0;\n" ::: "memory");
}

// A request's record, leader and table set, staged in shared memory per warp.
struct __align__(16) MemberSlot {
  ulonglong2 rc;
  uint32_t lead;
  int32_t set;
  uint32_t pad[2];
};

// Persistent member pass of pools of one decode group: every warp takes chunks of 8
// consecutive requests from a global counter (fetched one chunk ahead), so a warp that
// finishes early takes more work instead of idling until its block ends.  The next
// request's record, leader and table set are copied into the warp's shared-memory slot
// with cp.async while the current one is matched, so they cost no round trip of their own.
__global__ void __launch_bounds__(kMatchBlock, 8) match_members_kernel(
    const void* __restrict__ index, uint32_t D, uint32_t log2_cap,
    const uint64_t* __restrict__ chains, uint32_t R, const uint32_t* __restrict__ leader_of,
    const int32_t* __restrict__ set_of, const ulonglong2* __restrict__ rec,
    MatchCounters* counters, uint16_t* __restrict__ M, int* status) {
  __shared__ MemberSlot slots[kMatchBlock / 32];
  MemberSlot& slot = slots[threadIdx.x >> 5];
  const uint32_t lane = threadIdx.x & 31;
  const unsigned long long n_chunks = ((unsigned long long)R + kMemberChunk - 1) / kMemberChunk;
  // request rr's record into the slot (a leader's record is not written and not used)
  auto fetch = [&](uint64_t rr) {
    if (lane == 0) {
      cp_async16(&slot.rc, rec + rr);
      cp_async4(&slot.lead, leader_of + rr);
      cp_async4(&slot.set, set_of + rr);
      cp_async_commit();
    }
  };
  unsigned long long c = 0, c_next = 0;
  if (lane == 0) c = atomicAdd(&counters->next_member, 1ull);
  c = __shfl_sync(0xffffffffu, c, 0);
  if (c >= n_chunks) return;
  if (lane == 0) c_next = atomicAdd(&counters->next_member, 1ull);  // the chunk after
  uint64_t r = c * kMemberChunk;
  uint64_t end = min(r + kMemberChunk, (uint64_t)R);
  fetch(r);
  for (;;) {
    if (lane == 0) cp_async_wait_all();  // request r's record has landed
    __syncwarp();
    const ulonglong2 rc = slot.rc;
    const uint32_t lead = slot.lead;
    const int32_t set = slot.set;
    __syncwarp();  // every lane has read the slot before it is refilled
    uint64_t rn = r + 1;
    if (rn >= end) {  // this chunk is done: take the one fetched ahead, and fetch the next
      const unsigned long long cn = __shfl_sync(0xffffffffu, c_next, 0);
      rn = cn < n_chunks ? cn * kMemberChunk : (uint64_t)R;
      end = min(rn + kMemberChunk, (uint64_t)R);
      if (lane == 0 && cn < n_chunks) c_next = atomicAdd(&counters->next_member, 1ull);
    }
    if (rn < R) fetch(rn);
    if (lead != (uint32_t)r)  // leaders were matched by the leader pass
      member_match(index, D, log2_cap, chains, (uint32_t)r, lead, set, rc, M, lane, status);
    if (rn >= R) break;
    r = rn;
  }
}

// Member pass for pools of several decode groups: one warp per member.  With
// lcp = |common prefix of h_r and h_L| capped at min(n_r, n_L, max_d M_L[d] + 1), every
// decode has M_r[d] = min(M_L[d], lcp) unless M_L[d] >= lcp and block lcp of h_r is
// cached on d.  So the member's row is one elementwise pass over the leader's row (16
// bytes a lane when the rows are 16-byte aligned), and block lcp is then probed in the
// groups where some leader hit reaches lcp, up to 32 groups at once with one lane per
// group; a group whose probe finds the block is walked again by the whole warp.
__global__ void __launch_bounds__(kMatchBlock, 6) match_members_wide_kernel(
    const void* __restrict__ index, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off, uint32_t R,
    const uint32_t* __restrict__ set_off, const uint32_t* __restrict__ leader_of,
    const int32_t* __restrict__ set_of, uint16_t* __restrict__ M, int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t n_dgroups = (D + kGroup - 1) / kGroup;
  const bool vec = (D % 8u == 0) && ((reinterpret_cast<uintptr_t>(M) & 15u) == 0);
  const uint32_t n8 = D / 8u;  // 16-byte chunks of a row (vector form)

  for (uint64_t rr = warp; rr < R; rr += n_warps) {
    const uint32_t r = (uint32_t)rr;
    const uint32_t lead = __ldg(leader_of + r);
    if (lead == r) continue;  // leaders were matched by the leader pass
    const uint64_t row = (uint64_t)r * D;
    int32_t set;
    uint64_t c0, n;
    if (!chain_extent(chain_off, set_off, n_sets, set_of, r, lane, status, set, c0, n)) {
      const GroupHits z = {0u, 0u};
      for (uint32_t q = 0; q < n_dgroups; ++q)
        store_hits(M, row, q * kGroup, min(kGroup, D - q * kGroup), lane, z);
      continue;
    }
    const uint64_t l0 = __ldg(chain_off + lead);
    const uint64_t nl = min(__ldg(chain_off + lead + 1) - l0, (uint64_t)65535);
    const uint64_t* __restrict__ own = chains + c0;
    const uint64_t* __restrict__ lch = chains + l0;
    const uint16_t* __restrict__ ml = M + (uint64_t)lead * D;
    uint16_t* __restrict__ mr = M + row;

    // the leader's largest hit
    uint32_t mmax = 0;
    if (vec) {
      for (uint32_t c = lane; c < n8; c += 32) {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(ml) + c);
        const uint32_t m2 = __vmaxu2(__vmaxu2(v.x, v.y), __vmaxu2(v.z, v.w));
        mmax = max(mmax, max(m2 & 0xffffu, m2 >> 16));
      }
    } else {
      for (uint32_t d = lane; d < D; d += 32) mmax = max(mmax, (uint32_t)__ldg(ml + d));
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) mmax = max(mmax, __shfl_xor_sync(0xffffffffu, mmax, o));

    // common prefix with the leader, capped, 128 blocks a step
    const uint64_t cap = min(n, min(nl, (uint64_t)mmax + 1));
    uint64_t lcp = cap;
    for (uint64_t base = 0; base < cap; base += 128) {
      uint64_t a[4], b[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const uint64_t i = base + 32 * k + lane;
        a[k] = i < cap ? __ldg(own + i) : 0ull;
        b[k] = i < cap ? __ldg(lch + i) : 0ull;
      }
      uint64_t found = cap;
#pragma unroll
      for (int k = 3; k >= 0; --k) {
        const uint32_t diff = __ballot_sync(0xffffffffu, a[k] != b[k]);
        if (diff) found = base + 32 * k + (uint64_t)(__ffs(diff) - 1);
      }
      if (found < cap) {
        lcp = found;
        break;
      }
    }
    const bool probe = lcp < n;  // decodes with M_L >= lcp may hit block lcp

    uint32_t pend_q = 0;  // lane j: the j-th group waiting for its probe of block lcp
    uint32_t n_pend = 0;
    auto flush = [&]() {
      __syncwarp();
      unsigned long long pos = kNotFound;
      if (lane < n_pend) {
        const uint64_t key = __ldg(own + lcp);
        if (key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
        else pos = lookup(index_view(index, (uint64_t)set * n_dgroups + pend_q, log2_cap, 8u).hash,
                          key, log2_cap, status);
      }
      uint32_t hit = __ballot_sync(0xffffffffu, lane < n_pend && pos != kNotFound);
      while (hit) {
        const uint32_t j = __ffs(hit) - 1;
        hit &= hit - 1;
        const uint32_t q = __shfl_sync(0xffffffffu, pend_q, j);
        const unsigned long long pj = __shfl_sync(0xffffffffu, pos, j);
        const uint32_t q0 = q * kGroup, ng = min(kGroup, D - q0);
        const uint32_t mlo = lane < ng ? (uint32_t)__ldg(ml + q0 + lane) : 0u;
        const uint32_t mhi = lane + 32 < ng ? (uint32_t)__ldg(ml + q0 + lane + 32) : 0u;
        GroupHits h;
        h.lo = (uint64_t)mlo < lcp ? mlo : (uint32_t)n;
        h.hi = (uint64_t)mhi < lcp ? mhi : (uint32_t)n;
        const uint32_t alo = __ballot_sync(0xffffffffu, lane < ng && (uint64_t)mlo >= lcp);
        const uint32_t ahi = __ballot_sync(0xffffffffu, lane + 32 < ng && (uint64_t)mhi >= lcp);
        const unsigned long long alive = (unsigned long long)alo | ((unsigned long long)ahi << 32);
        scan_chain<8>(index_view(index, (uint64_t)set * n_dgroups + q, log2_cap, 8u),
                   log2_cap, own, lcp, n, alive, h, lane, status, pj);
        store_hits(M, row, q0, ng, lane, h);
      }
      n_pend = 0;
    };
    auto pend = [&](uint32_t q) {
      if (lane == n_pend) pend_q = q;
      if (++n_pend == 32) flush();
    };

    // M_r = min(M_L, lcp); note the groups where a leader hit reaches lcp
    const uint32_t lcp_u = (uint32_t)lcp;
    if (vec) {
      const uint32_t lcp2 = lcp_u | (lcp_u << 16);
      for (uint32_t c0v = 0; c0v < n8; c0v += 32) {
        const uint32_t c = c0v + lane;
        bool reach = false;
        if (c < n8) {
          uint4 v = __ldg(reinterpret_cast<const uint4*>(ml) + c);
          const uint32_t m2 = __vmaxu2(__vmaxu2(v.x, v.y), __vmaxu2(v.z, v.w));
          reach = max(m2 & 0xffffu, m2 >> 16) >= lcp_u;
          v.x = __vminu2(v.x, lcp2);
          v.y = __vminu2(v.y, lcp2);
          v.z = __vminu2(v.z, lcp2);
          v.w = __vminu2(v.w, lcp2);
          reinterpret_cast<uint4*>(mr)[c] = v;
        }
        // 8 chunks per group: lanes 8k .. 8k+7 hold group c0v / 8 + k
        const uint32_t fb = __ballot_sync(0xffffffffu, probe && reach);
#pragma unroll
        for (int k = 0; k < 4; ++k)
          if ((fb >> (8 * k)) & 0xffu) pend(c0v / 8u + (uint32_t)k);
      }
    } else {
      for (uint32_t q = 0; q < n_dgroups; ++q) {
        const uint32_t q0 = q * kGroup, ng = min(kGroup, D - q0);
        const uint32_t mlo = lane < ng ? (uint32_t)__ldg(ml + q0 + lane) : 0u;
        const uint32_t mhi = lane + 32 < ng ? (uint32_t)__ldg(ml + q0 + lane + 32) : 0u;
        GroupHits h;
        h.lo = min(mlo, lcp_u);
        h.hi = min(mhi, lcp_u);
        store_hits(M, row, q0, ng, lane, h);
        const bool reach = (lane < ng && mlo >= lcp_u) || (lane + 32 < ng && mhi >= lcp_u);
        if (__any_sync(0xffffffffu, probe && reach)) pend(q);
      }
    }
    if (n_pend) flush();
  }
}

uint32_t group_log2_slots(uint32_t R) {
  uint32_t l = 1;
  while ((1ull << l) < 2ull * R) ++l;
  return l;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace: group table | leader_of [R] | set_of [R] | leader list [R] | member records [R]
// | counters.
struct WorkspaceLayout {
  size_t table, leader_of, set_of, leaders, rec, counters, total;
};

WorkspaceLayout workspace_layout(uint32_t R) {
  WorkspaceLayout w;
  w.table = 0;
  w.leader_of = align_up(sizeof(GroupSlot) << group_log2_slots(R), 256);
  w.set_of = w.leader_of + align_up(sizeof(uint32_t) * (size_t)R, 256);
  w.leaders = w.set_of + align_up(sizeof(int32_t) * (size_t)R, 256);
  w.rec = w.leaders + align_up(sizeof(uint32_t) * (size_t)R, 256);
  w.counters = w.rec + align_up(sizeof(ulonglong2) * (size_t)R, 256);
  w.total = w.counters + align_up(sizeof(MatchCounters), 256);
  return w;
}

// Blocks of a persistent grid: every SM filled to the kernel's occupancy.
template <typename Kernel>
int persistent_grid(Kernel kernel) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kMatchBlock, 0);
  return (sms > 0 ? sms : 1) * (per_sm > 0 ? per_sm : 1);
}
int leader_grid() { return persistent_grid(match_leaders_kernel); }
int member_grid() { return persistent_grid(match_members_kernel); }

}  // namespace

extern "C" size_t netkv_cache_index_bytes(uint32_t n_sets, uint32_t D, uint32_t log2_capacity) {
  if (log2_capacity < 1 || log2_capacity > 31) return 0;
  return (size_t)n_sets * ((D + kGroup - 1) / kGroup) *
         index_stride(log2_capacity, mask_bytes_of(D));
}

extern "C" netkv_status netkv_cache_build(void* d_index, uint32_t n_sets, uint32_t D,
                                          uint32_t log2_capacity, const uint64_t* d_keys,
                                          const uint64_t* d_key_off, int* d_status,
                                          netkv_stream_t stream) {
  if (!d_index || !d_key_off || D == 0 || log2_capacity < 1 || log2_capacity > 31)
    return NETKV_EINVAL;
  if (!aligned_to(d_index, 16) || !aligned_to(d_key_off, 8) || (d_keys && !aligned_to(d_keys, 8)))
    return NETKV_EINVAL;
  if (n_sets == 0) return NETKV_OK;
  cudaStream_t s = (cudaStream_t)stream;
  NETKV_CUDA_TRY(cudaMemsetAsync(d_index, 0, netkv_cache_index_bytes(n_sets, D, log2_capacity), s));
  if (!d_keys) return NETKV_OK;
  const uint64_t n_index = (uint64_t)n_sets * ((D + kGroup - 1) / kGroup);
  const unsigned grid = (unsigned)(n_index < (1u << 20) ? n_index : (1u << 20));
  cache_build_kernel<<<grid, kBuildBlock, 0, s>>>(d_index, n_sets, D, log2_capacity, d_keys,
                                                  d_key_off, d_status);
  return netkv_launch_status();
}

extern "C" size_t netkv_prefix_match_workspace_size(uint32_t R) {
  if (R == 0) return 0;
  return workspace_layout(R).total;
}

extern "C" netkv_status netkv_prefix_match(const void* d_index, uint32_t D,
                                           uint32_t log2_capacity, uint32_t n_sets,
                                           const uint64_t* d_chains, const uint64_t* d_chain_off,
                                           uint32_t R, const uint32_t* d_set_off,
                                           void* d_workspace, size_t workspace_bytes,
                                           uint16_t* d_M, int* d_status, netkv_stream_t stream) {
  if (!d_index || !d_chain_off || !d_M || D == 0 || n_sets == 0) return NETKV_EINVAL;
  if (log2_capacity < 1 || log2_capacity > 31) return NETKV_EINVAL;
  if (n_sets > 1 && !d_set_off) return NETKV_EINVAL;
  if (!aligned_to(d_index, 16) || !aligned_to(d_chain_off, 8) || !aligned_to(d_M, 2) ||
      (d_chains && !aligned_to(d_chains, 8)) || (d_set_off && !aligned_to(d_set_off, 4)) ||
      (d_workspace && !aligned_to(d_workspace, 256)))
    return NETKV_EINVAL;
  if (R == 0) return NETKV_OK;
  if (!d_chains || R > 0x7fffffffu) return NETKV_EINVAL;
  if (d_workspace && workspace_bytes < netkv_prefix_match_workspace_size(R)) return NETKV_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  const void* index = d_index;
  const uint64_t tasks = (uint64_t)R * ((D + kGroup - 1) / kGroup);
  const uint64_t warps_per_block = kMatchBlock / 32;
  const uint64_t blocks = (tasks + warps_per_block - 1) / warps_per_block;
  const unsigned grid = (unsigned)(blocks < (1u << 24) ? blocks : (1u << 24));
  if (!d_workspace) {
    match_kernel<<<grid, kMatchBlock, 0, s>>>(index, D, log2_capacity, n_sets, d_chains,
                                              d_chain_off, R, d_set_off, d_M, d_status);
    return netkv_launch_status();
  }
  const uint32_t lg = group_log2_slots(R);
  const WorkspaceLayout L = workspace_layout(R);
  char* ws = reinterpret_cast<char*>(d_workspace);
  GroupSlot* tab = reinterpret_cast<GroupSlot*>(ws + L.table);
  uint32_t* leader_of = reinterpret_cast<uint32_t*>(ws + L.leader_of);
  int32_t* set_of = reinterpret_cast<int32_t*>(ws + L.set_of);
  uint32_t* leaders = reinterpret_cast<uint32_t*>(ws + L.leaders);
  ulonglong2* rec = reinterpret_cast<ulonglong2*>(ws + L.rec);
  MatchCounters* counters = reinterpret_cast<MatchCounters*>(ws + L.counters);
  NETKV_CUDA_TRY(cudaMemsetAsync(tab, 0, sizeof(GroupSlot) << lg, s));
  NETKV_CUDA_TRY(cudaMemsetAsync(counters, 0, sizeof(MatchCounters), s));
  const unsigned rgrid = (unsigned)((R + 255) / 256 < 65535u * 16 ? (R + 255) / 256 : 65535u * 16);
  group_insert_kernel<<<rgrid, 256, 0, s>>>(tab, lg, d_chains, d_chain_off, R, d_set_off, n_sets,
                                            set_of, rec);
  group_resolve_kernel<<<rgrid, 256, 0, s>>>(tab, lg, d_chain_off, R, leader_of, set_of, leaders,
                                             rec, counters, d_status);
  match_leaders_kernel<<<leader_grid(), kMatchBlock, 0, s>>>(
      index, D, log2_capacity, n_sets, d_chains, d_chain_off, R, d_set_off, set_of, leaders,
      counters, d_M, d_status);
  if (D <= kGroup) {
    match_members_kernel<<<member_grid(), kMatchBlock, 0, s>>>(
        index, D, log2_capacity, d_chains, R, leader_of, set_of, rec, counters, d_M, d_status);
  } else {
    const uint64_t mblocks = ((uint64_t)R + warps_per_block - 1) / warps_per_block;
    const unsigned mgrid = (unsigned)(mblocks < (1u << 24) ? mblocks : (1u << 24));
    match_members_wide_kernel<<<mgrid, kMatchBlock, 0, s>>>(index, D, log2_capacity, n_sets,
                                                            d_chains, d_chain_off, R, d_set_off,
                                                            leader_of, set_of, d_M, d_status);
  }
  return netkv_launch_status();
}

// ---------------------------------------------------------------------------------
// netkv_prefix_match_static: the prefix match for callers that cannot allocate device
// memory (see include/netkv.h).  Its workspace is this fixed device array, shared by
// every call on a device.  Host code cannot use the array's name as a device address, so
// the address is looked up with the device current: on every call made outside a stream
// capture (a device reset reloads the module and may move the array), and from the
// last lookup on that device during a capture.
// ---------------------------------------------------------------------------------
#include <mutex>

namespace {

constexpr size_t kStaticScratchBytes = 32ull << 20;  // 32 MiB per device
static __device__ __align__(256) unsigned char g_prefix_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_prefix_scratch on the current device.
netkv_status static_scratch(cudaStream_t stream, void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return NETKV_ECUDA;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(stream, &cap) != cudaSuccess) {
    cudaGetLastError();
    return NETKV_ECUDA;
  }
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (cap == cudaStreamCaptureStatusNone || !g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_prefix_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return NETKV_ECUDA;
    }
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return NETKV_OK;
}

}  // namespace

static_assert(NETKV_PREFIX_MATCH_STATIC_MAX_R > 0, "limit must be positive");

extern "C" netkv_status netkv_prefix_match_static(const void* d_index, uint32_t D,
                                                  uint32_t log2_capacity, uint32_t n_sets,
                                                  const uint64_t* d_chains,
                                                  const uint64_t* d_chain_off, uint32_t R,
                                                  const uint32_t* d_set_off, uint16_t* d_M,
                                                  int* d_status, netkv_stream_t stream) {
  if (R > NETKV_PREFIX_MATCH_STATIC_MAX_R ||
      netkv_prefix_match_workspace_size(R) > kStaticScratchBytes)
    return NETKV_ELIMIT;
  void* scratch = nullptr;
  const netkv_status st = static_scratch((cudaStream_t)stream, &scratch);
  if (st != NETKV_OK) return st;
  return netkv_prefix_match(d_index, D, log2_capacity, n_sets, d_chains, d_chain_off, R,
                            d_set_off, scratch, kStaticScratchBytes, d_M, d_status, stream);
}
