// Decode caches K_d and the block-level prefix hit of Sec. III-B:
// M[r][d] = |LCP_block(h_r, K_d)|, the number of leading blocks of request r's hash chain
// that are all cached on decode d.
//
// Cache index.  The caches of a table set are stored as an inverted index: one
// open-addressing table per group of up to 64 decodes, whose 16-byte slots hold a block
// hash and a 64-bit mask of the group's decodes that cache it.  One probe therefore
// answers the membership question for every decode of the group at once; the decodes
// of a set mostly cache the same shared prefixes, so this also keeps the index small.
//   cache_insert_kernel: one block per (set, decode) key list; linear probing from a
//   Fibonacci-hashed home slot, atomicCAS to claim the slot, atomicOr to add the decode.
//
// Match.  One warp per (request, decode group).  The warp first probes the block at the
// starting position (one probe serves the whole group), then walks the chain in chunks of
// 32 consecutive blocks: a 256-byte coalesced chain load, one index probe per lane, and one
// ballot per live decode to find its first missing block; a decode leaves once its first
// miss is known and the warp stops when every decode of the group has missed.  Probes are
// bounded by the table size.
//
// Prefix sharing.  Requests that share leading blocks have the same membership answers
// on those blocks, so with a workspace the match runs in three steps:
//   group_insert_kernel / group_resolve_kernel: requests are grouped by (table set,
//     first block hash) in an open-addressing table; each group's leader is its
//     longest chain (lowest index among equals); leaders go to a compact list.
//   match_leaders_kernel: leaders (and ungrouped requests) run the full match, one task
//     per (leader, decode group) taken in order from a counter.
//   match_kernel<kMembers>: a member r with leader L compares chains to get
//     lcp = |common prefix of h_r and h_L| (capped at max_d M_L[d] + 1).  For a decode
//     with M_L[d] < lcp the first missing block of L lies inside the common prefix, so
//     M_r[d] = M_L[d] exactly; otherwise blocks [0, lcp) are all cached and the probe
//     resumes at block lcp.  The result equals the full match whatever the grouping;
//     grouping only decides how much probing is saved.
#include "netkv_internal.cuh"

namespace {

constexpr int kInsertBlock = 256;
constexpr int kMatchBlock = 256;
constexpr uint32_t kGroup = 64;  // decodes per index table (bits of the mask)

struct __align__(16) IndexSlot {
  unsigned long long key;
  unsigned long long mask;
};

__global__ void __launch_bounds__(kInsertBlock) cache_insert_kernel(
    IndexSlot* __restrict__ index, uint32_t n_sets, uint32_t D, uint32_t log2_cap,
    const uint64_t* __restrict__ keys, const uint64_t* __restrict__ key_off, int* status) {
  const uint64_t cap = 1ull << log2_cap, mask = cap - 1;
  const uint32_t n_dgroups = (D + kGroup - 1) / kGroup;
  const uint64_t n_lists = (uint64_t)n_sets * D;
  for (uint64_t t = blockIdx.x; t < n_lists; t += gridDim.x) {
    const uint64_t beg = __ldg(key_off + t), end = __ldg(key_off + t + 1);
    if (end < beg) {
      if (threadIdx.x == 0) flag_status(status, NETKV_DEV_ERANGE);
      continue;
    }
    const uint64_t g = t / D;
    const uint32_t d = (uint32_t)(t - g * D);
    IndexSlot* tab = index + ((g * n_dgroups + d / kGroup) << log2_cap);
    const unsigned long long bit = 1ull << (d % kGroup);
    for (uint64_t j = beg + threadIdx.x; j < end; j += blockDim.x) {
      const unsigned long long key = __ldg(keys + j);
      if (key == 0ull) {
        flag_status(status, NETKV_DEV_EDOMAIN);
        continue;
      }
      uint64_t slot = home_slot(key, log2_cap);
      uint64_t step = 0;
      for (; step < cap; ++step) {
        const unsigned long long prev = atomicCAS(&tab[slot].key, 0ull, key);
        if (prev == 0ull || prev == key) {
          atomicOr(&tab[slot].mask, bit);
          break;
        }
        slot = (slot + 1) & mask;
      }
      if (step == cap) flag_status(status, NETKV_DEV_EFULL);
    }
  }
}

// Decodes of the group that cache `key` (non-zero); 0 when absent.
__device__ __forceinline__ unsigned long long lookup(const IndexSlot* __restrict__ tab,
                                                     uint64_t key, uint32_t log2_cap,
                                                     int* status) {
  const uint64_t mask = (1ull << log2_cap) - 1;
  uint64_t slot = home_slot(key, log2_cap);
  for (uint64_t seen = 0; seen <= mask; ++seen) {
    const ulonglong2 s = __ldg(reinterpret_cast<const ulonglong2*>(tab + slot));
    if (s.x == key) return s.y;
    if (s.x == 0ull) return 0ull;
    slot = (slot + 1) & mask;
  }
  flag_status(status, NETKV_DEV_EFULL);
  return 0ull;
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

// First-miss scan of blocks [start, n) of one chain for the `alive` decodes of a group.
// Decodes found missing at position p get p; decodes never missing keep their value.
__device__ __forceinline__ void scan_chain(const IndexSlot* __restrict__ tab, uint32_t log2_cap,
                                           const uint64_t* __restrict__ chain, uint64_t start,
                                           uint64_t n, unsigned long long alive, GroupHits& h,
                                           uint32_t lane, int* status) {
  if (!alive || start >= n) return;
  {  // the first block: one probe for the whole group
    const uint64_t key = __ldg(chain + start);
    unsigned long long mk = 0ull;
    if (key == 0ull) {
      if (lane == 0) flag_status(status, NETKV_DEV_EDOMAIN);
    } else if (lane == 0) {
      mk = lookup(tab, key, log2_cap, status);
    }
    mk = __shfl_sync(0xffffffffu, mk, 0);
    unsigned long long miss = alive & ~mk;
    while (miss) {
      const uint32_t j = __ffsll((long long)miss) - 1;
      miss &= miss - 1;
      set_hit(h, lane, j, (uint32_t)start);
    }
    alive &= mk;
    ++start;
  }
  for (uint64_t base = start; base < n && alive; base += 32) {
    const uint64_t i = base + lane;
    const bool in = i < n;
    const uint64_t key = in ? __ldcs(chain + i) : 0ull;
    if (in && key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
    const unsigned long long mk = (in && key != 0ull) ? lookup(tab, key, log2_cap, status) : 0ull;
    const uint32_t valid = __ballot_sync(0xffffffffu, in);
    unsigned long long a = alive;
    while (a) {
      const uint32_t j = __ffsll((long long)a) - 1;
      a &= a - 1;
      const uint32_t miss = valid & ~__ballot_sync(0xffffffffu, (mk >> j) & 1ull);
      if (miss) {
        set_hit(h, lane, j, (uint32_t)base + (uint32_t)(__ffs(miss) - 1));
        alive &= ~(1ull << j);
      }
    }
  }
}

enum MatchMode { kAll = 0, kMembers = 2 };

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
  unsigned long long n_leaders;  // entries of the leader list
  unsigned long long next_task;  // next (leader, decode group) task of the leader pass
};

__global__ void group_insert_kernel(GroupSlot* __restrict__ tab, uint32_t log2_slots,
                                    const uint64_t* __restrict__ chains,
                                    const uint64_t* __restrict__ chain_off, uint32_t R,
                                    const uint32_t* __restrict__ set_off, uint32_t n_sets) {
  const uint64_t mask = (1ull << log2_slots) - 1;
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    const int32_t set = find_set(set_off, n_sets, r);
    if (c1 <= c0 || set < 0) continue;
    const uint64_t n = c1 - c0;
    const uint64_t key = group_key(__ldg(chains + c0), (uint32_t)set);
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

__global__ void group_resolve_kernel(const GroupSlot* __restrict__ tab, uint32_t log2_slots,
                                     const uint64_t* __restrict__ chains,
                                     const uint64_t* __restrict__ chain_off, uint32_t R,
                                     const uint32_t* __restrict__ set_off, uint32_t n_sets,
                                     uint32_t* __restrict__ leader_of,
                                     uint32_t* __restrict__ leaders, MatchCounters* counters) {
  const uint64_t mask = (1ull << log2_slots) - 1;
  for (uint32_t r = blockIdx.x * blockDim.x + threadIdx.x; r < R; r += gridDim.x * blockDim.x) {
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    const int32_t set = find_set(set_off, n_sets, r);
    uint32_t lead = r;
    if (c1 > c0 && set >= 0) {
      const uint64_t key = group_key(__ldg(chains + c0), (uint32_t)set);
      uint64_t slot = home_slot(key, log2_slots);
      for (uint64_t step = 0; step <= mask; ++step) {
        const unsigned long long k = tab[slot].key;
        if (k == key) {
          const uint32_t L = 0xffffffffu - (uint32_t)(tab[slot].code & 0xffffffffull);
          // a leader from another table set (64-bit key collision) is never used
          if (L < R && find_set(set_off, n_sets, L) == set) lead = L;
          break;
        }
        if (k == 0ull) break;
        slot = (slot + 1) & mask;
      }
    }
    leader_of[r] = lead;
    if (lead == r) leaders[atomicAdd(&counters->n_leaders, 1ull)] = r;
  }
}

// Chain r's extent clamped to 65535 blocks; false on a bad request (flagged).
__device__ __forceinline__ bool chain_extent(const uint64_t* __restrict__ chain_off,
                                             const uint32_t* __restrict__ set_off,
                                             uint32_t n_sets, uint32_t r, uint32_t lane,
                                             int* status, int32_t& set, uint64_t& c0,
                                             uint64_t& n) {
  set = find_set(set_off, n_sets, r);
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
__global__ void __launch_bounds__(kMatchBlock) match_leaders_kernel(
    const IndexSlot* __restrict__ index, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off,
    const uint32_t* __restrict__ set_off, const uint32_t* __restrict__ leaders,
    MatchCounters* counters, uint16_t* __restrict__ M, int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t n_dgroups = (D + kGroup - 1) / kGroup;
  const unsigned long long total =
      *((volatile unsigned long long*)&counters->n_leaders) * n_dgroups;
  for (;;) {
    unsigned long long t = 0;
    if (lane == 0) t = atomicAdd(&counters->next_task, 1ull);
    t = __shfl_sync(0xffffffffu, t, 0);
    if (t >= total) break;
    const uint32_t r = __ldg(leaders + t / n_dgroups);
    const uint32_t q = (uint32_t)(t % n_dgroups);
    const uint32_t q0 = q * kGroup, ng = min(kGroup, D - q0);
    GroupHits h = {0u, 0u};
    int32_t set;
    uint64_t c0, n;
    if (chain_extent(chain_off, set_off, n_sets, r, lane, status, set, c0, n)) {
      h.lo = h.hi = (uint32_t)n;
      const unsigned long long alive = ng >= 64 ? ~0ull : ((1ull << ng) - 1);
      const IndexSlot* tab = index + (((uint64_t)set * n_dgroups + q) << log2_cap);
      scan_chain(tab, log2_cap, chains + c0, 0, n, alive, h, lane, status);
    }
    store_hits(M, (uint64_t)r * D, q0, ng, lane, h);
  }
}

template <int kMode>
__global__ void __launch_bounds__(kMatchBlock) match_kernel(
    const IndexSlot* __restrict__ index, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off, uint32_t R,
    const uint32_t* __restrict__ set_off, const uint32_t* __restrict__ leader_of,
    uint16_t* __restrict__ M, int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t n_dgroups = (D + kGroup - 1) / kGroup;
  const uint64_t total = (uint64_t)R * n_dgroups;

  for (uint64_t task = warp; task < total; task += n_warps) {
    const uint32_t r = (uint32_t)(task / n_dgroups);
    uint32_t lead = r;
    if (kMode == kMembers) {
      lead = __ldg(leader_of + r);
      if (lead == r) continue;  // leaders were matched by the leader pass
    }
    const uint32_t q = (uint32_t)(task - (uint64_t)r * n_dgroups);
    const uint32_t q0 = q * kGroup, ng = min(kGroup, D - q0);
    GroupHits h = {0u, 0u};
    int32_t set;
    uint64_t c0, n;
    if (!chain_extent(chain_off, set_off, n_sets, r, lane, status, set, c0, n)) {
      store_hits(M, (uint64_t)r * D, q0, ng, lane, h);
      continue;
    }
    h.lo = h.hi = (uint32_t)n;
    unsigned long long alive = ng >= 64 ? ~0ull : ((1ull << ng) - 1);
    uint64_t start = 0;
    if (kMode == kMembers) {
      // the leader's hits for this group and the common prefix of the two chains
      const uint64_t lrow = (uint64_t)lead * D + q0;
      const uint32_t mlo = lane < ng ? (uint32_t)__ldg(M + lrow + lane) : 0u;
      const uint32_t mhi = lane + 32 < ng ? (uint32_t)__ldg(M + lrow + lane + 32) : 0u;
      uint32_t mmax = max(mlo, mhi);
#pragma unroll
      for (int o = 16; o; o >>= 1) mmax = max(mmax, __shfl_xor_sync(0xffffffffu, mmax, o));
      const uint64_t l0 = __ldg(chain_off + lead), l1 = __ldg(chain_off + lead + 1);
      const uint64_t cap = min(n, min(l1 - l0, (uint64_t)mmax + 1));
      uint64_t lcp = cap;  // common prefix, 128 blocks per step
      for (uint64_t base = 0; base < cap; base += 128) {
        uint64_t a[4], b[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const uint64_t i = base + 32 * k + lane;
          a[k] = i < cap ? __ldcs(chains + c0 + i) : 0ull;
          b[k] = i < cap ? __ldg(chains + l0 + i) : 0ull;
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
      // decodes whose leader missed inside the common prefix copy the leader's answer
      const uint32_t clo = __ballot_sync(0xffffffffu, lane < ng && (uint64_t)mlo < lcp);
      const uint32_t chi = __ballot_sync(0xffffffffu, lane + 32 < ng && (uint64_t)mhi < lcp);
      const unsigned long long copy = (unsigned long long)clo | ((unsigned long long)chi << 32);
      if ((clo >> lane) & 1u) h.lo = mlo;
      if ((chi >> lane) & 1u) h.hi = mhi;
      alive &= ~copy;
      start = lcp;
    }
    const IndexSlot* tab = index + (((uint64_t)set * n_dgroups + q) << log2_cap);
    scan_chain(tab, log2_cap, chains + c0, start, n, alive, h, lane, status);
    store_hits(M, (uint64_t)r * D, q0, ng, lane, h);
  }
}

uint32_t group_log2_slots(uint32_t R) {
  uint32_t l = 1;
  while ((1ull << l) < 2ull * R) ++l;
  return l;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Workspace: group table | leader_of [R] | leader list [R] | counters.
struct WorkspaceLayout {
  size_t table, leader_of, leaders, counters, total;
};

WorkspaceLayout workspace_layout(uint32_t R) {
  WorkspaceLayout w;
  w.table = 0;
  w.leader_of = align_up(sizeof(GroupSlot) << group_log2_slots(R), 256);
  w.leaders = w.leader_of + align_up(sizeof(uint32_t) * (size_t)R, 256);
  w.counters = w.leaders + align_up(sizeof(uint32_t) * (size_t)R, 256);
  w.total = w.counters + align_up(sizeof(MatchCounters), 256);
  return w;
}

int leader_grid() {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, match_leaders_kernel, kMatchBlock, 0);
  return (sms > 0 ? sms : 1) * (per_sm > 0 ? per_sm : 1);
}

}  // namespace

extern "C" size_t netkv_cache_index_bytes(uint32_t n_sets, uint32_t D, uint32_t log2_capacity) {
  if (log2_capacity < 1 || log2_capacity > 32) return 0;
  return (size_t)n_sets * ((D + kGroup - 1) / kGroup) * (sizeof(IndexSlot) << log2_capacity);
}

extern "C" netkv_status netkv_cache_build(void* d_index, uint32_t n_sets, uint32_t D,
                                          uint32_t log2_capacity, const uint64_t* d_keys,
                                          const uint64_t* d_key_off, int* d_status,
                                          netkv_stream_t stream) {
  if (!d_index || !d_key_off || D == 0 || log2_capacity < 1 || log2_capacity > 32)
    return NETKV_EINVAL;
  if (!aligned_to(d_index, 16) || !aligned_to(d_key_off, 8) || (d_keys && !aligned_to(d_keys, 8)))
    return NETKV_EINVAL;
  if (n_sets == 0) return NETKV_OK;
  cudaStream_t s = (cudaStream_t)stream;
  NETKV_CUDA_TRY(cudaMemsetAsync(d_index, 0, netkv_cache_index_bytes(n_sets, D, log2_capacity), s));
  if (!d_keys) return NETKV_OK;
  const uint64_t lists = (uint64_t)n_sets * D;
  const unsigned grid = (unsigned)(lists < (1u << 20) ? lists : (1u << 20));
  cache_insert_kernel<<<grid, kInsertBlock, 0, s>>>(reinterpret_cast<IndexSlot*>(d_index), n_sets,
                                                    D, log2_capacity, d_keys, d_key_off, d_status);
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
  if (log2_capacity < 1 || log2_capacity > 32) return NETKV_EINVAL;
  if (n_sets > 1 && !d_set_off) return NETKV_EINVAL;
  if (!aligned_to(d_index, 16) || !aligned_to(d_chain_off, 8) || !aligned_to(d_M, 2) ||
      (d_chains && !aligned_to(d_chains, 8)) || (d_set_off && !aligned_to(d_set_off, 4)) ||
      (d_workspace && !aligned_to(d_workspace, 256)))
    return NETKV_EINVAL;
  if (R == 0) return NETKV_OK;
  if (!d_chains || R > 0x7fffffffu) return NETKV_EINVAL;
  if (d_workspace && workspace_bytes < netkv_prefix_match_workspace_size(R)) return NETKV_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  const IndexSlot* index = reinterpret_cast<const IndexSlot*>(d_index);
  const uint64_t tasks = (uint64_t)R * ((D + kGroup - 1) / kGroup);
  const uint64_t warps_per_block = kMatchBlock / 32;
  const uint64_t blocks = (tasks + warps_per_block - 1) / warps_per_block;
  const unsigned grid = (unsigned)(blocks < (1u << 24) ? blocks : (1u << 24));
  if (!d_workspace) {
    match_kernel<kAll><<<grid, kMatchBlock, 0, s>>>(index, D, log2_capacity, n_sets, d_chains,
                                                    d_chain_off, R, d_set_off, nullptr, d_M,
                                                    d_status);
    return netkv_launch_status();
  }
  const uint32_t lg = group_log2_slots(R);
  const WorkspaceLayout L = workspace_layout(R);
  char* ws = reinterpret_cast<char*>(d_workspace);
  GroupSlot* tab = reinterpret_cast<GroupSlot*>(ws + L.table);
  uint32_t* leader_of = reinterpret_cast<uint32_t*>(ws + L.leader_of);
  uint32_t* leaders = reinterpret_cast<uint32_t*>(ws + L.leaders);
  MatchCounters* counters = reinterpret_cast<MatchCounters*>(ws + L.counters);
  NETKV_CUDA_TRY(cudaMemsetAsync(tab, 0, sizeof(GroupSlot) << lg, s));
  NETKV_CUDA_TRY(cudaMemsetAsync(counters, 0, sizeof(MatchCounters), s));
  const unsigned rgrid = (unsigned)((R + 255) / 256 < 65535u * 16 ? (R + 255) / 256 : 65535u * 16);
  group_insert_kernel<<<rgrid, 256, 0, s>>>(tab, lg, d_chains, d_chain_off, R, d_set_off, n_sets);
  group_resolve_kernel<<<rgrid, 256, 0, s>>>(tab, lg, d_chains, d_chain_off, R, d_set_off, n_sets,
                                             leader_of, leaders, counters);
  match_leaders_kernel<<<leader_grid(), kMatchBlock, 0, s>>>(
      index, D, log2_capacity, n_sets, d_chains, d_chain_off, d_set_off, leaders, counters, d_M,
      d_status);
  match_kernel<kMembers><<<grid, kMatchBlock, 0, s>>>(index, D, log2_capacity, n_sets, d_chains,
                                                      d_chain_off, R, d_set_off, leader_of, d_M,
                                                      d_status);
  return netkv_launch_status();
}

// ---------------------------------------------------------------------------------
// netkv_prefix_match_static: the prefix match for callers that cannot allocate device
// memory (see include/netkv.h).  Its workspace is this fixed device array, shared by
// every call on a device; the device address is looked up once per device.
// ---------------------------------------------------------------------------------
#include <mutex>

namespace {

constexpr size_t kStaticScratchBytes = 24ull << 20;  // 24 MiB per device
static __device__ __align__(256) unsigned char g_prefix_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_prefix_scratch on the current device (looked up on first use).
netkv_status static_scratch(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return NETKV_ECUDA;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (!g_scratch_addr[dev]) {
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
  const netkv_status st = static_scratch(&scratch);
  if (st != NETKV_OK) return st;
  return netkv_prefix_match(d_index, D, log2_capacity, n_sets, d_chains, d_chain_off, R,
                            d_set_off, scratch, kStaticScratchBytes, d_M, d_status, stream);
}
