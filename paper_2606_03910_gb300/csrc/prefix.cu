// Decode caches K_d as open-addressing hash tables and the block-level prefix hit of
// Sec. III-B: M[r][d] = |LCP_block(h_r, K_d)|, the number of leading blocks of request
// r's hash chain that are all cached on decode d.
//
// cache_insert_kernel: one block per table, threads stride over that table's keys,
//   linear probing with atomicCAS from a Fibonacci-hashed home slot.
// match_kernel: one warp per (request, group of up to 8 decode tables).  The warp first
//   probes the chain's first block in every table of the group at once (one lane per
//   table), then walks the rest in chunks of 32 consecutive blocks (one 256-byte
//   coalesced load); every live decode of the group probes with all 32 keys and a
//   ballot finds the first miss; a decode whose first miss is found leaves the group
//   and the warp stops as soon as every decode has missed.  Probes read 16-byte slot
//   pairs, bounded by the table size.
//
// Prefix sharing.  Requests that share leading blocks have the same membership answers
// on those blocks, so with a workspace the match runs in three steps:
//   group_insert_kernel / group_resolve_kernel: requests are grouped by (table set,
//     first block hash) in an open-addressing table; each group's leader is its
//     longest chain (lowest index among equals).
//   match_leaders_kernel: leaders (and ungrouped requests) run the full match, one task
//     per (leader, decode) taken in order from a counter.
//   match_kernel<kMembers>: a member r with leader L compares chains to get
//     lcp = |common prefix of h_r and h_L| (capped at max_d M_L[d] + 1).  For a decode
//     with M_L[d] < lcp the first missing block of L lies inside the common prefix,
//     so M_r[d] = M_L[d] exactly; otherwise blocks [0, lcp) are all cached and the
//     probe resumes at block lcp.  The result equals the full match whatever the
//     grouping; grouping only decides how much probing is saved.
#include "netkv_internal.cuh"

namespace {

constexpr int kInsertBlock = 256;
constexpr int kMatchBlock = 256;
constexpr int kGroup = 8;

__global__ void __launch_bounds__(kInsertBlock) cache_insert_kernel(
    unsigned long long* __restrict__ tables, uint64_t n_tables, uint32_t log2_cap,
    const uint64_t* __restrict__ keys, const uint64_t* __restrict__ key_off, int* status) {
  const uint64_t cap = 1ull << log2_cap, mask = cap - 1;
  for (uint64_t t = blockIdx.x; t < n_tables; t += gridDim.x) {
    const uint64_t beg = __ldg(key_off + t), end = __ldg(key_off + t + 1);
    if (end < beg) {
      if (threadIdx.x == 0) flag_status(status, NETKV_DEV_ERANGE);
      continue;
    }
    unsigned long long* tab = tables + (t << log2_cap);
    for (uint64_t j = beg + threadIdx.x; j < end; j += blockDim.x) {
      const unsigned long long key = __ldg(keys + j);
      if (key == 0ull) {
        flag_status(status, NETKV_DEV_EDOMAIN);
        continue;
      }
      uint64_t slot = home_slot(key, log2_cap);
      uint64_t step = 0;
      for (; step < cap; ++step) {
        const unsigned long long prev = atomicCAS(tab + slot, 0ull, key);
        if (prev == 0ull || prev == key) break;
        slot = (slot + 1) & mask;
      }
      if (step == cap) flag_status(status, NETKV_DEV_EFULL);
    }
  }
}

// Membership of `key` (non-zero) in one table; reads aligned slot pairs.
__device__ __forceinline__ bool probe(const uint64_t* __restrict__ tab, uint64_t key,
                                      uint32_t log2_cap, int* status) {
  const uint64_t mask = (1ull << log2_cap) - 1;
  uint64_t slot = home_slot(key, log2_cap);
  // visit slot, slot+1, ... in pairs [2q, 2q+1]; the first pair may start at its odd half
  for (uint64_t seen = 0; seen <= mask;) {
    const ulonglong2 pr = __ldg(reinterpret_cast<const ulonglong2*>(tab + (slot & ~1ull)));
    if (!(slot & 1)) {
      if (pr.x == key) return true;
      if (pr.x == 0) return false;
      ++seen;
    }
    if (pr.y == key) return true;
    if (pr.y == 0) return false;
    ++seen;
    slot = ((slot | 1ull) + 1) & mask;
  }
  flag_status(status, NETKV_DEV_EFULL);
  return false;
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

enum MatchMode { kAll = 0, kLeaders = 1, kMembers = 2 };

constexpr uint32_t kNoLeader = 0xffffffffu;

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

// Work counters at the end of the workspace.
struct MatchCounters {
  unsigned long long n_leaders;   // entries of the leader list
  unsigned long long next_task;   // next (leader, decode) task of the leader pass
};

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

// Leader pass: one task per (leader, decode), taken in order from a global counter by
// whole warps, so long and short chains balance across the GPU and the eight decodes
// of a leader run in parallel.  Each task is the full first-miss scan of one chain
// against one table: block 0 alone, then chunks of 32 blocks with a ballot.
__global__ void __launch_bounds__(kMatchBlock) match_leaders_kernel(
    const uint64_t* __restrict__ tables, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off,
    const uint32_t* __restrict__ set_off, const uint32_t* __restrict__ leaders,
    MatchCounters* counters, uint16_t* __restrict__ M, int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const unsigned long long total = *((volatile unsigned long long*)&counters->n_leaders) * D;
  for (;;) {
    unsigned long long t = 0;
    if (lane == 0) t = atomicAdd(&counters->next_task, 1ull);
    t = __shfl_sync(0xffffffffu, t, 0);
    if (t >= total) break;
    const uint32_t r = __ldg(leaders + t / D);
    const uint32_t d = (uint32_t)(t % D);
    const int32_t set = find_set(set_off, n_sets, r);
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    if (set < 0 || c1 < c0) {
      if (lane == 0) {
        flag_status(status, NETKV_DEV_ERANGE);
        M[(uint64_t)r * D + d] = 0;
      }
      continue;
    }
    uint64_t n = c1 - c0;
    if (n > 65535) {
      if (lane == 0) flag_status(status, NETKV_DEV_EDOMAIN);
      n = 65535;
    }
    const uint64_t* tab = tables + (((uint64_t)set * D + d) << log2_cap);
    uint64_t m = n;
    for (uint64_t base = 0; base < n; base += 32) {
      const uint64_t i = base + lane;
      const bool in = i < n;
      const uint64_t key = in ? __ldcs(chains + c0 + i) : 0ull;
      if (in && key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
      const bool hit = in && key != 0ull && probe(tab, key, log2_cap, status);
      const uint32_t miss = __ballot_sync(0xffffffffu, in && !hit);
      if (miss) {
        m = base + (uint64_t)(__ffs(miss) - 1);
        break;
      }
    }
    if (lane == 0) M[(uint64_t)r * D + d] = (uint16_t)m;
  }
}

template <int kMode>
__global__ void __launch_bounds__(kMatchBlock) match_kernel(
    const uint64_t* __restrict__ tables, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off, uint32_t R,
    const uint32_t* __restrict__ set_off, const uint32_t* __restrict__ leader_of,
    uint16_t* __restrict__ M, int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t n_groups = (D + kGroup - 1) / kGroup;
  const uint64_t total = (uint64_t)R * n_groups;

  for (uint64_t task = warp; task < total; task += n_warps) {
    const uint32_t r = (uint32_t)(task / n_groups);
    uint32_t lead = r;
    if (kMode != kAll) {
      lead = __ldg(leader_of + r);
      if ((kMode == kLeaders) != (lead == r)) continue;   // warp-uniform
    }
    const uint32_t g0 = (uint32_t)(task - (uint64_t)r * n_groups) * kGroup;
    const uint32_t ng = min((uint32_t)kGroup, D - g0);
    const int32_t set = find_set(set_off, n_sets, r);
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    uint32_t m_lane = 0;
    if (set < 0 || c1 < c0) {
      if (lane == 0) flag_status(status, NETKV_DEV_ERANGE);
      if (lane < ng) M[(uint64_t)r * D + g0 + lane] = 0;
      continue;
    }
    uint64_t n = c1 - c0;
    if (n > 65535) {
      if (lane == 0) flag_status(status, NETKV_DEV_EDOMAIN);
      n = 65535;
    }
    uint32_t alive = (1u << ng) - 1;
    uint64_t start = 0;
    if (kMode == kMembers) {
      // leader's hits for this group and the common prefix of the two chains
      const uint32_t mL = lane < ng ? (uint32_t)__ldg(M + (uint64_t)lead * D + g0 + lane) : 0u;
      uint32_t mmax = mL;
#pragma unroll
      for (int o = 16; o; o >>= 1) mmax = max(mmax, __shfl_xor_sync(0xffffffffu, mmax, o));
      const uint64_t l0 = __ldg(chain_off + lead), l1 = __ldg(chain_off + lead + 1);
      uint64_t cap = min(n, min(l1 - l0, (uint64_t)mmax + 1));
      // common prefix, 128 blocks (four independent loads per lane and chain) per step
      uint64_t lcp = cap;
      for (uint64_t base = 0; base < cap; base += 128) {
        uint64_t a[4], b[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint64_t i = base + 32 * q + lane;
          a[q] = i < cap ? __ldcs(chains + c0 + i) : 0ull;
          b[q] = i < cap ? __ldg(chains + l0 + i) : 0ull;
        }
        uint64_t found = cap;
#pragma unroll
        for (int q = 3; q >= 0; --q) {
          const uint32_t diff = __ballot_sync(0xffffffffu, a[q] != b[q]);
          if (diff) found = base + 32 * q + (uint64_t)(__ffs(diff) - 1);
        }
        if (found < cap) {
          lcp = found;
          break;
        }
      }
      // decodes whose leader missed inside the common prefix copy the leader's answer
      const uint32_t copy = __ballot_sync(0xffffffffu, lane < ng && (uint64_t)mL < lcp);
      if (lane < ng && ((copy >> lane) & 1u)) m_lane = mL;
      alive &= ~copy;
      start = lcp;
    }
    if (lane < ng && ((alive >> lane) & 1u)) m_lane = (uint32_t)n;
    const uint64_t* tab0 = tables + (((uint64_t)set * D + g0) << log2_cap);
    // first block after `start`: one lane per table
    if (alive && start < n) {
      const uint64_t key = __ldg(chains + c0 + start);
      if (key == 0ull && lane == 0) flag_status(status, NETKV_DEV_EDOMAIN);
      const bool hit = lane < ng && ((alive >> lane) & 1u) && key != 0ull &&
                       probe(tab0 + ((uint64_t)lane << log2_cap), key, log2_cap, status);
      const uint32_t miss = alive & ~__ballot_sync(0xffffffffu, hit);
      if ((miss >> lane) & 1u) m_lane = (uint32_t)start;
      alive &= ~miss;
      ++start;
    }
    for (uint64_t base = start; base < n && alive; base += 32) {
      const uint64_t i = base + lane;
      const bool in = i < n;
      const uint64_t key = in ? __ldcs(chains + c0 + i) : 0ull;
      if (in && key == 0ull) flag_status(status, NETKV_DEV_EDOMAIN);
      const uint32_t valid = __ballot_sync(0xffffffffu, in);
      uint32_t a = alive;
      while (a) {
        const int j = __ffs(a) - 1;
        a &= a - 1;
        const bool hit = in && key != 0ull &&
                         probe(tab0 + ((uint64_t)j << log2_cap), key, log2_cap, status);
        const uint32_t miss = valid & ~__ballot_sync(0xffffffffu, hit);
        if (miss) {
          if (lane == (uint32_t)j) m_lane = (uint32_t)base + (uint32_t)(__ffs(miss) - 1);
          alive &= ~(1u << j);
        }
      }
    }
    if (lane < ng) M[(uint64_t)r * D + g0 + lane] = (uint16_t)m_lane;
  }
}

}  // namespace

extern "C" netkv_status netkv_cache_build(uint64_t* d_tables, uint64_t n_tables,
                                          uint32_t log2_capacity, const uint64_t* d_keys,
                                          const uint64_t* d_key_off, int* d_status,
                                          netkv_stream_t stream) {
  if (!d_tables || !d_key_off || log2_capacity < 1 || log2_capacity > 32) return NETKV_EINVAL;
  if (!aligned_to(d_tables, 16) || !aligned_to(d_key_off, 8) || (d_keys && !aligned_to(d_keys, 8)))
    return NETKV_EINVAL;
  if (n_tables == 0) return NETKV_OK;
  if (n_tables > (UINT64_MAX >> 3 >> log2_capacity)) return NETKV_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  NETKV_CUDA_TRY(cudaMemsetAsync(d_tables, 0, (n_tables << log2_capacity) * sizeof(uint64_t), s));
  if (!d_keys) return NETKV_OK;
  const unsigned grid = (unsigned)(n_tables < (1u << 20) ? n_tables : (1u << 20));
  cache_insert_kernel<<<grid, kInsertBlock, 0, s>>>(
      reinterpret_cast<unsigned long long*>(d_tables), n_tables, log2_capacity, d_keys, d_key_off,
      d_status);
  return netkv_launch_status();
}

namespace {

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

extern "C" size_t netkv_prefix_match_workspace_size(uint32_t R) {
  if (R == 0) return 0;
  return workspace_layout(R).total;
}

extern "C" netkv_status netkv_prefix_match(const uint64_t* d_tables, uint32_t D,
                                           uint32_t log2_capacity, uint32_t n_sets,
                                           const uint64_t* d_chains, const uint64_t* d_chain_off,
                                           uint32_t R, const uint32_t* d_set_off,
                                           void* d_workspace, size_t workspace_bytes,
                                           uint16_t* d_M, int* d_status, netkv_stream_t stream) {
  if (!d_tables || !d_chain_off || !d_M || D == 0 || n_sets == 0) return NETKV_EINVAL;
  if (log2_capacity < 1 || log2_capacity > 32) return NETKV_EINVAL;
  if (n_sets > 1 && !d_set_off) return NETKV_EINVAL;
  if (!aligned_to(d_tables, 16) || !aligned_to(d_chain_off, 8) || !aligned_to(d_M, 2) ||
      (d_chains && !aligned_to(d_chains, 8)) || (d_set_off && !aligned_to(d_set_off, 4)) ||
      (d_workspace && !aligned_to(d_workspace, 256)))
    return NETKV_EINVAL;
  if (R == 0) return NETKV_OK;
  if (!d_chains || R > 0x7fffffffu) return NETKV_EINVAL;
  if (d_workspace && workspace_bytes < netkv_prefix_match_workspace_size(R)) return NETKV_EINVAL;
  cudaStream_t s = (cudaStream_t)stream;
  const uint64_t tasks = (uint64_t)R * ((D + kGroup - 1) / kGroup);
  const uint64_t warps_per_block = kMatchBlock / 32;
  const uint64_t blocks = (tasks + warps_per_block - 1) / warps_per_block;
  const unsigned grid = (unsigned)(blocks < (1u << 24) ? blocks : (1u << 24));
  if (!d_workspace) {
    match_kernel<kAll><<<grid, kMatchBlock, 0, s>>>(d_tables, D, log2_capacity, n_sets, d_chains,
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
      d_tables, D, log2_capacity, n_sets, d_chains, d_chain_off, d_set_off, leaders, counters, d_M,
      d_status);
  match_kernel<kMembers><<<grid, kMatchBlock, 0, s>>>(d_tables, D, log2_capacity, n_sets, d_chains,
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

extern "C" netkv_status netkv_prefix_match_static(const uint64_t* d_tables, uint32_t D,
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
  return netkv_prefix_match(d_tables, D, log2_capacity, n_sets, d_chains, d_chain_off, R,
                            d_set_off, scratch, kStaticScratchBytes, d_M, d_status, stream);
}
