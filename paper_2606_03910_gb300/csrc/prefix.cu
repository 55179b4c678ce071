// Decode caches K_d as open-addressing hash tables and the block-level prefix hit of
// Sec. III-B: M[r][d] = |LCP_block(h_r, K_d)|, the number of leading blocks of request
// r's hash chain that are all cached on decode d.
//
// cache_insert_kernel: one block per table, threads stride over that table's keys,
//   linear probing with atomicCAS from a Fibonacci-hashed home slot.
// prefix_match_kernel: one warp per (request, group of up to 8 decode tables).  The
//   warp loads 32 consecutive chain blocks (one 256-byte coalesced load), every live
//   decode of the group probes its table with all 32 keys at once, and a ballot finds
//   the first block that missed; a decode whose first miss is found leaves the group,
//   and the warp stops as soon as every decode of the group has missed, so at most 31
//   blocks past the first miss are probed.  The chain chunk is reused by every decode
//   of the group.  Probes read 16-byte slot pairs (two slots per load), bounded by the
//   table size so no probe can loop forever.
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

__global__ void __launch_bounds__(kMatchBlock) prefix_match_kernel(
    const uint64_t* __restrict__ tables, uint32_t D, uint32_t log2_cap, uint32_t n_sets,
    const uint64_t* __restrict__ chains, const uint64_t* __restrict__ chain_off, uint32_t R,
    const uint32_t* __restrict__ set_off, uint16_t* __restrict__ M, int* status) {
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t warp = ((uint64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const uint64_t n_warps = ((uint64_t)gridDim.x * blockDim.x) >> 5;
  const uint32_t n_groups = (D + kGroup - 1) / kGroup;
  const uint64_t total = (uint64_t)R * n_groups;

  for (uint64_t task = warp; task < total; task += n_warps) {
    const uint32_t r = (uint32_t)(task / n_groups);
    const uint32_t g0 = (uint32_t)(task - (uint64_t)r * n_groups) * kGroup;
    const uint32_t ng = min((uint32_t)kGroup, D - g0);
    const int32_t set = find_set(set_off, n_sets, r);
    const uint64_t c0 = __ldg(chain_off + r), c1 = __ldg(chain_off + r + 1);
    uint32_t m_lane = 0;
    if (set < 0 || c1 < c0) {
      if (lane == 0) flag_status(status, NETKV_DEV_ERANGE);
    } else {
      uint64_t n = c1 - c0;
      if (n > 65535) {
        if (lane == 0) flag_status(status, NETKV_DEV_EDOMAIN);
        n = 65535;
      }
      m_lane = (uint32_t)n;
      const uint64_t* tab0 = tables + (((uint64_t)set * D + g0) << log2_cap);
      uint32_t alive = (ng >= 32) ? 0xffffffffu : ((1u << ng) - 1);
      for (uint64_t base = 0; base < n && alive; base += 32) {
        const uint64_t i = base + lane;
        const bool in = i < n;
        const uint64_t key = in ? __ldg(chains + c0 + i) : 0ull;
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

extern "C" netkv_status netkv_prefix_match(const uint64_t* d_tables, uint32_t D,
                                           uint32_t log2_capacity, uint32_t n_sets,
                                           const uint64_t* d_chains, const uint64_t* d_chain_off,
                                           uint32_t R, const uint32_t* d_set_off, uint16_t* d_M,
                                           int* d_status, netkv_stream_t stream) {
  if (!d_tables || !d_chain_off || !d_M || D == 0 || n_sets == 0) return NETKV_EINVAL;
  if (log2_capacity < 1 || log2_capacity > 32) return NETKV_EINVAL;
  if (n_sets > 1 && !d_set_off) return NETKV_EINVAL;
  if (!aligned_to(d_tables, 16) || !aligned_to(d_chain_off, 8) || !aligned_to(d_M, 2) ||
      (d_chains && !aligned_to(d_chains, 8)) || (d_set_off && !aligned_to(d_set_off, 4)))
    return NETKV_EINVAL;
  if (R == 0) return NETKV_OK;
  if (!d_chains) return NETKV_EINVAL;
  const uint64_t tasks = (uint64_t)R * ((D + kGroup - 1) / kGroup);
  const uint64_t warps_per_block = kMatchBlock / 32;
  const uint64_t blocks = (tasks + warps_per_block - 1) / warps_per_block;
  const unsigned grid = (unsigned)(blocks < (1u << 24) ? blocks : (1u << 24));
  prefix_match_kernel<<<grid, kMatchBlock, 0, (cudaStream_t)stream>>>(
      d_tables, D, log2_capacity, n_sets, d_chains, d_chain_off, R, d_set_off, d_M, d_status);
  return netkv_launch_status();
}
