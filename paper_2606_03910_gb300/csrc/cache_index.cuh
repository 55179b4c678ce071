// Layout of the decode-cache index (the block-level prefix caches K_d of Sec. III-B) and
// its lookup, used by the cache build and the prefix match.  (The greedy with evolving
// caches keeps its own per-decode state and does not read this index.)
//
// The caches of a table set are indexed per group of up to 64 decodes:
//   hash table  2^L open-addressing slots {hash, position in the run array};
//   run array   2^L entries {hash, mask of the group's decodes that cache it}, the
//               group's distinct cached hashes in the order the key lists give them.
// Index idx = set * n_groups + group occupies 2^(L+1) 16-byte records: slots, then runs.
#pragma once

#include "netkv_internal.cuh"

namespace {

constexpr uint32_t kGroup = 64;  // decodes per index (bits of the mask)
constexpr unsigned long long kNotFound = ~0ull;

struct __align__(16) IndexSlot {
  unsigned long long key;
  unsigned long long pos;  // position of the key in the run array
};

struct __align__(16) RunEntry {
  unsigned long long key;
  unsigned long long mask;  // decodes of the group that cache the key
};

// Hash table and run array of index (set g, decode group q): 2^L slots then 2^L entries.
__device__ __forceinline__ IndexSlot* index_hash(void* index, uint64_t idx, uint32_t L) {
  return reinterpret_cast<IndexSlot*>(index) + (idx << (L + 1));
}
__device__ __forceinline__ const IndexSlot* index_hash(const void* index, uint64_t idx,
                                                       uint32_t L) {
  return reinterpret_cast<const IndexSlot*>(index) + (idx << (L + 1));
}

// Run position of `key` (non-zero) in one index, or kNotFound.
__device__ __forceinline__ unsigned long long lookup(const IndexSlot* __restrict__ hash,
                                                     uint64_t key, uint32_t log2_cap,
                                                     int* status) {
  const uint64_t mask = (1ull << log2_cap) - 1;
  uint64_t slot = home_slot(key, log2_cap);
  for (uint64_t seen = 0; seen <= mask; ++seen) {
    const ulonglong2 s = __ldg(reinterpret_cast<const ulonglong2*>(hash + slot));
    if (s.x == key) return s.y;
    if (s.x == 0ull) return kNotFound;
    slot = (slot + 1) & mask;
  }
  flag_status(status, NETKV_DEV_EFULL);
  return kNotFound;
}

}  // namespace
