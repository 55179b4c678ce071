// Layout of the decode-cache index (the block-level prefix caches K_d of Sec. III-B) and
// its lookup, used by the cache build and the prefix match.  (The greedy with evolving
// caches keeps its own per-decode state and does not read this index.)
//
// The caches of a table set are indexed per group of up to 64 decodes:
//   hash table  2^L open-addressing slots {hash, position in the run array};
//   run keys    2^L hashes: the group's distinct cached hashes in the order the key lists
//               give them;
//   run masks   2^L masks of W bytes, bit (d mod 64) set when decode d caches the hash at
//               that run position.  W = 1, 2, 4 or 8 for pools of up to 8, 16, 32 or more
//               decodes, so a pool of 8 decodes reads 9 bytes per run position, not 16.
// Index idx = set * n_groups + group occupies index_stride(L, W) bytes (a multiple of 256):
// slots, then keys, then masks.
#pragma once

#include "netkv_internal.cuh"

namespace {

constexpr uint32_t kGroup = 64;  // decodes per index (bits of the mask)
constexpr unsigned long long kNotFound = ~0ull;

struct __align__(16) IndexSlot {
  unsigned long long key;
  unsigned long long pos;  // position of the key in the run array
};

// Bytes of one run mask for a pool of D decodes.
__host__ __device__ __forceinline__ uint32_t mask_bytes_of(uint32_t D) {
  const uint32_t g = D < kGroup ? D : kGroup;
  return g <= 8 ? 1u : g <= 16 ? 2u : g <= 32 ? 4u : 8u;
}

// Bytes of one index (slots, keys, masks), rounded up to 256.
__host__ __device__ __forceinline__ uint64_t index_stride(uint32_t log2_cap, uint32_t mask_bytes) {
  return (((uint64_t)(sizeof(IndexSlot) + 8u + mask_bytes) << log2_cap) + 255u) & ~255ull;
}

// One index: its hash table, run keys and run masks.
struct IndexView {
  IndexSlot* hash;
  unsigned long long* keys;
  unsigned char* masks;
  uint32_t mask_bytes;
};

__device__ __forceinline__ IndexView index_view(const void* index, uint64_t idx, uint32_t log2_cap,
                                                uint32_t mask_bytes) {
  unsigned char* base = reinterpret_cast<unsigned char*>(const_cast<void*>(index)) +
                        idx * index_stride(log2_cap, mask_bytes);
  IndexView v;
  v.hash = reinterpret_cast<IndexSlot*>(base);
  v.keys = reinterpret_cast<unsigned long long*>(base + (sizeof(IndexSlot) << log2_cap));
  v.masks = base + ((sizeof(IndexSlot) + 8u) << log2_cap);
  v.mask_bytes = mask_bytes;
  return v;
}

// Mask of run position p (read-only path).  kMB: the mask width when the caller knows it
// at compile time (pools of more than 32 decodes: 8), 0 to read it from the view.
template <int kMB = 0>
__device__ __forceinline__ unsigned long long run_mask(const IndexView& v, uint64_t p) {
  if (kMB == 8) return __ldg(reinterpret_cast<const unsigned long long*>(v.masks) + p);
  switch (v.mask_bytes) {
    case 1: return __ldg(v.masks + p);
    case 2: return __ldg(reinterpret_cast<const unsigned short*>(v.masks) + p);
    case 4: return __ldg(reinterpret_cast<const unsigned int*>(v.masks) + p);
    default: return __ldg(reinterpret_cast<const unsigned long long*>(v.masks) + p);
  }
}

// Adds decode bit `bit` (bit d mod 64 of the group) to the mask of run position p.
__device__ __forceinline__ void run_mask_or(const IndexView& v, uint64_t p, unsigned long long bit) {
  if (v.mask_bytes == 8) {
    atomicOr(reinterpret_cast<unsigned long long*>(v.masks) + p, bit);
  } else {  // the 32-bit word holding the mask; groups of <= 32 decodes, so bit < 2^32
    const uint64_t byte = p * v.mask_bytes;
    atomicOr(reinterpret_cast<unsigned int*>(v.masks) + (byte >> 2),
             (unsigned int)bit << (8u * (uint32_t)(byte & 3u)));
  }
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
