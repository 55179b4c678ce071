// Internal definitions shared by the NetKV CUDA translation units.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/netkv.h"

struct netkv_topology {
  uint32_t fanout[4];
  uint32_t N, P, D;
  uint32_t used_links, n_links;
  double bw[4], lat[4];
  float bw_f[4], lat_f[4];
  int device;
  // device mirror
  uint4* d_links;      // [N] (level-0, level-1, level-2, level-3 link of instance i)
  uint32_t* d_pre;     // [P] instance of prefill rank p
  uint32_t* d_dec;     // [D] instance of decode rank d
  uint8_t* d_role;     // [N] 0 = prefill, 1 = decode
};

// fp32 constants of a topology passed to kernels by value
struct TopoArgs {
  const uint4* links;
  const uint32_t* pre;
  const uint32_t* dec;
  const uint8_t* role;
  uint32_t N, P, D, n_links;
  float bw[4];
  float lat[4];
};

inline TopoArgs topo_args(const netkv_topology* t) {
  TopoArgs a;
  a.links = t->d_links;
  a.pre = t->d_pre;
  a.dec = t->d_dec;
  a.role = t->d_role;
  a.N = t->N;
  a.P = t->P;
  a.D = t->D;
  a.n_links = t->n_links;
  for (int k = 0; k < 4; ++k) {
    a.bw[k] = t->bw_f[k];
    a.lat[k] = t->lat_f[k];
  }
  return a;
}

#define NETKV_CUDA_TRY(expr)                          \
  do {                                                \
    if ((expr) != cudaSuccess) return NETKV_ECUDA;    \
  } while (0)

inline netkv_status netkv_launch_status() {
  return cudaPeekAtLastError() == cudaSuccess ? NETKV_OK : NETKV_ECUDA;
}

inline bool aligned_to(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

__device__ __forceinline__ void flag_status(int* status, int bits) {
  if (status) atomicOr(status, bits);
}

// Locality tier from the links of two instances: same node iff same level-1 link,
// same leaf iff same level-2 link, same pod iff same level-3 link.
__device__ __forceinline__ int tier_of(const uint4& a, const uint4& b) {
  return (a.y == b.y) ? 0 : (a.z == b.z) ? 1 : (a.w == b.w) ? 2 : 3;
}

__device__ __forceinline__ float pick4(const float4& v, int k) {
  return k == 0 ? v.x : k == 1 ? v.y : k == 2 ? v.z : v.w;
}

// Home slot of a key: Fibonacci (multiplicative) hashing, top log2_cap bits.
__device__ __forceinline__ uint64_t home_slot(uint64_t key, uint32_t log2_cap) {
  return (key * 0x9E3779B97F4A7C15ull) >> (64 - log2_cap);
}
