// Topology handle: the four-tier instance tree of Sec. III-A with the link numbering
// documented in netkv.h, mirrored to the device once at creation.
#include <math.h>
#include <stdlib.h>
#include <string.h>

#include <vector>

#include "netkv_internal.cuh"

extern "C" uint32_t netkv_version(void) { return 1u; }

extern "C" netkv_status netkv_topology_create(const netkv_topology_desc* desc,
                                              netkv_topology_t* out) {
  if (!desc || !out || !desc->role) return NETKV_EINVAL;
  *out = nullptr;
  uint64_t n = 1;
  for (int k = 0; k < 4; ++k) {
    if (desc->fanout[k] == 0) return NETKV_EINVAL;
    n *= desc->fanout[k];
    if (n >= (1ull << 31)) return NETKV_EINVAL;
  }
  for (int k = 0; k < 4; ++k) {
    const double b = desc->tier_bw_Bps[k], l = desc->tier_lat_s[k];
    if (!(b > 0) || !isfinite(b) || !(l >= 0) || !isfinite(l)) return NETKV_EINVAL;
  }
  const uint32_t N = (uint32_t)n;
  const uint32_t f0 = desc->fanout[0], f1 = desc->fanout[1], f2 = desc->fanout[2];
  const uint32_t n_node = N / f0, n_leaf = n_node / f1, n_pod = desc->fanout[3];
  const uint64_t used = (uint64_t)N + n_node + n_leaf + n_pod;
  if (used >= (1ull << 32) || desc->n_links < used) return NETKV_EINVAL;

  std::vector<uint4> links(N);
  std::vector<uint32_t> pre, dec;
  for (uint32_t i = 0; i < N; ++i) {
    const uint8_t r = desc->role[i];
    if (r > 1) return NETKV_EINVAL;
    (r ? dec : pre).push_back(i);
    const uint32_t node = i / f0, leaf = node / f1, pod = leaf / f2;
    links[i] = make_uint4(i, N + node, N + n_node + leaf, N + n_node + n_leaf + pod);
  }
  if (pre.empty() || dec.empty()) return NETKV_EINVAL;

  netkv_topology* t = (netkv_topology*)calloc(1, sizeof(netkv_topology));
  if (!t) return NETKV_ENOMEM;
  memcpy(t->fanout, desc->fanout, sizeof(t->fanout));
  t->N = N;
  t->P = (uint32_t)pre.size();
  t->D = (uint32_t)dec.size();
  t->used_links = (uint32_t)used;
  t->n_links = desc->n_links;
  for (int k = 0; k < 4; ++k) {
    t->bw[k] = desc->tier_bw_Bps[k];
    t->lat[k] = desc->tier_lat_s[k];
    t->bw_f[k] = (float)t->bw[k];
    t->lat_f[k] = (float)t->lat[k];
  }
  netkv_status st = NETKV_OK;
  if (cudaGetDevice(&t->device) != cudaSuccess ||
      cudaMalloc(&t->d_links, sizeof(uint4) * N) != cudaSuccess ||
      cudaMalloc(&t->d_pre, sizeof(uint32_t) * t->P) != cudaSuccess ||
      cudaMalloc(&t->d_dec, sizeof(uint32_t) * t->D) != cudaSuccess ||
      cudaMalloc(&t->d_role, N) != cudaSuccess) {
    st = NETKV_ENOMEM;
  } else if (cudaMemcpy(t->d_links, links.data(), sizeof(uint4) * N,
                        cudaMemcpyHostToDevice) != cudaSuccess ||
             cudaMemcpy(t->d_pre, pre.data(), sizeof(uint32_t) * t->P,
                        cudaMemcpyHostToDevice) != cudaSuccess ||
             cudaMemcpy(t->d_dec, dec.data(), sizeof(uint32_t) * t->D,
                        cudaMemcpyHostToDevice) != cudaSuccess ||
             cudaMemcpy(t->d_role, desc->role, N, cudaMemcpyHostToDevice) != cudaSuccess) {
    st = NETKV_ECUDA;
  }
  if (st != NETKV_OK) {
    cudaGetLastError();
    netkv_topology_destroy(t);
    return st;
  }
  *out = t;
  return NETKV_OK;
}

extern "C" netkv_status netkv_topology_destroy(netkv_topology_t t) {
  if (!t) return NETKV_EINVAL;
  cudaFree(t->d_links);
  cudaFree(t->d_pre);
  cudaFree(t->d_dec);
  cudaFree(t->d_role);
  free(t);
  return NETKV_OK;
}

extern "C" netkv_status netkv_topology_query(netkv_topology_t t, uint32_t* n_instances,
                                             uint32_t* P, uint32_t* D, uint32_t* used_links) {
  if (!t) return NETKV_EINVAL;
  if (n_instances) *n_instances = t->N;
  if (P) *P = t->P;
  if (D) *D = t->D;
  if (used_links) *used_links = t->used_links;
  return NETKV_OK;
}
