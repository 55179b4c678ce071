// Network cost oracle (Sec. III-D Eq. 3 and Eq. 4, Sec. III-E) with per-link congestion.
//
// level_bottleneck_kernel: UB[s][i][k] = min_{h<=k} B_h (1 - u[s][link_h(i)]), one
//   thread per (snapshot, instance), one 16-byte store each.  With directed links
//   (kDir) a prefill instance's climb reads the upward row and a decode instance's the
//   downward row: the directions a transfer from prefill to decode crosses them in.
// oracle_build_kernel: C[s][p][d] = kv / min(UB[s][p][tau], UB[s][d][tau]) + L_tau.
//   In the paper-literal per-tier mode (kTier) UB[s][i][k] = B_k (1 - c[s][k]) for every
//   instance, from four congestion values per snapshot.
//   Division is monotone (correctly rounded, positive operands), so
//   kv / min(a, b) == max(kv / a, kv / b) exactly; each block therefore divides once per
//   (instance, level) it touches and the per-pair work is a tier test, a max and an
//   add.  Each block owns one snapshot and 1024 consecutive decode ranks (4 per
//   thread, kept in registers) and walks every prefill rank, staged 1024 at a time in
//   shared memory; every warp store writes 512 contiguous bytes of a C row with an
//   evict-first hint.  No scratch memory: the quotients of the block's instances are
//   recomputed from the utilisation row.
#include "netkv_internal.cuh"

namespace {

constexpr int kBlock = 256;
constexpr int kPerThread = 4;
constexpr int kDChunk = kBlock * kPerThread;
constexpr int kPTile = 1024;

__device__ __forceinline__ bool util_ok(float u) { return u >= 0.0f && u < 1.0f; }

// Level bottlenecks of instance `links` in one utilisation row.
__device__ __forceinline__ float4 level_bottlenecks(const TopoArgs& t, const float* __restrict__ row,
                                                    const uint4& l, int* status) {
  const float u0 = __ldg(row + l.x), u1 = __ldg(row + l.y);
  const float u2 = __ldg(row + l.z), u3 = __ldg(row + l.w);
  if (!(util_ok(u0) && util_ok(u1) && util_ok(u2) && util_ok(u3)))
    flag_status(status, NETKV_DEV_EDOMAIN);
  float4 b;
  b.x = t.bw[0] * (1.0f - u0);
  b.y = fminf(b.x, t.bw[1] * (1.0f - u1));
  b.z = fminf(b.y, t.bw[2] * (1.0f - u2));
  b.w = fminf(b.z, t.bw[3] * (1.0f - u3));
  return b;
}

// Paper-literal per-tier maps (Sec. III-E): level k's bandwidth B_k (1 - c_k) from the
// snapshot's four per-tier congestion values, with no minimum over lower levels.
__device__ __forceinline__ float4 tier_bandwidths(const TopoArgs& t, const float* __restrict__ c,
                                                  int* status) {
  const float c0 = __ldg(c), c1 = __ldg(c + 1), c2 = __ldg(c + 2), c3 = __ldg(c + 3);
  if (!(util_ok(c0) && util_ok(c1) && util_ok(c2) && util_ok(c3)))
    flag_status(status, NETKV_DEV_EDOMAIN);
  return make_float4(t.bw[0] * (1.0f - c0), t.bw[1] * (1.0f - c1), t.bw[2] * (1.0f - c2),
                     t.bw[3] * (1.0f - c3));
}

__device__ __forceinline__ float4 quotients(float kv, const float4& b) {
  return make_float4(kv / b.x, kv / b.y, kv / b.z, kv / b.w);
}

template <bool kDir, bool kTier = false>
__global__ void __launch_bounds__(kBlock) level_bottleneck_kernel(
    TopoArgs t, const float* __restrict__ util, const float* __restrict__ util_down,
    uint32_t n_snap, float4* __restrict__ UB, int* status) {
  const uint64_t total = (uint64_t)n_snap * t.N;
  for (uint64_t idx = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; idx < total;
       idx += (uint64_t)gridDim.x * blockDim.x) {
    const uint64_t s = idx / t.N;
    const uint32_t i = (uint32_t)(idx - s * t.N);
    const uint4 l = __ldg(t.links + i);
    const float* rows = (kDir && __ldg(t.role + i)) ? util_down : util;
    UB[idx] = kTier ? tier_bandwidths(t, util + s * 4, status)
                    : level_bottlenecks(t, rows + s * t.n_links, l, status);
  }
}

// util_down: the decode side's rows (the downward utilisations of directed links; the
// same pointer as util for undirected links).
template <bool kVec, bool kTier = false>
__global__ void __launch_bounds__(kBlock) oracle_build_kernel(
    TopoArgs t, const float* __restrict__ util, const float* __restrict__ util_down,
    uint32_t n_snap, float kv, float* __restrict__ C, int* status) {
  __shared__ float4 s_q[kPTile];
  __shared__ uint4 s_l[kPTile];
  const float4 lat = make_float4(t.lat[0], t.lat[1], t.lat[2], t.lat[3]);
  const uint32_t d0 = blockIdx.x * kDChunk + threadIdx.x * kPerThread;

  for (uint32_t s = blockIdx.y; s < n_snap; s += gridDim.y) {
    const float* row = util + (uint64_t)s * t.n_links;
    const float* row_d = util_down + (uint64_t)s * t.n_links;
    uint4 ld[kPerThread];
    float4 qd[kPerThread];
#pragma unroll
    for (int j = 0; j < kPerThread; ++j) {
      const uint32_t d = d0 + j;
      if (d < t.D) {
        ld[j] = __ldg(t.links + __ldg(t.dec + d));
        qd[j] = quotients(kv, kTier ? tier_bandwidths(t, util + (uint64_t)s * 4, status)
                                    : level_bottlenecks(t, row_d, ld[j], status));
      } else {
        ld[j] = make_uint4(0, 0, 0, 0);
        qd[j] = make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
    float* crow = C + (uint64_t)s * t.P * t.D;
    for (uint32_t p0 = 0; p0 < t.P; p0 += kPTile) {
      const uint32_t np = min((uint32_t)kPTile, t.P - p0);
      __syncthreads();
      for (uint32_t k = threadIdx.x; k < np; k += kBlock) {
        const uint4 l = __ldg(t.links + __ldg(t.pre + p0 + k));
        s_l[k] = l;
        s_q[k] = quotients(kv, kTier ? tier_bandwidths(t, util + (uint64_t)s * 4, status)
                                     : level_bottlenecks(t, row, l, status));
      }
      __syncthreads();
      if (d0 >= t.D) continue;
      for (uint32_t k = 0; k < np; ++k) {
        const float4 qp = s_q[k];
        const uint4 lp = s_l[k];
        float c[kPerThread];
#pragma unroll
        for (int j = 0; j < kPerThread; ++j) {
          const int tau = tier_of(lp, ld[j]);
          c[j] = fmaxf(pick4(qp, tau), pick4(qd[j], tau)) + pick4(lat, tau);
        }
        float* out = crow + (uint64_t)(p0 + k) * t.D + d0;
        if (kVec) {
          __stcs(reinterpret_cast<float4*>(out), make_float4(c[0], c[1], c[2], c[3]));
        } else {
#pragma unroll
          for (int j = 0; j < kPerThread; ++j)
            if (d0 + j < t.D) __stcs(out + j, c[j]);
        }
      }
    }
  }
}

}  // namespace

enum OracleMode { kLinks = 0, kDirected = 1, kTiers = 2 };

static netkv_status oracle_build(netkv_topology_t topo, const float* d_util, const float* d_util_down,
                          int mode, uint32_t n_snap, double kv_bytes, float* d_C,
                          float* d_UB, int* d_status, netkv_stream_t stream) {
  if (!topo || !d_util || !d_util_down || (!d_C && !d_UB)) return NETKV_EINVAL;
  if (!(kv_bytes > 0) || !(kv_bytes < 3.0e38)) return NETKV_EINVAL;
  if (!aligned_to(d_util, 4) || !aligned_to(d_util_down, 4) || (d_C && !aligned_to(d_C, 4)) ||
      (d_UB && !aligned_to(d_UB, 16)))
    return NETKV_EINVAL;
  if (n_snap == 0) return NETKV_OK;
  const TopoArgs t = topo_args(topo);
  cudaStream_t s = (cudaStream_t)stream;
  if (d_UB) {
    const uint64_t total = (uint64_t)n_snap * t.N;
    const uint64_t blocks = (total + kBlock - 1) / kBlock;
    const unsigned grid = (unsigned)(blocks < (1u << 20) ? blocks : (1u << 20));
    if (mode == kTiers)
      level_bottleneck_kernel<false, true><<<grid, kBlock, 0, s>>>(
          t, d_util, d_util, n_snap, reinterpret_cast<float4*>(d_UB), d_status);
    else if (mode == kDirected)
      level_bottleneck_kernel<true><<<grid, kBlock, 0, s>>>(
          t, d_util, d_util_down, n_snap, reinterpret_cast<float4*>(d_UB), d_status);
    else
      level_bottleneck_kernel<false><<<grid, kBlock, 0, s>>>(
          t, d_util, d_util, n_snap, reinterpret_cast<float4*>(d_UB), d_status);
    if (netkv_launch_status() != NETKV_OK) return NETKV_ECUDA;
  }
  if (d_C) {
    const dim3 grid((t.D + kDChunk - 1) / kDChunk, n_snap < 65535u ? n_snap : 65535u);
    const bool vec = (t.D % 4 == 0) && aligned_to(d_C, 16);
    if (mode == kTiers && vec)
      oracle_build_kernel<true, true><<<grid, kBlock, 0, s>>>(t, d_util, d_util, n_snap,
                                                              (float)kv_bytes, d_C, d_status);
    else if (mode == kTiers)
      oracle_build_kernel<false, true><<<grid, kBlock, 0, s>>>(t, d_util, d_util, n_snap,
                                                               (float)kv_bytes, d_C, d_status);
    else if (vec)
      oracle_build_kernel<true><<<grid, kBlock, 0, s>>>(t, d_util, d_util_down, n_snap,
                                                        (float)kv_bytes, d_C, d_status);
    else
      oracle_build_kernel<false><<<grid, kBlock, 0, s>>>(t, d_util, d_util_down, n_snap,
                                                         (float)kv_bytes, d_C, d_status);
    if (netkv_launch_status() != NETKV_OK) return NETKV_ECUDA;
  }
  return NETKV_OK;
}

extern "C" netkv_status netkv_oracle_build(netkv_topology_t topo, const float* d_util,
                                           uint32_t n_snap, double kv_bytes, float* d_C,
                                           float* d_UB, int* d_status, netkv_stream_t stream) {
  return oracle_build(topo, d_util, d_util, kLinks, n_snap, kv_bytes, d_C, d_UB, d_status, stream);
}

extern "C" netkv_status netkv_oracle_build_directed(netkv_topology_t topo, const float* d_util_up,
                                                    const float* d_util_down, uint32_t n_snap,
                                                    double kv_bytes, float* d_C, float* d_UB,
                                                    int* d_status, netkv_stream_t stream) {
  return oracle_build(topo, d_util_up, d_util_down, kDirected, n_snap, kv_bytes, d_C, d_UB,
                      d_status, stream);
}

extern "C" netkv_status netkv_oracle_build_tiers(netkv_topology_t topo, const float* d_c,
                                                 uint32_t n_snap, double kv_bytes, float* d_C,
                                                 float* d_UB, int* d_status,
                                                 netkv_stream_t stream) {
  return oracle_build(topo, d_c, d_c, kTiers, n_snap, kv_bytes, d_C, d_UB, d_status, stream);
}
