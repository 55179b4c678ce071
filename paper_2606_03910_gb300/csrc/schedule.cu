// The greedy of Algorithm 1 (Sec. V-A) over independent scheduling streams.
//
// One CTA per stream walks that stream's events in order.  Each thread owns NPT
// consecutive decode ranks and keeps their load (active tokens) and instance links in
// registers, so the state of a stream never leaves the SM.  An arrival scores every
// candidate in parallel (the per-candidate work is the tier test, the bottleneck min of
// two level bottlenecks, one division for T_xfer and one for the missed fraction), then
// a (score, index) argmin that also carries the second-best score: a shuffle butterfly
// inside each warp and, for CTAs of several warps, one barrier and a second butterfly
// over the per-warp partials (double-buffered so one barrier per arrival suffices).
// Ties go to the lowest decode rank (line 13).  The decision is written by lane 0 of
// every warp, so a later departure event is resolved by the same lanes that wrote it.
// No scratch memory: network, prefix and load terms are combined on the fly from the
// level bottlenecks UB and the prefix hits M.
#include <math.h>

#include "netkv_internal.cuh"

namespace {

constexpr uint32_t kNone = 0xffffffffu;

__device__ __forceinline__ void combine(float& b, uint32_t& i, float& s, float b2, uint32_t i2,
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

__device__ __forceinline__ void warp_argmin(float& b, uint32_t& i, float& s) {
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float b2 = __shfl_xor_sync(0xffffffffu, b, o);
    const uint32_t i2 = __shfl_xor_sync(0xffffffffu, i, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
    combine(b, i, s, b2, i2, s2);
  }
}

template <int NPT, int BLOCK>
__global__ void __launch_bounds__(BLOCK) schedule_kernel(
    TopoArgs t, const netkv_weights* __restrict__ W, uint32_t R, const uint32_t* __restrict__ len,
    const uint32_t* __restrict__ prefill, const uint32_t* __restrict__ snap,
    const uint16_t* __restrict__ M, const float* __restrict__ UB, uint32_t n_snap,
    const uint32_t* __restrict__ events, const uint64_t* __restrict__ event_off,
    const int64_t* __restrict__ load_init, int32_t* dec, float* __restrict__ best,
    float* __restrict__ second, int64_t* __restrict__ load_final, int* status) {
  constexpr int NW = BLOCK / 32;
  __shared__ float s_b[2][NW];
  __shared__ uint32_t s_i[2][NW];
  __shared__ float s_s[2][NW];
  const uint32_t stream = blockIdx.x;
  const uint32_t tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  const uint32_t D = t.D, N = t.N;
  const netkv_weights w = W[stream];
  const float4 lat = make_float4(t.lat[0], t.lat[1], t.lat[2], t.lat[3]);
  const float inf = __int_as_float(0x7f800000);

  int64_t load[NPT];
  uint4 ld[NPT];  // links of the decode instance; .x is the instance index itself
#pragma unroll
  for (int j = 0; j < NPT; ++j) {
    const uint32_t d = tid * NPT + j;
    load[j] = 0;
    ld[j] = make_uint4(0, 0, 0, 0);
    if (d < D) {
      ld[j] = __ldg(t.links + __ldg(t.dec + d));
      if (load_init) load[j] = load_init[(uint64_t)stream * D + d];
    }
  }

  const uint64_t e0 = event_off[stream], e1 = event_off[stream + 1];
  uint32_t parity = 0;
  for (uint64_t e = e0; e < e1; ++e) {
    const uint32_t code = __ldg(events + e);
    const uint32_t r = code & 0x7fffffffu;
    if (r >= R) {
      if (tid == 0) flag_status(status, NETKV_DEV_ERANGE);
      continue;
    }
    const uint32_t l = __ldg(len + r);
    if (code >> 31) {  // departure: release the tokens of a dispatched request
      int32_t dd = 0;
      if (lane == 0) dd = *((volatile int32_t*)(dec + r));
      dd = __shfl_sync(0xffffffffu, dd, 0);
      if (dd >= 0 && (uint32_t)dd < D) {
#pragma unroll
        for (int j = 0; j < NPT; ++j)
          if (tid * NPT + j == (uint32_t)dd) load[j] -= l;
      }
      continue;
    }
    const uint32_t pr = __ldg(prefill + r), k = __ldg(snap + r);
    if (pr >= t.P || k >= n_snap || l == 0) {
      if (tid == 0) {
        flag_status(status, l == 0 ? NETKV_DEV_EDOMAIN : NETKV_DEV_ERANGE);
        best[r] = inf;
        second[r] = inf;
      }
      if (lane == 0) dec[r] = -1;
      continue;
    }
    const uint32_t pinst = __ldg(t.pre + pr);
    const uint4 lp = __ldg(t.links + pinst);
    const float4 ubp = __ldg(reinterpret_cast<const float4*>(UB) + (uint64_t)k * N + pinst);
    const float* ub_row = UB + (uint64_t)k * N * 4;
    const uint16_t* m_row = M + (uint64_t)r * D;

    float b = inf, s2 = inf;
    uint32_t bi = kNone;
#pragma unroll
    for (int j = 0; j < NPT; ++j) {
      const uint32_t d = tid * NPT + j;
      if (d < D) {
        const uint32_t m = __ldg(m_row + d);
        uint32_t lam = 16u * m;
        if (m > l / 16u) {
          flag_status(status, NETKV_DEV_EDOMAIN);
          lam = lam < l ? lam : l;
        }
        const uint32_t miss_tok = l - lam;
        const bool feasible = load[j] + (int64_t)l <= w.cap_tokens;
        const int tau = tier_of(lp, ld[j]);
        const float bb = fminf(pick4(ubp, tau), __ldg(ub_row + (uint64_t)ld[j].x * 4 + tau));
        const float s_eff = (float)((int64_t)miss_tok * (int64_t)w.bytes_per_token);
        const float T = s_eff / bb + pick4(lat, tau);
        const float miss = (float)miss_tok / (float)l;
        const float sc = w.w_net * T + w.w_prefix * miss + w.w_load * (w.theta_s_per_token * (float)load[j]);
        if (feasible) {
          if (bi == kNone || sc < b) {
            s2 = b;
            b = sc;
            bi = d;
          } else if (sc < s2) {
            s2 = sc;
          }
        }
      }
    }
    warp_argmin(b, bi, s2);
    if (NW > 1) {
      if (lane == 0) {
        s_b[parity][wid] = b;
        s_i[parity][wid] = bi;
        s_s[parity][wid] = s2;
      }
      __syncthreads();
      b = inf;
      s2 = inf;
      bi = kNone;
      if (lane < (uint32_t)NW) {
        b = s_b[parity][lane];
        bi = s_i[parity][lane];
        s2 = s_s[parity][lane];
      }
      warp_argmin(b, bi, s2);
      parity ^= 1u;
    }
    const int32_t dstar = bi == kNone ? -1 : (int32_t)bi;
    if (dstar >= 0) {
#pragma unroll
      for (int j = 0; j < NPT; ++j)
        if (tid * NPT + j == (uint32_t)dstar) load[j] += l;
    }
    if (lane == 0) *((volatile int32_t*)(dec + r)) = dstar;
    if (tid == 0) {
      best[r] = b;
      second[r] = s2;
    }
  }
#pragma unroll
  for (int j = 0; j < NPT; ++j) {
    const uint32_t d = tid * NPT + j;
    if (d < D) load_final[(uint64_t)stream * D + d] = load[j];
  }
}

template <int NPT, int BLOCK>
netkv_status launch(const TopoArgs& t, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
                    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap,
                    const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
                    const uint32_t* d_events, const uint64_t* d_event_off,
                    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
                    int64_t* d_load_final, int* d_status, cudaStream_t s) {
  schedule_kernel<NPT, BLOCK><<<n_streams, BLOCK, 0, s>>>(
      t, d_w, R, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, d_events, d_event_off, d_load_init,
      d_dec, d_best, d_second, d_load_final, d_status);
  return netkv_launch_status();
}

}  // namespace

extern "C" netkv_status netkv_schedule_streams(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap, const uint16_t* d_M,
    const float* d_UB, uint32_t n_snap, const uint32_t* d_events, const uint64_t* d_event_off,
    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
    int64_t* d_load_final, int* d_status, netkv_stream_t stream) {
  if (!topo || !d_w || !d_event_off || !d_load_final) return NETKV_EINVAL;
  if (n_streams == 0) return NETKV_OK;
  if (n_streams > 0x7fffffffu) return NETKV_EINVAL;
  if (R > 0 && (!d_len || !d_prefill || !d_snap || !d_M || !d_UB || !d_dec || !d_best ||
                !d_second || !d_events))
    return NETKV_EINVAL;
  if (!aligned_to(d_w, 8) || !aligned_to(d_UB, 16) || !aligned_to(d_event_off, 8) ||
      !aligned_to(d_load_final, 8) || (d_load_init && !aligned_to(d_load_init, 8)))
    return NETKV_EINVAL;
  const TopoArgs t = topo_args(topo);
  const uint32_t D = t.D;
  cudaStream_t s = (cudaStream_t)stream;
#define NETKV_SCHED(NPT, BLOCK)                                                                  \
  return launch<NPT, BLOCK>(t, n_streams, d_w, R, d_len, d_prefill, d_snap, d_M, d_UB, n_snap, \
                            d_events, d_event_off, d_load_init, d_dec, d_best, d_second,       \
                            d_load_final, d_status, s)
  if (D <= 32) NETKV_SCHED(1, 32);
  if (D <= 256) NETKV_SCHED(1, 256);
  if (D <= 1024) NETKV_SCHED(4, 256);
  if (D <= 4096) NETKV_SCHED(4, 1024);
#undef NETKV_SCHED
  return NETKV_EINVAL;
}
