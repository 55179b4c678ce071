// The decision-independent part of a candidate's score, shared by the greedy kernels.
#pragma once

#include "netkv_internal.cuh"

// Decision-independent part of a candidate's score (Algorithm 1 lines 5-8, Eq. 2, Eq. 3):
// w_net * (s_eff / min(UB_p[tau], UB_d[tau]) + L_tau) + w_prefix * (l - 16 M) / l.
__device__ __forceinline__ float base_score(const netkv_weights& w, uint32_t l, uint32_t m,
                                            float ub_p, float ub_d, float lat_tau, int* status) {
  uint32_t lam = 16u * m;
  if (m > l / 16u) {
    flag_status(status, NETKV_DEV_EDOMAIN);
    lam = lam < l ? lam : l;
  }
  const uint32_t miss_tok = l - lam;
  const float bb = fminf(ub_p, ub_d);
  const float s_eff = (float)((int64_t)miss_tok * (int64_t)w.bytes_per_token);
  const float T = s_eff / bb + lat_tau;
  const float miss = (float)miss_tok / (float)l;
  return w.w_net * T + w.w_prefix * miss;
}

// Level bottlenecks of an instance with links `l` in one utilisation row:
// (B_0 (1-u_0), min with B_1 (1-u_1), ...), the same fp32 expression as the oracle build's
// level-bottleneck pass, so a score computed from the row equals one computed from UB.
__device__ __forceinline__ float4 level_bottlenecks_of(const TopoArgs& t,
                                                       const float* __restrict__ row,
                                                       const uint4& l, int* status) {
  const float u0 = __ldg(row + l.x), u1 = __ldg(row + l.y);
  const float u2 = __ldg(row + l.z), u3 = __ldg(row + l.w);
  if (!(u0 >= 0.0f && u0 < 1.0f && u1 >= 0.0f && u1 < 1.0f && u2 >= 0.0f && u2 < 1.0f &&
        u3 >= 0.0f && u3 < 1.0f))
    flag_status(status, NETKV_DEV_EDOMAIN);
  float4 b;
  b.x = t.bw[0] * (1.0f - u0);
  b.y = fminf(b.x, t.bw[1] * (1.0f - u1));
  b.z = fminf(b.y, t.bw[2] * (1.0f - u2));
  b.w = fminf(b.z, t.bw[3] * (1.0f - u3));
  return b;
}
