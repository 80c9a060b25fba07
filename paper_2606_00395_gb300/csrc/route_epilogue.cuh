// Warp-cooperative finish of one token's routing, shared by the fp32 SIMT kernel and the
// split-K tensor-core kernel.  The token's logits are spread over the warp: lane l holds expert
// e = 32 j + l in zr[j] (z = p_old + b in predict mode, p in replay mode; -FLT_MAX beyond N)
// and the router part p in pr[j].
//   predict (Eqs. pr2_predict, pr2_route): rho_hat = Softmax(z); idx = TopK(rho_hat, k) by k
//            rounds of warp argmax (ties to the lower expert); gates = rho_hat[idx];
//            aux = p_old row (feature-cache logits); returns whether
//            rho_hat_(k) - rho_hat_(k+1) < PR2_NEAR_TIE_GAP.
//   replay  (Sec. 4.1): rho = Softmax(z); gates = rho[idx_in] (0 for an invalid slot, which is
//            flagged in *status); aux = the full rho row.
#pragma once

#include <float.h>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {

constexpr int kRoutePerLane = kMaxExperts / 32;

__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Largest value over the warp, lowest index among equal values.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (ov > v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
    }
  }
}

__device__ __forceinline__ bool route_warp_finish(bool predict, int64_t t, int N, int k,
                                                  const float (&zr)[kRoutePerLane],
                                                  const float (&pr)[kRoutePerLane],
                                                  const int32_t* __restrict__ idx_in,
                                                  int32_t* __restrict__ idx_out,
                                                  float* __restrict__ gates,
                                                  float* __restrict__ aux, int32_t* status,
                                                  bool norm) {
  const int lane = threadIdx.x & 31;
  float gsum = 0.f;  // sum of the written gates (lane 0), for PR2_F_NORMALIZE_TOPK
  float mx = -FLT_MAX;
#pragma unroll
  for (int j = 0; j < kRoutePerLane; ++j) mx = fmaxf(mx, zr[j]);
  mx = warp_max_f(mx);
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < kRoutePerLane; ++j)
    if (j * 32 + lane < N) s += expf(zr[j] - mx);
  s = warp_sum_f(s);
  const float inv_s = 1.0f / s;

  if (aux != nullptr) {
    float* row = aux + t * N;
#pragma unroll
    for (int j = 0; j < kRoutePerLane; ++j) {
      const int e = j * 32 + lane;
      if (e < N) row[e] = predict ? pr[j] : expf(zr[j] - mx) * inv_s;
    }
  }

  bool tie = false;
  if (predict) {
    unsigned taken = 0u;
    float prev = 0.f;
    const int rounds = (k < N) ? k + 1 : k;
    for (int r = 0; r < rounds; ++r) {
      float bv = -FLT_MAX;
      int bi = 0x7fffffff;
#pragma unroll
      for (int j = 0; j < kRoutePerLane; ++j) {
        const int e = j * 32 + lane;
        if (e < N && !((taken >> j) & 1u) && (zr[j] > bv || (zr[j] == bv && e < bi))) {
          bv = zr[j];
          bi = e;
        }
      }
      warp_argmax(bv, bi);
      if ((bi & 31) == lane) taken |= 1u << (bi >> 5);
      const float prob = expf(bv - mx) * inv_s;
      if (r < k) {
        if (lane == 0) {
          idx_out[t * k + r] = bi;
          gates[t * k + r] = prob;
          gsum += prob;
        }
        prev = prob;
      } else {
        tie = prev - prob < (float)PR2_NEAR_TIE_GAP;
      }
    }
  } else {
    for (int sl = 0; sl < k; ++sl) {
      const int e = idx_in[t * k + sl];
      bool ok = (e >= 0 && e < N);
      for (int s2 = 0; ok && s2 < sl; ++s2)
        if (idx_in[t * k + s2] == e) ok = false;
      float v = -FLT_MAX;
      const int ej = ok ? (e >> 5) : 0;
#pragma unroll
      for (int j = 0; j < kRoutePerLane; ++j)
        if (j == ej) v = zr[j];
      v = __shfl_sync(0xffffffffu, v, ok ? (e & 31) : 0);
      if (lane == 0) {
        const float g = ok ? expf(v - mx) * inv_s : 0.f;
        gates[t * k + sl] = g;
        gsum += g;
        if (!ok && status != nullptr) atomicOr(status, PR2_STATUS_BAD_INDEX);
      }
    }
  }
  if (norm && lane == 0 && gsum > 0.f) {  // renormalise the row just written (this thread's stores)
    const float sc = 1.0f / gsum;
    for (int r = 0; r < k; ++r) gates[t * k + r] *= sc;
  }
  return tie;
}

}  // namespace pr2
