// fp32 routing kernels (exact fp32 SIMT arithmetic; TF32 tensor cores would not meet the fp32
// tolerance).  One warp per token.
//   predict (Eqs. pr2_predict, pr2_route): z = h W^T + h W_p^T, rho_hat = Softmax(z),
//            idx = TopK(rho_hat, k) (ties to the lower expert), gates = rho_hat[idx].
//   replay  (Sec. 4.1 "Replay During Training"): rho = Softmax(h W^T), gates = rho[idx_in].
#include <float.h>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kWarps = 8;
constexpr int kPerLane = kMaxExperts / 32;  // expert slots per lane

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Largest (value, lowest index on ties) over the warp.
__device__ __forceinline__ void warp_argmax(float& v, int& i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    float ov = __shfl_xor_sync(0xffffffffu, v, o);
    int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (ov > v || (ov == v && oi < i)) {
      v = ov;
      i = oi;
    }
  }
}

__global__ void __launch_bounds__(kWarps * 32)
    route_simt_kernel(int T, int d, int N, int k, int predict, const float* __restrict__ h,
                      const float* __restrict__ W, const float* __restrict__ Wp,
                      const int32_t* __restrict__ idx_in, int32_t* __restrict__ idx_out,
                      float* __restrict__ gates, float* __restrict__ aux,
                      unsigned long long* near_tie, int32_t* status) {
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (t >= T) return;
  const float* ht = h + static_cast<int64_t>(t) * d;

  // z for experts e = j*32 + lane lives in zr[j]; p (router part alone) in pr[j].
  float zr[kPerLane], pr[kPerLane];
#pragma unroll
  for (int j = 0; j < kPerLane; ++j) {
    zr[j] = -FLT_MAX;
    pr[j] = 0.f;
    for (int l = 0; l < 32; ++l) {
      const int e = j * 32 + l;
      if (e >= N) break;
      const float* we = W + static_cast<int64_t>(e) * d;
      float p = 0.f, b = 0.f;
      if (predict) {
        const float* wq = Wp + static_cast<int64_t>(e) * d;
        for (int i = lane; i < d; i += 32) {
          const float x = ht[i];
          p = fmaf(x, we[i], p);
          b = fmaf(x, wq[i], b);
        }
        b = warp_sum(b);
      } else {
        for (int i = lane; i < d; i += 32) p = fmaf(ht[i], we[i], p);
      }
      p = warp_sum(p);
      if (lane == l) {
        pr[j] = p;
        zr[j] = p + b;
      }
    }
  }

  float mx = -FLT_MAX;
#pragma unroll
  for (int j = 0; j < kPerLane; ++j) mx = fmaxf(mx, zr[j]);
  mx = warp_max(mx);
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < kPerLane; ++j)
    if (j * 32 + lane < N) s += expf(zr[j] - mx);
  s = warp_sum(s);
  const float inv_s = 1.0f / s;

  if (aux != nullptr) {  // predict: p_old; replay: rho
    float* row = aux + static_cast<int64_t>(t) * N;
#pragma unroll
    for (int j = 0; j < kPerLane; ++j) {
      const int e = j * 32 + lane;
      if (e < N) row[e] = predict ? pr[j] : expf(zr[j] - mx) * inv_s;
    }
  }

  if (predict) {
    // k (+1 for the margin) rounds of warp argmax over the not yet selected experts.
    unsigned taken = 0u;
    float prev = 0.f;
    const int rounds = (k < N) ? k + 1 : k;
    for (int r = 0; r < rounds; ++r) {
      float bv = -FLT_MAX;
      int bi = 0x7fffffff;
#pragma unroll
      for (int j = 0; j < kPerLane; ++j) {
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
          idx_out[static_cast<int64_t>(t) * k + r] = bi;
          gates[static_cast<int64_t>(t) * k + r] = prob;
        }
        prev = prob;
      } else if (lane == 0 && near_tie != nullptr && prev - prob < (float)PR2_NEAR_TIE_GAP) {
        atomicAdd(near_tie, 1ull);
      }
    }
  } else {
    for (int sl = 0; sl < k; ++sl) {
      const int e = idx_in[static_cast<int64_t>(t) * k + sl];
      bool ok = (e >= 0 && e < N);
      for (int s2 = 0; ok && s2 < sl; ++s2)
        if (idx_in[static_cast<int64_t>(t) * k + s2] == e) ok = false;
      float v = -FLT_MAX;
      const int ej = ok ? (e >> 5) : 0;
#pragma unroll
      for (int j = 0; j < kPerLane; ++j)
        if (j == ej) v = zr[j];
      v = __shfl_sync(0xffffffffu, v, ok ? (e & 31) : 0);
      if (lane == 0) {
        gates[static_cast<int64_t>(t) * k + sl] = ok ? expf(v - mx) * inv_s : 0.f;
        if (!ok && status != nullptr) atomicOr(status, PR2_STATUS_BAD_INDEX);
      }
    }
  }
}

}  // namespace

cudaError_t launch_route_simt(const pr2_dims& dm, bool predict, const float* h, const float* W,
                              const float* Wp, const int32_t* idx_in, int32_t* idx_out,
                              float* gates, float* aux, int64_t* near_tie, int32_t* status,
                              cudaStream_t st) {
  const int T = static_cast<int>(dm.T);
  if (T == 0) return cudaSuccess;
  dim3 grid((T + kWarps - 1) / kWarps);
  route_simt_kernel<<<grid, kWarps * 32, 0, st>>>(
      T, dm.d, dm.N, dm.k, predict ? 1 : 0, h, W, Wp, idx_in, idx_out, gates, aux,
      reinterpret_cast<unsigned long long*>(near_tie), status);
  return cudaGetLastError();
}

}  // namespace pr2
