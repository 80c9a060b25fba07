// fp32 routing kernels (exact fp32 SIMT arithmetic; TF32 tensor cores would not meet the fp32
// tolerance).  One warp per token.
//   predict (Eqs. pr2_predict, pr2_route): z = h W^T + h W_p^T, rho_hat = Softmax(z),
//            idx = TopK(rho_hat, k) (ties to the lower expert), gates = rho_hat[idx].
//   replay  (Sec. 4.1 "Replay During Training"): rho = Softmax(h W^T), gates = rho[idx_in].
// PR2_F_NORMALIZE_TOPK divides a token's gates by their sum (over its valid slots).
#include <float.h>

#include "route_epilogue.cuh"

namespace pr2 {
namespace {

constexpr int kWarps = 8;

__global__ void __launch_bounds__(kWarps * 32)
    route_simt_kernel(int T, int d, int N, int k, int predict, const float* __restrict__ h,
                      const float* __restrict__ W, const float* __restrict__ Wp,
                      const int32_t* __restrict__ idx_in, int32_t* __restrict__ idx_out,
                      float* __restrict__ gates, float* __restrict__ aux,
                      unsigned long long* near_tie, int32_t* status, int norm) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int t = blockIdx.x * kWarps + (threadIdx.x >> 5);
  if (t >= T) return;
  const float* ht = h + static_cast<int64_t>(t) * d;

  // z for experts e = j*32 + lane lives in zr[j]; p (router part alone) in pr[j].
  float zr[kRoutePerLane], pr[kRoutePerLane];
#pragma unroll
  for (int j = 0; j < kRoutePerLane; ++j) {
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
        b = warp_sum_f(b);
      } else {
        for (int i = lane; i < d; i += 32) p = fmaf(ht[i], we[i], p);
      }
      p = warp_sum_f(p);
      if (lane == l) {
        pr[j] = p;
        zr[j] = p + b;
      }
    }
  }
  const bool tie = route_warp_finish(predict != 0, t, N, k, zr, pr, idx_in, idx_out, gates, aux,
                                     status, norm != 0);
  if (tie && lane == 0 && near_tie != nullptr) atomicAdd(near_tie, 1ull);
}

}  // namespace

cudaError_t launch_route_simt(const pr2_dims& dm, bool predict, const float* h, const float* W,
                              const float* Wp, const int32_t* idx_in, int32_t* idx_out,
                              float* gates, float* aux, int64_t* near_tie, int32_t* status,
                              cudaStream_t st) {
  const int T = static_cast<int>(dm.T);
  if (T == 0) return cudaSuccess;
  dim3 grid((T + kWarps - 1) / kWarps);
  return launch_pdl(route_simt_kernel, grid, dim3(kWarps * 32), 0, st, 1, T, dm.d, dm.N, dm.k,
                    predict ? 1 : 0, h, W, Wp, idx_in, idx_out, gates, aux,
                    reinterpret_cast<unsigned long long*>(near_tie), status,
                    (dm.flags & PR2_F_NORMALIZE_TOPK) ? 1 : 0);
}

}  // namespace pr2
