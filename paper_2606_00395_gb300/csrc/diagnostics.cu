// Route-tracking diagnostics (Sec. 5 "Top-k Agreement and Route KL", "Deviation Tails") and the
// fixed-length feature-cache writer (Algorithm 2, App. "uniform sub-sampling").
//
// Diagnostics: one warp per token.  Lane l holds rho[t, 32 j + l] and cached slot l.  A cached
// expert e lies in I_t = TopK(rho_t, k) (largest values, the lower expert first on equal
// values, as TopK of Eq. pr2_route) exactly when fewer than k experts beat it, where j beats e
// if rho_j > rho_e or rho_j = rho_e and j < e, i.e. if j's 64-bit rank key (orderable value
// bits, inverted index) is larger; the warp counts the experts that beat each cached entry
// with one ballot per 32 experts.
// overlap_t = |Î_t ∩ I_t| counts the cached entries (in range, not repeated) that pass.
// hist[k - overlap_t] and sum_t overlap_t are accumulated per block in shared memory and then
// with 64-bit integer atomics (order-independent, so exact and deterministic); the
// grid is at most two blocks per SM, each looping over tokens, so that the k + 2 global
// counters see few atomics.
// Feature cache: row c of the cache is row pos_c = floor(c T / T_c) of the batch; one warp per
// cached row copies h (16-byte vectors, eight in flight per lane) and the fp32 router logits.
#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kWarps = 16;

// Rank key of expert e with probability x: a larger key ranks higher (larger x; on equal x the
// lower expert).  -0 is taken as +0, so that equal values compare equal as floats do.
__device__ __forceinline__ uint64_t rank_key(float x, int e) {
  const uint32_t u = __float_as_uint(x + 0.0f);
  const uint32_t ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return (static_cast<uint64_t>(ord) << 32) | static_cast<uint32_t>(~e);
}

// kNJ = experts per lane (N <= 32 kNJ).
template <int kNJ>
__global__ void __launch_bounds__(kWarps * 32)
    diagnostics_kernel(const float* __restrict__ rho, const int32_t* __restrict__ cached,
                       int64_t T, int N, int k, unsigned long long* __restrict__ hist,
                       unsigned long long* __restrict__ overlap_sum) {
  __shared__ unsigned int sh_hist[kMaxTopKSimt + 1];
  __shared__ unsigned int sh_sum;
  pdl_wait();
  pdl_trigger();
  for (int i = threadIdx.x; i <= k; i += blockDim.x) sh_hist[i] = 0u;
  if (threadIdx.x == 0) sh_sum = 0u;
  __syncthreads();
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kWarps;
  for (int64_t t = static_cast<int64_t>(blockIdx.x) * kWarps + (threadIdx.x >> 5); t < T;
       t += nwarps) {
    const float* row = rho + t * N;
    // One round of loads per token: the row of rho and the k cached entries (lane sl holds
    // slot sl), so that nothing below waits on a dependent global load.
    const int e_l = lane < k ? cached[t * k + lane] : -1;
    float v[kNJ];
#pragma unroll
    for (int j = 0; j < kNJ; ++j) {
      const int e = j * 32 + lane;
      v[j] = e < N ? row[e] : 0.f;
    }
    uint64_t key[kNJ];  // experts beyond N get key 0, below every real key
#pragma unroll
    for (int j = 0; j < kNJ; ++j) key[j] = j * 32 + lane < N ? rank_key(v[j], j * 32 + lane) : 0ull;
    // slot sl counts if its entry is in range and no earlier slot holds the same expert
    bool ok_l = lane < k && e_l >= 0 && e_l < N;
    for (int s2 = 0; s2 < k - 1; ++s2) {
      const int es = __shfl_sync(0xffffffffu, e_l, s2);
      if (s2 < lane && es == e_l) ok_l = false;
    }
    // the rank key of this lane's slot, from the lane that holds rho[t, e_l]
    const int src = ok_l ? e_l : 0;
    uint64_t ks_l = 0;
#pragma unroll
    for (int j = 0; j < kNJ; ++j) {
      const uint64_t x = __shfl_sync(0xffffffffu, key[j], src & 31);
      if (j == (src >> 5)) ks_l = x;
    }
    const unsigned okmask = __ballot_sync(0xffffffffu, ok_l);
    // a cached expert is in TopK(rho_t, k) iff fewer than k experts rank above it
    int ov = 0;
    for (int sl = 0; sl < k; ++sl) {  // uniform over the warp
      const uint64_t ks = __shfl_sync(0xffffffffu, ks_l, sl);
      if (!((okmask >> sl) & 1u)) continue;
      int beat = 0;
#pragma unroll
      for (int j = 0; j < kNJ; ++j) beat += __popc(__ballot_sync(0xffffffffu, key[j] > ks));
      ov += beat < k ? 1 : 0;
    }
    if (lane == 0) {
      atomicAdd(&sh_hist[k - ov], 1u);
      atomicAdd(&sh_sum, static_cast<unsigned int>(ov));
    }
  }
  __syncthreads();
  for (int i = threadIdx.x; i <= k; i += blockDim.x)
    if (sh_hist[i] != 0u) atomicAdd(&hist[i], static_cast<unsigned long long>(sh_hist[i]));
  if (threadIdx.x == 0 && sh_sum != 0u)
    atomicAdd(overlap_sum, static_cast<unsigned long long>(sh_sum));
}

// cache_h[c] = h[pos_c], cache_p[c] = logits[pos_c], pos_c = floor(c T / Tc); one warp per row.
__global__ void __launch_bounds__(256)
    feature_cache_kernel(const uint4* __restrict__ h, const float* __restrict__ logits,
                         int64_t T, int64_t Tc, int row_vec, int N, int32_t* __restrict__ pos,
                         uint4* __restrict__ cache_h, float* __restrict__ cache_p) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  for (int64_t c = warp0; c < Tc; c += nwarps) {
    const int64_t p = (c * T) / Tc;
    if (lane == 0) pos[c] = static_cast<int32_t>(p);
    const uint4* src = h + p * row_vec;
    uint4* dst = cache_h + c * row_vec;
    // eight 16-byte loads in flight per lane before the stores (a 4 KB row in one round)
    for (int v0 = 0; v0 < row_vec; v0 += 8 * 32) {
      uint4 r[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int v = v0 + j * 32 + lane;
        if (v < row_vec) r[j] = __ldg(src + v);
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int v = v0 + j * 32 + lane;
        if (v < row_vec) dst[v] = r[j];
      }
    }
    if (logits != nullptr) {
      const float* ls = logits + p * N;
      float* ld = cache_p + c * N;
      for (int v = lane; v < N; v += 32) ld[v] = __ldg(ls + v);
    }
  }
}

}  // namespace

cudaError_t launch_diagnostics(const float* rho, const int32_t* cached, int64_t T, int N, int k,
                               int64_t* hist, int64_t* overlap_sum, int num_sms,
                               cudaStream_t st) {
  if (T == 0) return cudaSuccess;
  int64_t want = (T + kWarps - 1) / kWarps;
  if (want > 2 * static_cast<int64_t>(num_sms)) want = 2 * static_cast<int64_t>(num_sms);
  const unsigned blocks = static_cast<unsigned>(want);
  auto* h64 = reinterpret_cast<unsigned long long*>(hist);
  auto* o64 = reinterpret_cast<unsigned long long*>(overlap_sum);
  const dim3 grid(blocks), block(kWarps * 32);
  if (N <= 32) return launch_pdl(diagnostics_kernel<1>, grid, block, 0, st, 1, rho, cached, T, N, k, h64, o64);
  if (N <= 64) return launch_pdl(diagnostics_kernel<2>, grid, block, 0, st, 1, rho, cached, T, N, k, h64, o64);
  if (N <= 128) return launch_pdl(diagnostics_kernel<4>, grid, block, 0, st, 1, rho, cached, T, N, k, h64, o64);
  return launch_pdl(diagnostics_kernel<8>, grid, block, 0, st, 1, rho, cached, T, N, k, h64, o64);
}

cudaError_t launch_feature_cache(const void* h, const float* logits, int64_t T, int64_t Tc,
                                 int d, int N, int esz, int32_t* pos, void* cache_h,
                                 float* cache_p, int num_sms, cudaStream_t st) {
  if (Tc == 0) return cudaSuccess;
  int64_t blocks = (Tc + 7) / 8;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  if (blocks > cap) blocks = cap;
  return launch_pdl(feature_cache_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, 1,
                    static_cast<const uint4*>(h), logits, T, Tc, d * esz / 16, N, pos,
                    static_cast<uint4*>(cache_h), cache_p);
}

}  // namespace pr2
