// bf16 routing on the tcgen05 tensor cores.  One CTA = 128 tokens.
//
//   predict (Eqs. pr2_predict, pr2_route; Algorithm 2 first two steps):
//     [p_old | b] = h [W ; W_p]^T   one M=128 x N=2N accumulator in TMEM (fp32), K = d,
//     z = p_old + b, rho_hat = Softmax(z), idx = TopK(rho_hat, k), gates = rho_hat[idx],
//     p_old optionally written as the feature-cache logits.
//   replay (Sec. 4.1 "Replay During Training"):
//     p = h W^T, rho = Softmax(p), gates = rho[idx_in]   (no top-k, no predictor).
//
// Warp roles: warp 0 = TMA producer (h tile + weight tile per 64-wide K block), warp 1 = TMEM
// owner and MMA issuer, warps 2..5 = epilogue, one thread per token row (TMEM lane).
// The epilogue selects on z in fp32 (softmax is monotone, so the order equals the order of
// rho_hat); ties go to the lower expert index.
#include <float.h>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kThreads = 192;
constexpr int kBK = 64;                          // bf16 elements per 128-byte swizzle row
constexpr int kATileBytes = kTileM * kBK * 2;    // 16 KB
constexpr int kKeep = kMaxTopK + 1;              // top-(k+1) kept for the margin

struct RouteSmemLayout {
  int stages;
  int b_rows;        // rows of the weight tile: 2N (predict) or N (replay)
  int stage_bytes;   // A + B
  int bar_offset;    // after all stages
  int total;         // dynamic smem bytes requested (incl. 1 KB alignment slack)
};

__host__ __device__ inline RouteSmemLayout route_layout(int N, bool predict) {
  RouteSmemLayout L;
  L.b_rows = predict ? 2 * N : N;
  L.stage_bytes = kATileBytes + L.b_rows * kBK * 2;
  L.stages = (200 * 1024) / L.stage_bytes;
  if (L.stages > 6) L.stages = 6;
  if (L.stages < 2) L.stages = 2;
  L.bar_offset = L.stages * L.stage_bytes;
  L.total = 1024 + L.bar_offset + 256;
  return L;
}

__host__ __device__ inline uint32_t tmem_cols_for(int cols) {
  uint32_t c = 32;
  while (c < static_cast<uint32_t>(cols)) c <<= 1;
  return c;
}

__global__ void __launch_bounds__(kThreads, 1)
    route_tc_kernel(const __grid_constant__ CUtensorMap tm_h,
                    const __grid_constant__ CUtensorMap tm_w,
                    const __grid_constant__ CUtensorMap tm_wp, RouteTcArgs a, int predict) {
  extern __shared__ uint8_t smem_raw[];
  const RouteSmemLayout L = route_layout(a.N, predict != 0);
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bar_offset);
  uint64_t* empty = full + L.stages;
  uint64_t* acc_full = empty + L.stages;
  uint64_t* drain = acc_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int t0 = blockIdx.x * kTileM;
  const int KB = a.d / kBK;
  const uint32_t ncols = tmem_cols_for(L.b_rows);

  if (threadIdx.x == 0) {
    for (int s = 0; s < L.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tm_h);
    tma_prefetch_desc(&tm_w);
    if (predict) tma_prefetch_desc(&tm_wp);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, ncols);
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    const uint32_t bytes = static_cast<uint32_t>(L.stage_bytes);
    uint32_t issued = 0, last_par = 0;
    int stage = 0;
    uint32_t phase = 0;
    const uint64_t keep = l2_policy_evict_last();    // weights are re-read by every CTA
    const uint64_t stream = l2_policy_evict_first(); // h is read once
    for (int kb = 0; kb < KB; ++kb) {
      if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, a.status)) break;
      uint8_t* sa = smem + stage * L.stage_bytes;
      uint8_t* sb = sa + kATileBytes;
      mbar_arrive_expect_tx(&full[stage], bytes);
      tma_load_2d_hint(sa, &tm_h, &full[stage], kb * kBK, t0, stream);
      tma_load_2d_hint(sb, &tm_w, &full[stage], kb * kBK, 0, keep);
      if (predict) tma_load_2d_hint(sb + a.N * kBK * 2, &tm_wp, &full[stage], kb * kBK, 0, keep);
      issued |= 1u << stage;
      last_par = (last_par & ~(1u << stage)) | (phase << stage);
      if (++stage == L.stages) {
        stage = 0;
        phase ^= 1u;
      }
    }
    // Drain: every issued copy must have landed before the CTA can exit.
    for (int s = 0; s < L.stages; ++s)
      if ((issued >> s) & 1u)
        mbar_wait_slow(&full[s], (last_par >> s) & 1u, nullptr, nullptr, kDrainLimitNs);
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int kb = 0; kb < KB && ok; ++kb) {
      if (!mbar_wait(&full[stage], phase, abort_flag, a.status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + stage * L.stage_bytes);
      const uint32_t sb = sa + kATileBytes;
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk) {
        const uint64_t adesc = umma_desc_sw128(sa + kk * 32);
        for (int n0 = 0; n0 < L.b_rows; n0 += 256) {
          const int nc = (L.b_rows - n0) < 256 ? (L.b_rows - n0) : 256;
          const uint64_t bdesc = umma_desc_sw128(sb + n0 * (kBK * 2) + kk * 32);
          umma_bf16(tmem + n0, adesc, bdesc, umma_idesc_bf16(kTileM, nc),
                    (kb > 0 || kk > 0) ? 1u : 0u);
        }
      }
      umma_commit(&empty[stage]);
      if (++stage == L.stages) {
        stage = 0;
        phase ^= 1u;
      }
    }
    if (ok) umma_commit(acc_full);
    umma_commit(drain);
    mbar_wait_slow(drain, 0, nullptr, nullptr, kDrainLimitNs);
  } else if (warp >= 2) {
    // ---------------- epilogue: one thread per token ----------------
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int t = t0 + row;
    const bool live = t < a.T;
    const uint32_t trow = tmem + (static_cast<uint32_t>(q * 32) << 16);
    if (mbar_wait(acc_full, 0, abort_flag, a.status)) {
      tc_fence_after();
      const int N = a.N, k = a.k;
      if (predict) {
        float tv[kKeep];
        int ti[kKeep];
#pragma unroll
        for (int j = 0; j < kKeep; ++j) {
          tv[j] = -FLT_MAX;
          ti[j] = 0x7fffffff;
        }
        float* lrow = a.logits_or_probs ? a.logits_or_probs + static_cast<int64_t>(t) * N : nullptr;
        for (int c0 = 0; c0 < N; c0 += 16) {
          uint32_t rp[16], rb[16];
          tmem_ld16(trow + c0, rp);
          tmem_ld16(trow + N + c0, rb);
          tmem_wait_ld(rp);
          reg_fence(rb);
          if (live && lrow != nullptr) {
            float4* dst = reinterpret_cast<float4*>(lrow + c0);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              dst[j] = make_float4(__uint_as_float(rp[4 * j]), __uint_as_float(rp[4 * j + 1]),
                                   __uint_as_float(rp[4 * j + 2]), __uint_as_float(rp[4 * j + 3]));
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            float cv = __uint_as_float(rp[j]) + __uint_as_float(rb[j]);
            if (cv > tv[kKeep - 1]) {
              int ci = c0 + j;
#pragma unroll
              for (int s = 0; s < kKeep; ++s) {
                const bool sw = cv > tv[s];
                const float ov = tv[s];
                const int oi = ti[s];
                tv[s] = sw ? cv : ov;
                ti[s] = sw ? ci : oi;
                cv = sw ? ov : cv;
                ci = sw ? oi : ci;
              }
            }
          }
        }
        const float mx = tv[0];
        float sum = 0.f;
        for (int c0 = 0; c0 < N; c0 += 16) {
          uint32_t rp[16], rb[16];
          tmem_ld16(trow + c0, rp);
          tmem_ld16(trow + N + c0, rb);
          tmem_wait_ld(rp);
          reg_fence(rb);
#pragma unroll
          for (int j = 0; j < 16; ++j)
            sum += expf(__uint_as_float(rp[j]) + __uint_as_float(rb[j]) - mx);
        }
        const float inv_s = 1.0f / sum;
        bool tie = false;
        if (live) {
          int32_t* irow = a.idx_out + static_cast<int64_t>(t) * k;
          float* grow = a.gates + static_cast<int64_t>(t) * k;
          float pk = 0.f, pk1 = 0.f;
#pragma unroll
          for (int s = 0; s < kKeep; ++s) {
            const float pr = expf(tv[s] - mx) * inv_s;
            if (s < k) {
              irow[s] = ti[s];
              grow[s] = pr;
            }
            if (s == k - 1) pk = pr;
            if (s == k) pk1 = pr;
          }
          tie = (k < N) && (pk - pk1 < (float)PR2_NEAR_TIE_GAP);
        }
        const unsigned ties = __ballot_sync(0xffffffffu, tie);
        if (lane == 0 && ties != 0u && a.near_tie != nullptr)
          atomicAdd(reinterpret_cast<unsigned long long*>(a.near_tie),
                    static_cast<unsigned long long>(__popc(ties)));
      } else {
        // replay: cached indices, validated, their probabilities captured in the second pass
        int e_s[kMaxTopK];
        float z_s[kMaxTopK];
        bool bad = false;
#pragma unroll
        for (int s = 0; s < kMaxTopK; ++s) {
          int e = -1;
          if (live && s < k) {
            e = a.idx_in[static_cast<int64_t>(t) * k + s];
            bool ok = e >= 0 && e < N;
#pragma unroll
            for (int s2 = 0; s2 < kMaxTopK; ++s2)
              if (s2 < s && e_s[s2] == e) ok = false;
            if (!ok) {
              bad = true;
              e = -1;
            }
          }
          e_s[s] = e;
          z_s[s] = 0.f;
        }
        float mx = -FLT_MAX;
        for (int c0 = 0; c0 < N; c0 += 16) {
          uint32_t rp[16];
          tmem_ld16(trow + c0, rp);
          tmem_wait_ld(rp);
#pragma unroll
          for (int j = 0; j < 16; ++j) mx = fmaxf(mx, __uint_as_float(rp[j]));
        }
        float sum = 0.f;
        for (int c0 = 0; c0 < N; c0 += 16) {
          uint32_t rp[16];
          tmem_ld16(trow + c0, rp);
          tmem_wait_ld(rp);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            const float z = __uint_as_float(rp[j]);
            sum += expf(z - mx);
#pragma unroll
            for (int s = 0; s < kMaxTopK; ++s)
              if (e_s[s] == c0 + j) z_s[s] = z;
          }
        }
        const float inv_s = 1.0f / sum;
        if (live) {
          float* grow = a.gates + static_cast<int64_t>(t) * k;
#pragma unroll
          for (int s = 0; s < kMaxTopK; ++s)
            if (s < k) grow[s] = (e_s[s] >= 0) ? expf(z_s[s] - mx) * inv_s : 0.f;
          if (bad && a.status != nullptr) atomicOr(a.status, PR2_STATUS_BAD_INDEX);
        }
        if (a.logits_or_probs != nullptr) {
          float* prow = a.logits_or_probs + static_cast<int64_t>(t) * N;
          for (int c0 = 0; c0 < N; c0 += 16) {
            uint32_t rp[16];
            tmem_ld16(trow + c0, rp);
            tmem_wait_ld(rp);
            if (live) {
              float4* dst = reinterpret_cast<float4*>(prow + c0);
#pragma unroll
              for (int j = 0; j < 4; ++j)
                dst[j] = make_float4(expf(__uint_as_float(rp[4 * j]) - mx) * inv_s,
                                     expf(__uint_as_float(rp[4 * j + 1]) - mx) * inv_s,
                                     expf(__uint_as_float(rp[4 * j + 2]) - mx) * inv_s,
                                     expf(__uint_as_float(rp[4 * j + 3]) - mx) * inv_s);
            }
          }
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, ncols);
  }
}

}  // namespace

cudaError_t launch_route_tc(bool predict, const CUtensorMap& tm_h, const CUtensorMap& tm_w,
                            const CUtensorMap& tm_wp, const RouteTcArgs& a, cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  const RouteSmemLayout L = route_layout(a.N, predict);
  cudaError_t err = cudaFuncSetAttribute(route_tc_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, L.total);
  if (err != cudaSuccess) return err;
  dim3 grid((a.T + kTileM - 1) / kTileM);
  route_tc_kernel<<<grid, kThreads, L.total, st>>>(tm_h, tm_w, tm_wp, a, predict ? 1 : 0);
  return cudaGetLastError();
}

}  // namespace pr2
