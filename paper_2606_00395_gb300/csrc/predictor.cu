// Gradient of the predictive loss w.r.t. the evolution predictor (Eq. pr2_loss, Algorithm 3):
//   grad_Wp[j, i] = (1/T_c) sum_c G[c, j] h_old[c, i],   G = dKL/dz = pred - target,
// and the loss (1/T_c) sum_c KL_c.  G and the per-token KL come from the routing kernel in its
// loss mode (route_tc.cu), G stored transposed in bf16 ([N, Tpad]).
//
// bf16: one tcgen05 GEMM D[N x d] = Gt[N x T] h_old[T x d].  The A operand (Gt) is K-major;
// h_old is used as it is stored ([T, d], d contiguous), i.e. as an MN-major B operand: each
// stage holds four 64 x 64 TMA boxes (64 tokens x 64 columns of d) side by side along d.  The
// token dimension is split over `split` CTAs per output tile (each K block chain is short), the
// fp32 partials go to a workspace and a second kernel sums them in split order and scales by
// 1/T_c (deterministic); it also sums the per-token KL in double in a fixed tree order.
// fp32: exact-fp32 SIMT kernels (one warp per cached token, one thread per gradient entry).
#include <float.h>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kThreads = 192;
constexpr int kBK = 64;                          // tokens per K block
constexpr int kBN = 256;                         // d columns per output tile
constexpr int kATile = kTileM * kBK * 2;         // 16 KB: 128 experts x 64 tokens
constexpr int kBBox = kBK * 64 * 2;              // 8 KB: 64 tokens x 64 columns
constexpr int kBTile = (kBN / 64) * kBBox;       // 32 KB
constexpr int kStageBytes = kATile + kBTile;
constexpr int kStages = 4;
constexpr int kBarOffset = kStages * kStageBytes;
constexpr int kSmemBytes = 1024 + kBarOffset + 256;

__global__ void __launch_bounds__(kThreads, 1)
    loss_grad_tc_kernel(const __grid_constant__ CUtensorMap tm_gt,
                        const __grid_constant__ CUtensorMap tm_h, GradArgs g) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  const uint32_t pad = (1024u - (smem_u32(smem_raw) & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kBarOffset);
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;
  uint64_t* drain = acc_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_tiles_n = (g.d + kBN - 1) / kBN;
  const int m_tiles = (g.N + kTileM - 1) / kTileM;
  const int nt = static_cast<int>(blockIdx.x) % n_tiles_n;
  const int rest = static_cast<int>(blockIdx.x) / n_tiles_n;
  const int mt = rest % m_tiles;
  const int sp = rest / m_tiles;
  const int KBper = (g.Tpad / kBK) / g.split;
  const int kb0 = sp * KBper, kb1 = kb0 + KBper;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tm_gt);
    tma_prefetch_desc(&tm_h);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kBN);
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();  // G comes from the routing kernel in loss mode
  pdl_trigger();

  if (warp == 0 && lane == 0) {
    // ---------------- TMA producer ----------------
    uint32_t issued = 0, last_par = 0;
    int stage = 0;
    uint32_t phase = 0;
    for (int kb = kb0; kb < kb1; ++kb) {
      if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, g.status)) break;
      uint8_t* sa = smem + stage * kStageBytes;
      uint8_t* sb = sa + kATile;
      mbar_arrive_expect_tx(&full[stage], kStageBytes);
      tma_load_2d(sa, &tm_gt, &full[stage], kb * kBK, mt * kTileM);
      for (int q = 0; q < kBN / 64; ++q)
        tma_load_2d(sb + q * kBBox, &tm_h, &full[stage], nt * kBN + q * 64, kb * kBK);
      issued |= 1u << stage;
      last_par = (last_par & ~(1u << stage)) | (phase << stage);
      if (++stage == kStages) {
        stage = 0;
        phase ^= 1u;
      }
    }
    for (int s = 0; s < kStages; ++s)
      if ((issued >> s) & 1u)
        mbar_wait_slow(&full[s], (last_par >> s) & 1u, nullptr, nullptr, kDrainLimitNs);
  } else if (warp == 1 && lane == 0) {
    // ---------------- MMA issuer ----------------
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int kb = kb0; kb < kb1 && ok; ++kb) {
      if (!mbar_wait(&full[stage], phase, abort_flag, g.status)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + stage * kStageBytes);
      const uint32_t sb = sa + kATile;
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk)
        umma_bf16(tmem, umma_desc_sw128(sa + kk * 32), umma_desc_sw128_mn(sb + kk * 2048, kBBox),
                  umma_idesc_bf16_bmn(kTileM, kBN), (kb > kb0 || kk > 0) ? 1u : 0u);
      umma_commit(&empty[stage]);
      if (++stage == kStages) {
        stage = 0;
        phase ^= 1u;
      }
    }
    if (ok) umma_commit(acc_full);
    umma_commit(drain);
    mbar_wait_slow(drain, 0, nullptr, nullptr, kDrainLimitNs);
  } else if (warp >= 2) {
    // ---------------- epilogue: TMEM lane = expert row ----------------
    const int q = warp & 3;
    const int j = mt * kTileM + q * 32 + lane;
    const uint32_t trow = tmem + (static_cast<uint32_t>(q * 32) << 16);
    const bool have = __all_sync(0xffffffffu, mbar_wait(acc_full, 0, abort_flag, g.status));
    if (have) {
      tc_fence_after();
      float* dst = g.partial + (static_cast<int64_t>(sp) * g.N + j) * g.d + nt * kBN;
      for (int c0 = 0; c0 < kBN; c0 += 16) {
        uint32_t r[16];
        tmem_ld16(trow + c0, r);
        tmem_wait_ld(r);
        if (j < g.N && nt * kBN + c0 < g.d) {
          float4* o = reinterpret_cast<float4*>(dst + c0);
#pragma unroll
          for (int v = 0; v < 4; ++v)
            o[v] = make_float4(__uint_as_float(r[4 * v]), __uint_as_float(r[4 * v + 1]),
                               __uint_as_float(r[4 * v + 2]), __uint_as_float(r[4 * v + 3]));
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kBN);
  }
}

// grad = (1/T_c) sum over splits (split order, the split loop unrolled against its compile-time
// maximum so that every partial's load is in flight at once); the last block sums the
// per-token KL in double in a fixed tree order instead.
__global__ void __launch_bounds__(256)
    loss_finish_kernel(const float* __restrict__ partial, int split, int64_t n4, float scale,
                       float* __restrict__ grad, const float* __restrict__ kl_tok, int Tc,
                       float* __restrict__ loss) {
  pdl_wait();
  pdl_trigger();
  if (blockIdx.x == gridDim.x - 1) {
    __shared__ double sh[256];
    double acc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = 0.0;
    for (int c0 = 0; c0 < Tc; c0 += 8 * 256) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int c = c0 + j * 256 + static_cast<int>(threadIdx.x);
        if (c < Tc) acc[j] += static_cast<double>(kl_tok[c]);
      }
    }
    double s = 0.0;
#pragma unroll
    for (int j = 0; j < 8; ++j) s += acc[j];
    sh[threadIdx.x] = s;
    __syncthreads();
    for (int w = 128; w > 0; w >>= 1) {
      if (static_cast<int>(threadIdx.x) < w) sh[threadIdx.x] += sh[threadIdx.x + w];
      __syncthreads();
    }
    if (threadIdx.x == 0) *loss = Tc > 0 ? static_cast<float>(sh[0] / Tc) : 0.f;
    return;
  }
  const int64_t stride = static_cast<int64_t>(gridDim.x - 1) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4;
       i += stride) {
    float4 v[kLossMaxSplit];
#pragma unroll
    for (int s = 0; s < kLossMaxSplit; ++s)
      if (s < split) v[s] = reinterpret_cast<const float4*>(partial)[s * n4 + i];
    float4 acc = v[0];
#pragma unroll
    for (int s = 1; s < kLossMaxSplit; ++s) {
      if (s < split) {
        acc.x += v[s].x;
        acc.y += v[s].y;
        acc.z += v[s].z;
        acc.w += v[s].w;
      }
    }
    reinterpret_cast<float4*>(grad)[i] =
        make_float4(acc.x * scale, acc.y * scale, acc.z * scale, acc.w * scale);
  }
}

// ---- fp32 path ----------------------------------------------------------------------------

constexpr int kPerLane = kMaxExperts / 32;

__device__ __forceinline__ float wsum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float wmax(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// One warp per cached token c; lane l holds experts e = 32 jj + l.
__global__ void __launch_bounds__(256)
    loss_simt_kernel(const float* __restrict__ h_old, const float* __restrict__ p_old,
                     const float* __restrict__ Wp, const float* __restrict__ rho, int64_t T_rho,
                     const int32_t* __restrict__ pos, int delta, int Tc, int d, int N,
                     float* __restrict__ kl_tok, float* __restrict__ G, int32_t* status) {
  pdl_wait();
  pdl_trigger();
  const int lane = threadIdx.x & 31;
  const int c = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (c >= Tc) return;
  const int64_t r = pos != nullptr ? static_cast<int64_t>(pos[c]) : c;
  float* grow = G + static_cast<int64_t>(c) * N;
  if (r < 0 || r >= T_rho) {
    for (int e = lane; e < N; e += 32) grow[e] = 0.f;
    if (lane == 0) {
      kl_tok[c] = 0.f;
      if (status != nullptr) atomicOr(status, PR2_STATUS_BAD_INDEX);
    }
    return;
  }
  const float* hc = h_old + static_cast<int64_t>(c) * d;
  float v[kPerLane], u[kPerLane], rv[kPerLane];
#pragma unroll
  for (int jj = 0; jj < kPerLane; ++jj) {
    v[jj] = -INFINITY;
    u[jj] = -INFINITY;
    rv[jj] = 0.f;
    for (int l = 0; l < 32; ++l) {
      const int e = jj * 32 + l;
      if (e >= N) break;
      const float* we = Wp + static_cast<int64_t>(e) * d;
      float b = 0.f;
      for (int i = lane; i < d; i += 32) b = fmaf(hc[i], we[i], b);
      b = wsum(b);
      if (lane == l) {
        const float po = p_old[static_cast<int64_t>(c) * N + e];
        const float tr = rho[r * N + e];
        rv[jj] = tr;
        v[jj] = delta ? b : po + b;
        u[jj] = tr > 0.f ? logf(tr) - po : -INFINITY;
      }
    }
  }
  float m1 = -INFINITY, m2 = -INFINITY;
#pragma unroll
  for (int jj = 0; jj < kPerLane; ++jj) {
    m1 = fmaxf(m1, v[jj]);
    m2 = fmaxf(m2, u[jj]);
  }
  m1 = wmax(m1);
  m2 = wmax(m2);
  float s1 = 0.f, s2 = 0.f;
#pragma unroll
  for (int jj = 0; jj < kPerLane; ++jj) {
    if (jj * 32 + lane < N) {
      s1 += expf(v[jj] - m1);
      if (u[jj] != -INFINITY) s2 += expf(u[jj] - m2);
    }
  }
  const float l1 = m1 + logf(wsum(s1));
  const float l2 = m2 + logf(wsum(s2));
  float kl = 0.f;
#pragma unroll
  for (int jj = 0; jj < kPerLane; ++jj) {
    const int e = jj * 32 + lane;
    if (e >= N) continue;
    const float lp = v[jj] - l1;
    float tg, lt;
    if (delta) {
      lt = u[jj] - l2;
      tg = rv[jj] > 0.f ? expf(lt) : 0.f;
    } else {
      tg = rv[jj];
      lt = rv[jj] > 0.f ? logf(rv[jj]) : 0.f;
    }
    if (tg > 0.f) kl += tg * (lt - lp);
    grow[e] = expf(lp) - tg;
  }
  kl = wsum(kl);
  if (lane == 0) kl_tok[c] = kl;
}

// grad[j, i] = (1/T_c) sum_c G[c, j] h_old[c, i]; one thread per entry, consecutive i.
__global__ void __launch_bounds__(256)
    loss_grad_simt_kernel(const float* __restrict__ G, const float* __restrict__ h_old, int Tc,
                          int d, int N, float* __restrict__ grad) {
  pdl_wait();
  pdl_trigger();
  const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= static_cast<int64_t>(N) * d) return;
  const int j = static_cast<int>(idx / d), i = static_cast<int>(idx % d);
  float acc = 0.f;
  for (int c = 0; c < Tc; ++c)
    acc = fmaf(G[static_cast<int64_t>(c) * N + j], h_old[static_cast<int64_t>(c) * d + i], acc);
  grad[idx] = Tc > 0 ? acc / static_cast<float>(Tc) : 0.f;
}

}  // namespace

int loss_grad_split(int N, int d, int Tpad, int num_sms) {
  const int tiles = ((N + kTileM - 1) / kTileM) * ((d + kBN - 1) / kBN);
  const int KB = Tpad / kBK;
  int s = 1;
  while (s * 2 <= kLossMaxSplit && KB % (s * 2) == 0 && tiles * s * 2 <= num_sms) s *= 2;
  return s;
}

cudaError_t launch_loss_grad_tc(const CUtensorMap& tm_gt, const CUtensorMap& tm_h,
                                const GradArgs& g, cudaStream_t st) {
  cudaError_t err = cudaFuncSetAttribute(loss_grad_tc_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (err != cudaSuccess) return err;
  const int tiles = ((g.N + kTileM - 1) / kTileM) * ((g.d + kBN - 1) / kBN);
  return launch_pdl(loss_grad_tc_kernel, dim3(tiles * g.split), dim3(kThreads), kSmemBytes, st,
                    1, tm_gt, tm_h, g);
}

cudaError_t launch_loss_finish(const GradArgs& g, cudaStream_t st) {
  // without partials (fp32 path) only the loss is summed
  const int64_t n4 = g.partial != nullptr ? static_cast<int64_t>(g.N) * g.d / 4 : 0;
  int64_t blocks = (n4 + 255) / 256;
  if (blocks > 1024) blocks = 1024;
  blocks += 1;  // the last block sums the loss
  const float scale = g.Tc > 0 ? 1.0f / static_cast<float>(g.Tc) : 0.f;
  return launch_pdl(loss_finish_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, 1,
                    static_cast<const float*>(g.partial), g.split, n4, scale, g.grad, g.kl_tok,
                    g.Tc, g.loss);
}

cudaError_t launch_loss_simt(const float* h_old, const float* p_old, const float* Wp,
                             const float* rho, int64_t T_rho, const int32_t* pos, int delta,
                             int Tc, int d, int N, float* kl_tok, float* G, int32_t* status,
                             cudaStream_t st) {
  if (Tc == 0) return cudaSuccess;
  return launch_pdl(loss_simt_kernel, dim3((Tc + 7) / 8), dim3(256), 0, st, 1, h_old, p_old, Wp,
                    rho, T_rho, pos, delta, Tc, d, N, kl_tok, G, status);
}

cudaError_t launch_loss_grad_simt(const float* G, const float* h_old, int Tc, int d, int N,
                                  float* grad, cudaStream_t st) {
  const int64_t n = static_cast<int64_t>(N) * d;
  return launch_pdl(loss_grad_simt_kernel, dim3(static_cast<unsigned>((n + 255) / 256)),
                    dim3(256), 0, st, 1, G, h_old, Tc, d, N, grad);
}

}  // namespace pr2
