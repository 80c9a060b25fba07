// Gradient of the predictive loss w.r.t. the evolution predictor (Eq. pr2_loss, Algorithm 3):
//   grad_Wp[j, i] = (1/T_c) sum_c G[c, j] h_old[c, i],   G = dKL/dz = pred - target,
// and the loss (1/T_c) sum_c KL_c.  G and the per-token KL come from the routing kernel in its
// loss mode (route_tc.cu), G stored transposed in bf16 ([N, Tpad]).
//
// bf16: one tcgen05 GEMM D[N x d] = Gt[N x T] h_old[T x d].  The A operand (Gt) is K-major;
// h_old is used as it is stored ([T, d], d contiguous), i.e. as an MN-major B operand: each
// stage holds four 64 x 64 TMA boxes (64 tokens x 64 columns of d) side by side along d.  The
// token dimension is split over the `split` CTAs of a cluster per output tile (each K block
// chain is short); the cluster sums its fp32 partials, exchanged through L2, in split order and
// scales by 1/T_c (deterministic), and the same launch sums the per-token KL in double in a fixed
// order, so the loss call is two launches.
// fp32: exact-fp32 SIMT kernels (one warp per cached token, one thread per gradient entry).
#include <float.h>

#include <mutex>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kThreads = 192;
constexpr int kBK = 64;                          // tokens per K block
constexpr int kBN = 128;                         // d columns per output tile
constexpr int kATile = kTileM * kBK * 2;         // 16 KB: 128 experts x 64 tokens
constexpr int kBBox = kBK * 64 * 2;              // 8 KB: 64 tokens x 64 columns
constexpr int kBTile = (kBN / 64) * kBBox;       // 16 KB
constexpr int kStageBytes = kATile + kBTile;
constexpr int kStages = 4;
constexpr int kBarOffset = kStages * kStageBytes;
constexpr int kSmemBytes = 1024 + kBarOffset + 256;

// (1/T_c) sum_c kl_tok[c] in double, in one fixed order: thread t of 64 adds c = t + 64 j + 512 i
// into its accumulator j (j < 8, i ascending), then sums its 8 accumulators, then the 64 partial
// sums meet in a tree.  The values are loaded 32 per thread at a time (one round trip for
// T_c <= 2048).  `sh` holds 64 doubles; the 64 threads (two whole warps) meet on hardware
// barrier `bar`.
__device__ void sum_kl_tokens(const float* __restrict__ kl_tok, int Tc, float* __restrict__ loss,
                              double* sh, int t, int bar) {
  double acc[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) acc[j] = 0.0;
  for (int c0 = 0; c0 < Tc; c0 += 4 * 8 * 64) {
    float x[4][8];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int c = c0 + i * 512 + j * 64 + t;
        x[i][j] = c < Tc ? kl_tok[c] : 0.f;
      }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 8; ++j)
        if (c0 + i * 512 + j * 64 + t < Tc) acc[j] += static_cast<double>(x[i][j]);
  }
  double s = 0.0;
#pragma unroll
  for (int j = 0; j < 8; ++j) s += acc[j];
  sh[t] = s;
  named_bar_sync(bar, 64);
  for (int w = 32; w > 0; w >>= 1) {
    if (t < w) sh[t] += sh[t + w];
    named_bar_sync(bar, 64);
  }
  if (t == 0) *loss = Tc > 0 ? static_cast<float>(sh[0] / Tc) : 0.f;
}

// One 128 x 128 output tile per cluster of kSplit CTAs, which split the token dimension K.
// With kSplit > 1 every CTA writes its fp32 accumulator tile to the workspace (L2-resident, 64 KB
// per CTA, coalesced), the cluster meets at a barrier, and CTA r sums columns
// [r 128 / kSplit, (r + 1) 128 / kSplit) of the kSplit partial tiles in rank order (= token
// order), scales by 1/T_c and writes the gradient.  One extra cluster after the tiles sums the
// per-token KL into the loss (warps 0-1 of its first CTA), off the tiles' path.
template <int kSplit>
__global__ void __launch_bounds__(kThreads, 1)
    loss_grad_tc_kernel(const __grid_constant__ CUtensorMap tm_gt,
                        const __grid_constant__ CUtensorMap tm_h, GradArgs g) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  __shared__ double kl_sh[64];
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
  const int sp = static_cast<int>(blockIdx.x) % kSplit;  // the CTA's rank in its cluster
  const int tile = static_cast<int>(blockIdx.x) / kSplit;
  if (tile >= ((g.N + kTileM - 1) / kTileM) * n_tiles_n) {
    // the extra cluster after the output tiles: its first CTA sums the per-token KL into the
    // loss, beside the GEMM instead of after it
    pdl_wait();  // the per-token KL comes from the routing kernel in loss mode
    pdl_trigger();
    if (sp == 0 && warp < 2) sum_kl_tokens(g.kl_tok, g.Tc, g.loss, kl_sh, threadIdx.x, 2);
    return;
  }
  const int nt = tile % n_tiles_n;
  const int mt = tile / n_tiles_n;
  const int KBper = (g.Tpad / kBK) / kSplit;
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
  pdl_wait();  // G and the per-token KL come from the routing kernel in loss mode
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
  }
  __syncwarp();

  // ---------------- epilogue: TMEM lane = expert row ----------------
  const bool epi = warp >= 2;
  const int q = warp & 3;
  const int row = q * 32 + lane;  // row of the tile = TMEM lane
  const uint32_t trow = tmem + (static_cast<uint32_t>(q * 32) << 16);
  const float scale = g.Tc > 0 ? 1.0f / static_cast<float>(g.Tc) : 0.f;
  bool have = false;
  if (epi) {
    // tcgen05.ld is warp-collective: the whole warp reads TMEM or none of it does.
    have = __all_sync(0xffffffffu, mbar_wait(acc_full, 0, abort_flag, g.status));
    if (have) tc_fence_after();
  }
  if (kSplit == 1) {
    const int j = mt * kTileM + row;
    if (have) {
      float* dst = g.grad + static_cast<int64_t>(j) * g.d + nt * kBN;
      for (int c0 = 0; c0 < kBN; c0 += 16) {
        uint32_t r[16];
        tmem_ld16(trow + c0, r);
        tmem_wait_ld(r);
        if (j < g.N && nt * kBN + c0 < g.d) {
          float4* o = reinterpret_cast<float4*>(dst + c0);
#pragma unroll
          for (int v = 0; v < 4; ++v)
            o[v] = make_float4(__uint_as_float(r[4 * v]) * scale,
                               __uint_as_float(r[4 * v + 1]) * scale,
                               __uint_as_float(r[4 * v + 2]) * scale,
                               __uint_as_float(r[4 * v + 3]) * scale);
        }
      }
    }
  } else {
    constexpr int kCw = kBN / kSplit;  // columns summed by one CTA of the cluster
    constexpr int kC4 = kBN / 4;       // 16-byte words of one partial row
    // partial tile of source sp: word (c4, row) at [(tile kSplit + sp) kC4 + c4] 128 + row,
    // so that consecutive rows (lanes) write consecutive 16-byte words
    float4* part = reinterpret_cast<float4*>(g.partial) +
                   static_cast<int64_t>(tile) * kSplit * kC4 * kTileM;
    if (have) {
      // 64 columns per round: four TMEM loads in flight, one wait, sixteen 16-byte stores
      float4* mine = part + static_cast<int64_t>(sp) * kC4 * kTileM + row;
      for (int c0 = 0; c0 < kBN; c0 += 64) {
        uint32_t r[4][16];
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4) tmem_ld16(trow + c0 + q4 * 16, r[q4]);
        tmem_wait_ld(r[0]);
#pragma unroll
        for (int q4 = 1; q4 < 4; ++q4) reg_fence(r[q4]);
#pragma unroll
        for (int q4 = 0; q4 < 4; ++q4)
#pragma unroll
          for (int j = 0; j < 4; ++j)
            mine[((c0 + q4 * 16) / 4 + j) * kTileM] = make_float4(
                __uint_as_float(r[q4][4 * j]), __uint_as_float(r[q4][4 * j + 1]),
                __uint_as_float(r[q4][4 * j + 2]), __uint_as_float(r[q4][4 * j + 3]));
      }
      __threadfence();  // the partial tile is visible GPU-wide before the cluster barrier
    }
    cluster_sync();  // every partial tile of the cluster is written
    if (epi) {
      // this CTA's words: (kCw / 4) column words x 128 rows, kIter per thread, all of their
      // kSplit x kIter loads in flight before the sums
      constexpr int kWords = (kCw / 4) * kTileM;
      constexpr int kIter = kWords / 128;
      static_assert(kWords % 128 == 0, "whole rounds of 128 threads");
      float4 w[kIter][kSplit];
#pragma unroll
      for (int it = 0; it < kIter; ++it) {
        const int i = it * 128 + threadIdx.x - 64;
        const int c4 = sp * (kCw / 4) + i / kTileM;
#pragma unroll
        for (int src = 0; src < kSplit; ++src)
          w[it][src] = __ldcg(part + (static_cast<int64_t>(src) * kC4 + c4) * kTileM + i % kTileM);
      }
#pragma unroll
      for (int it = 0; it < kIter; ++it) {
        const int i = it * 128 + threadIdx.x - 64;
        float4 v = w[it][0];
#pragma unroll
        for (int src = 1; src < kSplit; ++src) {
          v.x += w[it][src].x;
          v.y += w[it][src].y;
          v.z += w[it][src].z;
          v.w += w[it][src].w;
        }
        const int j = mt * kTileM + i % kTileM;
        const int col = nt * kBN + (sp * (kCw / 4) + i / kTileM) * 4;
        if (j < g.N && col < g.d)
          *reinterpret_cast<float4*>(g.grad + static_cast<int64_t>(j) * g.d + col) =
              make_float4(v.x * scale, v.y * scale, v.z * scale, v.w * scale);
      }
    }
  }
  if (epi) tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kBN);
  }
}

// The loss of the fp32 path: one block of 64 threads sums the per-token KL (same order as the
// bf16 path's gradient kernel).
__global__ void __launch_bounds__(64)
    loss_finish_kernel(const float* __restrict__ kl_tok, int Tc, float* __restrict__ loss) {
  __shared__ double sh[64];
  pdl_wait();
  pdl_trigger();
  sum_kl_tokens(kl_tok, Tc, loss, sh, threadIdx.x, 1);
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

int64_t loss_grad_rows(int N) { return static_cast<int64_t>((N + kTileM - 1) / kTileM) * kTileM; }
int64_t loss_grad_cols(int d) { return static_cast<int64_t>((d + kBN - 1) / kBN) * kBN; }

namespace {

// Clusters of kSplit gradient CTAs that can be resident at once on the current device (cached).
template <int kSplit>
int grad_clusters_resident() {
  static std::mutex mu;
  static int cached_dev[8] = {-1, -1, -1, -1, -1, -1, -1, -1};
  static int cached_n[8] = {};
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < 8; ++i)
    if (cached_dev[i] == dev) return cached_n[i];
  int n = 0;
  if (cudaFuncSetAttribute(loss_grad_tc_kernel<kSplit>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) == cudaSuccess) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kSplit);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = kSmemBytes;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kSplit;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaOccupancyMaxActiveClusters(&n, loss_grad_tc_kernel<kSplit>, &cfg) != cudaSuccess)
      n = 0;
  }
  (void)cudaGetLastError();
  for (int i = 0; i < 8; ++i)
    if (cached_dev[i] < 0) {
      cached_dev[i] = dev;
      cached_n[i] = n;
      break;
    }
  return n;
}

int clusters_resident(int split) {
  switch (split) {
    case 2: return grad_clusters_resident<2>();
    case 4: return grad_clusters_resident<4>();
    case 8: return grad_clusters_resident<8>();
    default: return 0;
  }
}

}  // namespace

// The largest token split (a power of two up to kLossMaxSplit that divides the K blocks) whose
// (tiles + 1) x split CTAs (the output tiles and the loss-summing cluster) all fit on the GPU at
// once as clusters of `split`.
int loss_grad_split(int N, int d, int Tpad, int num_sms) {
  const int tiles = ((N + kTileM - 1) / kTileM) * ((d + kBN - 1) / kBN);
  const int KB = Tpad / kBK;
  int s = 1;
  while (s * 2 <= kLossMaxSplit && KB % (s * 2) == 0 && (tiles + 1) * s * 2 <= num_sms &&
         clusters_resident(s * 2) >= tiles + 1)
    s *= 2;
  return s;
}

template <int kSplit>
cudaError_t launch_grad_split(const CUtensorMap& tm_gt, const CUtensorMap& tm_h,
                              const GradArgs& g, int tiles, cudaStream_t st) {
  cudaError_t err = cudaFuncSetAttribute(loss_grad_tc_kernel<kSplit>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (err != cudaSuccess) return err;
  return launch_pdl(loss_grad_tc_kernel<kSplit>, dim3((tiles + 1) * kSplit), dim3(kThreads),
                    kSmemBytes, st, kSplit, tm_gt, tm_h, g);
}

cudaError_t launch_loss_grad_tc(const CUtensorMap& tm_gt, const CUtensorMap& tm_h,
                                const GradArgs& g, cudaStream_t st) {
  const int tiles = ((g.N + kTileM - 1) / kTileM) * ((g.d + kBN - 1) / kBN);
  switch (g.split) {
    case 1: return launch_grad_split<1>(tm_gt, tm_h, g, tiles, st);
    case 2: return launch_grad_split<2>(tm_gt, tm_h, g, tiles, st);
    case 4: return launch_grad_split<4>(tm_gt, tm_h, g, tiles, st);
    case 8: return launch_grad_split<8>(tm_gt, tm_h, g, tiles, st);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_loss_finish(const GradArgs& g, cudaStream_t st) {
  return launch_pdl(loss_finish_kernel, dim3(1), dim3(64), 0, st, 1, g.kl_tok, g.Tc, g.loss);
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
