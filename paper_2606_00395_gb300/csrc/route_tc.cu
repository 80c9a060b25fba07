// bf16 routing on the tcgen05 tensor cores.
//
//   predict (Eqs. pr2_predict, pr2_route; Algorithm 2 first two steps):
//     [p_old | b] = h [W ; W_p]^T   (fp32 accumulators in TMEM, K = d),
//     z = p_old + b, rho_hat = Softmax(z), idx = TopK(rho_hat, k), gates = rho_hat[idx],
//     p_old optionally written as the feature-cache logits.
//   replay (Sec. 4.1 "Replay During Training"):
//     p = h W^T, rho = Softmax(p), gates = rho[idx_in]   (no top-k, no predictor).
//
// A 128-token tile is handled by a cluster of S CTAs (S = 1, 2, 4 or 8) that split K = d.  Each
// tcgen05.mma costs the same issue time for any N <= 256 (one M=128 x N x K=16 step), so a lone
// tile's chain of d/16 MMAs, not bandwidth, bounds it, and only a K split shortens that chain:
// CTA r multiplies K blocks [r KB/S, (r+1) KB/S) into a partial [128 x NB] fp32 accumulator
// (NB = 2N columns [p_old | b] for predict, N for replay).  When the tiles outnumber the SMs
// (S = 1), each CTA takes half the pipeline stages so that two run on an SM side by side, one
// CTA's loads and finishing overlapping the other's MMAs (RouteTcArgs::compact).
//
// Warp roles: warp 0 = TMA producer, warp 1 = TMEM owner and MMA issuer, warps 2..5 = epilogue.
// With S > 1 the partials are reduce-scattered by rows through distributed shared memory: CTA q
// receives rows [q 128/S, (q+1) 128/S) of every CTA's partial, stored [source][column/4][row][4]
// so that each warp store moves contiguous bytes; the four epilogue warps then sum the S copies
// once, in source order (deterministic), walking consecutive 16-byte words so that no two lanes
// of a warp hit one bank.  Each row is then finished by S consecutive threads, thread `part` owning experts
// [part N/S, (part+1) N/S); with S = 1 one thread finishes its row straight from TMEM.  A thread
// reduces its experts to a max, a sum of exp(z - max) and (predict) its top-16 by 64-bit keys
// (orderable z bits, inverted expert index: z descending, ties to the lower expert), built by
// bitonic sorting 16 experts at a time and merging, in one pass with a running (online) softmax
// sum; the S threads of a row then combine max and sum (sum_q s_q exp(m_q - max), fixed shuffle
// order) and merge their lists by shuffles.
// Selection is on z in fp32 (softmax is monotone, so the order equals the order of rho_hat).
#include <float.h>

#include <mutex>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kThreads = 192;
constexpr int kBK = 64;                          // bf16 elements per 128-byte swizzle row
constexpr int kATileBytes = kTileM * kBK * 2;    // 16 KB
constexpr int kKeep = kMaxTopK + 1;              // top-(k+1) kept for the margin
constexpr int kMaxSplit = 8;
static_assert(kMaxSplit == kRouteMaxSplit, "histogram rows per routing tile");
constexpr int kMaxStages = 12;
constexpr int kStageBudget = 192 * 1024;    // pipeline stages of a CTA alone on its SM
constexpr int kCompactBudget = 96 * 1024;   // two CTAs per SM (more token tiles than SMs)

struct RouteSmemLayout {
  int stages;
  int b_rows;        // rows of the weight tile: 2N (predict) or N (replay)
  int passes;        // passes over K: 2 streams [W] then [W_p] (predict, N > 128), else 1
  int pass_rows;     // weight rows of a stage: b_rows / passes
  int stage_bytes;   // A + B
  int bar_offset;    // after all stages
  int total;         // dynamic smem bytes requested (incl. 1 KB alignment slack)
};

__host__ __device__ inline RouteSmemLayout route_layout(int N, bool predict, bool compact) {
  RouteSmemLayout L;
  L.b_rows = predict ? 2 * N : N;
  // Predict with more than 128 experts: [W; W_p] would make 80 KB stages (two in flight at
  // most), so the router and the predictor weights stream in two passes over K instead, each
  // stage holding N weight rows; h is read twice, but four stages overlap loads and MMAs.
  L.passes = (L.b_rows > 256 && N % 32 == 0) ? 2 : 1;
  L.pass_rows = L.b_rows / L.passes;
  L.stage_bytes = kATileBytes + L.pass_rows * kBK * 2;
  L.stages = (compact ? kCompactBudget : kStageBudget) / L.stage_bytes;
  if (L.stages > kMaxStages) L.stages = kMaxStages;
  if (L.stages < 2) L.stages = 2;
  L.bar_offset = L.stages * L.stage_bytes;
  L.total = 1024 + L.bar_offset + 256;
  return L;
}

// Bytes of the reduce-scatter buffer, [S][NB/S/4][128][4] fp32, placed over the pipeline
// stages once every CTA of the cluster has finished its K blocks.
__host__ __device__ inline int route_recv_bytes(int b_rows) { return b_rows * kTileM * 4; }

__host__ __device__ inline uint32_t tmem_cols_for(int cols) {
  uint32_t c = 32;
  while (c < static_cast<uint32_t>(cols)) c <<= 1;
  return c;
}

// Compare-exchange leaving the larger key in a.
__device__ __forceinline__ void cas_desc(uint64_t& a, uint64_t& b) {
  const bool sw = b > a;
  const uint64_t hi = sw ? b : a;
  const uint64_t lo = sw ? a : b;
  a = hi;
  b = lo;
}

// Bitonic sort of 16 keys into descending order.
__device__ __forceinline__ void sort16_desc(uint64_t (&v)[16]) {
#pragma unroll
  for (int kk = 2; kk <= 16; kk <<= 1)
#pragma unroll
    for (int j = kk >> 1; j > 0; j >>= 1)
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int l = i ^ j;
        if (l > i) {
          if ((i & kk) == 0)
            cas_desc(v[i], v[l]);
          else
            cas_desc(v[l], v[i]);
        }
      }
}

// top <- the 16 largest of top and c, both sorted descending (c is clobbered): the elementwise
// max of top and reversed c is a bitonic sequence holding them, then a bitonic merge sorts it.
__device__ __forceinline__ void merge16_desc(uint64_t (&top)[16], const uint64_t (&c)[16]) {
#pragma unroll
  for (int i = 0; i < 16; ++i) top[i] = top[i] > c[15 - i] ? top[i] : c[15 - i];
#pragma unroll
  for (int j = 8; j > 0; j >>= 1)
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int l = i ^ j;
      if (l > i) cas_desc(top[i], top[l]);
    }
}

// 64-bit key ordering (z descending, expert ascending).  An empty slot is key 0, below every
// real key.
__device__ __forceinline__ uint64_t topk_key(float z, int e) {
  const uint32_t u = __float_as_uint(z);
  const uint32_t ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return (static_cast<uint64_t>(ord) << 32) | static_cast<uint32_t>(~static_cast<uint32_t>(e));
}
__device__ __forceinline__ float key_z(uint64_t key) {
  const uint32_t ord = static_cast<uint32_t>(key >> 32);
  return __uint_as_float((ord & 0x80000000u) ? (ord & 0x7fffffffu) : ~ord);
}
__device__ __forceinline__ int key_e(uint64_t key) {
  return static_cast<int>(~static_cast<uint32_t>(key));
}

// Write a finished predict row: idx and gates of the k best keys (divided by their sum under
// PR2_F_NORMALIZE_TOPK); returns the near-tie flag rho_hat_(k) - rho_hat_(k+1) <
// PR2_NEAR_TIE_GAP, always on the unnormalised probabilities.
__device__ __forceinline__ bool predict_write(const uint64_t (&key)[16], float mx, float inv_s,
                                              int64_t t, const RouteTcArgs& a) {
  int32_t* irow = a.idx_out + t * a.k;
  float* grow = a.gates + t * a.k;
  float pr[kKeep];
  float sk = 0.f;
#pragma unroll
  for (int j = 0; j < kKeep; ++j) {
    pr[j] = expf(key_z(key[j]) - mx) * inv_s;
    if (j < a.k) sk += pr[j];
  }
  const float sc = a.norm ? 1.0f / sk : 1.0f;
  float pk = 0.f, pk1 = 0.f;
#pragma unroll
  for (int j = 0; j < kKeep; ++j) {
    if (j < a.k) {
      irow[j] = key_e(key[j]);
      grow[j] = pr[j] * sc;
    }
    if (j == a.k - 1) pk = pr[j];
    if (j == a.k) pk1 = pr[j];
  }
  return (a.k < a.N) && (pk - pk1 < (float)PR2_NEAR_TIE_GAP);
}

template <int kMode, int split>
__global__ void __launch_bounds__(kThreads, 1)
    route_tc_kernel(const __grid_constant__ CUtensorMap tm_h,
                    const __grid_constant__ CUtensorMap tm_w,
                    const __grid_constant__ CUtensorMap tm_wp, RouteTcArgs a) {
  constexpr bool predict = kMode == kModePredict;
  constexpr bool loss = kMode == kModeLoss;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  const int N = a.N, k = a.k;
  const RouteSmemLayout L = route_layout(N, predict, a.compact != 0);
  // 1024-B aligned base, kept as an offset into the shared array so the compiler knows every
  // derived pointer is shared memory.
  const uint32_t pad = (1024u - (smem_u32(smem_raw) & 1023u)) & 1023u;
  uint8_t* smem = smem_raw + pad;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bar_offset);
  uint64_t* empty = full + L.stages;
  uint64_t* acc_full = empty + L.stages;
  uint64_t* drain = acc_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const float4* recv = reinterpret_cast<const float4*>(smem);  // valid after the exchange

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int rank = split > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int t0 = (blockIdx.x / split) * kTileM;
  const int R = kTileM / split;             // rows finished by this CTA
  const int nr = N / split;                 // experts of one finishing thread
  const int nb4 = L.b_rows / 4;             // float4 columns of a partial row
  // Pass split: predict whose weights stream in two passes (N > 128) run by a 2-CTA cluster in
  // which CTA r streams pass r ([W], then [W_p]) over all of K; the two column halves of every
  // row then meet in the CTA that finishes it, through distributed shared memory, and are not
  // summed.  Otherwise the cluster splits K and the S partial rows are summed.
  const bool psplit = predict && L.passes == 2 && split == 2;
  const int KBper = psplit ? a.d / kBK : (a.d / kBK) / split;
  const int kb0 = psplit ? 0 : rank * KBper, kb1 = kb0 + KBper;
  const int npass = psplit ? 1 : L.passes;  // passes this CTA streams
  const int pass0 = psplit ? rank : 0;      // the first of them
  const int acc_cols = psplit ? L.pass_rows : L.b_rows;
  const uint32_t ncols = tmem_cols_for(acc_cols);

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
  // h, the weights and the cached route may come from the previous kernels.  With late_wait
  // the caller guarantees they are complete already (the kernel before is a grouped GEMM whose
  // own inputs came after them), so the CTAs start on the SMs that GEMM frees and wait for it
  // only before they exit: a kernel launched after this one then sees the GEMM's results too.
  if (!a.late_wait) pdl_wait();
  pdl_trigger();

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      const uint32_t bytes = static_cast<uint32_t>(L.stage_bytes);
      uint32_t issued = 0, last_par = 0;
      int stage = 0;
      uint32_t phase = 0;
      const uint64_t keep = l2_policy_evict_last();    // weights are re-read by every tile
      const uint64_t once = l2_policy_evict_first();   // h is read once
      bool ok = true;
      for (int pass = pass0; pass < pass0 + npass && ok; ++pass)
      for (int kb = kb0; kb < kb1; ++kb) {
        if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, a.status)) {
          ok = false;
          break;
        }
        uint8_t* sa = smem + stage * L.stage_bytes;
        uint8_t* sb = sa + kATileBytes;
        mbar_arrive_expect_tx(&full[stage], bytes);
        tma_load_2d_hint(sa, &tm_h, &full[stage], kb * kBK, t0, once);
        if (!predict || L.passes == 1) {  // replay never takes two passes
          tma_load_2d_hint(sb, &tm_w, &full[stage], kb * kBK, 0, keep);
          if (predict) tma_load_2d_hint(sb + N * kBK * 2, &tm_wp, &full[stage], kb * kBK, 0, keep);
        } else if (pass == 0) {
          // Each map is named directly: with one pointer selected between the two maps here,
          // even the replay kernel's mainloop (which never gets here) ran 25 % slower.
          tma_load_2d_hint(sb, &tm_w, &full[stage], kb * kBK, 0, keep);
        } else {
          tma_load_2d_hint(sb, &tm_wp, &full[stage], kb * kBK, 0, keep);
        }
        issued |= 1u << stage;
        last_par = (last_par & ~(1u << stage)) | (phase << stage);
        if (++stage == L.stages) {
          stage = 0;
          phase ^= 1u;
        }
      }
      // Drain: every issued copy must have landed before the stages are reused or the CTA exits.
      for (int s = 0; s < L.stages; ++s)
        if ((issued >> s) & 1u)
          mbar_wait_slow(&full[s], (last_par >> s) & 1u, nullptr, nullptr, kDrainLimitNs);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int pass = pass0; pass < pass0 + npass && ok; ++pass)
      for (int kb = kb0; kb < kb1 && ok; ++kb) {
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
          const uint32_t acc = (kb > kb0 || kk > 0) ? 1u : 0u;
          if (!predict || L.passes == 1) {  // replay never takes two passes
            for (int n0 = 0; n0 < L.b_rows; n0 += 256) {
              const int nc = (L.b_rows - n0) < 256 ? (L.b_rows - n0) : 256;
              const uint64_t bdesc = umma_desc_sw128(sb + n0 * (kBK * 2) + kk * 32);
              umma_bf16(tmem + n0, adesc, bdesc, umma_idesc_bf16(kTileM, nc), acc);
            }
          } else {  // pass p fills accumulator columns [p N, (p + 1) N): p_old, then b
            umma_bf16(tmem + (psplit ? 0 : pass * L.pass_rows), adesc,
                      umma_desc_sw128(sb + kk * 32), umma_idesc_bf16(kTileM, L.pass_rows), acc);
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
    }
    __syncwarp();
  }

  // ---------------- epilogue ----------------
  const bool epi = warp >= 2;
  // predict: experts of the rows this CTA finishes, for the dispatch that follows
  __shared__ int hist_s[kMaxExperts];
  const bool count = predict && a.hist != nullptr;
  if (count && epi) {
    for (int e = threadIdx.x - 64; e < N; e += 128) hist_s[e] = 0;
    named_bar_sync(1, 128);
  }
  const int q = warp & 3;
  const int row = q * 32 + lane;  // TMEM lane of this thread
  const uint32_t trow = tmem + (static_cast<uint32_t>(q * 32) << 16);
  // Finishing coordinates: row lr of this CTA's R rows, experts [part nr, (part+1) nr).
  const int et = threadIdx.x - 64;
  const int lr = split == 1 ? row : et / split;
  const int part = split == 1 ? 0 : et - lr * split;
  const int fe0 = part * nr;
  const int64_t t = static_cast<int64_t>(t0) + static_cast<int64_t>(rank) * R + lr;
  const bool live = epi && t < a.T;

  // replay: cached indices, validated (range, duplicates) while the K blocks run
  int e_s[kMaxTopK];
  bool bad = false;
  if (kMode == kModeReplay) {
#pragma unroll
    for (int s = 0; s < kMaxTopK; ++s) {
      int e = -1;
      if (live && s < k) {
        e = a.idx_in[t * k + s];
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
    }
  }

  // loss: the first kLossPre experts of this thread's segment of its p_old row and of its
  // teacher row (row pos[t] of rho), loaded while the K blocks run
  constexpr int kLossPre = loss ? 32 : 4;
  float po_s[kLossPre], tr_s[kLossPre];
  int64_t lrow = 0;
  bool okp = false;
  if (loss && live) {
    lrow = a.pos != nullptr ? static_cast<int64_t>(a.pos[t]) : t;
    okp = lrow >= 0 && lrow < a.T_rho;
    if (okp) {
      const float4* p4 = reinterpret_cast<const float4*>(a.p_old + t * N + fe0);
      const float4* r4 = reinterpret_cast<const float4*>(a.rho + lrow * N + fe0);
#pragma unroll
      for (int j = 0; j < kLossPre / 4; ++j) {
        if (4 * j < nr) {
          const float4 x = p4[j], y = r4[j];
          po_s[4 * j] = x.x;
          po_s[4 * j + 1] = x.y;
          po_s[4 * j + 2] = x.z;
          po_s[4 * j + 3] = x.w;
          tr_s[4 * j] = y.x;
          tr_s[4 * j + 1] = y.y;
          tr_s[4 * j + 2] = y.z;
          tr_s[4 * j + 3] = y.w;
        }
      }
    }
  }

  bool have = false;
  if (epi) {
    // tcgen05.ld is warp-collective: the whole warp reads TMEM or none of it does.
    have = __all_sync(0xffffffffu, mbar_wait(acc_full, 0, abort_flag, a.status));
    if (have) tc_fence_after();
  }
  if (split > 1) {
    cluster_sync();  // every CTA has finished its K blocks: the pipeline stages are free
    if (epi && have) {
      // Reduce-scatter by rows: this TMEM row goes to CTA row / R as its row row % R, into the
      // slot of source `rank` (K split) or into columns [rank N, (rank + 1) N) (pass split).
      float4* recv_w = reinterpret_cast<float4*>(smem);
      const uint32_t dst = static_cast<uint32_t>(row / R);
      const int drow = row - static_cast<int>(dst) * R;
      const int off4 = psplit ? L.pass_rows / 4 : nb4;
      const uint32_t rbase =
          mapa_shared(smem_u32(recv_w + (rank * off4) * R + drow), dst);
      for (int c0 = 0; c0 < acc_cols; c0 += 32) {
        uint32_t r0[16], r1[16];
        tmem_ld16(trow + c0, r0);
        tmem_ld16(trow + c0 + 16, r1);
        tmem_wait_ld(r0);
        reg_fence(r1);
#pragma unroll
        for (int j = 0; j < 4; ++j)
          st_cluster_v4(rbase + static_cast<uint32_t>(((c0 / 4 + j) * R) * 16), r0[4 * j],
                        r0[4 * j + 1], r0[4 * j + 2], r0[4 * j + 3]);
        if (c0 + 16 < acc_cols) {  // a multiple of 16, not always of 32
#pragma unroll
          for (int j = 0; j < 4; ++j)
            st_cluster_v4(rbase + static_cast<uint32_t>(((c0 / 4 + 4 + j) * R) * 16), r1[4 * j],
                          r1[4 * j + 1], r1[4 * j + 2], r1[4 * j + 3]);
        }
      }
    }
    cluster_sync();  // every partial row has landed
    if (epi && !psplit) {
      // Sum the S received copies of this CTA's rows once, in source order, into source 0's
      // slots: consecutive threads take consecutive 16-byte words (no bank conflicts), so the
      // finishing threads then read one value per column instead of S strided ones.
      float4* red = reinterpret_cast<float4*>(smem);
      const int n4 = nb4 * R;  // 16-byte words of one source
      for (int i = threadIdx.x - 64; i < n4; i += 128) {
        float4 v = red[i];
#pragma unroll
        for (int src = 1; src < split; ++src) {
          const float4 w = red[src * n4 + i];
          v.x += w.x;
          v.y += w.y;
          v.z += w.z;
          v.w += w.w;
        }
        red[i] = v;
      }
      named_bar_sync(1, 128);  // the four epilogue warps
    }
  }
  // Columns [c, c + 16) of the finished row: the summed partials (S > 1) or TMEM (S = 1).
  auto load16 = [&](int c, uint32_t (&r)[16]) {
    if (split == 1) {
      tmem_ld16(trow + c, r);
      tmem_wait_ld(r);
      return;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float4 v = recv[(c / 4 + j) * R + lr];
      r[4 * j] = __float_as_uint(v.x);
      r[4 * j + 1] = __float_as_uint(v.y);
      r[4 * j + 2] = __float_as_uint(v.z);
      r[4 * j + 3] = __float_as_uint(v.w);
    }
  };

  // One pass over this thread's experts, 16 at a time: running max m and sum of exp(z - m),
  // (predict) the top-16 keys, (replay) the z of the cached slots.
  if (epi && !loss) {
    bool tie = false;
    float m = -FLT_MAX, sum = 0.f;
    uint64_t top[16];
    float z_s[kMaxTopK];
#pragma unroll
    for (int j = 0; j < 16; ++j) top[j] = 0ull;
#pragma unroll
    for (int s = 0; s < kMaxTopK; ++s) z_s[s] = 0.f;
    if (have) {
      float* lrow = (predict && a.logits_or_probs != nullptr && live) ? a.logits_or_probs + t * N
                                                                      : nullptr;
      for (int c0 = fe0; c0 < fe0 + nr; c0 += 16) {
        float z[16];
        if (predict) {
          uint32_t rp[16], rb[16];
          load16(c0, rp);
          load16(N + c0, rb);
          if (lrow != nullptr) {
            float4* dst = reinterpret_cast<float4*>(lrow + c0);
#pragma unroll
            for (int j = 0; j < 4; ++j)
              dst[j] = make_float4(__uint_as_float(rp[4 * j]), __uint_as_float(rp[4 * j + 1]),
                                   __uint_as_float(rp[4 * j + 2]), __uint_as_float(rp[4 * j + 3]));
          }
#pragma unroll
          for (int j = 0; j < 16; ++j) z[j] = __uint_as_float(rp[j]) + __uint_as_float(rb[j]);
        } else {
          uint32_t rp[16];
          load16(c0, rp);
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            z[j] = __uint_as_float(rp[j]);
#pragma unroll
            for (int s = 0; s < kMaxTopK; ++s)
              if (e_s[s] == c0 + j) z_s[s] = z[j];
          }
        }
        float cm = z[0];
#pragma unroll
        for (int j = 1; j < 16; ++j) cm = fmaxf(cm, z[j]);
        const float nm = fmaxf(m, cm);
        float cs = 0.f;
#pragma unroll
        for (int j = 0; j < 16; ++j) cs += expf(z[j] - nm);
        sum = sum * expf(m - nm) + cs;
        m = nm;
        if (predict) {
          uint64_t ck[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) ck[j] = topk_key(z[j], c0 + j);
          sort16_desc(ck);
          merge16_desc(top, ck);
        }
      }
    }
    // Combine the S threads of the row (consecutive lanes): max, rescaled sum, merged lists.
    float mx = m;
#pragma unroll
    for (int o = 1; o < split; o <<= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float fs = have ? sum * expf(m - mx) : 0.f;
#pragma unroll
    for (int o = 1; o < split; o <<= 1) fs += __shfl_xor_sync(0xffffffffu, fs, o);
    const float inv_s = 1.0f / fs;
    if (predict) {
#pragma unroll
      for (int o = 1; o < split; o <<= 1) {
        uint64_t other[16];
#pragma unroll
        for (int j = 0; j < 16; ++j)
          other[j] = j < kKeep ? __shfl_xor_sync(0xffffffffu, top[j], o) : 0ull;
        merge16_desc(top, other);
      }
      if (have && live && part == 0) {
        tie = predict_write(top, mx, inv_s, t, a);
        if (count)
          for (int j = 0; j < k; ++j) atomicAdd(&hist_s[key_e(top[j])], 1);
      }
    } else if (!loss) {
      // Each valid slot's z is held by the one thread owning its expert; the others hold 0.
#pragma unroll
      for (int s = 0; s < kMaxTopK; ++s)
#pragma unroll
        for (int o = 1; o < split; o <<= 1) z_s[s] += __shfl_xor_sync(0xffffffffu, z_s[s], o);
      if (have && live && part == 0) {
        float* grow = a.gates + t * k;
        float gv[kMaxTopK];
        float sk = 0.f;
#pragma unroll
        for (int s = 0; s < kMaxTopK; ++s) {
          gv[s] = (s < k && e_s[s] >= 0) ? expf(z_s[s] - mx) * inv_s : 0.f;
          sk += gv[s];
        }
        const float sc = (a.norm && sk > 0.f) ? 1.0f / sk : 1.0f;  // over the valid slots
#pragma unroll
        for (int s = 0; s < kMaxTopK; ++s)
          if (s < k) grow[s] = gv[s] * sc;
        if (bad && a.status != nullptr) atomicOr(a.status, PR2_STATUS_BAD_INDEX);
      }
      if (have && a.logits_or_probs != nullptr) {
        float* prow = a.logits_or_probs + t * N;
        for (int c0 = fe0; c0 < fe0 + nr; c0 += 16) {
          uint32_t rp[16];
          load16(c0, rp);
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
    const unsigned ties = __ballot_sync(0xffffffffu, tie);
    if (lane == 0 && ties != 0u && a.near_tie != nullptr)
      atomicAdd(reinterpret_cast<unsigned long long*>(a.near_tie),
                static_cast<unsigned long long>(__popc(ties)));
    if (count) {  // every row of this CTA counted: publish its histogram row (zeros included)
      named_bar_sync(1, 128);
      int32_t* hrow = a.hist + static_cast<int64_t>(blockIdx.x) * N;
      for (int e = threadIdx.x - 64; e < N; e += 128) hrow[e] = hist_s[e];
    }
    tc_fence_before();
  }
  if (epi && loss) {
    // Predictive loss (Eq. pr2_loss, Algorithm 3) of cached row t over experts [fe0, fe0+nr):
    //   standard: prediction Softmax(v), v = p_old + b;  target rho (row pos[t] of the teacher)
    //   delta:    prediction Softmax(b);  target Softmax(u), u = log rho - p_old
    // KL_t = sum_j tgt_j (log tgt_j - log pred_j);  dKL_t/dv_j = pred_j - tgt_j, stored bf16
    // and transposed for the gradient GEMM.  Two passes: normalisers, then terms.  The first
    // kLossPre experts come from registers, any further ones from global memory.  Exponentials
    // and logarithms use the hardware approximations (__expf, __logf: a few ulp over the ranges
    // met here, far inside the loss's tolerance), which cut this phase from ~10 to ~4 us.
    const bool delta = a.delta != 0;
    if (live && !okp && part == 0 && a.status != nullptr) atomicOr(a.status, PR2_STATUS_BAD_INDEX);
    const bool use = have && okp;
    const float* po = a.p_old + (live ? t : 0) * N;
    const float* tr = a.rho + (okp ? lrow : 0) * N;
    auto row16 = [&](const float* src, int c, float (&v)[16]) {
      const float4* q = reinterpret_cast<const float4*>(src + c);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float4 x = q[j];
        v[4 * j] = x.x;
        v[4 * j + 1] = x.y;
        v[4 * j + 2] = x.z;
        v[4 * j + 3] = x.w;
      }
    };
    float m1 = -FLT_MAX, s1 = 0.f, m2 = -FLT_MAX, s2 = 0.f;
    auto normalisers = [&](const uint32_t (&rb)[16], const float (&pv)[16],
                           const float (&rv)[16]) {
      float v[16], u[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const float b = __uint_as_float(rb[j]);
        v[j] = delta ? b : pv[j] + b;
        u[j] = rv[j] > 0.f ? __logf(rv[j]) - pv[j] : -INFINITY;
      }
      float cm = v[0];
#pragma unroll
      for (int j = 1; j < 16; ++j) cm = fmaxf(cm, v[j]);
      float nm = fmaxf(m1, cm), cs = 0.f;
#pragma unroll
      for (int j = 0; j < 16; ++j) cs += __expf(v[j] - nm);
      s1 = s1 * __expf(m1 - nm) + cs;
      m1 = nm;
      if (delta) {
        cm = u[0];
#pragma unroll
        for (int j = 1; j < 16; ++j) cm = fmaxf(cm, u[j]);
        nm = fmaxf(m2, cm);
        cs = 0.f;
#pragma unroll
        for (int j = 0; j < 16; ++j) cs += __expf(u[j] - nm);
        s2 = s2 * __expf(m2 - nm) + cs;
        m2 = nm;
      }
    };
#pragma unroll
    for (int ch = 0; ch < kLossPre / 16; ++ch) {
      if (ch * 16 < nr) {
        uint32_t rb[16];
        load16(fe0 + ch * 16, rb);
        if (use) {
          float pv[16], rv[16];
#pragma unroll
          for (int j = 0; j < 16; ++j) {
            pv[j] = po_s[ch * 16 + j];
            rv[j] = tr_s[ch * 16 + j];
          }
          normalisers(rb, pv, rv);
        }
      }
    }
    for (int c0 = fe0 + kLossPre; c0 < fe0 + nr; c0 += 16) {
      uint32_t rb[16];
      load16(c0, rb);
      if (use) {
        float pv[16], rv[16];
        row16(po, c0, pv);
        row16(tr, c0, rv);
        normalisers(rb, pv, rv);
      }
    }
    float mx1 = m1, mx2 = m2;
#pragma unroll
    for (int o = 1; o < split; o <<= 1) {
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, o));
      mx2 = fmaxf(mx2, __shfl_xor_sync(0xffffffffu, mx2, o));
    }
    float f1 = s1 * __expf(m1 - mx1), f2 = s2 * __expf(m2 - mx2);
#pragma unroll
    for (int o = 1; o < split; o <<= 1) {
      f1 += __shfl_xor_sync(0xffffffffu, f1, o);
      f2 += __shfl_xor_sync(0xffffffffu, f2, o);
    }
    const float l1 = mx1 + __logf(f1), l2 = mx2 + __logf(f2);  // log normalisers
    float kl = 0.f;
    auto terms = [&](int c0, const uint32_t (&rb)[16], const float (&pv)[16],
                     const float (&rv)[16]) {
      float g[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) g[j] = 0.f;
      if (use) {
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          const float b = __uint_as_float(rb[j]);
          const float lp = (delta ? b : pv[j] + b) - l1;  // log prediction
          float tg, lt;
          if (delta) {
            lt = rv[j] > 0.f ? __logf(rv[j]) - pv[j] - l2 : -INFINITY;
            tg = rv[j] > 0.f ? __expf(lt) : 0.f;
          } else {
            tg = rv[j];
            lt = rv[j] > 0.f ? __logf(rv[j]) : 0.f;
          }
          if (tg > 0.f) kl += tg * (lt - lp);
          g[j] = __expf(lp) - tg;
        }
      }
#pragma unroll
      for (int j = 0; j < 16; ++j)
        a.gt[static_cast<int64_t>(c0 + j) * a.Tpad + t] =
            __bfloat16_as_ushort(__float2bfloat16_rn(g[j]));
    };
#pragma unroll
    for (int ch = 0; ch < kLossPre / 16; ++ch) {
      if (ch * 16 < nr) {
        uint32_t rb[16];
        load16(fe0 + ch * 16, rb);
        float pv[16], rv[16];
#pragma unroll
        for (int j = 0; j < 16; ++j) {
          pv[j] = use ? po_s[ch * 16 + j] : 0.f;
          rv[j] = use ? tr_s[ch * 16 + j] : 0.f;
        }
        terms(fe0 + ch * 16, rb, pv, rv);
      }
    }
    for (int c0 = fe0 + kLossPre; c0 < fe0 + nr; c0 += 16) {
      uint32_t rb[16];
      load16(c0, rb);
      float pv[16], rv[16];
      if (use) {
        row16(po, c0, pv);
        row16(tr, c0, rv);
      }
      terms(c0, rb, pv, rv);
    }
#pragma unroll
    for (int o = 1; o < split; o <<= 1) kl += __shfl_xor_sync(0xffffffffu, kl, o);
    if (live && part == 0) a.kl_tok[t] = use ? kl : 0.f;
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, ncols);
  }
  if (a.late_wait) pdl_wait();
}

template <int kMode, int kSplit>
cudaError_t set_smem_attr(int N) {
  const cudaError_t err = cudaFuncSetAttribute(route_tc_kernel<kMode, kSplit>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               route_layout(N, kMode == kModePredict, false).total);
  if (err != cudaSuccess) return err;
  // all of the SM's unified L1 / shared storage as shared memory, so that two compact CTAs fit
  return cudaFuncSetAttribute(route_tc_kernel<kMode, kSplit>,
                              cudaFuncAttributePreferredSharedMemoryCarveout,
                              cudaSharedmemCarveoutMaxShared);
}

template <int kMode, int kSplit>
cudaError_t launch_split(const CUtensorMap& tm_h, const CUtensorMap& tm_w,
                         const CUtensorMap& tm_wp, const RouteTcArgs& a, int tiles,
                         cudaStream_t st, int* max_clusters) {
  cudaError_t err = set_smem_attr<kMode, kSplit>(a.N);
  if (err != cudaSuccess) return err;
  const size_t smem = route_layout(a.N, kMode == kModePredict, a.compact != 0).total;
  if (max_clusters != nullptr) {  // occupancy query only
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(tiles * kSplit);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kSplit;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaOccupancyMaxActiveClusters(max_clusters, route_tc_kernel<kMode, kSplit>, &cfg);
  }
  return launch_pdl(route_tc_kernel<kMode, kSplit>, dim3(tiles * kSplit), dim3(kThreads), smem,
                    st, kSplit, tm_h, tm_w, tm_wp, a);
}

template <int kMode>
cudaError_t launch_splits(const CUtensorMap& tm_h, const CUtensorMap& tm_w,
                          const CUtensorMap& tm_wp, const RouteTcArgs& a, int split, int tiles,
                          cudaStream_t st, int* max_clusters) {
  switch (split) {
    case 1: return launch_split<kMode, 1>(tm_h, tm_w, tm_wp, a, tiles, st, max_clusters);
    case 2: return launch_split<kMode, 2>(tm_h, tm_w, tm_wp, a, tiles, st, max_clusters);
    case 4: return launch_split<kMode, 4>(tm_h, tm_w, tm_wp, a, tiles, st, max_clusters);
    case 8: return launch_split<kMode, 8>(tm_h, tm_w, tm_wp, a, tiles, st, max_clusters);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_any(int mode, const CUtensorMap& tm_h, const CUtensorMap& tm_w,
                       const CUtensorMap& tm_wp, const RouteTcArgs& a, int split, int tiles,
                       cudaStream_t st, int* max_clusters) {
  switch (mode) {
    case kModeReplay:
      return launch_splits<kModeReplay>(tm_h, tm_w, tm_wp, a, split, tiles, st, max_clusters);
    case kModePredict:
      return launch_splits<kModePredict>(tm_h, tm_w, tm_wp, a, split, tiles, st, max_clusters);
    case kModeLoss:
      return launch_splits<kModeLoss>(tm_h, tm_w, tm_wp, a, split, tiles, st, max_clusters);
    default: return cudaErrorInvalidValue;
  }
}

// CTAs of route_tc_kernel<mode, 1> with the compact layout that fit on one SM by its shared
// memory, registers, threads and TMEM columns (0 on error).  Counted from the kernel's attributes and the
// device limits: the occupancy query answers 1 for this kernel although two CTAs do run on
// one SM side by side (a per-CTA %smid / %globaltimer record of a T = 32768 launch).
template <int kMode>
int compact_blocks_per_sm(int N) {
  if (set_smem_attr<kMode, 1>(N) != cudaSuccess) return 0;
  cudaFuncAttributes fa{};
  if (cudaFuncGetAttributes(&fa, route_tc_kernel<kMode, 1>) != cudaSuccess) return 0;
  int dev = 0, smem_sm = 0, reserved = 0, regs_sm = 0, threads_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&smem_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&reserved, cudaDevAttrReservedSharedMemoryPerBlock, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&regs_sm, cudaDevAttrMaxRegistersPerMultiprocessor, dev) !=
          cudaSuccess ||
      cudaDeviceGetAttribute(&threads_sm, cudaDevAttrMaxThreadsPerMultiProcessor, dev) !=
          cudaSuccess)
    return 0;
  const size_t smem = route_layout(N, kMode == kModePredict, true).total + fa.sharedSizeBytes +
                      static_cast<size_t>(reserved);
  const int regs = ((fa.numRegs + 7) / 8) * 8 * kThreads;  // allocated per warp in 256s
  int n = static_cast<int>(static_cast<size_t>(smem_sm) / smem);
  if (regs > 0 && regs_sm / regs < n) n = regs_sm / regs;
  if (threads_sm / kThreads < n) n = threads_sm / kThreads;
  // each CTA holds its accumulator columns for its whole life: more CTAs than fit in the SM's
  // 512 TMEM columns would only wait in tcgen05.alloc for a neighbour to leave
  const int b_rows = route_layout(N, kMode == kModePredict, true).b_rows;
  const int by_tmem = static_cast<int>(512u / tmem_cols_for(b_rows));
  if (by_tmem < n) n = by_tmem;
  return n;
}

// Clusters of `split` CTAs of this kernel that can be resident at once (0 on error), cached
// per device and shape.
int max_active_clusters(int mode, int split, int N, bool compact = false) {
  struct Entry {
    int dev, mode, split, N, compact, clusters;
  };
  static std::mutex mu;
  static Entry cache[64];
  static int used = 0;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  std::lock_guard<std::mutex> lock(mu);
  for (int i = 0; i < used; ++i)
    if (cache[i].dev == dev && cache[i].mode == mode && cache[i].split == split &&
        cache[i].N == N && cache[i].compact == static_cast<int>(compact))
      return cache[i].clusters;
  int clusters = 0;
  if (compact) {  // clusters of one CTA: CTAs per SM, times the SMs
    const int per_sm = mode == kModePredict ? compact_blocks_per_sm<kModePredict>(N)
                                            : compact_blocks_per_sm<kModeReplay>(N);
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess)
      clusters = per_sm * sms;
    (void)cudaGetLastError();
  } else {
    RouteTcArgs probe{};
    probe.N = N;
    CUtensorMap none{};
    const cudaError_t err =
        launch_any(mode, none, none, none, probe, split, 1, nullptr, &clusters);
    if (err != cudaSuccess) {
      (void)cudaGetLastError();
      clusters = 0;
    }
  }
  if (used < 64) cache[used++] = Entry{dev, mode, split, N, static_cast<int>(compact), clusters};
  return clusters;
}

}  // namespace

bool route_compact(int T, int N, int mode, int num_sms) {
  const int tiles = (T + kTileM - 1) / kTileM;
  if (tiles <= num_sms) return false;
  const RouteSmemLayout L = route_layout(N, mode == kModePredict, true);
  if (L.stages * L.stage_bytes > kCompactBudget) return false;  // not even two stages fit
  if (2 * tmem_cols_for(L.b_rows) > 512) return false;           // two accumulators in TMEM
  return max_active_clusters(mode, 1, N, true) >= 2 * num_sms;
}

int route_split(int T, int N, int d, int mode, int num_sms) {
  const RouteSmemLayout L = route_layout(N, mode == kModePredict, false);
  const int tiles = (T + kTileM - 1) / kTileM;
  const int KB = d / kBK;
  if (L.passes == 2) {
    // predict with N > 128: the pass split (two CTAs per tile, each receiving its 64 rows' two
    // column halves) when it fits in one wave, else one CTA per tile streaming both passes
    const bool fits = route_recv_bytes(L.b_rows) / 2 <= L.stages * L.stage_bytes &&
                      KB % 2 == 0 && (N / 2) % 16 == 0 && tiles * 2 <= num_sms &&
                      max_active_clusters(mode, 2, N) >= tiles;
    return fits ? 2 : 1;
  }
  if (route_recv_bytes(L.b_rows) > L.stages * L.stage_bytes) return 1;
  for (int s = kMaxSplit; s > 1; s >>= 1) {
    if (N % s != 0 || (N / s) % 16 != 0 || KB % s != 0 || tiles * s > num_sms) continue;
    if (max_active_clusters(mode, s, N) < tiles) continue;  // must fit in one wave
    return s;
  }
  return 1;
}

cudaError_t launch_route_tc(int mode, const CUtensorMap& tm_h, const CUtensorMap& tm_w,
                            const CUtensorMap& tm_wp, const RouteTcArgs& a, int split,
                            cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  if (split < 1 || split > kMaxSplit || a.N % split != 0 || (a.N / split) % 16 != 0 ||
      (a.d / kBK) % split != 0 || (a.compact != 0 && split != 1))
    return cudaErrorInvalidValue;
  const int tiles = (a.T + kTileM - 1) / kTileM;
  return launch_any(mode, tm_h, tm_w, tm_wp, a, split, tiles, st, nullptr);
}

}  // namespace pr2
