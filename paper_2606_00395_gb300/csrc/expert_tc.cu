// Grouped expert GEMMs on the tcgen05 tensor cores (bf16 operands, fp32 accumulation in TMEM).
//
// The gated-MLP expert of App. E.2 with the SwiGLU activation, over the rows that dispatch
// grouped by expert:
//   gate/up GEMM:  H[r, :] = silu(X[r] Wg_e^T) * (X[r] Wu_e^T)     (K = d, 128 H columns / tile)
//   down GEMM:     Y[r, :] = H[r] Wd_e^T                           (K = m, 256 Y columns / tile)
// where X[r] = h[perm[r] / k] is the token that dispatch placed at row r.
//
// Persistent kernel: one CTA per SM walks the (M-tile, N-tile) list in M-major order, so the
// CTAs running at the same time share the weight tiles of the same few experts through L2.
// The A rows and the expert weight tiles (streamed from DRAM) travel in two separate rings of
// 128-byte-swizzled K-major tiles (A 4 x 16 KB, B 5 x 32 KB), each filled by its own producers,
// so the long-latency weight stream runs further ahead of the tensor core.  Warp roles (warp w runs on SM sub-partition w % 4):
//   warps 0-2, 4  A producers.  Gate/up GEMM of the routed experts: all 128 threads gather the
//              tile's rows straight from h with 16-byte cp.async (each thread owns 8 rows and
//              one 16-byte column chunk, written to its swizzled position), so neither a
//              permuted copy of h nor a gather launch exists; h (T x d) stays in L2.  Other
//              GEMMs: one thread of warp 0 issues TMA loads of the A tile.
//   warp 3     TMEM owner and tcgen05.mma issuer (M=128, N=256, K=16) into one of two
//              256-column fp32 accumulators.  It shares its sub-partition with one epilogue
//              warp only: next to a gather warp as well it issued late enough to cost the
//              gate/up GEMM 4 %.
//   warp 5     TMA producer of the weight ring.
//   warps 6-9  epilogue: drain the other accumulator (one thread per tile row) while the next
//              tile is being multiplied.
// Each tcgen05.commit costs the tensor pipe about 25 ns (a third of one MMA), so the MMA thread
// commits once per K block, to one release barrier shared by both rings (ReleaseCursor).
#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kThreads = 320;
constexpr int kWarpMma = 3;
constexpr int kWarpB = 5;
constexpr int kBK = 64;
constexpr int kBN = 256;
constexpr int kGatherThreads = 128;         // warps 0-2 and 4
constexpr int kATile = kTileM * kBK * 2;    // 16 KB
constexpr int kBTile = kBN * kBK * 2;       // 32 KB
constexpr int kAccCols = kBN;               // one accumulator
constexpr uint32_t kTmemCols = 2 * kAccCols;
constexpr int kRel = 8;                     // release barriers, one per K block mod 8

constexpr int kStagesA = 4;                 // 4 x 16 KB A ring + 5 x 32 KB weight ring = 224 KB
constexpr int kStagesB = 5;
constexpr int kBRing = kStagesA * kATile;   // offset of the weight ring
constexpr int kBarOffset = kBRing + kStagesB * kBTile;
constexpr int kSmemBytes = 1024 + kBarOffset + 256;
static_assert(kStagesA < kRel && kStagesB < kRel, "a ring of kRel stages could see a release twice");
static_assert((kStagesA + kStagesB + kRel + 5) * 8 + 8 <= 256, "barrier area");

// Stage release.  The MMA thread commits once per K block (each tcgen05.commit costs the tensor
// pipe ~25 ns, a third of an MMA), to rel[n % kRel] for the n-th K block.  A producer whose ring
// has S stages may refill the stage of K block n once K block n - S has completed, i.e. phase
// (n - S) / kRel of rel[(n - S) % kRel].  That barrier cannot be a phase further on: its next
// completion is K block n - S + kRel, whose data this producer has not issued yet (S < kRel).
template <int S>
struct ReleaseCursor {
  int n = 0;  // K blocks issued so far
  __device__ __forceinline__ bool wait(uint64_t* rel, volatile int* abort_flag, int32_t* status) {
    if (n < S) return true;
    const int j = n - S;
    return mbar_wait(&rel[j % kRel], static_cast<uint32_t>(j / kRel) & 1u, abort_flag, status);
  }
  __device__ __forceinline__ void advance() { ++n; }
};

// A producer of the gathered gate/up GEMM: thread `tid` of warps 0-2, 4 copies, for every K
// block, the 16-byte chunk `c = tid % 8` of tile rows r = tid / 8 + 16 i (i = 0..7).  In the
// 128-byte swizzled K-major tile, chunk c of row r sits at r * 128 + ((c ^ (r % 8)) * 16), and
// r % 8 is the same for all eight rows of a thread.  After its eight copies of a stage the thread
// registers an arrival on that stage's full barrier (count 128) that fires when they have
// landed; the MMA thread, after acquiring the barrier, fences the stage into the async proxy.
// A tile's rows are tokens perm[a_row0 + r] / k of h.  The next tile's table entry is loaded
// when a tile starts and its perm entries halfway through the tile, as raw values that are
// only turned into pointers when the next tile starts: no load result is waited for while the
// ring needs refilling.
__device__ __forceinline__ void gather_a_producer(const GemmArgs& g, uint8_t* smem,
                                                  uint64_t* full_a, uint64_t* rel_bar,
                                                  volatile int* abort_flag, int n_tiles_n,
                                                  int num_tiles, int KB) {
  const int tid = threadIdx.x < 96 ? threadIdx.x : threadIdx.x - 32;  // warps 0-2, 4
  const int c = tid & 7;
  const int r0 = tid >> 3;
  const uint32_t soff = static_cast<uint32_t>(r0 * 128 + ((c ^ (r0 & 7)) << 4));
  const __nv_bfloat16* h = static_cast<const __nv_bfloat16*>(g.a_src);
  const int64_t ld = g.K;
  const uint64_t keep = l2_policy_evict_last();  // h: every token row is read k times
  const int stride = static_cast<int>(gridDim.x);
  auto entry = [&](int tile) {
    return tile < num_tiles ? g.tiles[tile / n_tiles_n] : TileEntry{0, 0, 0, 0};
  };
  // perm entries of a tile's rows (padding rows: none, they are zero-filled)
  auto fetch = [&](const TileEntry& te, int32_t (&slot)[8], uint32_t& live) {
    live = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int row = r0 + 16 * i;
      const bool on = row < te.rows;
      slot[i] = on ? g.perm[te.a_row0 + row] : 0;
      live |= (on ? 1u : 0u) << i;
    }
  };
  int32_t slot[8], slot_next[8];
  uint32_t live = 0, live_next = 0;
  fetch(entry(blockIdx.x), slot, live);
  TileEntry te_next = entry(blockIdx.x + stride);
  const int kb_fetch = KB / 2;
  int stage = 0;
  ReleaseCursor<kStagesA> rc;
  bool ok = true;
  for (int tile = blockIdx.x; tile < num_tiles && ok; tile += stride) {
    const __nv_bfloat16* src[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) src[i] = h + static_cast<int64_t>(slot[i] / g.k) * ld + c * 8;
    const TileEntry te_after = entry(tile + 2 * stride);  // used by the next tile's fetch
    for (int kb = 0; kb < KB; ++kb) {
      if (!rc.wait(rel_bar, abort_flag, g.status)) {
        ok = false;
        break;
      }
      rc.advance();
      const uint32_t dst = smem_u32(smem + stage * kATile) + soff;
#pragma unroll
      for (int i = 0; i < 8; ++i)
        cp_async_16_hint(dst + i * 2048, src[i] + kb * kBK, ((live >> i) & 1u) * 16u, keep);
      cp_async_arrive_noinc(&full_a[stage]);
      if (++stage == kStagesA) stage = 0;
      if (kb == kb_fetch) fetch(te_next, slot_next, live_next);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) slot[i] = slot_next[i];
    live = live_next;
    te_next = te_after;
  }
  cp_async_commit();
  cp_async_wait<0>();  // nothing may still be writing shared memory when the CTA leaves
}

template <bool kSwiGLU, bool kGatherA>
__global__ void __launch_bounds__(kThreads, 1)
    expert_tc_kernel(const __grid_constant__ CUtensorMap tm_a,
                     const __grid_constant__ CUtensorMap tm_b0,
                     const __grid_constant__ CUtensorMap tm_b1, GemmArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full_a = reinterpret_cast<uint64_t*>(smem + kBarOffset);
  uint64_t* full_b = full_a + kStagesA;
  uint64_t* rel = full_b + kStagesB;         // [kRel]
  uint64_t* acc_full = rel + kRel;           // [2]
  uint64_t* acc_empty = acc_full + 2;    // [2]
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  constexpr int kColsPerTile = kSwiGLU ? kBN / 2 : kBN;  // output columns per N-tile
  const int n_tiles_n = (g.n_out + kColsPerTile - 1) / kColsPerTile;
  const int KB = g.K / kBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesA; ++s) mbar_init(&full_a[s], kGatherA ? kGatherThreads : 1);
    for (int s = 0; s < kStagesB; ++s) mbar_init(&full_b[s], 1);
    for (int s = 0; s < kRel; ++s) mbar_init(&rel[s], 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);  // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    if (!kGatherA) tma_prefetch_desc(&tm_a);
    tma_prefetch_desc(&tm_b0);
    if (kSwiGLU) tma_prefetch_desc(&tm_b1);
  }
  if (warp == kWarpMma) {
    tmem_alloc(tmem_slot, kTmemCols);
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();  // the tile table and the A operand come from the previous kernels
  pdl_trigger();
  const int num_tiles = (*g.num_tiles) * n_tiles_n;

  if (kGatherA && (warp < 3 || warp == 4)) {
    gather_a_producer(g, smem, full_a, rel, abort_flag, n_tiles_n, num_tiles, KB);
  } else if ((warp == 0 || warp == kWarpB) && lane == 0) {
    // ---------------- TMA producers: warp 0 the A ring, warp 5 the B ring ----------------
    const bool is_a = warp == 0;
    const int nst = is_a ? kStagesA : kStagesB;
    uint64_t* fullr = is_a ? full_a : full_b;
    uint32_t issued = 0, last_par = 0;
    int stage = 0;
    uint32_t phase = 0;
    ReleaseCursor<kStagesA> rca;
    ReleaseCursor<kStagesB> rcb;
    // Expert weights are reused only by the M-tiles of their expert, which run at about the
    // same time, so they take the normal L2 policy (an evict_last hint on them pushes out h,
    // H and Y, which later tiles and kernels read again).
    bool ok = true;
    // the next tile's entry is loaded while this tile streams
    TileEntry te_next = g.tiles[blockIdx.x / n_tiles_n];
    for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
      const int mt = tile / n_tiles_n;
      const int nt = tile - mt * n_tiles_n;
      const TileEntry te = te_next;
      const int nxt = tile + static_cast<int>(gridDim.x);
      if (nxt < num_tiles) te_next = g.tiles[nxt / n_tiles_n];
      const int brow = te.expert * g.b_rows_per_expert + nt * kColsPerTile;
      for (int kb = 0; kb < KB; ++kb) {
        const bool free = is_a ? rca.wait(rel, abort_flag, g.status)
                               : rcb.wait(rel, abort_flag, g.status);
        if (!free) {
          ok = false;
          break;
        }
        rca.advance();
        rcb.advance();
        if (is_a) {
          uint8_t* sa = smem + stage * kATile;
          mbar_arrive_expect_tx(&fullr[stage], kATile);
          tma_load_2d(sa, &tm_a, &fullr[stage], kb * kBK, te.a_row0);
        } else {
          uint8_t* sb = smem + kBRing + stage * kBTile;
          mbar_arrive_expect_tx(&fullr[stage], kBTile);
          tma_load_2d(sb, &tm_b0, &fullr[stage], kb * kBK, brow);
          if (kSwiGLU) tma_load_2d(sb + kBTile / 2, &tm_b1, &fullr[stage], kb * kBK, brow);
        }
        issued |= 1u << stage;
        last_par = (last_par & ~(1u << stage)) | (phase << stage);
        if (++stage == nst) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    for (int s = 0; s < nst; ++s)
      if ((issued >> s) & 1u)
        mbar_wait_slow(&fullr[s], (last_par >> s) & 1u, nullptr, nullptr, kDrainLimitNs);
  } else if (warp == kWarpMma && lane == 0) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t idesc = umma_idesc_bf16(kTileM, kBN);
    int sa_i = 0, sb_i = 0;
    uint32_t pha = 0, phb = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    int kn = 0;  // K blocks issued: K block kn releases through rel[kn % kRel]
    bool ok = true;
    for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
      if (!mbar_wait(&acc_empty[acc], acc_phase ^ 1u, abort_flag, g.status)) break;
      tc_fence_after();
      const uint32_t d_tmem = tmem + acc * kAccCols;
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(&full_a[sa_i], pha, abort_flag, g.status) ||
            !mbar_wait(&full_b[sb_i], phb, abort_flag, g.status)) {
          ok = false;
          break;
        }
        if (kGatherA) fence_proxy_async_smem();  // rows written by cp.async (generic proxy)
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + sa_i * kATile);
        const uint32_t sb = smem_u32(smem + kBRing + sb_i * kBTile);
#pragma unroll
        for (int kk = 0; kk < kBK / 16; ++kk)
          umma_bf16(d_tmem, umma_desc_sw128(sa + kk * 32), umma_desc_sw128(sb + kk * 32), idesc,
                    (kb > 0 || kk > 0) ? 1u : 0u);
        umma_commit(&rel[kn % kRel]);  // frees this K block's A and weight stages
        ++kn;
        if (++sa_i == kStagesA) {
          sa_i = 0;
          pha ^= 1u;
        }
        if (++sb_i == kStagesB) {
          sb_i = 0;
          phb ^= 1u;
        }
      }
      if (!ok) break;
      umma_commit(&acc_full[acc]);
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
    umma_commit(drain);
    mbar_wait_slow(drain, 0, nullptr, nullptr, kDrainLimitNs);
  } else if (warp >= 6) {
    // ---------------- epilogue (warp w reads TMEM lanes 32 (w % 4) .. +31) ----------------
    const int q = warp & 3;
    const int row = q * 32 + lane;
    int acc = 0;
    uint32_t acc_phase = 0;
    __nv_bfloat16* out = static_cast<__nv_bfloat16*>(g.out);
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x) {
      const int mt = tile / n_tiles_n;
      const int nt = tile - mt * n_tiles_n;
      const TileEntry te = g.tiles[mt];
      if (!mbar_wait(&acc_full[acc], acc_phase, abort_flag, g.status)) break;
      tc_fence_after();
      const bool live = row < te.rows;
      __nv_bfloat16* orow = out + static_cast<int64_t>(te.out_row0 + row) * g.n_out;
      const uint32_t tacc = tmem + acc * kAccCols + (static_cast<uint32_t>(q * 32) << 16);
      if (kSwiGLU) {
#pragma unroll 1
        for (int c0 = 0; c0 < kBN / 2; c0 += 16) {
          uint32_t rg[16], ru[16];
          tmem_ld16(tacc + c0, rg);
          tmem_ld16(tacc + kBN / 2 + c0, ru);
          tmem_wait_ld(rg);
          reg_fence(ru);
          const int col = nt * (kBN / 2) + c0;
          if (live && col < g.n_out) {
            uint32_t pk[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float g0 = __uint_as_float(rg[2 * j]), g1 = __uint_as_float(rg[2 * j + 1]);
              const float u0 = __uint_as_float(ru[2 * j]), u1 = __uint_as_float(ru[2 * j + 1]);
              const float h0 = __fdividef(g0, 1.0f + __expf(-g0)) * u0;
              const float h1 = __fdividef(g1, 1.0f + __expf(-g1)) * u1;
              pk[j] = pack_bf16x2(h0, h1);
            }
            st_global_v8(orow + col, pk);  // 16 columns = one 32-byte sector
          }
        }
      } else {
#pragma unroll 1
        for (int c0 = 0; c0 < kBN; c0 += 16) {
          uint32_t rv[16];
          tmem_ld16(tacc + c0, rv);
          tmem_wait_ld(rv);
          const int col = nt * kBN + c0;
          if (live && col < g.n_out) {
            uint32_t pk[8];
#pragma unroll
            for (int j = 0; j < 8; ++j)
              pk[j] = pack_bf16x2(__uint_as_float(rv[2 * j]), __uint_as_float(rv[2 * j + 1]));
            st_global_v8(orow + col, pk);  // 16 columns = one 32-byte sector
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[acc]);
      if (++acc == 2) {
        acc = 0;
        acc_phase ^= 1u;
      }
    }
  }
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace

cudaError_t launch_expert_tc(bool swiglu, bool gather_a, const CUtensorMap& tm_a,
                             const CUtensorMap& tm_b0, const CUtensorMap& tm_b1,
                             const GemmArgs& g, int num_sms, cudaStream_t st) {
  if (g.max_tiles <= 0) return cudaSuccess;
  if (gather_a && (!swiglu || g.a_src == nullptr || g.perm == nullptr || g.k <= 0))
    return cudaErrorInvalidValue;
  const int cols = swiglu ? kBN / 2 : kBN;
  const int64_t bound = static_cast<int64_t>(g.max_tiles) * ((g.n_out + cols - 1) / cols);
  const int grid = static_cast<int>(bound < num_sms ? bound : num_sms);
  auto* kernel = gather_a ? expert_tc_kernel<true, true>
                          : (swiglu ? expert_tc_kernel<true, false> : expert_tc_kernel<false, false>);
  const cudaError_t err =
      cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (err != cudaSuccess) return err;
  return launch_pdl(kernel, dim3(grid), dim3(kThreads), kSmemBytes, st, 1, tm_a, tm_b0, tm_b1, g);
}

}  // namespace pr2
