// Grouped expert GEMMs on the tcgen05 tensor cores (bf16 operands, fp32 accumulation in TMEM).
//
// The gated-MLP expert of App. E.2 with the SwiGLU activation, over the rows that dispatch
// grouped by expert:
//   phase 0, gate/up:  H[r, :] = silu(X[r] Wg_e^T) * (X[r] Wu_e^T)   (K = d, 128 H columns / tile)
//   phase 1, down:     Y[r, :] = H[r] Wd_e^T                         (K = m, 256 Y columns / tile)
// where X[r] = h[perm[r] / k] is the token that dispatch placed at row r.
//
// Persistent kernel: one CTA per SM walks a list of jobs (M-tile, N-tile, phase) in M-major
// order, so the CTAs running at the same time share the weight tiles of the same few experts
// through L2.  The routed experts run both phases in one cooperative launch, every gate/up job
// before every down job, so an SM that has run out of gate/up jobs starts on down jobs instead
// of idling until the last gate/up job of the launch ends.  A down job waits until the gate/up
// epilogues of its M-tile have counted themselves done (an acquire on a per-M-tile counter;
// every CTA takes its jobs in increasing order and a down job only waits on gate/up jobs earlier
// in the list, so the waits always end).  Interleaving groups of M-tiles instead (so that down
// jobs find H in L2) measured slower: the two phases then compete and down jobs wait.  A rows and expert weight tiles travel in two separate rings of 128-byte-
// swizzled K-major tiles (A 4 x 16 KB, B 5 x 32 KB), each filled by its own producers, so the
// long-latency weight stream runs further ahead of the tensor core.  Warp roles (warp w runs on
// SM sub-partition w % 4):
//   warps 0-2, 4  A producers (128 threads).  Gathered rows: every thread copies 8 rows x one
//              16-byte column chunk straight from h with cp.async, written to its swizzled
//              position, so neither a permuted copy of h nor a gather launch exists; h (T x d)
//              stays in L2.  TMA rows: thread 0 issues the copy, the others only arrive.
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

struct Job {
  int phase;  // 0: gate/up + SwiGLU, 1: down
  int mt;     // M-tile (entry of the tile table)
  int nt;     // N-tile
};

// Job f of a launch, M-major (n N-tiles per M-tile).  Non-fused kinds: their single phase.
// Fused: every gate/up job (n1 per M-tile) first, then every down job (n2 per M-tile).
__device__ __forceinline__ Job job_of(int f, int kind, int nm, int n1, int n2) {
  if (kind != kExpertFused) {
    const int ph = kind == kExpertDown ? 1 : 0;
    const int n = ph ? n2 : n1;
    return Job{ph, f / n, f % n};
  }
  if (f < nm * n1) return Job{0, f / n1, f % n1};
  f -= nm * n1;
  return Job{1, f / n2, f % n2};
}

struct Launch {
  int kind, nm, n1, n2, num_jobs, kb0, kb1;  // kb0 / kb1: K blocks of a phase-0 / 1 job
  __device__ __forceinline__ Job job(int f) const { return job_of(f, kind, nm, n1, n2); }
  __device__ __forceinline__ bool gathered(const Job& j) const {
    return j.phase == 0 && kind != kExpertGateUpTma;
  }
};

// A producer (warps 0-2, 4; 128 threads; each full_a stage completes on 128 arrivals).
// Gathered rows: thread `tid` copies, for every K block, the 16-byte chunk `c = tid % 8` of tile
// rows r = tid / 8 + 16 i (i = 0..7).  In the 128-byte swizzled K-major tile, chunk c of row r
// sits at r * 128 + ((c ^ (r % 8)) * 16), and r % 8 is the same for all eight rows of a
// thread.  After its eight copies of a stage the thread registers an arrival that fires when
// they have landed; the MMA thread, after acquiring the barrier, fences the stage into the async
// proxy.  A tile's rows are tokens perm[a_row0 + r] / k of h: the next job's table entry is
// loaded when a job starts and its perm entries halfway through the job, as raw values turned
// into pointers only when that job starts, so no load result is waited for while the ring needs
// refilling.  TMA rows: thread 0 issues one 128-row box per K block (after, for a fused down
// job, the M-tile's gate/up epilogues have all finished); the other threads only arrive.
__device__ __forceinline__ void a_producer(const MlpArgs& ma, const GemmArgs& gs, const Launch& L,
                                           const CUtensorMap* tm_a, uint8_t* smem,
                                           uint64_t* full_a, uint64_t* rel_bar,
                                           volatile int* abort_flag) {
  const GemmArgs& g0 = ma.p[0];  // gathered rows (a_src, perm, k, K) belong to phase 0
  int32_t* status = gs.status;
  const int tid = threadIdx.x < 96 ? threadIdx.x : threadIdx.x - 32;  // warps 0-2, 4
  const int c = tid & 7;
  const int r0 = tid >> 3;
  const uint32_t soff = static_cast<uint32_t>(r0 * 128 + ((c ^ (r0 & 7)) << 4));
  const __nv_bfloat16* h = static_cast<const __nv_bfloat16*>(g0.a_src);
  const int64_t ld = g0.K;
  const uint64_t keep = l2_policy_evict_last();  // h: every token row is read k times
  const int stride = static_cast<int>(gridDim.x);
  const int ready_need = 4 * L.n1;  // four epilogue warps per gate/up N-tile
  auto entry = [&](int f) {
    return f < L.num_jobs ? gs.tiles[L.job(f).mt] : TileEntry{0, 0, 0, 0};
  };
  // perm entries of a tile's rows (padding rows: none, they are zero-filled)
  auto fetch = [&](const TileEntry& te, int32_t (&slot)[8], uint32_t& live) {
    live = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int row = r0 + 16 * i;
      const bool on = row < te.rows;
      slot[i] = on ? g0.perm[te.a_row0 + row] : 0;
      live |= (on ? 1u : 0u) << i;
    }
  };
  int32_t slot[8], slot_next[8];
  uint32_t live = 0, live_next = 0;
  int f = blockIdx.x;
  TileEntry te = entry(f);
  if (f < L.num_jobs && L.gathered(L.job(f))) fetch(te, slot, live);
  TileEntry te_next = entry(f + stride);
  int stage = 0;
  ReleaseCursor<kStagesA> rc;
  bool ok = true;
  for (; f < L.num_jobs && ok; f += stride) {
    const Job job = L.job(f);
    const bool gat = L.gathered(job);
    const int nxt = f + stride;
    const bool next_gat = nxt < L.num_jobs && L.gathered(L.job(nxt));
    const TileEntry te_after = entry(f + 2 * stride);  // used by the next job's fetch
    const __nv_bfloat16* src[8];
    if (gat) {
#pragma unroll
      for (int i = 0; i < 8; ++i) src[i] = h + static_cast<int64_t>(slot[i] / g0.k) * ld + c * 8;
    }
    if (!gat && tid == 0 && L.kind == kExpertFused) {
      // H rows of this M-tile: written by other CTAs' gate/up epilogues
      const int* cnt = ma.ready + job.mt;
      const uint64_t t0 = globaltimer_ns();
      while (ld_acquire_gpu(cnt) < ready_need) {
        if (*abort_flag || globaltimer_ns() - t0 > kWaitLimitNs) {
          *abort_flag = 1;
          if (status != nullptr) atomicOr(status, PR2_STATUS_TIMEOUT);
          ok = false;
          break;
        }
        __nanosleep(64);
      }
      fence_proxy_async_global();
    }
    const int KB = job.phase ? L.kb1 : L.kb0;
    const int kb_fetch = KB / 2;
    for (int kb = 0; kb < KB && ok; ++kb) {
      if (!rc.wait(rel_bar, abort_flag, status)) {
        ok = false;
        break;
      }
      rc.advance();
      if (gat) {
        const uint32_t dst = smem_u32(smem + stage * kATile) + soff;
#pragma unroll
        for (int i = 0; i < 8; ++i)
          cp_async_16_hint(dst + i * 2048, src[i] + kb * kBK, ((live >> i) & 1u) * 16u, keep);
        cp_async_arrive_noinc(&full_a[stage]);
      } else if (tid == 0) {
        mbar_arrive_expect_tx(&full_a[stage], kATile);
        tma_load_2d(smem + stage * kATile, tm_a, &full_a[stage], kb * kBK, te.a_row0);
      } else {
        mbar_arrive(&full_a[stage]);
      }
      if (++stage == kStagesA) stage = 0;
      if (kb == kb_fetch && next_gat) fetch(te_next, slot_next, live_next);
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) slot[i] = slot_next[i];
    live = live_next;
    te = te_next;
    te_next = te_after;
  }
  cp_async_commit();
  cp_async_wait<0>();  // nothing may still be writing shared memory when the CTA leaves
  // TMA copies of thread 0 land on full barriers that the MMA thread waits for before the CTA
  // leaves (it drains every issued K block), so they need no drain here.
}

template <int kKind>
__global__ void __launch_bounds__(kThreads, 1)
    expert_tc_kernel(const __grid_constant__ CUtensorMap tm_a,
                     const __grid_constant__ CUtensorMap tm_b0,
                     const __grid_constant__ CUtensorMap tm_b1,
                     const __grid_constant__ CUtensorMap tm_b2, MlpArgs ma) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* full_a = reinterpret_cast<uint64_t*>(smem + kBarOffset);
  uint64_t* full_b = full_a + kStagesA;
  uint64_t* rel = full_b + kStagesB;         // [kRel]
  uint64_t* acc_full = rel + kRel;           // [2]
  uint64_t* acc_empty = acc_full + 2;        // [2]
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  constexpr bool kHas0 = kKind != kExpertDown;                                   // gate/up jobs
  constexpr bool kHas1 = kKind == kExpertDown || kKind == kExpertFused;          // down jobs
  const GemmArgs& g0 = ma.p[0];
  const GemmArgs& g1 = ma.p[1];
  const GemmArgs& gs = kHas0 ? g0 : g1;  // tile table, count and status word
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStagesA; ++s) mbar_init(&full_a[s], kGatherThreads);
    for (int s = 0; s < kStagesB; ++s) mbar_init(&full_b[s], 1);
    for (int s = 0; s < kRel; ++s) mbar_init(&rel[s], 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);  // one arrival per epilogue warp
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    tma_prefetch_desc(&tm_a);
    if (kHas0) {
      tma_prefetch_desc(&tm_b0);
      tma_prefetch_desc(&tm_b1);
    }
    if (kHas1) tma_prefetch_desc(&tm_b2);
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
  __shared__ int nm_s;
  if (threadIdx.x == 0) {
    const int nm = status_timed_out(gs.status) ? 0 : *gs.num_tiles;
    nm_s = nm < 0 ? 0 : (nm > gs.max_tiles ? gs.max_tiles : nm);
  }
  __syncthreads();
  Launch L;
  L.kind = kKind;
  L.nm = nm_s;  // dispatch's count, never above the host bound; 0 after a timeout
  L.n1 = kHas0 ? (g0.n_out + kBN / 2 - 1) / (kBN / 2) : 0;
  L.n2 = kHas1 ? (g1.n_out + kBN - 1) / kBN : 0;
  L.num_jobs = L.nm * (L.n1 + L.n2);
  L.kb0 = kHas0 ? g0.K / kBK : 0;
  L.kb1 = kHas1 ? g1.K / kBK : 0;

  if (warp < 3 || warp == 4) {
    a_producer(ma, gs, L, &tm_a, smem, full_a, rel, abort_flag);
  } else if (warp == kWarpB && lane == 0) {
    // ---------------- TMA producer of the weight ring ----------------
    // Expert weights are reused only by the M-tiles of their expert, which run at about the
    // same time, so they take the normal L2 policy (an evict_last hint on them pushes out h,
    // H and Y, which later tiles and kernels read again).
    uint32_t issued = 0, last_par = 0;
    int stage = 0;
    uint32_t phase = 0;
    ReleaseCursor<kStagesB> rcb;
    bool ok = true;
    const int stride = static_cast<int>(gridDim.x);
    // the next job's entry is loaded while this job streams
    Job jn = L.job(blockIdx.x < L.num_jobs ? blockIdx.x : 0);
    TileEntry te_next = gs.tiles[jn.mt];
    for (int f = blockIdx.x; f < L.num_jobs && ok; f += stride) {
      const Job job = jn;
      const TileEntry te = te_next;
      if (f + stride < L.num_jobs) {
        jn = L.job(f + stride);
        te_next = gs.tiles[jn.mt];
      }
      const int brow = job.phase == 0 ? te.expert * g0.b_rows_per_expert + job.nt * (kBN / 2)
                                      : te.expert * g1.b_rows_per_expert + job.nt * kBN;
      const int KB = job.phase ? L.kb1 : L.kb0;
      for (int kb = 0; kb < KB; ++kb) {
        if (!rcb.wait(rel, abort_flag, gs.status)) {
          ok = false;
          break;
        }
        rcb.advance();
        uint8_t* sb = smem + kBRing + stage * kBTile;
        mbar_arrive_expect_tx(&full_b[stage], kBTile);
        if (job.phase == 0) {
          tma_load_2d(sb, &tm_b0, &full_b[stage], kb * kBK, brow);
          tma_load_2d(sb + kBTile / 2, &tm_b1, &full_b[stage], kb * kBK, brow);
        } else {
          tma_load_2d(sb, &tm_b2, &full_b[stage], kb * kBK, brow);
        }
        issued |= 1u << stage;
        last_par = (last_par & ~(1u << stage)) | (phase << stage);
        if (++stage == kStagesB) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    for (int s = 0; s < kStagesB; ++s)
      if ((issued >> s) & 1u)
        mbar_wait_slow(&full_b[s], (last_par >> s) & 1u, nullptr, nullptr, kDrainLimitNs);
  } else if (warp == kWarpMma && lane == 0) {
    // ---------------- MMA issuer ----------------
    constexpr uint32_t idesc = umma_idesc_bf16(kTileM, kBN);
    int sa_i = 0, sb_i = 0;
    uint32_t pha = 0, phb = 0;
    int acc = 0;
    uint32_t acc_phase = 0;
    int kn = 0;  // K blocks issued: K block kn releases through rel[kn % kRel]
    bool ok = true;
    for (int f = blockIdx.x; f < L.num_jobs && ok; f += gridDim.x) {
      const Job job = L.job(f);
      const bool gat = L.gathered(job);
      const int KB = job.phase ? L.kb1 : L.kb0;
      if (!mbar_wait(&acc_empty[acc], acc_phase ^ 1u, abort_flag, gs.status)) break;
      tc_fence_after();
      const uint32_t d_tmem = tmem + acc * kAccCols;
      for (int kb = 0; kb < KB; ++kb) {
        if (!mbar_wait(&full_a[sa_i], pha, abort_flag, gs.status) ||
            !mbar_wait(&full_b[sb_i], phb, abort_flag, gs.status)) {
          ok = false;
          break;
        }
        if (gat) fence_proxy_async_smem();  // rows written by cp.async (generic proxy)
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
    for (int f = blockIdx.x; f < L.num_jobs; f += gridDim.x) {
      const Job job = L.job(f);
      const TileEntry te = gs.tiles[job.mt];
      if (!mbar_wait(&acc_full[acc], acc_phase, abort_flag, gs.status)) break;
      tc_fence_after();
      const bool live = row < te.rows;
      const uint32_t tacc = tmem + acc * kAccCols + (static_cast<uint32_t>(q * 32) << 16);
      if (job.phase == 0) {
        __nv_bfloat16* orow =
            static_cast<__nv_bfloat16*>(g0.out) + static_cast<int64_t>(te.out_row0 + row) * g0.n_out;
#pragma unroll 1
        for (int c0 = 0; c0 < kBN / 2; c0 += 16) {
          uint32_t rg[16], ru[16];
          tmem_ld16(tacc + c0, rg);
          tmem_ld16(tacc + kBN / 2 + c0, ru);
          tmem_wait_ld(rg);
          reg_fence(ru);
          const int col = job.nt * (kBN / 2) + c0;
          if (live && col < g0.n_out) {
            uint32_t pk[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) {
              const float a0 = __uint_as_float(rg[2 * j]), a1 = __uint_as_float(rg[2 * j + 1]);
              const float u0 = __uint_as_float(ru[2 * j]), u1 = __uint_as_float(ru[2 * j + 1]);
              const float h0 = __fdividef(a0, 1.0f + __expf(-a0)) * u0;
              const float h1 = __fdividef(a1, 1.0f + __expf(-a1)) * u1;
              pk[j] = pack_bf16x2(h0, h1);
            }
            st_global_v8(orow + col, pk);  // 16 columns = one 32-byte sector
          }
        }
      } else {
        __nv_bfloat16* orow =
            static_cast<__nv_bfloat16*>(g1.out) + static_cast<int64_t>(te.out_row0 + row) * g1.n_out;
#pragma unroll 1
        for (int c0 = 0; c0 < kBN; c0 += 16) {
          uint32_t rv[16];
          tmem_ld16(tacc + c0, rv);
          tmem_wait_ld(rv);
          const int col = job.nt * kBN + c0;
          if (live && col < g1.n_out) {
            uint32_t pk[8];
#pragma unroll
            for (int j = 0; j < 8; ++j)
              pk[j] = pack_bf16x2(__uint_as_float(rv[2 * j]), __uint_as_float(rv[2 * j + 1]));
            st_global_v8(orow + col, pk);  // 16 columns = one 32-byte sector
          }
        }
      }
      tc_fence_before();
      if (kKind == kExpertFused && job.phase == 0) __threadfence();  // H rows before the count
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&acc_empty[acc]);
        if (kKind == kExpertFused && job.phase == 0) atomicAdd(ma.ready + job.mt, 1);
      }
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

cudaError_t launch_expert_tc(ExpertKind kind, const CUtensorMap& tm_a, const CUtensorMap& tm_b0,
                             const CUtensorMap& tm_b1, const CUtensorMap& tm_b2,
                             const MlpArgs& a, int num_sms, cudaStream_t st) {
  const bool has0 = kind != kExpertDown, has1 = kind == kExpertDown || kind == kExpertFused;
  const GemmArgs& gs = has0 ? a.p[0] : a.p[1];
  if (gs.max_tiles <= 0) return cudaSuccess;
  if (kind == kExpertFused &&
      (a.p[0].a_src == nullptr || a.p[0].perm == nullptr || a.p[0].k <= 0))
    return cudaErrorInvalidValue;
  if (kind == kExpertFused && a.ready == nullptr) return cudaErrorInvalidValue;
  int per_tile = 0;
  if (has0) per_tile += (a.p[0].n_out + kBN / 2 - 1) / (kBN / 2);
  if (has1) per_tile += (a.p[1].n_out + kBN - 1) / kBN;
  const int64_t bound = static_cast<int64_t>(gs.max_tiles) * per_tile;
  const int grid = static_cast<int>(bound < num_sms ? bound : num_sms);
  void (*kernel)(CUtensorMap, CUtensorMap, CUtensorMap, CUtensorMap, MlpArgs) =
      kind == kExpertGateUpTma ? expert_tc_kernel<kExpertGateUpTma>
      : kind == kExpertDown    ? expert_tc_kernel<kExpertDown>
                               : expert_tc_kernel<kExpertFused>;
  cudaError_t err =
      cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
  if (err != cudaSuccess) return err;
  if (kind != kExpertFused)
    return launch_pdl(kernel, dim3(grid), dim3(kThreads), kSmemBytes, st, 1, tm_a, tm_b0, tm_b1,
                      tm_b2, a);
  // CTAs of the fused launch wait on one another: a cooperative launch guarantees that all of
  // them are resident (one per SM at this shared-memory size).
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  err = cudaLaunchKernelEx(&cfg, kernel, tm_a, tm_b0, tm_b1, tm_b2, a);
  if (err == cudaSuccess) return err;
  (void)cudaGetLastError();  // cooperative + programmatic serialization refused: drop the latter
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, tm_a, tm_b0, tm_b1, tm_b2, a);
}

}  // namespace pr2
