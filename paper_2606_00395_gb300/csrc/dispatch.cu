// Dispatch of (token, slot) pairs to experts and the gate-weighted combine.
//
// Dispatch ("dispatch to experts", Algorithm 1) is a stable counting sort of the flat slot ids
// f = t*k + s by expert id, deterministic and bit-exact:
//   1. hist   - one block per 256 slots: validate each slot (expert in [0,N), not repeated in
//               its token) and count per expert in shared memory -> blk_hist[b][e].
//   2. scan   - one block: per expert an exclusive scan over blocks (in place), the expert
//               totals (counts), their exclusive scan (offsets), the M-tile table of the
//               grouped GEMM, and the static tile tables of the shared experts.
//   3. place  - one block per 256 slots again: per-warp counts via __match_any_sync, a scan
//               over the 8 warps, then rank = popc(lanes below with the same expert):
//               perm[offsets[e] + r] = f, inv[f] = its position (-1 for an invalid slot).
//   4. gather - X[p, :] = h[perm[p] / k, :], 16-byte vectors, one warp per row; fp32 path only
//               (the bf16 gate/up GEMM reads its rows from h through perm itself).
// Steps 1-3 normally run as one cooperative launch (dispatch_fused_kernel): every block counts
// its slots, one bounded grid barrier, then each block derives the expert totals, its own
// per-expert bases and the expert offsets from the whole block histogram (identical in every
// block), block 0 writes counts, offsets and the tile tables (and clears the grouped GEMM's
// per-M-tile readiness counters), and every block places its slots.  Shapes whose grid cannot
// be resident at once use the three kernels above.
// Combine (the sums of Eqs. pr2_old_output / pr2_output):
//   out[t, :] = sum_s gates[t,s] * Y[inv[t*k+s], :] + sum_j Ys[j, t, :], fp32 accumulation,
//   plus, when given, a residual row r[t, :] (the multi-layer loop's h_l; may alias out).
//   bf16: combine_bulk_kernel (rows streamed into shared memory with bulk copies); fp32 and
//   layers whose rows do not fit its ring: combine_kernel (rows through registers).
#include <mutex>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

constexpr int kWarps = kDispatchChunk / 32;

__device__ __forceinline__ bool slot_valid(const int32_t* __restrict__ idx, int64_t f, int k, int N,
                                           int* e_out) {
  const int e = idx[f];
  bool ok = e >= 0 && e < N;
  const int64_t base = f - (f % k);
  for (int64_t f2 = base; ok && f2 < f; ++f2)
    if (idx[f2] == e) ok = false;
  *e_out = ok ? e : -1;
  return ok;
}

__global__ void __launch_bounds__(kDispatchChunk)
    hist_kernel(const int32_t* __restrict__ idx, int64_t F, int k, int N,
                int32_t* __restrict__ blk_hist, int32_t* status) {
  __shared__ int hist[kMaxExpertsDispatch];
  for (int e = threadIdx.x; e < N; e += blockDim.x) hist[e] = 0;
  pdl_wait();
  pdl_trigger();
  __syncthreads();
  const int64_t f = static_cast<int64_t>(blockIdx.x) * kDispatchChunk + threadIdx.x;
  if (f < F) {
    int e;
    if (slot_valid(idx, f, k, N, &e))
      atomicAdd(&hist[e], 1);
    else if (status != nullptr)
      atomicOr(status, PR2_STATUS_BAD_INDEX);
  }
  __syncthreads();
  int32_t* out = blk_hist + static_cast<int64_t>(blockIdx.x) * N;
  for (int e = threadIdx.x; e < N; e += blockDim.x) out[e] = hist[e];
}

// Exclusive block-wide scan of one int per thread (blockDim.x == 1024).
__device__ __forceinline__ int block_exclusive_scan(int v, int* sh, int* total) {
  const int tid = threadIdx.x;
  const int lane = tid & 31, w = tid >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[w] = x;
  __syncthreads();
  if (w == 0) {
    int s = sh[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    sh[lane] = s;  // inclusive warp totals
  }
  __syncthreads();
  const int incl = x + (w > 0 ? sh[w - 1] : 0);
  *total = sh[31];
  __syncthreads();
  return incl - v;
}

// The grouped GEMM's tile table: each expert's rows split into ceil(rows / tile_rows) tiles of
// near-equal size (entry i belongs to the expert whose tile range contains i; its per-tile
// readiness counter is cleared) and the static tile tables of the shared experts
// (every token: gate/up reads rows of h, down rows of Hs), from the experts' row offsets ex_off
// and first tiles ex_tile (N + 1 entries each, in shared memory); num_tiles[0..1] = their
// lengths.  Called by every thread of one block.
__device__ void write_tile_tables(int N, int64_t T, int n_shared, int tile_rows,
                                  const int* ex_off, const int* ex_tile,
                                  TileEntry* __restrict__ tiles,
                                  int32_t* __restrict__ num_tiles,
                                  TileEntry* __restrict__ stiles1,
                                  TileEntry* __restrict__ stiles2, int32_t* __restrict__ ready) {
  const int tid = threadIdx.x;
  const int all_tiles = ex_tile[N];
  const int mt_T = static_cast<int>((T + kTileM - 1) / kTileM);
  if (tid == 0) {
    num_tiles[0] = all_tiles;
    num_tiles[1] = n_shared * mt_T;
  }
  for (int i = tid; i < all_tiles; i += blockDim.x) {
    int lo = 0, hi = N - 1;
    while (lo < hi) {  // last expert with ex_tile[ex] <= i
      const int mid = (lo + hi + 1) >> 1;
      if (ex_tile[mid] <= i) lo = mid; else hi = mid - 1;
    }
    // the expert's c rows split into nch = ceil(c / tile_rows) tiles of near-equal size
    const int j = i - ex_tile[lo];
    const int nch = ex_tile[lo + 1] - ex_tile[lo];
    const int c = ex_off[lo + 1] - ex_off[lo];
    const int sz = (c + nch - 1) / nch;
    const int r0 = ex_off[lo] + j * sz;
    const int left = ex_off[lo + 1] - r0;
    tiles[i] = TileEntry{lo, r0, left < sz ? left : sz, r0};
    if (ready != nullptr) ready[i] = 0;  // per M-tile counter of the fused expert GEMM
  }
  for (int i = tid; i < n_shared * mt_T; i += blockDim.x) {
    const int j = i / mt_T, m = i - j * mt_T;
    const int r0 = m * kTileM;
    const int rows = (T - r0) < kTileM ? static_cast<int>(T - r0) : kTileM;
    const int o0 = static_cast<int>(j * T) + r0;
    stiles1[i] = TileEntry{j, r0, rows, o0};
    stiles2[i] = TileEntry{j, o0, rows, o0};
  }
}

// One block of 1024 threads = G groups of N_pad threads: thread (g, e) owns expert e over the
// block range of group g, so the per-expert scans over blocks run G-way parallel.
__global__ void __launch_bounds__(1024)
    scan_kernel(int32_t* __restrict__ blk_hist, int nblk, int N, int64_t T, int n_shared,
                int tile_rows,
                int32_t* __restrict__ counts, int32_t* __restrict__ offsets,
                TileEntry* __restrict__ tiles, int32_t* __restrict__ num_tiles,
                TileEntry* __restrict__ stiles1, TileEntry* __restrict__ stiles2,
                int32_t* __restrict__ ready) {
  __shared__ int sh[32];
  __shared__ int part[1024];  // [G][N_pad] partial sums, then their exclusive scan over g
  __shared__ int ex_off[kMaxExpertsDispatch + 1];
  __shared__ int ex_tile[kMaxExpertsDispatch + 1];
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x;
  int n_pad = 32;
  while (n_pad < N) n_pad <<= 1;
  const int G = 1024 / n_pad;
  const int g = tid / n_pad, e = tid - g * n_pad;
  const int per = (nblk + G - 1) / G;
  const int b0 = g * per, b1 = min(nblk, b0 + per);
  // Column slices are read 8 rows at a time with every load in flight (one L2 round trip per
  // 8 rows instead of a dependent chain).
  int sum = 0;
  if (e < N) {
    for (int c0 = b0; c0 < b1; c0 += 8) {
      int v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j)
        v[j] = (c0 + j < b1) ? blk_hist[static_cast<int64_t>(c0 + j) * N + e] : 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) sum += v[j];
    }
  }
  part[tid] = sum;
  __syncthreads();
  int total = 0;
  if (tid < N) {  // exclusive scan over the groups of expert tid
    for (int gg = 0; gg < G; ++gg) {
      const int v = part[gg * n_pad + tid];
      part[gg * n_pad + tid] = total;
      total += v;
    }
    counts[tid] = total;
  }
  __syncthreads();
  int all_rows, all_tiles;
  const int off = block_exclusive_scan(tid < N ? total : 0, sh, &all_rows);
  const int ntile_e = tid < N ? (total + tile_rows - 1) / tile_rows : 0;
  const int tstart = block_exclusive_scan(ntile_e, sh, &all_tiles);
  if (tid < N) {
    offsets[tid] = off;
    ex_off[tid] = off;
    ex_tile[tid] = tstart;
  }
  if (tid == 0) {
    offsets[N] = all_rows;
    ex_off[N] = all_rows;
    ex_tile[N] = all_tiles;
  }
  __syncthreads();
  // per-block bases: expert offset + rows of this expert in all earlier blocks
  if (e < N) {
    int run = ex_off[e] + part[g * n_pad + e];
    for (int c0 = b0; c0 < b1; c0 += 8) {
      int v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j)
        v[j] = (c0 + j < b1) ? blk_hist[static_cast<int64_t>(c0 + j) * N + e] : 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        if (c0 + j < b1) blk_hist[static_cast<int64_t>(c0 + j) * N + e] = run;
        run += v[j];
      }
    }
  }
  write_tile_tables(N, T, n_shared, tile_rows, ex_off, ex_tile, tiles, num_tiles, stiles1,
                    stiles2, ready);
}

__global__ void __launch_bounds__(kDispatchChunk)
    place_kernel(const int32_t* __restrict__ idx, int64_t F, int k, int N,
                 const int32_t* __restrict__ blk_base, int32_t* __restrict__ perm,
                 int32_t* __restrict__ inv) {
  __shared__ int wcnt[kWarps][kMaxExpertsDispatch];
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < kWarps * N; i += blockDim.x) wcnt[i / N][i % N] = 0;
  pdl_wait();
  pdl_trigger();
  __syncthreads();
  const int64_t f = static_cast<int64_t>(blockIdx.x) * kDispatchChunk + threadIdx.x;
  int e = -1;
  if (f < F) slot_valid(idx, f, k, N, &e);
  const unsigned same = __match_any_sync(0xffffffffu, e);
  if (e >= 0 && lane == __ffs(same) - 1) wcnt[w][e] = __popc(same);
  __syncthreads();
  const int32_t* base = blk_base + static_cast<int64_t>(blockIdx.x) * N;
  for (int x = threadIdx.x; x < N; x += blockDim.x) {
    int run = base[x];
    for (int ww = 0; ww < kWarps; ++ww) {
      const int c = wcnt[ww][x];
      wcnt[ww][x] = run;
      run += c;
    }
  }
  __syncthreads();
  if (f < F) {
    if (e >= 0) {
      const int pos = wcnt[w][e] + __popc(same & lanemask_lt());
      perm[pos] = static_cast<int32_t>(f);
      inv[f] = pos;
    } else {
      inv[f] = -1;
    }
  }
}

// Exclusive scan of one int per thread over a 256-thread block (8 warps).
__device__ __forceinline__ int block256_exclusive_scan(int v, int* sh, int* total) {
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[w] = x;
  __syncthreads();
  if (w == 0) {
    int s = lane < kWarps ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < kWarps) sh[lane] = s;
  }
  __syncthreads();
  const int incl = x + (w > 0 ? sh[w - 1] : 0);
  *total = sh[kWarps - 1];
  __syncthreads();
  return incl - v;
}

// Hist, scan and place in one cooperative launch (N % 4 == 0, N <= 256; grid resident).
__global__ void __launch_bounds__(kDispatchChunk)
    dispatch_fused_kernel(const int32_t* __restrict__ idx, int64_t F, int k, int N, int64_t T,
                          int n_shared, int tile_rows, int32_t* blk_hist, int32_t* __restrict__ counts,
                          int32_t* __restrict__ offsets, int32_t* __restrict__ perm,
                          int32_t* __restrict__ inv, TileEntry* __restrict__ tiles,
                          int32_t* __restrict__ num_tiles, TileEntry* __restrict__ stiles1,
                          TileEntry* __restrict__ stiles2, unsigned int* sync_ctr,
                          int32_t* status, int32_t* __restrict__ ready) {
  extern __shared__ int dsm[];
  int* wcnt = dsm;                   // [kWarps][N] per-warp counts, then per-warp bases
  int* tot = wcnt + kWarps * N;      // [N] slots of each expert over all blocks
  int* pre = tot + N;                // [N] slots of each expert in the blocks before this one
  int* ex_off = pre + N;             // [N+1]
  int* ex_tile = ex_off + N + 1;     // [N+1]
  __shared__ int sh[32];
  __shared__ int abort_s;
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31;
  const int nblk = static_cast<int>(gridDim.x), b = static_cast<int>(blockIdx.x);
  for (int i = tid; i < kWarps * N; i += blockDim.x) wcnt[i] = 0;
  for (int i = tid; i < N; i += blockDim.x) {
    tot[i] = 0;
    pre[i] = 0;
  }
  __syncthreads();
  // ---- 1. this block's slots: validity, per-warp counts, block histogram
  const int64_t f = static_cast<int64_t>(b) * kDispatchChunk + tid;
  int e = -1;
  if (f < F && !slot_valid(idx, f, k, N, &e) && status != nullptr)
    atomicOr(status, PR2_STATUS_BAD_INDEX);
  const unsigned same = __match_any_sync(0xffffffffu, e);
  if (e >= 0 && lane == __ffs(same) - 1) wcnt[w * N + e] = __popc(same);
  __syncthreads();
  for (int x = tid; x < N; x += blockDim.x) {
    int c = 0;
    for (int ww = 0; ww < kWarps; ++ww) c += wcnt[ww * N + x];
    blk_hist[static_cast<int64_t>(b) * N + x] = c;
  }
  // ---- grid barrier (every block is resident: cooperative launch); bounded
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    atomicAdd(sync_ctr, 1u);
    const uint64_t t0 = globaltimer_ns();
    int ok = 1;
    while (atomicAdd(sync_ctr, 0u) < static_cast<unsigned>(nblk)) {
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        ok = 0;
        if (status != nullptr) atomicOr(status, PR2_STATUS_TIMEOUT);
        break;
      }
    }
    __threadfence();
    abort_s = !ok;
  }
  __syncthreads();
  if (abort_s) return;
  // ---- 2. expert totals and this block's prefix from the whole histogram (int4 columns)
  const int n4 = N / 4, G = kDispatchChunk / n4;
  const int q = tid % n4, g = tid / n4;
  if (g < G) {
    int4 all = make_int4(0, 0, 0, 0), before = make_int4(0, 0, 0, 0);
    const int4* col = reinterpret_cast<const int4*>(blk_hist) + q;
    for (int r0 = g; r0 < nblk; r0 += 8 * G) {
      int4 v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int r = r0 + j * G;
        v[j] = r < nblk ? __ldcg(col + static_cast<int64_t>(r) * n4) : make_int4(0, 0, 0, 0);
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int r = r0 + j * G;
        all.x += v[j].x;
        all.y += v[j].y;
        all.z += v[j].z;
        all.w += v[j].w;
        if (r < b) {
          before.x += v[j].x;
          before.y += v[j].y;
          before.z += v[j].z;
          before.w += v[j].w;
        }
      }
    }
    atomicAdd(&tot[4 * q], all.x);
    atomicAdd(&tot[4 * q + 1], all.y);
    atomicAdd(&tot[4 * q + 2], all.z);
    atomicAdd(&tot[4 * q + 3], all.w);
    atomicAdd(&pre[4 * q], before.x);
    atomicAdd(&pre[4 * q + 1], before.y);
    atomicAdd(&pre[4 * q + 2], before.z);
    atomicAdd(&pre[4 * q + 3], before.w);
  }
  __syncthreads();
  int all_rows, all_tiles;
  const int total = tid < N ? tot[tid] : 0;
  const int off = block256_exclusive_scan(total, sh, &all_rows);
  const int tstart =
      block256_exclusive_scan(tid < N ? (total + tile_rows - 1) / tile_rows : 0, sh,
                              &all_tiles);
  if (tid < N) {
    ex_off[tid] = off;
    ex_tile[tid] = tstart;
  }
  if (tid == 0) {
    ex_off[N] = all_rows;
    ex_tile[N] = all_tiles;
  }
  __syncthreads();
  if (b == 0) {
    if (tid < N) {
      counts[tid] = total;
      offsets[tid] = off;
    }
    if (tid == 0) offsets[N] = all_rows;
    write_tile_tables(N, T, n_shared, tile_rows, ex_off, ex_tile, tiles, num_tiles, stiles1,
                      stiles2, ready);
  }
  // ---- 3. stable placement: per-warp bases, then ranks within the warp
  for (int x = tid; x < N; x += blockDim.x) {
    int run = ex_off[x] + pre[x];
    for (int ww = 0; ww < kWarps; ++ww) {
      const int c = wcnt[ww * N + x];
      wcnt[ww * N + x] = run;
      run += c;
    }
  }
  __syncthreads();
  if (f < F) {
    if (e >= 0) {
      const int pos = wcnt[w * N + e] + __popc(same & lanemask_lt());
      perm[pos] = static_cast<int32_t>(f);
      inv[f] = pos;
    } else {
      inv[f] = -1;
    }
  }
}

// Dispatch of a route that the routing kernel just wrote, from its per-CTA histograms: block b
// handles the slots of routing tile b (128 tokens x k slots, one thread per slot).  Every block
// derives the expert totals and its own prefix from the histogram rows (int4 column reads),
// then places its slots in stable order exactly as dispatch_fused_kernel does; block 0 writes
// counts, offsets and the tile tables.  Every slot is valid (the routing kernel wrote k distinct
// experts in [0, N) per token), which is what the histograms counted.
constexpr int kHistBlock = kTileM * kMaxTopK;  // 1024 threads: the slots of one routing tile
constexpr int kHistWarps = kHistBlock / 32;

__global__ void __launch_bounds__(kHistBlock)
    dispatch_hist_kernel(const int32_t* __restrict__ idx, int64_t T, int k, int N, int n_shared,
                         int tile_rows, const int32_t* __restrict__ hist, int hist_rows,
                         int split, int32_t* __restrict__ counts, int32_t* __restrict__ offsets,
                         int32_t* __restrict__ perm, int32_t* __restrict__ inv,
                         TileEntry* __restrict__ tiles, int32_t* __restrict__ num_tiles,
                         TileEntry* __restrict__ stiles1, TileEntry* __restrict__ stiles2,
                         int32_t* __restrict__ ready) {
  extern __shared__ int dsm[];
  int* wcnt = dsm;                     // [kHistWarps][N] per-warp counts, then per-warp bases
  int* tot = wcnt + kHistWarps * N;    // [N]
  int* pre = tot + N;                  // [N] slots of each expert in earlier tiles
  int* ex_off = pre + N;               // [N+1]
  int* ex_tile = ex_off + N + 1;       // [N+1]
  __shared__ int sh[32];
  const int tid = threadIdx.x, w = tid >> 5, lane = tid & 31;
  const int b = static_cast<int>(blockIdx.x);
  for (int i = tid; i < kHistWarps * N; i += kHistBlock) wcnt[i] = 0;
  for (int i = tid; i < N; i += kHistBlock) {
    tot[i] = 0;
    pre[i] = 0;
  }
  pdl_wait();  // the route and its histograms come from the routing kernel
  pdl_trigger();
  __syncthreads();
  // ---- expert totals and this tile's prefix: hist rows [0, hist_rows), before = rows < b*split
  const int n4 = N / 4, G = kHistBlock / n4;
  const int q = tid % n4, g = tid / n4;
  const int before_rows = b * split;
  if (g < G) {
    int4 all = make_int4(0, 0, 0, 0), bef = make_int4(0, 0, 0, 0);
    const int4* col = reinterpret_cast<const int4*>(hist) + q;
    for (int r0 = g; r0 < hist_rows; r0 += 8 * G) {
      int4 v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int r = r0 + j * G;
        v[j] = r < hist_rows ? __ldcg(col + static_cast<int64_t>(r) * n4) : make_int4(0, 0, 0, 0);
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int r = r0 + j * G;
        all.x += v[j].x;
        all.y += v[j].y;
        all.z += v[j].z;
        all.w += v[j].w;
        if (r < before_rows) {
          bef.x += v[j].x;
          bef.y += v[j].y;
          bef.z += v[j].z;
          bef.w += v[j].w;
        }
      }
    }
    atomicAdd(&tot[4 * q], all.x);
    atomicAdd(&tot[4 * q + 1], all.y);
    atomicAdd(&tot[4 * q + 2], all.z);
    atomicAdd(&tot[4 * q + 3], all.w);
    atomicAdd(&pre[4 * q], bef.x);
    atomicAdd(&pre[4 * q + 1], bef.y);
    atomicAdd(&pre[4 * q + 2], bef.z);
    atomicAdd(&pre[4 * q + 3], bef.w);
  }
  // ---- this tile's slots: per-warp counts
  const int64_t F = T * k;
  const int64_t f = static_cast<int64_t>(b) * kTileM * k + tid;
  const bool own = tid < kTileM * k && f < F;
  const int e = own ? idx[f] : -1;
  const unsigned same = __match_any_sync(0xffffffffu, e);
  if (e >= 0 && lane == __ffs(same) - 1) wcnt[w * N + e] = __popc(same);
  __syncthreads();
  int all_rows, all_tiles;
  const int total = tid < N ? tot[tid] : 0;
  const int off = block_exclusive_scan(total, sh, &all_rows);
  const int tstart =
      block_exclusive_scan(tid < N ? (total + tile_rows - 1) / tile_rows : 0, sh, &all_tiles);
  if (tid < N) {
    ex_off[tid] = off;
    ex_tile[tid] = tstart;
  }
  if (tid == 0) {
    ex_off[N] = all_rows;
    ex_tile[N] = all_tiles;
  }
  __syncthreads();
  if (b == 0) {
    if (tid < N) {
      counts[tid] = total;
      offsets[tid] = off;
    }
    if (tid == 0) offsets[N] = all_rows;
    write_tile_tables(N, T, n_shared, tile_rows, ex_off, ex_tile, tiles, num_tiles, stiles1,
                      stiles2, ready);
  }
  // ---- stable placement: per-warp bases, then ranks within the warp
  for (int x = tid; x < N; x += kHistBlock) {
    int run = ex_off[x] + pre[x];
    for (int ww = 0; ww < kHistWarps; ++ww) {
      const int c = wcnt[ww * N + x];
      wcnt[ww * N + x] = run;
      run += c;
    }
  }
  __syncthreads();
  if (own) {
    const int pos = wcnt[w * N + e] + __popc(same & lanemask_lt());
    perm[pos] = static_cast<int32_t>(f);
    inv[f] = pos;
  }
}

size_t hist_smem_bytes(int N) { return sizeof(int) * (static_cast<size_t>(kHistWarps) * N + 4 * N + 2); }

size_t fused_smem_bytes(int N) { return sizeof(int) * (static_cast<size_t>(kWarps) * N + 4 * N + 2); }

// Whether the fused dispatch can run (shape, and every block resident at once), cached per
// device and N.
bool fused_dispatch_ok(int N, int nblk, int num_sms) {
  if (N % 4 != 0 || N > kDispatchChunk || nblk < 1) return false;
  struct Entry {
    int dev, N, blocks_per_sm;
  };
  static std::mutex mu;
  static Entry cache[32];
  static int used = 0;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  std::lock_guard<std::mutex> lock(mu);
  int per_sm = -1;
  for (int i = 0; i < used; ++i)
    if (cache[i].dev == dev && cache[i].N == N) per_sm = cache[i].blocks_per_sm;
  if (per_sm < 0) {
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, dispatch_fused_kernel,
                                                      kDispatchChunk, fused_smem_bytes(N)) !=
        cudaSuccess) {
      (void)cudaGetLastError();
      per_sm = 0;
    }
    if (used < 32) cache[used++] = Entry{dev, N, per_sm};
  }
  return static_cast<int64_t>(per_sm) * num_sms >= nblk;
}

// X[p, :] = h[perm[p] / k, :] for p < offsets[N]; row_vec = 16-byte vectors per row.
__global__ void __launch_bounds__(256)
    gather_kernel(const uint4* __restrict__ h, const int32_t* __restrict__ perm,
                  const int32_t* __restrict__ nrows_ptr, int k, int row_vec,
                  uint4* __restrict__ X) {
  pdl_wait();
  pdl_trigger();
  const int nrows = *nrows_ptr;
  const int lane = threadIdx.x & 31;
  const int warp0 = static_cast<int>((blockIdx.x * blockDim.x + threadIdx.x) >> 5);
  const int nwarps = static_cast<int>((gridDim.x * blockDim.x) >> 5);
  for (int p = warp0; p < nrows; p += nwarps) {
    const int t = perm[p] / k;
    const uint4* src = h + static_cast<int64_t>(t) * row_vec;
    uint4* dst = X + static_cast<int64_t>(p) * row_vec;
#pragma unroll 8
    for (int v = lane; v < row_vec; v += 32) dst[v] = __ldg(src + v);
  }
}

template <typename T, int V, int KMAX>  // V elements per 16-byte vector, k <= KMAX
__global__ void __launch_bounds__(256)
    combine_kernel(const T* __restrict__ Y, const T* __restrict__ Ys,
                   const int32_t* __restrict__ inv, const float* __restrict__ gates, int64_t Tn,
                   int k, int d, int n_shared, const T* residual, T* out,
                   const int32_t* status) {
  pdl_wait();
  pdl_trigger();
  if (status_timed_out(status)) return;  // dispatch gave up: inv may be unwritten
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
  const int nvec = d / V;
  for (int64_t t = warp0; t < Tn; t += nwarps) {
    int my_pos = -1;
    float my_g = 0.f;
    if (lane < k) {
      my_pos = inv[t * k + lane];
      my_g = gates[t * k + lane];
    }
    int pos[KMAX];
    float gs[KMAX];
#pragma unroll
    for (int s = 0; s < KMAX; ++s) {
      pos[s] = __shfl_sync(0xffffffffu, my_pos, s);
      gs[s] = __shfl_sync(0xffffffffu, my_g, s);
      if (s >= k) pos[s] = -1;
    }
    for (int c = lane; c < nvec; c += 32) {
      uint4 raw[KMAX];
#pragma unroll
      for (int s = 0; s < KMAX; ++s)
        if (pos[s] >= 0)
          raw[s] = __ldg(reinterpret_cast<const uint4*>(Y + static_cast<int64_t>(pos[s]) * d) + c);
      float acc[V];
#pragma unroll
      for (int j = 0; j < V; ++j) acc[j] = 0.f;
      if (residual != nullptr) {  // read before the same thread overwrites it (in place)
        const uint4 r = reinterpret_cast<const uint4*>(residual + t * d)[c];
        const T* v = reinterpret_cast<const T*>(&r);
#pragma unroll
        for (int j = 0; j < V; ++j) acc[j] = to_f32<T>(v[j]);
      }
#pragma unroll
      for (int s = 0; s < KMAX; ++s) {
        if (pos[s] < 0) continue;
        const T* v = reinterpret_cast<const T*>(&raw[s]);
#pragma unroll
        for (int j = 0; j < V; ++j) acc[j] = fmaf(gs[s], to_f32<T>(v[j]), acc[j]);
      }
      for (int j2 = 0; j2 < n_shared; ++j2) {
        const uint4 r = __ldg(
            reinterpret_cast<const uint4*>(Ys + (static_cast<int64_t>(j2) * Tn + t) * d) + c);
        const T* v = reinterpret_cast<const T*>(&r);
#pragma unroll
        for (int j = 0; j < V; ++j) acc[j] += to_f32<T>(v[j]);
      }
      uint4 o;
      T* ov = reinterpret_cast<T*>(&o);
#pragma unroll
      for (int j = 0; j < V; ++j) ov[j] = from_f32<T>(acc[j]);
      reinterpret_cast<uint4*>(out + t * d)[c] = o;
    }
  }
}

// ---- combine through shared memory (bf16) ---------------------------------------------------
// out[t] = round(residual[t] + sum_s g[t,s] Y[inv[t,s]] + sum_j Ys[j,t]), the same arithmetic in
// the same order as combine_kernel.  Persistent, one CTA per SM, tokens t = blockIdx.x + i *
// gridDim.x.  Warp 0 is the producer: for each token it copies the token's rows (its k expert
// rows, its shared-expert rows and the residual row) into one slot of a ring in shared memory
// with 1-D bulk copies, so that a few hundred KB per SM are in flight; warps 1-8 sum a slot,
// each thread one 16-byte column chunk per pass, and release it.
constexpr int kCbConsumers = 8;
constexpr int kCbThreads = 32 * (kCbConsumers + 1);
constexpr int kCbMaxSlots = 8;
constexpr int kCbAhead = 4;  // tokens whose route entries the producer holds in advance
constexpr int kCbDataBytes = 196 * 1024;  // ring of token slots
constexpr int kCbSmemBytes = 128 + kCbDataBytes + kCbMaxSlots * (32 * 4 + 8) + 2 * kCbMaxSlots * 8;

struct CombineRing {
  int slots, rows, row_bytes;
};

__host__ __device__ inline CombineRing combine_ring(int k, int d, int n_shared, bool residual) {
  CombineRing r;
  r.rows = k + n_shared + (residual ? 1 : 0);
  r.row_bytes = d * 2;
  const int64_t slot = static_cast<int64_t>(r.rows) * r.row_bytes;
  const int64_t n = slot > 0 ? kCbDataBytes / slot : 0;
  r.slots = static_cast<int>(n < kCbMaxSlots ? n : kCbMaxSlots);
  return r;
}

constexpr int kCbMaxK = 8;  // the bf16 layer supports k <= 8

__global__ void __launch_bounds__(kCbThreads, 1)
    combine_bulk_kernel(const __nv_bfloat16* __restrict__ Y, const __nv_bfloat16* __restrict__ Ys,
                        const int32_t* __restrict__ inv, const float* __restrict__ gates,
                        int64_t Tn, int k, int d, int n_shared, const __nv_bfloat16* residual,
                        __nv_bfloat16* out, int32_t* status) {
  extern __shared__ uint8_t cb_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(cb_raw) + 127) & ~static_cast<uintptr_t>(127));
  const CombineRing ring = combine_ring(k, d, n_shared, residual != nullptr);
  const int S = ring.slots;
  const int slot_bytes = ring.rows * ring.row_bytes;
  float* meta_gate = reinterpret_cast<float*>(base + kCbDataBytes);             // [S][32]
  uint32_t* meta_mask = reinterpret_cast<uint32_t*>(meta_gate + kCbMaxSlots * 32);  // [S]
  uint64_t* full = reinterpret_cast<uint64_t*>(
      (reinterpret_cast<uintptr_t>(meta_mask + kCbMaxSlots) + 7) & ~static_cast<uintptr_t>(7));
  uint64_t* empty = full + kCbMaxSlots;
  __shared__ int abort_flag_s;
  volatile int* abort_flag = &abort_flag_s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCbConsumers);
    }
    abort_flag_s = 0;
    fence_mbar_init();
  }
  pdl_wait();
  pdl_trigger();
  if (threadIdx.x == 0) abort_flag_s = status_timed_out(status) ? 1 : 0;  // no tables to read
  __syncthreads();
  if (abort_flag_s) return;
  const int nvec = d / 8;
  if (warp == 0) {
    // ---------------- producer ----------------
    uint32_t issued = 0, last_par = 0;
    int slot = 0;
    uint32_t phase = 0;
    // Route entries of this CTA's next kCbAhead tokens, loaded ahead so that no token waits for
    // a global-memory round trip before its copies are issued (lane s: slot s).  The token loop
    // is unrolled by kCbAhead, so entry j is read kCbAhead tokens after its load was issued.
    int q_pos[kCbAhead];
    float q_g[kCbAhead];
    auto fetch = [&](int64_t tt, int& p, float& gg) {
      p = -1;
      gg = 0.f;
      if (lane < k && tt < Tn) {
        p = inv[tt * k + lane];
        gg = gates[tt * k + lane];
      }
    };
    const int64_t stride = gridDim.x;
#pragma unroll
    for (int j = 0; j < kCbAhead; ++j) fetch(blockIdx.x + j * stride, q_pos[j], q_g[j]);
    bool ok = true;
    for (int64_t t0 = blockIdx.x; t0 < Tn && ok; t0 += kCbAhead * stride) {
#pragma unroll
      for (int j = 0; j < kCbAhead; ++j) {
        const int64_t t = t0 + j * stride;
        if (t >= Tn || !ok) break;
        const int pos = q_pos[j];
        const float gt = q_g[j];
        fetch(t + kCbAhead * stride, q_pos[j], q_g[j]);
        if (!mbar_wait(&empty[slot], phase ^ 1u, abort_flag, status)) {
          ok = false;
          break;
        }
        const uint32_t vmask = __ballot_sync(0xffffffffu, pos >= 0);
        if (lane < k) meta_gate[slot * 32 + lane] = gt;
        if (lane == 0) meta_mask[slot] = vmask;
        __syncwarp();
        const uint32_t nrows = __popc(vmask) + n_shared + (residual != nullptr ? 1 : 0);
        const uint32_t dst = smem_u32(base + slot * slot_bytes);
        const uint32_t rb = static_cast<uint32_t>(ring.row_bytes);
        if (lane == 0) mbar_arrive_expect_tx(&full[slot], nrows * rb);  // releases the meta data
        __syncwarp();
        if (pos >= 0)
          bulk_load(dst + lane * rb, Y + static_cast<int64_t>(pos) * d, rb, &full[slot]);
        if (lane < n_shared)
          bulk_load(dst + (k + lane) * rb, Ys + (static_cast<int64_t>(lane) * Tn + t) * d, rb,
                    &full[slot]);
        if (lane == 0 && residual != nullptr)
          bulk_load(dst + (k + n_shared) * rb, residual + t * d, rb, &full[slot]);
        issued |= 1u << slot;
        last_par = (last_par & ~(1u << slot)) | (phase << slot);
        if (++slot == S) {
          slot = 0;
          phase ^= 1u;
        }
      }
    }
    // no copy may still be landing when the CTA leaves (the consumers may have given up)
    if (lane == 0)
      for (int s = 0; s < S; ++s)
        if ((issued >> s) & 1u)
          mbar_wait_slow(&full[s], (last_par >> s) & 1u, nullptr, nullptr, kDrainLimitNs);
  } else {
    // ---------------- consumers ----------------
    const int ct = threadIdx.x - 32;
    int slot = 0;
    uint32_t phase = 0;
    for (int64_t t = blockIdx.x; t < Tn; t += gridDim.x) {
      if (!mbar_wait(&full[slot], phase, abort_flag, status)) break;
      const uint8_t* sbase = base + slot * slot_bytes;
      const uint32_t vmask = meta_mask[slot];
      const float* gs = meta_gate + slot * 32;
      for (int c = ct; c < nvec; c += 32 * kCbConsumers) {
        float acc[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] = 0.f;
        if (residual != nullptr) {
          const uint4 r = reinterpret_cast<const uint4*>(sbase + (k + n_shared) * ring.row_bytes)[c];
          const __nv_bfloat16* v = reinterpret_cast<const __nv_bfloat16*>(&r);
#pragma unroll
          for (int j = 0; j < 8; ++j) acc[j] = __bfloat162float(v[j]);
        }
#pragma unroll
        for (int s = 0; s < kCbMaxK; ++s) {
          if (s >= k || !((vmask >> s) & 1u)) continue;
          const uint4 r = reinterpret_cast<const uint4*>(sbase + s * ring.row_bytes)[c];
          const __nv_bfloat16* v = reinterpret_cast<const __nv_bfloat16*>(&r);
#pragma unroll
          for (int j = 0; j < 8; ++j) acc[j] = fmaf(gs[s], __bfloat162float(v[j]), acc[j]);
        }
        for (int j2 = 0; j2 < n_shared; ++j2) {
          const uint4 r = reinterpret_cast<const uint4*>(sbase + (k + j2) * ring.row_bytes)[c];
          const __nv_bfloat16* v = reinterpret_cast<const __nv_bfloat16*>(&r);
#pragma unroll
          for (int j = 0; j < 8; ++j) acc[j] += __bfloat162float(v[j]);
        }
        uint4 o;
        o.x = pack_bf16x2(acc[0], acc[1]);
        o.y = pack_bf16x2(acc[2], acc[3]);
        o.z = pack_bf16x2(acc[4], acc[5]);
        o.w = pack_bf16x2(acc[6], acc[7]);
        reinterpret_cast<uint4*>(out + t * d)[c] = o;
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[slot]);
      if (++slot == S) {
        slot = 0;
        phase ^= 1u;
      }
    }
  }
}

}  // namespace

cudaError_t launch_dispatch(const DispatchArgs& a, int num_sms, cudaStream_t st) {
  const int64_t F = a.T * a.k;
  const int nblk = static_cast<int>((F + kDispatchChunk - 1) / kDispatchChunk);
  cudaError_t err = cudaSuccess;
  if (nblk > 0 && a.sync_ctr != nullptr && fused_dispatch_ok(a.N, nblk, num_sms)) {
    err = cudaMemsetAsync(a.sync_ctr, 0, sizeof(unsigned int), st);
    if (err != cudaSuccess) return err;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(nblk);
    cfg.blockDim = dim3(kDispatchChunk);
    cfg.dynamicSmemBytes = fused_smem_bytes(a.N);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;  // blocks wait on one another once
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    err = cudaLaunchKernelEx(&cfg, dispatch_fused_kernel, a.idx, F, a.k, a.N, a.T, a.n_shared,
                             a.tile_rows, a.blk_hist, a.counts, a.offsets, a.perm, a.inv, a.tiles,
                             a.num_tiles, a.stiles1, a.stiles2, a.sync_ctr, a.status, a.ready);
    if (err != cudaSuccess) return err;
  } else {
    if (nblk > 0) {
      err = launch_pdl(hist_kernel, dim3(nblk), dim3(kDispatchChunk), 0, st, 1, a.idx, F, a.k,
                       a.N, a.blk_hist, a.status);
      if (err != cudaSuccess) return err;
    }
    err = launch_pdl(scan_kernel, dim3(1), dim3(1024), 0, st, 1, a.blk_hist, nblk, a.N, a.T,
                     a.n_shared, a.tile_rows, a.counts, a.offsets, a.tiles, a.num_tiles, a.stiles1,
                     a.stiles2, a.ready);
    if (err != cudaSuccess) return err;
    if (nblk > 0) {
      err = launch_pdl(place_kernel, dim3(nblk), dim3(kDispatchChunk), 0, st, 1, a.idx, F, a.k,
                       a.N, static_cast<const int32_t*>(a.blk_hist), a.perm, a.inv);
      if (err != cudaSuccess) return err;
    }
  }
  if (nblk > 0 && a.xperm != nullptr) {
    const int row_vec = a.d * a.esz / 16;
    int64_t warps_needed = F;
    int64_t blocks = (warps_needed + 7) / 8;
    const int64_t cap = static_cast<int64_t>(num_sms) * 8;
    if (blocks > cap) blocks = cap;
    err = launch_pdl(gather_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, 1,
                     static_cast<const uint4*>(a.h), static_cast<const int32_t*>(a.perm),
                     static_cast<const int32_t*>(a.offsets + a.N), a.k, row_vec,
                     static_cast<uint4*>(a.xperm));
    if (err != cudaSuccess) return err;
  }
  return cudaSuccess;
}

cudaError_t launch_dispatch_from_hist(const DispatchArgs& a, const int32_t* hist, int split,
                                      cudaStream_t st) {
  const int tiles_r = static_cast<int>((a.T + kTileM - 1) / kTileM);
  if (tiles_r == 0) return cudaSuccess;
  if (a.N % 4 != 0 || a.k > kMaxTopK || hist == nullptr || split < 1) return cudaErrorInvalidValue;
  const size_t smem = hist_smem_bytes(a.N);
  cudaError_t err = cudaFuncSetAttribute(dispatch_hist_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
  if (err != cudaSuccess) return err;
  return launch_pdl(dispatch_hist_kernel, dim3(tiles_r), dim3(kHistBlock), smem, st, 1, a.idx,
                    a.T, a.k, a.N, a.n_shared, a.tile_rows, hist, tiles_r * split, split,
                    a.counts, a.offsets, a.perm, a.inv, a.tiles, a.num_tiles, a.stiles1,
                    a.stiles2, a.ready);
}

cudaError_t launch_combine(const CombineArgs& a, int num_sms, cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  const int32_t* status = a.status;
  int64_t blocks = (a.T + 7) / 8;
  const int64_t cap = static_cast<int64_t>(num_sms) * 8;
  if (blocks > cap) blocks = cap;
  const dim3 grid(static_cast<unsigned>(blocks)), block(256);
  if (a.bf16) {
    auto* Y = static_cast<const __nv_bfloat16*>(a.Y);
    auto* Ys = static_cast<const __nv_bfloat16*>(a.Ys);
    auto* out = static_cast<__nv_bfloat16*>(a.out);
    auto* res = static_cast<const __nv_bfloat16*>(a.residual);
    const CombineRing ring = combine_ring(a.k, a.d, a.n_shared, res != nullptr);
    const bool aligned = ((reinterpret_cast<uintptr_t>(res) | reinterpret_cast<uintptr_t>(Y) |
                           reinterpret_cast<uintptr_t>(Ys)) & 15u) == 0;
    if (ring.slots >= 3 && a.k <= kCbMaxK && a.n_shared <= 32 && (a.d * 2) % 16 == 0 &&
        aligned) {
      const int ctas = static_cast<int>(a.T < num_sms ? a.T : num_sms);
      auto* kern = combine_bulk_kernel;
      const cudaError_t err =
          cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kCbSmemBytes);
      if (err != cudaSuccess) return err;
      return launch_pdl(kern, dim3(ctas), dim3(kCbThreads), kCbSmemBytes, st, 1, Y, Ys, a.inv,
                        a.gates, a.T, a.k, a.d, a.n_shared, res, out, a.status);
    }
    // (bf16 layers have k <= 8, checked at the ABI)
    return launch_pdl(combine_kernel<__nv_bfloat16, 8, 8>, grid, block, 0, st, 1, Y, Ys, a.inv,
                      a.gates, a.T, a.k, a.d, a.n_shared, res, out, status);
  }
  auto* Y = static_cast<const float*>(a.Y);
  auto* Ys = static_cast<const float*>(a.Ys);
  auto* out = static_cast<float*>(a.out);
  auto* res = static_cast<const float*>(a.residual);
  return a.k <= 8 ? launch_pdl(combine_kernel<float, 4, 8>, grid, block, 0, st, 1, Y, Ys, a.inv,
                               a.gates, a.T, a.k, a.d, a.n_shared, res, out, status)
                  : launch_pdl(combine_kernel<float, 4, 32>, grid, block, 0, st, 1, Y, Ys, a.inv,
                               a.gates, a.T, a.k, a.d, a.n_shared, res, out, status);
}

}  // namespace pr2
