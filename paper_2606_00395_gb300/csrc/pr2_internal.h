// Host-side interface between the C ABI (api.cu) and the kernel launchers of each .cu file.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "pr2.h"

namespace pr2 {

// Launch with programmatic stream serialization (the kernel calls pdl_wait() before touching
// global memory) and, for cluster > 1, a 1-D thread-block cluster.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, unsigned cluster, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  unsigned n = 1;
  if (cluster > 1) {
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = cluster;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    n = 2;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// One M-tile of a grouped GEMM: rows [a_row0, a_row0 + rows) of the A operand, multiplied by
// the weights of `expert`, written to rows [out_row0, out_row0 + rows) of the output.
struct TileEntry {
  int32_t expert, a_row0, rows, out_row0;
};

constexpr int kTileM = 128;         // rows per M-tile (one tcgen05 M=128 accumulator)
constexpr int kDispatchChunk = 256; // flat slots per dispatch block (8 warps x 32 lanes)
constexpr int kMaxTopK = 8;         // slots kept by the tensor-core routing epilogue
constexpr int kMaxTopKSimt = 32;    // slots of the fp32 SIMT routing kernel
constexpr int kMaxExperts = 256;    // routed experts supported by the routing kernels
constexpr int kMaxExpertsDispatch = 1024;
constexpr int kRouteMaxSplit = 8;   // most CTAs splitting one routing tile (histogram rows)

// ---- routing (route_simt.cu, route_tc.cu) -------------------------------------------------
cudaError_t launch_route_simt(const pr2_dims& dm, bool predict, const float* h, const float* W,
                              const float* Wp, const int32_t* idx_in, int32_t* idx_out,
                              float* gates, float* logits_or_probs, int64_t* near_tie,
                              int32_t* status, cudaStream_t st);

// Modes of the tensor-core routing kernel (route_tc.cu).
enum RouteMode : int {
  kModeReplay = 0,   // rho = Softmax(h W^T), gates = rho[idx_in]
  kModePredict = 1,  // z = h W^T + h W_p^T, top-k, gates = rho_hat[idx]
  kModeLoss = 2,     // predictive loss: z = p_old + h_old W_p^T against a teacher rho
};

struct RouteTcArgs {
  int T, d, N, k;
  const int32_t* idx_in;   // replay: cached route
  int32_t* idx_out;        // predict: route out
  float* gates;
  float* logits_or_probs;  // predict: p_old [T,N]; replay: rho [T,N]; nullable
  int64_t* near_tie;
  int32_t* status;
  int norm;                // PR2_F_NORMALIZE_TOPK: gates divided by their sum over the route
  int compact;             // 1: half the pipeline stages, so two CTAs share an SM (split 1)
  int late_wait;           // 1: the inputs are known ready; wait for the previous kernel only
                           // before exiting (the launch overlaps it; see pr2_moe_replay_forward)
  int32_t* hist;           // predict, nullable: [CTAs][N] experts of each CTA's finished rows
                           // (CTA tile * split + rank), read by dispatch_from_hist
  // kModeLoss only (h = h_old, W = W_p)
  const float* p_old;      // [T, N] cached router logits
  const float* rho;        // [T_rho, N] teacher probabilities
  const int32_t* pos;      // [T] teacher row of each cached row (nullable: row t)
  int64_t T_rho;
  int delta;               // 1: delta-matching variant
  float* kl_tok;           // [T] per-token KL
  uint16_t* gt;            // [N, Tpad] bf16 bits of dKL/dz, transposed; rows t >= T hold 0
  int Tpad;                // multiple of 128, >= T
};
// CTAs of the cluster that splits K for one 128-token tile (1 = no split).
int route_split(int T, int N, int d, int mode, int num_sms);
// Whether a launch over T tokens runs two CTAs per SM, each with half the pipeline stages and
// no K split: when the 128-token tiles outnumber the SMs, so that one CTA's loads and finishing
// overlap the other's MMAs instead of the tiles running as a second wave.
bool route_compact(int T, int N, int mode, int num_sms);
cudaError_t launch_route_tc(int mode, const CUtensorMap& tm_h, const CUtensorMap& tm_w,
                            const CUtensorMap& tm_wp, const RouteTcArgs& a, int split,
                            cudaStream_t st);

// ---- dispatch and combine (dispatch.cu) ----------------------------------------------------
struct DispatchArgs {
  const int32_t* idx;
  int64_t T;
  int k, N, d, esz, n_shared;
  int32_t* blk_hist;     // [nblk, N] block histograms, scanned in place into block bases
  int32_t* counts;       // [N]
  int32_t* offsets;      // [N+1]
  int32_t* perm;         // [T*k]
  int32_t* inv;          // [T*k]
  TileEntry* tiles;      // [max_mtiles]
  int32_t* num_tiles;    // [2]: routed M-tiles, shared M-tiles
  TileEntry* stiles1;    // [n_shared * ceil(T/128)] gate/up GEMM of the shared experts
  TileEntry* stiles2;    // same, down GEMM
  const void* h;
  void* xperm;           // [T*k, d] permuted copy of h (fp32 path); nullptr: no gather launch
  int32_t* status;
  unsigned int* sync_ctr;  // grid-barrier counter of the fused dispatch (zeroed per call)
  int32_t* ready;          // [max_mtiles] per M-tile counters of the fused GEMM, cleared here
                           // (nullable)
  int tile_rows;           // most rows of one routed tile (an expert's rows are split evenly)
};
cudaError_t launch_dispatch(const DispatchArgs& a, int num_sms, cudaStream_t st);
// Dispatch of a route the routing kernel just wrote (every slot valid), from the per-CTA
// expert histograms it wrote: hist rows [tile * split + r], `split` rows per 128-token tile.
// No histogram pass and no grid barrier, so it is an ordinary launch behind the routing kernel.
cudaError_t launch_dispatch_from_hist(const DispatchArgs& a, const int32_t* hist, int split,
                                      cudaStream_t st);

struct CombineArgs {
  const void* Y;        // [T*k, d] expert outputs in dispatch order
  const void* Ys;       // [n_shared, T, d] shared-expert outputs (nullable)
  const int32_t* inv;   // [T*k]
  const float* gates;   // [T*k]
  int64_t T;
  int k, d, n_shared, bf16;
  void* out;            // [T, d]
  const void* residual; // [T, d] added to the sum (nullable); may equal `out`
  int32_t* status;      // PR2_STATUS_TIMEOUT if a bounded wait ran out (nullable)
};
cudaError_t launch_combine(const CombineArgs& a, int num_sms, cudaStream_t st);

// ---- grouped expert GEMMs (expert_tc.cu, expert_simt.cu) -----------------------------------
struct GemmArgs {
  const TileEntry* tiles;
  const int32_t* num_tiles;  // device count of valid entries in `tiles`
  int max_tiles;             // host bound on that count
  int K;                     // reduction length
  int n_out;                 // output columns
  int b_rows_per_expert;     // rows of one expert's weight matrix (m for gate/up, d for down)
  void* out;                 // [rows, n_out]
  int32_t* status;
  // Gathered A (gate/up GEMM of the routed experts): row r of a tile is token perm[r] / k of
  // `a_src` [T, K] instead of row r of a permuted copy.  Unused when the A operand comes from
  // the tensor map.
  const void* a_src;
  const int32_t* perm;
  int k;
};
// Launch kinds of the tcgen05 grouped GEMM (expert_tc.cu).  Phase 0 is a gate/up GEMM with the
// SwiGLU epilogue (weights tm_b0 = gate, tm_b1 = up), phase 1 a down GEMM (weights tm_b2).
enum ExpertKind : int {
  kExpertGateUpTma = 1,     // phase 0, A rows from tm_a (shared experts: rows of h)
  kExpertDown = 2,          // phase 1, A rows from tm_a
  kExpertFused = 3,         // phase 0, A rows gathered from p[0].a_src through p[0].perm,
                            // then phase 1 (A = p[0].out through tm_a), in one cooperative
                            // launch (the routed experts)
};
struct MlpArgs {
  GemmArgs p[2];     // arguments of phase 0 and phase 1 (only the launched phases are read)
  int32_t* ready;    // kExpertFused: per M-tile count of finished gate/up epilogue warps,
                     // zero on entry (dispatch clears it)
};
cudaError_t launch_expert_tc(ExpertKind kind, const CUtensorMap& tm_a, const CUtensorMap& tm_b0,
                             const CUtensorMap& tm_b1, const CUtensorMap& tm_b2,
                             const MlpArgs& a, int num_sms, cudaStream_t st);
cudaError_t launch_expert_simt(bool swiglu, const float* A, const float* Wb0, const float* Wb1,
                               const GemmArgs& g, cudaStream_t st);

// ---- predictive loss gradient (predictor.cu) ---------------------------------------------
// grad_Wp = (1/T_c) G^T h_old with G = dKL/dz.  bf16: split-K tcgen05 GEMM over tokens into
// `partial` [split, N, d] fp32, then a fixed-order reduction.  fp32: SIMT kernels.
struct GradArgs {
  int N, d, Tc, Tpad;
  int split;              // token-block split of the GEMM: CTAs per cluster (1, 2, 4 or 8)
  float* partial;         // [split, N, d] fp32 split partials (split > 1)
  float* grad;            // [N, d]
  const float* kl_tok;    // [Tc]
  float* loss;            // [1]
  int32_t* status;
};
constexpr int kLossMaxSplit = 8;
int loss_grad_split(int N, int d, int Tpad, int num_sms);
// Rows (experts) and columns (d) of the gradient rounded up to whole output tiles.
int64_t loss_grad_rows(int N);
int64_t loss_grad_cols(int d);
cudaError_t launch_loss_grad_tc(const CUtensorMap& tm_gt, const CUtensorMap& tm_h,
                                const GradArgs& g, cudaStream_t st);
// fp32 path: the loss from the per-token KL (the bf16 gradient kernel sums it itself).
cudaError_t launch_loss_finish(const GradArgs& g, cudaStream_t st);
// fp32 path: per-token KL and G [Tc, N] (row-major), then the gradient.
cudaError_t launch_loss_simt(const float* h_old, const float* p_old, const float* Wp,
                             const float* rho, int64_t T_rho, const int32_t* pos, int delta,
                             int Tc, int d, int N, float* kl_tok, float* G, int32_t* status,
                             cudaStream_t st);
cudaError_t launch_loss_grad_simt(const float* G, const float* h_old, int Tc, int d, int N,
                                  float* grad, cudaStream_t st);

// ---- diagnostics and feature cache (diagnostics.cu) ---------------------------------------
cudaError_t launch_diagnostics(const float* rho, const int32_t* cached, int64_t T, int N, int k,
                               int64_t* hist, int64_t* overlap_sum, int num_sms,
                               cudaStream_t st);
cudaError_t launch_feature_cache(const void* h, const float* logits, int64_t T, int64_t Tc,
                                 int d, int N, int esz, int32_t* pos, void* cache_h,
                                 float* cache_p, int num_sms, cudaStream_t st);

// ---- self test (api.cu) --------------------------------------------------------------------
cudaError_t launch_wait_selftest(int32_t* status, int64_t timeout_ns, cudaStream_t st);

}  // namespace pr2
