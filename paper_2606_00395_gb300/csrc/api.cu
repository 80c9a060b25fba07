// C ABI of the Pr^2 MoE layer (declared in include/pr2.h): argument validation, workspace
// layout, TMA descriptor encoding and the launch sequence of each entry point.
#include <cudaTypedefs.h>

#include <cstring>

#include "pr2_device.cuh"
#include "pr2_internal.h"

namespace pr2 {
namespace {

// ---- TMA descriptor encoding through the driver entry point (no libcuda link needed) ------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// 2-D bf16 tensor [outer, inner] (row-major, row pitch = inner elements), 128-byte swizzled
// boxes of box_inner x box_outer elements.
bool make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                    uint32_t box_inner, uint32_t box_outer) {
  auto fn = encode_fn();
  if (fn == nullptr) return false;
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {inner * 2};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int num_sms_of_current_device() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
  return n;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

pr2_status check_dims(const pr2_dims* dm) {
  if (dm == nullptr) return PR2_ERR_INVALID_ARG;
  if (dm->T < 0 || dm->d <= 0 || dm->N <= 0 || dm->k <= 0 || dm->k > dm->N || dm->m <= 0 ||
      dm->n_shared < 0)
    return PR2_ERR_INVALID_ARG;
  if (dm->dtype != PR2_FP32 && dm->dtype != PR2_BF16) return PR2_ERR_INVALID_ARG;
  if (dm->flags & ~(PR2_F_SYNC_STATUS | PR2_F_DELTA_LOSS | PR2_F_NORMALIZE_TOPK))
    return PR2_ERR_INVALID_ARG;  // an unknown flag is a caller error, not a no-op
  if (dm->T * static_cast<int64_t>(dm->k) > (int64_t{1} << 30)) return PR2_ERR_UNSUPPORTED;
  if (dm->N > kMaxExperts) return PR2_ERR_UNSUPPORTED;
  if (dm->dtype == PR2_FP32) {
    if (dm->k > kMaxTopKSimt || dm->d % 4 != 0) return PR2_ERR_UNSUPPORTED;
  } else {
    if (dm->k > kMaxTopK || dm->d % 64 != 0 || dm->m % 64 != 0 || dm->N % 16 != 0)
      return PR2_ERR_UNSUPPORTED;
  }
  return PR2_OK;
}

size_t esize(const pr2_dims& dm) { return dm.dtype == PR2_FP32 ? 4 : 2; }

// ---- workspace layout of pr2_moe_forward ----------------------------------------------------
struct Workspace {
  int32_t* status;
  int32_t* blk_hist;
  int32_t* counts;
  int32_t* offsets;
  int32_t* perm;
  int32_t* inv;
  int32_t* num_tiles;
  unsigned int* sync_ctr;
  int32_t* ready;
  TileEntry* tiles;
  TileEntry* stiles1;
  TileEntry* stiles2;
  int32_t* route_hist;  // per-CTA expert histograms of the rollout routing (pr2_moe_rollout_forward)
  void* xperm;
  void* hbuf;
  void* ybuf;
  void* hs;
  void* ys;
  int nblk, max_tiles, shared_tiles;
  size_t total;
};

Workspace carve(const pr2_dims& dm, uint8_t* base) {
  Workspace w{};
  size_t off = 0;
  auto take = [&](size_t bytes) -> uint8_t* {
    uint8_t* p = base ? base + off : nullptr;
    off += (bytes + 255) & ~size_t{255};
    return p;
  };
  const int64_t F = dm.T * dm.k;
  const size_t es = esize(dm);
  w.nblk = static_cast<int>((F + kDispatchChunk - 1) / kDispatchChunk);
  w.max_tiles = static_cast<int>(F / kTileM + dm.N + 1);
  const int mt_T = static_cast<int>((dm.T + kTileM - 1) / kTileM);
  w.shared_tiles = dm.n_shared * mt_T;
  w.status = reinterpret_cast<int32_t*>(take(sizeof(int32_t)));
  w.blk_hist = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * (size_t)w.nblk * dm.N));
  w.counts = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * dm.N));
  w.offsets = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * (dm.N + 1)));
  w.perm = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * F));
  w.inv = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * F));
  w.num_tiles = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * 2));
  w.sync_ctr = reinterpret_cast<unsigned int*>(take(sizeof(unsigned int)));
  w.ready = reinterpret_cast<int32_t*>(take(sizeof(int32_t) * w.max_tiles));
  w.tiles = reinterpret_cast<TileEntry*>(take(sizeof(TileEntry) * w.max_tiles));
  w.stiles1 = reinterpret_cast<TileEntry*>(take(sizeof(TileEntry) * (w.shared_tiles + 1)));
  w.stiles2 = reinterpret_cast<TileEntry*>(take(sizeof(TileEntry) * (w.shared_tiles + 1)));

  // permuted copy of h: only the fp32 path reads it; the bf16 gate/up GEMM gathers from h
  w.xperm = dm.dtype == PR2_FP32 ? take(es * F * dm.d) : nullptr;
  // H [Tk, m].  The rollout routing's per-CTA histograms share its first bytes: dispatch reads
  // them before the gate/up GEMM (which waits for dispatch) writes H.
  const size_t hist_bytes = sizeof(int32_t) * (size_t)mt_T * kRouteMaxSplit * dm.N;
  const size_t h_bytes = es * F * dm.m;
  w.hbuf = take(h_bytes > hist_bytes ? h_bytes : hist_bytes);
  w.route_hist = static_cast<int32_t*>(w.hbuf);
  w.ybuf = take(es * F * dm.d);
  w.hs = take(es * dm.n_shared * dm.T * dm.m);
  w.ys = take(es * dm.n_shared * dm.T * dm.d);
  w.total = off;
  return w;
}

pr2_status finish(cudaError_t err, uint32_t flags, int32_t* status_dev, cudaStream_t st) {
  if (err != cudaSuccess) return PR2_ERR_CUDA;
  if (flags & PR2_F_SYNC_STATUS) {
    if (status_dev == nullptr) return PR2_ERR_INVALID_ARG;
    int32_t hst = 0;
    if (cudaMemcpyAsync(&hst, status_dev, sizeof(hst), cudaMemcpyDeviceToHost, st) != cudaSuccess)
      return PR2_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return PR2_ERR_CUDA;
    if (hst & PR2_STATUS_TIMEOUT) return PR2_ERR_TIMEOUT;
    if (hst & PR2_STATUS_BAD_INDEX) return PR2_ERR_BAD_INDEX;
  }
  return PR2_OK;
}

pr2_status route_common(const pr2_dims* dims, bool predict, const void* h, const void* W,
                        const void* Wp, const int32_t* idx_in, int32_t* idx_out, float* gates,
                        float* aux, int64_t* near_tie, int32_t* status_dev, void* stream,
                        bool late_wait = false, int32_t* hist = nullptr,
                        int* split_out = nullptr) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  const pr2_dims& dm = *dims;
  if (dm.T == 0) return PR2_OK;  // nothing to route; empty tensors may have NULL data
  if (h == nullptr || W == nullptr || gates == nullptr) return PR2_ERR_INVALID_ARG;
  if (predict && (Wp == nullptr || idx_out == nullptr)) return PR2_ERR_INVALID_ARG;
  if (!predict && idx_in == nullptr) return PR2_ERR_INVALID_ARG;
  if ((dm.flags & PR2_F_SYNC_STATUS) && status_dev == nullptr) return PR2_ERR_INVALID_ARG;
  if (!aligned16(h) || !aligned16(W) || (Wp && !aligned16(Wp)) || (aux && !aligned16(aux)))
    return PR2_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t err;
  if (dm.dtype == PR2_FP32) {
    err = launch_route_simt(dm, predict, static_cast<const float*>(h),
                            static_cast<const float*>(W), static_cast<const float*>(Wp), idx_in,
                            idx_out, gates, aux, near_tie, status_dev, st);
  } else {
    if (dm.T > (int64_t{1} << 30)) return PR2_ERR_UNSUPPORTED;
    const int num_sms = num_sms_of_current_device();
    if (num_sms <= 0) return PR2_ERR_CUDA;
    const int mode = predict ? kModePredict : kModeReplay;
    const bool compact = route_compact(static_cast<int>(dm.T), dm.N, mode, num_sms);
    const int split =
        compact ? 1 : route_split(static_cast<int>(dm.T), dm.N, dm.d, mode, num_sms);
    CUtensorMap tm_h, tm_w, tm_wp;
    if (!make_tmap_bf16(&tm_h, h, dm.d, dm.T, 64, kTileM) ||
        !make_tmap_bf16(&tm_w, W, dm.d, dm.N, 64, dm.N))
      return PR2_ERR_CUDA;
    if (predict) {
      if (!make_tmap_bf16(&tm_wp, Wp, dm.d, dm.N, 64, dm.N)) return PR2_ERR_CUDA;
    } else {
      tm_wp = tm_w;
    }
    RouteTcArgs a{};
    a.T = static_cast<int>(dm.T);
    a.d = dm.d;
    a.N = dm.N;
    a.k = dm.k;
    a.idx_in = idx_in;
    a.idx_out = idx_out;
    a.gates = gates;
    a.logits_or_probs = aux;
    a.near_tie = near_tie;
    a.status = status_dev;
    a.norm = (dm.flags & PR2_F_NORMALIZE_TOPK) ? 1 : 0;
    a.compact = compact ? 1 : 0;
    a.late_wait = late_wait ? 1 : 0;
    a.hist = predict ? hist : nullptr;
    if (split_out != nullptr) *split_out = split;
    err = launch_route_tc(mode, tm_h, tm_w, tm_wp, a, split, st);
  }
  return finish(err, dm.flags, status_dev, st);
}

// ---- workspace of pr2_predictor_loss ---------------------------------------------------------
struct LossWorkspace {
  int32_t* status;
  uint16_t* gt;     // bf16: [N, Tpad] dKL/dz transposed
  float* G;         // fp32: [Tc, N] dKL/dz
  float* kl;        // [Tpad] per-token KL when the caller passes none
  float* partial;   // bf16: split partial tiles of the gradient, [kLossMaxSplit, Npad, dpad]
  int Tpad;
  size_t total;
};

LossWorkspace carve_loss(const pr2_dims& dm, uint8_t* base) {
  LossWorkspace w{};
  size_t off = 0;
  auto take = [&](size_t bytes) -> uint8_t* {
    uint8_t* p = base ? base + off : nullptr;
    off += (bytes + 255) & ~size_t{255};
    return p;
  };
  w.Tpad = static_cast<int>((dm.T + kTileM - 1) / kTileM) * kTileM;
  w.status = reinterpret_cast<int32_t*>(take(sizeof(int32_t)));
  w.kl = reinterpret_cast<float*>(take(sizeof(float) * (size_t)(w.Tpad > 0 ? w.Tpad : 1)));
  if (dm.dtype == PR2_BF16) {
    w.gt = reinterpret_cast<uint16_t*>(take(sizeof(uint16_t) * (size_t)dm.N * w.Tpad));
    w.partial = reinterpret_cast<float*>(
        take(sizeof(float) * (size_t)kLossMaxSplit * loss_grad_rows(dm.N) * loss_grad_cols(dm.d)));
  } else {
    w.G = reinterpret_cast<float*>(take(sizeof(float) * (size_t)dm.T * dm.N));
  }
  w.total = off;
  return w;
}

}  // namespace
}  // namespace pr2

using namespace pr2;

extern "C" {

pr2_status pr2_route_predict(const pr2_dims* dims, const void* h, const void* W_router,
                             const void* W_pred, int32_t* idx, float* gates, float* logits_old,
                             int64_t* near_tie, int32_t* status_dev, void* stream) {
  return route_common(dims, true, h, W_router, W_pred, nullptr, idx, gates, logits_old, near_tie,
                      status_dev, stream);
}

pr2_status pr2_route_replay(const pr2_dims* dims, const void* h, const void* W_router,
                            const int32_t* idx, float* gates, float* probs, int32_t* status_dev,
                            void* stream) {
  return route_common(dims, false, h, W_router, nullptr, idx, nullptr, gates, probs, nullptr,
                      status_dev, stream);
}

size_t pr2_predictor_loss_workspace_bytes(const pr2_dims* dims) {
  if (check_dims(dims) != PR2_OK) return 0;
  return carve_loss(*dims, nullptr).total;
}

pr2_status pr2_predictor_loss(const pr2_dims* dims, const void* h_old, const float* p_old,
                              const void* W_pred, const float* rho, int64_t T_rho,
                              const int32_t* pos, float* loss, float* kl_tok, float* grad_Wp,
                              void* workspace, size_t ws_bytes, int32_t* status_dev,
                              void* stream) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  const pr2_dims& dm = *dims;
  if (dm.T > (int64_t{1} << 30) - kTileM) return PR2_ERR_UNSUPPORTED;
  if (loss == nullptr || grad_Wp == nullptr || W_pred == nullptr) return PR2_ERR_INVALID_ARG;
  if (dm.T > 0 && (h_old == nullptr || p_old == nullptr || rho == nullptr || T_rho < 1))
    return PR2_ERR_INVALID_ARG;
  if ((dm.flags & PR2_F_SYNC_STATUS) && status_dev == nullptr) return PR2_ERR_INVALID_ARG;
  const void* al[] = {h_old, p_old, W_pred, rho, loss, kl_tok, grad_Wp};
  for (const void* p : al)
    if (p != nullptr && !aligned16(p)) return PR2_ERR_INVALID_ARG;
  const LossWorkspace probe = carve_loss(dm, nullptr);
  if (workspace == nullptr || ws_bytes < probe.total ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return PR2_ERR_WORKSPACE;
  const LossWorkspace w = carve_loss(dm, static_cast<uint8_t*>(workspace));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int32_t* status = status_dev ? status_dev : w.status;
  cudaError_t err = cudaSuccess;
  if (status_dev == nullptr) err = cudaMemsetAsync(w.status, 0, sizeof(int32_t), st);
  if (err == cudaSuccess && dm.T == 0) {  // no cached token: loss 0, gradient 0
    err = cudaMemsetAsync(loss, 0, sizeof(float), st);
    if (err == cudaSuccess)
      err = cudaMemsetAsync(grad_Wp, 0, sizeof(float) * (size_t)dm.N * dm.d, st);
    return finish(err, dm.flags, status_dev, st);
  }
  if (err != cudaSuccess) return PR2_ERR_CUDA;
  const int Tc = static_cast<int>(dm.T);
  float* kl = kl_tok ? kl_tok : w.kl;
  const int delta = (dm.flags & PR2_F_DELTA_LOSS) ? 1 : 0;
  GradArgs g{dm.N, dm.d, Tc, w.Tpad, 1, w.partial, grad_Wp, kl, loss, status};
  if (dm.dtype == PR2_FP32) {
    err = launch_loss_simt(static_cast<const float*>(h_old), p_old,
                           static_cast<const float*>(W_pred), rho, T_rho, pos, delta, Tc, dm.d,
                           dm.N, kl, w.G, status, st);
    if (err == cudaSuccess)
      err = launch_loss_grad_simt(w.G, static_cast<const float*>(h_old), Tc, dm.d, dm.N,
                                  grad_Wp, st);
    if (err == cudaSuccess) err = launch_loss_finish(g, st);
    return finish(err, dm.flags, status_dev, st);
  }
  const int num_sms = num_sms_of_current_device();
  if (num_sms <= 0) return PR2_ERR_CUDA;
  CUtensorMap tm_h, tm_w, tm_gt, tm_hmn;
  if (!make_tmap_bf16(&tm_h, h_old, dm.d, dm.T, 64, kTileM) ||
      !make_tmap_bf16(&tm_w, W_pred, dm.d, dm.N, 64, dm.N) ||
      !make_tmap_bf16(&tm_gt, w.gt, w.Tpad, dm.N, 64, kTileM) ||
      !make_tmap_bf16(&tm_hmn, h_old, dm.d, dm.T, 64, 64))
    return PR2_ERR_CUDA;
  RouteTcArgs a{};
  a.T = Tc;
  a.d = dm.d;
  a.N = dm.N;
  a.k = dm.k;
  a.status = status;
  a.p_old = p_old;
  a.rho = rho;
  a.pos = pos;
  a.T_rho = T_rho;
  a.delta = delta;
  a.kl_tok = kl;
  a.gt = w.gt;
  a.Tpad = w.Tpad;
  const int split = route_split(Tc, dm.N, dm.d, kModeLoss, num_sms);
  err = launch_route_tc(kModeLoss, tm_h, tm_w, tm_w, a, split, st);
  g.split = loss_grad_split(dm.N, dm.d, w.Tpad, num_sms);
  if (err == cudaSuccess) err = launch_loss_grad_tc(tm_gt, tm_hmn, g, st);
  return finish(err, dm.flags, status_dev, st);
}

pr2_status pr2_route_diagnostics(const pr2_dims* dims, const float* rho, const int32_t* idx_cached,
                                 int64_t* hist, int64_t* overlap_sum, void* stream) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  const pr2_dims& dm = *dims;
  if (dm.k > kMaxTopKSimt) return PR2_ERR_UNSUPPORTED;
  if (hist == nullptr || overlap_sum == nullptr) return PR2_ERR_INVALID_ARG;
  if (dm.T == 0) return PR2_OK;
  if (rho == nullptr || idx_cached == nullptr || !aligned16(rho)) return PR2_ERR_INVALID_ARG;
  const int num_sms = num_sms_of_current_device();
  if (num_sms <= 0) return PR2_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return finish(launch_diagnostics(rho, idx_cached, dm.T, dm.N, dm.k, hist, overlap_sum, num_sms,
                                   st),
                dm.flags & ~PR2_F_SYNC_STATUS, nullptr, st);
}

pr2_status pr2_feature_cache_write(const pr2_dims* dims, int64_t T_c, const void* h,
                                   const float* logits_old, int32_t* pos, void* cache_h,
                                   float* cache_p, void* stream) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  const pr2_dims& dm = *dims;
  if (T_c < 0 || T_c > dm.T || dm.T > (int64_t{1} << 31) - 1) return PR2_ERR_INVALID_ARG;
  if (T_c == 0) return PR2_OK;
  if (h == nullptr || pos == nullptr || cache_h == nullptr) return PR2_ERR_INVALID_ARG;
  if ((logits_old == nullptr) != (cache_p == nullptr)) return PR2_ERR_INVALID_ARG;
  if (!aligned16(h) || !aligned16(cache_h)) return PR2_ERR_INVALID_ARG;
  const int esz = static_cast<int>(esize(dm));
  if ((static_cast<int64_t>(dm.d) * esz) % 16 != 0) return PR2_ERR_UNSUPPORTED;
  const int num_sms = num_sms_of_current_device();
  if (num_sms <= 0) return PR2_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return finish(launch_feature_cache(h, logits_old, dm.T, T_c, dm.d, dm.N, esz, pos, cache_h,
                                     cache_p, num_sms, st),
                dm.flags & ~PR2_F_SYNC_STATUS, nullptr, st);
}

size_t pr2_moe_workspace_bytes(const pr2_dims* dims) {
  if (check_dims(dims) != PR2_OK) return 0;
  return carve(*dims, nullptr).total;
}

}  // extern "C"

namespace pr2 {
namespace {

// Replay routing run inside the layer forward (pr2_moe_replay_forward): the current router and
// the gates / probabilities it writes.
struct ReplayRoute {
  const void* W_router;
  float* probs;
};

// The layer forward of pr2_moe_forward; `residual` (nullable, [T, d] in the layer dtype, may
// alias `out`) is added to the combined output.  With `replay`, the replay gates of the route
// `idx` are computed into `gates` after the expert GEMMs and before the combine, which is the
// only step that reads them.
// Host-side checks of pr2_moe_forward's arguments (dims already checked, T > 0).
pr2_status forward_args(const pr2_dims& dm, const void* h, const int32_t* idx, const float* gates,
                        const void* W_gate, const void* W_up, const void* W_down,
                        const void* Ws_gate, const void* Ws_up, const void* Ws_down, void* out,
                        void* workspace, size_t ws_bytes) {
  if (h == nullptr || idx == nullptr || gates == nullptr || W_gate == nullptr ||
      W_up == nullptr || W_down == nullptr || out == nullptr)
    return PR2_ERR_INVALID_ARG;
  if (dm.n_shared > 0 && (Ws_gate == nullptr || Ws_up == nullptr || Ws_down == nullptr))
    return PR2_ERR_INVALID_ARG;
  if (dm.n_shared == 0 && (Ws_gate != nullptr || Ws_up != nullptr || Ws_down != nullptr))
    return PR2_ERR_INVALID_ARG;
  const void* ptrs[] = {h, W_gate, W_up, W_down, out};
  for (const void* p : ptrs)
    if (!aligned16(p)) return PR2_ERR_INVALID_ARG;
  if (dm.n_shared > 0 && (!aligned16(Ws_gate) || !aligned16(Ws_up) || !aligned16(Ws_down)))
    return PR2_ERR_INVALID_ARG;
  const Workspace probe = carve(dm, nullptr);
  if (workspace == nullptr || ws_bytes < probe.total ||
      (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
    return PR2_ERR_WORKSPACE;
  return PR2_OK;
}

// Per-CTA expert histograms that the rollout routing kernel wrote for this layer's route
// (pr2_moe_rollout_forward): dispatch then needs no histogram pass of its own.
struct RouteHist {
  const int32_t* hist;
  int split;
};

pr2_status moe_forward_impl(const pr2_dims* dims, const void* h, const int32_t* idx,
                            const float* gates, const void* W_gate, const void* W_up,
                            const void* W_down, const void* Ws_gate, const void* Ws_up,
                            const void* Ws_down, void* out, const void* residual,
                            int32_t* counts, int32_t* perm, void* workspace, size_t ws_bytes,
                            int32_t* status_dev, const pr2_stage_events* events,
                            void* stream, const ReplayRoute* replay = nullptr,
                            const RouteHist* rhist = nullptr) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  const pr2_dims& dm = *dims;
  if (dm.T == 0) return PR2_OK;  // empty layer: nothing to write
  s = forward_args(dm, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down, out,
                   workspace, ws_bytes);
  if (s != PR2_OK) return s;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const Workspace w = carve(dm, static_cast<uint8_t*>(workspace));
  int32_t* status = status_dev ? status_dev : w.status;
  const int num_sms = num_sms_of_current_device();
  if (num_sms <= 0) return PR2_ERR_CUDA;
  cudaError_t err = cudaSuccess;
  if (status_dev == nullptr) err = cudaMemsetAsync(w.status, 0, sizeof(int32_t), st);
  if (err != cudaSuccess) return PR2_ERR_CUDA;
  auto mark = [&](void* ev) {
    if (ev != nullptr && err == cudaSuccess)
      err = cudaEventRecord(static_cast<cudaEvent_t>(ev), st);
  };
  mark(events ? events->start : nullptr);

  const int es = static_cast<int>(esize(dm));
  DispatchArgs da{idx,       dm.T,       dm.k,      dm.N,    dm.d,   es,     dm.n_shared,
                  w.blk_hist, w.counts,  w.offsets, w.perm,  w.inv,  w.tiles, w.num_tiles,
                  w.stiles1, w.stiles2,  h,         w.xperm, status, w.sync_ctr,
                  dm.dtype == PR2_BF16 ? w.ready : nullptr, kTileM};
  // (w.xperm is nullptr on the bf16 path: dispatch then launches no gather)
  if (err == cudaSuccess)
    err = (rhist != nullptr && dm.dtype == PR2_BF16)
              ? launch_dispatch_from_hist(da, rhist->hist, rhist->split, st)
              : launch_dispatch(da, num_sms, st);
  mark(events ? events->dispatched : nullptr);
  if (err != cudaSuccess) return PR2_ERR_CUDA;

  const int64_t F = dm.T * dm.k;
  GemmArgs g1{w.tiles, w.num_tiles, w.max_tiles, dm.d, dm.m, dm.m, w.hbuf, status,
              h, w.perm, dm.k};  // gathered A (bf16); the fp32 GEMM reads w.xperm
  GemmArgs g2{w.tiles, w.num_tiles, w.max_tiles, dm.m, dm.d, dm.d, w.ybuf, status,
              nullptr, nullptr, 0};
  GemmArgs s1{w.stiles1, w.num_tiles + 1, w.shared_tiles, dm.d, dm.m, dm.m, w.hs, status,
              nullptr, nullptr, 0};
  GemmArgs s2{w.stiles2, w.num_tiles + 1, w.shared_tiles, dm.m, dm.d, dm.d, w.ys, status,
              nullptr, nullptr, 0};
  if (dm.dtype == PR2_BF16) {
    CUtensorMap b1g, b1u, a2, b2, sa1, sb1g, sb1u, sa2, sb2;
    bool ok = make_tmap_bf16(&b1g, W_gate, dm.d, (uint64_t)dm.N * dm.m, 64, 128) &&
              make_tmap_bf16(&b1u, W_up, dm.d, (uint64_t)dm.N * dm.m, 64, 128) &&
              make_tmap_bf16(&a2, w.hbuf, dm.m, F, 64, kTileM) &&
              make_tmap_bf16(&b2, W_down, dm.m, (uint64_t)dm.N * dm.d, 64, 256);
    if (ok && dm.n_shared > 0) {
      ok = make_tmap_bf16(&sa1, h, dm.d, dm.T, 64, kTileM) &&
           make_tmap_bf16(&sb1g, Ws_gate, dm.d, (uint64_t)dm.n_shared * dm.m, 64, 128) &&
           make_tmap_bf16(&sb1u, Ws_up, dm.d, (uint64_t)dm.n_shared * dm.m, 64, 128) &&
           make_tmap_bf16(&sa2, w.hs, dm.m, (uint64_t)dm.n_shared * dm.T, 64, kTileM) &&
           make_tmap_bf16(&sb2, Ws_down, dm.m, (uint64_t)dm.n_shared * dm.d, 64, 256);
    }
    if (!ok) return PR2_ERR_CUDA;
    // routed experts: gate/up then down in one cooperative launch
    MlpArgs routed{{g1, g2}, w.ready};
    err = launch_expert_tc(kExpertFused, a2, b1g, b1u, b2, routed, num_sms, st);
    if (err == cudaSuccess && dm.n_shared > 0) {
      MlpArgs sh1{{s1, s1}, nullptr};
      err = launch_expert_tc(kExpertGateUpTma, sa1, sb1g, sb1u, sb1g, sh1, num_sms, st);
    }
    mark(events ? events->gate_up_done : nullptr);
    if (err == cudaSuccess && dm.n_shared > 0) {
      MlpArgs sh2{{s2, s2}, nullptr};
      err = launch_expert_tc(kExpertDown, sa2, sb2, sb2, sb2, sh2, num_sms, st);
    }
    mark(events ? events->down_done : nullptr);
  } else {
    err = launch_expert_simt(true, static_cast<const float*>(w.xperm),
                             static_cast<const float*>(W_gate), static_cast<const float*>(W_up),
                             g1, st);
    if (err == cudaSuccess && dm.n_shared > 0)
      err = launch_expert_simt(true, static_cast<const float*>(h),
                               static_cast<const float*>(Ws_gate),
                               static_cast<const float*>(Ws_up), s1, st);
    mark(events ? events->gate_up_done : nullptr);
    if (err == cudaSuccess)
      err = launch_expert_simt(false, static_cast<const float*>(w.hbuf),
                               static_cast<const float*>(W_down), nullptr, g2, st);
    if (err == cudaSuccess && dm.n_shared > 0)
      err = launch_expert_simt(false, static_cast<const float*>(w.hs),
                               static_cast<const float*>(Ws_down), nullptr, s2, st);
    mark(events ? events->down_done : nullptr);
  }
  if (err != cudaSuccess) return PR2_ERR_CUDA;
  if (replay != nullptr) {
    // Its inputs (h, the router, the route) are complete before the GEMMs start, so on the
    // tensor-core path its CTAs take the SMs the GEMM's last CTAs free and wait for the GEMMs
    // only before exiting; the combine launched behind it then sees both.
    pr2_dims dr = dm;
    dr.flags &= ~PR2_F_SYNC_STATUS;
    s = route_common(&dr, false, h, replay->W_router, nullptr, idx, nullptr,
                     const_cast<float*>(gates), replay->probs, nullptr, status, stream,
                     dm.dtype == PR2_BF16);
    if (s != PR2_OK) return s;
  }

  CombineArgs ca{w.ybuf, dm.n_shared > 0 ? w.ys : nullptr, w.inv, gates, dm.T, dm.k, dm.d,
                 dm.n_shared, dm.dtype == PR2_BF16 ? 1 : 0, out, residual, status};
  err = launch_combine(ca, num_sms, st);
  mark(events ? events->end : nullptr);
  if (err == cudaSuccess && counts != nullptr)
    err = cudaMemcpyAsync(counts, w.counts, sizeof(int32_t) * dm.N, cudaMemcpyDeviceToDevice, st);
  if (err == cudaSuccess && perm != nullptr)
    err = cudaMemcpyAsync(perm, w.perm, sizeof(int32_t) * F, cudaMemcpyDeviceToDevice, st);
  return finish(err, dm.flags, status, st);
}

}  // namespace
}  // namespace pr2

extern "C" {

pr2_status pr2_moe_forward(const pr2_dims* dims, const void* h, const int32_t* idx,
                           const float* gates, const void* W_gate, const void* W_up,
                           const void* W_down, const void* Ws_gate, const void* Ws_up,
                           const void* Ws_down, void* out, int32_t* counts, int32_t* perm,
                           void* workspace, size_t ws_bytes, int32_t* status_dev,
                           const pr2_stage_events* events, void* stream) {
  return moe_forward_impl(dims, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down,
                          out, nullptr, counts, perm, workspace, ws_bytes, status_dev, events,
                          stream);
}

pr2_status pr2_moe_rollout_forward(const pr2_dims* dims, const void* h, const void* W_router,
                                   const void* W_pred, int32_t* idx, float* gates,
                                   float* logits_old, int64_t* near_tie, const void* W_gate,
                                   const void* W_up, const void* W_down, const void* Ws_gate,
                                   const void* Ws_up, const void* Ws_down, void* out,
                                   int32_t* counts, int32_t* perm, void* workspace,
                                   size_t ws_bytes, int32_t* status_dev,
                                   const pr2_stage_events* events, void* stream) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  const pr2_dims& dm = *dims;
  if (dm.T == 0) return PR2_OK;
  if ((dm.flags & PR2_F_SYNC_STATUS) && status_dev == nullptr) return PR2_ERR_INVALID_ARG;
  // everything both steps need is checked before anything is launched
  if (W_router == nullptr || W_pred == nullptr || !aligned16(W_router) || !aligned16(W_pred) ||
      (logits_old != nullptr && !aligned16(logits_old)))
    return PR2_ERR_INVALID_ARG;
  s = forward_args(dm, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down, out,
                   workspace, ws_bytes);
  if (s != PR2_OK) return s;
  pr2_dims dr = dm;
  dr.flags &= ~PR2_F_SYNC_STATUS;
  if (dm.dtype != PR2_BF16) {  // fp32: the two calls in sequence
    s = route_common(&dr, true, h, W_router, W_pred, nullptr, idx, gates, logits_old, near_tie,
                     status_dev, stream);
    if (s != PR2_OK) return s;
    return moe_forward_impl(dims, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down,
                            out, nullptr, counts, perm, workspace, ws_bytes, status_dev, events,
                            stream);
  }
  const Workspace w = carve(dm, static_cast<uint8_t*>(workspace));
  int split = 1;
  s = route_common(&dr, true, h, W_router, W_pred, nullptr, idx, gates, logits_old, near_tie,
                   status_dev, stream, false, w.route_hist, &split);
  if (s != PR2_OK) return s;
  const RouteHist rh{w.route_hist, split};
  return moe_forward_impl(dims, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down,
                          out, nullptr, counts, perm, workspace, ws_bytes, status_dev, events,
                          stream, nullptr, &rh);
}

pr2_status pr2_moe_replay_forward(const pr2_dims* dims, const void* h, const void* W_router,
                                  const int32_t* idx, float* gates, float* probs,
                                  const void* W_gate, const void* W_up, const void* W_down,
                                  const void* Ws_gate, const void* Ws_up, const void* Ws_down,
                                  void* out, int32_t* counts, int32_t* perm, void* workspace,
                                  size_t ws_bytes, int32_t* status_dev,
                                  const pr2_stage_events* events, void* stream) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  if (dims->T == 0) return PR2_OK;
  // everything the routing step needs is checked here, before the forward launches anything
  if (W_router == nullptr || gates == nullptr || !aligned16(W_router) ||
      (probs != nullptr && !aligned16(probs)))
    return PR2_ERR_INVALID_ARG;
  const ReplayRoute rr{W_router, probs};
  return moe_forward_impl(dims, h, idx, gates, W_gate, W_up, W_down, Ws_gate, Ws_up, Ws_down,
                          out, nullptr, counts, perm, workspace, ws_bytes, status_dev, events,
                          stream, &rr);
}

pr2_status pr2_rollout_layers(const pr2_dims* dims, int32_t L, void* h, const void* W_router,
                              const void* W_pred, const void* W_gate, const void* W_up,
                              const void* W_down, const void* Ws_gate, const void* Ws_up,
                              const void* Ws_down, int32_t* idx, float* gates,
                              float* logits_old, int64_t* near_tie, void* workspace,
                              size_t ws_bytes, int32_t* status_dev, void* stream) {
  pr2_status s = check_dims(dims);
  if (s != PR2_OK) return s;
  const pr2_dims& dm = *dims;
  if (L < 1) return PR2_ERR_INVALID_ARG;
  if ((dm.flags & PR2_F_SYNC_STATUS) && status_dev == nullptr) return PR2_ERR_INVALID_ARG;
  if (dm.T == 0) return PR2_OK;
  if (h == nullptr || W_router == nullptr || W_pred == nullptr || W_gate == nullptr ||
      W_up == nullptr || W_down == nullptr || idx == nullptr || gates == nullptr)
    return PR2_ERR_INVALID_ARG;
  const size_t es = esize(dm);
  const size_t r_sz = (size_t)dm.N * dm.d * es;            // one layer's router / predictor
  const size_t gu_sz = (size_t)dm.N * dm.m * dm.d * es;    // gate or up (and down) stack
  const size_t sgu_sz = (size_t)dm.n_shared * dm.m * dm.d * es;
  auto base = [](const void* p, size_t off) -> const void* {
    return p == nullptr ? nullptr : static_cast<const uint8_t*>(p) + off;
  };
  // Each layer's status goes to the caller's word (or the forward's own), read once at the end.
  const uint32_t lf = dm.flags & ~PR2_F_SYNC_STATUS;
  pr2_dims dl = dm;
  dl.flags = lf;
  for (int32_t l = 0; l < L; ++l) {
    int32_t* idx_l = idx + (size_t)l * dm.T * dm.k;
    float* gates_l = gates + (size_t)l * dm.T * dm.k;
    float* logits_l = logits_old ? logits_old + (size_t)l * dm.T * dm.N : nullptr;
    s = pr2_route_predict(&dl, h, base(W_router, l * r_sz), base(W_pred, l * r_sz), idx_l,
                          gates_l, logits_l, near_tie, status_dev, stream);
    if (s != PR2_OK) return s;
    s = moe_forward_impl(&dl, h, idx_l, gates_l, base(W_gate, l * gu_sz), base(W_up, l * gu_sz),
                         base(W_down, l * gu_sz), base(Ws_gate, l * sgu_sz),
                         base(Ws_up, l * sgu_sz), base(Ws_down, l * sgu_sz), h, h, nullptr,
                         nullptr, workspace, ws_bytes, status_dev, nullptr, stream);
    if (s != PR2_OK) return s;
  }
  return finish(cudaSuccess, dm.flags, status_dev, static_cast<cudaStream_t>(stream));
}

const char* pr2_strerror(pr2_status s) {
  switch (s) {
    case PR2_OK: return "ok";
    case PR2_ERR_INVALID_ARG: return "invalid argument";
    case PR2_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case PR2_ERR_CUDA: return "CUDA error";
    case PR2_ERR_BAD_INDEX: return "invalid expert index in route";
    case PR2_ERR_TIMEOUT: return "device wait timed out";
    case PR2_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
  }
  return "unknown status";
}

pr2_status pr2_selftest_wait_timeout(int32_t* status_dev, int64_t timeout_ns, void* stream) {
  if (status_dev == nullptr || timeout_ns < 1000 || timeout_ns > 1000000000) return PR2_ERR_INVALID_ARG;
  cudaError_t err = launch_wait_selftest(status_dev, timeout_ns, static_cast<cudaStream_t>(stream));
  return err == cudaSuccess ? PR2_OK : PR2_ERR_CUDA;
}

}  // extern "C"

namespace pr2 {
namespace {
// One thread waits on an mbarrier that expects an arrival nobody makes; the bounded wait gives
// up after timeout_ns and records PR2_STATUS_TIMEOUT.
__global__ void wait_selftest_kernel(int32_t* status, int64_t timeout_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0)
    mbar_wait_slow(&bar, 0, &abort_flag, status, static_cast<uint64_t>(timeout_ns));
}
}  // namespace

cudaError_t launch_wait_selftest(int32_t* status, int64_t timeout_ns, cudaStream_t st) {
  wait_selftest_kernel<<<1, 32, 0, st>>>(status, timeout_ns);
  return cudaGetLastError();
}
}  // namespace pr2
