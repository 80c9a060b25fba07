/*
 * pr2.h - C ABI of the Pr^2 (Predictive Routing Replay) MoE-layer forward for GB300 (sm_103a).
 *
 * The layer has two modes (Sec. 4.1 of arxiv 2606.00395):
 *   rollout:  pr2_route_predict  then  pr2_moe_forward   (Eqs. pr2_predict, pr2_route,
 *             pr2_old_output; Algorithm 1 rollout steps, Algorithm 2)
 *   training: pr2_route_replay   then  pr2_moe_forward   (Sec. 4.1 "Replay During Training",
 *             Eq. pr2_output; Algorithm 1 replay steps, Algorithm 3)
 *
 * Conventions shared by every entry point:
 *  - Every tensor argument is a DEVICE pointer to a contiguous row-major buffer owned by the
 *    caller; the library allocates nothing, keeps no state between calls and is re-entrant per
 *    stream.  All work is enqueued asynchronously on `stream` (a cudaStream_t; NULL = legacy
 *    default stream).  Pointers must be 16-byte aligned.
 *  - h, the weights and the layer output share dims->dtype (PR2_FP32 or PR2_BF16).  Gates,
 *    logits and probabilities are always fp32; expert indices are int32 (App. E.2 stores the
 *    replay indices as int32).
 *  - Weights are stored [out, in]: W_router[e*d + i] is entry (i, e) of the paper's d x N
 *    router matrix W, so the logits p = h W of Sec. 4.1 are p[t,e] = sum_i h[t,i] W_router[e*d+i].
 *    W_pred has the same layout for the evolution predictor W_p.  Expert weights are stacked:
 *    W_gate, W_up [N, m, d]; W_down [N, d, m]; shared experts Ws_* the same with n_shared rows.
 *  - Host-detectable problems (NULL pointer, unsupported shape, short workspace) return an
 *    error before anything is launched.  Data-dependent problems found on the device (a replay
 *    index outside [0, N) or repeated within a token; a bounded device wait that ran out) are
 *    OR-ed into the caller's device status word as PR2_STATUS_* bits; the offending slot then
 *    contributes nothing.  After a timeout the layer output is unspecified: the kernels of
 *    pr2_moe_forward that find PR2_STATUS_TIMEOUT in the word when they start (the grouped
 *    GEMMs and the combine, which read tables an aborted dispatch may not have written) do no
 *    work.  With PR2_F_SYNC_STATUS in dims->flags the call synchronises the
 *    stream, reads the status word and returns PR2_ERR_BAD_INDEX / PR2_ERR_TIMEOUT.  No C++
 *    exception crosses this ABI and no kernel traps.
 *  - Supported shapes: 1 <= k <= min(N, 32).  PR2_FP32 runs exact-fp32 SIMT kernels (N <= 256).
 *    PR2_BF16 runs tcgen05 tensor-core kernels (fp32 accumulation) and needs d % 64 == 0,
 *    m % 64 == 0, N % 16 == 0, N <= 256 and k <= 8.  Anything else returns PR2_ERR_UNSUPPORTED.
 */
#ifndef PR2_H
#define PR2_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PR2_OK = 0,
    PR2_ERR_INVALID_ARG = 1,  /* NULL pointer, k > N, T < 0, ...                             */
    PR2_ERR_UNSUPPORTED = 2,  /* valid but outside the shapes/dtypes listed above              */
    PR2_ERR_CUDA = 3,         /* a CUDA runtime call or launch failed                          */
    PR2_ERR_BAD_INDEX = 4,    /* (PR2_F_SYNC_STATUS only) invalid replay index seen on device  */
    PR2_ERR_TIMEOUT = 5,      /* (PR2_F_SYNC_STATUS only) a bounded device wait ran out        */
    PR2_ERR_WORKSPACE = 6     /* workspace NULL or smaller than pr2_moe_workspace_bytes()      */
} pr2_status;

typedef enum { PR2_FP32 = 0, PR2_BF16 = 1 } pr2_dtype;

/* dims->flags bits */
#define PR2_F_SYNC_STATUS 0x1u /* synchronise `stream` and turn the status word into a code */
#define PR2_F_DELTA_LOSS 0x2u  /* pr2_predictor_loss: the delta-matching variant              */
#define PR2_F_NORMALIZE_TOPK 0x4u /* routing: gates renormalised over the selected experts    */

/* device status word bits (OR-ed in by the kernels; the caller zeroes the word) */
#define PR2_STATUS_BAD_INDEX 0x1
#define PR2_STATUS_TIMEOUT 0x2

/* A token counts as a near tie when its k-th and (k+1)-th predicted probabilities differ by
 * less than this (the top-k margin Delta_k of Lemma topk_regret, App. B). */
#define PR2_NEAR_TIE_GAP 1e-4

/* Problem size of one MoE layer: T tokens, d = d_model, N routed experts, top-k, m = expert
 * hidden size (d_ff), n_shared always-on shared experts (App. E.2, "s"). */
typedef struct {
    int64_t T;
    int32_t d, N, k, m, n_shared;
    int32_t dtype;   /* pr2_dtype */
    uint32_t flags;  /* PR2_F_* (any other bit: PR2_ERR_INVALID_ARG) */
} pr2_dims;

/*
 * Rollout routing, Eqs. pr2_predict and pr2_route (Sec. 4.1 "Route Prediction During Rollout"),
 * with the route record of Algorithm 2:
 *     p_old = h W_old,  b = h W_p,  rho_hat = Softmax(p_old + b),  I_hat = TopK(rho_hat, k).
 *  h          [T, d]  dtype     router input h_old
 *  W_router   [N, d]  dtype     old-snapshot router (transposed W_old)
 *  W_pred     [N, d]  dtype     evolution predictor (transposed W_p)
 *  idx        [T, k]  int32     out: I_hat, slots by descending rho_hat, ties to the lower index
 *  gates      [T, k]  fp32      out: rho_hat at idx (full-softmax probability; divided by its
 *                               sum over the k slots only with PR2_F_NORMALIZE_TOPK in dims->flags,
 *                               the Qwen3 reading: the paper weights with rho_hat itself)
 *  logits_old [T, N]  fp32      out, nullable: p_old, the feature-cache logits of Algorithm 2
 *  near_tie   [1]     int64     in/out, nullable: += #tokens whose rho_hat_(k) - rho_hat_(k+1)
 *                               < PR2_NEAR_TIE_GAP (k < N)
 *  status_dev [1]     int32     in/out, nullable: PR2_STATUS_* bits
 */
pr2_status pr2_route_predict(const pr2_dims* dims, const void* h, const void* W_router,
                             const void* W_pred, int32_t* idx, float* gates, float* logits_old,
                             int64_t* near_tie, int32_t* status_dev, void* stream);

/*
 * Training-time replay gates, Sec. 4.1 "Replay During Training" (Algorithm 3, first step):
 *     rho = Softmax(h W),  gates[t,s] = rho[t, idx[t,s]];  no fresh top-k, no predictor.
 *  h [T,d], W_router [N,d] (current router, dtype); idx [T,k] int32 the cached route;
 *  gates [T,k] fp32 out (0 for an invalid slot; with PR2_F_NORMALIZE_TOPK divided by the sum
 *  over the token's valid slots); probs [T,N] fp32 out, nullable: the full rho (never divided);
 *  status_dev nullable (PR2_STATUS_BAD_INDEX for an index outside [0,N) or repeated in a token).
 */
pr2_status pr2_route_replay(const pr2_dims* dims, const void* h, const void* W_router,
                            const int32_t* idx, float* gates, float* probs, int32_t* status_dev,
                            void* stream);

/* Optional stage markers of pr2_moe_forward for profiling: each non-NULL member is a
 * cudaEvent_t (created by the caller on the current device) that the call records on `stream`
 * at that point of the launch sequence.  NULL members and a NULL struct pointer are ignored. */
typedef struct {
    void* start;         /* before dispatch                                              */
    void* dispatched;    /* after histogram, scan and stable placement (+ the row gather
                          * on the fp32 path; the bf16 gate/up GEMM gathers its rows)    */
    void* gate_up_done;  /* after the routed experts' GEMMs (bf16: gate/up and down run as
                          * one launch) and the shared experts' gate/up GEMM              */
    void* down_done;     /* after the shared experts' down GEMM (the routed down GEMM on
                          * the fp32 path)                                               */
    void* end;           /* after the gate-weighted combine                              */
} pr2_stage_events;

/* Bytes of device workspace pr2_moe_forward needs for `dims` (0 for invalid dims). */
size_t pr2_moe_workspace_bytes(const pr2_dims* dims);

/*
 * MoE layer output on a given route, Eq. pr2_old_output (rollout gates rho_hat[idx]) and
 * Eq. pr2_output (replay gates rho[idx]); experts are gated MLPs (App. E.2) with SwiGLU:
 *     out[t] = sum_{s<k} gates[t,s] * E_{idx[t,s]}(h_t) + sum_{j<n_shared} E^shared_j(h_t),
 *     E(x) = W_down (silu(W_gate x) * (W_up x)).
 *  h [T,d] dtype; idx [T,k] int32; gates [T,k] fp32; W_gate, W_up [N,m,d]; W_down [N,d,m];
 *  Ws_gate, Ws_up [n_shared,m,d], Ws_down [n_shared,d,m] (NULL iff n_shared == 0);
 *  out [T,d] dtype (written, fp32 accumulation, rounded once);
 *  counts [N] int32 out, nullable: tokens per expert (valid slots only);
 *  perm [T*k] int32 out, nullable: flat slot ids t*k+s grouped by expert, stable in slot order
 *      (entries past sum(counts) are unspecified);
 *  workspace/ws_bytes: device scratch of at least pr2_moe_workspace_bytes(dims) bytes, 256-byte
 *      aligned, owned by the caller and reused freely between calls on the same stream;
 *  status_dev nullable (a status word inside the workspace is used when NULL);
 *  events nullable: stage markers recorded for profiling (see pr2_stage_events).
 */
pr2_status pr2_moe_forward(const pr2_dims* dims, const void* h, const int32_t* idx,
                           const float* gates, const void* W_gate, const void* W_up,
                           const void* W_down, const void* Ws_gate, const void* Ws_up,
                           const void* Ws_down, void* out, int32_t* counts, int32_t* perm,
                           void* workspace, size_t ws_bytes, int32_t* status_dev,
                           const pr2_stage_events* events, void* stream);

/*
 * Rollout-mode layer in one call: pr2_route_predict followed by pr2_moe_forward on the route
 * and gates it records (Eqs. pr2_predict, pr2_route, pr2_old_output; Algorithm 2), with
 * identical results.  On the tensor-core path the routing kernel also counts, per CTA, the
 * experts of the rows it finishes into the workspace, so dispatch needs neither a histogram
 * pass nor a grid-wide barrier and runs as an ordinary launch right behind the routing kernel.
 * Arguments as in pr2_route_predict (idx, gates, logits_old, near_tie written) and
 * pr2_moe_forward (the rest; the workspace is the same size).
 */
pr2_status pr2_moe_rollout_forward(const pr2_dims* dims, const void* h, const void* W_router,
                                   const void* W_pred, int32_t* idx, float* gates,
                                   float* logits_old, int64_t* near_tie, const void* W_gate,
                                   const void* W_up, const void* W_down, const void* Ws_gate,
                                   const void* Ws_up, const void* Ws_down, void* out,
                                   int32_t* counts, int32_t* perm, void* workspace,
                                   size_t ws_bytes, int32_t* status_dev,
                                   const pr2_stage_events* events, void* stream);

/*
 * Training-mode layer in one call: pr2_route_replay followed by pr2_moe_forward on its gates
 * (Sec. 4.1 "Replay During Training", Eq. pr2_output), with identical results.  Only the
 * gate-weighted combine reads the replay gates, so the call launches dispatch and the expert
 * GEMMs first and the replay routing behind them; on the tensor-core path the routing kernel
 * runs on the SMs the GEMM's last CTAs free instead of in front of the whole layer.
 * Arguments as in pr2_route_replay (W_router, idx, gates written, probs nullable) and
 * pr2_moe_forward (the rest).  status_dev collects the bits of both steps.
 */
pr2_status pr2_moe_replay_forward(const pr2_dims* dims, const void* h, const void* W_router,
                                  const int32_t* idx, float* gates, float* probs,
                                  const void* W_gate, const void* W_up, const void* W_down,
                                  const void* Ws_gate, const void* Ws_up, const void* Ws_down,
                                  void* out, int32_t* counts, int32_t* perm, void* workspace,
                                  size_t ws_bytes, int32_t* status_dev,
                                  const pr2_stage_events* events, void* stream);

/*
 * pr2_moe_forward without a caller-provided workspace.  The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory where they run the layer
 * (a runtime whose pool owns all device memory, a hot path on which cudaMalloc/cudaFree and
 * their device-wide synchronisation are not allowed, a plug-in with a fixed memory budget).
 * Same arguments and results as pr2_moe_forward minus workspace/ws_bytes/events; the scratch
 * is one array of pr2_static_scratch_bytes() bytes (32 MiB) compiled into the library, which
 * every GPU that loads the library keeps reserved until the process exits.  The call allocates
 * nothing.
 *  - Layers whose pr2_moe_workspace_bytes(dims) exceeds pr2_static_scratch_bytes() are
 *    rejected with PR2_ERR_WORKSPACE before anything is launched (e.g. the Qwen3-shaped layer
 *    up to 743 tokens fits; a 4096-token batch does not).
 *  - The first call on a device looks up the array's device address (cudaGetSymbolAddress,
 *    with that device current); make that first call before any stream capture.
 *  - All calls on a device share the one array: calls whose kernels overlap on the GPU (other
 *    streams, other host threads) race on it and corrupt each other's results.  Serialise them,
 *    e.g. by issuing them on one stream.
 */
pr2_status pr2_moe_forward_static(const pr2_dims* dims, const void* h, const int32_t* idx,
                                  const float* gates, const void* W_gate, const void* W_up,
                                  const void* W_down, const void* Ws_gate, const void* Ws_up,
                                  const void* Ws_down, void* out, int32_t* counts,
                                  int32_t* perm, int32_t* status_dev, void* stream);

/* Size in bytes of the scratch array used by pr2_moe_forward_static (no paper counterpart). */
size_t pr2_static_scratch_bytes(void);

/*
 * Predictive loss of one layer and its gradient w.r.t. the evolution predictor (Sec. 4.2 Eq.
 * pr2_loss; Algorithm 3 "reconstruct the predictive distribution", "predictive KL loss").
 * dims->T is the number T_c of cached tokens; d, N and dtype are the layer's (k is unused
 * beyond the usual checks).
 *  h_old [T_c, d] dtype, p_old [T_c, N] fp32: the cached route-recording features (Algorithm 2
 *    feature cache).  W_pred [N, d] dtype: the predictor W_p.
 *  rho [T_rho, N] fp32: the teacher, the current routing distribution Softmax(h W) of the
 *    batch (e.g. the `probs` output of pr2_route_replay); a stop-gradient target.  Cached row c
 *    is compared with row pos[c] (pos [T_c] int32; NULL: row c).  A pos entry outside
 *    [0, T_rho) sets PR2_STATUS_BAD_INDEX and that row contributes nothing.
 *  Default (Eq. pr2_loss):  z = p_old + h_old W_p^T,  rho_hat = Softmax(z),
 *      KL_c = sum_j rho_j (log rho_j - log rho_hat_j),   dKL_c/dz = rho_hat - rho.
 *  PR2_F_DELTA_LOSS (the appendix delta-matching variant): target q = Softmax(p - p_old),
 *      computed as Softmax(log rho - p_old); prediction Softmax(h_old W_p^T);
 *      KL_c = KL(q || Softmax(b)),  dKL_c/db = Softmax(b) - q.
 *  Outputs: loss[0] = (1/T_c) sum_c KL_c (fp32, summed in double in a fixed order);
 *    kl_tok [T_c] fp32 per-token KL_c (nullable);
 *    grad_Wp [N, d] fp32 = (1/T_c) sum_c (dKL_c/dz)^T h_old[c] (overwritten).
 *  T_c = 0 writes loss 0 and a zero gradient.  bf16 runs the predictor projection on tcgen05
 *  (fp32 accumulation) and the gradient as a tcgen05 GEMM on bf16-rounded dKL/dz; fp32 runs
 *  exact-fp32 SIMT kernels.  Deterministic.
 *  workspace/ws_bytes: device scratch of at least pr2_predictor_loss_workspace_bytes(dims)
 *    bytes, 256-byte aligned, not used concurrently by another call.
 */
size_t pr2_predictor_loss_workspace_bytes(const pr2_dims* dims);
pr2_status pr2_predictor_loss(const pr2_dims* dims, const void* h_old, const float* p_old,
                              const void* W_pred, const float* rho, int64_t T_rho,
                              const int32_t* pos, float* loss, float* kl_tok, float* grad_Wp,
                              void* workspace, size_t ws_bytes, int32_t* status_dev,
                              void* stream);

/*
 * Route tracking of a cached route against the current router (Sec. 5 "Top-k Agreement and
 * Route KL", "Deviation Tails").  For each of the dims->T tokens: I_t = TopK(rho_t, k) of the
 * current routing distribution rho [T, N] fp32 (e.g. the probs output of pr2_route_replay;
 * ties to the lower expert as in Eq. pr2_route), Î_t = idx_cached[t] ([T, k] int32, the
 * replayed route); overlap_t = |Î_t ∩ I_t|, where a cached entry outside [0, N) or repeated in
 * its token never matches.  ACCUMULATES hist[k - overlap_t] += 1 (int64 [k+1], the deviation
 * count of "Deviation Tails") and overlap_sum[0] += overlap_t; the caller zeroes both, so that
 * layers can be summed.  Top-k agreement = overlap_sum / (T k).  Exact (integer atomics).
 * Needs k <= 32.  The route KL of Sec. 5 is the loss value of pr2_predictor_loss.
 */
pr2_status pr2_route_diagnostics(const pr2_dims* dims, const float* rho,
                                 const int32_t* idx_cached, int64_t* hist, int64_t* overlap_sum,
                                 void* stream);

/*
 * Fixed-length feature-cache writer (Algorithm 2: store the route-recording features
 * (h_old, p_old) of the retained positions; App.: T_c positions drawn by uniform sub-sampling
 * along the rollout).  The T_c <= dims->T retained positions are evenly spaced,
 * pos[c] = floor(c T / T_c) (int32 [T_c]; T_c = T keeps every token), and
 * cache_h[c] = h[pos[c]] ([T_c, d], dims->dtype, bits copied), cache_p[c] = logits_old[pos[c]]
 * ([T_c, N] fp32; both NULL to skip).  logits_old is the p_old output of pr2_route_predict.
 * Cache size T_c (2 d + 4 N) bytes per layer for bf16 h (Table 4).
 */
pr2_status pr2_feature_cache_write(const pr2_dims* dims, int64_t T_c, const void* h,
                                   const float* logits_old, int32_t* pos, void* cache_h,
                                   float* cache_p, void* stream);

/*
 * Multi-layer rollout decode: L Pr^2 MoE layers in rollout mode applied in sequence to one
 * batch of T tokens, as the route-recording phase runs them layer after layer (Algorithm 2 for
 * l = 1..L: predict the route, record it and the features, compute o_old^(l); App. "Pr^3"
 * uses the same rollout-engine pass).  Between layers the residual stream
 * h^(l+1) = h^(l) + o_old^(l) (rounded once to dims->dtype) stands in for the rest of the
 * transformer block; attention and normalisation are outside this library.
 *  h [T, d] dims->dtype: h^(1) on entry, h^(L+1) on return (updated in place).
 *  Weights stacked by layer: W_router, W_pred [L, N, d]; W_gate, W_up [L, N, m, d];
 *    W_down [L, N, d, m]; shared experts Ws_gate, Ws_up [L, n_shared, m, d],
 *    Ws_down [L, n_shared, d, m] (NULL iff n_shared == 0).
 *  Outputs per layer, as pr2_route_predict writes them: idx [L, T, k], gates [L, T, k],
 *    logits_old [L, T, N] (nullable: the feature-cache logits p_old); near_tie (nullable) counts
 *    over all layers.
 *  workspace: pr2_moe_workspace_bytes(dims) bytes, reused by every layer.
 * Every step is an asynchronous launch on `stream` (no host synchronisation unless
 * PR2_F_SYNC_STATUS), so the whole loop can be captured into a CUDA graph by the caller and
 * replayed; results equal those of L pairs of pr2_route_predict / pr2_moe_forward calls.
 */
pr2_status pr2_rollout_layers(const pr2_dims* dims, int32_t L, void* h, const void* W_router,
                              const void* W_pred, const void* W_gate, const void* W_up,
                              const void* W_down, const void* Ws_gate, const void* Ws_up,
                              const void* Ws_down, int32_t* idx, float* gates,
                              float* logits_old, int64_t* near_tie, void* workspace,
                              size_t ws_bytes, int32_t* status_dev, void* stream);

/* Static, human-readable name of a status code. */
const char* pr2_strerror(pr2_status s);

/*
 * Self-test of the bounded device wait used by every pipelined kernel (no paper counterpart):
 * launches one CTA that waits on a barrier nothing will ever complete, gives up after
 * `timeout_ns` nanoseconds, ORs PR2_STATUS_TIMEOUT into status_dev[0] and returns normally.
 * timeout_ns must lie in [1e3, 1e9].  Lets a caller check that a stalled pipeline reports an
 * error instead of hanging.
 */
pr2_status pr2_selftest_wait_timeout(int32_t* status_dev, int64_t timeout_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* PR2_H */
