/*
 * Pr^2 MoE-layer oracle: a plain, slow, fp64 CPU restatement of what the layer computes.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or call this file;
 * only the tests, the smoke check and the bench's CPU-baseline / reference arm use it.  It
 * shares no code, header, table or helper with the CUDA library.
 *
 * Every input is read in its stored precision (fp32, or bf16 given as raw 16-bit patterns)
 * and widened exactly to double; all arithmetic below is fp64 with no intermediate rounding.
 * Weight layout: [out, in] row-major, i.e. W[e*d + i] is entry (i, e) of the paper's d x N
 * router matrix, so  p_e = sum_i h_i W[e*d + i]  is the paper's  p = h W  (Sec. 4.1).
 *
 * Readings taken where the paper is silent (each also listed in the design notes):
 *  - TopK ties go to the lower expert index; the k slots are ordered by descending probability.
 *  - Gates are the full-softmax probabilities at the selected indices, never renormalised
 *    (Eq. pr2_old_output / Eq. pr2_output weight by rho-hat_j and rho_j directly).
 *  - The gated-MLP expert of App. E.2 is SwiGLU: y = W_down (silu(W_gate h) * (W_up h)).
 *  - Shared experts are added with weight 1 and never appear in the routed indices (App. E.2).
 *  - A replay index outside [0, N) or repeated within a token is invalid: it is counted and
 *    that slot contributes nothing.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* ---- exact widening of stored values to double ------------------------------------------ */

enum { ORC_FP32 = 0, ORC_BF16 = 1 };

static double widen(const void* base, int64_t i, int dtype) {
    if (dtype == ORC_FP32) return (double)((const float*)base)[i];
    /* bf16 is the top half of an IEEE binary32: shift the 16 stored bits into place. */
    uint32_t bits = ((uint32_t)((const uint16_t*)base)[i]) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ---- Sec. 4.1: router logits, softmax, top-k ---------------------------------------------- */

/* p[e] = sum_i h[t,i] W[e,i]  (the row-vector product h W of Sec. 4.1). */
static void project(const void* h, int64_t t, int d, int N, const void* W, int dtype, double* p) {
    for (int e = 0; e < N; ++e) {
        double acc = 0.0;
        for (int i = 0; i < d; ++i)
            acc += widen(h, t * (int64_t)d + i, dtype) * widen(W, (int64_t)e * d + i, dtype);
        p[e] = acc;
    }
}

/* Softmax(z)_e = exp(z_e - max z) / sum_j exp(z_j - max z)  (Eq. pr2_predict). */
static void softmax(const double* z, int N, double* rho) {
    double mx = z[0];
    for (int e = 1; e < N; ++e) if (z[e] > mx) mx = z[e];
    double sum = 0.0;
    for (int e = 0; e < N; ++e) { rho[e] = exp(z[e] - mx); sum += rho[e]; }
    for (int e = 0; e < N; ++e) rho[e] /= sum;
}

/* TopK(rho, k) (Eq. pr2_route): repeated selection of the largest remaining probability,
 * lower index first on equal values.  Returns the margin rho_(k) - rho_(k+1) (the Delta_k of
 * Lemma topk_regret; +inf when k == N) and writes the k+1 ordered values to `top_vals`. */
static double topk(const double* rho, int N, int k, int32_t* sel, double* top_vals, char* taken) {
    memset(taken, 0, (size_t)N);
    int kk = (k < N) ? k + 1 : k;
    for (int s = 0; s < kk; ++s) {
        int best = -1;
        for (int e = 0; e < N; ++e)
            if (!taken[e] && (best < 0 || rho[e] > rho[best])) best = e;
        taken[best] = 1;
        if (s < k) sel[s] = best;
        top_vals[s] = rho[best];
    }
    return (k < N) ? top_vals[k - 1] - top_vals[k] : INFINITY;
}

/*
 * Rollout mode, Algorithm 1 (route prediction) / Algorithm 2 steps on one layer:
 *   p_old = h_old W_old,  b = h_old W_p,  rho_hat = Softmax(p_old + b),  I_hat = TopK(rho_hat, k),
 *   gates[t,s] = rho_hat[t, I_hat[t,s]].
 * Outputs (all [T, ...] row-major; `logits`, `probs`, `margin`, `top_vals` may be NULL):
 *   idx[T,k], gates[T,k], logits[T,N] = p_old (the feature-cache logits), probs[T,N] = rho_hat,
 *   margin[T] = rho_hat_(k) - rho_hat_(k+1), top_vals[T, k+1] = the ordered top probabilities.
 */
void oracle_route_predict(int64_t T, int d, int N, int k, int dtype, const void* h, const void* W,
                          const void* Wp, int32_t* idx, double* gates, double* logits,
                          double* probs, double* margin, double* top_vals) {
    #pragma omp parallel
    {
        double* p = (double*)malloc(sizeof(double) * (size_t)N);
        double* b = (double*)malloc(sizeof(double) * (size_t)N);
        double* z = (double*)malloc(sizeof(double) * (size_t)N);
        double* rho = (double*)malloc(sizeof(double) * (size_t)N);
        double* tv = (double*)malloc(sizeof(double) * (size_t)(k + 1));
        char* taken = (char*)malloc((size_t)N);
        #pragma omp for schedule(dynamic, 4)
        for (int64_t t = 0; t < T; ++t) {
            project(h, t, d, N, W, dtype, p);   /* p_old = h_old W_old */
            project(h, t, d, N, Wp, dtype, b);  /* b = h_old W_p       */
            for (int e = 0; e < N; ++e) z[e] = p[e] + b[e];
            softmax(z, N, rho);
            double mg = topk(rho, N, k, idx + t * k, tv, taken);
            for (int s = 0; s < k; ++s) gates[t * k + s] = rho[idx[t * k + s]];
            if (logits) memcpy(logits + t * N, p, sizeof(double) * (size_t)N);
            if (probs) memcpy(probs + t * N, rho, sizeof(double) * (size_t)N);
            if (margin) margin[t] = mg;
            if (top_vals)
                for (int s = 0; s < ((k < N) ? k + 1 : k); ++s) top_vals[t * (k + 1) + s] = tv[s];
        }
        free(p); free(b); free(z); free(rho); free(tv); free(taken);
    }
}

/*
 * Training (replay) mode, Sec. 4.1 "Replay During Training" / Algorithm 3:
 *   rho = Softmax(h W) with the current router; no fresh top-k; the predictor is not used;
 *   gates[t,s] = rho[t, idx[t,s]] for the cached indices.
 * An index outside [0,N) or repeated within its token is invalid: its gate is 0 and it is
 * counted in the return value.  `probs` ([T,N]) may be NULL.
 */
int64_t oracle_route_replay(int64_t T, int d, int N, int k, int dtype, const void* h,
                            const void* W, const int32_t* idx, double* gates, double* probs) {
    int64_t bad = 0;
    #pragma omp parallel reduction(+ : bad)
    {
        double* p = (double*)malloc(sizeof(double) * (size_t)N);
        double* rho = (double*)malloc(sizeof(double) * (size_t)N);
        #pragma omp for schedule(dynamic, 4)
        for (int64_t t = 0; t < T; ++t) {
            project(h, t, d, N, W, dtype, p);
            softmax(p, N, rho);
            for (int s = 0; s < k; ++s) {
                int32_t e = idx[t * k + s];
                int ok = (e >= 0 && e < N);
                for (int s2 = 0; ok && s2 < s; ++s2) if (idx[t * k + s2] == e) ok = 0;
                gates[t * k + s] = ok ? rho[e] : 0.0;
                bad += !ok;
            }
            if (probs) memcpy(probs + t * N, rho, sizeof(double) * (size_t)N);
        }
        free(p); free(rho);
    }
    return bad;
}

/*
 * Dispatch of (token, slot) pairs to experts ("dispatch to experts", Algorithm 1): a stable
 * counting sort of the flat slot ids f = t*k + s by expert id.
 *   counts[e]  = #{f : idx[f] = e}                       (valid slots only)
 *   offsets[e] = sum_{e' < e} counts[e'],  offsets[N] = number of valid slots
 *   perm[offsets[e] + r] = the r-th f (in increasing f) with idx[f] = e
 *   inv[f] = the position of f in perm, or -1 for an invalid slot.
 * Invalid slots (index outside [0,N) or repeated within the token) are skipped and counted.
 */
int64_t oracle_permute(int64_t T, int k, int N, const int32_t* idx, int32_t* counts,
                       int32_t* offsets, int32_t* perm, int32_t* inv) {
    int64_t F = T * k, bad = 0;
    char* valid = (char*)malloc((size_t)(F > 0 ? F : 1));
    for (int e = 0; e < N; ++e) counts[e] = 0;
    for (int64_t f = 0; f < F; ++f) {
        int32_t e = idx[f];
        int ok = (e >= 0 && e < N);
        int64_t t = f / k;
        for (int64_t f2 = t * k; ok && f2 < f; ++f2) if (idx[f2] == e) ok = 0;
        valid[f] = (char)ok;
        if (ok) counts[e] += 1; else bad += 1;
    }
    offsets[0] = 0;
    for (int e = 0; e < N; ++e) offsets[e + 1] = offsets[e] + counts[e];
    int32_t* next = (int32_t*)malloc(sizeof(int32_t) * (size_t)N);
    for (int e = 0; e < N; ++e) next[e] = offsets[e];
    for (int64_t f = 0; f < F; ++f) {
        if (!valid[f]) { inv[f] = -1; continue; }
        int32_t pos = next[idx[f]]++;
        perm[pos] = (int32_t)f;
        inv[f] = pos;
    }
    free(next); free(valid);
    return bad;
}

/* silu(x) = x * sigma(x), sigma(x) = 1 / (1 + exp(-x)). */
static double silu(double x) { return x / (1.0 + exp(-x)); }

/* Gated-MLP expert (App. E.2, SwiGLU): y = Wd (silu(Wg x) * (Wu x)); Wg, Wu: [m,d]; Wd: [d,m].
 * `ex` selects expert ex inside stacked [E, ...] weight tensors. */
static void expert_ffn(const void* h, int64_t t, int d, int m, int dtype, const void* Wg,
                       const void* Wu, const void* Wd, int64_t ex, double* a, double* y) {
    const int64_t gu = ex * (int64_t)m * d, dn = ex * (int64_t)d * m;
    for (int j = 0; j < m; ++j) {
        double g = 0.0, u = 0.0;
        for (int i = 0; i < d; ++i) {
            double x = widen(h, t * (int64_t)d + i, dtype);
            g += x * widen(Wg, gu + (int64_t)j * d + i, dtype);
            u += x * widen(Wu, gu + (int64_t)j * d + i, dtype);
        }
        a[j] = silu(g) * u;
    }
    for (int c = 0; c < d; ++c) {
        double acc = 0.0;
        for (int j = 0; j < m; ++j) acc += a[j] * widen(Wd, dn + (int64_t)c * m + j, dtype);
        y[c] = acc;
    }
}

/*
 * MoE layer output on given routes (Eq. pr2_old_output in rollout mode, Eq. pr2_output in
 * replay mode; the two differ only in where idx and gates come from):
 *   out[t] = sum_{s<k} gates[t,s] * E_{idx[t,s]}(h_t)  +  sum_{sh < n_shared} E^shared_sh(h_t)
 * summed in slot order, then the shared experts.  Only the n_tok tokens listed in `tokens`
 * are computed; out is [n_tok, d] in that order.  Invalid slots contribute nothing.
 */
void oracle_moe_forward(int64_t n_tok, const int64_t* tokens, int64_t T, int d, int N, int k,
                        int m, int n_shared, int dtype, const void* h, const int32_t* idx,
                        const double* gates, const void* Wg, const void* Wu, const void* Wd,
                        const void* Wsg, const void* Wsu, const void* Wsd, double* out) {
    (void)T;
    #pragma omp parallel
    {
        double* a = (double*)malloc(sizeof(double) * (size_t)m);
        double* y = (double*)malloc(sizeof(double) * (size_t)d);
        #pragma omp for schedule(dynamic, 1)
        for (int64_t i = 0; i < n_tok; ++i) {
            int64_t t = tokens[i];
            double* o = out + i * d;
            for (int c = 0; c < d; ++c) o[c] = 0.0;
            for (int s = 0; s < k; ++s) {
                int32_t e = idx[t * k + s];
                int ok = (e >= 0 && e < N);
                for (int s2 = 0; ok && s2 < s; ++s2) if (idx[t * k + s2] == e) ok = 0;
                if (!ok) continue;
                expert_ffn(h, t, d, m, dtype, Wg, Wu, Wd, e, a, y);
                for (int c = 0; c < d; ++c) o[c] += gates[t * k + s] * y[c];
            }
            for (int sh = 0; sh < n_shared; ++sh) {
                expert_ffn(h, t, d, m, dtype, Wsg, Wsu, Wsd, sh, a, y);
                for (int c = 0; c < d; ++c) o[c] += y[c];
            }
        }
        free(a); free(y);
    }
}

/* ---- Sec. 4.2 "Predictive Loss" (Eq. pr2_loss) and Algorithm 3 ---------------------------- */

/* log Softmax(v)_j = v_j - max - log sum_i exp(v_i - max) for finite v_j; entries equal to
 * -inf get -inf.  Writes the probabilities to `pr` and their logs to `lg`. */
static void log_softmax(const double* v, int N, double* pr, double* lg) {
    double mx = -INFINITY;
    for (int j = 0; j < N; ++j) if (v[j] > mx) mx = v[j];
    double s = 0.0;
    for (int j = 0; j < N; ++j) s += (v[j] == -INFINITY) ? 0.0 : exp(v[j] - mx);
    double ls = log(s);
    for (int j = 0; j < N; ++j) {
        lg[j] = (v[j] == -INFINITY) ? -INFINITY : v[j] - mx - ls;
        pr[j] = (v[j] == -INFINITY) ? 0.0 : exp(lg[j]);
    }
}

/*
 * Predictive loss of one layer over the T_c cached tokens and its gradient w.r.t. W_p.
 * Cached route-recording features (Algorithm 2, feature cache F): h_old[T_c,d] in the stored
 * dtype and p_old[T_c,N] fp32.  Teacher (stop-gradient): the current routing distribution
 * rho = Softmax(h W) (Algorithm 3, first step) of the token each cached row belongs to, row
 * pos[c] of rho_full[T_rho,N] (fp32; pos NULL means row c).
 *
 * kind 0, Eq. pr2_loss / Algorithm 3 ("reconstruct", "KL"):
 *   z = p_old + h_old W_p^T,  rho_hat = Softmax(z),
 *   KL_c = sum_j rho_j (log rho_j - log rho_hat_j)   (terms with rho_j = 0 are 0),
 *   dKL_c / dz_j = rho_hat_j - rho_j                  (softmax Jacobian, sum_j rho_j = 1).
 * kind 1, the delta-matching alternative (App. "Predictive Objective Ablation"):
 *   target q = Softmax(Delta p), Delta p = p - p_old.  The teacher is given as probabilities,
 *   and Softmax(log rho - p_old) = Softmax(p - logsumexp(p) - p_old) = Softmax(Delta p);
 *   prediction Softmax(b), b = h_old W_p^T;  KL_c = KL(q || Softmax(b)),
 *   dKL_c / db_j = Softmax(b)_j - q_j.
 * loss = (1/T_c) sum_c KL_c  (the expectation over cached tokens of Eq. pr2_loss, one layer);
 * grad[j*d + i] = (1/T_c) sum_c dKL_c/dz_j h_old[c,i]  (b_j = sum_i h_old[c,i] W_p[j*d + i]).
 * A pos entry outside [0, T_rho) is invalid: that row contributes nothing and is counted in
 * the return value.  kl_tok[T_c] may be NULL.  T_c = 0 gives loss 0 and a zero gradient.
 */
int64_t oracle_predictor_loss(int64_t Tc, int d, int N, int dtype, int kind, const void* h_old,
                              const float* p_old, const void* Wp, const float* rho_full,
                              int64_t T_rho, const int32_t* pos, double* loss, double* kl_tok,
                              double* grad) {
    double* dz = (double*)calloc((size_t)(Tc > 0 ? Tc : 1) * (size_t)N, sizeof(double));
    double* kl = (double*)calloc((size_t)(Tc > 0 ? Tc : 1), sizeof(double));
    int64_t bad = 0;
    #pragma omp parallel reduction(+ : bad)
    {
        double* b = (double*)malloc(sizeof(double) * (size_t)N);
        double* v = (double*)malloc(sizeof(double) * (size_t)N);
        double* tgt = (double*)malloc(sizeof(double) * (size_t)N);
        double* ltgt = (double*)malloc(sizeof(double) * (size_t)N);
        double* pred = (double*)malloc(sizeof(double) * (size_t)N);
        double* lpred = (double*)malloc(sizeof(double) * (size_t)N);
        #pragma omp for schedule(dynamic, 4)
        for (int64_t c = 0; c < Tc; ++c) {
            int64_t r = pos ? (int64_t)pos[c] : c;
            if (r < 0 || r >= T_rho) { bad += 1; continue; }
            project(h_old, c, d, N, Wp, dtype, b);              /* b = h_old W_p */
            const float* rho = rho_full + r * (int64_t)N;
            const float* po = p_old + c * (int64_t)N;
            if (kind == 0) {
                for (int j = 0; j < N; ++j) {
                    tgt[j] = (double)rho[j];
                    ltgt[j] = (rho[j] > 0.0f) ? log((double)rho[j]) : -INFINITY;
                    v[j] = (double)po[j] + b[j];                    /* z = p_old + b */
                }
                log_softmax(v, N, pred, lpred);                     /* rho_hat */
            } else {
                for (int j = 0; j < N; ++j)
                    v[j] = (rho[j] > 0.0f) ? log((double)rho[j]) - (double)po[j] : -INFINITY;
                log_softmax(v, N, tgt, ltgt);                       /* q = Softmax(Delta p) */
                log_softmax(b, N, pred, lpred);                     /* Softmax(b) */
            }
            double acc = 0.0;
            for (int j = 0; j < N; ++j) {
                if (tgt[j] > 0.0) acc += tgt[j] * (ltgt[j] - lpred[j]);
                dz[c * N + j] = pred[j] - tgt[j];
            }
            kl[c] = acc;
        }
        free(b); free(v); free(tgt); free(ltgt); free(pred); free(lpred);
    }
    double tot = 0.0;
    for (int64_t c = 0; c < Tc; ++c) tot += kl[c];
    *loss = (Tc > 0) ? tot / (double)Tc : 0.0;
    if (kl_tok) for (int64_t c = 0; c < Tc; ++c) kl_tok[c] = kl[c];
    #pragma omp parallel for schedule(static)
    for (int j = 0; j < N; ++j)
        for (int i = 0; i < d; ++i) {
            double acc = 0.0;
            for (int64_t c = 0; c < Tc; ++c)
                acc += dz[c * N + j] * widen(h_old, c * (int64_t)d + i, dtype);
            grad[(int64_t)j * d + i] = (Tc > 0) ? acc / (double)Tc : 0.0;
        }
    free(dz); free(kl);
    return bad;
}

/* ---- Sec. 5 "Top-k Agreement and Route KL", "Deviation Tails" ----------------------------- */

/*
 * Route tracking of a cached route against the current router.  I_t = TopK(rho_t, k) of the
 * current routing distribution (rho[T,N] fp32 as stored, exact in double; ties to the lower
 * expert, as in Eq. pr2_route), Î_t = idx_cached[t].  overlap_t = |Î_t ∩ I_t|, where an entry
 * outside [0,N) or repeated within its token never matches.  hist[k - overlap_t] += 1 (the
 * deviation count of "Deviation Tails", 0..k); returns sum_t overlap_t, so the top-k agreement
 * averaged over tokens is that sum / (T k).
 */
int64_t oracle_route_diagnostics(int64_t T, int N, int k, const float* rho,
                                 const int32_t* idx_cached, int64_t* hist) {
    for (int c = 0; c <= k; ++c) hist[c] = 0;
    int64_t total = 0;
    double* r = (double*)malloc(sizeof(double) * (size_t)N);
    double* tv = (double*)malloc(sizeof(double) * (size_t)(k + 1));
    int32_t* sel = (int32_t*)malloc(sizeof(int32_t) * (size_t)k);
    char* taken = (char*)malloc((size_t)N);
    for (int64_t t = 0; t < T; ++t) {
        for (int j = 0; j < N; ++j) r[j] = (double)rho[t * (int64_t)N + j];
        topk(r, N, k, sel, tv, taken);                 /* sets taken[e] for the k+1 best */
        memset(taken, 0, (size_t)N);
        for (int s = 0; s < k; ++s) taken[sel[s]] = 1;  /* keep exactly I_t */
        int ov = 0;
        for (int s = 0; s < k; ++s) {
            int32_t e = idx_cached[t * k + s];
            int ok = (e >= 0 && e < N);
            for (int s2 = 0; ok && s2 < s; ++s2) if (idx_cached[t * k + s2] == e) ok = 0;
            if (ok && taken[e]) ++ov;
        }
        hist[k - ov] += 1;
        total += ov;
    }
    free(r); free(tv); free(sel); free(taken);
    return total;
}

/* ---- Algorithm 2 feature cache, App. "uniform sub-sampling" --------------------------------- */

/*
 * Feature-cache writer: store the route-recording features (h_old, p_old) of the T_c retained
 * positions of a T-token rollout (Algorithm 2: "store route-recording features when (tau,l) is
 * retained by the fixed-length feature cache").  Reading of "drawn by uniform sub-sampling along
 * the rollout": evenly spaced positions pos_c = floor(c T / T_c), c < T_c <= T, so the whole
 * rollout is covered (T_c = T keeps every token).  cache_h[c] = h[pos_c] (esz-byte elements,
 * bits copied), cache_p[c] = logits[pos_c] (fp32).
 */
void oracle_feature_cache(int64_t T, int64_t Tc, int d, int N, int esz, const void* h,
                          const float* logits, int32_t* pos, void* cache_h, float* cache_p) {
    for (int64_t c = 0; c < Tc; ++c) {
        int64_t p = (c * T) / Tc;
        pos[c] = (int32_t)p;
        memcpy((char*)cache_h + c * (int64_t)d * esz, (const char*)h + p * (int64_t)d * esz,
               (size_t)d * (size_t)esz);
        memcpy(cache_p + c * (int64_t)N, logits + p * (int64_t)N, sizeof(float) * (size_t)N);
    }
}
