"""Pins for the CPU oracle: each check compares it with something other than itself.

The paper prints no worked numeric example of the layer, so the pins are closed forms, special
cases that reduce to a textbook or library routine, brute force on tiny inputs, and the
inequalities of App. B (Lemma topk_regret, Pinsker).  ``test_oracle_mutants.py`` plants
plausible mistakes in copies of the oracle and checks that these pins catch each one.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2606_00395_gb300 import synth


def _rand(shape, seed, scale=1.0):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(*shape, generator=g) * scale).contiguous()


def _f64(t):
    return t.double().numpy()


# ------------------------------------------------------------------ routing (Sec. 4.1)

def test_softmax_rows_sum_to_one():
    h, W, Wp = _rand((64, 32), 1), _rand((16, 32), 2, 0.3), _rand((16, 32), 3, 0.3)
    r = oracle.route_predict(h, W, Wp, 4)
    assert np.all(np.abs(r["probs"].sum(1) - 1.0) < 1e-12)
    assert np.all(r["probs"] > 0)


def test_selector_rows_give_closed_form_logits_and_softmax():
    """W rows are basis vectors: p_e = h[pi(e)] exactly, so rho-hat has a closed form.

    A transposed weight read, a wrong row index, or a dropped predictor term changes these."""
    T, d, N, k = 8, 12, 5, 2
    pi = [7, 0, 11, 3, 5]
    h = _rand((T, d), 4)
    W = torch.zeros(N, d)
    for e, i in enumerate(pi):
        W[e, i] = 1.0
    Wp = torch.zeros(N, d)
    Wp[2, 1] = 0.5  # b_2 = 0.5 * h[:, 1]
    r = oracle.route_predict(h, W, Wp, k)
    hd = _f64(h)
    logits = np.stack([hd[:, i] for i in pi], 1)
    assert np.array_equal(r["logits"], logits)
    for t in range(T):
        z = [hd[t, pi[e]] + (0.5 * hd[t, 1] if e == 2 else 0.0) for e in range(N)]
        den = sum(math.exp(v) for v in z)
        for e in range(N):
            assert abs(r["probs"][t, e] - math.exp(z[e]) / den) < 1e-14


def test_two_experts_is_a_sigmoid_of_the_logit_gap():
    h, W, Wp = _rand((32, 8), 5), _rand((2, 8), 6, 0.5), _rand((2, 8), 7, 0.5)
    r = oracle.route_predict(h, W, Wp, 1)
    z = _f64(h) @ _f64(W).T + _f64(h) @ _f64(Wp).T
    sig = 1.0 / (1.0 + np.exp(z[:, 1] - z[:, 0]))
    assert np.max(np.abs(r["probs"][:, 0] - sig)) < 1e-14


@pytest.mark.parametrize("N", [1, 2, 5, 16])
def test_topk_equals_brute_force_sort(N):
    T, d = 48, 6
    h, W, Wp = _rand((T, d), 10 + N), _rand((N, d), 20 + N), _rand((N, d), 30 + N, 0.2)
    for k in range(1, N + 1):
        r = oracle.route_predict(h, W, Wp, k)
        for t in range(T):
            order = sorted(range(N), key=lambda e: (-r["probs"][t, e], e))
            assert list(r["idx"][t]) == order[:k]
            assert np.array_equal(r["gates"][t], r["probs"][t, order[:k]])
            want = r["probs"][t, order[k - 1]] - r["probs"][t, order[k]] if k < N else math.inf
            assert r["margin"][t] == want


def test_uniform_router_breaks_ties_to_lower_index():
    """W = W_p = 0 gives rho-hat = 1/N; W_p = -W cancels the router exactly (sign of b)."""
    T, d, N, k = 6, 10, 7, 3
    h = _rand((T, d), 40)
    W = _rand((N, d), 41)
    for Wr, Wq in ((torch.zeros(N, d), torch.zeros(N, d)), (W, -W)):
        r = oracle.route_predict(h, Wr, Wq, k)
        assert np.array_equal(r["idx"], np.tile(np.arange(k, dtype=np.int32), (T, 1)))
        assert np.all(r["gates"] == 1.0 / N)
        assert np.all(r["margin"] == 0.0)


def test_zero_predictor_is_plain_topk_routing():
    """W_p = 0 reduces Pr^2 rollout routing to the router's own top-k (routing replay, R2)."""
    T, d, N, k = 40, 16, 12, 3
    h, W = _rand((T, d), 50), _rand((N, d), 51, 0.4)
    r = oracle.route_predict(h, W, torch.zeros(N, d), k)
    p = _f64(h) @ _f64(W).T
    ref = np.argsort(-p, axis=1, kind="stable")[:, :k]
    assert np.array_equal(r["idx"], ref)
    rep = oracle.route_replay(h, W, r["idx"])
    assert np.array_equal(rep["gates"], r["gates"]) and rep["bad"] == 0


def test_predictor_alone_routes_by_its_own_projection():
    """W = 0: the route is the top-k of h W_p (the predictor term is present and added)."""
    T, d, N, k = 40, 16, 12, 3
    h, Wp = _rand((T, d), 52), _rand((N, d), 53, 0.4)
    r = oracle.route_predict(h, torch.zeros(N, d), Wp, k)
    b = _f64(h) @ _f64(Wp).T
    assert np.array_equal(r["idx"], np.argsort(-b, axis=1, kind="stable")[:, :k])
    assert np.all(r["logits"] == 0.0)  # p_old excludes the predictor bias


def test_replay_gates_gather_current_router_probabilities():
    T, d, N, k = 30, 16, 10, 4
    h, W = _rand((T, d), 60), _rand((N, d), 61, 0.4)
    idx = np.stack([np.random.default_rng(t).permutation(N)[:k] for t in range(T)]).astype(np.int32)
    rep = oracle.route_replay(h, W, idx)
    p = _f64(h) @ _f64(W).T
    ref = np.exp(p - p.max(1, keepdims=True))
    ref /= ref.sum(1, keepdims=True)
    assert np.max(np.abs(rep["probs"] - ref)) < 1e-14
    assert np.array_equal(rep["gates"], np.take_along_axis(rep["probs"], idx, 1))


def test_normalized_gates_sum_to_one_and_reduce_in_special_cases():
    """The optional renormalisation (PR2_F_NORMALIZE_TOPK): each row of selected gates sums to
    1; k = 1 gives exactly 1; k = N leaves the gates (rho-hat sums to 1 over all experts); a
    uniform router gives 1/k; invalid replay slots stay 0 and the valid ones sum to 1."""
    T, d, N, k = 24, 16, 9, 3
    h, W, Wp = _rand((T, d), 70), _rand((N, d), 71, 0.4), _rand((N, d), 72, 0.4)
    r = oracle.route_predict(h, W, Wp, k, normalize=True)
    plain = oracle.route_predict(h, W, Wp, k)
    assert np.array_equal(r["idx"], plain["idx"]) and np.array_equal(r["probs"], plain["probs"])
    assert np.max(np.abs(r["gates"].sum(1) - 1.0)) < 1e-14
    assert np.all(r["gates"] > plain["gates"])  # k < N: the sum of the selected is below 1
    one = oracle.route_predict(h, W, Wp, 1, normalize=True)
    assert np.all(one["gates"] == 1.0)
    full = oracle.route_predict(h, W, Wp, N, normalize=True)
    assert np.max(np.abs(full["gates"] - np.take_along_axis(full["probs"], full["idx"], 1))) < 1e-14
    uni = oracle.route_predict(h, torch.zeros(N, d), torch.zeros(N, d), k, normalize=True)
    assert np.max(np.abs(uni["gates"] - 1.0 / k)) < 1e-15
    idx = plain["idx"].copy()
    idx[0, 1] = N            # invalid
    idx[1, :] = -1           # every slot invalid
    rep = oracle.route_replay(h, W, idx, normalize=True)
    assert rep["gates"][0, 1] == 0.0 and abs(rep["gates"][0].sum() - 1.0) < 1e-14
    assert np.all(rep["gates"][1] == 0.0)
    assert np.max(np.abs(rep["gates"][2:].sum(1) - 1.0)) < 1e-14


def test_replay_flags_invalid_and_duplicate_indices():
    T, d, N = 4, 8, 6
    h, W = _rand((T, d), 62), _rand((N, d), 63)
    idx = np.array([[0, 1], [6, 2], [-1, 3], [4, 4]], np.int32)
    rep = oracle.route_replay(h, W, idx)
    assert rep["bad"] == 3
    assert rep["gates"][1, 0] == 0 and rep["gates"][2, 0] == 0 and rep["gates"][3, 1] == 0
    assert rep["gates"][3, 0] == rep["probs"][3, 4]


def _kl(p, q):
    return float(np.sum(p * (np.log(p) - np.log(q))))


def test_lemma_topk_regret_and_margin_condition():
    """App. B, Lemma topk_regret: p(S*) - p(S_hat) <= sqrt(2 KL(p||p_hat)); if
    KL < Delta_k(p)^2 / 2 the supports coincide; Pinsker: ||p - p_hat||_inf <= sqrt(KL/2)."""
    T, d, N, k = 400, 24, 16, 4
    h = _rand((T, d), 70)
    W = _rand((N, d), 71, 0.5)
    hits = 0
    for trial, scale in enumerate((0.002, 0.02, 0.1, 0.5)):
        Wp = _rand((N, d), 72 + trial, scale)
        pred = oracle.route_predict(h, W, Wp, k)                     # rho-hat = Softmax(p + b)
        cur = oracle.route_predict(h, W, torch.zeros(N, d), k)       # rho = Softmax(p), TopK
        for t in range(T):
            p, q = cur["probs"][t], pred["probs"][t]
            kl = _kl(p, q)
            s_star, s_hat = cur["idx"][t], pred["idx"][t]
            assert p[s_star].sum() - p[s_hat].sum() <= math.sqrt(2 * kl) + 1e-15
            assert np.max(np.abs(p - q)) <= math.sqrt(kl / 2) + 1e-15
            if kl < cur["margin"][t] ** 2 / 2:
                hits += 1
                assert set(s_star) == set(s_hat)
    assert hits > 100  # the margin branch is exercised


# ------------------------------------------------------------------ dispatch

@pytest.mark.parametrize("T,k,N", [(1, 1, 1), (37, 3, 5), (64, 8, 16), (0, 2, 4)])
def test_permute_is_a_stable_counting_sort(T, k, N):
    rng = np.random.default_rng(T * 100 + k)
    idx = np.array([rng.permutation(N)[:k] for _ in range(T)], np.int32).reshape(T, k)
    r = oracle.permute(idx, N)
    flat = idx.reshape(-1)
    assert np.array_equal(r["counts"], np.bincount(flat, minlength=N))
    assert r["counts"].sum() == T * k and r["offsets"][N] == T * k
    assert list(r["perm"]) == sorted(range(T * k), key=lambda f: (flat[f], f))
    assert np.array_equal(r["inv"][r["perm"]], np.arange(T * k))


def test_permute_skips_invalid_slots():
    idx = np.array([[1, 1], [0, 9], [2, -3]], np.int32)
    r = oracle.permute(idx, 3)
    assert r["bad"] == 3 and list(r["counts"]) == [1, 1, 1]
    assert list(r["perm"]) == [2, 0, 4] and list(r["inv"]) == [1, -1, 0, -1, 2, -1]


# ------------------------------------------------------------------ experts (App. E.2)

def _swiglu_np(x, Wg, Wu, Wd):
    g = x @ Wg.T
    return ((g / (1.0 + np.exp(-g))) * (x @ Wu.T)) @ Wd.T


def test_single_expert_top1_is_a_dense_swiglu_mlp():
    """N = k = 1: the gate is Softmax of one logit = 1 and the layer is one dense gated MLP."""
    cfg = synth.LayerConfig("t", T=20, d=24, N=1, k=1, m=40, dtype="fp32")
    L = synth.make_layer(cfg, seed=3)
    r = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], 1)
    assert np.all(r["gates"] == 1.0) and np.all(r["idx"] == 0)
    out = oracle.moe_forward(L["x"], r["idx"], r["gates"], L["W_gate"], L["W_up"], L["W_down"])
    ref = _swiglu_np(_f64(L["x"]), _f64(L["W_gate"][0]), _f64(L["W_up"][0]), _f64(L["W_down"][0]))
    assert np.max(np.abs(out - ref)) <= 1e-12 * np.max(np.abs(ref))


def test_permutation_matrix_experts_have_a_closed_form():
    """Wg, Wu, Wd permutation matrices (m = d): y = P3 (silu(P1 x) * (P2 x)) exactly; the
    permutations are not involutions, so any transposed weight read changes the result."""
    d = 7
    p1, p2, p3 = [1, 2, 3, 4, 5, 6, 0], [3, 0, 6, 1, 4, 2, 5], [2, 4, 6, 1, 3, 5, 0]
    def pm(p):
        M = torch.zeros(d, d)
        for r_, c in enumerate(p):
            M[r_, c] = 1.0
        return M
    x = _rand((3, d), 80)
    Wg, Wu, Wd = pm(p1)[None], pm(p2)[None], pm(p3)[None]
    idx = np.zeros((3, 1), np.int32)
    gates = np.array([[1.0], [0.5], [2.0]])
    out = oracle.moe_forward(x, idx, gates, Wg, Wu, Wd)
    for t in range(3):
        xt = [float(v) for v in x[t]]
        a = [xt[p1[j]] / (1.0 + math.exp(-xt[p1[j]])) * xt[p2[j]] for j in range(d)]
        y = [a[p3[c]] for c in range(d)]
        assert np.allclose(out[t], gates[t, 0] * np.array(y), rtol=1e-15, atol=1e-16)


def test_zero_up_projection_gives_zero_output():
    cfg = synth.LayerConfig("t", T=10, d=16, N=4, k=2, m=8, dtype="fp32")
    L = synth.make_layer(cfg, seed=4)
    r = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], 2)
    out = oracle.moe_forward(L["x"], r["idx"], r["gates"], L["W_gate"],
                             torch.zeros_like(L["W_up"]), L["W_down"])
    assert np.all(out == 0.0)


def test_dense_uniform_mixture_is_the_expert_mean():
    """k = N with W = W_p = 0: every gate is 1/N and the layer is the mean of all experts."""
    cfg = synth.LayerConfig("t", T=6, d=16, N=4, k=4, m=8, dtype="fp32")
    L = synth.make_layer(cfg, seed=5)
    Z = torch.zeros(4, 16)
    r = oracle.route_predict(L["x"], Z, Z, 4)
    out = oracle.moe_forward(L["x"], r["idx"], r["gates"], L["W_gate"], L["W_up"], L["W_down"])
    x = _f64(L["x"])
    ref = sum(_swiglu_np(x, _f64(L["W_gate"][e]), _f64(L["W_up"][e]), _f64(L["W_down"][e]))
              for e in range(4)) / 4
    assert np.max(np.abs(out - ref)) <= 1e-12 * np.max(np.abs(ref))


def test_routed_sum_follows_slot_gates_and_experts():
    """Two-slot routing against per-expert dense MLPs (catches a wrong expert offset or a gate
    applied to the wrong slot)."""
    cfg = synth.LayerConfig("t", T=9, d=16, N=5, k=2, m=12, dtype="fp32")
    L = synth.make_layer(cfg, seed=6)
    rng = np.random.default_rng(0)
    idx = np.stack([rng.permutation(5)[:2] for _ in range(9)]).astype(np.int32)
    gates = rng.random((9, 2))
    out = oracle.moe_forward(L["x"], idx, gates, L["W_gate"], L["W_up"], L["W_down"])
    x = _f64(L["x"])
    for t in range(9):
        ref = sum(gates[t, s] * _swiglu_np(x[t:t + 1], _f64(L["W_gate"][e]), _f64(L["W_up"][e]),
                                            _f64(L["W_down"][e]))[0]
                  for s, e in enumerate(idx[t]))
        assert np.max(np.abs(out[t] - ref)) <= 1e-12 * np.max(np.abs(ref))


def test_shared_expert_alone_when_routed_gates_are_zero():
    cfg = synth.LayerConfig("t", T=8, d=16, N=4, k=2, m=8, n_shared=1, dtype="fp32")
    L = synth.make_layer(cfg, seed=7)
    r = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], 2)
    out = oracle.moe_forward(L["x"], r["idx"], np.zeros((8, 2)), L["W_gate"], L["W_up"],
                             L["W_down"], L["Ws_gate"], L["Ws_up"], L["Ws_down"])
    ref = _swiglu_np(_f64(L["x"]), _f64(L["Ws_gate"][0]), _f64(L["Ws_up"][0]),
                     _f64(L["Ws_down"][0]))
    assert np.max(np.abs(out - ref)) <= 1e-12 * np.max(np.abs(ref))


def test_rollout_then_replay_of_its_route_reproduces_the_output():
    """W_p = 0 and the same router: replaying the recorded route gives the rollout output."""
    cfg = synth.LayerConfig("t", T=24, d=16, N=6, k=2, m=8, dtype="fp32")
    L = synth.make_layer(cfg, seed=8)
    Z = torch.zeros_like(L["W_pred"])
    r = oracle.route_predict(L["x"], L["W_router"], Z, 2)
    rep = oracle.route_replay(L["x"], L["W_router"], r["idx"])
    o1 = oracle.moe_forward(L["x"], r["idx"], r["gates"], L["W_gate"], L["W_up"], L["W_down"])
    o2 = oracle.moe_forward(L["x"], r["idx"], rep["gates"], L["W_gate"], L["W_up"], L["W_down"])
    assert np.array_equal(o1, o2)


def test_token_subset_matches_full_run_and_bf16_inputs_widen_exactly():
    cfg = synth.LayerConfig("t", T=12, d=16, N=4, k=2, m=8, dtype="bf16")
    L = synth.make_layer(cfg, seed=9)
    r = oracle.route_predict(L["x"], L["W_router"], L["W_pred"], 2)
    full = oracle.moe_forward(L["x"], r["idx"], r["gates"], L["W_gate"], L["W_up"], L["W_down"])
    sub = oracle.moe_forward(L["x"], r["idx"], r["gates"], L["W_gate"], L["W_up"], L["W_down"],
                             tokens=[11, 0, 5])
    assert np.array_equal(sub, full[[11, 0, 5]])
    # bf16 -> double widening is exact: same values given as fp32 give identical results
    r32 = oracle.route_predict(L["x"].float(), L["W_router"].float(), L["W_pred"].float(), 2)
    assert np.array_equal(r32["logits"], r["logits"]) and np.array_equal(r32["idx"], r["idx"])


# ---- Eq. pr2_loss / Algorithm 3: predictive loss and its W_p gradient ----------------------

def _loss_inputs(Tc=5, d=6, N=4, seed=7):
    g = torch.Generator().manual_seed(seed)
    # W_p on a 2^-10 grid: the +-2^-8 and +-2^-9 finite-difference steps are exact in fp32
    Wp = torch.randint(-64, 65, (N, d), generator=g).float() / 1024
    h = torch.randn(Tc, d, generator=g)
    p_old = torch.randn(Tc, N, generator=g)
    rho = torch.softmax(torch.randn(Tc, N, generator=g).double(), -1).float()
    return h, p_old, Wp, rho


def _dyadic_rho(T, N, g):
    """Teacher rows on a 2^-10 grid summing to exactly 1 (in fp32 and in double)."""
    c = torch.randint(1, 1024 // N, (T, N), generator=g)
    c[:, -1] = 1024 - c[:, :-1].sum(1)
    return (c.double() / 1024).float()


@pytest.mark.parametrize("delta", [False, True])
def test_loss_gradient_matches_finite_differences(delta):
    h, p_old, Wp, rho = _loss_inputs()
    r = oracle.predictor_loss(h, p_old, Wp, rho, delta=delta)
    N, d = Wp.shape
    eps = 2.0 ** -8
    fd = np.zeros((N, d))
    for j in range(N):
        for i in range(d):
            def L(e):
                W = Wp.clone()
                W[j, i] += e
                return oracle.predictor_loss(h, p_old, W, rho, delta=delta)["loss"]
            d1 = (L(eps) - L(-eps)) / (2 * eps)
            d2 = (L(eps / 2) - L(-eps / 2)) / eps
            fd[j, i] = (4 * d2 - d1) / 3  # Richardson: O(eps^4)
    assert np.max(np.abs(fd - r["grad"])) <= 1e-7 * max(1.0, np.max(np.abs(r["grad"])))
    assert r["loss"] > 0 and np.all(r["kl"] >= 0)


@pytest.mark.parametrize("delta", [False, True])
def test_loss_vanishes_at_the_teacher(delta):
    """Teacher rho = Softmax(p_old + h W*^T): the standard loss is 0 at W_p = W*; the delta
    target Softmax(log rho - p_old) = Softmax(h W*^T) is matched by Softmax(b) at W_p = W* too."""
    h, p_old, Wp, _ = _loss_inputs(Tc=7, d=8, N=5, seed=3)
    z = p_old.double() + h.double() @ Wp.double().T
    rho = torch.softmax(z, -1).float()
    r = oracle.predictor_loss(h, p_old, Wp, rho, delta=delta)
    # only the fp32 rounding of rho remains: its rows sum to 1 within ~1e-7
    assert abs(r["loss"]) < 1e-7
    assert np.max(np.abs(r["grad"])) < 1e-6
    other = oracle.predictor_loss(h, p_old, torch.zeros_like(Wp), rho, delta=delta)
    assert other["loss"] > 1e-4


def test_loss_two_experts_closed_form():
    """N = 2: KL of two Bernoulli laws, q = sigmoid(z_1 - z_0)."""
    h, p_old, Wp, _ = _loss_inputs(Tc=6, d=5, N=2, seed=11)
    rho = _dyadic_rho(6, 2, torch.Generator().manual_seed(1))
    r = oracle.predictor_loss(h, p_old, Wp, rho)
    z = p_old.double().numpy() + h.double().numpy() @ Wp.double().numpy().T
    q = 1.0 / (1.0 + np.exp(-(z[:, 1] - z[:, 0])))
    a = rho.double().numpy()[:, 1]
    kl = a * np.log(a / q) + (1 - a) * np.log((1 - a) / (1 - q))
    assert np.max(np.abs(r["kl"] - kl)) <= 1e-12
    assert abs(r["loss"] - kl.mean()) <= 1e-12


def test_loss_shift_invariance_and_delta_equals_standard_at_zero_p_old():
    h, _, Wp, _ = _loss_inputs(Tc=6, d=7, N=5, seed=5)
    g = torch.Generator().manual_seed(2)
    rho = _dyadic_rho(6, 5, g)
    p_old = torch.randint(-128, 128, (6, 5), generator=g).float() / 64  # exact +2 shifts
    a = oracle.predictor_loss(h, p_old, Wp, rho)
    b = oracle.predictor_loss(h, p_old + 2.0, Wp, rho)
    assert abs(a["loss"] - b["loss"]) <= 1e-12
    assert np.max(np.abs(a["grad"] - b["grad"])) <= 1e-12
    z = torch.zeros_like(p_old)
    s = oracle.predictor_loss(h, z, Wp, rho)
    t = oracle.predictor_loss(h, z, Wp, rho, delta=True)
    assert abs(s["loss"] - t["loss"]) <= 1e-12
    assert np.max(np.abs(s["grad"] - t["grad"])) <= 1e-12


def test_loss_rows_follow_pos_and_invalid_rows_are_skipped():
    h, p_old, Wp, rho = _loss_inputs(Tc=4, d=5, N=3, seed=9)
    g = torch.Generator().manual_seed(4)
    full = torch.softmax(torch.randn(9, 3, generator=g).double(), -1).float()
    pos = np.array([7, 0, 3, 5], np.int32)
    a = oracle.predictor_loss(h, p_old, Wp, full, pos=pos)
    b = oracle.predictor_loss(h, p_old, Wp, full[torch.from_numpy(pos).long()])
    assert a["bad"] == 0 and abs(a["loss"] - b["loss"]) <= 1e-15
    assert np.array_equal(a["grad"], b["grad"])
    bad = np.array([7, 9, 3, -1], np.int32)
    c = oracle.predictor_loss(h, p_old, Wp, full, pos=bad)
    keep = oracle.predictor_loss(h[[0, 2]], p_old[[0, 2]], Wp, full[[7, 3]])
    assert c["bad"] == 2 and c["kl"][1] == 0 and c["kl"][3] == 0
    assert abs(c["loss"] * 4 - keep["loss"] * 2) <= 1e-12
    empty = oracle.predictor_loss(h[:0], p_old[:0], Wp, full)
    assert empty["loss"] == 0 and not np.any(empty["grad"])


# ---- Sec. 5: top-k agreement and deviation histogram ----------------------------------------

def test_route_diagnostics_match_brute_force():
    g = torch.Generator().manual_seed(12)
    T, N, k = 40, 9, 3
    # probabilities on a coarse grid so that exact ties occur
    raw = torch.randint(0, 6, (T, N), generator=g).double()
    rho = (raw / raw.sum(1, keepdim=True).clamp(min=1)).float()
    cached = torch.stack([torch.randperm(N, generator=g)[:k] for _ in range(T)]).int().numpy()
    cached[3, 1] = N        # invalid
    cached[5, 2] = cached[5, 0]  # repeated
    r = oracle.route_diagnostics(rho, cached)
    hist = np.zeros(k + 1, np.int64)
    total = 0
    rv = rho.numpy()
    for t in range(T):
        cur = set(sorted(range(N), key=lambda e: (-float(rv[t, e]), e))[:k])
        seen, ov = set(), 0
        for e in cached[t]:
            if 0 <= e < N and e not in seen and e in cur:
                ov += 1
            seen.add(int(e))
        hist[k - ov] += 1
        total += ov
    assert np.array_equal(r["hist"], hist) and r["overlap"] == total
    assert r["agreement"] == total / (T * k)


def test_route_diagnostics_identity_and_disjoint_routes():
    g = torch.Generator().manual_seed(13)
    T, N, k = 16, 10, 4
    rho = torch.softmax(torch.randn(T, N, generator=g).double(), -1).float()
    order = torch.argsort(-rho.double(), dim=1, stable=True).int().numpy()
    same = oracle.route_diagnostics(rho, order[:, :k])
    assert same["hist"][0] == T and same["agreement"] == 1.0
    far = oracle.route_diagnostics(rho, order[:, -k:])
    assert far["hist"][k] == T and far["agreement"] == 0.0


# ---- Algorithm 2: fixed-length feature cache ------------------------------------------------

@pytest.mark.parametrize("Tc", [1, 5, 37])
def test_feature_cache_evenly_spaced_rows(Tc):
    g = torch.Generator().manual_seed(14)
    T, d, N = 37, 8, 6
    h = torch.randn(T, d, generator=g).bfloat16()
    lg = torch.randn(T, N, generator=g)
    r = oracle.feature_cache(h, lg, Tc)
    pos = r["pos"]
    assert list(pos) == [c * T // Tc for c in range(Tc)] and pos[0] == 0
    assert np.all(np.diff(pos) >= 1) and pos[-1] <= T - 1
    assert torch.equal(r["h"], h[torch.from_numpy(pos).long()])
    assert np.array_equal(r["p"], lg.numpy()[pos])


# ---- Algorithm 2 over stacked layers (residual stream) ---------------------------------------

def test_bf16_rounding_of_the_residual_stream_is_round_to_nearest_even():
    x = np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8, 1 + 2.0 ** -8 + 2.0 ** -40, -0.0, 0.0,
                  -(1 + 2.0 ** -8 + 2.0 ** -40), 3.0 * 2.0 ** -20])
    got = oracle._round_to(x, torch.bfloat16).float().numpy()
    want = np.array([1.0, 1 + 2.0 ** -6, 1 + 2.0 ** -7, 0.0, 0.0, -(1 + 2.0 ** -7),
                     3.0 * 2.0 ** -20])
    assert np.array_equal(got, want)
    r = np.random.default_rng(1).standard_normal(4096).astype(np.float32).astype(np.float64)
    assert torch.equal(oracle._round_to(r, torch.bfloat16), torch.from_numpy(r).float().bfloat16())


def test_rollout_layers_compose_single_layers():
    cfg = synth.LayerConfig("t", T=16, d=16, N=4, k=2, m=8, dtype="fp32")
    layers = [synth.make_layer(cfg, seed=20 + l) for l in range(3)]
    h0 = layers[0]["x"]
    r = oracle.rollout_layers(h0, layers, 2)
    cur = h0.double().numpy()
    for l, lw in enumerate(layers):
        one = oracle.route_predict(torch.from_numpy(cur).float(), lw["W_router"], lw["W_pred"], 2)
        assert np.array_equal(one["idx"], r["idx"][l])
        o = oracle.moe_forward(torch.from_numpy(cur).float(), one["idx"], one["gates"],
                               lw["W_gate"], lw["W_up"], lw["W_down"])
        cur = (cur + o).astype(np.float32).astype(np.float64)
    assert np.array_equal(r["h"].numpy(), cur.astype(np.float32))
    # zero up-projections: every layer adds 0, the stream is unchanged, routes stay those of h0
    zl = [dict(lw, W_up=torch.zeros_like(lw["W_up"])) for lw in layers]
    z = oracle.rollout_layers(h0, zl, 2)
    assert torch.equal(z["h"], h0)
    for l, lw in enumerate(zl):
        assert np.array_equal(z["idx"][l],
                              oracle.route_predict(h0, lw["W_router"], lw["W_pred"], 2)["idx"])
