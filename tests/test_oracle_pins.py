"""Pins of the fp64 oracle against what the paper and the mathematics fix (CPU only).

Each check is independent of the oracle's own code path: hand-worked examples (tests/golden),
closed forms, a library routine for the quantile, brute force over all subsets for Eq. 6, the
degenerate settings that reduce EAT to fixed Top-K or to a fixed probability threshold, and
invariants of the account state.  The mutation tests at the end plant plausible mistakes in the
oracle and check that some pin catches each one.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

import oracle.eat_oracle as orc

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "worked_examples.json")))
REL = 1e-12


def close(a, b, tol=REL):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return np.allclose(a, b, rtol=tol, atol=tol)


def acc_from(d):
    return orc.Accounts(np.array(d["N"], np.int64), np.array(d["P"], np.float64),
                        np.array(d["C"], np.float64))


P0 = orc.Params(max_k=2)


# ---------------------------------------------------------------- worked examples (tests/golden)
def check_w1(m):
    w = GOLD["W1"]
    acc = m.Accounts.zeros(4)
    s_h = m.history_score(acc, P0)
    assert close(s_h, np.zeros(4))
    sels = []
    for tok in w["tokens"]:
        p = np.array(tok["p"])
        th = m.threshold(p, P0, 0)
        assert close(th.mu, tok["mu"]) and close(th.sigma, tok["sigma"])
        assert close(th.tau, tok["tau"])
        assert close(th.q_lo, tok["q_lo"]) and close(th.q_hi, tok["q_hi"])
        assert close(th.tau_final, tok["tau_final"])
        I = m.importance(p, s_h, P0.beta)
        assert close(I, tok["I"])
        sel = m.select(I, th.tau_final, P0.max_k)
        assert sel == tok["selected"]
        assert close(m.renormalize(p, sel, P0.eps), tok["g_norm"])
        sels.append(sel)
    p = np.array([t["p"] for t in w["tokens"]])
    norms = {(int(k.split(",")[0]), int(k.split(",")[1])): v for k, v in w["norms"].items()}
    after = m.account_update(acc, sels, p, norms, P0.alpha)
    exp = w["state_after"]
    assert list(after.N) == exp["N"]
    assert close(after.P, exp["P"]) and close(after.C, exp["C"])


def check_w2(m):
    w = GOLD["W2"]
    acc = acc_from(w["state"])
    s_h = m.history_score(acc, P0)
    assert close(s_h, w["s_h_sum"])
    assert close(m.history_score(acc, P0.with_(c_mode="raw")), w["s_h_raw"])
    for tok in w["tokens"]:
        p = np.array(tok["p"])
        th = m.threshold(p, P0, 0)
        assert close(th.tau_final, tok["tau_final"])
        I = m.importance(p, s_h, P0.beta)
        assert close(I, tok["I_sum"])
        sel = m.select(I, th.tau_final, P0.max_k)
        assert sel == tok["selected"]
        assert close(m.renormalize(p, sel, P0.eps), tok["g_norm"])
        raw = m.importance(p, m.history_score(acc, P0.with_(c_mode="raw")), P0.beta)
        assert m.select(raw, th.tau_final, P0.max_k) == tok["selected"]
        if "selected_reset_state" in tok:
            I0 = m.importance(p, m.history_score(m.Accounts.zeros(4), P0), P0.beta)
            assert m.select(I0, th.tau_final, P0.max_k) == tok["selected_reset_state"]


def check_w3(m):
    w = GOLD["W3"]
    p = np.array(w["p"])
    I = m.importance(p, np.zeros(4), P0.beta)
    for case in w["cases"]:
        th = m.threshold(p, P0, case["ppl_sign"])
        assert close(th.tau_final, case["tau_final"])
        assert m.select(I, th.tau_final, P0.max_k) == case["selected"]


def check_w4(m):
    w = GOLD["W4"]
    p = np.array(w["p"])
    I = m.importance(p, np.zeros(4), P0.beta)
    for case in w["cases"]:
        th = m.threshold(p, P0, case["ppl_sign"])
        assert close(th.tau, case["tau"]) and close(th.tau_smoothed, case["tau_smoothed"])
        assert close(th.tau_final, case["tau_final"])
        assert m.select(I, th.tau_final, P0.max_k) == case["selected"]


def check_swiglu(m):
    s = GOLD["SWIGLU"]
    out = m.expert_ffn(np.array([s["x"]]), np.array(s["w_gate"]), np.array(s["w_up"]),
                       np.array(s["w_down"]))[0]
    assert close(out, s["out"])
    assert close(np.sqrt((out ** 2).sum()), s["norm"])


def test_w1_reset_state_routing_and_update():
    check_w1(orc)


def test_w2_history_changes_selection():
    check_w2(orc)


def test_w3_ppl_adjustment_flips_selection():
    check_w3(orc)


def test_w4_lower_and_upper_clamp():
    check_w4(orc)


def test_swiglu_hand_example():
    check_swiglu(orc)


# ---------------------------------------------------------------- closed forms
def test_softmax_closed_forms():
    assert close(orc.softmax(np.zeros((1, 7))), np.full((1, 7), 1 / 7))
    z = np.array([[0.3, -1.2]])
    assert close(orc.softmax(z)[0, 0], 1.0 / (1.0 + math.exp(-1.5)))
    big = orc.softmax(np.array([[1000.0, 999.0, -1000.0]]))
    assert np.isfinite(big).all()
    assert close(big[0, 0], 1.0 / (1.0 + math.exp(-1.0) + math.exp(-2000.0)))


def test_router_logits_temperature_and_bias():
    x = np.array([[1.0, 2.0]])
    w = np.array([[0.5, -1.0], [2.0, 0.25]])
    b = np.array([0.1, -0.2])
    # (1*0.5 + 2*-1 + 0.1) / 0.5 = -2.8 ; (1*2 + 2*0.25 - 0.2) / 0.5 = 4.6
    assert close(orc.router_logits(x, w, b, 0.5), [[-2.8, 4.6]])


@pytest.mark.parametrize("n", [1, 2, 3, 4, 7, 8, 60, 64])
def test_quantile_matches_numpy_linear(n):
    rng = np.random.default_rng(n)
    v = rng.random(n)
    for q in (0.0, 0.1, 0.25, 0.5, 0.9, 1.0):
        assert close(orc.quantile_type7(v, q), np.percentile(v, 100 * q, method="linear"))


def test_silu_closed_form():
    assert orc.silu(np.array([0.0]))[0] == 0.0
    assert close(orc.silu(np.array([1.0]))[0], math.e / (1.0 + math.e))
    assert close(orc.silu(np.array([-40.0]))[0], -40.0 * math.exp(-40.0), 1e-9)


def test_ema_closed_form():
    """Repeated calls with a constant norm r: C_n = r (1 - (1 - alpha)^n)."""
    acc = orc.Accounts.zeros(3)
    r, a = 2.5, 0.95
    p = np.array([[0.2, 0.7, 0.1]])
    for n in range(1, 6):
        acc = orc.account_update(acc, [[1]], p, {(0, 1): r}, a)
        assert close(acc.C[1], r * (1.0 - (1.0 - a) ** n))
        assert acc.N[1] == n and close(acc.P[1], 0.7 * n)
        assert acc.C[0] == 0.0 and acc.C[2] == 0.0


def test_ema_uses_batch_mean():
    acc = orc.Accounts(np.array([3, 0]), np.array([1.0, 0.0]), np.array([4.0, 0.0]))
    p = np.array([[0.6, 0.4], [0.3, 0.7]])
    out = orc.account_update(acc, [[0], [0]], p, {(0, 0): 1.0, (1, 0): 3.0}, 0.95)
    assert out.N[0] == 5 and close(out.P[0], 1.9)
    assert close(out.C[0], 0.05 * 4.0 + 0.95 * 2.0)
    assert out.N[1] == 0 and out.C[1] == 0.0


# ---------------------------------------------------------------- brute force of Eq. 6
def brute_force_eq6(I, tau, K):
    """All subsets S of the experts; with the strict order i > j  <=>  I_i > I_j or (I_i == I_j
    and i < j), Eq. 6 picks S = {i in E : #{j in E : j > i} < K} when E is non-empty and
    S = {the maximum of the order} when E is empty.  Returns every subset meeting that."""
    n = len(I)
    above = lambda j, i: I[j] > I[i] or (I[j] == I[i] and j < i)
    cand = {i for i in range(n) if I[i] > tau}
    hits = []
    for r in range(1, n + 1):
        for S in itertools.combinations(range(n), r):
            S = set(S)
            if not cand:
                ok = len(S) == 1 and all(not above(j, next(iter(S))) for j in range(n))
            else:
                ok = S == {i for i in cand if sum(above(j, i) for j in cand) < K}
            if ok:
                hits.append(sorted(S))
    return hits


@pytest.mark.parametrize("E", [1, 2, 3, 5, 8, 10])
def test_select_brute_force(E):
    rng = np.random.default_rng(100 + E)
    for trial in range(40):
        I = rng.random(E)
        if trial % 4 == 0 and E > 2:           # planted ties
            I[rng.integers(E)] = I[0]
            I[-1] = I[1]
        if trial % 5 == 0:
            I = np.round(I, 1)
        tau = float(rng.choice([0.0, 0.3, 0.5, 0.8, 1.1]))
        for K in range(1, E + 1):
            hits = brute_force_eq6(list(I), tau, K)
            assert len(hits) == 1
            assert orc.select(I, tau, K) == hits[0]


# ---------------------------------------------------------------- degenerate settings
def random_accounts(rng, E):
    N = rng.integers(0, 50, E)
    P = rng.random(E) * N
    C = rng.random(E) * 10
    return orc.Accounts(N.astype(np.int64), P, C)


def test_degenerate_fixed_topk():
    """beta = 0, alpha1 = 0, alpha2 huge, no clamp, f = 1: tau = 0, every expert is a candidate
    and the K cap leaves vanilla Top-K with Mixtral-style renormalised weights."""
    prm = orc.Params(beta=0.0, alpha1=0.0, alpha2=1e30, clamp=False, max_k=3)
    rng = np.random.default_rng(5)
    E, d = 8, 16
    layer = orc.Layer(rng.normal(size=(E, d)), rng.normal(size=E), None, None, None)
    x = rng.normal(size=(50, d))
    r = orc.route(x, layer, random_accounts(rng, E), prm, 0)
    p = r.p
    for t in range(50):
        order = np.lexsort((np.arange(E), -p[t]))   # by p desc, index asc
        top = sorted(order[:3].tolist())
        assert r.selected[t] == top
        ref = np.zeros(E)
        ref[top] = p[t, top] / (p[t, top].sum() + 1e-8)
        assert close(r.g_norm[t], ref)


def test_degenerate_fixed_probability_threshold():
    """beta = 0, alpha2 = 0, alpha1 = P E, no clamp, f = 1: tau = max(P, 1/E) = P for P >= 1/E,
    so E_final = {p_i > P} capped to K (argmax when empty): a fixed-probability-threshold router
    of the Top-P family."""
    rng = np.random.default_rng(6)
    E, d, K = 8, 12, 4
    for P in (0.125, 0.2, 0.4):
        prm = orc.Params(beta=0.0, alpha1=P * E, alpha2=0.0, clamp=False, max_k=K)
        layer = orc.Layer(rng.normal(size=(E, d)) * 2, None, None, None, None)
        x = rng.normal(size=(40, d))
        r = orc.route(x, layer, random_accounts(rng, E), prm, 0)
        for t in range(40):
            above = [i for i in range(E) if r.p[t, i] > P]
            order = sorted(above, key=lambda i: -r.p[t, i])
            exp = sorted(order[:K]) if above else [int(np.argmax(r.p[t]))]
            assert r.selected[t] == exp
            desc = sorted(range(E), key=lambda i: (-r.p[t, i], i))
            assert r.selected[t] == sorted(desc[:len(exp)])       # a descending-p prefix


def test_topp_router():
    assert orc.topp_select(np.array([0.1, 0.5, 0.3, 0.1]), 0.6) == [1, 2]
    assert orc.topp_select(np.array([0.1, 0.5, 0.3, 0.1]), 0.4) == [1]
    assert orc.topp_select(np.array([0.25, 0.25, 0.25, 0.25]), 1.0) == [0, 1, 2, 3]
    rng = np.random.default_rng(9)
    for _ in range(50):
        p = orc.softmax(rng.normal(size=(1, 8)) * 2)[0]
        for P in (0.2, 0.4, 0.6):
            s = orc.topp_select(p, P)
            desc = sorted(range(8), key=lambda i: (-p[i], i))
            assert s == sorted(desc[:len(s)])
            assert p[s].sum() >= P
            assert len(s) == 1 or p[sorted(desc[:len(s) - 1])].sum() < P
            # when some expert alone exceeds P (the fixed-threshold router's candidate set is
            # non-empty), the smallest prefix reaching P is that expert alone
            thr = [i for i in range(8) if p[i] > P]
            if thr:
                assert s == [desc[0]]


def test_beta_zero_ignores_history():
    rng = np.random.default_rng(11)
    E, d = 16, 10
    layer = orc.Layer(rng.normal(size=(E, d)), rng.normal(size=E), None, None, None)
    x = rng.normal(size=(30, d))
    prm = orc.Params(beta=0.0, max_k=4)
    base = orc.route(x, layer, orc.Accounts.zeros(E), prm, 1).selected
    for _ in range(5):
        assert orc.route(x, layer, random_accounts(rng, E), prm, 1).selected == base


# ---------------------------------------------------------------- layer output
def tiny_layer(rng, E, d, F, S=0):
    mk = lambda *s: rng.normal(size=s) * 0.3
    return orc.Layer(mk(E, d), mk(E), mk(E, F, d), mk(E, F, d), mk(E, d, F),
                     mk(S, F, d) if S else None, mk(S, F, d) if S else None,
                     mk(S, d, F) if S else None)


def test_identical_experts_output():
    """All experts equal: y_t = FFN(x_t) * sum_e g_norm,t,e for any selection."""
    rng = np.random.default_rng(3)
    E, d, F = 4, 6, 5
    base = tiny_layer(rng, 1, d, F)
    layer = orc.Layer(rng.normal(size=(E, d)), rng.normal(size=E),
                      np.repeat(base.w_gate, E, 0), np.repeat(base.w_up, E, 0),
                      np.repeat(base.w_down, E, 0))
    x = rng.normal(size=(9, d))
    res = orc.moe_forward(x, layer, orc.Accounts.zeros(E), orc.Params(max_k=3))
    ffn = orc.expert_ffn(x, base.w_gate[0], base.w_up[0], base.w_down[0])
    assert close(res.y, ffn * res.routing.g_norm.sum(1, keepdims=True), 1e-12)


def test_single_expert_hand_output():
    """E = 2, the router forces expert 1 alone: y = g_norm * SwiGLU hand example, and the shared
    expert (weight 1) adds the same hand value again."""
    s = GOLD["SWIGLU"]
    wg, wu, wd = (np.array(s[k]) for k in ("w_gate", "w_up", "w_down"))
    z = np.zeros((1, 2, 2))
    layer = orc.Layer(np.zeros((2, 2)), np.array([-50.0, 50.0]), np.concatenate([z, wg[None]]),
                      np.concatenate([z, wu[None]]), np.concatenate([z, wd[None]]))
    x = np.array([s["x"]])
    res = orc.moe_forward(x, layer, orc.Accounts.zeros(2), orc.Params(max_k=2))
    assert res.routing.selected == [[1]]
    g = res.routing.g_norm[0, 1]
    assert close(g, 1.0 / (1.0 + math.exp(-100.0)) / (1.0 / (1.0 + math.exp(-100.0)) + 1e-8))
    assert close(res.y[0], g * np.array(s["out"]))
    assert close(res.norms[(0, 1)], s["norm"])
    layer.ws_gate, layer.ws_up, layer.ws_down = wg[None], wu[None], wd[None]
    res2 = orc.moe_forward(x, layer, orc.Accounts.zeros(2), orc.Params(max_k=2))
    assert close(res2.y[0], (g + 1.0) * np.array(s["out"]))
    assert res2.accounts_after.N.tolist() == [0, 1]


def test_token_output_matches_forward():
    rng = np.random.default_rng(4)
    layer = tiny_layer(rng, 6, 8, 7, S=2)
    x = rng.normal(size=(12, 8))
    acc = random_accounts(rng, 6)
    prm = orc.Params(max_k=3)
    res = orc.moe_forward(x, layer, acc, prm)
    for t in (0, 5, 11):
        y, norms = orc.token_output(x[t], layer, res.routing, t)
        assert close(y, res.y[t], 1e-12)
        for e, v in norms.items():
            assert close(v, res.norms[(t, e)])


# ---------------------------------------------------------------- invariants over a run
def test_invariants_multi_step():
    rng = np.random.default_rng(21)
    E, d, F, K = 8, 16, 12, 3
    layer = tiny_layer(rng, E, d, F)
    prm = orc.Params(max_k=K)
    acc = orc.Accounts.zeros(E)
    max_norm = 0.0
    for step in range(12):
        x = rng.normal(size=(10, d))
        sign = int(rng.choice([-1, 0, 1]))
        res = orc.moe_forward(x, layer, acc, prm, sign)
        k = res.routing.k
        assert (k >= 1).all() and (k <= min(K, E)).all()
        gs = res.routing.g_norm.sum(1)
        assert ((gs > 1 - 1e-7) & (gs <= 1.0)).all()
        for th in res.routing.thresholds:
            assert th.q_lo - 1e-15 <= th.tau_final <= th.q_hi + 1e-15
        max_norm = max([max_norm] + list(res.norms.values()))
        new = res.accounts_after
        assert (new.N >= acc.N).all() and new.N.dtype == np.int64
        assert (new.P >= acc.P).all() and (new.P <= new.N + 1e-12).all() and (new.P >= 0).all()
        assert (new.C >= 0).all() and (new.C <= max_norm + 1e-12).all()
        assert new.N.sum() == acc.N.sum() + k.sum()
        assert close((new.N / new.N.sum()).sum(), 1.0)
        acc = new


def test_reset_is_reproducible():
    rng = np.random.default_rng(8)
    layer = tiny_layer(rng, 5, 6, 4)
    x = rng.normal(size=(7, 6))
    a = orc.moe_forward(x, layer, orc.Accounts.zeros(5), orc.Params(max_k=2))
    b = orc.moe_forward(x, layer, orc.Accounts.zeros(5), orc.Params(max_k=2))
    assert np.array_equal(a.y, b.y)
    assert a.routing.selected == b.routing.selected
    for f in ("N", "P", "C"):
        assert np.array_equal(getattr(a.accounts_after, f), getattr(b.accounts_after, f))


# ---------------------------------------------------------------- planted mistakes
def _pins(m):
    """Run every pin against module m; returns the names that fail."""
    failed = []
    for name, fn in (("w1", check_w1), ("w2", check_w2), ("w3", check_w3), ("w4", check_w4),
                     ("swiglu", check_swiglu), ("w6", check_w6)):
        try:
            fn(m)
        except AssertionError:
            failed.append(name)
    rng = np.random.default_rng(1)
    try:
        for _ in range(30):
            I = np.round(rng.random(6), 1)
            for K in (1, 2, 3):
                if m.select(I, 0.3, K) != brute_force_eq6(list(I), 0.3, K)[0]:
                    raise AssertionError
    except AssertionError:
        failed.append("brute")
    return failed


MUTANTS = {
    "drop_w3_term": ("history_score",
                     lambda orig: lambda acc, prm: orig(acc, prm.with_(w3=0.0))),
    "sample_std": ("threshold", None),
    "non_strict_compare": ("select", None),
    "gate_up_swapped": ("expert_ffn",
                        lambda orig: lambda x, g, u, d: orig(x, u, g, d)),
    "clamp_before_smoothing": ("threshold", None),
    "ema_alpha_on_old": ("account_update",
                         lambda orig: lambda acc, sel, p, n, a: orig(acc, sel, p, n, 1.0 - a)),
    "importance_beta_swapped": ("importance",
                                lambda orig: lambda p, s, b: orig(p, s, 1.0 - b)),
    "drop_w1_term": ("history_score",
                     lambda orig: lambda acc, prm: orig(acc, prm.with_(w1=0.0))),
    "renorm_over_all_experts": ("renormalize",
                                lambda orig: lambda g, sel, eps: (np.asarray(g, np.float64) *
                                                                  orig(g, sel, eps).astype(bool)) /
                                (np.asarray(g, np.float64).sum() + eps)),
    "ppl_factor_sign_flipped": ("ppl_factor",
                                lambda orig: lambda sign, prm: orig(-sign, prm)),
    "perplexity_of_summed_nll": ("perplexity",
                                 lambda orig: lambda nll: float(math.exp(np.sum(nll)))),
    "norm_squared_in_account": ("account_update",
                                lambda orig: lambda acc, sel, p, n, a:
                                orig(acc, sel, p, {k: v * v for k, v in n.items()}, a)),
}


def _threshold_sample_std(g, prm, ppl_sign=0):
    g = np.asarray(g, np.float64)
    n = g.shape[0]
    mu = g.mean()
    sigma = math.sqrt(((g - mu) ** 2).sum() / (n - 1))
    tau = max(prm.alpha1 * mu, mu - prm.alpha2 * sigma)
    tau_s = prm.kappa1 * orc.ppl_factor(ppl_sign, prm) * tau + prm.kappa2 * tau
    lo, hi = orc.quantile_type7(g, prm.q_lo), orc.quantile_type7(g, prm.q_hi)
    return orc.Threshold(mu, sigma, tau, tau_s, lo, hi, min(max(tau_s, lo), hi))


def _threshold_clamp_first(g, prm, ppl_sign=0):
    g = np.asarray(g, np.float64)
    mu = g.mean()
    sigma = math.sqrt(((g - mu) ** 2).mean())
    tau = max(prm.alpha1 * mu, mu - prm.alpha2 * sigma)
    lo, hi = orc.quantile_type7(g, prm.q_lo), orc.quantile_type7(g, prm.q_hi)
    tau_ppl = min(max(orc.ppl_factor(ppl_sign, prm) * tau, lo), hi)
    tau_s = prm.kappa1 * tau_ppl + prm.kappa2 * tau
    return orc.Threshold(mu, sigma, tau, tau_s, lo, hi, tau_s)


def _select_non_strict(I, tau, K):
    cand = [i for i in range(len(I)) if I[i] >= tau]
    if not cand:
        return [int(np.argmax(I))]
    return sorted(sorted(cand, key=lambda i: (-I[i], i))[:K])


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, monkeypatch):
    attr, wrap = MUTANTS[name]
    if name == "sample_std":
        repl = _threshold_sample_std
    elif name == "clamp_before_smoothing":
        repl = _threshold_clamp_first
    elif name == "non_strict_compare":
        repl = _select_non_strict
    else:
        repl = wrap(getattr(orc, attr))
    assert _pins(orc) == []
    monkeypatch.setattr(orc, attr, repl)
    assert _pins(orc) != [], f"mutant {name} survived every pin"


# ---------------------------------------------------------------- baselines and OPD (§3.5, §4.1)
def test_topk_router_equals_degenerate_eat():
    """router "topk" and the degenerate EAT setting (beta 0, alpha1 0, alpha2 huge, no clamp)
    are two formulations of vanilla Top-K: same selections and gates."""
    rng = np.random.default_rng(31)
    E, d = 12, 9
    layer = orc.Layer(rng.normal(size=(E, d)), rng.normal(size=E), None, None, None)
    x = rng.normal(size=(40, d))
    acc = random_accounts(rng, E)
    a = orc.route(x, layer, acc, orc.Params(router="topk", max_k=3), 1)
    b = orc.route(x, layer, acc, orc.Params(beta=0.0, alpha1=0.0, alpha2=1e30, clamp=False,
                                            max_k=3), 0)
    assert a.selected == b.selected
    assert close(a.g_norm, b.g_norm)


def test_topp_router_hand_and_cap():
    p = np.array([0.1, 0.5, 0.3, 0.1])
    assert orc.topp_select(p, 0.6) == [1, 2]            # 0.5 < 0.6, 0.5 + 0.3 >= 0.6
    assert orc.topp_select(p, 0.85, K=2) == [1, 2]      # would need a third expert; capped at K
    assert orc.topp_select(p, 0.85) == [0, 1, 2]        # ties 0.1/0.1 -> lower index first
    layer = orc.Layer(np.zeros((4, 1)), np.log(p), None, None, None)
    r = orc.route(np.zeros((1, 1)), layer, orc.Accounts.zeros(4),
                  orc.Params(router="topp", top_p=0.6, max_k=4))
    assert r.selected == [[1, 2]]
    assert close(r.g_norm[0], [0.0, 0.5 / (0.8 + 1e-8), 0.3 / (0.8 + 1e-8), 0.0])


def test_opd_reweighting():
    p = np.array([[0.5, 0.5], [0.2, 0.8]])
    assert close(orc.opd_reweight(p, np.array([3.0, 1.0])), [[0.75, 0.25], [3 * 0.2 / 1.4, 0.8 / 1.4]])
    assert close(orc.opd_reweight(p, np.array([2.0, 2.0])), p)   # uniform scales: identity
    assert close(orc.opd_reweight(p, None), p)
    # the reweighted distribution drives selection: a large scale on expert 0 flips token 2
    layer = orc.Layer(np.zeros((2, 1)), np.log(np.array([0.2, 0.8])), None, None, None,
                      opd_scale=np.array([9.0, 1.0]))
    r = orc.route(np.zeros((1, 1)), layer, orc.Accounts.zeros(2), orc.Params(router="topk",
                                                                             max_k=1))
    assert r.selected == [[0]] and close(r.p[0], [1.8 / 2.6, 0.8 / 2.6])


# ---------------------------------------------------------------- temporal smoothing (W5)
def check_w5(m):
    w = GOLD["W5"]
    p = np.array(w["p"])
    prm = P0.with_(smoothing="temporal")
    I = m.importance(p, np.zeros(4), prm.beta)
    for case in w["cases"]:
        prev = float("nan") if case["tau_prev"] is None else case["tau_prev"]
        th = m.threshold(p, prm, 0, prev)
        assert close(th.tau_final, case["tau_final"])
        assert m.select(I, th.tau_final, prm.max_k) == case["selected"]


def test_w5_temporal_smoothing():
    check_w5(orc)


def check_w6(m):
    prev = float("nan")
    for win in GOLD["W6"]["windows"]:
        sign, curr = m.ppl_sign_update(prev, np.array(win["nll"]))
        assert sign == win["sign"] and close(curr, win["ppl"])
        prev = curr


def test_w6_ppl_sign_from_likelihoods():
    check_w6(orc)


def test_perplexity_closed_forms():
    """PPL of a constant likelihood c is e^c; the sign follows the mean NLL (exp is monotone), a
    window no worse than the last gives -1 ('otherwise'), and a NaN likelihood gives no signal."""
    rng = np.random.default_rng(21)
    for c in (0.0, 0.3, 2.5, 7.0):
        assert close(orc.perplexity(np.full(5, c)), math.exp(c))
    for _ in range(50):
        a, b = rng.uniform(0, 5, 7), rng.uniform(0, 5, 3)
        s, _ = orc.ppl_sign_update(orc.perplexity(a), b)
        assert s == (1 if b.mean() > a.mean() else -1)
    assert orc.ppl_sign_update(math.exp(1.0), np.array([1.0]))[0] == -1
    assert orc.ppl_sign_update(1.0, np.array([np.nan, 1.0]))[0] == 0
    assert orc.ppl_sign_update(float("nan"), np.array([1.0])) == (0, math.e)


def test_temporal_equals_call_when_prev_is_tau():
    rng = np.random.default_rng(44)
    for _ in range(20):
        p = orc.softmax(rng.normal(size=(1, 8)))[0]
        a = orc.threshold(p, P0, 1)
        b = orc.threshold(p, P0.with_(smoothing="temporal"), 1, a.tau)
        assert close(a.tau_final, b.tau_final)


def test_nan_token_selects_nothing_and_leaves_accounts():
    """Reading R15: a token with a non-finite hidden state has NaN routing probabilities; in every
    router mode it selects no expert, its output row is NaN, and the other tokens' outputs and the
    account update equal those of the same call without it."""
    import oracle.eat_oracle as orc
    rng = np.random.default_rng(13)
    E, d, F, T = 6, 16, 12, 9
    layer = orc.Layer(rng.normal(0, 0.3, (E, d)), rng.normal(0, 0.5, E),
                      rng.normal(0, 0.2, (E, F, d)), rng.normal(0, 0.2, (E, F, d)),
                      rng.normal(0, 0.2, (E, d, F)))
    x = rng.normal(0, 1, (T, d))
    x[2, 5] = np.nan
    x[6, 0] = np.inf
    keep = [t for t in range(T) if t not in (2, 6)]
    acc = orc.Accounts(np.array([3, 0, 5, 1, 2, 4], np.int64), rng.uniform(0, 2, E),
                       rng.uniform(0, 1, E))
    for router in ("eat", "topk", "topp"):
        prm = orc.Params(max_k=2, router=router)
        full = orc.moe_forward(x, layer, acc, prm)
        part = orc.moe_forward(x[keep], layer, acc, prm)
        assert full.routing.selected[2] == [] and full.routing.selected[6] == []
        assert np.isnan(full.y[2]).all() and np.isnan(full.y[6]).all()
        assert np.allclose(full.y[keep], part.y, rtol=1e-12, atol=1e-14)
        assert np.array_equal(full.accounts_after.N, part.accounts_after.N)
        assert np.allclose(full.accounts_after.P, part.accounts_after.P, rtol=1e-13)
        assert np.allclose(full.accounts_after.C, part.accounts_after.C, rtol=1e-13)
        assert np.array_equal(full.accounts_after.N, acc.N + np.bincount(
            [e for t in keep for e in full.routing.selected[t]], minlength=E))
