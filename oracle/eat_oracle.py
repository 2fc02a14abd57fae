"""Plain fp64 CPU oracle of one MoE layer forward under EAT (Expert Account Tracker) routing.

TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference leg of ``bench.py`` may import this module.  The CUDA library and its
Python binding never import it, and it imports nothing from them: the two share no code.

Every function restates one step of the method as the paper defines it, in float64 numpy, with
no blocking, fusion or reordering beyond what the definition states.  Inputs stored in bf16 or
fp32 are widened to float64 exactly; nothing is rounded in between.

Paper: "EAT: Expert Account Tracker for Efficient MoE Inference" (arxiv 2609.33614).
  * §3.1  vanilla MoE layer: router -> selected experts -> renormalised weighted sum
  * §3.2  expert account (N, P_total, C_s), history score S_h (Eq. 1), importance I (Eq. 2)
  * §3.3  threshold tau (Eq. 3-5), PPL adjustment (and the perplexity it reads), boundedness,
          smoothing
  * §3.4  candidate set / K cap (Eq. 6), mask and renormalisation (Eq. 7-8)
  * Table 1  hyper-parameter defaults
  * §3.5  OPD inference reweighting of the routing probabilities (scales supplied by the caller)
  * §4.1  Top-P comparison router (P = 0.6 / 0.2 / 0.4) and the vanilla fixed Top-K router

Readings taken where the paper is silent or ambiguous (each is also listed in the design notes):
  R1  the raw gating score g that §3.3 thresholds is the softmax probability p of §3.2 (g == p).
  R2  empty-history terms of Eq. 1 are 0 (N_i/sum N with sum N = 0, P_i/N_i with N_i = 0).
  R3  c_mode "sum" (default): the C_s term of Eq. 1 enters as the share C_i / sum_j C_j;
      c_mode "raw": the literal C_i.
  R4  tau_PPL = f * tau (f = 1.2 after a PPL rise, 0.9 otherwise, 1 without a signal) and the
      smoothing is the same-call blend kappa1 * tau_PPL + kappa2 * tau.
  R4' (optional, smoothing "temporal") the smoothing is an EMA over calls of one token stream:
      kappa1 * tau_PPL + kappa2 * (that stream's previous tau_final).
  R5  tau_min / tau_max are the linear-interpolation ("type 7") 10th / 90th percentiles of the
      token's E routing probabilities, applied after smoothing so tau_final lies in range.
  R6  argmax ties (empty candidate set) go to the lowest expert index.
  R7  the K cap keeps exactly K experts ordered by (I descending, index ascending).
  R8  the renormalised weights use g = p, not I.
  R9  shared experts (configs with always-on experts) are added with weight 1, are not routed
      and have no account.
  R10 routing in one call reads the account snapshot taken before the call; the account update
      is applied after the whole call.
  R11 P_total accumulates the raw probability p of each activation.
  R12 C_s takes one EMA step per call with the batch mean of the unweighted expert-output L2
      norms of that expert's activations; experts with no activation keep C_s.
  R15 a token whose routing probabilities are not all numbers (NaN: a non-finite hidden state
      or router weight) selects no expert, in every router mode; its output row is NaN and it
      adds nothing to the accounts.
  SwiGLU experts: E_e(x) = W_down (silu(W_gate x) * (W_up x)), silu(z) = z / (1 + exp(-z)).

Parity pins (tests/test_oracle_pins.py): hand-worked examples of Eq. 1-8 (tests/golden),
closed forms (softmax, silu, EMA), brute force of Eq. 6 over all subsets, the degenerate
settings that reduce to fixed Top-K and to a fixed probability threshold, invariants of the
account state.  No function here is "parity unpinned".
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
import math

import numpy as np

F64 = np.float64


# ----------------------------------------------------------------------------------------------
# Hyper-parameters (Table 1, §3.3 factors and bounds, Eq. 7 epsilon)
# ----------------------------------------------------------------------------------------------
@dataclass(frozen=True)
class Params:
    alpha: float = 0.95      # EMA smoothing factor of C_s (§3.2, Table 1)
    w1: float = 0.3          # Eq. 1 weights (Table 1)
    w2: float = 0.3
    w3: float = 0.4
    beta: float = 0.6        # Eq. 2 balance (Table 1)
    alpha1: float = 0.5      # Eq. 5 scalings (Table 1)
    alpha2: float = 1.0
    kappa1: float = 0.7      # smoothing weights (§3.3, Table 1)
    kappa2: float = 0.3
    ppl_up: float = 1.2      # tau * (1 + 20%) after a PPL rise (§3.3)
    ppl_down: float = 0.9    # tau * (1 - 10%) otherwise (§3.3)
    q_lo: float = 0.10       # tau_min / tau_max quantiles (§3.3, reading R5)
    q_hi: float = 0.90
    eps: float = 1e-8        # Eq. 7
    temperature: float = 1.0  # logits are divided by it before the softmax
    max_k: int = 2           # K of Eq. 6 (Table 1: 2 for Mixtral/Phi, 8 for Qwen)
    clamp: bool = True       # boundedness enforcement on/off
    c_mode: str = "sum"      # reading R3: "sum" or "raw"
    router: str = "eat"      # "eat" (§3.2-§3.4), or the baselines "topk" / "topp" (§4.1)
    top_p: float = 0.6       # P of the Top-P baseline (§4.1: 0.6 / 0.2 / 0.4)
    smoothing: str = "call"  # reading R4 ("call") or the temporal reading ("temporal", R4')

    def with_(self, **kw) -> "Params":
        return replace(self, **kw)


@dataclass
class Accounts:
    """Per-expert account of §3.2: activation count N, total gating probability P_total and
    the EMA contribution C_s."""
    N: np.ndarray   # int64 [E]
    P: np.ndarray   # float64 [E]
    C: np.ndarray   # float64 [E]

    @staticmethod
    def zeros(n_experts: int) -> "Accounts":
        return Accounts(np.zeros(n_experts, np.int64), np.zeros(n_experts, F64),
                        np.zeros(n_experts, F64))

    def copy(self) -> "Accounts":
        return Accounts(self.N.copy(), self.P.copy(), self.C.copy())


@dataclass
class Layer:
    """One MoE layer in nn.Linear layout: w_router [E, d], b_router [E] or None,
    w_gate / w_up [E, F, d], w_down [E, d, F]; optional always-on shared experts ws_* [S, ...]."""
    w_router: np.ndarray
    b_router: np.ndarray | None
    w_gate: np.ndarray
    w_up: np.ndarray
    w_down: np.ndarray
    ws_gate: np.ndarray | None = None
    ws_up: np.ndarray | None = None
    ws_down: np.ndarray | None = None
    opd_scale: np.ndarray | None = None   # [E] per-expert OPD reweighting scales (§3.5)

    @property
    def n_experts(self) -> int:
        return self.w_router.shape[0]


# ----------------------------------------------------------------------------------------------
# Router (§3.1, §3.2)
# ----------------------------------------------------------------------------------------------
def router_logits(x: np.ndarray, w_router: np.ndarray, b_router: np.ndarray | None,
                  temperature: float = 1.0) -> np.ndarray:
    """Raw routing scores of §3.1: z_t,i = (x_t . w_r,i + b_i) / temperature.  [T, E]."""
    z = np.asarray(x, F64) @ np.asarray(w_router, F64).T
    if b_router is not None:
        z = z + np.asarray(b_router, F64)[None, :]
    return z / F64(temperature)


def opd_reweight(p: np.ndarray, scale: np.ndarray | None) -> np.ndarray:
    """§3.5 OPD inference reweighting: scale each routing probability by the expert's factor and
    renormalise the distribution, p'_i = s_i p_i / sum_j s_j p_j (identity without scales)."""
    if scale is None:
        return np.asarray(p, F64)
    q = np.asarray(p, F64) * np.asarray(scale, F64)[None, :]
    return q / q.sum(axis=-1, keepdims=True)


def softmax(z: np.ndarray) -> np.ndarray:
    """p_i, the router-assigned selection probability of expert i among all experts (§3.2),
    the softmax of the routing scores along the last axis (max subtracted first)."""
    z = np.asarray(z, F64)
    e = np.exp(z - z.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


# ----------------------------------------------------------------------------------------------
# History score and importance (§3.2, Eq. 1 and 2)
# ----------------------------------------------------------------------------------------------
def history_score(acc: Accounts, prm: Params) -> np.ndarray:
    """Eq. 1: S_h,i = w1 * N_i / sum N + w2 * P_total,i / N_i + w3 * C_s,i.

    Readings R2 (empty-history terms are 0) and R3 (c_mode "sum" uses C_i / sum_j C_j)."""
    N = acc.N.astype(F64)
    P = np.asarray(acc.P, F64)
    C = np.asarray(acc.C, F64)
    total_n = N.sum()
    a = N / total_n if total_n > 0 else np.zeros_like(N)
    b = np.zeros_like(N)
    used = N > 0
    b[used] = P[used] / N[used]
    if prm.c_mode == "sum":
        total_c = C.sum()
        c = C / total_c if total_c > 0 else np.zeros_like(C)
    elif prm.c_mode == "raw":
        c = C.copy()
    else:
        raise ValueError(f"unknown c_mode {prm.c_mode!r}")
    return prm.w1 * a + prm.w2 * b + prm.w3 * c


def importance(p: np.ndarray, s_h: np.ndarray, beta: float) -> np.ndarray:
    """Eq. 2: I_i = (1 - beta) * p_i + beta * S_h,i (broadcast over tokens)."""
    return (1.0 - beta) * np.asarray(p, F64) + beta * np.asarray(s_h, F64)


# ----------------------------------------------------------------------------------------------
# Adaptive threshold (§3.3, Eq. 3-5, adjustment, boundedness, smoothing)
# ----------------------------------------------------------------------------------------------
def quantile_type7(v: np.ndarray, q: float) -> float:
    """Linear-interpolation quantile of the values v (reading R5): sort ascending v_(0..n-1),
    h = (n - 1) q, result v_(floor h) + (h - floor h) (v_(floor h + 1) - v_(floor h))."""
    s = np.sort(np.asarray(v, F64))
    n = s.shape[0]
    h = (n - 1) * q
    lo = int(math.floor(h))
    hi = min(lo + 1, n - 1)
    return float(s[lo] + (h - lo) * (s[hi] - s[lo]))


def ppl_factor(ppl_sign: int, prm: Params) -> float:
    """§3.3 performance-based adjustment: PPL rose (sign > 0) -> tau * 1.2, otherwise
    (sign < 0) -> tau * 0.9; sign 0 means no PPL signal for this call -> factor 1."""
    if ppl_sign > 0:
        return prm.ppl_up
    if ppl_sign < 0:
        return prm.ppl_down
    return 1.0


def perplexity(nll: np.ndarray) -> float:
    """The model perplexity §3.3 calibrates tau with: PPL = exp of the mean token negative
    log-likelihood over the tokens of the current window (at least one)."""
    nll = np.asarray(nll, F64)
    return float(math.exp(nll.sum() / nll.shape[0]))


def ppl_sign_update(ppl_prev: float, nll: np.ndarray) -> tuple[int, float]:
    """The sign the §3.3 adjustment reads: +1 when PPL_curr - PPL_prev > 0 (a drop in
    performance), -1 otherwise; 0 when there is no previous perplexity (NaN) or the current one is
    not a number.  Returns (sign, PPL_curr); PPL_curr is the next window's PPL_prev."""
    curr = perplexity(nll)
    if math.isnan(ppl_prev) or math.isnan(curr):
        return 0, curr
    return (1 if curr - ppl_prev > 0 else -1), curr


@dataclass
class Threshold:
    mu: float
    sigma: float
    tau: float
    tau_smoothed: float
    q_lo: float
    q_hi: float
    tau_final: float


def threshold(g: np.ndarray, prm: Params, ppl_sign: int = 0,
              tau_prev: float | None = None) -> Threshold:
    """§3.3 for one token's gating scores g [E] (g = p, reading R1):
    mu = mean g (Eq. 3), sigma = population std (Eq. 4), tau = max(a1 mu, mu - a2 sigma) (Eq. 5),
    tau_PPL = f tau, smoothed kappa1 tau_PPL + kappa2 tau (R4), then clamped to the
    [q_lo, q_hi] quantiles of g (R5).  Temporal reading (R4', smoothing "temporal"): the second
    term is the previous call's tau_final of the same token stream, kappa1 tau_PPL + kappa2
    tau_prev; without a previous value (None or NaN) it falls back to tau."""
    g = np.asarray(g, F64)
    n = g.shape[0]
    mu = g.sum() / n
    sigma = math.sqrt(((g - mu) ** 2).sum() / n)
    tau = max(prm.alpha1 * mu, mu - prm.alpha2 * sigma)
    tau_ppl = ppl_factor(ppl_sign, prm) * tau
    second = tau
    if prm.smoothing == "temporal" and tau_prev is not None and not math.isnan(tau_prev):
        second = float(tau_prev)
    elif prm.smoothing not in ("call", "temporal"):
        raise ValueError(f"unknown smoothing {prm.smoothing!r}")
    tau_s = prm.kappa1 * tau_ppl + prm.kappa2 * second
    lo = quantile_type7(g, prm.q_lo)
    hi = quantile_type7(g, prm.q_hi)
    tau_final = min(max(tau_s, lo), hi) if prm.clamp else tau_s
    return Threshold(float(mu), float(sigma), float(tau), float(tau_s), lo, hi, float(tau_final))


# ----------------------------------------------------------------------------------------------
# Selection and renormalisation (§3.4, Eq. 6-8)
# ----------------------------------------------------------------------------------------------
def select(I: np.ndarray, tau_final: float, K: int) -> list[int]:
    """Eq. 6.  Candidate set E = {i : I_i > tau_final} (strict); empty -> {argmax I} (lowest
    index on ties, R6); more than K -> the K largest by (I desc, index asc) (R7).
    Returns the selected expert indices in ascending order."""
    I = np.asarray(I, F64)
    cand = [i for i in range(I.shape[0]) if I[i] > tau_final]
    if not cand:
        best = 0
        for i in range(1, I.shape[0]):
            if I[i] > I[best]:
                best = i
        return [best]
    if len(cand) <= K:
        return cand
    ranked = sorted(cand, key=lambda i: (-I[i], i))
    return sorted(ranked[:K])


def renormalize(g: np.ndarray, selected: list[int], eps: float) -> np.ndarray:
    """Eq. 7-8: m_i = 1 for selected experts, g_norm,i = g_i m_i / (sum_j g_j m_j + eps)."""
    g = np.asarray(g, F64)
    m = np.zeros_like(g)
    m[list(selected)] = 1.0
    return g * m / ((g * m).sum() + eps)


# ----------------------------------------------------------------------------------------------
# One routing call over T tokens (Eq. 1-8 from one account snapshot, R10)
# ----------------------------------------------------------------------------------------------
@dataclass
class Routing:
    logits: np.ndarray           # [T, E]
    p: np.ndarray                # [T, E]  (= g, R1)
    s_h: np.ndarray              # [E]
    I: np.ndarray                # [T, E]
    thresholds: list             # [T] Threshold
    selected: list               # [T] ascending expert lists
    g_norm: np.ndarray           # [T, E]

    @property
    def k(self) -> np.ndarray:
        return np.array([len(s) for s in self.selected], np.int64)

    @property
    def tau_final(self) -> np.ndarray:
        return np.array([t.tau_final for t in self.thresholds], F64)


def route(x: np.ndarray, layer: Layer, acc: Accounts, prm: Params, ppl_sign: int = 0,
          tau_prev: np.ndarray | None = None) -> Routing:
    """Router -> softmax (-> OPD reweighting, §3.5) -> S_h -> I -> tau_final -> E_final -> g_norm
    for every token, all from the same account snapshot (reading R10).  With router "topk" /
    "topp" the selection is the §4.1 baseline instead of Eq. 6; everything else is unchanged.
    tau_prev [T]: previous tau_final per token stream for the temporal smoothing (NaN: none)."""
    z = router_logits(x, layer.w_router, layer.b_router, prm.temperature)
    p = opd_reweight(softmax(z), layer.opd_scale)
    s_h = history_score(acc, prm)
    I = importance(p, s_h[None, :], prm.beta)
    ths, sels = [], []
    g_norm = np.zeros_like(p)
    for t in range(p.shape[0]):
        th = threshold(p[t], prm, ppl_sign, None if tau_prev is None else float(tau_prev[t]))
        if np.isnan(p[t]).any():
            sel = []  # reading R15
        elif prm.router == "eat":
            sel = select(I[t], th.tau_final, prm.max_k)
        elif prm.router == "topk":
            sel = topk_select(p[t], prm.max_k)
        elif prm.router == "topp":
            sel = topp_select(p[t], prm.top_p, prm.max_k)
        else:
            raise ValueError(f"unknown router {prm.router!r}")
        ths.append(th)
        sels.append(sel)
        g_norm[t] = renormalize(p[t], sel, prm.eps)
    return Routing(z, p, s_h, I, ths, sels, g_norm)


# ----------------------------------------------------------------------------------------------
# Experts and the layer output (§3.1, §3.4 last paragraph)
# ----------------------------------------------------------------------------------------------
def silu(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, F64)
    return z / (1.0 + np.exp(-z))


def expert_ffn(x_rows: np.ndarray, w_gate: np.ndarray, w_up: np.ndarray,
               w_down: np.ndarray) -> np.ndarray:
    """SwiGLU expert on rows x [n, d]: W_down (silu(W_gate x) * (W_up x)) -> [n, d]."""
    x_rows = np.asarray(x_rows, F64)
    gate = x_rows @ np.asarray(w_gate, F64).T
    up = x_rows @ np.asarray(w_up, F64).T
    return (silu(gate) * up) @ np.asarray(w_down, F64).T


def shared_output(x: np.ndarray, layer: Layer) -> np.ndarray:
    """Sum of the always-on shared experts, each with weight 1 (reading R9)."""
    y = np.zeros((x.shape[0], layer.w_router.shape[1]), F64)
    if layer.ws_gate is None:
        return y
    for s in range(layer.ws_gate.shape[0]):
        y += expert_ffn(x, layer.ws_gate[s], layer.ws_up[s], layer.ws_down[s])
    return y


def account_update(acc: Accounts, selected: list, p: np.ndarray, norms: dict,
                   alpha: float) -> Accounts:
    """§3.2 account update after a call (R10-R12):
    N_e += n_e;  P_total,e += sum of p_t,e over the activations of e;
    C_e <- (1 - alpha) C_e + alpha * mean ||E_e(x_t)||_2 over those activations (n_e > 0)."""
    E = acc.N.shape[0]
    out = acc.copy()
    for e in range(E):
        toks = [t for t in range(len(selected)) if e in selected[t]]
        if not toks:
            continue
        out.N[e] += len(toks)
        out.P[e] += sum(float(p[t, e]) for t in toks)
        mean_norm = sum(norms[(t, e)] for t in toks) / len(toks)
        out.C[e] = (1.0 - alpha) * acc.C[e] + alpha * mean_norm
    return out


@dataclass
class ForwardResult:
    y: np.ndarray             # [T, d] float64
    routing: Routing
    norms: dict               # (t, e) -> ||E_e(x_t)||_2
    accounts_after: Accounts


def moe_forward(x: np.ndarray, layer: Layer, acc: Accounts, prm: Params,
                ppl_sign: int = 0, tau_prev: np.ndarray | None = None) -> ForwardResult:
    """One MoE layer call: y_t = sum_{e in E_final(t)} g_norm,t,e E_e(x_t) + shared(x_t), then the
    account update.  One call is one EMA timestep t of §3.2."""
    x = np.asarray(x, F64)
    r = route(x, layer, acc, prm, ppl_sign, tau_prev)
    T = x.shape[0]
    y = np.zeros((T, layer.w_router.shape[1]), F64)
    norms = {}
    for e in range(layer.n_experts):
        toks = [t for t in range(T) if e in r.selected[t]]
        if not toks:
            continue
        out = expert_ffn(x[toks], layer.w_gate[e], layer.w_up[e], layer.w_down[e])
        for row, t in enumerate(toks):
            y[t] += r.g_norm[t, e] * out[row]
            norms[(t, e)] = float(np.sqrt((out[row] ** 2).sum()))
    y += shared_output(x, layer)
    for t in range(T):
        if not r.selected[t]:
            y[t] = np.nan  # reading R15
    new_acc = account_update(acc, r.selected, r.p, norms, prm.alpha)
    return ForwardResult(y, r, norms, new_acc)


def token_output(x_t: np.ndarray, layer: Layer, routing: Routing, t: int) -> tuple:
    """Layer output of one token t given a routing of the call (for sampled checks at sizes where
    the full forward is too slow): returns (y_t [d], {e: ||E_e(x_t)||})."""
    x_t = np.asarray(x_t, F64)[None, :]
    y = np.zeros(layer.w_router.shape[1], F64)
    norms = {}
    for e in routing.selected[t]:
        out = expert_ffn(x_t, layer.w_gate[e], layer.w_up[e], layer.w_down[e])[0]
        y += routing.g_norm[t, e] * out
        norms[e] = float(np.sqrt((out ** 2).sum()))
    y += shared_output(x_t, layer)[0]
    if not routing.selected[t]:
        y[:] = np.nan  # reading R15
    return y, norms


# ----------------------------------------------------------------------------------------------
# Comparison router of §4.1 (Top-P, Huang et al.) -- oracle only
# ----------------------------------------------------------------------------------------------
def topp_select(p: np.ndarray, P: float, K: int | None = None) -> list[int]:
    """Top-P routing: take experts in descending probability (index ascending on ties) until
    their cumulative probability reaches P; the smallest such prefix, at most K experts when K is
    given.  Ascending indices."""
    p = np.asarray(p, F64)
    order = sorted(range(p.shape[0]), key=lambda i: (-p[i], i))
    chosen, acc = [], 0.0
    for i in order:
        if K is not None and len(chosen) == K:
            break
        chosen.append(i)
        acc += p[i]
        if acc >= P:
            break
    return sorted(chosen)


def topk_select(p: np.ndarray, K: int) -> list[int]:
    """Vanilla fixed Top-K routing (§2, §4.1): the K largest probabilities, index ascending on
    ties.  Ascending indices."""
    p = np.asarray(p, F64)
    return sorted(sorted(range(p.shape[0]), key=lambda i: (-p[i], i))[:K])
