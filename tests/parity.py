"""Parity protocol between the CUDA path (through the C ABI) and the fp64 oracle.

Selection: expert sets and k bit-exact on every token whose importance lies more than
delta = 1e-5 * max(1, |tau_final|) from its threshold (and from the K-th / (K+1)-th candidate and
the top-two argmax decisions); the remaining "ambiguous" tokens must hold a selection that is valid
for importances and threshold perturbed by delta.  Accounts: each step starts from the GPU's own
pre-step accounts (teacher forcing); N exact, P_total within 1e-6 relative, the C_s update rule
within 1e-6 relative given the GPU's per-expert norm sums, C_s against the oracle's norms within a
dtype-dependent bound.  Layer output: max over tokens of ||y_gpu - y_ref||_inf / ||y_ref||_inf.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

import oracle.eat_oracle as orc

from tests.helpers import np64

# one line per full-size parity step (worst output error, near-tie tokens), printed at the end of
# the session by tests/conftest.py
REPORT: list = []


def delta_of(tau):
    return 1e-5 * max(1.0, abs(tau))


def ambiguous(I: np.ndarray, tau: float, K: int) -> bool:
    dl = delta_of(tau)
    if np.min(np.abs(I - tau)) <= dl:
        return True
    cand = np.sort(I[I > tau])[::-1]
    if cand.size > K and cand[K - 1] - cand[K] <= dl:
        return True
    if cand.size == 0:
        top = np.sort(I)[::-1]
        if top.size > 1 and top[0] - top[1] <= dl:
            return True
    return False


def valid_selection(sel: list, I: np.ndarray, tau: float, K: int) -> bool:
    """Could `sel` be the Eq. 6 result for importances / threshold within delta of (I, tau)?"""
    dl = delta_of(tau)
    if not 1 <= len(sel) <= K or len(set(sel)) != len(sel):
        return False
    if len(sel) == 1 and I[sel[0]] >= I.max() - dl:
        argmax_ok = True
    else:
        argmax_ok = False
    for i in sel:
        if not (I[i] > tau - dl or argmax_ok):
            return False
    lo = min(I[i] for i in sel)
    for j in range(I.shape[0]):
        if j in sel:
            continue
        if I[j] > tau + dl and not (len(sel) == K and I[j] <= lo + dl):
            return False
    return True


@dataclass
class StepReport:
    n_ambiguous: int
    max_rel_y: float
    max_rel_w: float
    n_tokens: int


def gpu_selection(idx: torch.Tensor, k: torch.Tensor) -> list:
    idx = idx.cpu().numpy()
    k = k.cpu().numpy()
    return [idx[t, :k[t]].tolist() for t in range(idx.shape[0])]


def _desc(p):
    return sorted(range(p.shape[0]), key=lambda i: (-p[i], i))


def ambiguous_baseline(p: np.ndarray, K: int, mode: str, top_p: float) -> bool:
    """Top-K: the K-th and (K+1)-th probabilities within delta.  Top-P: additionally any
    cumulative probability before the first K + 1 ranks within delta of P."""
    dl = 1e-5
    order = _desc(p)
    q = p[order]
    if any(q[i] - q[i + 1] <= dl for i in range(min(K, q.size - 1))):
        return True
    if mode == "topp":
        cum = np.concatenate([[0.0], np.cumsum(q)])
        if np.any(np.abs(cum[:K + 1] - top_p) <= dl):
            return True
    return False


def valid_baseline(sel: list, p: np.ndarray, K: int, mode: str, top_p: float) -> bool:
    """A descending-p prefix (within delta) of admissible length."""
    dl = 1e-5
    L = len(sel)
    if not 1 <= L <= K or len(set(sel)) != L:
        return False
    lo = min(p[i] for i in sel)
    if any(p[j] > lo + dl for j in range(p.shape[0]) if j not in sel):
        return False
    if mode == "topk":
        return L == K
    tot = sum(p[i] for i in sel)
    return (L == K or tot >= top_p - dl) and tot - lo < top_p + dl


def check_routing(routing: orc.Routing, sel_gpu: list, w_gpu: np.ndarray, K: int,
                  w_tol: float = 1e-5, mode: str = "eat", top_p: float = 0.6):
    """Returns (ambiguous token list, max relative gate error on the others)."""
    amb = []
    max_w = 0.0
    for t, sel in enumerate(sel_gpu):
        I, tau = routing.I[t], routing.tau_final[t]
        assert sel == sorted(sel), f"token {t}: idx not ascending {sel}"
        if np.isnan(routing.p[t]).any():  # reading R15: no expert, zero gates
            assert sel == [] and np.all(w_gpu[t] == 0.0), f"token {t}: NaN p selected {sel}"
            continue
        if mode != "eat":
            if ambiguous_baseline(routing.p[t], K, mode, top_p):
                amb.append(t)
                assert valid_baseline(sel, routing.p[t], K, mode, top_p), \
                    f"token {t}: GPU {mode} selection {sel} invalid"
                continue
        elif ambiguous(I, tau, K):
            amb.append(t)
            assert valid_selection(sel, I, tau, K), \
                f"token {t}: GPU selection {sel} invalid near the threshold (tau={tau})"
            continue
        assert sel == routing.selected[t], \
            f"token {t}: GPU {sel} != oracle {routing.selected[t]} (tau={tau:.9g})"
        ref = routing.g_norm[t, sel]
        got = w_gpu[t, :len(sel)]
        max_w = max(max_w, float(np.max(np.abs(got - ref) / np.abs(ref))))
        assert np.all(w_gpu[t, len(sel):] == 0.0)
    assert max_w <= w_tol, f"gate error {max_w} > {w_tol}"
    return amb, max_w


def substituted(routing: orc.Routing, sel_gpu: list, amb: list, eps: float) -> list:
    """The oracle's selections with the GPU's choice on the ambiguous tokens."""
    sel = [list(s) for s in routing.selected]
    for t in amb:
        sel[t] = list(sel_gpu[t])
    return sel


def oracle_outputs(x64: np.ndarray, layer: orc.Layer, routing: orc.Routing, sel: list,
                   eps: float, tokens=None):
    """Layer outputs and norms of the oracle for a given selection (all tokens or a sample)."""
    T = x64.shape[0]
    toks = range(T) if tokens is None else tokens
    g_norm = {t: orc.renormalize(routing.p[t], sel[t], eps) for t in toks}
    y = {}
    norms = {}
    for t in toks:
        yt = np.zeros(x64.shape[1])
        for e in sel[t]:
            o = orc.expert_ffn(x64[t:t + 1], layer.w_gate[e], layer.w_up[e], layer.w_down[e])[0]
            yt += g_norm[t][e] * o
            norms[(t, e)] = float(np.sqrt((o ** 2).sum()))
        y[t] = yt
    if layer.ws_gate is not None:
        idx = list(toks)
        sh = orc.shared_output(x64[idx], layer)
        for r, t in enumerate(idx):
            y[t] = y[t] + sh[r]
    for t in toks:
        if not sel[t]:
            y[t] = np.full(x64.shape[1], np.nan)  # reading R15
    return y, norms


def oracle_outputs_batched(x64, layer, routing, sel, eps):
    """Same as oracle_outputs over all tokens, batching rows per expert (library matmuls)."""
    T, d = x64.shape
    y = np.zeros((T, d))
    norms = {}
    for e in range(layer.n_experts):
        toks = [t for t in range(T) if e in sel[t]]
        if not toks:
            continue
        o = orc.expert_ffn(x64[toks], layer.w_gate[e], layer.w_up[e], layer.w_down[e])
        for r, t in enumerate(toks):
            g = orc.renormalize(routing.p[t], sel[t], eps)[e]
            y[t] += g * o[r]
            norms[(t, e)] = float(np.sqrt((o[r] ** 2).sum()))
    y += orc.shared_output(x64, layer)
    for t in range(T):
        if not sel[t]:
            y[t] = np.nan  # reading R15
    return y, norms


def rel_err_rows(y_gpu: np.ndarray, y_ref: np.ndarray) -> np.ndarray:
    """Per row: max |gpu - ref| / max |ref|; a NaN reference row (reading R15) matches only an
    all-NaN GPU row (error 0, else inf)."""
    nan_ref = np.isnan(y_ref).all(axis=1)
    yr = np.where(nan_ref[:, None], 0.0, y_ref)
    yg = np.where(nan_ref[:, None], 0.0, y_gpu)
    den = np.abs(yr).max(axis=1)
    den[den == 0] = 1.0
    err = np.abs(yg - yr).max(axis=1) / den
    err[nan_ref] = np.where(np.isnan(y_gpu[nan_ref]).all(axis=1), 0.0, np.inf)
    err[np.isnan(err)] = np.inf
    return err


def check_accounts(acc_before: orc.Accounts, acc_gpu_after, stats_gpu, routing, sel, norms_ref,
                   alpha, c_tol):
    """acc_gpu_after = (N, P, C) numpy after the GPU step; stats_gpu = (n_e, sum_p, sum_norm)."""
    N_g, P_g, C_g = acc_gpu_after
    n_g, sp_g, sn_g = stats_gpu
    E = acc_before.N.shape[0]
    T = len(sel)
    n_ref = np.zeros(E, np.int64)
    for s in sel:
        for e in s:
            n_ref[e] += 1
    assert np.array_equal(n_g.astype(np.int64), n_ref), f"n_e {n_g} != {n_ref}"
    assert np.array_equal(N_g, acc_before.N + n_ref)
    p_ref = acc_before.P + np.array([sum(routing.p[t, e] for t in range(T) if e in sel[t])
                                     for e in range(E)])
    den = np.maximum(np.abs(p_ref), 1e-30)
    assert np.all(np.abs(P_g - p_ref) / den <= 1e-6), f"P_total {P_g} vs {p_ref}"
    # update rule given the GPU's own norm sums
    C_rule = acc_before.C.copy()
    used = n_g > 0
    C_rule[used] = (1 - alpha) * acc_before.C[used] + alpha * sn_g[used] / n_g[used]
    den = np.maximum(np.abs(C_rule), 1e-30)
    assert np.all(np.abs(C_g - C_rule) / den <= 1e-6), f"C update rule {C_g} vs {C_rule}"
    if norms_ref is not None:
        C_ref = acc_before.C.copy()
        for e in range(E):
            toks = [t for t in range(T) if e in sel[t]]
            if toks:
                C_ref[e] = (1 - alpha) * acc_before.C[e] + \
                    alpha * sum(norms_ref[(t, e)] for t in toks) / len(toks)
        den = np.maximum(np.abs(C_ref), 1e-30)
        err = np.max(np.abs(C_g - C_ref) / den)
        assert err <= c_tol, f"C_s vs oracle norms: {err} > {c_tol}"
