"""Thin ctypes binding of libeat.so (include/eat.h), same names as the C ABI.

Argument marshalling only: every step of the layer runs in the CUDA library.  torch tensors are
used for device memory and streams; pointers are passed as ``tensor.data_ptr()`` and the stream
as ``torch.cuda.current_stream().cuda_stream``.  Loading fails loudly when the library is missing:
there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libeat.so")

EAT_OK, EAT_ERR_INVALID_ARG, EAT_ERR_UNSUPPORTED, EAT_ERR_OOM, EAT_ERR_CUDA, EAT_ERR_STATE = range(6)
EAT_F32, EAT_BF16, EAT_FP8_E4M3 = 0, 1, 2
EAT_C_SUM, EAT_C_RAW = 0, 1
EAT_ROUTER_EAT, EAT_ROUTER_TOPK, EAT_ROUTER_TOPP = 0, 1, 2
EAT_SMOOTH_CALL, EAT_SMOOTH_TEMPORAL = 0, 1
KERNEL_KINDS = ("route", "permute", "ffn_up", "ffn_down", "shared_up", "shared_down", "combine",
                "account", "select", "gather")

c_i32, c_i64, c_dbl, c_vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p


class eat_params(ctypes.Structure):
    _fields_ = [(n, c_dbl) for n in ("alpha", "w1", "w2", "w3", "beta", "alpha1", "alpha2",
                                     "kappa1", "kappa2", "ppl_up", "ppl_down", "q_lo", "q_hi",
                                     "eps", "temperature")] + \
               [("max_k", c_i32), ("clamp_enabled", c_i32), ("c_mode", c_i32),
                ("router_mode", c_i32), ("top_p", c_dbl), ("smoothing_mode", c_i32)]


class eat_layer_desc(ctypes.Structure):
    _fields_ = [(n, c_i32) for n in ("d_model", "n_experts", "d_ff", "n_shared", "d_ff_shared",
                                     "max_tokens", "wdtype", "xdtype")] + \
               [(n, c_vp) for n in ("w_router", "b_router", "w_gate", "w_up", "w_down",
                                    "ws_gate", "ws_up", "ws_down", "opd_scale",
                                    "w_gate_scale", "w_up_scale", "w_down_scale",
                                    "ws_gate_scale", "ws_up_scale", "ws_down_scale")]


class EatError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{status_string(status)}: {msg}")
        self.status = status


_lib = None

# name -> (restype, argtypes)
_SIGS = {
    "eat_default_params": (c_i32, [ctypes.POINTER(eat_params)]),
    "eat_create": (c_i32, [ctypes.POINTER(eat_layer_desc), ctypes.POINTER(eat_params),
                           ctypes.POINTER(c_vp)]),
    "eat_reset_accounts": (c_i32, [c_vp, c_vp]),
    "eat_route": (c_i32, [c_vp, c_vp, c_i32, c_i32, c_vp, c_vp, c_vp, c_vp]),
    "eat_moe_forward": (c_i32, [c_vp, c_vp, c_i32, c_i32, c_vp, c_vp, c_vp, c_vp, c_vp]),
    "eat_moe_forward_host": (c_i32, [c_vp, c_vp, c_i32, c_i32, c_vp, c_vp]),
    "eat_moe_forward_host_async": (c_i32, [c_vp, c_vp, c_i32, c_i32, c_vp, c_vp]),
    "eat_route_noalloc": (c_i32, [c_vp, c_i32, c_i32, c_i32, c_i32, c_vp, c_vp, c_vp, c_vp, c_vp,
                                  ctypes.POINTER(eat_params), c_i32, c_vp, c_vp, c_vp, c_vp]),
    "eat_set_tau_state": (c_i32, [c_vp, c_vp]),
    "eat_ppl_update": (c_i32, [c_vp, c_i32, c_vp, c_vp, c_vp]),
    "eat_set_ppl_sign_source": (c_i32, [c_vp, c_vp]),
    "eat_layer_policy": (c_i32, [c_i32, c_i32, ctypes.POINTER(eat_params)]),
    "eat_destroy": (c_i32, [c_vp]),
    "eat_get_accounts": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_vp]),
    "eat_set_accounts": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_vp]),
    "eat_get_call_stats": (c_i32, [c_vp, c_vp, c_vp, c_vp, c_vp]),
    "eat_get_counters": (c_i32, [c_vp, ctypes.POINTER(c_i64), c_i32]),
    "eat_profile_begin": (c_i32, [c_vp, c_i32]),
    "eat_profile_end": (c_i32, [c_vp, ctypes.POINTER(c_dbl), ctypes.POINTER(c_i64), c_i32]),
    "eat_ffn_backend": (c_i32, [c_vp]),
    "eat_selftest_bounded_wait": (c_i32, [c_i64, ctypes.POINTER(ctypes.c_uint32)]),
    "eat_selftest_expire_wait": (c_i32, [c_vp, c_i64, c_vp]),
    "eat_last_error": (ctypes.c_char_p, [c_vp]),
    "eat_status_string": (ctypes.c_char_p, [c_i32]),
}


def lib():
    """Load libeat.so (built by ``paper_2609_33614_gb300.build``); raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it first "
                               "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def status_string(s: int) -> str:
    return lib().eat_status_string(s).decode()


def _check(status: int, handle=None):
    if status != EAT_OK:
        raise EatError(status, lib().eat_last_error(handle).decode())


def _ptr(t):
    return None if t is None else t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream


def eat_default_params(max_k: int = 2, **overrides) -> eat_params:
    p = eat_params()
    _check(lib().eat_default_params(ctypes.byref(p)))
    p.max_k = max_k
    for k, v in overrides.items():
        setattr(p, k, v)
    return p


def eat_create(desc: eat_layer_desc, params: eat_params) -> int:
    h = c_vp()
    _check(lib().eat_create(ctypes.byref(desc), ctypes.byref(params), ctypes.byref(h)))
    return h.value


def eat_reset_accounts(h, stream=None):
    _check(lib().eat_reset_accounts(h, _stream(stream)), h)


def eat_route(h, x, T, ppl_sign, idx, w, k, stream=None):
    _check(lib().eat_route(h, _ptr(x), T, ppl_sign, _ptr(idx), _ptr(w), _ptr(k),
                           _stream(stream)), h)


def eat_moe_forward(h, x, T, ppl_sign, y, idx=None, w=None, k=None, stream=None):
    _check(lib().eat_moe_forward(h, _ptr(x), T, ppl_sign, _ptr(y), _ptr(idx), _ptr(w), _ptr(k),
                                 _stream(stream)), h)


def eat_moe_forward_host(h, x_host, T, ppl_sign, y_host, stream=None):
    _check(lib().eat_moe_forward_host(h, _ptr(x_host), T, ppl_sign, _ptr(y_host),
                                      _stream(stream)), h)


def eat_moe_forward_host_async(h, x_host, T, ppl_sign, y_host, stream=None):
    """Enqueue-only variant (see include/eat.h): synchronise the stream before reading y_host."""
    _check(lib().eat_moe_forward_host_async(h, _ptr(x_host), T, ppl_sign, _ptr(y_host),
                                            _stream(stream)), h)


def eat_route_noalloc(x, T, d_model, n_experts, xdtype, w_router, b_router, N, P, C, params,
                      ppl_sign, idx, w, k, stream=None):
    """Routing with no device allocation (see include/eat.h): every buffer is the caller's."""
    _check(lib().eat_route_noalloc(_ptr(x), T, d_model, n_experts, xdtype, _ptr(w_router),
                                   _ptr(b_router), _ptr(N), _ptr(P), _ptr(C),
                                   ctypes.byref(params), ppl_sign, _ptr(idx), _ptr(w), _ptr(k),
                                   _stream(stream)))


def eat_set_tau_state(h, tau_state):
    _check(lib().eat_set_tau_state(h, _ptr(tau_state)), h)


def eat_ppl_update(nll, n, ppl_state, sign, stream=None):
    """Perplexity of a window of token NLLs and the sign of its change (see include/eat.h)."""
    _check(lib().eat_ppl_update(_ptr(nll), n, _ptr(ppl_state), _ptr(sign), _stream(stream)))


def eat_set_ppl_sign_source(h, sign):
    _check(lib().eat_set_ppl_sign_source(h, _ptr(sign)), h)


def eat_layer_policy(layer: int, n_layers: int, params: eat_params) -> eat_params:
    """The §5.2 layer-wise adjustment of ``params`` (in place, also returned)."""
    _check(lib().eat_layer_policy(layer, n_layers, ctypes.byref(params)))
    return params


def layer_policy(layer: int, n_layers: int, max_k: int) -> dict:
    """eat_layer_policy applied to the defaults with K = max_k, as eat_params overrides."""
    p = eat_layer_policy(layer, n_layers, eat_default_params(max_k))
    d = eat_default_params(max_k)
    return {"max_k": p.max_k, **({"alpha1": p.alpha1} if p.alpha1 != d.alpha1 else {})}


def eat_destroy(h):
    _check(lib().eat_destroy(h))


def eat_get_accounts(h, N, P, C, stream=None):
    _check(lib().eat_get_accounts(h, _ptr(N), _ptr(P), _ptr(C), _stream(stream)), h)


def eat_set_accounts(h, N, P, C, stream=None):
    _check(lib().eat_set_accounts(h, _ptr(N), _ptr(P), _ptr(C), _stream(stream)), h)


def eat_get_call_stats(h, n_e=None, sum_p=None, sum_norm=None, stream=None):
    _check(lib().eat_get_call_stats(h, _ptr(n_e), _ptr(sum_p), _ptr(sum_norm),
                                    _stream(stream)), h)


def eat_get_counters(h) -> dict:
    out = (c_i64 * 5)()
    _check(lib().eat_get_counters(h, out, 5), h)
    return {"calls": out[0], "union_sum": out[1], "activations": out[2], "launches": out[3],
            "status": out[4]}


def eat_profile_begin(h, capacity: int):
    _check(lib().eat_profile_begin(h, capacity), h)


def eat_profile_end(h) -> dict:
    n = len(KERNEL_KINDS)
    ms = (c_dbl * n)()
    cnt = (c_i64 * n)()
    _check(lib().eat_profile_end(h, ms, cnt, n), h)
    return {KERNEL_KINDS[i]: (ms[i], cnt[i]) for i in range(n)}


def eat_ffn_backend(h) -> int:
    return lib().eat_ffn_backend(h)


def eat_selftest_bounded_wait(limit_ns: int) -> int:
    out = ctypes.c_uint32(0)
    _check(lib().eat_selftest_bounded_wait(limit_ns, ctypes.byref(out)))
    return out.value


def eat_selftest_expire_wait(h, limit_ns: int, stream=None):
    _check(lib().eat_selftest_expire_wait(h, limit_ns, _stream(stream)), h)


# ------------------------------------------------------------------------------------------------
# Convenience wrapper: one layer from torch tensors (still only marshalling).
# ------------------------------------------------------------------------------------------------
class EatLayer:
    """Owns an eat_handle for one MoE layer whose weights are CUDA tensors (kept referenced)."""

    def __init__(self, w_router, b_router, w_gate, w_up, w_down, max_tokens, params,
                 ws_gate=None, ws_up=None, ws_down=None, opd_scale=None, scales=None):
        """Expert weights fp32, bf16, or torch.float8_e4m3fn with ``scales`` = dict of the fp32
        per-row scale tensors (w_gate_scale, w_up_scale, w_down_scale and, with shared experts,
        ws_gate_scale, ws_up_scale, ws_down_scale)."""
        import torch
        scales = scales or {}
        self._keep = [w_router, b_router, w_gate, w_up, w_down, ws_gate, ws_up, ws_down,
                      opd_scale] + list(scales.values())
        fp8 = w_gate.dtype == torch.float8_e4m3fn
        bf16 = w_gate.dtype == torch.bfloat16 or fp8
        E, F, d = w_gate.shape
        S = 0 if ws_gate is None else ws_gate.shape[0]
        Fs = 0 if ws_gate is None else ws_gate.shape[1]
        self.E, self.F, self.d, self.S, self.K = E, F, d, S, params.max_k
        self.dtype = torch.bfloat16 if fp8 else w_gate.dtype  # hidden-state dtype
        self.max_tokens = max_tokens
        wdt = EAT_FP8_E4M3 if fp8 else (EAT_BF16 if bf16 else EAT_F32)
        sc = [_ptr(scales.get(n)) for n in ("w_gate_scale", "w_up_scale", "w_down_scale",
                                             "ws_gate_scale", "ws_up_scale", "ws_down_scale")]
        desc = eat_layer_desc(d, E, F, S, Fs, max_tokens, wdt, EAT_BF16 if bf16 else EAT_F32,
                              _ptr(w_router), _ptr(b_router), _ptr(w_gate), _ptr(w_up),
                              _ptr(w_down), _ptr(ws_gate), _ptr(ws_up), _ptr(ws_down),
                              _ptr(opd_scale), *sc)
        self.params = params
        self.h = eat_create(desc, params)

    @classmethod
    def from_workload(cls, lw, max_tokens, params=None, device="cuda", opd_scale=None):
        """Build from a workloads.LayerWeights or workloads.Fp8LayerWeights (moved to
        ``device`` if needed)."""
        if params is None:
            params = eat_default_params(lw.shape.max_k, temperature=lw.shape.temperature)
        mv = lambda t: None if t is None else t.to(device).contiguous()
        scales = {n: mv(t) for n, t in getattr(lw, "scales", {}).items()}
        return cls(mv(lw.w_router), mv(lw.b_router), mv(lw.w_gate), mv(lw.w_up), mv(lw.w_down),
                   max_tokens, params, mv(lw.ws_gate), mv(lw.ws_up), mv(lw.ws_down),
                   mv(opd_scale), scales=scales)

    def close(self):
        if getattr(self, "h", None):
            eat_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def forward(self, x, ppl_sign=0, with_routing=False):
        import torch
        T = x.shape[0]
        y = torch.empty_like(x)
        if with_routing:
            idx = torch.empty(T, self.K, dtype=torch.int32, device=x.device)
            w = torch.empty(T, self.K, dtype=torch.float32, device=x.device)
            k = torch.empty(T, dtype=torch.int32, device=x.device)
            eat_moe_forward(self.h, x, T, ppl_sign, y, idx, w, k)
            return y, idx, w, k
        eat_moe_forward(self.h, x, T, ppl_sign, y)
        return y

    def route(self, x, ppl_sign=0):
        import torch
        T = x.shape[0]
        idx = torch.empty(T, self.K, dtype=torch.int32, device=x.device)
        w = torch.empty(T, self.K, dtype=torch.float32, device=x.device)
        k = torch.empty(T, dtype=torch.int32, device=x.device)
        eat_route(self.h, x, T, ppl_sign, idx, w, k)
        return idx, w, k

    def accounts(self):
        import torch
        N = torch.empty(self.E, dtype=torch.int64, device="cuda")
        P = torch.empty(self.E, dtype=torch.float64, device="cuda")
        C = torch.empty(self.E, dtype=torch.float64, device="cuda")
        eat_get_accounts(self.h, N, P, C)
        return N, P, C

    def set_accounts(self, N, P, C):
        eat_set_accounts(self.h, N.contiguous(), P.contiguous(), C.contiguous())

    def call_stats(self):
        import torch
        n = torch.empty(self.E, dtype=torch.int32, device="cuda")
        sp = torch.empty(self.E, dtype=torch.float64, device="cuda")
        sn = torch.empty(self.E, dtype=torch.float64, device="cuda")
        eat_get_call_stats(self.h, n, sp, sn)
        return n, sp, sn

    def reset(self):
        eat_reset_accounts(self.h)
