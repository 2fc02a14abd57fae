"""The C-ABI library: it loads, exports every entry point include/eat.h declares, and rejects
invalid arguments on the host before touching a device (no compute call is made here)."""
import ctypes
import os
import re

import pytest

from paper_2609_33614_gb300 import build, eat

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return eat.lib()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "eat.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\**\s+\**(eat_\w+)\s*\(", src, flags=re.M)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(eat._SIGS), "binding and header disagree"


def test_default_params_are_table1(lib):
    p = eat.eat_default_params()
    assert (p.alpha, p.w1, p.w2, p.w3, p.beta) == (0.95, 0.3, 0.3, 0.4, 0.6)
    assert (p.alpha1, p.alpha2, p.kappa1, p.kappa2) == (0.5, 1.0, 0.7, 0.3)
    assert (p.ppl_up, p.ppl_down, p.q_lo, p.q_hi, p.eps) == (1.2, 0.9, 0.1, 0.9, 1e-8)
    assert (p.temperature, p.max_k, p.clamp_enabled, p.c_mode) == (1.0, 2, 1, eat.EAT_C_SUM)
    assert (p.router_mode, p.top_p) == (eat.EAT_ROUTER_EAT, 0.6)
    assert lib.eat_default_params(None) == eat.EAT_ERR_INVALID_ARG


def _desc(**kw):
    base = dict(d_model=256, n_experts=8, d_ff=512, n_shared=0, d_ff_shared=0, max_tokens=64,
                wdtype=eat.EAT_F32, xdtype=eat.EAT_F32, w_router=16, b_router=None,
                w_gate=4096, w_up=8192, w_down=12288, ws_gate=None, ws_up=None, ws_down=None,
                opd_scale=None, w_gate_scale=None, w_up_scale=None, w_down_scale=None,
                ws_gate_scale=None, ws_up_scale=None, ws_down_scale=None)
    base.update(kw)
    return eat.eat_layer_desc(*[base[n] for n, _ in eat.eat_layer_desc._fields_])


@pytest.mark.parametrize("kw,params,status", [
    (dict(n_experts=0), {}, eat.EAT_ERR_UNSUPPORTED),
    (dict(n_experts=257), {}, eat.EAT_ERR_UNSUPPORTED),
    (dict(d_model=100), {}, eat.EAT_ERR_UNSUPPORTED),
    (dict(d_ff=96), {}, eat.EAT_ERR_UNSUPPORTED),
    (dict(n_shared=2, d_ff_shared=0), {}, eat.EAT_ERR_UNSUPPORTED),
    (dict(max_tokens=0), {}, eat.EAT_ERR_INVALID_ARG),
    (dict(wdtype=eat.EAT_BF16), {}, eat.EAT_ERR_UNSUPPORTED),
    (dict(wdtype=eat.EAT_FP8_E4M3), {}, eat.EAT_ERR_UNSUPPORTED),          # fp8 needs bf16 x
    (dict(wdtype=eat.EAT_FP8_E4M3, xdtype=eat.EAT_BF16), {}, eat.EAT_ERR_INVALID_ARG),  # no scales
    (dict(wdtype=eat.EAT_FP8_E4M3, xdtype=eat.EAT_BF16, w_gate_scale=64, w_up_scale=64,
          w_down_scale=64, n_shared=1, d_ff_shared=64, ws_gate=4096, ws_up=4096, ws_down=4096),
     {}, eat.EAT_ERR_INVALID_ARG),                                                   # shared scales
    (dict(w_gate=None), {}, eat.EAT_ERR_INVALID_ARG),
    (dict(w_up=4100), {}, eat.EAT_ERR_INVALID_ARG),
    (dict(n_shared=1, d_ff_shared=64), {}, eat.EAT_ERR_INVALID_ARG),
    ({}, dict(max_k=0), eat.EAT_ERR_INVALID_ARG),
    ({}, dict(max_k=9), eat.EAT_ERR_INVALID_ARG),
    ({}, dict(temperature=0.0), eat.EAT_ERR_INVALID_ARG),
    ({}, dict(q_lo=0.95), eat.EAT_ERR_INVALID_ARG),
    ({}, dict(c_mode=7), eat.EAT_ERR_INVALID_ARG),
    ({}, dict(alpha=1.5), eat.EAT_ERR_INVALID_ARG),
    ({}, dict(router_mode=3), eat.EAT_ERR_INVALID_ARG),
    ({}, dict(router_mode=eat.EAT_ROUTER_TOPP, top_p=0.0), eat.EAT_ERR_INVALID_ARG),
])
def test_create_rejects_invalid_layers(lib, kw, params, status):
    h = ctypes.c_void_p(1234)
    p = eat.eat_default_params(**params)
    r = lib.eat_create(ctypes.byref(_desc(**kw)), ctypes.byref(p), ctypes.byref(h))
    assert r == status, lib.eat_last_error(None)
    assert h.value is None
    assert lib.eat_last_error(None)


def test_null_handle_calls(lib):
    assert lib.eat_create(None, None, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_route(None, 1, 1, 0, 1, 1, 1, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_moe_forward(None, 1, 1, 0, 1, None, None, None, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_moe_forward_host(None, 1, 1, 0, 1, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_moe_forward_host_async(None, 1, 1, 0, 1, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_reset_accounts(None, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_destroy(None) == eat.EAT_OK
    assert lib.eat_ffn_backend(None) == -1
    assert lib.eat_status_string(eat.EAT_ERR_CUDA) == b"EAT_ERR_CUDA"
    assert lib.eat_status_string(99) == b"EAT_UNKNOWN_STATUS"
    out = ctypes.c_uint32(7)
    assert lib.eat_selftest_bounded_wait(10, ctypes.byref(out)) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_selftest_bounded_wait(10**6, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_selftest_expire_wait(None, 10**6, None) == eat.EAT_ERR_INVALID_ARG


def test_binding_raises_with_message(lib):
    with pytest.raises(eat.EatError) as ei:
        eat._check(lib.eat_route(None, 1, 1, 0, 1, 1, 1, None))
    assert ei.value.status == eat.EAT_ERR_INVALID_ARG
    assert "null handle" in str(ei.value)


def test_layer_policy_and_ppl_argument_checks(lib):
    """eat_layer_policy is host arithmetic on the params (§5.2: the lower three quarters of a
    stack sparser, the upper quarter unchanged); eat_ppl_update rejects bad arguments before any
    launch."""
    for n_layers, K in ((32, 2), (26, 6), (4, 8)):
        for layer in range(n_layers):
            p = eat.eat_layer_policy(layer, n_layers, eat.eat_default_params(K))
            low = layer < (3 * n_layers) // 4
            assert p.max_k == (max(1, K // 3) if low else K)
            assert p.alpha1 == (1.0 if low else 0.5)
            assert (p.beta, p.alpha2, p.kappa1) == (0.6, 1.0, 0.7)
    p = eat.eat_default_params(2)
    assert lib.eat_layer_policy(3, 3, ctypes.byref(p)) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_layer_policy(-1, 3, ctypes.byref(p)) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_layer_policy(0, 3, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_ppl_update(None, 4, 64, 64, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_ppl_update(64, 0, 64, 64, None) == eat.EAT_ERR_INVALID_ARG
    assert b"n >= 1" in lib.eat_last_error(None)
    assert lib.eat_ppl_update(64, 4, 68, 64, None) == eat.EAT_ERR_INVALID_ARG
    assert lib.eat_set_ppl_sign_source(None, None) == eat.EAT_ERR_INVALID_ARG

