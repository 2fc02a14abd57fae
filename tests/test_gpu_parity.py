"""GPU-vs-oracle parity of the EAT MoE layer through the C ABI (needs a GB300).

Every case draws seeded inputs (paper_2609_33614_gb300.workloads), runs steps through libeat.so and
checks each step against the fp64 oracle from the GPU's own pre-step accounts (teacher forcing):
selections and k bit-exact on non-ambiguous tokens, gates within 1e-5, n_e and N exact, P_total
and the C_s update rule within 1e-6 relative, C_s against the oracle's norms within 1e-6 (fp32)
or 2e-2 (bf16), layer outputs within 1e-5 (fp32) or 2e-2 (bf16) max relative error per token.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle.eat_oracle as orc
from paper_2609_33614_gb300 import eat, workloads as W
from tests import parity as par
from tests.helpers import np64, oracle_layer, oracle_layer_lazy

pytestmark = pytest.mark.gpu

Y_TOL = {torch.float32: 1e-5, torch.bfloat16: 2e-2}
C_TOL = {torch.float32: 1e-6, torch.bfloat16: 2e-2}


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_33614_gb300 import build
    build.build()
    torch.cuda.set_device(0)


def oracle_params(shape, **kw):
    """The oracle's Params for the same settings as the C ABI's eat_params overrides."""
    kw = dict(kw)
    if "c_mode" in kw:
        kw["c_mode"] = "raw" if kw["c_mode"] == eat.EAT_C_RAW else "sum"
    if "clamp_enabled" in kw:
        kw["clamp"] = bool(kw.pop("clamp_enabled"))
    if "smoothing_mode" in kw:
        kw["smoothing"] = "temporal" if kw.pop("smoothing_mode") == eat.EAT_SMOOTH_TEMPORAL \
            else "call"
    if "router_mode" in kw:
        kw["router"] = {eat.EAT_ROUTER_EAT: "eat", eat.EAT_ROUTER_TOPK: "topk",
                        eat.EAT_ROUTER_TOPP: "topp"}[kw.pop("router_mode")]
    return orc.Params(max_k=shape.max_k, temperature=shape.temperature, **kw)


def gpu_params(shape, **kw):
    return eat.eat_default_params(shape.max_k, temperature=shape.temperature, **kw)


def _acc(layer):
    N, P, C = layer.accounts()
    return orc.Accounts(N.cpu().numpy(), P.cpu().numpy(), C.cpu().numpy())


def run_parity(shape, lw, Ts, signs=None, prm_kw=None, layer=None, L=None, sample=None,
               x_device="cpu", max_tokens=None, inputs=None, opd_scale=None, tau_state=None,
               report=None):
    """Run len(Ts) steps and check each one.  sample: number of tokens whose outputs are checked
    (None: all).  inputs: optional list of x tensors replacing the seeded draws.  report: a label;
    when given, each step's worst output error and near-tie count are printed.  Returns the list of
    GPU outputs."""
    prm_kw = prm_kw or {}
    own = layer is None
    if own:
        layer = eat.EatLayer.from_workload(lw, max(Ts) if max_tokens is None else max_tokens,
                                           gpu_params(shape, **prm_kw), opd_scale=opd_scale)
    if L is None:
        L = oracle_layer(lw)
    if opd_scale is not None:
        L.opd_scale = np64(opd_scale)
    prm = oracle_params(shape, **prm_kw)
    if tau_state is not None:
        eat.eat_set_tau_state(layer.h, tau_state)
    outs = []
    rng = np.random.default_rng(99)
    for step, T in enumerate(Ts):
        sign = 0 if signs is None else signs[step]
        x = inputs[step] if inputs is not None else W.make_tokens(shape, T, step=step,
                                                                  device=x_device)
        acc0 = _acc(layer)
        tau_prev = None if tau_state is None else tau_state[:T].cpu().numpy().astype(np.float64)
        y, idx, w, k = layer.forward(x.cuda(), sign, with_routing=True)
        torch.cuda.synchronize()
        n_e, s_p, s_n = (t.cpu().numpy() for t in layer.call_stats())
        N1, P1, C1 = (t.cpu().numpy() for t in layer.accounts())
        x64 = np64(x)
        routing = orc.route(x64, L, acc0, prm, sign, tau_prev)
        if tau_state is not None:
            got = tau_state[:T].cpu().numpy().astype(np.float64)
            assert np.allclose(got, routing.tau_final, rtol=1e-5, atol=1e-9), \
                f"step {step}: stored tau_final differs from the oracle"
        sel_gpu = par.gpu_selection(idx, k)
        amb, _ = par.check_routing(routing, sel_gpu, w.cpu().numpy(), shape.max_k,
                                   mode=prm.router, top_p=prm.top_p)
        sel = par.substituted(routing, sel_gpu, amb, prm.eps)
        y_gpu = np64(y)
        # outputs of every token, with the GPU's (validated) selection on the ambiguous ones
        if sample is None:
            y_ref, norms = par.oracle_outputs_batched(x64, L, routing, sel, prm.eps)
            toks = list(range(T))
            err = par.rel_err_rows(y_gpu, y_ref)
            norms_ref = norms
        else:
            toks = sorted(set(rng.choice(T, size=min(sample, T), replace=False).tolist()))
            yd, _ = par.oracle_outputs(x64, L, routing, sel, prm.eps, toks)
            err = par.rel_err_rows(y_gpu[toks], np.stack([yd[t] for t in toks]))
            norms_ref = None
        assert err.max() <= Y_TOL[shape.xdtype], \
            f"step {step}: output rel err {err.max():.3g} (token {toks[int(err.argmax())]})"
        if report is not None:
            par.REPORT.append(f"parity {shape.name} {report} step {step}: T={T} checked {len(toks)} "
                              f"rows, max rel err {err.max():.3g}, near-tie tokens {len(amb)}")
        par.check_accounts(acc0, (N1, P1, C1), (n_e, s_p, s_n), routing, sel, norms_ref,
                           prm.alpha, C_TOL[shape.xdtype])
        outs.append(y)
    if own:
        layer.close()
    return outs


# ------------------------------------------------------------------ toy (fp32), the full config
def test_toy_16_steps():
    lw = W.make_layer(W.TOY)
    run_parity(W.TOY, lw, [64] * 16)


def test_toy_ppl_signs():
    lw = W.make_layer(W.TOY)
    run_parity(W.TOY, lw, [64] * 16, signs=W.ppl_signs(16))


def test_toy_large_calls():
    """fp32 layer, calls above 128 tokens: the fp32 router-score kernel over the slices the
    stream-K plan sets for the call, and the CUDA-core expert kernels."""
    lw = W.make_layer(W.TOY)
    run_parity(W.TOY, lw, [300, 1100, 64])


def test_toy_c_mode_raw_and_no_clamp():
    lw = W.make_layer(W.TOY)
    run_parity(W.TOY, lw, [64] * 6, prm_kw={"c_mode": eat.EAT_C_RAW})
    run_parity(W.TOY, lw, [64] * 6, prm_kw={"clamp_enabled": 0})


# ------------------------------------------------------------------ reduced bf16 layers
MIX_S = W.scaled(W.MIXTRAL, "mixtral-s", d_model=512, d_ff=704)
OLMOE_S = W.scaled(W.OLMOE, "olmoe-s", d_model=256, d_ff=192)
QWEN_S = W.scaled(W.QWEN, "qwen-s", d_model=256, d_ff=128, d_ff_shared=192)
DSV2L_S = W.scaled(W.DSV2L, "dsv2l-s", d_model=256, d_ff=192, n_layers=3)


def test_mixtral_shaped_ragged():
    lw = W.make_layer(MIX_S)
    run_parity(MIX_S, lw, [1, 37, 200, 64, 5], signs=[0, 1, -1, 0, 1])


def test_olmoe_shaped_k8_temperature():
    lw = W.make_layer(OLMOE_S)
    run_parity(OLMOE_S, lw, [333, 32, 32, 32])


def test_qwen_shaped_shared_experts():
    lw = W.make_layer(QWEN_S)
    run_parity(QWEN_S, lw, [300, 17, 1])


def test_shared_experts_in_the_routed_sm_pair_launches():
    """Calls of 1024 tokens or more run the always-on shared experts' units after the routed ones
    in the same SM-pair launches: full and ragged 256-token shared tiles (1024, 2100), shared
    d_ff (192) unlike the routed one (128), then a small call on the single-SM kernels."""
    lw = W.make_layer(QWEN_S)
    run_parity(QWEN_S, lw, [1024, 2100, 40])


@pytest.mark.parametrize("gate_first", [True, False])
def test_gate_up_interleave_from_one_allocation(gate_first):
    """The SM-pair gate/up tile interleaves 16 gate rows and 16 up rows through a 4D view whose
    stride between the two weight tensors is their distance, with either tensor at the lower
    address: here both are halves of one allocation, up first or gate first, for the routed and
    the shared experts (1100 and 2100 tokens: SM pairs with a ragged last tile)."""
    sh = QWEN_S
    lw = W.make_layer(sh)
    def pair_of(a, b):
        buf = torch.empty((2,) + tuple(a.shape), dtype=a.dtype, device="cuda")
        first, second = (buf[0], buf[1]) if gate_first else (buf[1], buf[0])
        first.copy_(a)
        second.copy_(b)
        return first, second
    wg, wu = pair_of(lw.w_gate, lw.w_up)
    wsg, wsu = pair_of(lw.ws_gate, lw.ws_up)
    assert (wg.data_ptr() < wu.data_ptr()) == gate_first
    layer = eat.EatLayer(lw.w_router.cuda(), lw.b_router.cuda(), wg, wu, lw.w_down.cuda(), 2100,
                         gpu_params(sh), wsg, wsu, lw.ws_down.cuda())
    run_parity(sh, lw, [1100, 2100], layer=layer)
    layer.close()


def test_dsv2l_shaped_residual_chain():
    """Three layers, independent accounts, x_{l+1} = bf16(x_l + y_l) with the GPU's x_l."""
    T = 96
    layers = [W.make_layer(DSV2L_S, l) for l in range(3)]
    x = W.make_tokens(DSV2L_S, T)
    for l, lw in enumerate(layers):
        outs = run_parity(DSV2L_S, lw, [T], inputs=[x])
        x = (x.cuda().float() + outs[0].float()).to(torch.bfloat16).cpu()


# ------------------------------------------------------------------ edge and degenerate cases
def test_single_expert_layer():
    sh = W.scaled(W.TOY, "one-expert", d_model=64, n_experts=1, d_ff=64, max_k=1)
    lw = W.make_layer(sh)
    run_parity(sh, lw, [1, 9, 33])


def test_k_equals_e():
    sh = W.scaled(W.TOY, "k-eq-e", d_model=128, n_experts=4, d_ff=128, max_k=4)
    lw = W.make_layer(sh)
    run_parity(sh, lw, [50, 50, 50])


@pytest.mark.parametrize("E,K,T", [(256, 8, 300), (100, 16, 130), (33, 5, 77)])
def test_expert_counts_and_max_k(E, K, T):
    """Up to 256 experts (8 per lane of the selection warp), a ragged lane layout, K = 16."""
    sh = W.scaled(W.OLMOE, f"e{E}", d_model=256, n_experts=E, d_ff=128, max_k=K)
    lw = W.make_layer(sh)
    run_parity(sh, lw, [T, 1, T // 3])


@pytest.mark.parametrize("E,d", [(64, 256), (100, 192), (256, 512)])
def test_router_runs_split_between_blocks(E, d):
    """Router scores of calls above 128 tokens: a persistent grid takes equal runs of
    (64-token x 64-expert tile, 32-column chunk) units, so tiles are split between blocks at
    chunk boundaries that depend on T, E and d, and the split slices are padded with zero pairs.
    Selections and gates against the oracle (routing only, from seeded accounts) for token
    counts around the tile size and the one-wave point, ragged expert tiles (E = 100) and
    several expert tiles (E = 256); eat_route_noalloc, which may use fewer slices, on the same
    inputs where its scratch holds the call."""
    sh = W.scaled(W.OLMOE, f"rt{E}-{d}", d_model=d, n_experts=E, d_ff=64, max_k=8)
    lw = W.make_layer(sh)
    ref = oracle_layer(lw)
    L = eat.EatLayer.from_workload(lw, 4099, gpu_params(sh))
    L.forward(W.make_tokens(sh, 300, step=9).cuda(), 0)  # some history in the accounts
    prm = orc.Params(max_k=sh.max_k, temperature=sh.temperature)
    for T in (129, 191, 640, 2047, 4099):
        x = W.make_tokens(sh, T, step=T).cuda()
        idx, w, k = L.route(x, 0)
        torch.cuda.synchronize()
        N, P, C = (t.cpu().numpy() for t in L.accounts())
        routing = orc.route(np64(x), ref, orc.Accounts(N, P, C), prm, 0)
        par.check_routing(routing, par.gpu_selection(idx, k), w.cpu().numpy(), sh.max_k)
        if T * E <= (1 << 20) // 8:
            N, P, C = L.accounts()
            idx2 = torch.empty_like(idx)
            w2 = torch.empty_like(w)
            k2 = torch.empty_like(k)
            eat.eat_route_noalloc(x, T, d, E, eat.EAT_BF16, L._keep[0], L._keep[1], N, P, C,
                                  L.params, 0, idx2, w2, k2)
            torch.cuda.synchronize()
            par.check_routing(routing, par.gpu_selection(idx2, k2), w2.cpu().numpy(), sh.max_k)
    L.close()


@pytest.mark.parametrize("E,K,T", [(256, 8, 1500), (64, 2, 1100)])
def test_sm_pair_small_groups(E, K, T):
    """Calls of >= 1024 tokens run the SM-pair GEMMs; with many experts nearly every group is a
    partial 256-token tile (MMA widths of 32..224, one CTA's half of the tile empty or partial),
    and the all-tokens-one-expert call below makes one group span several full tiles."""
    sh = W.scaled(W.OLMOE, f"pair{E}", d_model=256, n_experts=E, d_ff=384, max_k=K)
    lw = W.make_layer(sh)
    run_parity(sh, lw, [T, T])


def test_sm_pair_one_large_group():
    """One expert takes every token of a 2100-token call: 8 full SM-pair tiles and a partial one."""
    lw = W.make_layer(OLMOE_S)
    lw.b_router = torch.full_like(lw.b_router, -30.0)
    lw.b_router[7] = 30.0
    run_parity(OLMOE_S, lw, [2100])


@pytest.mark.parametrize("E,K,T", [(256, 8, 1500), (64, 2, 1100)])
def test_fp8_large_calls_small_groups(E, K, T):
    """e4m3 weights at call sizes where bf16 layers switch to the SM-pair kernels (fp8 layers keep
    the single-SM kernels, 128-token tiles): mostly partial tiles."""
    sh = W.scaled(W.OLMOE, f"pair8-{E}", d_model=256, n_experts=E, d_ff=384, max_k=K)
    lw8 = W.to_fp8(W.make_layer(sh))
    layer = eat.EatLayer.from_workload(lw8, T, gpu_params(sh))
    run_parity(sh, lw8.dequantized(), [T, T], layer=layer)
    layer.close()


def test_fp8_large_call_one_group():
    """e4m3 weights, one expert takes all 2100 tokens: 16 full 128-token tiles and a partial one."""
    lw = W.make_layer(OLMOE_S)
    lw.b_router = torch.full_like(lw.b_router, -30.0)
    lw.b_router[7] = 30.0
    lw8 = W.to_fp8(lw)
    layer = eat.EatLayer.from_workload(lw8, 2100, gpu_params(OLMOE_S))
    run_parity(OLMOE_S, lw8.dequantized(), [2100], layer=layer)
    layer.close()


# ------------------------------------------------------------------ fp8 (e4m3) expert weights
@pytest.mark.parametrize("name,Ts", [("mixtral", [1, 16, 64]), ("olmoe", [32, 300, 1100]),
                                     ("qwen", [64, 200, 1500])])
def test_fp8_weights(name, Ts):
    """e4m3 expert weights with per-row scales, decode sizes and calls of 1100 / 1500 tokens
    (qwen: routed and shared experts); the oracle runs on the dequantized weights."""
    shape = {"mixtral": MIX_S, "olmoe": OLMOE_S, "qwen": QWEN_S}[name]
    lw8 = W.to_fp8(W.make_layer(shape))
    layer = eat.EatLayer.from_workload(lw8, max(Ts), gpu_params(shape))
    assert eat.eat_ffn_backend(layer.h) == 1
    run_parity(shape, lw8.dequantized(), Ts, layer=layer)
    layer.close()


@pytest.mark.parametrize("mode", ["eat", "topk", "topp"])
def test_nonfinite_tokens_select_nothing(mode):
    """Tokens with a NaN or an infinite hidden-state element (reading R15): in every router mode
    they select no expert (k = 0, the rank-based modes included), their output rows are NaN, and
    the other tokens and the accounts follow the oracle."""
    kw = {"eat": {}, "topk": {"router_mode": eat.EAT_ROUTER_TOPK},
          "topp": {"router_mode": eat.EAT_ROUTER_TOPP, "top_p": 0.6}}[mode]
    lw = W.make_layer(QWEN_S)
    x = W.make_tokens(QWEN_S, 40)
    x[5, 3] = float("nan")
    x[9, 100] = float("inf")
    x[39] = float("nan")
    outs = run_parity(QWEN_S, lw, [40], prm_kw=kw, inputs=[x])
    y = outs[0]
    for t in (5, 9, 39):
        assert torch.isnan(y[t]).all()
    assert not torch.isnan(y[[0, 1, 2, 10, 38]]).any()


def test_toy_free_running_first_divergence():
    """The toy configuration run free for 16 steps: the GPU and the oracle each evolve their own
    accounts (no teacher forcing).  Selections must agree token for token until the first step
    that holds a near-tie token (the only legitimate source of a difference, which then feeds
    different accounts into every later step); the step reached is printed."""
    sh = W.TOY
    lw = W.make_layer(sh)
    layer = eat.EatLayer.from_workload(lw, 64, gpu_params(sh))
    L = oracle_layer(lw)
    prm = oracle_params(sh)
    acc = orc.Accounts.zeros(sh.n_experts)
    first = None
    for step in range(16):
        x = W.make_tokens(sh, 64, step=step)
        _, idx, w, k = layer.forward(x.cuda(), 0, with_routing=True)
        res = orc.moe_forward(np64(x), L, acc, prm)
        sel_gpu = par.gpu_selection(idx, k)
        near = [t for t in range(64)
                if par.ambiguous(res.routing.I[t], res.routing.tau_final[t], sh.max_k)]
        diff = [t for t in range(64) if sel_gpu[t] != res.routing.selected[t]]
        if diff:
            assert set(diff) <= set(near), f"step {step}: tokens {diff} differ without a near-tie"
            first = step
            break
        if near:  # a near-tie agreed this time; later accounts may still drift apart
            first = step
            break
        N, P, C = (t.cpu().numpy() for t in layer.accounts())
        assert np.array_equal(N, res.accounts_after.N)
        assert np.allclose(P, res.accounts_after.P, rtol=1e-6)
        assert np.allclose(C, res.accounts_after.C, rtol=1e-5, atol=1e-12)
        acc = res.accounts_after
    print(f"free-running toy: identical through step {15 if first is None else first - 1}")
    layer.close()


@pytest.mark.parametrize("shape,T", [("olmoe", 48), ("qwen", 48), ("olmoe", 1100),
                                     ("qwen", 1100)])
def test_two_handles_on_two_streams_interleaved(shape, T):
    """Two handles (one layer each) driven from two CUDA streams with their calls interleaved give
    the results of running each alone: a handle's workspace and accounts are its own (with shared
    experts, so are the stream and events their small calls fork onto).  At 1100 tokens the two
    handles' persistent SM-pair and stream-K router launches overlap on the GPU."""
    sh = OLMOE_S if shape == "olmoe" else QWEN_S
    lw = W.make_layer(sh)
    xs = [W.make_tokens(sh, T, step=s).cuda() for s in range(4)]
    ref = []
    solo = eat.EatLayer.from_workload(lw, T, gpu_params(sh))
    for x in xs:
        ref.append(solo.forward(x, 0).clone())
    solo.close()
    a = eat.EatLayer.from_workload(lw, T, gpu_params(sh))
    b = eat.EatLayer.from_workload(lw, T, gpu_params(sh))
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    ya = [torch.empty_like(x) for x in xs]
    yb = [torch.empty_like(x) for x in xs]
    torch.cuda.synchronize()
    for i, x in enumerate(xs):
        eat.eat_moe_forward(a.h, x, T, 0, ya[i], stream=sa)
        eat.eat_moe_forward(b.h, x, T, 0, yb[i], stream=sb)
    torch.cuda.synchronize()
    for i in range(4):
        assert torch.equal(ya[i], ref[i]) and torch.equal(yb[i], ref[i])
    a.close()
    b.close()


def test_workspace_allocation_failure_and_new_handle():
    """A layer whose workspace cannot be allocated (65536 tokens x 16 experts of d_ff 262144:
    over 500 GB of activations) fails with EAT_ERR_OOM, leaves no handle and no pending CUDA
    error; the context stays usable, and a handle created after another was destroyed works."""
    fields = dict(d_model=64, n_experts=16, d_ff=262144, n_shared=0, d_ff_shared=0,
                  max_tokens=65536, wdtype=eat.EAT_BF16, xdtype=eat.EAT_BF16, w_router=1 << 20,
                  b_router=None, w_gate=1 << 21, w_up=1 << 22, w_down=1 << 23, ws_gate=None,
                  ws_up=None, ws_down=None, opd_scale=None, w_gate_scale=None, w_up_scale=None,
                  w_down_scale=None, ws_gate_scale=None, ws_up_scale=None, ws_down_scale=None)
    big = eat.eat_layer_desc(*[fields[n] for n, _ in eat.eat_layer_desc._fields_])
    prm = eat.eat_default_params(16)
    h = ctypes.c_void_p()
    r = eat.lib().eat_create(ctypes.byref(big), ctypes.byref(prm), ctypes.byref(h))
    assert r == eat.EAT_ERR_OOM and h.value is None
    assert b"cudaMalloc" in eat.lib().eat_last_error(None)
    torch.cuda.synchronize()
    assert torch.cuda.is_available() and (torch.ones(4, device="cuda") * 2).sum().item() == 8
    lw = W.make_layer(MIX_S)
    layer0 = eat.EatLayer.from_workload(lw, 8, gpu_params(MIX_S))
    layer0.close()
    layer1 = eat.EatLayer.from_workload(lw, 8, gpu_params(MIX_S))
    run_parity(MIX_S, lw, [8], layer=layer1)
    layer1.close()


def test_fp8_hidden_state_magnitudes():
    """fp8 layer, hidden-state rows scaled by 1e-6 ... 1e4 and one all-zero row: each row of the
    GEMMs' other operand picks its own power-of-two scale before the e4m3 hi/lo split.  The router
    weights are zero (routing by the bias alone), so the magnitudes reach only the expert GEMMs
    (logits in the thousands would make the fp32 router, not the split, the limiting error)."""
    lw = W.make_layer(QWEN_S)
    lw.w_router = torch.zeros_like(lw.w_router)
    lw8 = W.to_fp8(lw)
    x = W.make_tokens(QWEN_S, 48)
    x = (x.float() * torch.logspace(-6, 4, 48).view(48, 1)).to(x.dtype)
    x[17] = 0
    layer = eat.EatLayer.from_workload(lw8, 48, gpu_params(QWEN_S))
    run_parity(QWEN_S, lw8.dequantized(), [48], layer=layer, inputs=[x])
    layer.close()


@pytest.mark.parametrize("fp8", [False, True])
def test_many_short_gate_up_units(fp8):
    """d_ff = 4096 over d_model = 256: 32 feature tiles per expert, so calls of 16 or more tokens
    hand every CTA several gate/up units of only 4 (bf16) or 2 (e4m3) k-blocks, and the weight
    prefetch of the down kernel spans units."""
    sh = W.scaled(W.MIXTRAL, "short-k", d_model=256, d_ff=4096)
    lw = W.make_layer(sh)
    if fp8:
        lw8 = W.to_fp8(lw)
        layer = eat.EatLayer.from_workload(lw8, 100, gpu_params(sh))
        run_parity(sh, lw8.dequantized(), [16, 64, 100, 1, 37], layer=layer)
        layer.close()
    else:
        run_parity(sh, lw, [16, 64, 100, 1, 37])


@pytest.mark.parametrize("d,F,E,K", [(1024, 320, 64, 8), (2048, 192, 16, 4), (512, 4096, 8, 2)])
def test_decode_calls_ragged_shapes(d, F, E, K):
    """Decode-sized calls (1 to 32 tokens: token tiles of 16 and 32, split-K down projections)
    on layers with ragged feature tiles (d_ff 320, 192), odd down k-block counts and many feature
    tiles per expert (d_ff 4096), with PPL signs of both kinds."""
    sh = W.scaled(W.OLMOE, f"fused-{d}-{F}", d_model=d, n_experts=E, d_ff=F, max_k=K)
    lw = W.make_layer(sh)
    run_parity(sh, lw, [32, 1, 7, 16, 32, 25], signs=[0, 1, -1, 0, 1, -1])


def test_partial_feature_tiles():
    """d = 320 and d_ff = 192: feature tiles of 128 end half-full in both expert GEMMs."""
    sh = W.scaled(W.QWEN, "ragged-d", d_model=320, n_experts=16, d_ff=192, n_shared=1,
                  d_ff_shared=320, max_k=3)
    lw = W.make_layer(sh)
    run_parity(sh, lw, [97, 3000, 5])


@pytest.mark.parametrize("fp8", [False, True])
def test_odd_k_block_counts(fp8):
    """d = 192 and d_ff = 320: 3 and 5 k-blocks of 64 bf16 elements (2 and 3 ragged k-blocks of 128
    e4m3 ones), so the kernels whose pipeline stages hold two k-blocks end every unit on a stage
    with one; batch 1, 50 and 1200 run the 16- and 64-token single-SM kernels and the SM pairs."""
    sh = W.scaled(W.MIXTRAL, "odd-kb", d_model=192, n_experts=8, d_ff=320, max_k=2)
    lw = W.make_layer(sh)
    if not fp8:
        run_parity(sh, lw, [1, 50, 1200])
        return
    lw8 = W.to_fp8(lw)
    layer = eat.EatLayer.from_workload(lw8, 1200, gpu_params(sh))
    run_parity(sh, lw8.dequantized(), [1, 50, 1200], layer=layer)
    layer.close()


def test_degenerate_fixed_topk_on_gpu():
    """beta = 0, alpha1 = 0, alpha2 huge, no clamp: vanilla Top-K by p (index tie-break)."""
    kw = {"beta": 0.0, "alpha1": 0.0, "alpha2": 1e30, "clamp_enabled": 0}
    lw = W.make_layer(MIX_S)
    layer = eat.EatLayer.from_workload(lw, 128, gpu_params(MIX_S, **kw))
    x = W.make_tokens(MIX_S, 128).cuda()
    idx, w, k = layer.route(x)
    L = oracle_layer(lw)
    r = orc.route(np64(x), L, orc.Accounts.zeros(8), oracle_params(MIX_S, **kw))
    for t in range(128):
        order = np.lexsort((np.arange(8), -r.p[t]))
        assert sorted(idx[t, :k[t]].tolist()) == sorted(order[:2].tolist())
    assert (k.cpu() == 2).all()
    layer.close()
    run_parity(MIX_S, lw, [128, 128], prm_kw=kw)


def test_all_tokens_one_expert():
    """Router bias forces one expert for every token: a single group of n_e = T rows (2500: SM
    pairs with a ragged last tile, and an account update over three 1024-slot chunks of one
    expert, finished by the last of its blocks)."""
    lw = W.make_layer(OLMOE_S)
    lw.b_router = torch.full_like(lw.b_router, -30.0)
    lw.b_router[5] = 30.0
    run_parity(OLMOE_S, lw, [257, 2500, 1])


def test_set_accounts_restore_and_route_is_pure():
    lw = W.make_layer(QWEN_S)
    layer = eat.EatLayer.from_workload(lw, 64, gpu_params(QWEN_S))
    g = torch.Generator().manual_seed(3)
    N = torch.randint(0, 100, (60,), generator=g).to(torch.int64)
    P = torch.rand(60, generator=g, dtype=torch.float64) * N
    C = torch.rand(60, generator=g, dtype=torch.float64) * 5
    layer.set_accounts(N.cuda(), P.cuda(), C.cuda())
    x = W.make_tokens(QWEN_S, 64).cuda()
    a = layer.route(x, 1)
    b = layer.route(x, 1)
    for u, v in zip(a, b):
        assert torch.equal(u, v)
    N1, P1, C1 = layer.accounts()
    assert torch.equal(N1.cpu(), N) and torch.equal(P1.cpu(), P) and torch.equal(C1.cpu(), C)
    _, idx, w, k = layer.forward(x, 1, with_routing=True)
    assert torch.equal(idx, a[0]) and torch.equal(w, a[1]) and torch.equal(k, a[2])
    layer.set_accounts(N.cuda(), P.cuda(), C.cuda())
    run_parity(QWEN_S, lw, [64, 64], layer=layer, signs=[1, -1])
    layer.reset()
    N2, P2, C2 = layer.accounts()
    assert int(N2.abs().sum()) == 0 and float(P2.abs().sum()) == 0 and float(C2.abs().sum()) == 0
    layer.close()


def test_max_tokens_bound_and_host_path():
    lw = W.make_layer(MIX_S)
    layer = eat.EatLayer.from_workload(lw, 40, gpu_params(MIX_S))
    x = W.make_tokens(MIX_S, 41).cuda()
    y = torch.empty_like(x)
    with pytest.raises(eat.EatError) as ei:
        eat.eat_moe_forward(layer.h, x, 41, 0, y)
    assert ei.value.status == eat.EAT_ERR_INVALID_ARG
    # an empty call is rejected, by the layer call and by routing alone, and changes nothing
    acc0 = layer.accounts()
    idx = torch.empty(1, MIX_S.max_k, dtype=torch.int32, device="cuda")
    w = torch.empty(1, MIX_S.max_k, dtype=torch.float32, device="cuda")
    k = torch.empty(1, dtype=torch.int32, device="cuda")
    for call in (lambda: eat.eat_moe_forward(layer.h, x, 0, 0, y),
                 lambda: eat.eat_route(layer.h, x, 0, 0, idx, w, k)):
        with pytest.raises(eat.EatError) as ei:
            call()
        assert ei.value.status == eat.EAT_ERR_INVALID_ARG
    for u, v in zip(acc0, layer.accounts()):
        assert torch.equal(u, v)
    acc = layer.accounts()
    y_dev = layer.forward(x[:40].contiguous(), 0)
    layer.set_accounts(*acc)
    xh = x[:40].cpu().pin_memory()
    yh = torch.empty_like(xh).pin_memory()
    eat.eat_moe_forward_host(layer.h, xh, 40, 0, yh)
    assert torch.equal(yh, y_dev.cpu())
    # the enqueue-only variant: two calls queued back to back, one synchronisation; the second
    # call routes with the accounts the first one updated
    layer.set_accounts(*acc)
    layer.forward(x[:40].contiguous(), 0)
    y_dev2 = layer.forward(x[:40].contiguous(), 0)
    layer.set_accounts(*acc)
    yh1, yh2 = torch.empty_like(yh).pin_memory(), torch.empty_like(yh).pin_memory()
    s = torch.cuda.current_stream()
    eat.eat_moe_forward_host_async(layer.h, xh, 40, 0, yh1, s)
    eat.eat_moe_forward_host_async(layer.h, xh, 40, 0, yh2, s)
    s.synchronize()
    assert torch.equal(yh1, y_dev.cpu()) and torch.equal(yh2, y_dev2.cpu())
    layer.close()


@pytest.mark.parametrize("name,Ts", [("olmoe", [32, 300, 1100]), ("qwen", [16, 300, 1100]),
                                     ("olmoe-fp8", [32, 300])])
def test_host_buffers_page_locked_and_pageable(name, Ts):
    """eat_moe_forward_host with page-locked buffers (the router kernel reads x over the host link
    and writes the device copy, the combine writes y to the host) and with pageable buffers (copy
    engine), against eat_moe_forward on device buffers: outputs and accounts bit for bit, for
    gathering decode tiles, single-SM tiles of 128 tokens and SM pairs; the Qwen-shaped layer's
    small calls run their shared experts beside the routing and take the copies."""
    sh = {"olmoe": OLMOE_S, "qwen": QWEN_S, "olmoe-fp8": OLMOE_S}[name]
    lw = W.make_layer(sh)
    if name.endswith("fp8"):
        lw = W.to_fp8(lw)
    layer = eat.EatLayer.from_workload(lw, max(Ts), gpu_params(sh))
    for s in range(2):  # some history in the accounts
        layer.forward(W.make_tokens(sh, 64, step=50 + s).cuda(), 0)
    s = torch.cuda.current_stream()
    for T in Ts:
        x = W.make_tokens(sh, T, step=T).cuda()
        acc = layer.accounts()
        y_dev = layer.forward(x, 0).cpu()
        acc_dev = [a.clone() for a in layer.accounts()]
        for pinned in (True, False):
            layer.set_accounts(*acc)
            xh = x.cpu().pin_memory() if pinned else x.cpu().clone()
            yh = torch.full_like(xh, float("nan"))
            if pinned:
                yh = yh.pin_memory()
            eat.eat_moe_forward_host(layer.h, xh, T, 0, yh)
            assert torch.equal(yh, y_dev), (name, T, pinned)
            for u, v in zip(layer.accounts(), acc_dev):
                assert torch.equal(u, v), (name, T, pinned)
        # two enqueue-only calls back to back (the two staging buffers in turn), one
        # synchronisation; the second routes with the accounts the first one updated
        layer.set_accounts(*acc)
        y2_dev = layer.forward(x, 0).cpu()
        layer.set_accounts(*acc)
        layer.forward(x, 0)
        y3_dev = layer.forward(x, 0).cpu()
        layer.set_accounts(*acc)
        xh = x.cpu().pin_memory()
        yh1 = torch.empty_like(xh).pin_memory()
        yh2 = torch.empty_like(xh).pin_memory()
        eat.eat_moe_forward_host_async(layer.h, xh, T, 0, yh1, s)
        eat.eat_moe_forward_host_async(layer.h, xh, T, 0, yh2, s)
        s.synchronize()
        assert torch.equal(yh1, y2_dev) and torch.equal(yh2, y3_dev), (name, T)
    layer.close()


def test_deterministic_repeat():
    lw = W.make_layer(OLMOE_S)
    outs = []
    for _ in range(2):
        layer = eat.EatLayer.from_workload(lw, 300, gpu_params(OLMOE_S))
        x = W.make_tokens(OLMOE_S, 300).cuda()
        ys = [layer.forward(x, 0) for _ in range(3)]
        outs.append((ys, layer.accounts()))
        layer.close()
    for a, b in zip(outs[0][0], outs[1][0]):
        assert torch.equal(a, b)
    for a, b in zip(outs[0][1], outs[1][1]):
        assert torch.equal(a, b)


# ------------------------------------------------------------------ baselines and OPD (§4.1, §3.5)
def test_topk_router_mode():
    lw = W.make_layer(MIX_S)
    run_parity(MIX_S, lw, [128, 7, 1], prm_kw={"router_mode": eat.EAT_ROUTER_TOPK})


@pytest.mark.parametrize("top_p", [0.2, 0.4, 0.6])
def test_topp_router_mode(top_p):
    lw = W.make_layer(OLMOE_S)
    run_parity(OLMOE_S, lw, [300, 32], prm_kw={"router_mode": eat.EAT_ROUTER_TOPP,
                                                "top_p": top_p})


def test_opd_reweighting_eat_and_topp():
    lw = W.make_layer(QWEN_S)
    g = torch.Generator().manual_seed(17)
    scale = (torch.rand(60, generator=g) * 3 + 0.25).to(torch.float32)
    run_parity(QWEN_S, lw, [200, 16], opd_scale=scale)
    run_parity(QWEN_S, lw, [200], opd_scale=scale,
               prm_kw={"router_mode": eat.EAT_ROUTER_TOPP, "top_p": 0.4})


# ------------------------------------------------------------------ threshold variants, layer policy
def test_temporal_smoothing_state():
    """EMA of tau_final over calls of each token stream (decode batch of 24 streams)."""
    lw = W.make_layer(OLMOE_S)
    state = torch.full((64,), float("nan"), device="cuda")
    run_parity(OLMOE_S, lw, [24] * 6, signs=[0, 1, 1, -1, 0, -1], max_tokens=64,
               prm_kw={"smoothing_mode": eat.EAT_SMOOTH_TEMPORAL}, tau_state=state)


def test_reversed_ppl_factors():
    """The other reading of §3.3's PPL adjustment (a PPL rise lowers the threshold)."""
    lw = W.make_layer(MIX_S)
    run_parity(MIX_S, lw, [64] * 4, signs=[1, -1, 1, 1], prm_kw={"ppl_up": 0.8, "ppl_down": 1.1})


def test_ppl_feed_on_device():
    """§3.3 fed from token likelihoods on the device: eat_ppl_update turns each window's NLLs into
    the perplexity and the sign of its change (against the oracle: the hand-worked windows of the
    golden example W6, then random windows), and a handle attached to that sign routes exactly as
    the same handle given the oracle's sign on the host."""
    import json
    import math
    import os
    gold = json.load(open(os.path.join(os.path.dirname(__file__), "golden",
                                       "worked_examples.json")))["W6"]["windows"]
    g = torch.Generator().manual_seed(5)
    windows = [w["nll"] for w in gold] + \
        [(torch.rand(n, generator=g) * 4).tolist() for n in (1, 7, 300, 5000)]
    state = torch.full((1,), float("nan"), dtype=torch.float64, device="cuda")
    sign = torch.zeros(1, dtype=torch.int32, device="cuda")
    lw = W.make_layer(MIX_S)
    a = eat.EatLayer.from_workload(lw, 64, gpu_params(MIX_S))
    b = eat.EatLayer.from_workload(lw, 64, gpu_params(MIX_S))
    eat.eat_set_ppl_sign_source(a.h, sign)
    prev = float("nan")
    for i, win in enumerate(windows):
        nll = torch.tensor(win, dtype=torch.float32)
        eat.eat_ppl_update(nll.cuda(), len(win), state, sign)
        x = W.make_tokens(MIX_S, 64, step=i).cuda()
        ya = a.forward(x, 0)  # the sign comes from the device
        torch.cuda.synchronize()
        ref_sign, curr = orc.ppl_sign_update(prev, nll.double().numpy())
        if i < len(gold):
            assert ref_sign == gold[i]["sign"]
        assert int(sign.item()) == ref_sign, f"window {i}"
        assert math.isclose(float(state.item()), curr, rel_tol=1e-13)
        yb = b.forward(x, ref_sign)
        assert torch.equal(ya, yb)
        prev = curr
    for u, v in zip(a.accounts(), b.accounts()):
        assert torch.equal(u, v)
    eat.eat_set_ppl_sign_source(a.h, None)
    a.close()
    b.close()


def test_layer_policy_stack():
    """Per-layer parameters on a stack (§5.2: lower layers sparser, upper layers up to full K)."""
    from paper_2609_33614_gb300.eat import layer_policy
    T, n = 64, 4
    sh = W.scaled(W.DSV2L, "dsv2l-policy", d_model=256, d_ff=192, n_layers=n)
    x = W.make_tokens(sh, T)
    for l in range(n):
        kw = layer_policy(l, n, sh.max_k)
        lw = W.make_layer(sh, l)
        outs = run_parity(W.scaled(sh, "p", max_k=kw["max_k"]), lw, [T], inputs=[x],
                          prm_kw={k: v for k, v in kw.items() if k != "max_k"})
        x = (x.cuda().float() + outs[0].float()).to(torch.bfloat16).cpu()


# ------------------------------------------------------------------ failure path
def test_bounded_wait_expires_and_context_survives():
    """A kernel wait that nothing satisfies gives up after its bound, reports through the status
    word, and the context keeps working (no trap, no hang)."""
    import time
    t0 = time.time()
    assert eat.eat_selftest_bounded_wait(20_000_000) == 64       # 20 ms bound
    assert time.time() - t0 < 10.0
    lw = W.make_layer(MIX_S)
    run_parity(MIX_S, lw, [16])
    layer = eat.EatLayer.from_workload(lw, 16, gpu_params(MIX_S))
    layer.forward(W.make_tokens(MIX_S, 16).cuda(), 0)
    assert eat.eat_get_counters(layer.h)["status"] == 0
    layer.close()


def test_expired_wait_leaves_accounts_and_fails_later_calls():
    """A wait that runs out on the handle's status word (the 20 ms bounded wait an expert kernel
    uses, on a barrier nothing arrives on): the next layer call writes NaN rows and leaves N,
    P_total and C_s unchanged; every later call returns EAT_ERR_STATE (the host-buffer call too)
    until eat_reset_accounts, after which the handle follows the oracle again.  No fault, trap or
    hang is involved."""
    lw = W.make_layer(MIX_S)
    layer = eat.EatLayer.from_workload(lw, 32, gpu_params(MIX_S))
    for s in range(2):
        layer.forward(W.make_tokens(MIX_S, 32, step=s).cuda(), 0)
    torch.cuda.synchronize()
    acc0 = [t.clone() for t in layer.accounts()]
    c0 = eat.eat_get_counters(layer.h)
    eat.eat_selftest_expire_wait(layer.h, 20_000_000)
    x = W.make_tokens(MIX_S, 32, step=5).cuda()
    y = layer.forward(x, 0)  # enqueued behind the expiring wait: accepted, then invalid
    torch.cuda.synchronize()
    assert torch.isnan(y.float()).all()
    for u, v in zip(acc0, layer.accounts()):
        assert torch.equal(u, v)
    c1 = eat.eat_get_counters(layer.h)
    assert c1["status"] == 64 and c1["calls"] == c0["calls"]
    idx = torch.empty(32, MIX_S.max_k, dtype=torch.int32, device="cuda")
    w = torch.empty(32, MIX_S.max_k, dtype=torch.float32, device="cuda")
    k = torch.empty(32, dtype=torch.int32, device="cuda")
    xh = x.cpu().pin_memory()
    yh = torch.empty_like(xh).pin_memory()
    for call in (lambda: layer.forward(x, 0), lambda: eat.eat_route(layer.h, x, 32, 0, idx, w, k),
                 lambda: eat.eat_moe_forward_host(layer.h, xh, 32, 0, yh),
                 lambda: eat.eat_moe_forward_host_async(layer.h, xh, 32, 0, yh)):
        with pytest.raises(eat.EatError) as ei:
            call()
        assert ei.value.status == eat.EAT_ERR_STATE
        assert "bounded wait" in str(ei.value)
    for u, v in zip(acc0, layer.accounts()):
        assert torch.equal(u, v)
    layer.reset()
    assert eat.eat_get_counters(layer.h)["status"] == 0
    run_parity(MIX_S, lw, [32, 7], layer=layer)
    # a host-buffer call that is itself the failing call reports it after its synchronisation
    eat.eat_selftest_expire_wait(layer.h, 20_000_000)
    with pytest.raises(eat.EatError) as ei:
        eat.eat_moe_forward_host(layer.h, xh, 32, 0, yh)
    assert ei.value.status == eat.EAT_ERR_STATE
    assert torch.isnan(yh.float()).all()
    layer.reset()
    layer.close()


# ------------------------------------------------------------------ CUDA graph capture
@pytest.mark.parametrize("shape,T", [("mixtral", 64), ("qwen", 64), ("qwen", 1100),
                                     ("olmoe", 1100)])
def test_forward_replays_as_cuda_graph(shape, T):
    """A layer call has no host synchronisation and decides its expert schedule on the device, so
    it can be captured once and replayed: the replays must match direct calls bit for bit, accounts
    included (two handles on the same weights, same inputs).  The qwen-shaped layer's 64-token call
    runs its shared experts on the handle's second stream, forked and joined inside the capture;
    the 1100-token calls capture the stream-K router, the chunked permute, the gather and the
    SM-pair expert kernels (with the shared experts in the routed launches for qwen)."""
    sh = {"mixtral": MIX_S, "qwen": QWEN_S, "olmoe": OLMOE_S}[shape]
    lw = W.make_layer(sh)
    a = eat.EatLayer.from_workload(lw, T, gpu_params(sh))
    b = eat.EatLayer.from_workload(lw, T, gpu_params(sh))
    x = W.make_tokens(sh, T).cuda()
    y_graph = torch.empty_like(x)
    stream = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(stream):
        eat.eat_moe_forward(a.h, x, T, 0, y_graph, stream=stream.cuda_stream)  # warm-up call
        torch.cuda.current_stream().synchronize()
        with torch.cuda.graph(g, stream=stream):
            eat.eat_moe_forward(a.h, x, T, 0, y_graph, stream=stream.cuda_stream)
    torch.cuda.synchronize()
    ys = [b.forward(x, 0)]  # matches the warm-up call of a
    for _ in range(4):
        g.replay()
        torch.cuda.synchronize()
        y_direct = b.forward(x, 0)
        assert torch.equal(y_graph, y_direct)
    for u, v in zip(a.accounts(), b.accounts()):
        assert torch.equal(u, v)
    a.close()
    b.close()


# ------------------------------------------------------------------ full-size layers, every token
# Every output row and every account of the call is checked against the oracle at the
# configurations' own sizes (C_s against the oracle's own norms as well as the update rule); the
# worst output error of each configuration is printed.
def _big(shape, layer_id=0):
    return W.make_layer(shape, layer_id, device="cuda")


def test_full_mixtral_decode_batches():
    """Mixtral-8x7B-shaped layer, decode at batch 1 / 16 / 64 (the benchmarked configuration)."""
    lw = _big(W.MIXTRAL)
    L = oracle_layer_lazy(lw)
    for B in (1, 16, 64):
        layer = eat.EatLayer.from_workload(lw, 64, gpu_params(W.MIXTRAL))
        run_parity(W.MIXTRAL, lw, [B] * 3, layer=layer, L=L, x_device="cuda", report=f"B{B}")
        layer.close()


def test_full_mixtral_decode_fp8():
    """The same layer with e4m3 expert weights (the fp8 decode configuration)."""
    lw8 = W.to_fp8(_big(W.MIXTRAL))
    dq = lw8.dequantized()
    L = oracle_layer_lazy(dq)
    for B in (1, 16, 64):
        layer = eat.EatLayer.from_workload(lw8, 64, gpu_params(W.MIXTRAL))
        run_parity(W.MIXTRAL, dq, [B] * 2, layer=layer, L=L, x_device="cuda", report=f"fp8 B{B}")
        layer.close()


def test_full_olmoe_prefill_then_decode():
    lw = _big(W.OLMOE)
    L = oracle_layer_lazy(lw)
    layer = eat.EatLayer.from_workload(lw, 4096, gpu_params(W.OLMOE))
    run_parity(W.OLMOE, lw, [4096, 32, 32], layer=layer, L=L, x_device="cuda", report="")
    layer.close()


def test_full_qwen_prefill():
    lw = _big(W.QWEN)
    L = oracle_layer_lazy(lw)
    layer = eat.EatLayer.from_workload(lw, 8192, gpu_params(W.QWEN))
    run_parity(W.QWEN, lw, [8192, 64], layer=layer, L=L, x_device="cuda", report="")
    layer.close()


@pytest.mark.parametrize("layer_id", [0, 12, 25])
def test_full_dsv2l_layer_prefill_then_decode(layer_id):
    """One DeepSeek-V2-Lite-shaped layer at full width: prefill of 16384 tokens, then a decode
    call of 128 routed by the accounts the prefill left.  Layer 0 has the flattest routing (bias
    scale 0.2: the most near-ties), layer 25 the most skewed (1.0)."""
    lw = _big(W.DSV2L, layer_id)
    L = oracle_layer_lazy(lw)
    layer = eat.EatLayer.from_workload(lw, 16384, gpu_params(W.DSV2L))
    run_parity(W.DSV2L, lw, [16384, 128], layer=layer, L=L, x_device="cuda",
               report=f"layer {layer_id}")
    layer.close()


@pytest.mark.parametrize("mode,top_p", [("topk", None), ("topp", 0.4)])
def test_full_olmoe_prefill_baseline_routers(mode, top_p):
    """The §4.1 baseline routers at full size: OLMoE-shaped prefill of 4096 tokens (SM pairs) and a
    decode call of 32, every token and account checked."""
    kw = {"router_mode": eat.EAT_ROUTER_TOPK} if mode == "topk" else \
        {"router_mode": eat.EAT_ROUTER_TOPP, "top_p": top_p}
    lw = _big(W.OLMOE)
    L = oracle_layer_lazy(lw)
    layer = eat.EatLayer.from_workload(lw, 4096, gpu_params(W.OLMOE, **kw))
    run_parity(W.OLMOE, lw, [4096, 32], layer=layer, L=L, x_device="cuda", prm_kw=kw,
               report=mode)
    layer.close()


def test_temporal_smoothing_large_calls():
    """EMA of tau_final over calls (temporal reading) with calls on the SM-pair path: 2048 token
    streams, three calls with PPL signs of both kinds."""
    lw = W.make_layer(OLMOE_S)
    state = torch.full((2048,), float("nan"), device="cuda")
    run_parity(OLMOE_S, lw, [2048, 2048, 1500], signs=[1, -1, 0], max_tokens=2048,
               prm_kw={"smoothing_mode": eat.EAT_SMOOTH_TEMPORAL}, tau_state=state)


def test_maximum_call_size():
    """The largest call a handle takes (max_tokens = 65536) on a small layer with shared experts:
    one 65536-token call on the SM pairs (routed and shared experts in the same launches, about
    4400 token tiles), then a decode call routed by the accounts it left."""
    sh = W.scaled(W.QWEN, "qwen-max", d_model=128, n_experts=60, d_ff=128, d_ff_shared=128)
    lw = W.make_layer(sh)
    run_parity(sh, lw, [65536, 8], max_tokens=65536)


def test_full_dsv2l_decode_stack_26_layers():
    """The 26-layer DeepSeek-V2-Lite-shaped stack in decode at batch 128, two steps, through the
    pre-norm residual chain the benchmark runs (reading R13): layer l reads h_l = RMSNorm(x_l)
    and x_{l+1} = x_l + y_l, with every layer's own accounts.  Each layer is checked on every
    token from the GPU's own h_l (teacher forcing).  Layer-major order: step s of layer l needs
    only layer l's earlier steps and layer l - 1's output of step s."""
    B, steps = 128, 2
    xs = [W.make_tokens(W.DSV2L, B, step=s, device="cuda") for s in range(steps)]
    for l in range(W.DSV2L.n_layers):
        lw = _big(W.DSV2L, l)
        L = oracle_layer_lazy(lw)
        layer = eat.EatLayer.from_workload(lw, B, gpu_params(W.DSV2L))
        hs = [torch.nn.functional.rms_norm(x, (W.DSV2L.d_model,), eps=1e-6) for x in xs]
        outs = run_parity(W.DSV2L, lw, [B] * steps, layer=layer, L=L, inputs=hs,
                          report=f"stack layer {l}")
        layer.close()
        xs = [x + y for x, y in zip(xs, outs)]
        del lw, L
    assert all(bool(torch.isfinite(x.float()).all()) for x in xs)
