"""Seeded synthetic inputs shaped like the MoE layers the EAT paper evaluates.

This module holds no arithmetic of the method: it only draws random tensors with fixed seeds so that
the CUDA path and the fp64 oracle see identical bytes.  The paper's models (Mixtral-8x7B,
Qwen-MoE, ...) and its OpenCompass benchmarks (§4.1) are not available; these synthetic layers and
hidden states stand in for them.

Recipe (one torch.Generator per layer, seed 1234 + 1000 * config_id + layer):
  router weight W_r ~ N(0, 0.02^2) fp32 [E, d]; per-expert logit bias as the config states
  (N(0, 0.5^2), Zipf popularity log(pi_e) with pi ~ rank^-s over a seeded permutation, or a depth-
  scaled N(0, 1)); expert weights W_gate, W_up [E, F, d] and W_down [E, d, F] ~ N(0, 0.02^2)
  stored in the config's weight dtype; hidden states x ~ N(0, 1) in the activation dtype, one
  generator per (config, stream) so step s of a decode run is reproducible on its own.
Small layers are drawn on the CPU; layers too large for a quick CPU draw may be drawn on a CUDA
generator instead (``device="cuda"``) -- both sides then read the same device tensors.
"""
from __future__ import annotations

from dataclasses import dataclass, field
import math

import torch


@dataclass(frozen=True)
class LayerShape:
    name: str
    config_id: int
    d_model: int
    n_experts: int
    d_ff: int
    max_k: int
    n_shared: int = 0
    d_ff_shared: int = 0
    wdtype: torch.dtype = torch.bfloat16
    xdtype: torch.dtype = torch.bfloat16
    bias: str = "normal"          # "normal" (N(0, 0.5^2)), "zipf", "depth"
    zipf_s: float = 1.0
    temperature: float = 1.0
    n_layers: int = 1


# The five configurations (sizes as the config list states them).
TOY = LayerShape("toy", 1, 256, 8, 512, 2, wdtype=torch.float32, xdtype=torch.float32)
MIXTRAL = LayerShape("mixtral", 2, 4096, 8, 14336, 2)
OLMOE = LayerShape("olmoe", 3, 2048, 64, 1024, 8, bias="zipf", zipf_s=1.1, temperature=0.5)
QWEN = LayerShape("qwen", 4, 2048, 60, 1408, 4, n_shared=4, d_ff_shared=1408, bias="zipf",
                  zipf_s=1.0)
DSV2L = LayerShape("dsv2l", 5, 2048, 64, 1408, 6, n_shared=2, d_ff_shared=1408, bias="depth",
                   n_layers=26)

SHAPES = {s.name: s for s in (TOY, MIXTRAL, OLMOE, QWEN, DSV2L)}


def scaled(shape: LayerShape, name: str, **kw) -> LayerShape:
    """A reduced copy of a shape (same structure and distributions) for tests."""
    from dataclasses import replace
    return replace(shape, name=name, **kw)


def layer_seed(shape: LayerShape, layer: int = 0) -> int:
    return 1234 + 1000 * shape.config_id + layer


def _normal(gen, shape, std, device, dtype):
    t = torch.randn(*shape, generator=gen, device=device, dtype=torch.float32)
    return (t * std).to(dtype)


def zipf_bias(n_experts: int, s: float, gen: torch.Generator) -> torch.Tensor:
    """Per-expert logit bias log(pi_e), pi_e proportional to rank_e^-s, rank a seeded permutation
    of 1..E (popularity skew of the router)."""
    rank = torch.randperm(n_experts, generator=gen).to(torch.float64) + 1.0
    pi = rank.pow(-s)
    pi = pi / pi.sum()
    return pi.log().to(torch.float32)


@dataclass
class LayerWeights:
    shape: LayerShape
    w_router: torch.Tensor
    b_router: torch.Tensor
    w_gate: torch.Tensor
    w_up: torch.Tensor
    w_down: torch.Tensor
    ws_gate: torch.Tensor | None = None
    ws_up: torch.Tensor | None = None
    ws_down: torch.Tensor | None = None


@dataclass
class Fp8LayerWeights(LayerWeights):
    """Expert weights as e4m3 with one fp32 scale per row (``scales`` keyed like the C ABI's
    descriptor fields: w_gate_scale, w_up_scale, w_down_scale, ws_gate_scale, ...)."""
    scales: dict | None = None

    def dequantized(self) -> LayerWeights:
        """The weights the fp8 layer computes with: scale[row] * e4m3 value, in fp32."""
        def dq(q, name):
            if q is None:
                return None
            return q.float() * self.scales[name].unsqueeze(-1).float()
        return LayerWeights(self.shape, self.w_router, self.b_router,
                            dq(self.w_gate, "w_gate_scale"), dq(self.w_up, "w_up_scale"),
                            dq(self.w_down, "w_down_scale"), dq(self.ws_gate, "ws_gate_scale"),
                            dq(self.ws_up, "ws_up_scale"), dq(self.ws_down, "ws_down_scale"))


def quantize_fp8(w: torch.Tensor):
    """Per-row e4m3 quantization of [..., rows, cols] weights: scale = max |row| / 448 (1 for an
    all-zero row), q = round-to-nearest e4m3 of w / scale.  Returns (q, scale fp32 [..., rows])."""
    wf = w.float()
    amax = wf.abs().amax(dim=-1)
    scale = torch.where(amax > 0, amax / 448.0, torch.ones_like(amax))
    q = (wf / scale.unsqueeze(-1)).to(torch.float8_e4m3fn)
    return q, scale


def to_fp8(lw: LayerWeights) -> Fp8LayerWeights:
    """The layer with its expert weights quantized to e4m3 per row (router unchanged)."""
    out, scales = {}, {}
    for name in ("w_gate", "w_up", "w_down", "ws_gate", "ws_up", "ws_down"):
        t = getattr(lw, name)
        if t is None:
            out[name] = None
            continue
        out[name], scales[name + "_scale"] = quantize_fp8(t)
    return Fp8LayerWeights(lw.shape, lw.w_router, lw.b_router, out["w_gate"], out["w_up"],
                           out["w_down"], out["ws_gate"], out["ws_up"], out["ws_down"],
                           scales=scales)


def make_layer(shape: LayerShape, layer: int = 0, device: str = "cpu") -> LayerWeights:
    """Draw one layer's router and expert weights.  The router (fp32) and its bias are always
    drawn on the CPU generator; the expert weights on ``device``'s generator."""
    seed = layer_seed(shape, layer)
    g_cpu = torch.Generator("cpu").manual_seed(seed)
    E, d, F = shape.n_experts, shape.d_model, shape.d_ff
    w_router = _normal(g_cpu, (E, d), 0.02, "cpu", torch.float32)
    if shape.bias == "normal":
        b = _normal(g_cpu, (E,), 0.5, "cpu", torch.float32)
    elif shape.bias == "zipf":
        b = zipf_bias(E, shape.zipf_s, g_cpu)
    elif shape.bias == "depth":
        s_l = 0.2 + 0.8 * layer / max(1, shape.n_layers - 1)
        b = _normal(g_cpu, (E,), 1.0, "cpu", torch.float32) * s_l
    else:
        raise ValueError(shape.bias)
    if device == "cpu":
        g_w = g_cpu
    else:
        g_w = torch.Generator(device).manual_seed(seed)
    wd = shape.wdtype
    w_gate = _normal(g_w, (E, F, d), 0.02, device, wd)
    w_up = _normal(g_w, (E, F, d), 0.02, device, wd)
    w_down = _normal(g_w, (E, d, F), 0.02, device, wd)
    ws = (None, None, None)
    if shape.n_shared:
        S, Fs = shape.n_shared, shape.d_ff_shared
        ws = (_normal(g_w, (S, Fs, d), 0.02, device, wd),
              _normal(g_w, (S, Fs, d), 0.02, device, wd),
              _normal(g_w, (S, d, Fs), 0.02, device, wd))
    return LayerWeights(shape, w_router, b, w_gate, w_up, w_down, *ws)


def make_tokens(shape: LayerShape, n_tokens: int, stream: int = 0, step: int = 0,
                device: str = "cpu") -> torch.Tensor:
    """Hidden states x [T, d] ~ N(0, 1) in the activation dtype for decode/prefill step ``step``
    of input stream ``stream``."""
    seed = layer_seed(shape) * 7919 + 104729 * stream + step
    g = torch.Generator(device).manual_seed(seed)
    return torch.randn(n_tokens, shape.d_model, generator=g, device=device,
                       dtype=torch.float32).to(shape.xdtype)


def ppl_signs(n_steps: int, seed: int = 77) -> list[int]:
    """Seeded +-1 sequence standing in for the sign of PPL_curr - PPL_prev (§3.3)."""
    g = torch.Generator("cpu").manual_seed(seed)
    return [1 if v else -1 for v in torch.randint(0, 2, (n_steps,), generator=g).tolist()]
