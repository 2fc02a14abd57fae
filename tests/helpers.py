"""Test helpers: convert seeded workload tensors to the oracle's float64 numpy layer."""
import numpy as np
import torch

import oracle.eat_oracle as orc


def np64(t):
    if t is None:
        return None
    return t.detach().to("cpu", torch.float64).numpy()


def oracle_layer(lw, experts=None):
    """Oracle Layer from workloads.LayerWeights (all experts, or only the listed ones filled)."""
    if experts is None:
        wg, wu, wd = np64(lw.w_gate), np64(lw.w_up), np64(lw.w_down)
    else:
        E = lw.w_gate.shape[0]
        wg = np.zeros((E,) + tuple(lw.w_gate.shape[1:]))
        wu = np.zeros_like(wg)
        wd = np.zeros((E,) + tuple(lw.w_down.shape[1:]))
        for e in experts:
            wg[e], wu[e], wd[e] = np64(lw.w_gate[e]), np64(lw.w_up[e]), np64(lw.w_down[e])
    return orc.Layer(np64(lw.w_router), np64(lw.b_router), wg, wu, wd,
                     np64(lw.ws_gate), np64(lw.ws_up), np64(lw.ws_down))


def oracle_params(shape, **kw):
    return orc.Params(max_k=shape.max_k, temperature=shape.temperature, **kw)


class LazyExperts:
    """Per-expert float64 view of a (possibly device-resident) weight tensor, converted on first
    use, so sampled oracle checks of large layers only widen the experts they touch."""

    def __init__(self, t):
        self.t = t
        self.shape = tuple(t.shape)
        self.cache = {}

    def __getitem__(self, e):
        e = int(e)
        if e not in self.cache:
            # widened to float64 on the device (exact) and copied once
            self.cache[e] = self.t[e].detach().to(torch.float64).cpu().numpy()
        return self.cache[e]


def oracle_layer_lazy(lw):
    lz = lambda t: None if t is None else LazyExperts(t)
    return orc.Layer(np64(lw.w_router), np64(lw.b_router), lz(lw.w_gate), lz(lw.w_up),
                     lz(lw.w_down), lz(lw.ws_gate), lz(lw.ws_up), lz(lw.ws_down))
