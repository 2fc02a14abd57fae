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
