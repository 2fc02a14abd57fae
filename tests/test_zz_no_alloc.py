"""eat_route_noalloc: routing for callers that cannot allocate device memory.

Callers such as a serving process whose memory pool already holds nearly all of HBM, or a decode
loop that cannot afford cudaMalloc's implicit synchronisation, cannot create a handle.  They call
eat_route_noalloc, which takes every buffer from the caller and keeps its scratch in a fixed array
inside the library.  This test checks, through the C ABI, two calls in a row (the second at the
largest batch the fixed scratch holds, T x E = 131072 router scores):
  - against the handle-based eat_route on the same inputs and accounts: selections and k equal,
    gates within the 1e-5 tolerance of the parity tests;
  - against the fp64 oracle on the same account snapshot: selections and k exact on every token
    away from a near-tie, gates within 1e-5 (eat_route_noalloc may use fewer router slices than
    eat_route, a difference only the oracle can judge);
and that a batch too large for the fixed scratch is rejected.  The file sorts last so that a run
stopping at the first failure has already run every other test.
"""
import pytest
import torch

import oracle.eat_oracle as orc
from paper_2609_33614_gb300 import eat, workloads as W
from tests import parity as par
from tests.helpers import np64, oracle_layer

pytestmark = pytest.mark.gpu

SHAPE = W.scaled(W.OLMOE, "olmoe-noalloc", d_model=1024, d_ff=256)


@pytest.fixture(scope="module")
def layer():
    from paper_2609_33614_gb300 import build
    build.build()
    torch.cuda.set_device(0)
    lw = W.make_layer(SHAPE)
    L = eat.EatLayer.from_workload(lw, 2048)
    for s in range(3):  # some routing history in the accounts
        L.forward(W.make_tokens(SHAPE, 256, step=100 + s).cuda(), 0)
    torch.cuda.synchronize()
    yield L, oracle_layer(lw)
    L.close()


def _noalloc(L, x, sign):
    T = x.shape[0]
    N, P, C = L.accounts()
    idx = torch.full((T, L.K), -7, dtype=torch.int32, device="cuda")
    w = torch.full((T, L.K), -7.0, dtype=torch.float32, device="cuda")
    k = torch.full((T,), -7, dtype=torch.int32, device="cuda")
    wr, br = L._keep[0], L._keep[1]
    eat.eat_route_noalloc(x, T, L.d, L.E, eat.EAT_BF16, wr, br, N, P, C, L.params, sign,
                          idx, w, k)
    return idx, w, k


@pytest.mark.parametrize("calls", [((300, 1), (2048, -1))])
def test_noalloc_matches_route_and_oracle_two_calls(layer, calls):
    L, ref_layer = layer
    assert calls[-1][0] * L.E == (1 << 20) // 8  # the scratch's largest batch
    prm = orc.Params(max_k=SHAPE.max_k, temperature=SHAPE.temperature)
    for step, (T, sign) in enumerate(calls):
        x = W.make_tokens(SHAPE, T, step=step).cuda()
        ref_idx, ref_w, ref_k = L.route(x, sign)
        idx, w, k = _noalloc(L, x, sign)
        torch.cuda.synchronize()
        assert torch.equal(k, ref_k)
        assert torch.equal(idx, ref_idx)
        assert torch.allclose(w, ref_w, rtol=1e-5, atol=0.0)
        N, P, C = (t.cpu().numpy() for t in L.accounts())
        routing = orc.route(np64(x), ref_layer, orc.Accounts(N, P, C), prm, sign)
        par.check_routing(routing, par.gpu_selection(idx, k), w.cpu().numpy(), SHAPE.max_k)


def test_noalloc_rejects_batches_beyond_its_scratch(layer):
    L, _ = layer
    T = (1 << 20) // 8 // L.E + 1   # T * E > 131072 router scores
    x = torch.zeros(T, L.d, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(eat.EatError) as ei:
        _noalloc(L, x, 0)
    assert ei.value.status == eat.EAT_ERR_INVALID_ARG
    assert "scratch" in str(ei.value)
