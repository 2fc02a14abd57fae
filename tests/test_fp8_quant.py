"""Per-row e4m3 quantization of expert weights (workloads.quantize_fp8): the format the fp8 layers
take.  Host logic only; the GPU path is checked against the oracle on the dequantized weights."""
import pytest
import torch

from paper_2609_33614_gb300 import workloads as W


def test_rows_map_their_largest_magnitude_to_448():
    torch.manual_seed(0)
    w = torch.randn(3, 16, 40) * torch.logspace(-3, 1, 16).view(1, 16, 1)
    q, s = W.quantize_fp8(w)
    assert q.dtype == torch.float8_e4m3fn and s.shape == (3, 16)
    assert torch.equal(q.float().abs().amax(-1), torch.full((3, 16), 448.0))
    assert torch.allclose(s, w.abs().amax(-1) / 448.0)


def test_dequantized_error_within_e4m3_rounding():
    torch.manual_seed(1)
    w = torch.randn(64, 256) * 0.02
    q, s = W.quantize_fp8(w)
    deq = q.float() * s.unsqueeze(-1)
    # e4m3 keeps 3 fraction bits: rounding to nearest errs by at most 2^-4 of the value for
    # normal numbers; below the normal range (2^-6 x scale) by at most half a subnormal step
    err = (deq - w).abs()
    bound = torch.maximum(w.abs() * 2.0 ** -4, s.unsqueeze(-1) * 2.0 ** -10)
    assert bool((err <= bound * (1 + 1e-6)).all())


def test_zero_rows_and_layer_conversion():
    w = torch.zeros(2, 4, 64)
    w[1, 2, 5] = -3.0
    q, s = W.quantize_fp8(w)
    assert s[0, 0] == 1.0 and bool((q[0].float() == 0).all())
    assert q[1, 2, 5].float() == -448.0 and s[1, 2] == pytest.approx(3.0 / 448.0)
    lw = W.make_layer(W.scaled(W.QWEN, "q8", d_model=128, n_experts=4, d_ff=64, n_shared=1,
                               d_ff_shared=64, max_k=2))
    lw8 = W.to_fp8(lw)
    assert set(lw8.scales) == {"w_gate_scale", "w_up_scale", "w_down_scale", "ws_gate_scale",
                               "ws_up_scale", "ws_down_scale"}
    deq = lw8.dequantized()
    rel = ((deq.w_down - lw.w_down.float()).abs().max() / lw.w_down.float().abs().max()).item()
    assert rel <= 2.0 ** -4


def _split_e4m3(v: torch.Tensor):
    """The two-part e4m3 split of bf16 rows that fp8 layers apply to the GEMMs' other operand,
    restated with torch's round-to-nearest-even casts: per row the power of two s that puts the
    largest magnitude in [128, 256), hi = e4m3(v / s), lo = e4m3(v / s - hi)."""
    m = v.float().abs().amax(-1, keepdim=True)
    ex = torch.floor(torch.log2(m))  # m in [2^ex, 2^(ex+1))
    s = torch.where(m > 0, torch.exp2(ex - 7), torch.ones_like(m))
    a = v.float() / s
    hi = a.to(torch.float8_e4m3fn).float()
    lo = (a - hi).to(torch.float8_e4m3fn).float()
    return hi, lo, s


def test_two_part_e4m3_split_of_bf16_rows_is_exact():
    """hi keeps a bf16 value's leading 4 significant bits and lo the remaining (at most 4), so
    (hi + lo) * s reproduces a value exactly while that remainder stays on the e4m3 grid: for
    scaled magnitudes of at least 1/4, which every value within 2^-9 of its row's largest
    magnitude has (the largest scales to at least 128); smaller values err by at most half an e4m3
    subnormal step (2^-10 after scaling)."""
    g = torch.Generator().manual_seed(5)
    rows = torch.randn(64, 4096, generator=g) * torch.logspace(-30, 30, 64).view(64, 1)
    rows[3] = 0.0
    rows[7, 100] = 1e4  # one large value over a row of small ones
    v = rows.to(torch.bfloat16)
    hi, lo, s = _split_e4m3(v)
    assert bool((hi.abs().amax(-1) <= 256).all())  # values below 256 round to at most 256 < 448
    rec = (hi + lo) * s
    vf = v.float()
    big = vf.abs() >= vf.abs().amax(-1, keepdim=True) * 2.0 ** -9
    assert torch.equal(rec[big], vf[big])
    assert bool(((rec - vf).abs()[~big] <= (s * 2.0 ** -10).expand_as(vf)[~big]).all())
    assert torch.equal(rec[3], torch.zeros(4096))
