"""Host logic of bench.py's multi-process path on CPU: world_size 2 over gloo (the job time is the
max over ranks, throughput sums the ranks' tokens), plus the reference-arm JSON shape."""
import json
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE="2", LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    world, r, _ = bench.dist_setup(2)
    bench.barrier(world)
    out[r] = (bench.max_over_ranks(1.5 + r, world), bench.sum_over_ranks(10.0 * (r + 1), world))
    import torch.distributed as dist
    dist.destroy_process_group()


def test_gloo_two_ranks_max_and_sum():
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(_free_port(), out), nprocs=2, join=True)
    assert out[0] == (2.5, 30.0) and out[1] == (2.5, 30.0)


def test_kernel_bytes_formula():
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_33614_gb300 import workloads as W
    sh = W.MIXTRAL
    # two activated experts for one token: gate+up weights of both experts dominate
    b = bench.kernel_bytes("ffn_up", sh, 2, 2, 1)
    assert b == 2 * 2 * 14336 * 4096 * 2 + 2 * 4096 * 2 + 2 * 14336 * 2
    assert bench.kernel_flops("ffn_down", sh, 2, 1) == 2 * 2 * 4096 * 14336


def test_roofline_units_and_peaks():
    """Decode lines are HBM-bound (GB/s of algorithmic bytes per event-timed launch), prefill lines
    tensor-bound against the burst bf16 peak (launches event-timed one by one), with the fraction
    of the sustained peak as a note, and e4m3 contractions against twice the bf16 figures (the
    nominal e4m3 / bf16 ratio)."""
    sys.path.insert(0, ROOT)
    import bench
    peaks = (6800.0, 1900.0, 1700.0, "measured")
    dk = {"ms": 2.0, "launches": 4, "bytes": 4 * 3.4e9, "flops": 4 * 8.5e11}  # 0.5 ms each
    hbm = bench.roofline(dk, True, False, peaks)
    assert hbm["bound"] == "hbm" and hbm["unit"] == "GB/s"
    assert abs(hbm["achieved"] - 6800.0) < 1e-6 and abs(hbm["frac"] - 1.0) < 1e-12
    ten = bench.roofline(dk, False, False, peaks)
    assert ten["unit"] == "TFLOP/s" and abs(ten["achieved"] - 1700.0) < 1e-6
    assert ten["peak"] == 1900.0 and abs(ten["frac"] - 1700.0 / 1900.0) < 1e-12
    assert abs(ten["note"]["frac_of_sustained"] - 1.0) < 1e-12
    f8 = bench.roofline(dk, False, True, peaks)
    assert f8["peak"] == 3800.0 and abs(f8["frac"] - 1700.0 / 3800.0) < 1e-12
    assert abs(f8["note"]["frac_of_sustained"] - 0.5) < 1e-12
    assert f8["mma_flops_per_algorithmic_flop"] == 2


def test_traffic_needs_the_current_kernel_sources(tmp_path):
    """A recorded DRAM capture counts only while the FFN kernel sources hash to the recorded value;
    decode captures scale per activated expert."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_33614_gb300 import build
    cur = build.ffn_source_hash()
    rec = {"w": {"ffn_up": {"dram_bytes_per_expert": 2.0e8, "source_hash": cur},
                 "ffn_down": {"dram_bytes_per_launch": 5.0e8, "source_hash": "0" * 64}}}
    path = tmp_path / "traffic.json"
    path.write_text(json.dumps(rec))
    assert bench.traffic_for("ffn_up", "w", 3.5, path=str(path)) == 7.0e8
    assert bench.traffic_for("ffn_down", "w", 1.0, path=str(path)) is None
    assert bench.traffic_for("ffn_up", "other", 1.0, path=str(path)) is None


def test_blas_thread_setter_found_or_none():
    """The single-thread oracle timing finds the BLAS library's thread setter, or reports that it
    cannot (then the line says so instead of timing all cores as one)."""
    sys.path.insert(0, ROOT)
    import bench
    fn = bench._blas_thread_setter()
    if fn is not None:
        fn(1)
        fn(os.cpu_count() or 1)
