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
