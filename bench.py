"""Benchmark of the EAT MoE-layer hot path on GB300 (one JSON line on rank 0).

Default workload: a Mixtral-8x7B-shaped layer (d=4096, 8 SwiGLU experts, d_ff=14336, K=2, bf16
weights, fp32 accumulate) in decode: one step = one layer call at each of batch 1, 16 and 64 tokens
(three handles sharing the weights, each with its own evolving expert accounts; 81 tokens/step).
Inputs are resident in HBM before the timed region; the 2.8 GB of expert weights are larger than
L2, so no flush is needed between steps.  Other workloads (--workload) are the prefill/decode
configurations of the OLMoE-, Qwen-MoE- and DeepSeek-V2-Lite-shaped layers.

--impl reference times the fp64 CPU oracle (the reference arm of this benchmark) on the host cores
on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

_CORES = os.cpu_count() or 1
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(_CORES))

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("MoE-layer tokens/s at 1 GB300 (decode & prefill); % HBM/tensor roofline; "
          "experts/token")
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0


# ------------------------------------------------------------------------------- workloads
def workload_spec(name):
    from paper_2609_33614_gb300 import workloads as W
    specs = {
        "mixtral-decode": dict(shape=W.MIXTRAL, batches=[1, 16, 64], layers=1,
                               desc="mixtral-8x7b-shaped MoE layer, decode, batch 1+16+64 per step"),
        "olmoe-prefill": dict(shape=W.OLMOE, batches=[4096], layers=1,
                              desc="olmoe-shaped MoE layer, prefill 4096 tokens per step"),
        "olmoe-decode": dict(shape=W.OLMOE, batches=[32], layers=1,
                             desc="olmoe-shaped MoE layer, decode batch 32 per step"),
        "qwen-prefill": dict(shape=W.QWEN, batches=[8192], layers=1,
                             desc="qwen1.5-moe-shaped layer (60 routed + 4 shared), prefill 8192"),
        "dsv2l-prefill": dict(shape=W.DSV2L, batches=[16384], layers=26,
                              desc="deepseek-v2-lite-shaped 26-layer MoE stack (pre-norm residual "
                                   "blocks), prefill 16384"),
        "dsv2l-decode": dict(shape=W.DSV2L, batches=[128], layers=26,
                             desc="deepseek-v2-lite-shaped 26-layer MoE stack (pre-norm residual "
                                  "blocks), decode batch 128"),
        # e4m3 expert weights with per-row scales (hidden states bf16, e4m3 x e4m3 GEMMs on the
        # hi/lo split of the other operand)
        "mixtral-decode-fp8": dict(shape=W.MIXTRAL, batches=[1, 16, 64], layers=1, fp8=True,
                                   desc="mixtral-8x7b-shaped MoE layer, e4m3 expert weights, "
                                        "decode, batch 1+16+64 per step"),
        "olmoe-decode-fp8": dict(shape=W.OLMOE, batches=[32], layers=1, fp8=True,
                                 desc="olmoe-shaped MoE layer, e4m3 expert weights, decode "
                                      "batch 32 per step"),
        "olmoe-prefill-fp8": dict(shape=W.OLMOE, batches=[4096], layers=1, fp8=True,
                                  desc="olmoe-shaped MoE layer, e4m3 expert weights, prefill "
                                       "4096 tokens per step"),
    }
    return specs[name]


def bench_config(args, spec):
    """The `config` object of the JSON line (identical for both arms)."""
    shape = spec["shape"]
    cfg = {"workload": spec["desc"], "router": args.router, "cuda_graph": args.graph}
    if args.router == "topp":
        cfg["top_p"] = args.top_p
    if spec.get("fp8"):
        cfg["expert_weights"] = ("e4m3, fp32 scale per row (e4m3 x e4m3 -> fp32 GEMMs, other "
                                 "operand split into e4m3 hi + lo per row)")
    cfg.update({"d_model": shape.d_model, "n_experts": shape.n_experts, "d_ff": shape.d_ff,
                "n_shared": shape.n_shared, "max_k": shape.max_k, "layers": spec["layers"],
                "batches": spec["batches"],
                "l2": "inputs larger than L2 (expert weights > 129 MB), no flush"})
    return cfg


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            pk = json.load(fh)
        return float(pk["hbm_gbs"]), float(pk["bf16_tflops"]), \
            float(pk.get("bf16_tflops_sustained", pk["bf16_tflops"])), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS, 1700.0, "fallback"


# ------------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index, interval_ms=20):
        self.gpu = gpu_index
        self.interval_ms = interval_ms
        self.proc = None
        self.lines = []  # (host time, csv line)

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", str(self.interval_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, window=None):
        """Median SM clock, max clock and throttle reasons over the samples (those read inside
        the host-time window (t0, t1) only, when given)."""
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, mx, reasons = [], [], set()
        for ts, ln in self.lines:
            if window is not None and not window[0] <= ts <= window[1]:
                continue
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------------------- distributed
def dist_setup(n_gpus):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(0)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(value, world):
    """Max of a float over all ranks (the slowest replica sets the job time)."""
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value, world):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ------------------------------------------------------------------------------- roofline
def kernel_bytes(kind, shape, union, acts, T, fp8=False):
    """Algorithmic HBM bytes of one launch: weights of the activated experts (bf16 2 B, or e4m3
    1 B plus a 4 B scale per row) plus the activation rows the kernel must read and write
    (16-bit = 2 B, fp32 partials = 4 B)."""
    d, F = shape.d_model, shape.d_ff
    wb = 1 if fp8 else 2
    rs = 4 if fp8 else 0  # scale bytes per weight row
    Fs = shape.d_ff_shared
    if kind == "ffn_up":
        return union * 2 * F * (d * wb + rs) + acts * d * 2 + acts * F * 2
    if kind == "ffn_down":
        return union * d * (F * wb + rs) + acts * F * 2 + acts * d * 4
    if kind == "shared_up":
        return shape.n_shared * 2 * Fs * (d * wb + rs) + T * d * 2 + shape.n_shared * T * Fs * 2
    if kind == "shared_down":
        return shape.n_shared * d * (Fs * wb + rs) + shape.n_shared * T * (Fs * 2 + d * 4)
    raise KeyError(kind)


def kernel_flops(kind, shape, acts, T):
    d, F = shape.d_model, shape.d_ff
    if kind == "ffn_up":
        return acts * 2 * 2 * d * F
    if kind == "ffn_down":
        return acts * 2 * d * F
    if kind == "shared_up":
        return shape.n_shared * T * 2 * 2 * d * shape.d_ff_shared
    if kind == "shared_down":
        return shape.n_shared * T * 2 * d * shape.d_ff_shared
    raise KeyError(kind)


def roofline(dk, decode, fp8, peaks):
    """The dominant kernel against its roofline.  dk: the kernel's event-timed total ms, launch
    count and algorithmic bytes and flops summed over its launches; decode calls are bound by HBM
    (bytes of the activated experts' weights and the activation rows), prefill calls by the
    tensor pipe (flops).  peaks: (HBM GB/s, bf16 burst TFLOP/s, bf16 sustained TFLOP/s, source).
    A contraction's launches are event-timed one by one inside sub-millisecond steps, a burst
    regime, so the burst peak is the denominator; the fraction of the sustained figure is kept
    beside it as a labelled note."""
    hbm, bf16_burst, bf16_sus, peak_src = peaks
    avg_launch_s = dk["ms"] / 1e3 / max(1, dk["launches"])
    if decode:
        achieved = dk["bytes"] / max(1, dk["launches"]) / avg_launch_s / 1e9
        return {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": achieved / hbm, "peak_source": peak_src}
    achieved = dk["flops"] / max(1, dk["launches"]) / avg_launch_s / 1e12
    if fp8:
        # an e4m3 contraction: the measured bf16 peak x the nominal e4m3 / bf16 ratio (4.5 /
        # 2.25 PFLOP/s dense); the kernels issue two e4m3 MMAs (hi and lo parts of the other
        # operand) per algorithmic product, so they cannot pass half of it
        peak, sus = 2.0 * bf16_burst, 2.0 * bf16_sus
        src = peak_src + " burst bf16 x 2 (nominal e4m3 / bf16)"
    else:
        peak, sus, src = bf16_burst, bf16_sus, peak_src + " burst"
    roof = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
            "frac": achieved / peak, "peak_source": src,
            "note": {"frac_of_sustained": achieved / sus, "sustained_peak": sus}}
    if fp8:
        roof["mma_flops_per_algorithmic_flop"] = 2
    return roof


def traffic_for(kind, workload, experts_per_launch, path=None):
    """DRAM bytes per launch from the committed ncu summary (profiles/traffic.json), if it was
    taken on the current FFN kernel sources (its source hash equals build.ffn_source_hash());
    else None.  Decode captures are stored per activated expert and scaled by this run's mean
    activated experts per launch."""
    path = path or os.path.join(ROOT, "profiles", "traffic.json")
    try:
        from paper_2609_33614_gb300 import build
        with open(path) as fh:
            tr = json.load(fh)
        ent = tr.get(workload, {}).get(kind)
        if ent and ent.get("source_hash") == build.ffn_source_hash():
            if "dram_bytes_per_expert" in ent:
                return ent["dram_bytes_per_expert"] * experts_per_launch
            return ent["dram_bytes_per_launch"]
    except Exception:
        pass
    return None


# ------------------------------------------------------------------------------- our arm
def run_ours(args, world, rank, local, workload, clk, soak_s=1.0, with_cpu_baseline=True):
    """Measure one workload on this rank's GPU: the timed pass (CUDA events on the launching
    stream), a pass with per-launch events (dominant kernel and its roofline), an untimed routing
    replay (k histogram), the end-to-end pass through the host-buffer entry point, for single-layer
    prefill workloads the cold and warm prefill passes, and a soak of the same steps that gives the
    clock sampler `clk` samples under this load.  Returns the result fields of the JSON line."""
    import torch
    from paper_2609_33614_gb300 import eat, workloads as W

    spec = workload_spec(workload)
    shape = spec["shape"]
    batches = spec["batches"]
    n_layers = spec["layers"]
    dev = torch.device("cuda", torch.cuda.current_device())
    stream = torch.cuda.current_stream()
    n_steps_total = args.warmup + args.steps
    t_start = time.time()

    # layers (weights drawn on the GPU generator) and one handle per (layer, batch)
    layer_w = [W.make_layer(shape, l, device="cuda") for l in range(n_layers)]
    if spec.get("fp8"):
        layer_w = [W.to_fp8(lw) for lw in layer_w]
    handles = []  # [layer][batch]
    mode = {"eat": eat.EAT_ROUTER_EAT, "topk": eat.EAT_ROUTER_TOPK,
            "topp": eat.EAT_ROUTER_TOPP}[args.router]
    for lw in layer_w:
        row = []
        for B in batches:
            prm = eat.eat_default_params(shape.max_k, temperature=shape.temperature,
                                         router_mode=mode, top_p=args.top_p)
            row.append(eat.EatLayer.from_workload(lw, B, prm))
        handles.append(row)
    # inputs resident in HBM before the timed region
    xs = {B: [W.make_tokens(shape, B, step=s, device="cuda") for s in range(min(n_steps_total, 64))]
          for B in batches}
    ys = {B: torch.empty(B, shape.d_model, dtype=shape.xdtype, device=dev) for B in batches}
    tokens_per_step = sum(batches)

    # stacks run pre-norm blocks: the MoE layer reads RMSNorm(x_l) (unit gain) and the residual
    # stream takes x_{l+1} = x_l + y_l, both outside the MoE layer.  (Without the norm the residual
    # of the random-weight SwiGLU stack grows layer by layer until it overflows.)
    xr = {B: [torch.empty(B, shape.d_model, dtype=shape.xdtype, device=dev) for _ in range(2)]
          for B in batches}

    def rms_norm(x):
        return torch.nn.functional.rms_norm(x, (shape.d_model,), eps=1e-6)

    def layers_fwd(bi, B, x, routing=None):
        for l in range(n_layers):
            h = rms_norm(x) if n_layers > 1 else x
            if routing is None:
                eat.eat_moe_forward(handles[l][bi].h, h, B, 0, ys[B])
            else:  # also write the routing (idx, w, k) and count the tokens per k
                idx, w, k, hist = routing
                eat.eat_moe_forward(handles[l][bi].h, h, B, 0, ys[B], idx[B], w[B], k[B])
                hist += torch.bincount(k[B].long(), minlength=hist.numel())
            if l + 1 < n_layers:
                nxt = xr[B][l % 2]
                torch.add(x, ys[B], out=nxt)
                x = nxt
        return ys[B]

    def step(s):
        for bi, B in enumerate(batches):
            layers_fwd(bi, B, xs[B][s % len(xs[B])])

    step_direct = step  # per-kernel event timing needs direct launches
    if args.graph:
        # one step captured as a CUDA graph over fixed input buffers; each step copies its inputs
        # in (device to device) and replays the graph
        xin = {B: torch.empty(B, shape.d_model, dtype=shape.xdtype, device=dev) for B in batches}
        for B in batches:
            xin[B].copy_(xs[B][0])
        for bi, B in enumerate(batches):
            layers_fwd(bi, B, xin[B])  # a call outside capture before capturing
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=torch.cuda.Stream()):
            for bi, B in enumerate(batches):
                layers_fwd(bi, B, xin[B])
        torch.cuda.synchronize()

        def step(s):  # noqa: F811
            for B in batches:
                xin[B].copy_(xs[B][s % len(xs[B])], non_blocking=True)
            graph.replay()

    def reset_all():
        for row in handles:
            for h in row:
                h.reset()

    def timed(fn, profile=False, window=None, before_step=None):
        reset_all()
        for s in range(args.warmup):
            if before_step:
                before_step()
            fn(s)
        if profile:
            for row in handles:
                for h in row:
                    eat.eat_profile_begin(h.h, 16 * n_steps_total + 64)
        before = [[eat.eat_get_counters(h.h) for h in row] for row in handles]
        barrier(world)
        torch.cuda.synchronize()
        t0 = time.time()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s in range(args.warmup, n_steps_total):
            if before_step:
                before_step()
            fn(s)
        e1.record(stream)
        torch.cuda.synchronize()
        if window is not None:
            window[:] = [t0, time.time()]
        barrier(world)
        ms = e0.elapsed_time(e1)
        after = [[eat.eat_get_counters(h.h) for h in row] for row in handles]
        prof = None
        if profile:
            prof = [[eat.eat_profile_end(h.h) for h in row] for row in handles]
        return ms, before, after, prof

    timed_window = [0.0, 0.0]
    ms, c0, c1, _ = timed(step, window=timed_window)
    job_ms = max_over_ranks(ms, world)
    total_tokens = sum_over_ranks(tokens_per_step * args.steps, world)
    value = total_tokens / (job_ms / 1e3)

    launches = sum(c1[l][b]["launches"] - c0[l][b]["launches"]
                   for l in range(n_layers) for b in range(len(batches)))
    acts = sum(c1[l][b]["activations"] - c0[l][b]["activations"]
               for l in range(n_layers) for b in range(len(batches)))
    unions = {B: (sum(c1[l][bi]["union_sum"] - c0[l][bi]["union_sum"] for l in range(n_layers)) /
                  max(1, sum(c1[l][bi]["calls"] - c0[l][bi]["calls"] for l in range(n_layers))))
              for bi, B in enumerate(batches)}

    # second pass with per-kernel CUDA events (roofline of the dominant kernel)
    ms_p, p0, p1, prof = timed(step_direct, profile=True)

    # tokens per number of selected experts over the timed steps: an untimed replay from the same
    # reset state with the routing written out (the routing is deterministic, so it is the timed
    # run's)
    reset_all()
    kmax = shape.max_k
    r_idx = {B: torch.empty(B, kmax, dtype=torch.int32, device=dev) for B in batches}
    r_w = {B: torch.empty(B, kmax, dtype=torch.float32, device=dev) for B in batches}
    r_k = {B: torch.empty(B, dtype=torch.int32, device=dev) for B in batches}
    k_hist = torch.zeros(kmax + 1, dtype=torch.int64, device=dev)
    scratch = torch.zeros_like(k_hist)
    for s in range(n_steps_total):
        for bi, B in enumerate(batches):
            layers_fwd(bi, B, xs[B][s % len(xs[B])],
                       (r_idx, r_w, r_k, k_hist if s >= args.warmup else scratch))
    k_hist = {str(i): int(c) for i, c in enumerate(k_hist.cpu().tolist())}
    kinds = {}
    for l in range(n_layers):
        for bi, B in enumerate(batches):
            dU = p1[l][bi]["union_sum"] - p0[l][bi]["union_sum"]
            dA = p1[l][bi]["activations"] - p0[l][bi]["activations"]
            dC = p1[l][bi]["calls"] - p0[l][bi]["calls"]
            for kind, (kms, n) in prof[l][bi].items():
                k = kinds.setdefault(kind, {"ms": 0.0, "launches": 0, "bytes": 0.0, "flops": 0.0})
                k["ms"] += kms
                k["launches"] += n
                k.setdefault("union", 0.0)
                if n and dC:
                    k["union"] += n * dU / dC
                if kind in ("ffn_up", "ffn_down", "shared_up", "shared_down") and n:
                    # per-launch average union / activations of this handle
                    k["bytes"] += n * kernel_bytes(kind, shape, dU / max(1, dC), dA / max(1, dC), B,
                                                   fp8=bool(spec.get("fp8")))
                    k["flops"] += n * kernel_flops(kind, shape, dA / max(1, dC), B)
                    folded = shape.n_shared and prof[l][bi]["shared_up"][1] == 0
                    if folded and kind in ("ffn_up", "ffn_down"):
                        # large calls run the shared experts inside the routed launches
                        sk = "shared_up" if kind == "ffn_up" else "shared_down"
                        k["bytes"] += n * kernel_bytes(sk, shape, 0, 0, B,
                                                       fp8=bool(spec.get("fp8")))
                        k["flops"] += n * kernel_flops(sk, shape, 0, B)
    total_kernel_ms = sum(k["ms"] for k in kinds.values())
    dom = max((k for k in kinds if k.startswith("ffn") or k.startswith("shared")),
              key=lambda k: kinds[k]["ms"])
    dk = kinds[dom]
    avg_launch_s = dk["ms"] / 1e3 / max(1, dk["launches"])
    roof = roofline(dk, max(batches) <= 256, bool(spec.get("fp8")), load_peaks())
    roof["traffic"] = traffic_for(dom, workload, dk["union"] / max(1, dk["launches"]))
    roof.update({"kernel": dom, "kernel_share": dk["ms"] / total_kernel_ms,
                 "avg_launch_us": avg_launch_s * 1e6,
                 "algorithmic_bytes_per_launch": dk["bytes"] / max(1, dk["launches"]),
                 "algorithmic_flops_per_launch": dk["flops"] / max(1, dk["launches"])})

    # end to end through the public host-buffer entry point (copies inside the timed region)
    xh = {B: [x.cpu().pin_memory() for x in xs[B]] for B in batches}
    yh = {B: torch.empty(B, shape.d_model, dtype=shape.xdtype).pin_memory() for B in batches}

    xd = {B: torch.empty(B, shape.d_model, dtype=shape.xdtype, device=dev) for B in batches}
    for B in batches:  # every pinned input has been copied once before the timed steps
        for x in xh[B]:
            xd[B].copy_(x, non_blocking=True)
    torch.cuda.synchronize()

    def step_host(s):
        # every call copies its x in and its y out inside the step; the step ends when the host
        # holds all of the step's outputs
        for bi, B in enumerate(batches):
            if n_layers == 1:
                eat.eat_moe_forward_host_async(handles[0][bi].h, xh[B][s % len(xh[B])], B, 0,
                                               yh[B], stream)
            else:
                xd[B].copy_(xh[B][s % len(xh[B])], non_blocking=True)
                yh[B].copy_(layers_fwd(bi, B, xd[B]), non_blocking=True)
        stream.synchronize()

    e2e_ms, _, _, _ = timed(step_host)
    e2e_ms = max_over_ranks(e2e_ms, world)
    elt = 2 if shape.xdtype == torch.bfloat16 else 4
    e2e = {"value": sum_over_ranks(tokens_per_step * args.steps, world) / (e2e_ms / 1e3),
           "unit": "tokens/s",
           "h2d_bytes_per_step": tokens_per_step * shape.d_model * elt,
           "d2h_bytes_per_step": tokens_per_step * shape.d_model * elt}

    # cold and warm prefill: every timed call starts from the same account state, the empty history
    # of a reset (cold) or the state left by 8 calls of 256 tokens (warm), restored in stream order
    # before each call (three small device copies inside the timed region)
    prefill_states = None
    if n_layers == 1 and len(batches) == 1 and batches[0] > 256:
        E = shape.n_experts
        h0 = handles[0][0]
        zero = (torch.zeros(E, dtype=torch.int64, device=dev),
                torch.zeros(E, dtype=torch.float64, device=dev),
                torch.zeros(E, dtype=torch.float64, device=dev))
        h0.reset()
        for s in range(8):
            h0.forward(xs[batches[0]][s % len(xs[batches[0]])][:256].contiguous(), 0)
        warm = tuple(t.clone() for t in h0.accounts())
        prefill_states = {}
        for name, snap in (("cold", zero), ("warm", warm)):
            st_ms, q0, q1, _ = timed(step, before_step=lambda snap=snap: h0.set_accounts(*snap))
            st_ms = max_over_ranks(st_ms, world)
            dC = q1[0][0]["calls"] - q0[0][0]["calls"]
            prefill_states[name] = {
                "value": sum_over_ranks(tokens_per_step * args.steps, world) / (st_ms / 1e3),
                "unit": "tokens/s", "ms_per_step": st_ms / args.steps,
                "union_per_call": (q1[0][0]["union_sum"] - q0[0][0]["union_sum"]) / max(1, dC),
                "experts_per_token": (q1[0][0]["activations"] - q0[0][0]["activations"]) /
                max(1, dC * batches[0])}
        prefill_states["warm"]["state"] = "accounts after 8 calls of 256 tokens from a reset"

    # soak: the same steps, untimed, so that the clock sampler sees this load for soak_s seconds
    t_soak = time.time()
    s = 0
    while time.time() - t_soak < soak_s:
        step(s)
        s += 1
        if s % 8 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    t_end = time.time()

    clocks = clk.summary((t_start, t_end))
    clocks["timed_region"] = clk.summary(tuple(timed_window))
    clocks["sampled"] = "nvidia-smi every 20 ms over this workload's timed, per-launch, e2e " \
                        f"passes and a {soak_s:.1f} s soak of the same steps"
    if clocks.get("sm_mhz"):
        roof["avg_launch_us_x_sm_mhz"] = avg_launch_s * 1e6 * clocks["sm_mhz"]

    result = {
        "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": job_ms / args.steps,
        "dtype": "e4m3" if spec.get("fp8") else "bf16",
        "config": bench_config(args, spec),
        "roofline": roof,
        "experts_per_token": acts / max(1, sum(B * args.steps for B in batches) * n_layers),
        "union_per_call": unions,
        "k_histogram": k_hist,
        "kernels_ms_per_step": {k: v["ms"] / args.steps for k, v in kinds.items()},
        "gpu_launches": launches,
        "clocks": clocks,
        "e2e": e2e,
    }
    if prefill_states is not None:
        result["prefill_states"] = prefill_states
    if rank == 0 and world == 1 and with_cpu_baseline and not args.no_cpu_baseline:
        # the oracle runs after every GPU measurement of the process (its BLAS threads would
        # compete with the host thread that issues the end-to-end copies): keep what it needs
        N, P, C = handles[0][0].accounts()
        result["_oracle_inputs"] = (workload, layer_w[0], (N.cpu(), P.cpu(), C.cpu()))
    for row in handles:
        for h in row:
            h.close()
    del layer_w, handles
    torch.cuda.empty_cache()
    return result


# ------------------------------------------------------------------------------- oracle arm
def _oracle_layer(lw):
    """The oracle's fp64 layer (an fp8 layer's dequantized weights: what its GPU path uses)."""
    import torch
    import oracle.eat_oracle as orc
    if hasattr(lw, "dequantized"):
        lw = lw.dequantized()
    f = lambda t: None if t is None else t.detach().to("cpu").to(torch.float64).numpy()
    return orc.Layer(f(lw.w_router), f(lw.b_router), f(lw.w_gate), f(lw.w_up), f(lw.w_down),
                     f(lw.ws_gate), f(lw.ws_up), f(lw.ws_down))


def oracle_sample(workload, lw, accounts=None, min_seconds=10.0, max_steps=None, batches=None):
    """Time the fp64 oracle, as it stands, on a bounded sample of the workload: successive layer
    calls cycling through the workload's batch sizes (prefill workloads: the first 256 tokens of
    the prefill batch), from the given accounts (N, P, C tensors, e.g. a GPU handle's after its
    timed steps) or the empty history, until min_seconds of CPU time have run (or max_steps
    calls)."""
    import numpy as np
    import torch
    import oracle.eat_oracle as orc
    from paper_2609_33614_gb300 import workloads as W

    spec = workload_spec(workload)
    shape = spec["shape"]
    bs = batches or [min(B, 256) for B in spec["batches"]]
    L = _oracle_layer(lw)
    prm = orc.Params(max_k=shape.max_k, temperature=shape.temperature)
    if accounts is not None:
        acc = orc.Accounts(*(t.cpu().numpy() for t in accounts))
    else:
        acc = orc.Accounts.zeros(shape.n_experts)
    toks, calls, el = 0, 0, 0.0
    while el < min_seconds and (max_steps is None or calls < max_steps):
        B = bs[calls % len(bs)]
        x = W.make_tokens(shape, B, step=calls).to(torch.float64).numpy()
        t0 = time.perf_counter()
        res = orc.moe_forward(x, L, acc, prm, 0)
        el += time.perf_counter() - t0
        acc = res.accounts_after
        toks += B
        calls += 1
    return {"value": toks / el, "unit": "tokens/s", "cores": int(os.environ["OPENBLAS_NUM_THREADS"]),
            "kind": "oracle",
            "sample": f"{calls} oracle layer calls cycling batches {bs} ({toks} tokens, "
                      f"{el:.1f} s), fp64 numpy, weights widened to fp64 before timing"}


def _blas_thread_setter():
    """openblas_set_num_threads (under any of its exported names) of the BLAS library numpy
    loaded into this process, found through /proc/self/maps; None when there is none."""
    import ctypes
    import numpy  # noqa: F401  (loads the BLAS library)
    paths = set()
    try:
        with open("/proc/self/maps") as fh:
            for ln in fh:
                f = ln.split()
                if len(f) >= 6 and "blas" in f[-1].lower() and ".so" in f[-1]:
                    paths.add(f[-1])
    except OSError:
        return None
    for path in sorted(paths):
        try:
            lib = ctypes.CDLL(path)
        except OSError:
            continue
        for name in ("openblas_set_num_threads", "scipy_openblas_set_num_threads64_",
                     "scipy_openblas_set_num_threads", "openblas_set_num_threads64_"):
            fn = getattr(lib, name, None)
            if fn is not None:
                fn.argtypes = [ctypes.c_int]
                fn.restype = None
                return fn
    return None


def oracle_sample_single_thread(workload, lw, accounts=None, min_seconds=5.0):
    """The same oracle sample with its BLAS library limited to one thread (restored after)."""
    setter = _blas_thread_setter()
    if setter is None:
        return {"unavailable": "no openblas_set_num_threads in the BLAS library numpy loaded"}
    setter(1)
    try:
        r = oracle_sample(workload, lw, accounts, min_seconds=min_seconds)
    finally:
        setter(int(os.environ["OPENBLAS_NUM_THREADS"]))
    r["cores"] = 1
    return r


def run_reference(args, world, rank):
    """The reference arm: the fp64 oracle on the host cores, rank 0 only."""
    if rank != 0:
        return None
    import torch
    from paper_2609_33614_gb300 import workloads as W
    spec = workload_spec(args.workload)
    shape = spec["shape"]
    lw = W.make_layer(shape, 0, device="cuda" if torch.cuda.is_available() else "cpu")
    if spec.get("fp8"):
        lw = W.to_fp8(lw)
    # each step: one oracle layer call at batch 1 (bounded so K steps end in minutes)
    bs = [1] if spec["batches"][0] <= 256 else [64]
    import oracle.eat_oracle as orc
    L = _oracle_layer(lw)
    del lw
    prm = orc.Params(max_k=shape.max_k, temperature=shape.temperature, router=args.router,
                     top_p=args.top_p)
    acc = orc.Accounts.zeros(shape.n_experts)
    toks, el = 0, 0.0
    for s in range(args.warmup + args.steps):
        B = bs[s % len(bs)]
        x = W.make_tokens(shape, B, step=s).to(torch.float64).numpy()
        t0 = time.perf_counter()
        res = orc.moe_forward(x, L, acc, prm, 0)
        dt = time.perf_counter() - t0
        acc = res.accounts_after
        if s >= args.warmup:
            el += dt
            toks += B
    value = toks / el
    cores = int(os.environ["OPENBLAS_NUM_THREADS"])
    return {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": el * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": bench_config(args, spec),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores,
                             "kind": "oracle",
                             "sample": f"{args.steps} timed oracle layer calls at batch {bs}"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=256)
    ap.add_argument("--warmup", type=int, default=16)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="mixtral-decode")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-prefill-record", action="store_true",
                    help="default workload only: skip the OLMoE prefill sub-record")
    ap.add_argument("--router", default="eat", choices=["eat", "topk", "topp"],
                    help="selection rule: EAT (default) or the paper's Top-K / Top-P baselines")
    ap.add_argument("--top-p", type=float, default=0.6)
    ap.add_argument("--graph", action="store_true",
                    help="replay each step as a captured CUDA graph")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world, rank, local = dist_setup(args.gpus)
    if args.impl == "reference":
        res = run_reference(args, world, rank)
    else:
        from paper_2609_33614_gb300 import build
        if rank == 0:
            build.build()
        barrier(world)
        with ClockSampler(local) as clk:
            res = run_ours(args, world, rank, local, args.workload, clk)
            if args.workload == "mixtral-decode" and not args.no_prefill_record:
                # the prefill half of the metric, measured in the same run: one OLMoE-shaped
                # prefill layer (4096 tokens per call)
                pre = run_ours(args, world, rank, local, "olmoe-prefill", clk, soak_s=0.5,
                               with_cpu_baseline=False)
                pre.pop("n_gpus")
                pre["workload"] = "olmoe-prefill"
                res["prefill"] = pre
            ctx = res.pop("_oracle_inputs", None)
            if ctx is not None:
                wl, lw, acc = ctx
                res["cpu_baseline"] = oracle_sample(wl, lw, acc, min_seconds=10.0)
                res["cpu_baseline"]["single_thread"] = oracle_sample_single_thread(
                    wl, lw, acc, min_seconds=5.0)
                del lw
        res = {"metric": METRIC, **res, "higher_is_better": True, "scaling": "weak",
               "vs_baseline": None,
               "data": "synthetic (seeded N(0,1) hidden states, N(0,0.02^2) weights" +
                       (", quantized to e4m3 per row)" if workload_spec(args.workload).get("fp8")
                        else ")")}
    if rank == 0 and res is not None:
        print(json.dumps(res))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
