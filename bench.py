"""Benchmark of the MC compressed MoE layer (PMQ mixed-bit experts + ODP routing)
on GB300.

Default workload: one Mixtral-8x7b-shaped MoE layer in decode -- H 4096, SwiGLU F
14336, 8 experts, top-2, 16 tokens, group 128, per-expert bits from {1,2,3}
(sum 20, mean 2.5), ODP off -- the configuration the decode tokens/s metric is
quoted on.  A step is one mc_moe_forward (gate, top-2, ODP, permutation, W1|W3
GEMV + SwiGLU, W2 GEMV, combine) on resident device inputs.  Packed weights
rotate over several device copies so that no step finds its weights in L2.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload decode16|decode1|decode4]
  python bench.py --impl reference ...   (the CPU oracle on the host cores)

Under torchrun every rank runs an independent replica (the layer does not need a
collective); rank 0 prints one JSON line with the aggregate over ranks.
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "Mixed-bit MoE-layer tokens/s; % HBM roofline (decode), % TC peak (prefill)"
WORKLOADS = {"decode16": 16, "decode4": 4, "decode1": 1}


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def _algorithmic_bytes(shape, bits, touched, T, H):
    """Packed weight bytes of the touched experts (codes + fp16 scale/zero) plus
    the gate, activations and output.  Returns (total, w13 part)."""
    per_mat = lambda b: H * shape.F * b / 8 + H * shape.F / shape.group * 4
    w13 = sum(2 * per_mat(int(bits[e])) for e in touched)
    w2 = sum(per_mat(int(bits[e])) for e in touched)
    other = shape.E * H * 2 + 2 * T * H * 2
    return w13 + w2 + other, w13


def cpu_baseline(L, budget_s=12.0, threads=None):
    """Time the oracle, as it stands, on a bounded sample of the workload's tokens
    (one token per host thread)."""
    import concurrent.futures as cf

    import oracle
    mats = [[oracle.QMat(*L.mat_shape(m), L.group, int(L.bits[e]), L.codes[e][m], L.scale[e][m], L.zero[e][m])
             for m in range(3)] for e in range(L.E)]
    xf, gf = L.x_f32(), L.gate_f32()
    t0 = time.perf_counter()
    oracle.moe_layer(xf, gf, mats, L.mu, L.protect, tokens=[0])
    one = time.perf_counter() - t0
    cores = threads or (os.cpu_count() or 1)
    n = int(max(1, min(L.T, cores, round(budget_s / max(one, 1e-3) * cores / 2))))
    toks = list(range(n))
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(min(n, cores)) as ex:
        list(ex.map(lambda t: oracle.moe_layer(xf, gf, mats, L.mu, L.protect, tokens=[t]), toks))
    dt = time.perf_counter() - t0
    return {"value": n / dt, "unit": "tokens/s", "cores": min(n, cores), "kind": "oracle",
            "sample": "%d of the workload's %d tokens (full layer per token, fp64, one token per thread)"
                      % (n, L.T)}


def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return 0
    T = WORKLOADS[args.workload]
    L = synth.config_decode(T=T)
    steps = []
    cb = None
    for i in range(args.warmup + args.steps):
        r = cpu_baseline(L, budget_s=4.0)
        if i >= args.warmup:
            steps.append(r["value"])
            cb = r
    v = statistics.median(steps)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * T / v, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": "mixtral-8x7b MoE layer decode, %d tokens, H 4096, F 14336, 8 experts, "
                                   "top-2, group 128, bits sum 20, ODP off" % T},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cb["cores"], "kind": "oracle",
                             "sample": cb["sample"]},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run(args):
    import torch
    import torch.distributed as dist

    import paper_2410_06270_gb300 as mc

    world, rank, local = _dist()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    T = WORKLOADS[args.workload]
    L = synth.config_decode(T=T)
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    flat = lambda a: [a[e][m] for e in range(L.E) for m in range(3)]
    packed_host = mc.pack_experts_host(shape, L.bits, flat(L.codes), flat(L.scale), flat(L.zero))
    # enough independent copies that one rotation exceeds L2 several times over
    nsets = max(2, int(np.ceil(4 * 132e6 / packed_host.nbytes)) + 1)
    packed = [torch.from_numpy(packed_host).to(dev) for _ in range(nsets)]
    x = torch.from_numpy(L.x.view(np.int16).copy()).view(torch.bfloat16).to(dev)
    gw = torch.from_numpy(L.gate.view(np.int16).copy()).view(torch.bfloat16).to(dev)
    ws = mc.alloc_workspace(shape, T, dev)
    y = torch.empty_like(x)
    idx = None

    def step(i):
        return mc.moe_forward(x, gw, shape, L.bits, packed[i % nsets], 0.0, None, y=y, workspace=ws)

    # routing once, to know which experts a step touches (fixed inputs)
    _, r = mc.moe_forward(x, gw, shape, L.bits, packed[0], 0.0, None, y=y, workspace=ws, routing=True)
    mc.check_status(ws)
    idx = r["idx"].cpu().numpy()
    touched = sorted(set(idx.reshape(-1).tolist()))
    alg_bytes, w13_bytes = _algorithmic_bytes(shape, L.bits, touched, T, L.H)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = Clocks(local)
    clocks.start()
    mc.profile_enable(True)
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for i in range(args.steps):
        step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    mc.profile_enable(False)
    prof = mc.profile_read()
    ms = e0.elapsed_time(e1)
    mc.check_status(ws)
    # end to end through the public API: pinned host input -> device -> layer -> host
    xh = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
    xh.copy_(x.cpu())
    yh = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
    torch.cuda.synchronize()
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e2.record(stream)
    for i in range(args.steps):
        x.copy_(xh, non_blocking=True)
        step(i)
        yh.copy_(y, non_blocking=True)
    e3.record(stream)
    torch.cuda.synchronize()
    ms_e2e = e2.elapsed_time(e3)
    cl = clocks.stop()

    t_local = torch.tensor([ms, ms_e2e], dtype=torch.float64, device=dev)
    if world > 1:
        dist.all_reduce(t_local, op=dist.ReduceOp.MAX)
        dist.barrier()
    ms, ms_e2e = float(t_local[0]), float(t_local[1])
    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return 0

    hbm, bf16, src = _peaks()
    w13_ms, w13_n = prof.get("gemv_w13", (0.0, 0))
    avg = w13_ms / max(w13_n, 1)
    achieved = w13_bytes / (avg * 1e-3) / 1e9 if avg > 0 else None
    launches = sum(n for _, n in prof.values())
    value = world * T * args.steps / (ms * 1e-3)
    e2e = world * T * args.steps / (ms_e2e * 1e-3)
    layer_gbs = alg_bytes * args.steps / (ms * 1e-3) / 1e9
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f16 x {1,2,3}-bit codes, fp32 accumulate", "data": "synthetic",
        "config": {"workload": "mixtral-8x7b MoE layer decode, %d tokens, H 4096, F 14336, 8 experts, top-2, "
                               "group 128, bits %s (mean %.2f), ODP off" % (T, list(map(int, L.bits)), L.mean_bits()),
                   "global_batch": T * world, "parallelism": "replicas" if world > 1 else "single",
                   "l2": "inputs larger than L2: %d rotating copies of the %.0f MB packed weights"
                         % (nsets, packed_host.nbytes / 1e6),
                   "touched_experts": len(touched)},
        "roofline": {"bound": "hbm", "kernel": "gemv_w13", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": (achieved / hbm) if achieved else None, "traffic": None,
                     "peak_source": "%s (MEASURED_PEAKS.json hbm_gbs)" % src if src == "measured" else src,
                     "algorithmic_bytes_per_launch": w13_bytes,
                     "layer_gbs": layer_gbs, "layer_frac": layer_gbs / hbm},
        "kernels_ms_per_step": {k: v[0] / max(v[1], 1) for k, v in prof.items()},
        "e2e": {"value": e2e, "unit": "tokens/s", "h2d_bytes_per_step": int(x.numel() * 2),
                "d2h_bytes_per_step": int(y.numel() * 2)},
        "gpu_launches": launches,
        "clocks": cl,
    }
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(L)
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="mc", choices=["mc", "reference"])
    ap.add_argument("--workload", default="decode16", choices=sorted(WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    return run(args)


if __name__ == "__main__":
    sys.exit(main())
