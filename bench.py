"""Benchmark of the MC compressed MoE layer (PMQ mixed-bit experts + ODP routing)
on GB300.

Default run: the headline line is one Mixtral-8x7b-shaped MoE layer in decode --
H 4096, SwiGLU F 14336, 8 experts, top-2, 16 tokens, group 128, per-expert bits
from {1,2,3} (sum 20, mean 2.5), ODP off -- the configuration the decode
tokens/s metric is quoted on; the same JSON line carries, under "workloads", the
other configurations measured the same way: the prefill layer (4096 tokens,
skewed expert loads), the ODP layer (256 tokens, 15% of secondaries pruned, 10%
protected) at bit sums 20 / 16 / 13, and the 32-layer stack at 32 tokens.  A
step is one pass of the whole layer (gate, top-2, ODP, permutation, W1|W3 +
SwiGLU, W2, combine; the stack: 32 of them with RMSNorm and residual adds) as a
CUDA graph replay on resident device inputs.  Packed weights rotate over several
device copies so that no step finds its weights in L2.

Timing: each workload replays K steps between CUDA events on the launching
stream, synchronised on both sides, in rounds until at least a second of timed
load has passed (so that the nvidia-smi sampler, started and read before the
first round, sees the GPU under load); the reported K-step time is the median
round.  The end-to-end figure (`e2e`) times K steps that each copy their input
from pinned host memory and their output back, in rounds (the median of at
least three), after one untimed replay of every graph it uses.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
      NAME: all (default: decode16 + the sub-records above) or one of
            decode16 decode1 decode4 decode16_8x22b decode16_fp16 prefill4096
            odp256 odp256_b16 odp256_b13 odp256_drop odp256_mask stack32
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
HBM_NOMINAL_GBS = 7900.0  # GB300 HBM3e nominal, reported beside the measured copy peak
WORKLOADS = {"decode16": ("decode", 16), "decode4": ("decode", 4), "decode1": ("decode", 1),
             "decode16_8x22b": ("decode", 16), "decode16_fp16": ("decode", 16),
             "prefill4096": ("prefill", 4096),
             "odp256": ("odp", 256), "odp256_b16": ("odp", 256), "odp256_b13": ("odp", 256),
             "odp256_drop": ("odp", 256), "odp256_mask": ("odp", 256),
             "stack32": ("stack", 32)}
# the default run: the headline workload, then the sub-records of the same line
HEADLINE = "decode16"
SUB_RECORDS = ("prefill4096", "odp256", "odp256_b16", "odp256_b13", "stack32")
NO_CPU_BASELINE = {"odp256_b16": "odp256", "odp256_b13": "odp256"}  # same layer shape and routing
STACK_LAYERS = 32
ODP_BITS = {"odp256": 20, "odp256_b16": 16, "odp256_b13": 13, "odp256_drop": 20, "odp256_mask": 20}
ODP_DROP = {"odp256_drop": 0.02}  # fraction of tokens whose experts are all masked (Sec. 3.2, Fig. 9)
# workloads whose step first computes the protect mask from an attention map (Eq. 6):
# heads of the synthetic causal attention, fraction of tokens protected
MASK_HEADS, MASK_PROTECT = 32, 0.02
ODP_PRUNE = 0.15  # fraction of unprotected tokens whose secondary expert the threshold drops
MIN_TIMED_S = 1.0  # timed load per workload (rounds of K steps)
CPU_BUDGET_S = 8.0  # host-core seconds of oracle work per workload's CPU baseline


def _peaks():
    """(HBM GB/s, bf16 TFLOP/s burst, bf16 TFLOP/s sustained, source)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons, read by a thread as
    the rows arrive (each row carries its own timestamp)."""

    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,utilization.gpu")
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.rows = []
        self.lock = threading.Lock()
        self.thread = None

    def _parse(self, line):
        f = [x.strip() for x in line.split(",")]
        if len(f) < 11:
            return None
        try:
            ts = time.mktime(time.strptime(f[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
            ts += float("0." + f[0].split(".")[1]) if "." in f[0] else 0.0
            util = float(f[10]) if f[10] not in ("[N/A]", "") else None
            return (ts, float(f[2]), float(f[3]), [n for n, v in zip(self.NAMES, f[6:10])
                                                   if v.lower().startswith("active")], util)
        except (ValueError, IndexError):
            return None

    def _reader(self):
        for line in self.proc.stdout:
            r = self._parse(line)
            if r is not None:
                with self.lock:
                    self.rows.append(r)

    def start(self, wait_s=5.0):
        """Start the sampler and return once its first row has arrived (or after
        wait_s seconds)."""
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return False
        self.thread = threading.Thread(target=self._reader, daemon=True)
        self.thread.start()
        t0 = time.time()
        while time.time() - t0 < wait_s:
            with self.lock:
                if self.rows:
                    return True
            time.sleep(0.02)
        return False

    def stop(self, window=None):
        """Median SM clock and the throttle reasons seen; samples restricted to
        `window` = (t0, t1) host wall-clock seconds when any fall inside it."""
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=5)
        with self.lock:
            rows = list(self.rows)
        if not rows:
            return None
        where = "run"
        if window is not None:
            inside = [r for r in rows if window[0] <= r[0] <= window[1]]
            if inside:
                rows, where = inside, "timed region"
        reasons = sorted({n for r in rows for n in r[3]})
        loaded = [r for r in rows if r[4] is not None and r[4] > 0]
        return {"sm_mhz": statistics.median(r[1] for r in rows), "sm_max_mhz": max(r[2] for r in rows),
                "samples": len(rows), "samples_under_load": len(loaded), "window": where, "reasons": reasons}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(values, device="cpu"):
    """Element-wise max of `values` over the ranks of the default process group
    (the slowest replica's times); the values themselves without one."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def job_throughput(world, units_per_rank, steps, ms):
    """Whole-job units per second: every rank processes units_per_rank per step;
    the job takes the slowest rank's `ms` for `steps` steps."""
    return world * units_per_rank * steps / (ms * 1e-3)


def _timed_rounds(torch, replay, steps, stream, world, min_s=MIN_TIMED_S, max_rounds=5000):
    """Rounds of exactly `steps` replays between CUDA events on `stream`,
    synchronised (and, with several ranks, barriered) on both sides, repeated
    until at least min_s seconds of rounds have passed.  Returns (median round
    ms, every round's ms, (wall t0, wall t1))."""
    import torch.distributed as dist
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    rounds = []
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    w0 = time.time()
    i = 0
    while True:
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(steps):
            replay(i)
            i += 1
        e1.record(stream)
        torch.cuda.synchronize()
        rounds.append(e0.elapsed_time(e1))
        if len(rounds) >= max_rounds or (len(rounds) >= 3 and time.time() - w0 >= min_s):
            break
    if world > 1:
        dist.barrier()
    w1 = time.time()
    return statistics.median(rounds), rounds, (w0, w1)


def _e2e_pipelined(torch, step, nsets, x, y, steps, stream, min_s=MIN_TIMED_S / 2, max_rounds=2000):
    """End to end: every step copies an input from pinned host memory to the
    device and an output back, over two device buffer pairs.  A step is one graph
    replay with three branches: the layer on pair b, the host->device copy of the
    next step's input into pair 1-b and the device->host copy of the previous
    step's output out of pair 1-b, so the copies overlap the layer with no
    cross-stream synchronisation between steps.  A round is `steps` such steps
    plus the first input's copy before them and the last output's copy after
    them, timed from before the first copy to after the last; each graph is
    replayed once before the first round (its first launch uploads it), and
    rounds repeat (at least 3) until `min_s` seconds have passed.  Returns the
    median round's milliseconds."""
    xh = [torch.empty(x.shape, dtype=x.dtype, pin_memory=True) for _ in range(2)]
    yh = [torch.empty(y.shape, dtype=y.dtype, pin_memory=True) for _ in range(2)]
    for b in range(2):
        xh[b].copy_(x.cpu())
    xd = [torch.empty_like(x) for _ in range(2)]
    yd = [torch.empty_like(y) for _ in range(2)]
    graphs = {}
    for k in range(nsets):
        for b in range(2):
            gr = torch.cuda.CUDAGraph()
            cs, side = torch.cuda.Stream(), torch.cuda.Stream()
            cs.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(cs):
                with torch.cuda.graph(gr, stream=cs):
                    fork, join = torch.cuda.Event(), torch.cuda.Event()
                    fork.record(cs)
                    side.wait_event(fork)
                    with torch.cuda.stream(side):
                        xd[1 - b].copy_(xh[1 - b], non_blocking=True)  # the next step's input
                        yh[1 - b].copy_(yd[1 - b], non_blocking=True)  # the previous step's output
                        join.record(side)
                    step(k, xd[b], yd[b])
                    cs.wait_event(join)
            torch.cuda.current_stream().wait_stream(cs)
            graphs[k, b] = gr
    for gr in graphs.values():
        gr.replay()
    torch.cuda.synchronize()
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    last = (steps - 1) % 2

    def one_round():
        e2.record(stream)
        xd[0].copy_(xh[0], non_blocking=True)
        for i in range(steps):
            graphs[i % nsets, i % 2].replay()
        yh[last].copy_(yd[last], non_blocking=True)
        e3.record(stream)
        torch.cuda.synchronize()
        return e2.elapsed_time(e3)

    rounds, w0 = [], time.time()
    while len(rounds) < 3 or (time.time() - w0 < min_s and len(rounds) < max_rounds):
        rounds.append(one_round())
    del graphs
    return statistics.median(rounds)


def _algorithmic_bytes(shape, bits, touched, T, H):
    """Packed weight bytes of the touched experts (codes + fp16 scale/zero) plus
    the gate, activations and output.  Returns (total, w13 part)."""
    # 16-bit (unquantised) experts carry no scale / zero
    per_mat = lambda b: H * shape.F * b / 8 + (0 if b == 16 else H * shape.F / shape.group * 4)
    w13 = sum(2 * per_mat(int(bits[e])) for e in touched)
    w2 = sum(per_mat(int(bits[e])) for e in touched)
    other = shape.E * H * 2 + 2 * T * H * 2
    return w13 + w2 + other, w13


def _oracle_mats(oracle, L):
    """The oracle's expert matrices of a synthetic layer (16-bit experts: dense fp16 weights)."""
    def one(e, m):
        if int(L.bits[e]) == 16:
            return oracle.QMat(*L.mat_shape(m), L.group, 16, dense=np.asarray(L.codes[e][m], np.float32))
        return oracle.QMat(*L.mat_shape(m), L.group, int(L.bits[e]), L.codes[e][m], L.scale[e][m], L.zero[e][m])
    return [[one(e, m) for m in range(3)] for e in range(L.E)]


def cpu_baseline(L, budget_s=CPU_BUDGET_S, threads=None):
    """Time the oracle, as it stands, on a bounded sample of the workload's tokens
    (one token per host thread)."""
    import concurrent.futures as cf

    import oracle
    mats = _oracle_mats(oracle, L)
    xf, gf = L.x_f32(), L.gate_f32()
    t_mask = 0.0
    if name_has_mask(L):  # the step's Eq. 6 mask, for all tokens (charged pro rata below)
        t0 = time.perf_counter()
        oracle.token_importance(xf, L.attn, MASK_PROTECT)
        t_mask = time.perf_counter() - t0
    t0 = time.perf_counter()
    oracle.moe_layer(xf, gf, mats, L.mu, L.protect, tokens=[0])
    one = time.perf_counter() - t0
    cores = threads or (os.cpu_count() or 1)
    n = int(max(1, min(L.T, cores, round(budget_s / max(one, 1e-3) * cores / 2))))
    toks = list(range(n))
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(min(n, cores)) as ex:
        list(ex.map(lambda t: oracle.moe_layer(xf, gf, mats, L.mu, L.protect, tokens=[t]), toks))
    dt = time.perf_counter() - t0 + t_mask * n / L.T
    return {"value": n / dt, "unit": "tokens/s", "cores": min(n, cores), "kind": "oracle",
            "single_thread_value": 1.0 / (one + t_mask / L.T),
            "sample": "%d of the workload's %d tokens (full layer per token, fp64, one token per thread%s); "
                      "single_thread_value: token 0 alone on one thread" % (
                          n, L.T, "; plus the Eq. 6 mask of all tokens, charged n/T of its time" if t_mask else "")}


def _oracle_stack_mus(L, gates, mats, nl, threads=None):
    """Per-layer thresholds of the first nl layers along the oracle's own
    trajectory (untimed calibration of the reference arm): at each layer, the
    ODP_PRUNE quantile of w1/w0 over the unprotected tokens' routing at mu = 0,
    then every token through that layer with it (one token per thread)."""
    import concurrent.futures as cf

    import oracle
    gf = [synth.bf16_bits_to_f32(g) for g in gates]
    h = L.x_f32().astype(np.float64)
    mus = []
    for l in range(nl):
        xn = oracle.bf16_round(np.stack([oracle.rmsnorm(h[t], np.ones(L.H, np.float32), 1e-5) for t in range(L.T)]))
        _, w, _ = oracle.route(xn, gf[l], 0.0, L.protect)
        ratio = w[:, 1].astype(np.float64) / w[:, 0]
        mus.append(float(np.quantile(ratio[L.protect == 0], ODP_PRUNE)))
        one = lambda t: oracle.stack(h[t:t + 1], [gf[l]], mats, [mus[-1]], L.protect[t:t + 1])[0][0]
        with cf.ThreadPoolExecutor(threads or os.cpu_count() or 1) as ex:
            h = np.stack(list(ex.map(one, range(L.T))))
    return mus


def cpu_baseline_stack(L, gates, mus=None, budget_s=CPU_BUDGET_S, threads=None):
    """The oracle's stack on a bounded sample of the workload: one token per host
    thread through the first `nl` of the stack's layers (nl sized to the budget;
    every layer has the same shape), scaled to whole-stack tokens/s by nl / layers.
    mus: the per-layer thresholds (None: calibrated along the oracle's own
    trajectory for the layers it runs, untimed)."""
    import concurrent.futures as cf

    import oracle
    mats = _oracle_mats(oracle, L)
    gf = [synth.bf16_bits_to_f32(g) for g in gates]
    xf = L.x_f32()
    layers = len(gates)
    cores = threads or (os.cpu_count() or 1)
    t0 = time.perf_counter()
    oracle.stack(xf[:1], gf[:1], mats, [0.0], L.protect[:1])
    one = time.perf_counter() - t0  # one token, one layer
    n = int(max(1, min(L.T, cores)))
    nl = int(max(1, min(layers, round(budget_s / max(one, 1e-3) / 2))))
    if mus is None:  # calibrated once per workload object
        mus = getattr(L, "oracle_mus", None)
        if mus is None or len(mus) < nl:
            mus = L.oracle_mus = _oracle_stack_mus(L, gates, mats, nl, threads)
    run = lambda t: oracle.stack(xf[t:t + 1], gf[:nl], mats, list(mus[:nl]), L.protect[t:t + 1])
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(n) as ex:
        list(ex.map(run, range(n)))
    dt = time.perf_counter() - t0
    return {"value": n * nl / layers / dt, "unit": "tokens/s", "cores": n, "kind": "oracle",
            "single_thread_value": 1.0 / (one * layers),
            "sample": "%d of the workload's %d tokens, one token per thread through the first %d of its %d layers "
                      "(fp64), scaled by %d/%d to whole-stack tokens/s; single_thread_value: token 0 through one "
                      "layer alone on one thread, times %d" % (n, L.T, nl, layers, nl, layers, layers)}


def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return 0
    name = HEADLINE if args.workload == "all" else args.workload
    kind, T, L = _workload(name)
    if kind == "stack":
        L, gates = L
        mus = None  # calibrated along the oracle's own trajectory
    if kind == "odp":
        import oracle
        if name_has_mask(L):
            L.protect = oracle.token_importance(L.x_f32(), L.attn, MASK_PROTECT)[1]
        _, w, _ = oracle.route(L.x_f32(), L.gate_f32(), 0.0, L.protect)
        L.mu = oracle.odp_threshold(w, L.protect, ODP_PRUNE)
    steps = args.steps if args.steps else 3
    vals = []
    cb = None
    budget = min(4.0, 150.0 / (args.warmup + steps))  # the whole run stays within a few minutes
    for i in range(args.warmup + steps):
        r = cpu_baseline_stack(L, gates, mus, budget_s=budget) if kind == "stack" else cpu_baseline(L, budget_s=budget)
        if i >= args.warmup:
            vals.append(r["value"])
            cb = r
    v = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": steps, "warmup": args.warmup, "ms_per_step": 1000.0 * T / v, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": _describe(kind, T, L)},
            "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cb["cores"], "kind": "oracle",
                             "sample": cb["sample"]},
            "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def _workload(name):
    kind, T = WORKLOADS[name]
    if kind == "decode":
        L = synth.config_decode_22b(T=T) if name.endswith("8x22b") else \
            synth.config_decode_fp16(T=T) if name.endswith("fp16") else synth.config_decode(T=T)
    elif kind == "prefill":
        L = synth.config_prefill(T=T)
    elif kind == "stack":
        L = synth.config_stack(T=T, layers=STACK_LAYERS)
    else:
        L = synth.config_odp(T=T, bits_total=ODP_BITS[name])
        if name in ODP_DROP:
            L.protect = synth.importance_mask(L.x, 0.10, ODP_DROP[name], 1238)
    if name.endswith("_mask"):
        # the step computes the protect mask from this attention map (Eq. 6)
        L.mask_step = True
        L.attn = synth.causal_attention(MASK_HEADS, T, 1240)
    return kind, T, L


def _describe(kind, T, L):
    if kind == "stack":
        L = L[0] if isinstance(L, tuple) else L
        return ("mixtral-8x7b stack of %d pre-norm MoE layers (h <- h + MoE(RMSNorm(h))), %d tokens, H 4096, "
                "F 14336, 8 experts, top-2, group 128, bits %s (mean %.2f), ODP on (per-layer mu dropping the "
                "secondary expert of %d%% of unprotected tokens), %d%% of tokens protected, whole stack in one "
                "CUDA graph" % (STACK_LAYERS, T, list(map(int, L.bits)), L.mean_bits(), round(100 * ODP_PRUNE),
                                round(100 * float((L.protect == 1).mean()))))
    if name_has_mask(L):
        return ("mixtral-8x7b MoE layer %s, %d tokens, H 4096, F 14336, 8 experts, top-2, group 128, bits %s "
                "(mean %.2f), the step computes the protect mask of the top %d%% tokens from a %d-head causal "
                "attention map (Eq. 6) and runs the layer with ODP (mu %.4g: drops the secondary expert of %d%% of "
                "unprotected tokens)%s" % (kind, T, list(map(int, L.bits)), L.mean_bits(), round(100 * MASK_PROTECT),
                                           MASK_HEADS, L.mu, round(100 * ODP_PRUNE),
                                           ", expert loads skewed ~4:1" if kind == "prefill" else ""))
    if kind == "odp":
        odp = "ODP on (mu %.4g: drops the secondary expert of %d%% of unprotected tokens), %d%% of tokens " \
              "protected by the importance surrogate" % (L.mu, round(100 * ODP_PRUNE),
                                                         round(100 * float((L.protect == 1).mean())))
        if (L.protect == 2).any():
            odp += ", the %d%% least important tokens dropped (all experts masked)" % round(
                100 * float((L.protect == 2).mean()))
    else:
        odp = "ODP off"
    model = "mixtral-8x22b" if L.H == synth.MIXTRAL22_H else "mixtral-8x7b"
    if int(L.bits[0]) == 16:
        odp += ", experts unquantised (fp16 weights: the baseline of the mixed-bit layer)"
    return ("%s MoE layer %s, %d tokens, H %d, F %d, 8 experts, top-2, group 128, bits %s "
            "(mean %.2f), %s%s" % (model, kind, T, L.H, L.F, list(map(int, L.bits)), L.mean_bits(), odp,
                                   ", expert loads skewed ~4:1" if kind == "prefill" else ""))


def name_has_mask(L):
    return getattr(L, "mask_step", False)


def _odp_threshold(mc, x, gw, shape, protect_np, protect_dev):
    """mu that prunes ODP_PRUNE of the prunable tokens: the library's quantile of
    w1/w0 (mc_odp_threshold_host) over its own routing weights at mu = 0."""
    r = mc.route(x, gw, shape, 0.0, protect_dev)
    return mc.odp_threshold(r["w"], protect_np, ODP_PRUNE)


def _traffic(kernel, workload):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if it was
    taken on the kernel's current source (else None)."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            d = json.load(f)[kernel + "/" + workload]
        with open(os.path.join(ROOT, "paper_2410_06270_gb300", "csrc", d["source"]), "rb") as f:
            sha = hashlib.sha256(f.read()).hexdigest()
        return float(d["bytes_per_launch"]) if sha == d["source_sha256"] else None
    except Exception:
        return None


def _graph_profile(mc, torch, step, nsets, kernels, rounds):
    """{kernel: (mean ms per launch, launches per step)} from CUDA graphs of the step
    captured with the library's profiling events (event nodes around the selected
    kernels), one graph per rotating weight copy; each round replays every graph
    once and reads the events of those replays."""
    mc.profile_clear()
    mc.profile_select(kernels)
    mc.profile_enable(True)
    graphs = []
    for k in range(nsets):
        gr = torch.cuda.CUDAGraph()
        cs = torch.cuda.Stream()
        cs.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(cs):
            with torch.cuda.graph(gr, stream=cs):
                step(k)
        torch.cuda.current_stream().wait_stream(cs)
        graphs.append(gr)
    mc.profile_enable(False)
    mc.profile_select(None)
    tot = {}
    for _ in range(rounds):
        for gr in graphs:
            gr.replay()
        for name, (ms, n) in mc.profile_read().items():
            a = tot.setdefault(name, [0.0, 0])
            a[0] += ms
            a[1] += n
    mc.profile_clear()
    del graphs
    return {name: (ms / max(n, 1), n / (rounds * nsets)) for name, (ms, n) in tot.items()}


def _clock_note(cl):
    if cl is None:
        return None
    cl = dict(cl)
    cl["note"] = "nvidia-smi -lms 50 rows read as they arrive; sampler started (first row received) before the " \
                 "first timed round; rows restricted to the timed rounds' wall-clock window"
    return cl


def measure_layer(name, args, torch, mc, dev, local, world, cpu=True):
    """One single-layer workload.  Returns the JSON record (the slowest rank's
    times; value = whole-job tokens/s)."""
    kind, T, L = _workload(name)
    steps = args.steps if args.steps else {"decode": 2000, "odp": 1000, "prefill": 100}[kind]
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    flat = lambda a: [a[e][m] for e in range(L.E) for m in range(3)]
    packed_host = mc.pack_experts_host(shape, L.bits, flat(L.codes), flat(L.scale), flat(L.zero))
    # enough independent copies that one rotation exceeds L2 several times over
    nsets = max(2, int(np.ceil(4 * 132e6 / packed_host.nbytes)) + 1)
    packed = [torch.from_numpy(packed_host).to(dev) for _ in range(nsets)]
    x = torch.from_numpy(L.x.view(np.int16).copy()).view(torch.bfloat16).to(dev)
    gw = torch.from_numpy(L.gate.view(np.int16).copy()).view(torch.bfloat16).to(dev)
    prot = None if L.protect is None else torch.from_numpy(L.protect.copy()).to(dev)
    attn = imp = iws = None
    if name_has_mask(L):
        # the protect mask comes from the step itself (Eq. 6 on the attention map)
        attn = torch.from_numpy(L.attn).to(dev)
        imp = torch.empty(T, dtype=torch.float32, device=dev)
        prot = torch.empty(T, dtype=torch.uint8, device=dev)
        iws = torch.empty(mc.load().mc_token_importance_workspace_size(T), dtype=torch.uint8, device=dev)
        mc.token_importance(x, attn, MASK_PROTECT, importance=imp, mask=prot, workspace=iws)
        L.protect = prot.cpu().numpy()
    if kind == "odp" or attn is not None:
        L.mu = _odp_threshold(mc, x, gw, shape, L.protect, prot)
    mu = float(L.mu)
    ws = mc.alloc_workspace(shape, T, dev)
    y = torch.empty_like(x)

    def step(i, xb=None, yb=None):
        xb = x if xb is None else xb
        yb = y if yb is None else yb
        if attn is not None:
            mc.token_importance(xb, attn, MASK_PROTECT, importance=imp, mask=prot, workspace=iws)
        return mc.moe_forward(xb, gw, shape, L.bits, packed[i % nsets], mu, prot, y=yb, workspace=ws)

    # routing once, to know which experts a step touches and how many pairs it keeps (fixed inputs)
    _, r = mc.moe_forward(x, gw, shape, L.bits, packed[0], mu, prot, y=y, workspace=ws, routing=True)
    mc.check_status(ws)
    idx = r["idx"].cpu().numpy()
    pr = r["pruned"].cpu().numpy()
    pairs = int(2 * T - int(np.minimum(pr, 1).sum()) - int((pr == 2).sum()))
    keep = np.stack([pr != 2, pr == 0], axis=1)
    touched = sorted(set(idx[keep].reshape(-1).tolist()))
    alg_bytes, w13_bytes = _algorithmic_bytes(shape, L.bits, touched, T, L.H)
    w13_flops = 4.0 * L.H * L.F * pairs          # W1 and W3: 2 x (2 H F) per kept pair
    layer_flops = 6.0 * L.H * L.F * pairs + 2.0 * L.H * L.E * T
    rk = "gemv_w13" if 2 * T < 240 else "gemm_w13"  # the path mc_moe_forward picks (kPrefillPairs)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    # one CUDA graph per rotating weight copy: a step is a graph replay
    graphs = []
    for k in range(nsets):
        gr = torch.cuda.CUDAGraph()
        cs = torch.cuda.Stream()
        cs.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(cs):
            with torch.cuda.graph(gr, stream=cs):
                step(k)
        torch.cuda.current_stream().wait_stream(cs)
        graphs.append(gr)
    for i in range(args.warmup):
        graphs[i % nsets].replay()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    clocks = Clocks(local)
    clocks.start()
    ms, rounds, window = _timed_rounds(torch, lambda i: graphs[i % nsets].replay(), steps, stream, world)
    cl = clocks.stop(window)
    mc.check_status(ws)
    # the roofline kernel's launch duration: CUDA events around that kernel only,
    # captured as event nodes of a profiling copy of the step graphs (events inside
    # the timed graphs would serialise the launches they bracket); then the
    # per-kernel breakdown from a second profiling copy with every kernel bracketed
    prof = _graph_profile(mc, torch, step, nsets, [rk], rounds=max(3, min(steps, 200)))
    breakdown = _graph_profile(mc, torch, step, nsets, None, rounds=max(3, min(steps, 50)))
    ms_e2e = _e2e_pipelined(torch, step, nsets, x, y, steps, stream)
    ms, ms_e2e, avg = max_over_ranks([ms, ms_e2e, prof.get(rk, (0.0, 0))[0]], dev)
    del graphs

    hbm, bf16, bf16_sus, src = _peaks()
    value = job_throughput(world, T, steps, ms)
    e2e = job_throughput(world, T, steps, ms_e2e)
    layer_s = ms * 1e-3 / steps
    layer_gbs = alg_bytes / layer_s / 1e9
    layer_tf = layer_flops / layer_s / 1e12
    t_hbm, t_tc = alg_bytes / (hbm * 1e9), layer_flops / (bf16 * 1e12)
    layer_roof = {"bytes": alg_bytes, "flops": layer_flops, "hbm_bound_us": t_hbm * 1e6, "tensor_bound_us": t_tc * 1e6,
                  "binding": "hbm" if t_hbm >= t_tc else "tensor", "measured_us": layer_s * 1e6,
                  "frac": max(t_hbm, t_tc) / layer_s, "gbs": layer_gbs, "hbm_frac": layer_gbs / hbm,
                  "tflops": layer_tf, "tensor_frac_burst": layer_tf / bf16,
                  "note": "whole-step roofline: max(algorithmic bytes / measured HBM peak, algorithmic flops / "
                          "measured bf16 burst peak) / measured step time"}
    if rk == "gemv_w13":
        achieved = w13_bytes / (avg * 1e-3) / 1e9 if avg > 0 else None
        roof = {"bound": "hbm", "kernel": rk, "achieved": achieved, "peak": hbm, "unit": "GB/s",
                "frac": (achieved / hbm) if achieved else None, "traffic": _traffic(rk, name),
                "peak_source": "%s (MEASURED_PEAKS.json hbm_gbs)" % src if src == "measured" else src,
                "frac_of_nominal_7900": (achieved / HBM_NOMINAL_GBS) if achieved else None,
                "algorithmic_bytes_per_launch": w13_bytes, "kernel_us": avg * 1e3,
                "layer_gbs": layer_gbs, "layer_frac": layer_gbs / hbm}
    else:
        achieved = w13_flops / (avg * 1e-3) / 1e12 if avg > 0 else None
        roof = {"bound": "tensor", "kernel": rk, "achieved": achieved, "peak": bf16, "unit": "TFLOP/s",
                "frac": (achieved / bf16) if achieved else None, "traffic": _traffic(rk, name),
                "peak_source": "%s (MEASURED_PEAKS.json bf16_tflops: the burst peak, the kernel runs for "
                               "milliseconds at most; fp16 has the bf16 rate)" % src if src == "measured" else src,
                "peak_sustained": bf16_sus, "frac_of_sustained": (achieved / bf16_sus) if achieved else None,
                "algorithmic_flops_per_launch": w13_flops, "kernel_us": avg * 1e3, "kept_pairs": pairs,
                "layer_tflops": layer_tf, "layer_frac": layer_tf / bf16,
                "layer_gbs": layer_gbs, "layer_hbm_frac": layer_gbs / hbm}
    rec = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": steps,
        "warmup": args.warmup, "ms_per_step": ms / steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "data": "synthetic",
        "dtype": "f16 x f16 (unquantised experts), fp32 accumulate" if int(L.bits[0]) == 16 else
                 "f16 x {1,2,3}-bit codes, fp32 accumulate",
        "config": {"workload": _describe(kind, T, L),
                   "global_batch": T * world, "parallelism": "replicas" if world > 1 else "single",
                   "l2": "inputs larger than L2: %d rotating copies of the %.0f MB packed weights"
                         % (nsets, packed_host.nbytes / 1e6),
                   "touched_experts": len(touched), "kept_pairs": pairs},
        "roofline": roof,
        "layer_roofline": layer_roof,
        "timing": {"rounds": len(rounds), "round_ms_median": ms, "round_ms_min": min(rounds),
                   "round_ms_max": max(rounds), "timed_s": window[1] - window[0],
                   "how": "rounds of exactly K CUDA graph replays between CUDA events on the launching stream, "
                          "synchronised on both sides, until >= %.1f s; median round reported" % MIN_TIMED_S},
        "kernels_ms_per_step": {k: v[0] * v[1] for k, v in breakdown.items()},
        "launch": "roofline kernel duration = mean of CUDA events around that kernel, captured as event nodes in "
                  "profiling copies of the step graphs (%d replays); kernels_ms_per_step from copies with every "
                  "kernel bracketed (each event node between two kernels removes their programmatic launch "
                  "overlap, so the sum exceeds ms_per_step)" % (nsets * max(3, min(steps, 200))),
        "e2e": {"value": e2e, "unit": "tokens/s", "h2d_bytes_per_step": int(x.numel() * 2),
                "d2h_bytes_per_step": int(y.numel() * 2),
                "copies": "pinned host buffers, two device buffer pairs; every step is one graph replay "
                          "whose branches copy step i+1's input in and step i-1's output out while step i's "
                          "layer runs (plus the first input before and the last output after the steps)"},
        "gpu_launches": int(round(sum(n for _, n in breakdown.values()))) * steps,
        "clocks": _clock_note(cl),
    }
    if cpu and not args.no_cpu_baseline:
        rec["cpu_baseline"] = cpu_baseline(L)
    del packed, ws, x, y
    torch.cuda.empty_cache()
    return rec


def measure_stack(name, args, torch, mc, dev, local, world, cpu=True):
    """The 32-layer stack: one mc_stack_forward captured into a CUDA graph (with the
    copy of the step's input into the residual stream), replayed."""
    kind, T, (L, gates) = _workload(name)
    layers = len(gates)
    steps = args.steps if args.steps else 100
    shape = mc.Shape(L.E, L.H, L.F, L.group)
    flat = lambda a: [a[e][m] for e in range(L.E) for m in range(3)]
    packed_host = mc.pack_experts_host(shape, L.bits, flat(L.codes), flat(L.scale), flat(L.zero))
    packs = [torch.from_numpy(packed_host).to(dev) for _ in range(layers)]  # every layer streams its own copy
    bf = lambda b: torch.from_numpy(b.view(np.int16).copy()).view(torch.bfloat16).to(dev)
    x0 = bf(L.x)
    gw = [bf(g) for g in gates]
    prot = torch.from_numpy(L.protect.copy()).to(dev)
    gamma = torch.ones((layers, L.H), dtype=torch.bfloat16, device=dev)
    # per-layer thresholds from this layer's own routing along the stack's trajectory at mu = 0
    mus, touched, pairs = [], [], 0
    h = x0.clone()
    wsl = mc.alloc_workspace(shape, T, dev)
    for l in range(layers):
        xn = mc.rmsnorm(h, gamma[l])
        r = mc.route(xn, gw[l], shape, 0.0, prot)
        w = r["w"].cpu().numpy().astype(np.float64)
        mus.append(float(np.quantile((w[:, 1] / w[:, 0])[L.protect == 0], ODP_PRUNE)))
        y, rr = mc.moe_forward(xn, gw[l], shape, L.bits, packs[l], mus[-1], prot, workspace=wsl, routing=True)
        pr = rr["pruned"].cpu().numpy()
        keep = np.stack([pr != 2, pr == 0], axis=1)
        touched.append(sorted(set(rr["idx"].cpu().numpy()[keep].reshape(-1).tolist())))
        pairs += int(keep.sum())
        h = mc.add(h, y)
    mc.check_status(wsl)
    del wsl
    args_s = mc.StackArgs(gw, [L.bits] * layers, packs, mus)
    ws = mc.stack_workspace(shape, T, dev)
    hs = x0.clone()
    mc.stack_forward(hs, shape, args_s, gamma, ws, prot)  # sets the kernels' attributes before capture
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    cs = torch.cuda.Stream()
    cs.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cs):
        with torch.cuda.graph(graph, stream=cs):
            hs.copy_(x0)
            mc.stack_forward(hs, shape, args_s, gamma, ws, prot)
    torch.cuda.current_stream().wait_stream(cs)
    alg = sum(_algorithmic_bytes(shape, L.bits, t, T, L.H)[0] for t in touched)
    flops = 6.0 * L.H * L.F * pairs + 2.0 * L.H * L.E * T * layers

    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    clocks = Clocks(local)
    clocks.start()
    ms, rounds, window = _timed_rounds(torch, lambda i: graph.replay(), steps, stream, world)
    cl = clocks.stop(window)
    mc.check_status(ws)
    # per-kernel breakdown: one eager profiled call
    mc.profile_select(None)
    mc.profile_enable(True)
    mc.stack_forward(hs, shape, args_s, gamma, ws, prot)
    torch.cuda.synchronize()
    mc.profile_enable(False)
    breakdown = mc.profile_read()
    # end to end: pinned host input -> device -> graph -> host
    xh = torch.empty(x0.shape, dtype=x0.dtype, pin_memory=True)
    xh.copy_(x0.cpu())
    yh = torch.empty(x0.shape, dtype=x0.dtype, pin_memory=True)
    torch.cuda.synchronize()
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e2e_rounds, w0 = [], time.time()
    while len(e2e_rounds) < 3 or time.time() - w0 < MIN_TIMED_S / 2:
        e2.record(stream)
        for _ in range(steps):
            x0.copy_(xh, non_blocking=True)
            graph.replay()
            yh.copy_(hs, non_blocking=True)
        e3.record(stream)
        torch.cuda.synchronize()
        e2e_rounds.append(e2.elapsed_time(e3))
    ms_e2e = statistics.median(e2e_rounds)
    ms, ms_e2e = max_over_ranks([ms, ms_e2e], dev)
    del graph
    hbm, bf16, _, src = _peaks()
    step_s = ms * 1e-3 / steps
    gbs = alg / step_s / 1e9
    rec = {
        "metric": METRIC, "value": job_throughput(world, T, steps, ms), "unit": "tokens/s", "n_gpus": world,
        "steps": steps, "warmup": args.warmup, "ms_per_step": ms / steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f16 x {1,2,3}-bit codes, fp32 accumulate",
        "data": "synthetic",
        "config": {"workload": _describe(kind, T, L), "global_batch": T * world,
                   "parallelism": "replicas" if world > 1 else "single",
                   "l2": "inputs larger than L2: %d layers x %.0f MB packed weights, one device copy per layer"
                         % (layers, packed_host.nbytes / 1e6),
                   "weights": "one seeded expert set shared by the layers (separate copies), per-layer gates",
                   "kept_pairs": pairs},
        "roofline": {"bound": "hbm", "kernel": "stack step (CUDA graph: %d layers of rmsnorm, route, permute, "
                                                "GEMV W1|W3, GEMV W2, combine; RMSNorm in the routing launch, residual add in the combine)" % layers,
                     "achieved": gbs, "peak": hbm, "unit": "GB/s", "frac": gbs / hbm, "traffic": None,
                     "frac_of_nominal_7900": gbs / HBM_NOMINAL_GBS,
                     "peak_source": "%s (MEASURED_PEAKS.json hbm_gbs)" % src if src == "measured" else src,
                     "algorithmic_bytes_per_step": alg, "tensor_frac_burst": flops / step_s / 1e12 / bf16},
        "timing": {"rounds": len(rounds), "round_ms_median": ms, "round_ms_min": min(rounds),
                   "round_ms_max": max(rounds), "timed_s": window[1] - window[0]},
        "kernels_ms_per_step": {k: v[0] for k, v in breakdown.items()},
        "e2e": {"value": job_throughput(world, T, steps, ms_e2e), "unit": "tokens/s",
                "h2d_bytes_per_step": int(x0.numel() * 2), "d2h_bytes_per_step": int(hs.numel() * 2)},
        # the profiled kernels of one call (each layer's RMSNorm runs in its routing
        # launch and its residual add in its combine)
        "gpu_launches": _launches_per_step(breakdown, 1) * steps,
        "clocks": _clock_note(cl),
    }
    if cpu and not args.no_cpu_baseline:
        rec["cpu_baseline"] = cpu_baseline_stack(L, gates, mus)
    del packs, ws, hs, x0
    torch.cuda.empty_cache()
    return rec


def _launches_per_step(breakdown, n):
    return int(round(sum(c for _, c in breakdown.values()) / max(n, 1)))


def _measure(name, args, torch, mc, dev, local, world, cpu=True):
    fn = measure_stack if WORKLOADS[name][0] == "stack" else measure_layer
    return fn(name, args, torch, mc, dev, local, world, cpu=cpu)


def run(args):
    import torch
    import torch.distributed as dist

    import paper_2410_06270_gb300 as mc

    world, rank, local = _dist()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    if args.workload == "all":
        line = _measure(HEADLINE, args, torch, mc, dev, local, world)
        subs = {}
        for name in SUB_RECORDS:
            rec = _measure(name, args, torch, mc, dev, local, world, cpu=name not in NO_CPU_BASELINE)
            if name in NO_CPU_BASELINE and "cpu_baseline" in subs.get(NO_CPU_BASELINE[name], {}):
                rec["cpu_baseline"] = dict(subs[NO_CPU_BASELINE[name]]["cpu_baseline"],
                                           sample="that of %s (same layer shape, routing and oracle work per "
                                                  "token)" % NO_CPU_BASELINE[name])
            for k in ("metric", "n_gpus", "steps", "warmup", "higher_is_better", "scaling", "vs_baseline", "data"):
                rec.pop(k, None)
            subs[name] = rec
        line["workloads"] = subs
        line["gpu_launches_all_workloads"] = line["gpu_launches"] + sum(r["gpu_launches"] for r in subs.values())
    else:
        line = _measure(args.workload, args, torch, mc, dev, local, world)
    if world > 1:
        dist.barrier()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0, help="timed steps per round (default: 2000 decode, 1000 ODP, "
                                                         "100 prefill and stack)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="mc", choices=["mc", "reference"])
    ap.add_argument("--workload", default="all", choices=["all"] + sorted(WORKLOADS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    return run(args)


if __name__ == "__main__":
    sys.exit(main())
