"""Benchmark of the compressed-MoE forward (LorExperts / BTExperts) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl lx|reference]

A step is one full forward (route, bucket, shared anchor and correction
products with SwiGLU, down projection, combine) over one batch of synthetic
tokens, inputs already resident in HBM.  The default workload is the
Qwen3-30B-A3B-shaped layer (H=2048, I=768, E=128 top-8, 32 clusters of 4,
rank-128 members, bf16) at a decode batch of 64 tokens.  Four device copies of
the layer (2 GB) rotate between steps and every step takes a fresh token batch,
so weights come from HBM, not L2.

Prints one JSON line (rank 0).  `--impl reference` times the CPU oracle (the
plain definition of the method) on the host cores instead, on a bounded sample.
Under torchrun every rank runs its own replica on its own batches (no
collective on the data path); the timing is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import shutil
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "compressed-MoE layer tokens/s (1 GB300); % HBM roofline decode, % bf16 peak prefill"

WORKLOADS = {
    # name: (layer maker, T, description)
    "decode64": ("qwen", 64, "Qwen3-30B-A3B-shaped compressed MoE layer, decode batch of 64 tokens"),
    "decode32": ("qwen", 32, "Qwen3-30B-A3B-shaped compressed MoE layer, decode batch of 32 tokens"),
    "decode8": ("qwen", 8, "Qwen3-30B-A3B-shaped compressed MoE layer, decode batch of 8 tokens"),
    "decode1": ("qwen", 1, "Qwen3-30B-A3B-shaped compressed MoE layer, decode batch of 1 token"),
    "prefill": ("qwen", 8192, "Qwen3-30B-A3B-shaped compressed MoE layer, prefill of 8192 tokens"),
    "high_e": ("high_e", 4096, "E=256 (32 clusters of 8, rank 64), H=2560, I=1536, 4096 tokens"),
    "tree": ("tree", 2048, "BTExperts depth-2 tree (8 roots, 32 rank-192 subs, 96 rank-64 leaves), 2048 tokens"),
    "binary_decode64": ("binary", 64, "BTExperts Fig. 2 binary trees with -1/+1 edges (16 roots, "
                        "rank-128/64 internal corrections, 128 rank-64 leaf experts), decode batch of 64 tokens"),
    "binary": ("binary", 2048, "BTExperts Fig. 2 binary trees with -1/+1 edges (16 roots, "
               "rank-128/64 internal corrections, 128 rank-64 leaf experts), 2048 tokens"),
    "single_base_decode64": ("single_base", 64, "single shared base with 128 rank-128 experts, "
                             "H=2048, I=768, top-8, decode batch of 64 tokens"),
    "single_base": ("single_base", 2048, "single shared base with 128 rank-128 experts, "
                    "H=2048, I=768, top-8, 2048 tokens"),
}


# standalone kernels of the compression pipeline (timed on their own)
OFFLINE = {
    "coact": "router profiling statistics: co-activation counts of 8192-token batches of the "
             "Qwen3-30B-A3B-shaped layer's top-8 routing (E=128)",
    "align": "neuron alignment of one member to its dominant at the Qwen3-30B-A3B expert shape "
             "(H=2048, I=768): cost matrix, exact assignment, permutation",
    "compress": "compression of one member at the Qwen3-30B-A3B expert shape (H=2048, I=768): "
                "rank-128 randomized SVD (oversampling 8, 2 power iterations) of the gate, up "
                "and down residuals with the symmetric split",
}


def make_layer(kind):
    import synth
    return {"qwen": synth.qwen_decode_layer, "high_e": synth.high_e_layer,
            "tree": synth.btexperts_tree_layer, "binary": synth.btexperts_binary_layer,
            "single_base": synth.d2moe_base_layer}[kind]()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# ----------------------------------------------------------------------------
# clocks sampler (nvidia-smi during the timed region)
# ----------------------------------------------------------------------------
class Clocks:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,"
             "utilization.gpu")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None
        self.windows = []

    def start(self):
        if not shutil.which("nvidia-smi"):
            return
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        self.f = open(self.path, "w")
        self.proc = subprocess.Popen(
            ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.QUERY}",
             "--format=csv,noheader,nounits", "-lms", "50"], stdout=self.f,
            stderr=subprocess.DEVNULL)

    def mark(self, t0, t1):
        self.windows.append((t0, t1))

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                util = float(parts[9])
                rows.append((float(parts[1]), float(parts[2]), parts[4:9], util))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        names = ["active", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        loaded = [r for r in rows if r[3] >= 50] or rows
        reasons = set()
        for _, _, flags, _ in loaded:
            for n, v in zip(names[1:], flags[1:]):
                if v.strip().lower() in ("active", "1", "yes"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(r[0] for r in loaded),
                "sm_max_mhz": max(r[1] for r in rows), "reasons": sorted(reasons),
                "samples": len(rows), "samples_under_load": len(loaded),
                "window": "warm-up + timed loops (50 ms sampling, utilization >= 50%)"}


# ----------------------------------------------------------------------------
# algorithmic bytes per kernel launch, from the realised routing
# ----------------------------------------------------------------------------
def routing_stats(src, node_off, T, k):
    cnt = np.diff(node_off.astype(np.int64))
    anchor = np.asarray(src.node_parent) < 0
    rank = np.asarray(src.node_rank, np.int64)
    return dict(cnt=cnt, anchor=anchor, rank=rank, T=T, k=k,
                touched_anchor=int(np.sum((cnt > 0) & anchor)),
                touched_corr=int(np.sum((cnt > 0) & ~anchor)),
                R_anchor=int(cnt[anchor].sum()), R_corr=int(cnt[~anchor].sum()),
                corr_r_touched=int(rank[(cnt > 0) & ~anchor].sum()),
                corr_r_rows=int((rank * cnt)[~anchor].sum()))


def kernel_bytes(name, st, src, esz):
    """Bytes a kernel must move per launch (its inputs read once, outputs written
    once), for the kernels whose traffic is dominated by weight streaming."""
    H, I, E = src.d_model, src.d_ff, src.n_experts
    Ra, Rc, ta = st["R_anchor"], st["R_corr"], st["touched_anchor"]
    rt, rr = st["corr_r_touched"], st["corr_r_rows"]
    T, k = st["T"], st["k"]
    Ra_c = Ra + Rc
    table = {
        "router": E * H * esz + T * H * esz + T * E * 4,
        "generic_up_anchor": ta * 2 * I * H * esz + Ra * H * esz + Ra * 2 * I * 4,
        "generic_up_V": rt * 2 * H * esz + Rc * H * esz + rr * 2 * 4,
        "generic_up_U": rt * 2 * I * esz + rr * 2 * 4 + Rc * 2 * I * 4,
        "generic_dn_anchor": ta * H * I * esz + Ra * I * 4 + Ra * H * 4,
        "generic_dn_V": rt * I * esz + Rc * I * 4 + rr * 4,
        "generic_dn_U": rt * H * esz + rr * 4 + Rc * H * 4,
        # streaming kernels: weights once, activations in, results out (bf16)
        "stream_up_anchor_V": (ta * 2 * I * H + rt * 2 * H) * esz + Ra_c * H * esz
                              + Ra * 2 * I * 2 + rr * 2 * 2,
        "stream_up_U": rt * 2 * I * esz + rr * 2 * 2 + Rc * 2 * I * 2,
        "stream_dn_anchor_V": (ta * H * I + rt * I) * esz + Ra_c * I * 2 + Ra * H * 2 + rr * 2,
        "stream_dn_U": rt * H * esz + rr * 2 + Rc * H * 2,
    }
    # the fused streaming launches: {V, anchor gate/up, U} and {Vd, anchor down, Ud}
    table["stream_up"] = table["stream_up_anchor_V"] + table["stream_up_U"]
    table["stream_dn"] = table["stream_dn_anchor_V"] + table["stream_dn_U"]
    return table.get(name)


def fp32_alu_peak_tflops(peaks):
    """fp32 FMA peak of the GB300: 152 SMs x 128 FP32 lanes x 2 FLOP x the
    maximum SM clock (MEASURED_PEAKS sm_max_mhz, else 2070 MHz)."""
    mhz = float(peaks.get("sm_max_mhz", 2070.0))
    return 152 * 128 * 2 * mhz * 1e6 / 1e12


def kernel_alu_flops(name, st, src):
    """fp32 multiply-add FLOPs of the CUDA-core kernels: the router's logits."""
    if name == "router":
        return 2 * st["T"] * src.n_experts * src.d_model
    return None


def kernel_flops(name, st, src):
    """Dense multiply-add FLOPs per launch of a tensor-core kernel: 2 x (rows of
    each node's bucket) x (its output columns) x (its K), over real rows only."""
    H, I = src.d_model, src.d_ff
    Ra, rr = st["R_anchor"], st["corr_r_rows"]
    table = {
        "tc_up_anchor": 2 * Ra * 2 * I * H,
        # screened routing: the approximate logits of every (token, expert)
        "router_screen": 2 * st["T"] * src.n_experts * H,
        "tc_up_V": 2 * rr * 2 * H,
        "tc_up_U": 2 * rr * 2 * I,
        # the fused correction + SwiGLU kernel of flat layers: the members' P U^T
        # products (the work tc_up_U does on the unfused path)
        "ct_swiglu": 2 * rr * 2 * I,
        "tc_dn_anchor": 2 * Ra * H * I,
        # flat layers: the members' Q Ud^T join the anchor's down tile along K
        "tc_dn_anchor_U": 2 * Ra * H * I + 2 * rr * H,
        "tc_dn_V": 2 * rr * I,
        "tc_dn_U": 2 * rr * H,
    }
    return table.get(name)


def step_bytes(st, src, esz):
    from paper_2608_07814_gb300 import cost
    c = cost.step_counts(src.d_model, src.d_ff, src.n_experts, src.node_parent, src.node_rank,
                         st["cnt"], st["T"], esz, esz)
    return c


def traffic_for(kernel, workload):
    """dram bytes per launch from the committed ncu summary, if it was taken on
    this workload and the kernel's source is unchanged since; else None."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    d = json.load(open(p)).get(kernel)
    if not d or d.get("workload") != workload:
        return None
    src = os.path.join(ROOT, d["source"])
    if not os.path.exists(src):
        return None
    if hashlib.sha256(open(src, "rb").read()).hexdigest() != d["sha256"]:
        return None
    return d["bytes_per_launch"]


# ----------------------------------------------------------------------------
# ranks: one replica per GPU on its own token batches (weak scaling)
# ----------------------------------------------------------------------------
def max_over_ranks(values, world, device=None):
    """Element-wise max of per-rank timings; every rank calls it and gets the max."""
    if world <= 1:
        return [float(v) for v in values]
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return [float(v) for v in t]


def whole_job_rate(units_per_rank_step, steps, world, ms):
    """Units processed by all ranks per second, over the slowest rank's time."""
    return units_per_rank_step * steps * world / (ms * 1e-3)


def batch_seed(rank, b):
    """Seed of batch b on a rank: every rank draws its own tokens."""
    return 1000 * rank + b


# ----------------------------------------------------------------------------
# the CUDA arm
# ----------------------------------------------------------------------------
def workload_config(src, T, desc):
    """The workload's `config` (identical in both arms)."""
    return {"workload": desc, "d_model": src.d_model, "d_ff": src.d_ff,
            "n_experts": src.n_experts, "top_k": src.top_k, "n_nodes": src.n_nodes,
            "tokens_per_step": T, "layer_bytes": src.weight_bytes(),
            "l2": "inputs larger than L2 (GPU arm: rotating device copies of the layer for "
                  "decode batches, 8 token batches; the reference arm runs on the host cores)"}


def time_steps(layers, xs, ys, k, steps, warmup, world, clocks, graph=True):
    """Step time and per-kernel device times of `steps` forwards.

    The step time comes from one CUDA graph of the forwards without
    instrumentation (dependent launch on); the kernel durations from a second
    graph of the same forwards with the library's CUDA events around every
    launch.  Barrier + synchronize on both sides of the timed region; the max
    over ranks is taken by the caller."""
    import torch
    n_copies, n_batches = len(layers), len(xs)
    stream = torch.cuda.current_stream()

    def run(n):
        for i in range(n):
            layers[i % n_copies].moe_forward(xs[i % n_batches], k, ys[i % n_batches])

    for i in range(warmup):
        layers[i % n_copies].moe_forward(xs[i % n_batches], k, ys[i % n_batches])
    torch.cuda.synchronize()
    # one profiled pass fills each layer's event pool, so that the instrumented
    # capture below creates no events
    for L in layers:
        L.read_profile()
        L.set_profiling(True)
    run(steps)
    torch.cuda.synchronize()
    for L in layers:
        L.read_profile(cap=1 << 20)
    g = gp = None
    if graph:
        gp = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gp):
            run(steps)
    for L in layers:
        L.set_profiling(False)
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            run(steps)
        g.replay()  # untimed replay: first-launch costs of the graph
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0 = time.time()
    ev0.record(stream)
    if g is not None:
        g.replay()
    else:
        run(steps)
    ev1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clocks.mark(t0, time.time())
    ms = ev0.elapsed_time(ev1)
    t1 = time.time()
    if gp is not None:
        gp.replay()
    else:
        for L in layers:
            L.set_profiling(True)
        run(steps)
        for L in layers:
            L.set_profiling(False)
    torch.cuda.synchronize()
    clocks.mark(t1, time.time())
    per_copy = [L.read_profile(cap=1 << 20) for L in layers]
    del g, gp
    return ms, per_copy


def kernel_tables(per_copy, steps, n_copies, stats, src):
    """Per-kernel totals, launch counts and algorithmic bytes / FLOPs of the
    timed launches (records are in launch order per layer copy)."""
    esz = 2 if src.dtype == "bf16" else 4
    totals, counts, kbytes, kflops, kalu = {}, {}, {}, {}, {}
    launches = 0
    for c, recs in enumerate(per_copy):
        steps_of_copy = [i for i in range(steps) if i % n_copies == c]
        per_step = len(recs) // max(1, len(steps_of_copy))
        for j, (name, kms) in enumerate(recs):
            totals[name] = totals.get(name, 0.0) + kms
            counts[name] = counts.get(name, 0) + 1
            if name != "bucket_clear":
                launches += 1
            st = stats[(steps_of_copy[j // per_step] if per_step else 0) % len(stats)]
            for table, f in ((kbytes, kernel_bytes(name, st, src, esz)),
                             (kflops, kernel_flops(name, st, src)),
                             (kalu, kernel_alu_flops(name, st, src))):
                if f is not None:
                    table[name] = table.get(name, 0.0) + f
    return totals, counts, kbytes, kflops, kalu, launches


def roofline_summary(src, T, ms, steps, stats, tabs, peaks, peak_kind, workload):
    """Dominant kernel's roofline, per-kernel fractions and the step roofline."""
    totals, counts, kbytes, kflops, kalu, launches = tabs
    esz = 2 if src.dtype == "bf16" else 4
    hbm = float(peaks["hbm_gbs"])
    tf, tfs = float(peaks["bf16_tflops"]), float(peaks["bf16_tflops_sustained"])
    alu = fp32_alu_peak_tflops(peaks)
    dom = max(totals, key=totals.get)
    avg_ms = totals[dom] / counts[dom]
    roof = None
    if dom in kalu and src.dtype == "bf16" and T > 256:
        # the large-batch router: fp32 FMAs on the CUDA cores
        fl = kalu[dom] / counts[dom]
        ach = fl / (avg_ms * 1e-3) / 1e12
        roof = {"kernel": dom, "bound": "alu", "achieved": round(ach, 2), "peak": round(alu, 1),
                "unit": "TFLOP/s", "frac": round(ach / alu, 4), "traffic": traffic_for(dom, workload),
                "algorithmic_flops_per_launch": round(fl), "avg_launch_us": round(avg_ms * 1e3, 2),
                "peak_source": "derived fp32 FMA peak (152 SMs x 128 lanes x 2 x max SM clock)"}
    elif dom in kbytes:
        b = kbytes[dom] / counts[dom]
        ach = b / (avg_ms * 1e-3) / 1e9
        roof = {"kernel": dom, "bound": "hbm", "achieved": round(ach, 1), "peak": hbm,
                "unit": "GB/s", "frac": round(ach / hbm, 4), "traffic": traffic_for(dom, workload),
                "algorithmic_bytes_per_launch": round(b), "avg_launch_us": round(avg_ms * 1e3, 2),
                "peak_source": f"{peak_kind} hbm_gbs"}
    elif dom in kflops:
        fl = kflops[dom] / counts[dom]
        ach = fl / (avg_ms * 1e-3) / 1e12
        roof = {"kernel": dom, "bound": "tensor", "achieved": round(ach, 1), "peak": tf,
                "unit": "TFLOP/s", "frac": round(ach / tf, 4), "traffic": traffic_for(dom, workload),
                "algorithmic_flops_per_launch": round(fl), "avg_launch_us": round(avg_ms * 1e3, 2),
                "peak_source": f"{peak_kind} bf16_tflops (burst)"}

    def kernel_frac(n):
        t = totals[n] / counts[n] * 1e-3
        if n in kflops:
            return {"frac_bf16": round(kflops[n] / counts[n] / t / 1e12 / tf, 4)}
        if n in kalu and src.dtype == "bf16" and T > 256:
            return {"frac_alu": round(kalu[n] / counts[n] / t / 1e12 / alu, 4)}
        if n in kbytes:
            return {"frac_hbm": round(kbytes[n] / counts[n] / t / 1e9 / hbm, 4)}
        return {}

    cs = [step_bytes(stats[i % len(stats)], src, esz) for i in range(steps)]
    sec = ms * 1e-3
    step_b = sum(c["bytes"] for c in cs)
    step_f = sum(c["flops"] for c in cs)
    step = {"algorithmic_bytes_per_step": round(step_b / steps),
            "algorithmic_flops_per_step": round(step_f / steps),
            "achieved_gbs": round(step_b / sec / 1e9, 1),
            "achieved_tflops": round(step_f / sec / 1e12, 1)}
    if T <= 256:
        step.update({"bound": "hbm", "frac": round(step_b / sec / 1e9 / hbm, 4),
                     "frac_nominal_8tbs": round(step_b / sec / 1e9 / 8000.0, 4),
                     "peak": f"{peak_kind} hbm_gbs {hbm}"})
    else:
        step.update({"bound": "tensor", "frac": round(step_f / sec / 1e12 / tf, 4),
                     "frac_sustained": round(step_f / sec / 1e12 / tfs, 4),
                     "peak": f"{peak_kind} bf16_tflops {tf} (burst), {tfs} (sustained)"})
    amort = float(np.mean([st["T"] * st["k"] / max(1, st["R_anchor"]) for st in stats]))
    kernels = {n: {"launches": counts[n], "avg_us": round(totals[n] / counts[n] * 1e3, 2),
                   "share": round(totals[n] / sum(totals.values()), 4), **kernel_frac(n)}
               for n in totals}
    return roof, kernels, step, round(amort, 3), launches


def setup_workload(src, T, n_copies, rank, dev, layers=None):
    """Installed layer copies, 8 token batches on the device and their hosts."""
    import synth
    from paper_2608_07814_gb300 import lx
    if layers is None:
        layers = [lx.Layer(src) for _ in range(n_copies)]
    for L in layers:
        L.reserve(T, src.top_k)
    xs_host = [synth.tokens(src, T, seed=batch_seed(rank, b)) for b in range(8)]
    xs = [lx.host_to_torch(x, src.dtype).to(dev) for x in xs_host]
    ys = [torch_empty_like(x) for x in xs]
    return layers, xs_host, xs, ys


def torch_empty_like(x):
    import torch
    return torch.empty_like(x)


def batch_stats(src, layer, xs, ys, T):
    """Routing statistics of every batch (outside the timed region)."""
    import torch
    stats = []
    for b in range(len(xs)):
        layer.moe_forward(xs[b], src.top_k, ys[b])
        bk = layer.get_buckets()
        torch.cuda.synchronize()
        stats.append(routing_stats(src, bk["node_off"].cpu().numpy(), T, src.top_k))
    return stats


def run_lx(args, rank, world, local_rank):
    import torch
    from paper_2608_07814_gb300 import lx

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    kind, T, desc = WORKLOADS[args.workload]
    src = make_layer(kind)
    k = src.top_k
    n_copies = args.copies if args.copies else (4 if T <= 512 else 1)
    layers, xs_host, xs, ys = setup_workload(src, T, n_copies, rank, dev)
    stats = batch_stats(src, layers[0], xs, ys, T)
    peaks, peak_kind = load_peaks()

    clocks = Clocks(local_rank)
    clocks.start()
    ms, per_copy = time_steps(layers, xs, ys, k, args.steps, args.warmup, world, clocks,
                              graph=not args.no_graph)

    # e2e: host buffers, copies inside the timed region, a read of every result
    stream = torch.cuda.current_stream()
    xh = [lx.host_to_torch(x, src.dtype).pin_memory() for x in xs_host]
    yh = [torch.empty_like(x).pin_memory() for x in xh]
    xd, yd = torch.empty_like(xs[0]), torch.empty_like(xs[0])
    k_e2e = max(3, min(args.steps, 200))
    for i in range(3):
        xd.copy_(xh[i % len(xh)], non_blocking=True)
        layers[i % n_copies].moe_forward(xd, k, yd)
        yh[i % len(xh)].copy_(yd, non_blocking=True)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_e2e0 = time.time()
    e0.record(stream)
    for i in range(k_e2e):
        xd.copy_(xh[i % len(xh)], non_blocking=True)
        layers[i % n_copies].moe_forward(xd, k, yd)
        yh[i % len(xh)].copy_(yd, non_blocking=True)
        stream.synchronize()
    e1.record(stream)
    torch.cuda.synchronize()
    clocks.mark(t_e2e0, time.time())
    ms_e2e = e0.elapsed_time(e1)

    # the other workloads of the metric, at one GPU, in the same run
    per_config = None
    if world == 1 and not args.no_per_config and args.workload == "decode64":
        per_config = run_per_config(args, rank, dev, src, layers, clocks, peaks, peak_kind)
    clk = clocks.stop()

    ms, ms_e2e = max_over_ranks([ms, ms_e2e], world, dev)
    if rank != 0:
        return None
    tabs = kernel_tables(per_copy, args.steps, n_copies, stats, src)
    roof, kernels, step, amort, launches = roofline_summary(
        src, T, ms, args.steps, stats, tabs, peaks, peak_kind, args.workload)
    config = workload_config(src, T, desc)
    config.update({"layer_copies": n_copies, "parallelism": f"replica per GPU x{world}",
                   "timing": ("one CUDA graph of the K forwards (kernel durations from a "
                              "second, event-instrumented graph of the same forwards)")
                             if not args.no_graph else "K forwards launched one by one"})
    line = {
        "metric": METRIC, "value": round(whole_job_rate(T, args.steps, world, ms), 1),
        "unit": "tokens/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms / args.steps, 5), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if src.dtype == "bf16" else "f32",
        "data": "synthetic (seeded Gaussian weights and tokens, Zipf-skewed cluster-correlated router)",
        "config": config,
        "roofline": roof,
        "kernels": kernels,
        "step_roofline": step,
        "amortisation": amort,
        "e2e": {"value": round(whole_job_rate(T, k_e2e, world, ms_e2e), 1), "unit": "tokens/s",
                "steps": k_e2e, "h2d_bytes_per_step": int(xs[0].numel() * xs[0].element_size()),
                "d2h_bytes_per_step": int(ys[0].numel() * ys[0].element_size())},
        "gpu_launches": launches,
        "clocks": clk,
        "impl": "lx",
    }
    if per_config is not None:
        line["per_config"] = per_config
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(src, xs_host, T, args.cpu_seconds, n_tokens=8)
    return line


# the other workloads reported beside the headline (name, layer kind, T, steps)
PER_CONFIG = [("decode1", 20), ("decode8", 20), ("decode32", 20), ("prefill", 10),
              ("high_e", 10), ("tree", 10)]


def run_per_config(args, rank, dev, qwen_src, qwen_layers, clocks, peaks, peak_kind):
    """Each of the metric's other workloads: tokens/s, the step roofline, the
    dominant kernel's roofline, the amortisation and a bounded oracle baseline.
    The Qwen-shaped layer copies of the headline are reused."""
    import torch
    out = {}
    made = {"qwen": qwen_src}
    for name, steps in PER_CONFIG:
        kind, T, desc = WORKLOADS[name]
        t_start = time.time()
        if kind not in made:
            made[kind] = make_layer(kind)
        src = made[kind]
        reuse = qwen_layers if kind == "qwen" else None
        layers, xs_host, xs, ys = setup_workload(src, T, len(reuse) if reuse else 1, rank, dev,
                                                 layers=reuse)
        stats = batch_stats(src, layers[0], xs, ys, T)
        ms, per_copy = time_steps(layers, xs, ys, src.top_k, steps, 3, 1, clocks,
                                  graph=not args.no_graph)
        tabs = kernel_tables(per_copy, steps, len(layers), stats, src)
        roof, kernels, step, amort, launches = roofline_summary(
            src, T, ms, steps, stats, tabs, peaks, peak_kind, name)
        entry = {"workload": desc, "tokens_per_step": T, "steps": steps, "warmup": 3,
                 "value": round(whole_job_rate(T, steps, 1, ms), 1), "unit": "tokens/s",
                 "ms_per_step": round(ms / steps, 5), "layer_copies": len(layers),
                 "step_roofline": step, "roofline": roof, "amortisation": amort,
                 "gpu_launches": launches,
                 "kernels": {n: v for n, v in kernels.items() if v["share"] >= 0.02}}
        if not args.no_cpu_baseline:
            entry["cpu_baseline"] = cpu_baseline(src, xs_host, T, args.cfg_cpu_seconds,
                                                 n_tokens=8 if T <= 8 else 4, n_batches=2)
        entry["wall_s"] = round(time.time() - t_start, 1)
        out[name] = entry
        if reuse is None:
            for L in layers:
                L.free()
        del xs, ys
        torch.cuda.empty_cache()
    return out


def _event_ms(fn, steps, warmup, world=1):
    """Average ms per call of fn() over `steps` calls on the current stream
    (CUDA events, synchronised on both sides), after `warmup` calls; with
    several ranks a barrier precedes the timed calls and the slowest rank's
    time is returned."""
    import torch
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(steps):
        fn()
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / steps
    if world > 1:
        ms = max_over_ranks([ms], world, torch.device("cuda", torch.cuda.current_device()))[0]
    return ms


def run_offline(args, rank, world, local_rank):
    import torch
    import synth
    import oracle
    from oracle import align as oalign, stats as ostats
    from paper_2608_07814_gb300 import lx

    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    line = {"n_gpus": world, "steps": args.steps, "warmup": args.warmup, "scaling": "weak",
            "vs_baseline": None, "data": "synthetic", "impl": "lx",
            "config": {"workload": OFFLINE[args.workload]}}
    if args.workload == "coact":
        src = make_layer("qwen")
        L = lx.Layer(src)
        T, k, E, nb = 8192, 8, src.n_experts, 16
        ids = []
        for b in range(nb):
            x = lx.host_to_torch(synth.tokens(src, T, seed=batch_seed(rank, b)), "bf16").to(dev)
            ids.append(L.route(x, k)[0])
        fire = torch.zeros(E, dtype=torch.int64, device=dev)
        coact = torch.zeros((E, E), dtype=torch.int64, device=dev)
        it = [0]

        def step():
            lx.coact_accumulate(ids[it[0] % nb], E, fire, coact)
            it[0] += 1
        ms = _event_ms(step, args.steps, args.warmup, world)
        byts = T * k * 4 + 2 * E * E * 8
        t_npmi = _event_ms(lambda: lx.coact_npmi(coact, T * nb), 20, 3)
        host_ids = [i.cpu().numpy() for i in ids[:2]]
        t0 = time.time()
        for h in host_ids:
            ostats.coact_counts(h[:1024], E)
        cpu = 2 * 1024 / (time.time() - t0)
        line.update({"metric": "router-statistics tokens/s (co-activation counts)",
                     "value": round(whole_job_rate(T, 1, world, ms), 1), "unit": "tokens/s",
                     "ms_per_step": round(ms, 5), "higher_is_better": True, "dtype": "int64",
                     "gpu_launches": args.steps,
                     "roofline": {"kernel": "k_coact_smem", "bound": "hbm",
                                  "achieved": round(byts / (ms * 1e-3) / 1e9, 1), "peak": hbm,
                                  "unit": "GB/s", "frac": round(byts / (ms * 1e-3) / 1e9 / hbm, 5),
                                  "traffic": None, "note": "latency-bound: 256 KB of ids per launch"},
                     "npmi_us": round(t_npmi * 1e3, 2),
                     "cpu_baseline": {"value": round(cpu, 1), "unit": "tokens/s", "cores": 1,
                                      "kind": "oracle", "sample": "2 x 1024 tokens"}})
        line["config"].update({"tokens_per_step": T, "n_experts": E, "top_k": k,
                               "l2": "16 rotating id batches (4 MB, L2-resident)"})
    elif args.workload == "compress":
        H, I, r, l, q = 2048, 768, 128, 136, 2
        rng = np.random.default_rng(rank)
        draw = lambda s: synth.to_storage(rng.standard_normal(s).astype(np.float32) * 0.02, "bf16")
        shapes = [(I, H), (I, H), (H, I)]
        dom = [draw(sh) for sh in shapes]
        mem = [draw(sh) for sh in shapes]
        oms = [rng.standard_normal((sh[1], l)).astype(np.float32) for sh in shapes]
        dd = [lx.host_to_torch(w, "bf16").to(dev) for w in dom]
        md = [lx.host_to_torch(w, "bf16").to(dev) for w in mem]
        od = [torch.from_numpy(o).to(dev) for o in oms]
        wsz = max(lx.compress_workspace_bytes(a, b, l, r) for a, b in shapes)
        ws = torch.empty(wsz, dtype=torch.uint8, device=dev)

        def step():
            for p in range(3):
                lx.compress_factor(dd[p], md[p], od[p], r, q, workspace=ws)
        ms_seq = _event_ms(step, max(3, args.steps // 4), args.warmup)
        # one member alone: its three projections concurrently on three streams
        wss1 = [torch.empty(wsz, dtype=torch.uint8, device=dev) for _ in range(3)]
        ms_one = _event_ms(lambda: lx.compress_member(dd, md, od, r, q, workspaces=wss1),
                           max(3, args.steps // 4), args.warmup)
        # a layer's members are independent: n_conc members (3 projections
        # each) in flight on their own streams, each with its own workspace
        n_conc = 8
        streams = [torch.cuda.Stream(device=dev) for _ in range(3 * n_conc)]
        wss = [torch.empty(wsz, dtype=torch.uint8, device=dev) for _ in streams]
        outs = [(torch.empty((a, r), dtype=torch.float32, device=dev),
                 torch.empty((b, r), dtype=torch.float32, device=dev),
                 torch.empty(r, dtype=torch.float32, device=dev))
                for _ in range(n_conc) for a, b in shapes]

        def step_conc():
            main = torch.cuda.current_stream()
            ev = torch.cuda.Event()
            ev.record(main)
            for j, st in enumerate(streams):
                st.wait_event(ev)
                p = j % 3
                lx.compress_factor(dd[p], md[p], od[p], r, q, workspace=wss[j], stream=st,
                                   out=outs[j])
            for st in streams:
                e = torch.cuda.Event()
                e.record(st)
                main.wait_event(e)
        ms = _event_ms(step_conc, args.steps, args.warmup, world) / n_conc
        # launches of one projection: the R products (split, transposes, MMA,
        # ordered sum), 2q single and 2 double CholeskyQR passes (Gram, Cholesky,
        # basis product each), then trmm, Jacobi, Ritz, finish, two factor
        # products and the sign rule
        launches_per_projection = ((1 + q) * 3 + (1 + q) * 5 + 3 * (2 * q + 4) + 7)
        big = sum((2 + 2 * q) * 2.0 * a * b * l for a, b in shapes)        # the R-sized products
        # CholeskyQR passes: q + 2 on each side (rows and cols), each a lower
        # Gram (n l^2) and a basis product (2 n l^2); then the two factor products
        small = sum(3.0 * l * l * (q + 2) * (a + b) + 2.0 * (a + b) * l * r for a, b in shapes)
        alu = fp32_alu_peak_tflops(peaks)
        ach = (big + small) / (ms * 1e-3) / 1e12
        t0 = time.time()
        for p in range(3):
            R = synth.from_storage(mem[p], "bf16") - synth.from_storage(dom[p], "bf16")
            from oracle import compress as ocomp
            ocomp.randomized_factors(R, r, oms[p].astype(np.float64), q)
        cpu_s = time.time() - t0
        line["sequential_ms_per_member"] = round(ms_seq, 3)
        line["one_member_ms"] = round(ms_one, 3)
        line.update({"metric": "members compressed/s (gate, up and down residuals, rank 128)",
                     "value": round(1e3 / ms * world, 3), "unit": "members/s",
                     "ms_per_step": round(ms, 4), "higher_is_better": True, "dtype": "f32",
                     "gpu_launches": args.steps * n_conc * 3 * launches_per_projection,
                     "roofline": {"kernel": "whole compression step", "bound": "alu",
                                  "achieved": round(ach, 2), "peak": round(alu, 1),
                                  "unit": "TFLOP/s", "frac": round(ach / alu, 4), "traffic": None,
                                  "algorithmic_flops_per_step": round(big + small),
                                  "peak_source": "fp32 FMA: 152 SMs x 128 lanes x 2 x sm_max_mhz"},
                     "cpu_baseline": {"value": round(1.0 / cpu_s, 4), "unit": "members/s",
                                      "cores": os.cpu_count(), "kind": "oracle",
                                      "sample": "one member (3 projections), float64 numpy"}})
        line["config"].update({"d_model": H, "d_ff": I, "rank": r, "oversampling": l - r,
                               "power_iters": q, "l2": "one member (L2-resident)",
                               "concurrency": f"{n_conc} members (x3 projections) on "
                                              f"{3 * n_conc} streams per step; value per member"})
    else:
        H, I = 2048, 768
        rng = np.random.default_rng(rank)
        draw = lambda s: synth.to_storage(rng.standard_normal(s).astype(np.float32) * 0.02, "bf16")
        dom = [draw((I, H)), draw((I, H)), draw((H, I))]
        mems = [[draw((I, H)), draw((I, H)), draw((H, I))] for _ in range(4)]
        dd = tuple(lx.host_to_torch(w, "bf16").to(dev) for w in dom)
        md = [tuple(lx.host_to_torch(w, "bf16").to(dev) for w in m) for m in mems]
        it = [0]

        def step():
            lx.align_cost(dd, md[it[0] % 4])
            it[0] += 1
        ms_loop = _event_ms(step, args.steps, args.warmup, world)
        # device throughput: four calls replayed from a CUDA graph (the host's
        # per-call launch work, which bounds the loop above, left out)
        timing = "CUDA graph of 4 calls (device time per call)"
        try:
            side = torch.cuda.Stream()
            side.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(side):
                for j in range(4):
                    lx.align_cost(dd, md[j])
            torch.cuda.current_stream().wait_stream(side)
            torch.cuda.synchronize()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph):
                kept = [lx.align_cost(dd, md[j]) for j in range(4)]
            ms = _event_ms(graph.replay, max(1, args.steps // 4), args.warmup, world) / 4
        except Exception as ex:  # capture not possible: the host loop's time
            ms, timing = ms_loop, f"host loop ({type(ex).__name__} in graph capture)"
        cost = lx.align_cost(dd, md[0]).cpu().numpy()
        t0 = time.time()
        P, _ = lx.lap_solve(cost)
        lap_s = time.time() - t0
        Pd = torch.from_numpy(P).to(dev)
        ms_perm = _event_ms(lambda: lx.permute_neurons(Pd, *md[1]), 20, 3)
        # a layer's members end to end: 16 members' costs on the GPU, one copy
        # of all costs to pinned host memory, the batched assignment on the host
        # cores, the permutations back and applied on the GPU
        nb = 16
        mb = [tuple(lx.host_to_torch(draw(sh), "bf16").to(dev) for sh in ((I, H), (I, H), (H, I)))
              for _ in range(nb)]
        costs_d = torch.empty((nb, I, I), dtype=torch.float32, device=dev)
        costs_h = torch.empty((nb, I, I), dtype=torch.float32).pin_memory()
        perms_h = torch.empty((nb, I), dtype=torch.int32).pin_memory()
        perms_d = torch.empty((nb, I), dtype=torch.int32, device=dev)
        outs = [tuple(torch.empty_like(w) for w in m) for m in mb]

        def layer_pass():
            for b in range(nb):
                costs_d[b].copy_(lx.align_cost(dd, mb[b]))
            costs_h.copy_(costs_d, non_blocking=True)
            torch.cuda.synchronize()
            Pb, _ = lx.lap_solve_batch(costs_h.numpy())
            perms_h.copy_(torch.from_numpy(Pb))
            perms_d.copy_(perms_h, non_blocking=True)
            for b in range(nb):
                lx.permute_neurons(perms_d[b], *mb[b], out=outs[b])
            torch.cuda.synchronize()
        layer_pass()
        t0 = time.time()
        for _ in range(3):
            layer_pass()
        e2e_s = (time.time() - t0) / 3
        flops = 2.0 * I * I * 3 * H + 2.0 * 2 * I * 3 * H
        tf = float(peaks["bf16_tflops"])       # bf16 experts take the tensor-core kernel
        ach = flops / (ms * 1e-3) / 1e12
        pbytes = 2 * 3 * I * H * 2 + I * 4
        t0 = time.time()
        oalign.assign(oalign.cost_matrix(tuple(synth.from_storage(w, "bf16") for w in dom),
                                         tuple(synth.from_storage(w, "bf16") for w in mems[0]),
                                         rows=np.arange(64)))
        cpu_rows = 64 / (time.time() - t0)
        line.update({"metric": "neuron-alignment cost matrices/s (one member vs its dominant)",
                     "value": round(1e3 / ms * world, 2), "unit": "matrices/s",
                     "ms_per_step": round(ms, 5), "higher_is_better": True, "dtype": "f32",
                     "gpu_launches": args.steps, "timing": timing,
                     "host_loop_ms_per_call": round(ms_loop, 5),
                     "roofline": {"kernel": "lx_align_cost (operand packing, tcgen05 split-K GEMM, "
                                            "ordered range sum)", "bound": "tensor",
                                  "achieved": round(ach, 2), "peak": tf, "unit": "TFLOP/s",
                                  "frac": round(ach / tf, 4), "traffic": None,
                                  "peak_source": f"{peak_kind} bf16_tflops (burst)"},
                     "lap_host_s": round(lap_s, 3),
                     "permute": {"us": round(ms_perm * 1e3, 2),
                                 "gbs": round(pbytes / (ms_perm * 1e-3) / 1e9, 1),
                                 "frac_hbm": round(pbytes / (ms_perm * 1e-3) / 1e9 / hbm, 4)},
                     "e2e": {"value": round(nb / e2e_s, 2),
                             "unit": "members aligned/s (16 members: GPU costs, batched host "
                                     f"assignment on {os.cpu_count()} cores, GPU permutations)",
                             "h2d_bytes_per_step": nb * I * 4, "d2h_bytes_per_step": nb * I * I * 4},
                     "one_member_s": round(ms * 1e-3 + lap_s + ms_perm * 1e-3, 4),
                     "cpu_baseline": {"value": round(cpu_rows / I, 5), "unit": "matrices/s",
                                      "cores": os.cpu_count(), "kind": "oracle",
                                      "sample": "64 of the 768 cost rows (float64 definition)"}})
        line["config"].update({"d_model": H, "d_ff": I, "l2": "4 rotating members (L2-resident)"})
    return line if rank == 0 else None


_RECON = {}   # id(layer) -> {expert: reconstructed float64 weights}


def cpu_baseline(src, xs_host, T, budget_s, n_tokens=8, n_batches=8):
    """The oracle, as it stands, on a bounded sample of the same workload:
    routing plus the standard MoE forward of the first `n_tokens` tokens of
    `n_batches` batches, from experts reconstructed beforehand (the
    reconstruction is timed separately, and shared by the workloads of one layer)."""
    import oracle
    n = min(T, n_tokens)
    samples = [x[:n] for x in xs_host[:n_batches]]
    t0 = time.time()
    ids = np.unique(np.concatenate([oracle.route(src, x)[0].ravel() for x in samples]))
    cache = _RECON.setdefault(id(src), {})
    missing = [int(e) for e in ids if int(e) not in cache]
    cache.update(oracle.reconstruct(src, missing) if missing else {})
    experts = {int(e): cache[int(e)] for e in ids}
    recon_s = time.time() - t0
    done, b, t0 = 0, 0, time.time()
    while True:
        oracle.moe_forward(src, samples[b % len(samples)], experts=experts)
        done += n
        b += 1
        if time.time() - t0 > budget_s or b >= 8 * len(samples):
            break
    el = time.time() - t0
    return {"value": round(done / el, 3), "unit": "tokens/s", "cores": os.cpu_count(),
            "kind": "oracle", "seconds": round(el, 2),
            "reconstruction_s": round(recon_s, 2),
            "sample": f"{b} batch(es) of the first {n} tokens of the workload's batches: "
                      "canonical-fp32 routing and the float64 standard MoE forward, timed; "
                      f"the float64 reconstruction of the {len(experts)} experts they select "
                      "is done beforehand (reconstruction_s: the part not already done for "
                      "an earlier workload of the same layer)"}


# ----------------------------------------------------------------------------
# the reference arm: the CPU oracle
# ----------------------------------------------------------------------------
def run_reference(args, rank, world):
    if rank != 0:
        return None
    import oracle
    import synth
    kind, T, desc = WORKLOADS[args.workload]
    src = make_layer(kind)
    n = min(T, args.ref_tokens)
    xs = [synth.tokens(src, T, seed=b)[:n] for b in range(4)]
    ids = np.concatenate([oracle.route(src, x)[0].ravel() for x in xs])
    t0 = time.time()
    experts = oracle.reconstruct(src, ids)
    recon_s = time.time() - t0
    for i in range(args.warmup):
        oracle.moe_forward(src, xs[i % 4], experts=experts)
    t0 = time.time()
    for i in range(args.steps):
        oracle.moe_forward(src, xs[i % 4], experts=experts)
    el = time.time() - t0
    v = n * args.steps / el
    sample = (f"{n} of the {T} tokens of each step's batch: canonical-fp32 routing and the "
              f"float64 standard MoE forward, from the {len(experts)} experts the samples "
              f"select, reconstructed beforehand in {recon_s:.1f} s")
    return {"metric": METRIC, "value": round(v, 3), "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(el / args.steps * 1e3, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(src, T, desc),
            "impl": "reference",
            "cpu_baseline": {"value": round(v, 3), "unit": "tokens/s", "cores": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(v, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default="decode64", choices=sorted(WORKLOADS) + sorted(OFFLINE))
    ap.add_argument("--impl", default="lx", choices=["lx", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--cfg-cpu-seconds", type=float, default=3.0,
                    help="oracle seconds per workload of per_config")
    ap.add_argument("--no-per-config", action="store_true",
                    help="report the headline workload only")
    ap.add_argument("--ref-tokens", type=int, default=8)
    ap.add_argument("--no-graph", action="store_true",
                    help="launch the timed steps one by one instead of as one CUDA graph")
    ap.add_argument("--copies", type=int, default=None,
                    help="device copies of the layer rotated between steps (default 4 for decode)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1 and args.impl == "lx":
        import torch
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl")
    if args.workload in OFFLINE:
        line = run_offline(args, rank, world, local_rank) if args.impl == "lx" else \
            {"impl": "reference", "unavailable": "the reference arm times the forward only"}
    elif args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        line = run_lx(args, rank, world, local_rank)
    if line is not None:
        print(json.dumps(line), flush=True)
    if world > 1 and args.impl == "lx":
        import torch
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
