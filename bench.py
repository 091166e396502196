#!/usr/bin/env python3
"""Benchmark of the block-quantised matmul hot path on GB300.

Default workload (one "step"): the action-token decode of a Gemma-style 2B backbone
at M=1 -- 18 layers x (q, k, v, o, gate, up, down) linears -- once with Q8_0 and once
with Q4_0 weights, each chain replayed as a CUDA graph of emb_qlayer_seq (fused
q/k/v and gate/up launches, programmatic dependent launch between launches). This is
the paper's latency-first batch-1 execution (Section 3.1 challenge 2, Section 3.2
principle 2) on its 8-bit / 4-bit configurations (Section 4, Table 3).

Metric: algorithmic HBM bytes (packed weights read once + bf16 X + fp32 Y) per second,
i.e. GB/s against the HBM roofline; for --workload with M >= 50 it is TFLOP/s against
the bf16 tensor-core roofline.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload NAME]

N > 1: one process per GPU (torchrun); every rank runs its own replica of the step
(weak scaling, no collective on the data path); time = max over ranks.
--impl reference: the CPU oracle timed on the host cores on a bounded sample of the
same workload (this build has no other reference implementation).
"""
from __future__ import annotations

import argparse
import concurrent.futures as cf
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads as wl  # noqa: E402

FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS = 1900.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0
BAD_CLOCK_REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")


# ------------------------------------------------------------------ helpers

def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def init_dist(world: int, backend: str):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)
    return dist if world > 1 else None


def barrier(dist):
    if dist is not None:
        dist.barrier()


def max_over_ranks(value: float, dist, device=None) -> float:
    """Largest value across ranks (the slowest rank sets the whole-job time)."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, dist, device=None) -> float:
    if dist is None:
        return value
    import torch
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            p = json.load(fh)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": FALLBACK_HBM_GBS, "bf16_tflops": FALLBACK_BF16_TFLOPS,
                "bf16_tflops_sustained": FALLBACK_BF16_TFLOPS_SUSTAINED, "source": "fallback"}


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.gpu), "-lms", "200"], stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.flush()
        self.out.seek(0)
        rows = [ln.strip().split(", ") for ln in self.out.read().splitlines() if ln.strip()]
        self.out.close()
        os.unlink(self.out.name)
        return summarize_clocks(rows)


def summarize_clocks(rows):
    names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
    sm, mx, reasons, power = [], None, set(), []
    for r in rows:
        if len(r) < 9:
            continue
        try:
            sm.append(float(r[1]))
            mx = float(r[2])
            power.append(float(r[3]))
        except ValueError:
            continue
        for name, val in zip(names, r[5:9]):
            if val.strip().lower() == "active":
                reasons.add(name)
    if not sm:
        return {"sm_mhz": None, "sm_max_mhz": mx, "reasons": ["no samples"]}
    # samples under load: the timed region keeps the GPU busy; drop idle-clock samples
    loaded = [v for v in sm if v >= 0.5 * max(sm)] or sm
    return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": mx, "reasons": sorted(reasons),
            "samples": len(sm), "power_w_max": max(power) if power else None}


# ------------------------------------------------------------------ workloads

WORKLOADS = {
    "gemma2b_decode": lambda: [wl.gemma2b_decode(wl.Q8_0), wl.gemma2b_decode(wl.Q4_0)],
    # the 2048 x 2048 Q8_0 linear, 100 calls per step on distinct weight copies
    "single_linear": lambda: [wl.single_linear_copies()],
    "action_expert": lambda: [wl.action_expert_denoise()],
    # the flow-matching loop recorded as one chain (10 steps x 18 layers, fused epilogues)
    "action_expert_fused": lambda: [wl.action_expert_fused()],
    "gemma2b_prefill": lambda: [wl.gemma2b_prefill(wl.Q8_0), wl.gemma2b_prefill(wl.Q4_0)],
    # the 6-bit configuration (Table 3), decode and prefill
    "gemma2b_decode_q6": lambda: [wl.gemma2b_decode(wl.Q6_0)],
    "gemma2b_prefill_q6": lambda: [wl.gemma2b_prefill(wl.Q6_0)],
    "vit": lambda: [wl.vit_tower(wl.Q8_0), wl.vit_tower(wl.Q4_0)],
    "llama7b_decode": lambda: [wl.llama7b(1)],
    "llama7b_prefill": lambda: [wl.llama7b(280)],
}


def build_chain(w: wl.Workload, device):
    """Device weights (generated, quantised once per distinct linear, fp32 freed),
    activations and outputs. All activations of the chain live in one device arena and all
    outputs in another (views at 256-byte offsets), so a step moves them with one copy each
    way. Outputs follow each layer's epilogue: fp32, bf16, gated bf16 (N/2 columns), or the
    one fp32 residual stream that every residual-add layer accumulates into; a layer with
    x_from > 0 reads the output of the group that many groups earlier. Layers of the same
    name (one layer of a loop run several times in the chain) share their weights, their
    activation buffer and their output buffer, as the loop itself would."""
    import torch
    import paper_2607_02501_gb300 as emb

    def r256(n):
        return (n + 255) // 256 * 256

    def out_shape(lin):
        if lin.epilogue in (wl.EPI_GEGLU, wl.EPI_SWIGLU):
            return (w.M, lin.N // 2), torch.bfloat16
        return (w.M, lin.N), (torch.bfloat16 if lin.epilogue == wl.EPI_BF16 else torch.float32)

    resid_n = {lin.N for g in w.groups for lin in g if lin.epilogue == wl.EPI_ADD}
    assert len(resid_n) <= 1, "one residual stream per workload"
    x_keys = {(g[0].name, g[0].K) for g in w.groups if g[0].x_from == 0}
    y_keys = {(lin.name, lin.N) for g in w.groups for lin in g if lin.epilogue != wl.EPI_ADD}
    x_bytes = sum(r256(w.M * K * 2) for _, K in x_keys)
    y_bytes = sum(r256(w.M * n * 4) for _, n in y_keys) + sum(r256(w.M * n * 4) for n in resid_n)
    x_arena = torch.empty(x_bytes, dtype=torch.uint8, device=device)
    y_arena = torch.zeros(y_bytes, dtype=torch.uint8, device=device)
    resid = None
    yo = 0
    if resid_n:
        n = resid_n.pop()
        resid = y_arena[:w.M * n * 4].view(torch.float32).view(w.M, n)
        yo = r256(w.M * n * 4)
    specs, xs, ys, outs, x_bufs, y_bufs = [], [], [], [], {}, {}
    images = build_chain.images
    xo = 0
    for group in w.groups:
        K = group[0].K
        if group[0].x_from > 0:
            X = outs[len(outs) - group[0].x_from]
            assert X.dtype == torch.bfloat16 and X.shape == (w.M, K)
        elif (group[0].name, K) in x_bufs:
            X = x_bufs[(group[0].name, K)]
        else:
            X = x_arena[xo:xo + w.M * K * 2].view(torch.bfloat16).view(w.M, K)
            X.copy_(wl.activation_torch(w.M, K, wl.activation_seed(group[0]), device=device))
            xo += r256(w.M * K * 2)
            xs.append(X)
            x_bufs[(group[0].name, K)] = X
        group_out = None
        for lin in group:
            key = (w.fmt, lin.name, lin.N, lin.K, lin.seed, lin.outliers)
            if key not in images:
                W = wl.weight_torch(lin, device=device)
                images[key] = emb.quantize(w.fmt, W)
                del W
            if lin.epilogue == wl.EPI_ADD:
                Y = resid
            elif (lin.name, lin.N) in y_bufs:
                Y = y_bufs[(lin.name, lin.N)]
            else:
                shape, dt = out_shape(lin)
                nbytes = shape[0] * shape[1] * (2 if dt == torch.bfloat16 else 4)
                Y = y_arena[yo:yo + nbytes].view(dt).view(*shape)
                yo += r256(nbytes)
                ys.append(Y)
                y_bufs[(lin.name, lin.N)] = Y
            group_out = Y
            specs.append((w.fmt, images[key], lin.N, lin.K, X, Y, lin.epilogue))
        outs.append(group_out)
    if resid is not None:
        ys.insert(0, resid)
    torch.cuda.synchronize()
    build_chain.arenas[id(specs)] = (x_arena, y_arena)
    return specs, xs, ys


build_chain.arenas = {}   # id(specs) -> (activation arena, output arena)
build_chain.images = {}   # (fmt, name, N, K, seed, outliers) -> packed device image, shared by chains


def count_launches(specs) -> int:
    """Kernel launches of one emb_qlayer_seq over these layers (fused groups)."""
    n, prev = 0, None
    size = 0
    for sp in specs:
        key = (sp[0], sp[3], sp[4].data_ptr())
        if key == prev and size < 4:
            size += 1
            continue
        n += 1
        prev, size = key, 1
    return n


def capture_graph(specs, M):
    """The chain recorded by the library (emb_chain_create) after one eager call (module
    load); returns an object whose replay() launches the whole chain with one call."""
    import torch
    import paper_2607_02501_gb300 as emb
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    rec = emb.RecordedChain(specs, M)
    rec.replay = rec.launch
    return rec, rec.layers


# ------------------------------------------------------------------ CPU oracle timing

def oracle_sample_images(w: wl.Workload, layers: int):
    """Host-side packed images (made by the oracle) for the first `layers` layers."""
    import oracle
    import torch
    lins = [lin for g in w.groups[:4 * layers] for lin in g]

    def one(lin):
        W = wl.weight_torch(lin, device="cpu").numpy()
        return lin, oracle.quantize(w.fmt, W)

    with cf.ThreadPoolExecutor(max_workers=max(1, oracle.host_threads())) as ex:
        imgs = list(ex.map(one, lins))
    xs = {}
    for g in w.groups[:4 * layers]:
        X = wl.activation_torch(w.M, g[0].K, wl.activation_seed(g[0]), device="cpu")
        bits = X.view(torch.int16).numpy().view("uint16")
        for lin in g:
            xs[lin.name] = bits
    return [(lin, img, xs[lin.name]) for lin, img in imgs]


def time_oracle(work, fmt, M, budget_s: float, min_rounds: int = 1, nthreads: int = 0):
    """Run the oracle matmul over `work` (list of (lin, img, X)) repeatedly until
    budget_s has passed; returns (bytes/s, elapsed, rounds). nthreads 0 = every host core."""
    import oracle
    nbytes = 0
    t0 = time.perf_counter()
    rounds = 0
    while True:
        for lin, img, X in work:
            oracle.qmatmul(fmt, img, X, lin.N, lin.K, nthreads)
            nbytes += lin.N * lin.K // 32 * wl.BLOCK_BYTES[fmt] + M * lin.K * 2 + M * lin.N * 4
        rounds += 1
        el = time.perf_counter() - t0
        if rounds >= min_rounds and el >= budget_s:
            return nbytes / el, el, rounds


def cpu_baseline(workloads, budget_s=8.0, layers=2):
    import oracle
    threads = oracle.host_threads()
    total_bytes, total_t = 0.0, 0.0
    one_bytes, one_t = 0.0, 0.0
    n_lin = []
    for w in workloads:
        work = oracle_sample_images(w, min(layers, w.layers))
        n_lin.append(len(work))
        bps, el, rounds = time_oracle(work, w.fmt, w.M, budget_s / len(workloads))
        total_bytes += bps * el
        total_t += el
        # the same sample on one host thread (a shorter budget: one linear at least)
        bps1, el1, _ = time_oracle(work[:1], w.fmt, w.M, budget_s / 4 / len(workloads), nthreads=1)
        one_bytes += bps1 * el1
        one_t += el1
    used = min(layers, workloads[0].layers)
    sample = (f"first {used} of {workloads[0].layers} layers "
              f"({'/'.join(map(str, n_lin))} linears) per format, repeated over ~{budget_s:.0f} s; "
              f"fp64 oracle matmul from oracle-packed weights, {threads} host threads")
    return {"value": total_bytes / total_t / 1e9, "unit": "GB/s", "cores": threads,
            "kind": "oracle", "sample": sample,
            "value_1core": one_bytes / one_t / 1e9,
            "sample_1core": "the first linear of the same sample, repeated on one host thread"}


# ------------------------------------------------------------------ arms

def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    ws = WORKLOADS[args.workload]()
    import oracle
    oracle.build()
    threads = oracle.host_threads()
    # one step = the oracle over a fixed sample of linears (layer 0 of each format),
    # sized so the whole run stays within a few minutes
    work = [(w, oracle_sample_images(w, 1)) for w in ws]
    per_step_target = min(1.0, 90.0 / max(1, args.steps + args.warmup))
    for _ in range(args.warmup):
        for w, items in work:
            time_oracle(items[:1], w.fmt, w.M, 0.0)
    # pick how many linears a step covers from one calibration pass
    t0 = time.perf_counter()
    for w, items in work:
        time_oracle(items[:1], w.fmt, w.M, 0.0)
    one = (time.perf_counter() - t0) / len(work)
    per_fmt = max(1, min(7, int(per_step_target / max(one, 1e-6) / len(work))))
    nbytes = 0
    t0 = time.perf_counter()
    for _ in range(args.steps):
        for w, items in work:
            for lin, img, X in items[:per_fmt]:
                oracle.qmatmul(w.fmt, img, X, lin.N, lin.K)
                nbytes += (lin.N * lin.K // 32 * wl.BLOCK_BYTES[w.fmt]
                           + w.M * lin.K * 2 + w.M * lin.N * 4)
    el = time.perf_counter() - t0
    value = nbytes / el / 1e9
    sample = (f"each step: the fp64 oracle over the first {per_fmt} linears of layer 0 "
              f"per format ({threads} host threads)")
    line = {"impl": "reference", "metric": metric_name(ws), "value": value, "unit": "GB/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": el / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_of(ws, args),
            "cpu_baseline": {"value": value, "unit": "GB/s", "cores": threads,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def truncate(w: wl.Workload, layers: int) -> wl.Workload:
    import dataclasses
    layers = max(1, min(layers, w.layers))
    per = len(w.groups) // w.layers
    return dataclasses.replace(w, layers=layers, groups=tuple(w.groups[:per * layers]))


def metric_name(ws) -> str:
    return "qmatmul µs & HBM GB/s (M=1) / TFLOP/s (M≥50), as fraction of roofline"


L2_BYTES = 126e6   # GB300 L2


def distinct_weight_bytes(ws) -> int:
    """Packed bytes of the distinct weight matrices a step reads (a loop that reuses a
    layer's weights, as the denoising steps do, counts them once)."""
    seen, total = set(), 0
    for w in ws:
        for lin in w.linears():
            key = (w.fmt, lin.name, lin.N, lin.K, lin.seed)
            if key not in seen:
                seen.add(key)
                total += lin.N * lin.K // 32 * wl.BLOCK_BYTES[w.fmt]
    return total


def l2_policy(distinct: int) -> str:
    """How the timed steps keep weights from being served by L2 between reads."""
    if distinct > 3 * L2_BYTES:
        return "inputs larger than L2 (distinct weights per step >> 126 MB L2)"
    if distinct > 2 * L2_BYTES:
        return ("weights rotate through L2 (distinct weights per step > 2 x 126 MB L2, "
                "read in the same order every pass)")
    return "weights partly L2-resident (distinct weights per step < 2 x 126 MB L2)"


def config_of(ws, args):
    w0 = ws[0]
    return {"workload": args.workload,
            "formats": [wl.FMT_NAMES[w.fmt] for w in ws],
            "M": w0.M, "layers": w0.layers, "linears_per_format": len(w0.linears()),
            "repeats": w0.repeats,
            "weight_bytes_per_step": sum(w.weight_bytes() * w.repeats for w in ws),
            "distinct_weight_bytes": distinct_weight_bytes(ws),
            "l2": l2_policy(distinct_weight_bytes(ws)),
            "parallelism": f"replica x{int(os.environ.get('WORLD_SIZE', '1'))}"}


def measure_workload(name, ws, args, dev, dist, steps, warmup, e2e_steps, clocks=True):
    """Build the workload's chains, record each once, and time `steps` passes (after
    `warmup`) with CUDA events on the launching stream: per pass and per chain. Returns the
    measured figures: value / unit (the workload's metric), roofline of the dominant chain
    and of every format, e2e through the public API, clocks."""
    import torch
    import paper_2607_02501_gb300 as emb
    world = dist.get_world_size() if dist is not None else 1
    chains = []
    for w in ws:
        specs, xs, ys = build_chain(w, dev)
        g, layers = capture_graph(specs, w.M)
        chains.append({"w": w, "specs": specs, "xs": xs, "ys": ys, "graph": g, "layers": layers,
                       "launches": count_launches(specs),
                       "bytes": w.algorithmic_bytes(), "flops": w.flops()})
    tensor_bound = ws[0].M >= 50   # the metric is TFLOP/s from M = 50 on
    # the binding roof: tensor cores above the ridge (peak flops / peak bytes), HBM below
    # (M = 50 has ~80 flop/B, under the ~250 flop/B ridge)
    peaks = load_peaks()
    ridge = peaks["bf16_tflops_sustained"] * 1e12 / (peaks["hbm_gbs"] * 1e9)
    roof_tensor = all(w.flops() / w.algorithmic_bytes() >= ridge for w in ws)
    for _ in range(warmup):
        for c in chains:
            for _ in range(c["w"].repeats):
                c["graph"].replay()
    torch.cuda.synchronize()
    assert emb.emb_device_status() == emb.EMB_OK

    sampler = ClockSampler(torch.cuda.current_device()) if clocks else None
    if sampler:
        sampler.start()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(chains) + 1)]
          for _ in range(steps)]
    barrier(dist)
    torch.cuda.synchronize()
    for i in range(steps):
        ev[i][0].record()
        for j, c in enumerate(chains):
            for _ in range(c["w"].repeats):
                c["graph"].replay()
            ev[i][j + 1].record()
    torch.cuda.synchronize()
    barrier(dist)
    clock = sampler.stop() if sampler else None
    total_ms = ev[0][0].elapsed_time(ev[-1][-1])
    chain_ms = [sum(ev[i][j].elapsed_time(ev[i][j + 1]) for i in range(steps))
                for j in range(len(chains))]
    per_step = step_stats([ev[i][0].elapsed_time(ev[i][-1]) for i in range(steps)])
    assert emb.emb_device_status() == emb.EMB_OK
    max_ms = max_over_ranks(total_ms, dist, dev)

    step_bytes = sum(c["bytes"] * c["w"].repeats for c in chains)
    step_flops = sum(c["flops"] * c["w"].repeats for c in chains)
    if tensor_bound:
        value = world * step_flops * steps / (max_ms / 1e3) / 1e12
        unit = "TFLOP/s"
    else:
        value = world * step_bytes * steps / (max_ms / 1e3) / 1e9
        unit = "GB/s"

    def roofline(k):
        """Roofline of chain k: its algorithmic bytes (or flops) per launch over its
        average launch duration in the timed region."""
        c = chains[k]
        launches = c["launches"] * c["w"].repeats * steps
        per_launch_ms = chain_ms[k] / launches
        if roof_tensor:
            achieved = c["flops"] * c["w"].repeats * steps / launches / (per_launch_ms / 1e3) / 1e12
            roof = {"bound": "tensor", "achieved": achieved, "peak": peaks["bf16_tflops_sustained"],
                    "unit": "TFLOP/s", "peak_source": f"{peaks['source']} bf16 dense (sustained)"}
        else:
            achieved = c["bytes"] * c["w"].repeats * steps / launches / (per_launch_ms / 1e3) / 1e9
            roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                    "peak_source": f"{peaks['source']} HBM copy bandwidth"}
        roof["frac"] = roof["achieved"] / roof["peak"]
        roof["traffic"] = kernel_traffic(name, c["w"])
        roof["kernel"] = ("GEMV (gemv_staged_kernel + gemv_ring_kernel + gemv_kernel + gemv_q4_mma_kernel)" if c["w"].M <= 4
                          else "gemm_tc_kernel") + f" <{wl.FMT_NAMES[c['w'].fmt]}>"
        roof["launches_per_step"] = c["launches"] * c["w"].repeats
        roof["per_launch_us"] = per_launch_ms * 1e3
        return roof

    # dominant kernel family: the chain that takes the most time
    dominant = max(range(len(chains)), key=lambda k: chain_ms[k])
    per_format = {}
    for k, cc in enumerate(chains):
        per_format[wl.FMT_NAMES[cc["w"].fmt]] = {
            "ms_per_step": chain_ms[k] / steps,
            unit: (cc["flops"] if tensor_bound else cc["bytes"]) * cc["w"].repeats * steps
            / (chain_ms[k] / 1e3) / (1e12 if tensor_bound else 1e9),
            "roofline": roofline(k)}
    e2e = measure_e2e(chains, e2e_steps, dev, dist, tensor_bound)
    return {"chains": chains, "ws": ws, "value": value, "unit": unit, "max_ms": max_ms,
            "ms_per_step": max_ms / steps, "step_ms": per_step, "roofline": roofline(dominant),
            "per_format": per_format, "e2e": e2e, "clocks": clock, "tensor_bound": tensor_bound,
            "gpu_launches": sum(cc["launches"] * cc["w"].repeats for cc in chains) * steps}


# Every configuration the bench reports beside its headline (one entry per configuration of
# the workload list: the single linear, the 2B decoder at M = 1 (the headline itself), the
# action expert's denoising loop at M = 50, the 2B prefill at M = 816 and the vision tower
# at M = 768, the 7B backbone at M = 1 and M = 280).
CONFIG_WORKLOADS = [("1_single_linear_q8_0_m1", "single_linear"),
                    ("2_gemma2b_decode_m1", "gemma2b_decode"),
                    ("3_action_expert_m50", "action_expert"),
                    ("4_gemma2b_prefill_m816", "gemma2b_prefill"),
                    ("4_vit_m768", "vit"),
                    ("5_llama7b_decode_m1", "llama7b_decode"),
                    ("5_llama7b_prefill_m280", "llama7b_prefill")]


def config_entry(m):
    """The per-configuration summary of a measure_workload result."""
    return {"value": m["value"], "unit": m["unit"], "ms_per_step": m["ms_per_step"],
            "roofline": {k: m["roofline"][k] for k in ("bound", "achieved", "peak", "unit", "frac",
                                                      "traffic", "kernel")},
            "per_format": {f: {"ms_per_step": v["ms_per_step"], m["unit"]: v[m["unit"]],
                               "roofline": {k: v["roofline"][k] for k in ("achieved", "peak", "frac",
                                                                         "traffic")}}
                           for f, v in m["per_format"].items()},
            "e2e": {k: m["e2e"][k] for k in ("value", "unit", "h2d_bytes_per_step", "d2h_bytes_per_step")},
            "formats": [wl.FMT_NAMES[w.fmt] for w in m["ws"]], "M": m["ws"][0].M}


def run_ours(args):
    import torch
    import paper_2607_02501_gb300 as emb
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = init_dist(world, "nccl")
    emb.lib()
    ws = WORKLOADS[args.workload]()
    if args.layers:
        ws = [truncate(w, args.layers) for w in ws]
    m = measure_workload(args.workload, ws, args, dev, dist, args.steps, args.warmup,
                         max(1, min(args.steps, 200)))
    isolated = isolated_launch_us(m["chains"][0]["specs"], ws[0].M) if args.workload == "single_linear" else None
    line = {"metric": metric_name(ws), "value": m["value"], "unit": m["unit"], "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": m["ms_per_step"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if m["tensor_bound"] else "f32", "data": "synthetic",
            "config": config_of(ws, args), "roofline": m["roofline"], "e2e": m["e2e"],
            "clocks": m["clocks"], "gpu_launches": m["gpu_launches"],
            "per_format": {f: {"ms_per_step": v["ms_per_step"], m["unit"]: v[m["unit"]],
                               "roofline": v["roofline"]} for f, v in m["per_format"].items()}}
    line["step_ms"] = m["step_ms"]
    if isolated is not None:
        line["isolated_launch_us"] = isolated
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        torch.cuda.synchronize()
        line["cpu_baseline"] = cpu_baseline(ws)
    if world == 1 and not args.no_configs and args.workload == "gemma2b_decode" and not args.layers:
        # every configuration, a few timed passes each (after the headline's timed region)
        cfg_steps = max(3, min(args.steps, 10))
        configs = {}
        for key, wname in CONFIG_WORKLOADS:
            if wname == args.workload:
                configs[key] = config_entry(m)
                continue
            cm = measure_workload(wname, WORKLOADS[wname](), args, dev, dist, cfg_steps, 3,
                                  max(1, min(cfg_steps, 5)), clocks=False)
            configs[key] = config_entry(cm)
            configs[key]["steps"] = cfg_steps
            for c in cm["chains"]:
                c["graph"].close()
                build_chain.arenas.pop(id(c["specs"]), None)
            del cm
        line["configs"] = configs
    if rank == 0:
        print(json.dumps(line))
    if dist is not None:
        dist.destroy_process_group()
    return 0


def step_stats(ms):
    """Median, minimum and maximum of the per-step device times (CUDA events at each
    step's start and end on this rank)."""
    v = sorted(float(x) for x in ms)
    n = len(v)
    med = v[n // 2] if n % 2 else 0.5 * (v[n // 2 - 1] + v[n // 2])
    return {"median": med, "min": v[0], "max": v[-1], "steps": n}


def isolated_launch_us(specs, M, n=50):
    """One linear at a time on an idle GPU: device time between CUDA events around one
    emb_qlayer_seq call (one launch), each call on the next weight copy; median and min."""
    import torch
    import paper_2607_02501_gb300 as emb
    times = []
    for i in range(n):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record()
        emb.emb_qlayer_seq([specs[i % len(specs)]], M)
        b.record()
        torch.cuda.synchronize()
        times.append(a.elapsed_time(b) * 1e3)
    times.sort()
    return {"median": times[len(times) // 2], "min": times[0], "calls": n,
            "how": "CUDA events around one emb_qlayer_seq call on an idle GPU, rotating weight copies"}


def kernel_traffic(workload, w):
    """DRAM bytes per launch of the dominant kernel from the committed ncu summary, if
    one exists for this workload and matches the current kernel build."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"traffic_{workload}.json")
    try:
        with open(path) as fh:
            d = json.load(fh)
        for src in d["sources"]:
            with open(os.path.join(ROOT, src["path"]), "rb") as fh:
                if hashlib.sha256(fh.read()).hexdigest() != src["sha256"]:
                    return None   # the kernels changed since the counters were taken
        return d.get(wl.FMT_NAMES[w.fmt])
    except (OSError, ValueError, KeyError):
        return None


def measure_e2e(chains, steps, dev, dist, tensor_bound):
    """Same metric through the public call a user makes: per step, copy every layer's
    activations from pinned host memory, run emb_qlayer_seq for each format, copy every
    output back, synchronise."""
    import torch
    import paper_2607_02501_gb300 as emb
    arenas = [build_chain.arenas[id(c["specs"])] for c in chains]
    host_x = [xa.cpu().pin_memory() for xa, _ in arenas]
    host_y = [torch.empty(ya.shape, dtype=ya.dtype).pin_memory() for _, ya in arenas]
    h2d = sum(x.numel() * x.element_size() for x in host_x)   # the bytes each step copies
    d2h = sum(y.numel() * y.element_size() for y in host_y)

    def one_step():
        # per chain: every activation in (one copy of the arena), the recorded chain
        # (one call), every output back (one copy)
        for k, c in enumerate(chains):
            arenas[k][0].copy_(host_x[k], non_blocking=True)
            for _ in range(c["w"].repeats):
                c["graph"].replay()
            host_y[k].copy_(arenas[k][1], non_blocking=True)
        torch.cuda.synchronize()

    for _ in range(3):
        one_step()
    barrier(dist)
    t0 = time.perf_counter()
    for _ in range(steps):
        one_step()
    el = max_over_ranks(time.perf_counter() - t0, dist, dev)
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if tensor_bound:
        work = sum(c["flops"] * c["w"].repeats for c in chains)
        val, unit = world * work * steps / el / 1e12, "TFLOP/s"
    else:
        work = sum(c["bytes"] * c["w"].repeats for c in chains)
        val, unit = world * work * steps / el / 1e9, "GB/s"
    return {"value": val, "unit": unit, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "steps": steps, "ms_per_step": el / steps * 1e3,
            "how": "per format: one pinned H2D copy of all activations, one emb_chain_launch "
                   "of the recorded chain, one D2H copy of all outputs; synchronise each step"}


# ------------------------------------------------------------------ whole-layer loops

LAYER_LOOPS = {"action_expert_layers": wl.action_expert_layers}


class LayerLoopState:
    """Device state of a LayerLoop: per layer its packed weights, norm gains and prefix
    cache; one residual stream and one buffer per intermediate, reused by every layer."""

    def __init__(self, L: "wl.LayerLoop", dev):
        import torch
        import paper_2607_02501_gb300 as emb
        self.L, self.dev = L, dev
        g = torch.Generator(device="cpu")
        self.imgs, self.g1, self.g2, self.K0, self.V0 = [], [], [], [], []
        for l in range(L.layers):
            imgs = {}
            for lin in L.linears(l):
                W = wl.weight_torch(lin, device=dev)
                imgs[lin.name.rsplit(".", 1)[1]] = emb.quantize(L.fmt, W)
                del W
            self.imgs.append(imgs)
            g.manual_seed(L.seed0 + 16 * l + 8)
            self.g1.append((1.0 + 0.1 * torch.randn(L.D, generator=g)).to(dev))
            self.g2.append((1.0 + 0.1 * torch.randn(L.D, generator=g)).to(dev))
            self.K0.append(torch.randn(L.prefix, L.Hk * L.d, generator=g).to(torch.bfloat16).to(dev))
            self.V0.append(torch.randn(L.prefix, L.Hk * L.d, generator=g).to(torch.bfloat16).to(dev))
        g.manual_seed(L.seed0 + 1)
        self.R0 = (torch.randn(L.M, L.D, generator=g) * 2.0)
        self.R = self.R0.to(dev)
        bf = lambda *sh: torch.zeros(*sh, dtype=torch.bfloat16, device=dev)
        M = L.M
        self.h, self.h2 = bf(M, L.D), bf(M, L.D)
        self.q, self.k, self.v = bf(M, L.H * L.d), bf(M, L.Hk * L.d), bf(M, L.Hk * L.d)
        self.a, self.gg = bf(M, L.H * L.d), bf(M, L.F)
        torch.cuda.synchronize()

    def layer(self, l, s, parts=("norm", "linear", "rope", "attention")):
        import paper_2607_02501_gb300 as emb
        L, w, fmt = self.L, self.imgs[l], self.L.fmt
        M, D, F = L.M, L.D, L.F
        qd, kd = L.H * L.d, L.Hk * L.d
        if "norm" in parts:
            emb.emb_rmsnorm(self.R, self.g1[l], self.h, 1e-6, stream=s)
        if "linear" in parts:
            emb.emb_qlayer_seq_chained([(fmt, w["q"], qd, D, self.h, self.q, emb.EMB_EPI_BF16),
                                (fmt, w["k"], kd, D, self.h, self.k, emb.EMB_EPI_BF16),
                                (fmt, w["v"], kd, D, self.h, self.v, emb.EMB_EPI_BF16)], M, stream=s)
        if "rope" in parts:
            emb.emb_rope_qk(self.q, L.H, self.k, L.Hk, L.d, L.prefix, 10000.0, stream=s)
        if "attention" in parts:
            emb.emb_attention(self.q, self.K0[l], self.V0[l], self.k, self.v, self.a, L.H, L.Hk,
                              L.d, 1.0 / math.sqrt(L.d), stream=s)
        if "linear" in parts:
            emb.emb_qlayer_seq_chained([(fmt, w["o"], D, qd, self.a, self.R, emb.EMB_EPI_ADD)], M, stream=s)
        if "norm" in parts:
            emb.emb_rmsnorm(self.R, self.g2[l], self.h2, 1e-6, stream=s)
        if "linear" in parts:
            emb.emb_qlayer_seq_chained([(fmt, w["gate_up"], 2 * F, D, self.h2, self.gg, emb.EMB_EPI_GEGLU)], M,
                               stream=s)
            emb.emb_qlayer_seq_chained([(fmt, w["down"], D, F, self.gg, self.R, emb.EMB_EPI_ADD)], M, stream=s)

    def record(self, s, parts=("norm", "linear", "rope", "attention")):
        """The loop (steps x layers) recorded as one chain on stream s."""
        import paper_2607_02501_gb300 as emb
        rec = emb.Recording(s)
        with rec:
            for _ in range(self.L.steps):
                for l in range(self.L.layers):
                    self.layer(l, s, parts)
        return rec


def layer_loop_oracle(L, budget_s: float):
    """The oracle over one layer of the loop (its six matmuls from oracle-packed weights,
    two norms, two rotaries, attention), repeated for about budget_s; flop/s."""
    import numpy as np
    import oracle
    import torch
    rng = np.random.default_rng(3)
    imgs = []
    for lin in L.linears(0):
        W = wl.weight_torch(lin, device="cpu").numpy()
        imgs.append((lin, oracle.quantize(L.fmt, W)))
    bf = lambda *sh: oracle.bf16_round(rng.standard_normal(sh))
    R = rng.standard_normal((L.M, L.D)).astype(np.float32)
    gam = np.ones(L.D, dtype=np.float32)
    K0, V0 = bf(L.prefix, L.Hk * L.d), bf(L.prefix, L.Hk * L.d)
    to_bits = lambda x: torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.bfloat16).view(
        torch.int16).numpy().view(np.uint16)
    t0 = time.perf_counter()
    rounds = 0
    while True:
        h, _ = oracle.rmsnorm_reference(R, gam, 1e-6)
        hb = to_bits(h)
        outs = {}
        for lin, img in imgs[:3]:
            outs[lin.name.rsplit(".", 1)[1]] = oracle.qmatmul(L.fmt, img, hb, lin.N, lin.K)[0]
        q, _ = oracle.rope_reference(oracle.bf16_round(outs["q"]), L.H, L.d, L.prefix, 10000.0)
        k, _ = oracle.rope_reference(oracle.bf16_round(outs["k"]), L.Hk, L.d, L.prefix, 10000.0)
        a, _ = oracle.attention_reference(q, K0, V0, k, oracle.bf16_round(outs["v"]), L.H, L.Hk, L.d,
                                          1.0 / math.sqrt(L.d))
        lin, img = imgs[3]
        Ro = R + oracle.qmatmul(L.fmt, img, to_bits(a), lin.N, lin.K)[0]
        h2, _ = oracle.rmsnorm_reference(Ro.astype(np.float32), gam, 1e-6)
        lin, img = imgs[4]
        gu = oracle.qmatmul(L.fmt, img, to_bits(h2), lin.N, lin.K)[0]
        gg, _ = oracle.epilogue_reference(oracle.EPI_GEGLU, gu, np.zeros_like(gu))
        lin, img = imgs[5]
        oracle.qmatmul(L.fmt, img, to_bits(gg), lin.N, lin.K)
        rounds += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            return L.layer_flops() * rounds / el, el, rounds


def run_layer_loop(args):
    import torch
    import paper_2607_02501_gb300 as emb
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = init_dist(world, "nccl")
    emb.lib()
    L = LAYER_LOOPS[args.workload]()
    st = LayerLoopState(L, dev)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        for l in range(L.layers):      # one eager pass (per-device setup happens here)
            st.layer(l, s)
        s.synchronize()
        full = st.record(s)
        # the same loop with only the linears, and with only the attention: the roofline's
        # per-launch figures for the kernel families
        lin_only = st.record(s, ("linear",))
        attn_only = st.record(s, ("attention",))
    torch.cuda.synchronize()
    assert emb.emb_device_status() == emb.EMB_OK

    def timed(rec, steps):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
        with torch.cuda.stream(s):
            ev[0].record(s)
            for i in range(steps):
                rec.launch(s)
                ev[i + 1].record(s)
        torch.cuda.synchronize()
        return ev[0].elapsed_time(ev[-1])

    with torch.cuda.stream(s):
        for _ in range(args.warmup):
            full.launch(s)
    torch.cuda.synchronize()
    sampler = ClockSampler(local)
    sampler.start()
    barrier(dist)
    torch.cuda.synchronize()
    total_ms = timed(full, args.steps)
    barrier(dist)
    clocks = sampler.stop()
    assert emb.emb_device_status() == emb.EMB_OK
    max_ms = max_over_ranks(total_ms, dist, dev)
    value = world * L.flops() * args.steps / (max_ms / 1e3) / 1e12

    # kernel families timed on their own (same launches, same buffers)
    k_steps = max(3, min(args.steps, 20))
    lin_ms = timed(lin_only, k_steps) / k_steps
    attn_ms = timed(attn_only, k_steps) / k_steps
    assert emb.emb_device_status() == emb.EMB_OK
    peaks = load_peaks()
    lin_launches = 4 * L.layers * L.steps
    lin_bytes = sum(lin.N * lin.K // 32 * wl.BLOCK_BYTES[L.fmt] for lin in L.linears(0)) * L.layers * L.steps
    if lin_ms >= attn_ms:
        per_launch = lin_ms / lin_launches
        achieved = lin_bytes / lin_launches / (per_launch / 1e3) / 1e9
        kernel = "gemm_tc_kernel <Q8_0> (q/k/v, o, gate/up, down)"
        nl = lin_launches
    else:
        qd, kd = L.H * L.d, L.Hk * L.d
        ab = 2 * L.M * qd * 2 + 2 * 2 * (L.prefix + L.M) * kd
        per_launch = attn_ms / (L.layers * L.steps)
        achieved = ab / (per_launch / 1e3) / 1e9
        kernel = "attention_kernel <128>"
        nl = L.layers * L.steps
    roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / peaks["hbm_gbs"], "traffic": None, "kernel": kernel,
            "peak_source": f"{peaks['source']} HBM copy bandwidth",
            "launches_per_step": nl, "per_launch_us": per_launch * 1e3,
            "family_ms_per_step": {"linears": lin_ms, "attention": attn_ms}}

    # e2e: per closed-loop step the host supplies the chunk's starting residual stream and
    # reads back the final one; the loop replays on the device in between
    host_r = st.R0.pin_memory()
    host_out = torch.empty_like(host_r).pin_memory()
    e2e_steps = max(1, min(args.steps, 100))
    with torch.cuda.stream(s):
        for _ in range(2):
            st.R.copy_(host_r, non_blocking=True)
            full.launch(s)
            host_out.copy_(st.R, non_blocking=True)
        s.synchronize()
        barrier(dist)
        t0 = time.perf_counter()
        for _ in range(e2e_steps):
            st.R.copy_(host_r, non_blocking=True)
            full.launch(s)
            host_out.copy_(st.R, non_blocking=True)
            s.synchronize()
        el = max_over_ranks(time.perf_counter() - t0, dist, dev)
    e2e = {"value": world * L.flops() * e2e_steps / el / 1e12, "unit": "TFLOP/s",
           "h2d_bytes_per_step": host_r.numel() * 4, "d2h_bytes_per_step": host_out.numel() * 4,
           "steps": e2e_steps, "ms_per_step": el / e2e_steps * 1e3,
           "how": "one pinned H2D copy of the starting residual, one replay of the recorded loop, "
                  "one D2H copy of the final residual; synchronise each step"}
    line = {"metric": "whole-layer loop TFLOP/s (linears + attention), M=50",
            "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": max_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": args.workload, "formats": [wl.FMT_NAMES[L.fmt]], "M": L.M,
                       "layers": L.layers, "denoise_steps": L.steps, "prefix_tokens": L.prefix,
                       "heads": [L.H, L.Hk, L.d], "flops_per_step": L.flops(),
                       "algorithmic_bytes_per_step": L.algorithmic_bytes(),
                       "l2": "weights per step 274 MB > 126 MB L2",
                       "parallelism": f"replica x{world}"},
            "roofline": roof, "e2e": e2e, "clocks": clocks,
            "gpu_launches": L.launches() * args.steps}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        fps, el_o, rounds = layer_loop_oracle(L, 8.0)
        line["cpu_baseline"] = {"value": fps / 1e12, "unit": "TFLOP/s", "cores": oracle.host_threads(),
                                "kind": "oracle",
                                "sample": f"one layer of the loop (six matmuls, two norms, two "
                                          f"rotaries, attention) x{rounds} over {el_o:.1f} s"}
    if rank == 0:
        print(json.dumps(line))
    full.close()
    lin_only.close()
    attn_only.close()
    if dist is not None:
        dist.destroy_process_group()
    return 0


def run_layer_loop_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    L = LAYER_LOOPS[args.workload]()
    per_step = min(2.0, 90.0 / max(1, args.steps + args.warmup))
    layer_loop_oracle(L, per_step * args.warmup)
    fps, el, rounds = layer_loop_oracle(L, per_step * args.steps)
    value = fps / 1e12
    sample = f"each step: the oracle over one layer of the loop, {rounds} layers in {el:.1f} s"
    line = {"impl": "reference", "metric": "whole-layer loop TFLOP/s (linears + attention), M=50",
            "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": args.workload, "M": L.M, "layers": L.layers},
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": oracle.host_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(list(WORKLOADS) + list(LAYER_LOOPS)),
                    default="gemma2b_decode")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the per-configuration section of the default line")
    ap.add_argument("--layers", type=int, default=0,
                    help="run only the first L layers (small cases for ncu captures; "
                         "a number taken this way is not the workload's bench value)")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.workload in LAYER_LOOPS:
        if args.layers:
            ap.error("--layers applies to the linear-chain workloads")
        return run_layer_loop_reference(args) if args.impl == "reference" else run_layer_loop(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
