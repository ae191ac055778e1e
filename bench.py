#!/usr/bin/env python3
"""Benchmark of RIS prefill sparse attention on GB300; prints one JSON line on rank 0.

Workload (one step = one pass of the whole hot path over one batch of synthetic input):
a Qwen2-1.5B-shaped prefill attention stack at N = 65536 tokens, 28 layers of (12 query
heads, 2 KV heads, head_dim 128), bf16 Q/K/V ~ N(0, 1) with 1% outlier channels scaled x8
(layer L drawn from seed L), RoPE theta 1e6 with YaRN extension (s = 65536 / 32768 = 2),
run once in Stochastic Mode and once in Structural Mode, each at density 1% with 10
ensemble seeds. Each mode builds its master mask once (all seeds OR-merged) and runs the
28 layers on it: RoPE of q and k, masked QK^T, one softmax per row, PV.

value      = sampled pair-heads per second over the whole job (all ranks): for each mode
             28 * (pairs of the master mask) * 12 query heads, per step.
e2e        = the same metric through the C ABI with host buffers: per step the 28 layers'
             q/k/v are copied from pinned host memory and all outputs copied back, the copies
             overlapped with the compute on two copy streams.
roofline   = the attention kernel's algorithmic gathered bytes (K and V rows of every sampled
             pair, both KV heads: pairs * 2 * 2 * 128 * 2 B) per launch over its CUDA-event
             duration, against the measured HBM copy bandwidth.

--impl reference times the fp64 CPU oracle on the host cores on a bounded sample of the
same workload (its own sample of rows per step) and prints the same line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "sampled attention pairs/s and ms/layer at N=32k/64k, 1% density; % of roofline"
UNIT = "pair-heads/s"
MODES = (("stochastic", 0), ("structural", 1))


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--N", type=int, default=65536)
    ap.add_argument("--layers", type=int, default=28)
    ap.add_argument("--seeds", type=int, default=10)
    ap.add_argument("--density", type=float, default=0.01)
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end measurement")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target oracle seconds per mode")
    return ap.parse_args()


def workload_config(a):
    return {
        "workload": f"Qwen2-1.5B-shaped prefill attention stack, N={a.N}, {a.layers} layers x (12 q heads, "
                    f"2 KV heads, head_dim 128), YaRN RoPE theta 1e6 (native 32768), Stochastic and Structural "
                    f"modes at {a.density:g} density x {a.seeds} seeds",
        "N": a.N, "layers": a.layers, "heads": 12, "kv_heads": 2, "head_dim": 128,
        "rope": "yarn", "rope_theta": 1e6, "native_len": 32768, "modes": [m for m, _ in MODES],
        "density": a.density, "seeds": a.seeds, "input_dtype": "bf16", "outlier_channels": "1% x8",
        "l2": "inputs larger than L2 (each layer's q/k/v is 268 MB; layers use distinct buffers)",
    }


# ----------------------------------------------------------------------------- distributed plumbing
def dist_init():
    """One process per GPU under torchrun; returns (rank, world, dist or None)."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if world <= 1:
        return 0, 1, None
    import torch
    import torch.distributed as dist

    backend = "nccl" if torch.cuda.is_available() else "gloo"
    if backend == "nccl":
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    dist.init_process_group(backend=backend)
    return rank, world, dist


def barrier(dist):
    if dist is not None:
        dist.barrier()


def max_over_ranks(x: float, dist) -> float:
    """Largest value of x over all ranks (the slowest rank sets the job's time)."""
    if dist is None:
        return float(x)
    import torch

    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------- clocks
CLOCK_FIELDS = ["index", "pci.bus_id", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
                "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
                "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]


class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs (read-only queries)."""

    def __init__(self, path):
        self.path = path
        self.proc = None

    def __enter__(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "--query-gpu=" + ",".join(CLOCK_FIELDS),
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.f.close()

    def summary(self, bus_id=None):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) != len(CLOCK_FIELDS):
                continue
            rows.append(dict(zip(CLOCK_FIELDS, parts)))
        if bus_id:
            sel = [r for r in rows if r["pci.bus_id"].lower().endswith(bus_id.lower()[-12:])]
            rows = sel or rows
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        idx = rows[0]["index"]
        rows = [r for r in rows if r["index"] == idx]

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r["clocks.sm"]) for r in rows if num(r["clocks.sm"])]
        reasons = set()
        for r in rows:
            for k in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"):
                if r["clocks_event_reasons." + k].lower() == "active":
                    reasons.add(k)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": num(rows[0]["clocks.max.sm"]), "reasons": sorted(reasons), "samples": len(rows),
                "power_w_max": max((num(r["power.draw"]) or 0.0) for r in rows)}


# ----------------------------------------------------------------------------- CPU oracle sample
def oracle_sample(q_host, k_host, v_host, N, mode, density, seeds, target_s, rng_seed):
    """Time the fp64 oracle on a random sample of rows of one layer; returns (pair-heads, seconds, rows)."""
    import numpy as np

    import oracle

    spec = oracle.MaskSpec(N=N, mode=mode, density=density, seeds=seeds)
    cfg = oracle.RopeCfg(kind=oracle.ROPE_YARN, theta=1e6, native_len=32768)
    rng = np.random.default_rng(rng_seed)
    nrows, total_ph, total_t, used = 8, 0, 0.0, 0
    while total_t < target_s and nrows <= N:
        rows = np.sort(rng.choice(N, size=nrows, replace=False))
        t0 = time.perf_counter()
        out, lse, off, cols = oracle.sparse_attention(q_host, k_host, v_host, spec, cfg, rows=rows)
        dt = time.perf_counter() - t0
        total_ph += int(off[-1]) * q_host.shape[1]
        total_t += dt
        used += nrows
        # grow the sample towards the time target
        nrows = int(min(N, max(2 * nrows, nrows * (target_s - total_t) / max(dt, 1e-3))))
        if total_t + dt * 2 > 2.5 * target_s:
            break
    return total_ph, total_t, used


def host_qkv(N, layer, device):
    import torch

    from paper_2607_21927_gb300 import inputs

    q, k, v = inputs.make_qkv(N, 12, 2, 128, dtype=torch.bfloat16, seed=layer, outliers=True, device=device)
    return [t.float().cpu().numpy().astype("float64") for t in (q, k, v)]


def cpu_baseline(a, device):
    import oracle

    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    qn, kn, vn = host_qkv(a.N, 0, device)
    ph, secs, rows = 0, 0.0, 0
    for name, mode in MODES:
        p, t, r = oracle_sample(qn, kn, vn, a.N, mode, a.density, list(range(a.seeds)), a.cpu_seconds, 1234 + mode)
        ph, secs, rows = ph + p, secs + t, rows + r
    return {"value": ph / secs, "unit": UNIT, "cores": oracle.get_threads(), "kind": "oracle",
            "sample": f"layer 0, {rows} random query rows (both modes), whole path per row: mask row, RoPE, "
                      f"masked softmax attention over all 12 heads; {ph} pair-heads in {secs:.1f} s"}


# ----------------------------------------------------------------------------- reference arm
def run_reference(a, rank):
    if rank != 0:
        return
    import oracle

    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    qn, kn, vn = host_qkv(a.N, 0, "cpu")
    per_step = max(2.0, a.cpu_seconds / 2)
    for w in range(a.warmup):
        for name, mode in MODES:
            oracle_sample(qn, kn, vn, a.N, mode, a.density, list(range(a.seeds)), 0.5, 99 + w)
    ph, secs, rows = 0, 0.0, 0
    for s in range(a.steps):
        for name, mode in MODES:
            p, t, r = oracle_sample(qn, kn, vn, a.N, mode, a.density, list(range(a.seeds)), per_step / 2, 7 * s + mode)
            ph, secs, rows = ph + p, secs + t, rows + r
    value = ph / secs
    sample = (f"per step: random query rows of layer 0 in both modes, whole path per row; {rows} rows, "
              f"{ph} pair-heads in {secs:.1f} s over {a.steps} steps")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": a.gpus,
            "steps": a.steps, "warmup": a.warmup, "ms_per_step": 1e3 * secs / a.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(a),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.get_threads(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- traffic record
def recorded_traffic(kernel_file: str):
    """DRAM bytes per launch from the committed ncu summary, if taken on the current kernel source."""
    rec = os.path.join(ROOT, "profiles", "traffic.json")
    src = os.path.join(ROOT, "paper_2607_21927_gb300", "csrc", kernel_file)
    try:
        data = json.load(open(rec))
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
        ent = data.get(kernel_file)
        if ent and ent.get("source_sha256_16") == h:
            return ent.get("dram_bytes_per_launch_full_size")
    except Exception:
        pass
    return None


# ----------------------------------------------------------------------------- our arm
def main():
    a = parse_args()
    rank, world, dist = dist_init()
    if a.impl == "reference":
        run_reference(a, rank)
        return

    import torch

    from paper_2607_21927_gb300 import inputs, ris

    dev = torch.device("cuda", torch.cuda.current_device())
    N, L, Hq, Hkv, D = a.N, a.layers, 12, 2, 128
    seeds = list(range(a.seeds))
    rope = ris.rope_cfg(ris.ROPE_YARN, 1e6, 32768)

    # inputs resident in HBM: one (q, k, v) per layer, layer L drawn from seed L
    qs, ks, vs = [], [], []
    for layer in range(L):
        q, k, v = inputs.make_qkv(N, Hq, Hkv, D, dtype=torch.bfloat16, seed=layer, outliers=True, device=dev)
        qs.append(q)
        ks.append(k)
        vs.append(v)
    outs = [[torch.empty(N, Hq, D, dtype=torch.bfloat16, device=dev) for _ in range(L)] for _ in MODES]
    stream = torch.cuda.current_stream()
    pairs, design = {}, {}

    def step():
        for mi, (name, mode) in enumerate(MODES):
            m = ris.ris_mask_generate(N, Hkv, mode, a.density, seeds)
            pairs[name] = m.info().n_pairs
            design[name] = ris.ris_attention_design(m, torch.bfloat16, D)
            for layer in range(L):
                ris.ris_attention_masked(m, qs[layer], ks[layer], vs[layer], rope=rope, out=outs[mi][layer])
            m.free()

    for _ in range(a.warmup):
        step()
    torch.cuda.synchronize()

    # ---- device-timed region
    import tempfile

    clocks_path = os.path.join(tempfile.gettempdir(), f"ris_bench_clocks_{os.getpid()}.csv")
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(dist)
    torch.cuda.synchronize()
    ris.ris_kernel_timer_enable(True)
    n0 = ris.ris_launch_count()
    with ClockSampler(clocks_path) as clk:
        ev0.record(stream)
        for _ in range(a.steps):
            step()
        ev1.record(stream)
        torch.cuda.synchronize()
    launches = ris.ris_launch_count() - n0
    k_ms, k_n = ris.ris_kernel_timer_read()
    ris.ris_kernel_timer_enable(False)
    barrier(dist)
    elapsed_ms = max_over_ranks(ev0.elapsed_time(ev1), dist)

    pair_heads_step = sum(pairs[name] for name, _ in MODES) * L * Hq
    value = world * pair_heads_step * a.steps / (elapsed_ms / 1e3)
    ms_step = elapsed_ms / a.steps

    # roofline of the attention kernel over the timed region: algorithmic bytes (gather) or
    # algorithmic FLOPs (tiles) per launch / mean launch time
    launches_per_step = len(MODES) * L
    mean_launch_ms = k_ms / max(k_n, 1)
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    hbm = peaks.get("hbm_gbs")
    peak_note = "measured" if hbm else "fallback"
    hbm = hbm or 6800.0
    tc = peaks.get("bf16_tflops_sustained") or 1700.0
    kinds = sorted(set(design.values()))
    if kinds == [2]:  # every launch on the tensor-core tile kernel
        flops_per_launch = 4 * D * Hq * sum(pairs.values()) * L / launches_per_step
        achieved = flops_per_launch / (mean_launch_ms / 1e3) / 1e12
        roofline = {"bound": "tensor", "achieved": achieved, "peak": tc, "unit": "TFLOP/s", "frac": achieved / tc,
                    "traffic": None, "kernel": "k_attn_tile (tcgen05 masked tiles)",
                    "peak_source": ("measured sustained bf16" if peaks.get("bf16_tflops_sustained") else "fallback"),
                    "flops": "algorithmic: 4 * head_dim * query heads per sampled pair",
                    "mean_launch_ms": mean_launch_ms, "launches_timed": k_n}
    else:
        bytes_per_step = sum(pairs[name] for name, _ in MODES) * L * Hkv * 2 * D * 2
        achieved = (bytes_per_step / launches_per_step) / (mean_launch_ms / 1e3) / 1e9
        roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                    "traffic": recorded_traffic("attn_bf16.cu") if kinds == [0] else None,
                    "kernel": "k_attn_bf16 (register gather)" if kinds == [0] else "mixed designs " + str(kinds),
                    "peak_source": peak_note, "bytes": "algorithmic: K and V rows of every sampled pair, both KV heads",
                    "mean_launch_ms": mean_launch_ms, "launches_timed": k_n}
    # the sampled-pair roofline: max(sampled FLOPs / tensor peak, tile-reuse K/V bytes / HBM)
    flops = 4 * D * Hq * sum(pairs.values()) * L
    b_tile = len(MODES) * L * (N / 128) * (N / 2) * Hkv * 2 * D * 2
    t_roof = max(flops / (tc * 1e12), b_tile / (hbm * 1e9))
    clocks = clk.summary(getattr(torch.cuda.get_device_properties(dev), "pci_bus_id", None))

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": a.steps, "warmup": a.warmup,
            "ms_per_step": ms_step, "ms_per_layer": ms_step / (len(MODES) * L), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": workload_config(a), "pairs_per_mask": pairs,
            "design_per_mode": {k: ris.DESIGNS.get(v, v) for k, v in design.items()}, "roofline": roofline,
            "pair_roofline": {"t_roof_ms_per_step": 1e3 * t_roof, "frac": 1e3 * t_roof / ms_step,
                                    "formula": "max(4*D*Hq*pairs / bf16 sustained, (N/128)*(N/2)*Hkv*2*D*2 B / HBM)"},
            "clocks": clocks, "gpu_launches": launches}

    # ---- end to end through the C ABI with host buffers
    if not a.no_e2e:
        hq = [t.cpu().pin_memory() for t in qs]
        hk = [t.cpu().pin_memory() for t in ks]
        hv = [t.cpu().pin_memory() for t in vs]
        ho = [[torch.empty(N, Hq, D, dtype=torch.bfloat16).pin_memory() for _ in range(L)] for _ in MODES]
        h2d = sum(t.numel() * t.element_size() for t in hq + hk + hv)
        d2h = sum(t.numel() * t.element_size() for row in ho for t in row)

        # Host transfers overlap the compute: one stream brings the layers' q/k/v in, another
        # takes the outputs out, both ordered against the compute stream with per-layer events.
        h2d_s, d2h_s = torch.cuda.Stream(), torch.cuda.Stream()
        in_ready = [torch.cuda.Event() for _ in range(L)]
        layer_free = [torch.cuda.Event() for _ in range(L)]
        out_ready = [[torch.cuda.Event() for _ in range(L)] for _ in MODES]
        out_free = [[torch.cuda.Event() for _ in range(L)] for _ in MODES]
        first = [True]

        def e2e_step():
            for layer in range(L):
                with torch.cuda.stream(h2d_s):
                    if not first[0]:
                        h2d_s.wait_event(layer_free[layer])
                    qs[layer].copy_(hq[layer], non_blocking=True)
                    ks[layer].copy_(hk[layer], non_blocking=True)
                    vs[layer].copy_(hv[layer], non_blocking=True)
                    in_ready[layer].record(h2d_s)
            for mi, (name, mode) in enumerate(MODES):
                m = ris.ris_mask_generate(N, Hkv, mode, a.density, seeds)
                for layer in range(L):
                    stream.wait_event(in_ready[layer])
                    if not first[0]:
                        stream.wait_event(out_free[mi][layer])
                    ris.ris_attention_masked(m, qs[layer], ks[layer], vs[layer], rope=rope, out=outs[mi][layer])
                    out_ready[mi][layer].record(stream)
                    if mi == len(MODES) - 1:
                        layer_free[layer].record(stream)
                    with torch.cuda.stream(d2h_s):
                        d2h_s.wait_event(out_ready[mi][layer])
                        ho[mi][layer].copy_(outs[mi][layer], non_blocking=True)
                        out_free[mi][layer].record(d2h_s)
                m.free()
            first[0] = False

        e2e_step()
        torch.cuda.synchronize()
        barrier(dist)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        h2d_s.wait_event(e0)
        d2h_s.wait_event(e0)
        for _ in range(a.steps):
            e2e_step()
        stream.wait_stream(h2d_s)
        stream.wait_stream(d2h_s)
        e1.record(stream)
        torch.cuda.synchronize()
        e_ms = max_over_ranks(e0.elapsed_time(e1), dist)
        line["e2e"] = {"value": world * pair_heads_step * a.steps / (e_ms / 1e3), "unit": UNIT,
                       "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": e_ms / a.steps}
    else:
        line["e2e"] = None

    if rank == 0 and world == 1 and not a.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(a, dev)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
