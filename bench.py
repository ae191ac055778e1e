#!/usr/bin/env python3
"""Benchmark of RIS prefill sparse attention on GB300; prints one JSON line on rank 0.

Default workload (C5; one step = one pass of the whole hot path over one batch of synthetic
input): a Qwen2-1.5B-shaped prefill attention stack at N = 65536 tokens, 28 layers of (12
query heads, 2 KV heads, head_dim 128), bf16 Q/K/V ~ N(0, 1) with 1% outlier channels scaled
x8 (layer L drawn from seed L), RoPE theta 1e6 with YaRN extension (s = 65536 / 32768 = 2),
run once in Stochastic Mode and once in Structural Mode, each at density 1% with 10 ensemble
seeds. Each run builds its master mask once (all seeds OR-merged) and runs the layers on it:
RoPE of q and k, masked QK^T, one softmax per row, PV. --workload selects the other
evaluation shapes (C1 .. C4c, one layer shape each, with enough distinct layers per step that
the inputs of a step exceed L2).

value      = sampled pair-heads per second over the whole job (all ranks): for each run
             layers * (pairs of the master mask) * query heads, per step.
e2e        = the same metric through the C ABI with host buffers: per step every layer's
             q/k/v is copied from pinned host memory and all outputs copied back, the copies
             overlapped with the compute on two copy streams.
mask_ms_per_step / attn_ms_per_layer
           = the mask builds of a step (CUDA events around each build inside the timed region)
             and the rest of the step per layer (RoPE + attention), so that the per-layer cost
             is reported with the mask build amortised separately.
roofline   = the dominant attention kernel: for the gathering designs its algorithmic bytes
             (K and V rows of every sampled pair, all KV heads) per launch over the mean
             CUDA-event launch time, against this library's L2 row-gather probe when the
             layer's K/V working set fits in L2 (bound "l2", the HBM fraction beside it), else
             the measured HBM copy bandwidth; for the tcgen05 tile design its algorithmic
             FLOPs (4 * head_dim per sampled pair-head) against the measured sustained bf16 peak.

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
L2_FLUSH_BYTES = 256 << 20  # distinct per-layer inputs of at least this size, so each layer starts cold in L2

# Workloads (names follow the configuration table of the method's evaluation shapes). Each run
# is (name, mode, density, n_seeds): one master mask built per run, every layer attended on it.
# Qwen2-1.5B shape: 12 query heads, 2 KV heads, head_dim 128, theta 1e6, native 32768 tokens;
# TinyLlama shape: 32 / 4 / 64, theta 1e4, native 2048 tokens.
WORKLOADS = {
    "C1": dict(N=2048, layers=0, Hq=1, Hkv=1, D=128, dtype="f32", outliers=False, rope=("plain", 1e6, 32768),
               runs=[("stochastic", 0, 0.05, 1)], title="single-head fp32 attention, N=2048"),
    "C2": dict(N=8192, layers=0, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
               runs=[("stochastic", 0, 0.01, 10)], title="Qwen2-1.5B-shaped attention layer, N=8192"),
    "C3": dict(N=16384, layers=0, Hq=32, Hkv=4, D=64, dtype="bf16", outliers=False, rope=("yarn", 1e4, 2048),
               runs=[("structural", 1, 0.01, 10)], title="TinyLlama-shaped attention layer, N=16384, YaRN s=8"),
    "C4a": dict(N=32768, layers=0, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
                runs=[("stochastic", 0, 0.01, 70)], title="Qwen2-1.5B-shaped attention layer, N=32768"),
    "C4b": dict(N=32768, layers=0, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
                runs=[("stochastic", 0, 0.05, 10)], title="Qwen2-1.5B-shaped attention layer, N=32768"),
    "C4c": dict(N=32768, layers=0, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
                runs=[("dense", 2, 1.0, 1)], title="Qwen2-1.5B-shaped attention layer, N=32768, dense causal"),
    "C5": dict(N=65536, layers=28, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
               runs=[("stochastic", 0, 0.01, 10), ("structural", 1, 0.01, 10)],
               title="Qwen2-1.5B-shaped prefill attention stack, N=65536, 28 layers, YaRN s=2"),
    # C5 with the index-draw sampler (the torch.randint reading): K = round(dN) draws per row and seed
    "C5r": dict(N=65536, layers=28, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
                runs=[("stochastic", 0, 0.01, 10), ("structural", 1, 0.01, 10)], sampler=1,
                title="C5 with the index-draw sampler"),
    # C5 with the paper's full geometry: local window 1024 and anchors over the first tokens
    "C6": dict(N=65536, layers=28, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
               runs=[("stochastic", 0, 0.01, 10), ("structural", 1, 0.01, 10)], geometry="paper",
               title="C5 with the paper's geometry (local window 1024 + 4 anchor tokens)"),
    # Hybrid Anchor decode after the C5 prefill: 32 generated tokens x 28 layers per run, the
    # anchor of each run frozen at the first token, a 1024-token sliding window
    "D5": dict(N=65536, layers=28, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
               runs=[("stochastic", 0, 0.01, 10), ("structural", 1, 0.01, 10)], kind="decode", gen=32, window=1024,
               title="Hybrid Anchor decode after the N=65536 prefill, 28 layers, YaRN s=2"),
    # per-seed ensembles (ris_ensemble_batch's mode): one output per seed, all seeds in one launch
    "E2": dict(N=8192, layers=0, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
               runs=[("stochastic", 0, 0.01, 10)], per_seed=True,
               title="C2 as a per-seed ensemble (10 outputs per layer)"),
    "E4a": dict(N=32768, layers=0, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
                runs=[("stochastic", 0, 0.01, 70)], per_seed=True,
                title="C4a as a per-seed ensemble (70 outputs per layer)"),
    "E5": dict(N=65536, layers=0, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
               runs=[("stochastic", 0, 0.01, 10)], per_seed=True,
               title="C5 Stochastic as a per-seed ensemble (10 outputs per layer)"),
    # the sub-1% Structural sweep at 64k: d = 0.1% .. 0.9%, 50 .. 200 seeds, one layer each
    "S1": dict(N=65536, layers=1, Hq=12, Hkv=2, D=128, dtype="bf16", outliers=True, rope=("yarn", 1e6, 32768),
               runs=[(f"structural_{d / 10:.1f}pct_x{s}", 1, d / 1000, s) for d in range(1, 10)
                     for s in (50, 100, 150, 200)],
               title="sub-1% Structural sweep at N=65536 (36 masks, one layer each)"),
}


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="C5")
    ap.add_argument("--N", type=int, default=None, help="override the workload's token count")
    ap.add_argument("--layers", type=int, default=None, help="override the number of layers per step")
    ap.add_argument("--seeds", type=int, default=None, help="override the ensemble size of every run")
    ap.add_argument("--density", type=float, default=None, help="override the density of every sparse run")
    ap.add_argument("--no-e2e", action="store_true", help="skip the host-buffer end-to-end measurement")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--no-probes", action="store_true", help="skip the L2 / FFMA ceiling probes")
    ap.add_argument("--cpu-seconds", type=float, default=12.0, help="target oracle seconds per step")
    ap.add_argument("--shard", choices=("replicas", "rows", "rows-kv"), default="replicas",
                    help="with several ranks: every rank runs the whole workload (weak scaling), or each "
                         "rank takes a balanced range of query rows of the same workload (strong scaling) "
                         "with all of K and V (rows), or holding only its own rows of q, k and v and "
                         "all-gathering each layer's K and V (rows-kv)")
    a = ap.parse_args()
    w = dict(WORKLOADS[a.workload])
    w["name"] = a.workload
    if a.N is not None:
        w["N"] = a.N
    runs = []
    for name, mode, dens, ns in w["runs"]:
        if mode != 2:
            dens = a.density if a.density is not None else dens
            ns = a.seeds if a.seeds is not None else ns
        runs.append((name, mode, dens, ns))
    w["runs"] = runs
    e = 4 if w["dtype"] == "f32" else 2
    per_layer = w["N"] * (w["Hq"] + 2 * w["Hkv"]) * w["D"] * e
    if a.layers is not None:
        w["layers"] = a.layers
    elif w["layers"] == 0:
        w["layers"] = max(1, -(-L2_FLUSH_BYTES // per_layer))
    a.w = w
    return a


def workload_config(a):
    w = a.w
    e = 4 if w["dtype"] == "f32" else 2
    per_layer = w["N"] * (w["Hq"] + 2 * w["Hkv"]) * w["D"] * e
    kind, theta, native = w["rope"]
    runs = ", ".join(f"{n}" + ("" if m == 2 else f" {d:g} x {s} seeds") for n, m, d, s in w["runs"])
    return {
        "workload": f"{w['name']}: {w['title']} ({w['Hq']} q heads, {w['Hkv']} KV heads, head_dim {w['D']}, "
                    f"{w['dtype']}{' with 1% x8 outlier channels' if w['outliers'] else ''}), {kind} RoPE "
                    f"theta {theta:g} native {native}; runs: {runs}; {w['layers']} layer(s) per run per step",
        "name": w["name"], "N": w["N"], "layers": w["layers"], "heads": w["Hq"], "kv_heads": w["Hkv"],
        "head_dim": w["D"], "rope": kind, "rope_theta": theta, "native_len": native,
        "runs": [{"name": n, "mode": m, "density": d, "seeds": s} for n, m, d, s in w["runs"]],
        "input_dtype": w["dtype"], "outlier_channels": "1% x8" if w["outliers"] else None,
        "geometry": ("local window 1024 + 4 anchors" if w.get("geometry") == "paper" else "diagonal only"),
        "sampler": "index draws (K = round(dN) per row and seed)" if w.get("sampler") else "Bernoulli per pair",
        "seed_outputs": "one per seed (per-seed masks)" if w.get("per_seed") else "one (union of the seeds)",
        "multi_gpu": {"rows": "balanced query-row ranges of one workload per rank",
                      "rows-kv": "balanced query-row ranges of one workload per rank, each rank holding only "
                                 "its rows of q, k and v and all-gathering each layer's K and V"}.get(
                          a.shard, "one whole workload per rank"),
        "l2": (f"inputs larger than L2: each layer has its own q/k/v ({per_layer / 2**20:.0f} MiB), "
               f"{w['layers']} layers = {w['layers'] * per_layer / 2**20:.0f} MiB per run"),
    } | ({"decode": {"generated_tokens": w["gen"], "window": w["window"],
                     "cache": "rotated K (bf16 hi + lo) and V of every layer, N + generated tokens rows",
                     "l2": "every token reads 28 layers' selected K/V rows (~300 MB), more than L2"}}
         if w.get("kind") == "decode" else {})


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
ROPE_KINDS = {"none": 0, "plain": 1, "linear": 2, "yarn": 3}


def oracle_rope(w):
    import oracle

    kind, theta, native = w["rope"]
    return oracle.RopeCfg(kind=ROPE_KINDS[kind], theta=theta, native_len=native)


def oracle_sample(q_host, k_host, v_host, w, run, target_s, rng_seed):
    """Time the fp64 oracle on a random sample of rows of one layer; returns (pair-heads, seconds, rows)."""
    import numpy as np

    import oracle

    N = w["N"]
    name, mode, density, n_seeds = run
    paper = w.get("geometry") == "paper"
    spec = oracle.MaskSpec(N=N, mode=mode, density=density, seeds=list(range(n_seeds)),
                           local_window=1024 if paper else 1, n_anchor=4 if paper else 0,
                           sampler=int(w.get("sampler", 0)))
    cfg = oracle_rope(w)
    rng = np.random.default_rng(rng_seed)
    nrows, total_ph, total_t, used = 8, 0, 0.0, 0
    while total_t < target_s and nrows <= N:
        rows = np.sort(rng.choice(N, size=nrows, replace=False))
        if w.get("per_seed"):  # one seed's own mask per sample
            spec.seed_index = int(rng.integers(n_seeds))
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


def host_qkv(w, layer, device):
    import torch

    from paper_2607_21927_gb300 import inputs

    dt = torch.float32 if w["dtype"] == "f32" else torch.bfloat16
    q, k, v = inputs.make_qkv(w["N"], w["Hq"], w["Hkv"], w["D"], dtype=dt, seed=layer, outliers=w["outliers"],
                              device=device)
    return [t.float().cpu().numpy().astype("float64") for t in (q, k, v)]


def cpu_baseline(a, device):
    import oracle

    w = a.w
    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    qn, kn, vn = host_qkv(w, 0, device)
    ph, secs, rows = 0, 0.0, 0
    for ri, run in enumerate(w["runs"]):
        p, t, r = oracle_sample(qn, kn, vn, w, run, a.cpu_seconds / len(w["runs"]), 1234 + ri)
        ph, secs, rows = ph + p, secs + t, rows + r
    return {"value": ph / secs, "unit": UNIT, "cores": oracle.get_threads(), "kind": "oracle",
            "sample": f"layer 0, {rows} random query rows (over {len(w['runs'])} run(s)), whole path per row: "
                      f"mask row, RoPE, masked softmax attention over all {w['Hq']} heads; {ph} pair-heads in "
                      f"{secs:.1f} s"}


# ----------------------------------------------------------------------------- reference arm
def run_reference(a, rank):
    if rank != 0:
        return
    import oracle

    w = a.w
    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    qn, kn, vn = host_qkv(w, 0, "cpu")
    per_step = max(2.0, a.cpu_seconds / 2)
    for s in range(a.warmup):
        for ri, run in enumerate(w["runs"]):
            oracle_sample(qn, kn, vn, w, run, 0.5, 99 + s)
    ph, secs, rows = 0, 0.0, 0
    for s in range(a.steps):
        for ri, run in enumerate(w["runs"]):
            p, t, r = oracle_sample(qn, kn, vn, w, run, per_step / len(w["runs"]), 7 * s + ri)
            ph, secs, rows = ph + p, secs + t, rows + r
    value = ph / secs
    sample = (f"per step: random query rows of layer 0 in every run, whole path per row; {rows} rows, "
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
def recorded_traffic(kernel_files, workload: str):
    """DRAM bytes per launch (per layer call, summed over its launches) of the kernels of
    `kernel_files` at `workload`, from the committed ncu record, if it was taken on the
    current sources."""
    rec = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        data = json.load(open(rec))
        hs = [hashlib.sha256(open(os.path.join(ROOT, "paper_2607_21927_gb300", "csrc", f), "rb").read()).hexdigest()[:16]
              for f in kernel_files]
        ent = data.get("+".join(kernel_files), {}).get(workload)
        if ent and ent.get("source_sha256_16") == (hs[0] if len(hs) == 1 else hs):
            return ent.get("dram_bytes_per_launch_full_size")
    except Exception:
        pass
    return None


# ----------------------------------------------------------------------------- decode workload
def oracle_decode_sample(w, target_s, rng_seed):
    """Time the fp64 oracle's decode step on random (run, generated token) samples of layer 0;
    returns (pair-heads, seconds, steps)."""
    import numpy as np

    import oracle
    from paper_2607_21927_gb300 import inputs

    import torch

    N, gen = w["N"], w["gen"]
    T = N + gen
    q, k, v = inputs.make_qkv(T, w["Hq"], w["Hkv"], w["D"], dtype=torch.bfloat16, seed=0, outliers=w["outliers"])
    qn, kn, vn = (x.float().numpy().astype("float64") for x in (q, k, v))
    cfg = oracle_rope(w)
    anchors = [oracle.decode_anchor(oracle.MaskSpec(N=N, mode=m, density=d, seeds=list(range(s))))
               for _, m, d, s in w["runs"]]
    rng = np.random.default_rng(rng_seed)
    ph, secs, steps = 0, 0.0, 0
    while secs < target_s:
        ri = int(rng.integers(len(anchors)))
        t = N + int(rng.integers(gen))
        t0 = time.perf_counter()
        out, lse, keys = oracle.decode_step(qn[t], kn, vn, t, anchors[ri], w["window"], cfg, N)
        secs += time.perf_counter() - t0
        ph += keys.shape[0] * w["Hq"]
        steps += 1
    return ph, secs, steps


def run_reference_decode(a, rank):
    if rank != 0:
        return
    import oracle

    w = a.w
    oracle.set_threads(os.cpu_count() or 1)
    oracle_decode_sample(w, 0.5, 99)
    ph, secs, steps = oracle_decode_sample(w, max(2.0, a.cpu_seconds / 2) * a.steps, 7)
    value = ph / secs
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": a.gpus,
            "steps": a.steps, "warmup": a.warmup, "ms_per_step": 1e3 * secs / a.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(a),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.get_threads(), "kind": "oracle",
                             "sample": f"{steps} decode steps of layer 0 (random run and token), {ph} pair-heads "
                                       f"in {secs:.1f} s"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main_decode(a, rank, world, dist):
    """Decode workload: per run, the anchor is frozen once (timed apart), then each step generates
    `gen` tokens through all layers; one CUDA graph per (run, token) position-independent chain of
    layers is captured once and replayed, the position living in device memory."""
    import tempfile

    import torch

    from paper_2607_21927_gb300 import inputs, ris

    w = a.w
    dev = torch.device("cuda", torch.cuda.current_device())
    N, L, Hq, Hkv, D, gen, W = w["N"], w["layers"], w["Hq"], w["Hkv"], w["D"], w["gen"], w["window"]
    T = N + gen
    kind, theta, native = w["rope"]
    rope = ris.rope_cfg(ROPE_KINDS[kind], theta, native)
    runs = w["runs"]
    # per layer: the rotated cache of N + gen positions (prefill and generated tokens' keys)
    k_hi, k_lo, vs = [], [], []
    for layer in range(L):
        _, k, v = inputs.make_qkv(T, Hq, Hkv, D, dtype=torch.bfloat16, seed=layer, outliers=w["outliers"], device=dev)
        hi, lo = ris.ris_rope_split(k, N, rope)
        k_hi.append(hi)
        k_lo.append(lo)
        vs.append(v)
        del k
    gq = torch.Generator(device=dev)
    gq.manual_seed(1234)
    qs = torch.randn(gen, L, Hq, D, generator=gq, device=dev).to(torch.bfloat16)
    outs = torch.empty(len(runs), gen, L, Hq, D, dtype=torch.float32, device=dev)
    qbuf = torch.empty(L, Hq, D, dtype=torch.bfloat16, device=dev)
    obuf = torch.empty(L, Hq, D, dtype=torch.float32, device=dev)
    t_dev = torch.zeros(1, dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream()

    ev_a0, ev_a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev_a0.record(stream)
    anchors = [ris.ris_decode_anchor(N, Hkv, m, d, list(range(s))) for _, m, d, s in runs]
    ev_a1.record(stream)
    torch.cuda.synchronize()
    anchor_ms = ev_a0.elapsed_time(ev_a1) / len(runs)
    n_anchor = [an.info()[2] for an in anchors]

    def token_chain(an):
        for layer in range(L):
            ris.ris_decode_step(an, qbuf[layer], k_hi[layer], k_lo[layer], vs[layer], N, W, N, rope,
                                out=obuf[layer], t_dev=t_dev, advance=(layer == L - 1))

    graphs = []
    for an in anchors:
        t_dev.fill_(N)
        token_chain(an)  # sizes the anchor's partials buffer before capture
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            token_chain(an)
        graphs.append(g)
    t_start = torch.tensor([N], dtype=torch.int64).pin_memory()

    def step():
        for ri, g in enumerate(graphs):
            t_dev.copy_(t_start, non_blocking=True)
            for tok in range(gen):
                qbuf.copy_(qs[tok])
                g.replay()
                outs[ri, tok].copy_(obuf)

    for _ in range(a.warmup):
        step()
    torch.cuda.synchronize()
    ris.ris_device_status()
    ceil = ceilings(ris, w, a.no_probes)

    clocks_path = os.path.join(tempfile.gettempdir(), f"ris_bench_clocks_{os.getpid()}.csv")
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(dist)
    torch.cuda.synchronize()
    with ClockSampler(clocks_path) as clk:
        ev0.record(stream)
        for _ in range(a.steps):
            step()
        ev1.record(stream)
        torch.cuda.synchronize()
    # graph replays bypass the library's host launch counter: two kernels per layer and token
    launches = 2 * L * gen * len(runs) * a.steps
    barrier(dist)
    elapsed_ms = max_over_ranks(ev0.elapsed_time(ev1), dist)
    ris.ris_device_status()

    # keys per token: the anchor keys below the window plus the window (t - W < j <= t)
    pairs = 0
    for an, na in zip(anchors, n_anchor):
        keys = an.info()[3].cpu()
        for tok in range(gen):
            t = N + tok
            lo = max(0, t - W + 1)
            pairs += int((keys < lo).sum()) + (t - lo + 1)
    pair_heads_step = pairs * L * Hq
    value = world * pair_heads_step * a.steps / (elapsed_ms / 1e3)
    ms_step = elapsed_ms / a.steps
    tokens_step = gen * len(runs)
    bytes_step = pairs * L * Hkv * 2 * D * 2  # K and V rows (bf16) of every selected key, all KV heads
    achieved = bytes_step / (ms_step / 1e3) / 1e9
    hbm = ceil["hbm_gbs"]
    roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "traffic": None, "kernel": "k_decode_partial + k_decode_combine (whole token chain)",
                "peak_source": ceil["hbm_source"],
                "bytes": "algorithmic: K and V rows (bf16) of every selected key, all KV heads, over the step time "
                         "(graph replays: no per-launch timer)"}
    clocks = clk.summary(getattr(torch.cuda.get_device_properties(dev), "pci_bus_id", None))
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": a.steps, "warmup": a.warmup,
            "ms_per_step": ms_step, "us_per_token": 1e3 * ms_step / tokens_step,
            "us_per_token_layer": 1e3 * ms_step / (tokens_step * L), "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "config": workload_config(a),
            "anchor_ms": anchor_ms, "anchor_keys": dict(zip([r[0] for r in runs], n_anchor)),
            "roofline": roofline, "ceilings": ceil, "clocks": clocks, "gpu_launches": launches}

    # host-driven loop (no graph) for comparison: one Python + C call per layer and token
    def host_step():
        for ri, an in enumerate(anchors):
            for tok in range(gen):
                for layer in range(L):
                    ris.ris_decode_step(an, qs[tok, layer], k_hi[layer], k_lo[layer], vs[layer], N + tok, W, N,
                                        rope, out=outs[ri, tok, layer])

    host_step()
    torch.cuda.synchronize()
    h0, h1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    h0.record(stream)
    host_step()
    h1.record(stream)
    torch.cuda.synchronize()
    line["host_loop_us_per_token"] = 1e3 * h0.elapsed_time(h1) / tokens_step

    if not a.no_e2e:
        hq = qs.cpu().pin_memory()
        ho = torch.empty(outs.shape, dtype=outs.dtype).pin_memory()

        def e2e_step():
            for ri, g in enumerate(graphs):
                t_dev.copy_(t_start, non_blocking=True)
                for tok in range(gen):
                    qbuf.copy_(hq[tok], non_blocking=True)
                    g.replay()
                    ho[ri, tok].copy_(obuf, non_blocking=True)

        e2e_step()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(a.steps):
            e2e_step()
        e1.record(stream)
        torch.cuda.synchronize()
        e_ms = max_over_ranks(e0.elapsed_time(e1), dist)
        line["e2e"] = {"value": world * pair_heads_step * a.steps / (e_ms / 1e3), "unit": UNIT,
                       "h2d_bytes_per_step": len(runs) * hq.numel() * hq.element_size(),
                       "d2h_bytes_per_step": ho.numel() * ho.element_size(), "ms_per_step": e_ms / a.steps}
    else:
        line["e2e"] = None
    if rank == 0 and world == 1 and not a.no_cpu_baseline:
        import oracle

        oracle.set_threads(os.cpu_count() or 1)
        ph, secs, steps = oracle_decode_sample(w, a.cpu_seconds, 5)
        line["cpu_baseline"] = {"value": ph / secs, "unit": UNIT, "cores": oracle.get_threads(), "kind": "oracle",
                                "sample": f"{steps} decode steps of layer 0 (random run and token), {ph} pair-heads "
                                          f"in {secs:.1f} s"}
    for an in anchors:
        an.free()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


# ----------------------------------------------------------------------------- our arm
def ceilings(ris, w, no_probes):
    """Peaks: MEASURED_PEAKS.json (HBM copy, bf16 GEMM) plus this library's L2 and FFMA probes."""
    peaks = {}
    try:
        peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        pass
    c = {"hbm_gbs": peaks.get("hbm_gbs") or 6800.0, "hbm_source": "measured" if peaks.get("hbm_gbs") else "fallback",
         "tc_tflops": peaks.get("bf16_tflops_sustained") or 1700.0,
         "tc_source": "measured sustained bf16" if peaks.get("bf16_tflops_sustained") else "fallback",
         "tc_burst_tflops": peaks.get("bf16_tflops") or 1900.0}
    c["l2_bytes"] = ris.ris_probe_l2_bytes()
    if not no_probes:
        e = 4 if w["dtype"] == "f32" else 2
        # the gather kernels' working set: rotated K (hi and lo for bf16) and V of one layer
        kv_set = w["N"] * w["Hkv"] * w["D"] * e * (3 if e == 2 else 2)
        c["l2_stream_gbs"] = ris.ris_probe_l2_read(64 << 20, 0)
        c["l2_rows_gbs"] = ris.ris_probe_l2_read(max(1 << 20, min(kv_set, c["l2_bytes"] * 3 // 4)), 1)
        c["l2_rows_set_bytes"] = max(1 << 20, min(kv_set, c["l2_bytes"] * 3 // 4))
        c["ffma_tflops"] = ris.ris_probe_ffma()
    return c


def main():
    a = parse_args()
    rank, world, dist = dist_init()
    if a.impl == "reference":
        if a.w.get("kind") == "decode":
            run_reference_decode(a, rank)
        else:
            run_reference(a, rank)
        return
    if a.w.get("kind") == "decode":
        main_decode(a, rank, world, dist)
        return

    import torch

    from paper_2607_21927_gb300 import inputs, ris

    w = a.w
    dev = torch.device("cuda", torch.cuda.current_device())
    N, L, Hq, Hkv, D = w["N"], w["layers"], w["Hq"], w["Hkv"], w["D"]
    tdt = torch.float32 if w["dtype"] == "f32" else torch.bfloat16
    e = 4 if w["dtype"] == "f32" else 2
    runs = w["runs"]
    kind, theta, native = w["rope"]
    rope = ris.rope_cfg(ROPE_KINDS[kind], theta, native)
    geom = ris.paper_geometry() if w.get("geometry") == "paper" else None
    if w.get("sampler"):
        geom = ris.mask_opts(sampler=w["sampler"])

    # inputs resident in HBM: one (q, k, v) per layer, layer L drawn from seed L
    qs, ks, vs = [], [], []
    for layer in range(L):
        q, k, v = inputs.make_qkv(N, Hq, Hkv, D, dtype=tdt, seed=layer, outliers=w["outliers"], device=dev)
        qs.append(q)
        ks.append(k)
        vs.append(v)
    per_seed = bool(w.get("per_seed"))
    oshape = lambda ns: (ns, N, Hq, D) if per_seed else (N, Hq, D)  # noqa: E731
    outs = [[torch.empty(oshape(ns), dtype=tdt, device=dev) for _ in range(L)] for (_, _, _, ns) in runs]
    stream = torch.cuda.current_stream()
    # rows-kv: each rank keeps only its own rows of every layer's q, k and v (for each run's
    # balanced partition, a pure function of the mask that every rank derives alike) and
    # all-gathers K and V per layer inside the step
    local = {}
    if a.shard == "rows-kv":
        from paper_2607_21927_gb300 import shard

        for ri, (name, mode, dens, ns) in enumerate(runs):
            m = ris.ris_mask_generate(N, Hkv, mode, dens, list(range(ns)), opts=geom, per_seed=per_seed)
            b = ris.ris_mask_row_split(m, world)
            m.free()
            r0, r1 = b[rank], b[rank + 1]
            local[ri] = (b, [qs[l][r0:r1].clone() for l in range(L)], [ks[l][r0:r1].clone() for l in range(L)],
                         [vs[l][r0:r1].clone() for l in range(L)],
                         [torch.empty((r1 - r0, Hq, D), dtype=tdt, device=dev) for _ in range(L)])
    pairs, design, suffix = {}, {}, {}
    mask_events = []  # (run, start, mask built, layers done) events of each run while `timing` is set
    timing = [False]

    def step():
        for ri, (name, mode, dens, ns) in enumerate(runs):
            if timing[0]:
                mask_events.append((name,) + tuple(torch.cuda.Event(enable_timing=True) for _ in range(3)))
                mask_events[-1][1].record(stream)
            m = ris.ris_mask_generate(N, Hkv, mode, dens, list(range(ns)), opts=geom, per_seed=per_seed)
            if timing[0]:
                mask_events[-1][2].record(stream)
            mi = m.info()
            pairs[name] = mi.n_pairs
            design[name] = ris.ris_attention_design(m, tdt, D)
            # the dense-suffix split attends the rows' dense suffixes (Structural blocks, local
            # window) on the tiles, not by gathering
            suffix[name] = mi.suffix_pairs * mi.n_masks if design[name] == 4 else 0
            if a.shard == "rows-kv":
                b, ql, kl, vl, ol = local[ri]
                for layer in range(L):
                    if world > 1:
                        kf, vf = shard.kv_allgather(kl[layer], vl[layer], b)
                    else:
                        kf, vf = kl[layer], vl[layer]
                    ris.ris_attention_masked_local(m, b[rank], b[rank + 1], ql[layer], kf, vf, out_rows=ol[layer],
                                                   rope=rope)
            elif a.shard == "rows" and world > 1:
                # every rank builds the same mask and attends its own balanced range of rows
                b = ris.ris_mask_row_split(m, world)
                for layer in range(L):
                    ris.ris_attention_masked_rows(m, b[rank], b[rank + 1], qs[layer], ks[layer], vs[layer],
                                                  outs[ri][layer], rope=rope)
            else:
                for layer in range(L):
                    ris.ris_attention_masked(m, qs[layer], ks[layer], vs[layer], rope=rope, out=outs[ri][layer])
            if timing[0]:
                mask_events[-1][3].record(stream)
            m.free()

    for _ in range(a.warmup):
        step()
    torch.cuda.synchronize()
    ceil = ceilings(ris, w, a.no_probes)
    torch.cuda.synchronize()

    # ---- device-timed region
    import tempfile

    clocks_path = os.path.join(tempfile.gettempdir(), f"ris_bench_clocks_{os.getpid()}.csv")
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.reset_peak_memory_stats(dev)
    ris.ris_memory_stats(reset_high_water=True)
    barrier(dist)
    torch.cuda.synchronize()
    ris.ris_kernel_timer_enable(True)
    n0 = ris.ris_launch_count()
    with ClockSampler(clocks_path) as clk:
        timing[0] = True
        ev0.record(stream)
        for _ in range(a.steps):
            step()
        ev1.record(stream)
        torch.cuda.synchronize()
        timing[0] = False
    launches = ris.ris_launch_count() - n0
    k_ms, k_n, k_each = ris.ris_kernel_timer_samples()
    ris.ris_kernel_timer_enable(False)
    barrier(dist)
    elapsed_ms = max_over_ranks(ev0.elapsed_time(ev1), dist)
    lib_cur, lib_high = ris.ris_memory_stats()
    torch_high = torch.cuda.max_memory_allocated(dev)

    mask_ms = max_over_ranks(sum(e0.elapsed_time(e1) for _, e0, e1, _ in mask_events) / a.steps, dist)
    layers_ms = {}  # per run: its layers' device time per step (RoPE + attention)
    for name, _, e1, e2 in mask_events:
        layers_ms[name] = layers_ms.get(name, 0.0) + e1.elapsed_time(e2) / a.steps
    total_pairs = sum(pairs.values())
    pair_heads_step = total_pairs * L * Hq
    strong = a.shard in ("rows", "rows-kv") and world > 1  # the ranks share one workload
    value = (1 if strong else world) * pair_heads_step * a.steps / (elapsed_ms / 1e3)
    ms_step = elapsed_ms / a.steps

    # roofline of the attention kernel over the timed region: algorithmic bytes (gather) or
    # algorithmic FLOPs (tiles) per launch / mean launch time
    launches_per_step = len(runs) * L
    mean_launch_ms = k_ms / max(k_n, 1)
    median_launch_ms = statistics.median(k_each) if k_each else None
    per_run_ms = {}  # launches are recorded run by run within each step, L per run
    if len(k_each) == launches_per_step * a.steps:
        for i, ms_i in enumerate(k_each):
            per_run_ms.setdefault(runs[(i % launches_per_step) // L][0], []).append(ms_i)
    median_per_run = {k: statistics.median(v) for k, v in per_run_ms.items()}
    kinds = sorted(set(design.values()))
    hbm, tc = ceil["hbm_gbs"], ceil["tc_tflops"]
    kv_row_bytes = Hkv * 2 * D * e  # K and V rows of one key, all KV heads
    kv_set = N * Hkv * D * e * (3 if e == 2 else 2)  # rotated K (hi + lo for bf16) and V of a layer
    gather_names = {0: "k_attn_bf16 (register gather)", 2: "k_attn_tile (tcgen05 masked tiles)",
                    3: "k_attn_f32 (fp32 gather)",
                    4: "k_attn_tile suffix pass + k_attn_bf16 (dense-suffix split: Structural blocks / local window "
                       "on the tiles, the rest gathered)"}
    traffic_file = {0: ("attn_bf16.cu",), 2: ("attn_tile.cu",), 4: ("attn_tile.cu", "attn_bf16.cu")}

    def design_roofline(kd, names):
        """Roofline of design kd's kernel over the launches of runs `names`: algorithmic work per
        launch / that kernel's mean CUDA-event launch time in the timed region."""
        each = [t for nm in names for t in per_run_ms.get(nm, [])]
        if each:
            mean_ms, med_ms, n_l = sum(each) / len(each), statistics.median(each), len(each)
        else:  # launch times not attributable to runs: all launches
            mean_ms, med_ms, n_l = mean_launch_ms, median_launch_ms, k_n
        pairs_launch = sum(pairs[nm] for nm in names) / len(names)
        traffic = recorded_traffic(traffic_file[kd], a.workload) if kd in traffic_file else None
        ent = {"kernel": gather_names.get(kd, "?"), "mean_launch_ms": mean_ms, "median_launch_ms": med_ms,
               "launches_timed": n_l, "traffic": traffic}
        if kd == 2:
            achieved = 4 * D * Hq * pairs_launch / (mean_ms / 1e3) / 1e12
            dense = 4 * D * Hq * N * (N + 1) / 2 * (max(r[3] for r in runs if r[0] in names) if per_seed else 1)
            ent.update({"bound": "tensor", "achieved": achieved, "peak": tc, "unit": "TFLOP/s", "frac": achieved / tc,
                        "peak_source": ceil["tc_source"],
                        "flops": "algorithmic: 4 * head_dim * query heads per sampled pair",
                        "design_frac": (dense / (tc * 1e12)) / (mean_ms / 1e3),
                        "design_note": "dense-causal tile FLOPs / sustained bf16 peak over the launch time (the "
                                       "kernel issues 1.5x that at head dim 128: an fp16 score product, two "
                                       "e4m3 score corrections at twice the rate, one fp16 value product)"})
            if rope is not None and w["dtype"] == "bf16":
                # rotated bf16 inputs at head dim 128 (bounds of |q~| |k~| well inside e4m3's range
                # here): per tile pair one fp16 score product, two e4m3 correction products (each
                # half the time of a 16-bit one) and one fp16 value product; at head dim 64, three
                # bf16 score products and the value product
                ent["issued_frac"] = (1.5 if D == 128 else 2.0) * ent["design_frac"]
                ent["issued_note"] = ("issued tensor-core work in 16-bit-equivalent products of 128x128x128 per "
                                      "causal tile pair (3 at head dim 128, 4 at 64) / sustained bf16 peak over the "
                                      "launch time")
        else:
            # gathered pairs: all of them, or with the dense-suffix split all but the suffixes
            # (whose tile pass is inside the launch time: the split's two launches are timed as one)
            gathered = pairs_launch - sum(suffix[nm] for nm in names) / len(names)
            achieved = gathered * kv_row_bytes / (mean_ms / 1e3) / 1e9
            ent.update({"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                        "peak_source": ceil["hbm_source"],
                        "bytes": "algorithmic: K and V rows of every gathered sampled pair, all KV heads"})
            if kd == 4:
                ent["suffix_pairs_per_launch"] = sum(suffix[nm] for nm in names) / len(names)
                ent["note"] = ("time of both launches (suffix pass on the tiles, then the gather); bytes of the "
                               "gathered pairs only")
            if "l2_rows_gbs" in ceil and kv_set < ceil["l2_bytes"]:
                # the K/V working set is L2-resident: the gathered rows are served from L2, so L2 is
                # the bound (HBM carries only the compulsory q/k/v/out traffic, `traffic`)
                ent.update({"bound": "l2", "peak": ceil["l2_rows_gbs"], "frac": achieved / ceil["l2_rows_gbs"],
                            "peak_source": "measured in this run by the library's L2 probe: whole 256-byte rows "
                                           f"at random indices over {ceil['l2_rows_set_bytes'] / 2**20:.0f} MiB "
                                           "(L2 is not in MEASURED_PEAKS.json)",
                            "hbm_peak": hbm, "frac_of_hbm": achieved / hbm,
                            "bytes_read_per_algorithmic_byte": 1.5 if e == 2 else 1.0})
        ent["device_ms_per_step"] = sum(each) / a.steps if each else None
        return ent

    by_design = {}
    for name, kd in design.items():
        by_design.setdefault(kd, []).append(name)
    per_design = {kd: design_roofline(kd, names) for kd, names in by_design.items()}
    if len(kinds) == 1:
        roofline = per_design[kinds[0]]
        roofline["median_launch_ms_per_run"] = median_per_run
    else:
        # several designs in one step: the headline is the design with the most kernel time
        dom = max(per_design, key=lambda kd: per_design[kd]["device_ms_per_step"] or 0.0)
        roofline = dict(per_design[dom])
        roofline["kernel"] = "mixed designs; headline = " + per_design[dom]["kernel"] + " (most kernel time)"
        roofline["median_launch_ms_per_run"] = median_per_run
        roofline["per_design"] = {ris.DESIGNS[kd]: ent for kd, ent in per_design.items()}
    # the sampled-pair roofline: max(sampled FLOPs / tensor peak, min(row, tile) K/V bytes / bandwidth)
    flops = 4 * D * Hq * total_pairs * L
    b_row = total_pairs * L * kv_row_bytes
    b_tile = sum((r[3] if per_seed else 1) for r in runs) * L * (N / 128) * (N / 2) * kv_row_bytes
    in_l2 = N * kv_row_bytes < ceil["l2_bytes"]
    bw = ceil.get("l2_stream_gbs", hbm) if in_l2 else hbm
    t_roof = max(flops / (tc * 1e12), min(b_row, b_tile) / (bw * 1e9))
    clocks = clk.summary(getattr(torch.cuda.get_device_properties(dev), "pci_bus_id", None))

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": a.steps, "warmup": a.warmup,
            "ms_per_step": ms_step, "ms_per_layer": ms_step / (len(runs) * L), "higher_is_better": True,
            "mask_ms_per_step": mask_ms, "layers_ms_per_run": layers_ms,
            "attn_ms_per_layer": (ms_step - mask_ms) / (len(runs) * L),
            "attn_pair_heads_per_s": (1 if strong else world) * pair_heads_step / ((ms_step - mask_ms) / 1e3),
            "scaling": "strong" if strong else "weak", "vs_baseline": None, "dtype": w["dtype"], "data": "synthetic",
            "config": workload_config(a), "pairs_per_mask": pairs,
            "design_per_run": {k: ris.DESIGNS.get(v, v) for k, v in design.items()}, "roofline": roofline,
            "pair_roofline": {"t_roof_ms_per_step": 1e3 * t_roof, "frac": 1e3 * t_roof / ms_step,
                              "bandwidth": ("L2 stream probe" if in_l2 and "l2_stream_gbs" in ceil else "HBM"),
                              "formula": "max(4*D*Hq*pairs / bf16 sustained, min(pairs, (N/128)*(N/2)) * "
                                         "Hkv*2*D*e / bandwidth)"},
            "ceilings": ceil, "clocks": clocks, "gpu_launches": launches,
            "memory": {"library_pool_high_water_bytes": lib_high, "torch_max_allocated_bytes": torch_high,
                       "note": "torch holds every layer's inputs and outputs resident; the library's high-water "
                               "mark is its masks plus per-call scratch"}}

    # ---- end to end through the C ABI with host buffers
    if not a.no_e2e:
        hq = [t.cpu().pin_memory() for t in qs]
        hk = [t.cpu().pin_memory() for t in ks]
        hv = [t.cpu().pin_memory() for t in vs]
        ho = [[torch.empty(oshape(ns), dtype=tdt).pin_memory() for _ in range(L)] for (_, _, _, ns) in runs]
        h2d = sum(t.numel() * t.element_size() for t in hq + hk + hv)
        d2h = sum(t.numel() * t.element_size() for row in ho for t in row)

        # Host transfers overlap the compute: one stream brings the layers' q/k/v in, another
        # takes the outputs out, both ordered against the compute stream with per-layer events.
        # Masks are built on their own stream: the mask call waits for its own kernels (to size
        # the key lists), which on the compute stream would also drain every queued layer at
        # each run boundary and leave the device idle while the host resumes.
        h2d_s, d2h_s, mask_s = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
        in_ready = [torch.cuda.Event() for _ in range(L)]
        layer_free = [torch.cuda.Event() for _ in range(L)]
        out_ready = [[torch.cuda.Event() for _ in range(L)] for _ in runs]
        out_free = [[torch.cuda.Event() for _ in range(L)] for _ in runs]
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
            for ri, (name, mode, dens, ns) in enumerate(runs):
                m = ris.ris_mask_generate(N, Hkv, mode, dens, list(range(ns)), opts=geom, per_seed=per_seed,
                                          stream=mask_s)
                stream.wait_stream(mask_s)
                b = ris.ris_mask_row_split(m, world) if strong else None
                for layer in range(L):
                    stream.wait_event(in_ready[layer])
                    if not first[0]:
                        stream.wait_event(out_free[ri][layer])
                    if strong:
                        ris.ris_attention_masked_rows(m, b[rank], b[rank + 1], qs[layer], ks[layer], vs[layer],
                                                      outs[ri][layer], rope=rope)
                    else:
                        ris.ris_attention_masked(m, qs[layer], ks[layer], vs[layer], rope=rope,
                                                 out=outs[ri][layer])
                    out_ready[ri][layer].record(stream)
                    if ri == len(runs) - 1:
                        layer_free[layer].record(stream)
                    with torch.cuda.stream(d2h_s):
                        d2h_s.wait_event(out_ready[ri][layer])
                        ho[ri][layer].copy_(outs[ri][layer], non_blocking=True)
                        out_free[ri][layer].record(d2h_s)
                mask_s.wait_stream(stream)  # the mask is released after its layers
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
        line["e2e"] = {"value": (1 if strong else world) * pair_heads_step * a.steps / (e_ms / 1e3), "unit": UNIT,
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
