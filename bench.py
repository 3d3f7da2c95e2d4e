#!/usr/bin/env python3
"""Decode benchmark of the TASP compiled sparse path on GB300.

Workload (default): Llama-3-70B shape, one dependency-closed mask at 0.57 active
FLOPs, batch-1 teacher-forced decode at context 4096 on a BF16 KV cache of
synthetic prior tokens, INT8 per-output-channel weights, dense BF16 LM head.
A step is one decode token: every layer's RMSNorm+QKV+RoPE+KV append, split-KV
attention over the retained KV heads, O-projection, gate/up+SiLU*up, down, then
the final norm and the LM head, replayed from one CUDA graph.

Prints one JSON line (ms/token, lower is better) with the per-kernel roofline of
the dominant kernel, an end-to-end figure through the host-buffer C-ABI call,
clock samples, and the CPU oracle timed on the host as a baseline.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config 1|2|3]
                    [--dense | --mask groups|qheads] [--quant-group 128]
                    [--workload decode|prefill|mixed|spectral] [--prompt T] [--union] [--layers L]

The default decode line also carries the other workloads' figures (prefill of a 2,048-token
prompt, the 16-turn union step) under "other_workloads" (--no-other-workloads skips them).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "decode ms/token (70B-shape, 43% mask, bs1); achieved HBM GB/s vs ~8 TB/s"
# DRAM traffic over algorithmic bytes of one launch, from one ncu capture of the kernel
# (dram__bytes_read.sum + dram__bytes_write.sum of a 70B-width gate/up launch with 18,432
# kept channels: 306,268,672 B against 302,137,344 algorithmic). Re-taken whenever the
# kernel changes.
TRAFFIC_PER_ALGORITHMIC = {"gate_up": 306268672 / 302137344}
PAPER_CONTEXT = {"ms_per_token_sparse": 31.3, "ms_per_token_dense": 45.2,
                 "hardware": "1x A100 80GB SXM, real Llama-3-70B, groupwise INT8, ~2k context"}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=3, choices=[1, 2, 3])
    ap.add_argument("--dense", action="store_true", help="time the dense fallback plan instead of the mask")
    ap.add_argument("--mask", choices=["groups", "qheads"], default="groups",
                    help="decode: whole GQA groups (the benchmark masks) or query-head candidates with KV closure")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--workload", choices=["decode", "prefill", "mixed", "spectral"], default="decode",
                    help="decode (the headline metric), the prefill of one prompt on the 8B shape, the spectral "
                         "descriptors of one 70B-shape layer, or "
                         "mixed-turn serving (70B shape, 16 turns over the dense plan and five masks)")
    ap.add_argument("--union", action="store_true",
                    help="mixed workload: one union-of-masks step for all turns (every weight row read once "
                         "for all plans) instead of one weight pass per plan group")
    ap.add_argument("--panels", choices=["row-indexed", "compact"], default="row-indexed",
                    help="mixed workload: Q/K/V and gate/up panels as row maps into the shared store "
                         "(zero copy) or materialized copies")
    ap.add_argument("--prompt", type=int, default=2048, help="prefill prompt length")
    ap.add_argument("--quant-group", type=int, default=0,
                    help="groupwise INT8 store with one BF16 scale per this many input columns (Table 1: 128)")
    ap.add_argument("--no-other-workloads", action="store_true",
                    help="decode: skip the short prefill and mixed-turn runs attached to the line")
    ap.add_argument("--layers", type=int, default=0,
                    help="keep the workload's widths but only this many layers (small cases for ncu captures)")
    return ap.parse_args()


def measured_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


# ------------------------------------------------------------------ distributed plumbing
def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, v):
    if world == 1:
        return v
    import torch
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ clocks
class ClockSampler:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join(tempfile.gettempdir(), f"tasp_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-lms", "100", "-i", str(self.gpu)], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, smax, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.remove(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ workload
def workload(args):
    import dataclasses
    wl = synth.CONFIGS[args.config]
    if args.layers:
        sh = dataclasses.replace(wl.shape, L=args.layers)
        wl = dataclasses.replace(wl, shape=sh, name=f"{wl.name}_{args.layers}layers")
    if args.quant_group:
        sh = dataclasses.replace(wl.shape, quant_group=args.quant_group)
        wl = dataclasses.replace(wl, shape=sh, name=f"{wl.name}_int8g{args.quant_group}")
    return wl, wl.shape, wl.masks[0]


def block_bounds(K: int, n: int = 5) -> list:
    """Step indices that cut K timed steps into min(n, K) consecutive blocks (the paper reports
    latency as mean and spread over five timing blocks); strictly increasing, first 0, last K."""
    nb = max(1, min(n, K))
    return [i * K // nb for i in range(nb + 1)]


def kv_bytes(plan_dims, dh, T):
    """KV bytes of one step at context T (keys+values read for T positions, one position written)."""
    m = sum(dm[0] for dm in plan_dims)
    return m * 2 * T * dh * 2 + m * 2 * dh * 2


def gemv_bytes(shape, plan_dims):
    """Algorithmic bytes per launch kind, summed over layers (weights, scales, activations in/out)."""
    d, dh, g = shape.d, shape.dh, shape.Hq // shape.Hkv
    b = {"qkv": 0, "o_proj": 0, "gate_up": 0, "down": 0}
    for dm in plan_dims:  # (kept KV groups, kept channels[, kept query heads])
        m_kv, c = dm[0], dm[1]
        m_q = dm[2] if len(dm) > 2 else m_kv * g
        rows = (m_q + 2 * m_kv) * dh
        b["qkv"] += rows * d + rows * 4 + d * 4 + d * 4 + m_q * dh * 4 + m_kv * 2 * dh * 2
        if m_kv:
            b["o_proj"] += d * m_q * dh + d * 4 + m_q * dh * 4 + 2 * d * 4
        if c:
            b["gate_up"] += 2 * c * d + 2 * c * 4 + d * 4 + d * 4 + c * 4
            b["down"] += d * c + d * 4 + c * 4 + 2 * d * 4
        G = getattr(shape, "quant_group", 0)
        if G:  # BF16 group scales: 2 bytes per G weights
            b["qkv"] += 2 * rows * (d // G)
            b["o_proj"] += 2 * d * (m_q * dh // G)
            b["gate_up"] += 2 * 2 * c * (d // G)
            b["down"] += 2 * d * (c // G)
    b["lm_head"] = shape.vocab * d * 2 + d * 4 + shape.vocab * 4
    return b


# ------------------------------------------------------------------ CPU oracle baseline
def oracle_bench_mask(shape, recipe, qheads=False, dense=False):
    """The oracle's compiled mask for the decode workload: whole GQA groups, or query-head
    candidates with KV closure (or everything kept, for the dense fallback)."""
    from oracle import maskc
    if dense:
        return maskc.all_keep(shape)
    tg = synth.layer_target_u24(recipe.mask_seed, shape.L)
    if qheads:
        sc = synth.mask_scores_u32(recipe.mask_seed, shape.L, shape.Hq + shape.n_chan_units)
        return maskc.compile_mask_qheads(shape, sc, tg, recipe.budget, recipe.r_lo, recipe.r_hi)
    sc = synth.mask_scores_u32(recipe.mask_seed, shape.L, shape.n_units)
    return maskc.compile_mask(shape, sc, tg, recipe.budget, recipe.r_lo, recipe.r_hi)


def cpu_oracle_sample(shape, recipe, wl, n_steps, layers=(0, None), lm_rows=1024, qheads=False, dense=False):
    """Time the oracle's decode arithmetic on host cores for a bounded sample.

    Sample: the given layers of the masked model (weights regenerated and
    dequantized once, outside the timing, like the GPU's resident store), one
    decode step each per timed step, plus a slice of LM-head rows; scaled to all
    layers and the full vocabulary. Returns (ms/token per step list, info).
    """
    from oracle import forward, weights
    mask = oracle_bench_mask(shape, recipe, qheads, dense)
    layers = [l if l is not None else shape.L - 1 for l in layers]
    layers = sorted(set(layers))
    t0 = time.perf_counter()
    W, KV = [], []
    for l in layers:
        lq = weights.gen_layer(shape, l)
        W.append(weights.dense_zeroed(shape, lq, mask.keep_groups[l], mask.keep_chans[l],
                                      keep_qheads=mask.qheads(shape, l)))
        KV.append(forward.prior_cache(shape, l, wl.kv_seed, wl.t_prior))
    lm = weights.lm_head_f32(shape, 0, lm_rows) if shape.vocab else None
    gf = weights.gamma_final(shape)
    regen_s = time.perf_counter() - t0
    x = synth.probe_f32(1, 0, shape.d, 4.0)
    per_step = []
    for _ in range(n_steps):
        t = time.perf_counter()
        for (Wl, (Kc, Vc)) in zip(W, KV):
            forward.layer_step(shape, Wl, x, Kc, Vc, wl.t_prior)
        tl = time.perf_counter() - t
        t = time.perf_counter()
        if lm is not None:
            xn = forward.rmsnorm(x, gf, shape.eps)
            _ = lm @ xn
        tlm = time.perf_counter() - t
        per_step.append(1e3 * (tl * shape.L / len(layers) + (tlm * shape.vocab / lm_rows if lm is not None else 0)))
    threads = None
    try:
        from threadpoolctl import threadpool_info
        threads = max((i.get("num_threads", 1) for i in threadpool_info()), default=None)
    except Exception:
        pass
    info = {"kind": "oracle", "cores": os.cpu_count(), "blas_threads": threads,
            "sample": f"layers {layers} of {shape.L} (one decode step each, context {wl.t_prior}) + "
                      f"{lm_rows} of {shape.vocab} LM-head rows, scaled to the full model; weights regenerated "
                      f"once outside timing ({regen_s:.1f} s)",
            "regen_s": round(regen_s, 2)}
    return per_step, info


def decode_config(wl, args, ratio, world):
    """The decode workload's config, the same on both arms: the prior context is the workload's
    (each timed step adds one token to it)."""
    qh = getattr(args, "mask", "groups") == "qheads" and not args.dense
    return {"workload": wl.name + ("_dense" if args.dense else "") + ("_qheads" if qh else ""),
            "mask": "all-keep dense fallback" if args.dense else
            f"greedy dependency-closed{' (query-head candidates)' if qh else ''}, active-FLOP ratio {ratio:.4f}",
            "context": wl.t_prior, "batch": 1, "parallelism": "replicas" if world > 1 else "single GPU",
            "l2": "inputs larger than L2 (each step streams the whole plan's weights)"}


# ------------------------------------------------------------------ reference arm (the oracle)
def run_reference(args):
    world, rank, _ = dist_setup(args)
    if rank != 0:
        return
    wl, shape, recipe = workload(args)
    qh = args.mask == "qheads"
    per_step, info = cpu_oracle_sample(shape, recipe, wl, args.warmup + args.steps, qheads=qh, dense=args.dense)
    if args.dense:
        ratio = 1.0
    else:
        m = oracle_bench_mask(shape, recipe, qh)
        ratio = m.info["total_flops"] / m.info["dense_flops"]
    timed = per_step[args.warmup:]
    v = float(np.mean(timed))
    info["value"] = v
    info["unit"] = "ms/token"
    out = {"impl": "reference", "metric": METRIC, "value": v, "unit": "ms/token", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": v, "higher_is_better": False,
           "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
           "config": decode_config(wl, args, ratio, world),
           "cpu_baseline": info,
           "e2e": {"value": v, "unit": "ms/token", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# ------------------------------------------------------------------ our arm
def run_ours(args):
    import torch

    world, rank, local = dist_setup(args)
    torch.cuda.set_device(local)
    from paper_2609_29499_gb300 import build
    if rank == 0 or world == 1:
        build.build()
    barrier(world)
    from paper_2609_29499_gb300 import tasp
    tasp.load()

    wl, shape, recipe = workload(args)
    K, Wm = args.steps, args.warmup
    t0 = time.perf_counter()
    if args.dense:
        plan = tasp.Plan(shape, tasp.all_keep_mask())
    elif args.mask == "qheads":  # query-head candidates with KV closure (Sec. 3.3, Table 1)
        sc = synth.mask_scores_u32(recipe.mask_seed, shape.L, shape.Hq + shape.n_chan_units)
        tg = synth.layer_target_u24(recipe.mask_seed, shape.L)
        plan = tasp.Plan(shape, tasp.greedy_qhead_mask(sc, tg, recipe.budget, recipe.r_lo, recipe.r_hi))
    else:
        sc = synth.mask_scores_u32(recipe.mask_seed, shape.L, shape.n_units)
        tg = synth.layer_target_u24(recipe.mask_seed, shape.L)
        plan = tasp.Plan(shape, tasp.greedy_mask(sc, tg, recipe.budget, recipe.r_lo, recipe.r_hi))
    setup_s = time.perf_counter() - t0
    info = plan.info()
    dims = [plan.layer_dims(l) + (plan.layer_qheads(l),) for l in range(shape.L)]
    extra = 4
    e2e_steps = 0 if args.no_e2e else K
    sess = tasp.Session(plan, wl.t_prior + Wm + K + extra + e2e_steps + 1)
    sess.fill_synthetic(wl.t_prior, wl.kv_seed + rank)
    total_steps = Wm + K + 1
    xb = synth.step_inputs_bf16(wl.x_seed + rank, total_steps, 1, shape.d)
    x = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
    logits = torch.empty((1, shape.vocab), dtype=torch.float32, device="cuda") if shape.vocab else None
    hidden = torch.empty((1, shape.d), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()

    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    for t in range(Wm):
        tasp.decode_step([sess], x[t], hidden, logits)
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    T_start = sess.position
    bounds = block_bounds(K)
    evs = [torch.cuda.Event(enable_timing=True) for _ in bounds]
    evs[0].record(stream)
    nxt = 1
    for t in range(K):
        tasp.decode_step([sess], x[Wm + t], hidden, logits)
        if nxt < len(bounds) and t + 1 == bounds[nxt]:
            evs[nxt].record(stream)
            nxt += 1
    torch.cuda.synchronize()
    barrier(world)
    clocks = sampler.stop()
    ms = evs[0].elapsed_time(evs[-1]) / K
    block_ms = [evs[i].elapsed_time(evs[i + 1]) / (bounds[i + 1] - bounds[i]) for i in range(len(bounds) - 1)]
    ms = max_over_ranks(world, ms)

    # per-kernel durations of one eager step (CUDA events around each launch, same stream)
    prof = tasp.profile_step([sess], x[Wm + K], logits)
    T_mid = T_start + K // 2
    step_bytes = info["weight_bytes_per_token"] + kv_bytes(dims, shape.dh, T_mid + 1)
    gb = gemv_bytes(shape, dims)
    peak, peak_kind = measured_peak()
    kinds = {k: v for k, v in prof.items() if v[1] > 0}
    dominant = max(kinds, key=lambda k: kinds[k][0])
    dur_ms, launches = kinds[dominant]
    per_launch_bytes = gb.get(dominant, 0) / max(1, launches)
    achieved = per_launch_bytes / (dur_ms / launches * 1e-3) / 1e9 if dominant in gb else None
    roofline = {"bound": "hbm", "kernel": dominant, "achieved": round(achieved, 1) if achieved else None,
                "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 4) if achieved else None,
                "peak_source": f"{peak_kind} hbm_gbs (copy bandwidth)",
                "bytes_per_launch": int(per_launch_bytes), "launch_us": round(dur_ms / launches * 1e3, 2),
                "traffic": (int(per_launch_bytes * TRAFFIC_PER_ALGORITHMIC[dominant])
                            if dominant in TRAFFIC_PER_ALGORITHMIC else None),
                "traffic_source": "ncu capture of a 70B-width launch, scaled by algorithmic bytes"}
    step_gbs = step_bytes / (ms * 1e-3) / 1e9
    kernels = {k: {"ms": round(v[0], 4), "launches": v[1],
                   "GB/s": round(gb[k] / (v[0] * 1e-3) / 1e9, 1) if k in gb and v[0] > 0 else None}
               for k, v in kinds.items()}

    # end to end through the host-buffer C-ABI call (pinned host input, logits read back)
    e2e = None
    if not args.no_e2e:
        xh = torch.from_numpy(xb[:K].view(np.int16)).view(torch.bfloat16).pin_memory()
        lh = torch.empty((1, shape.vocab), dtype=torch.float32).pin_memory() if shape.vocab else None
        hh = None if shape.vocab else torch.empty((1, shape.d), dtype=torch.float32).pin_memory()
        tasp.decode_step_host([sess], xh[0], hh, lh)  # records the host-path graph once
        barrier(world)
        te = time.perf_counter()
        for t in range(K - 1):
            tasp.decode_step_host([sess], xh[t + 1], hh, lh)
        e2e_ms = (time.perf_counter() - te) * 1e3 / max(1, K - 1)
        e2e_ms = max_over_ranks(world, e2e_ms)
        e2e = {"value": round(e2e_ms, 4), "unit": "ms/token", "h2d_bytes_per_step": shape.d * 2,
               "d2h_bytes_per_step": (shape.vocab * 4 if shape.vocab else shape.d * 4)}

    launches_per_step = tasp.step_launches([sess], with_logits=logits is not None)
    sess.release()
    plan.release()

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        per_step, cinfo = cpu_oracle_sample(shape, recipe, wl, 3, qheads=args.mask == "qheads", dense=args.dense)
        cinfo["value"] = round(float(np.mean(per_step)), 1)
        cinfo["unit"] = "ms/token"
        cpu = cinfo

    if rank == 0:
        out = {
            "metric": METRIC, "value": round(ms, 4), "unit": "ms/token", "n_gpus": world, "steps": K, "warmup": Wm,
            "ms_per_step": round(ms, 4), "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
            "dtype": "int8w-f32", "data": "synthetic",
            "config": decode_config(wl, args, info['flops_retained'] / info['flops_dense'], world),
            "context_first_timed_step": T_start,
            "tokens_per_s": round(1e3 / ms * world, 2),
            "roofline": roofline,
            "step_roofline": {"bytes_per_token": int(step_bytes), "achieved": round(step_gbs, 1), "peak": peak,
                              "unit": "GB/s", "frac": round(step_gbs / peak, 4),
                              "frac_of_8TBps": round(step_gbs / 8000.0, 4)},
            "kernels_eager_serialised": {
                "note": "one eager step with CUDA events around every launch: no graph, no programmatic "
                        "overlap, so the per-kind sums exceed the graph-replayed step",
                "per_kind": kernels},
            "timing_blocks": {"n": len(block_ms), "ms_per_token": [round(b, 4) for b in block_ms],
                              "std": round(statistics.pstdev(block_ms), 4) if len(block_ms) > 1 else 0.0},
            "e2e": e2e,
            "gpu_launches": launches_per_step * K,
            "clocks": clocks,
            "cpu_baseline": cpu,
            "paper_context": PAPER_CONTEXT,
            "setup_s": round(setup_s, 1),
            "memory": {"store_bytes": int(info["store_bytes"]), "plan_bytes": int(info["panel_bytes"]),
                       "library_bytes": int(tasp.memory_in_use()),
                       "torch_max_allocated_bytes": int(torch.cuda.max_memory_allocated())},
        }
        if world == 1 and not args.no_other_workloads and not args.layers and args.config == 3 and not args.dense:
            out["other_workloads"] = other_workloads(args)
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def measured_tensor_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["bf16_tflops"]), "measured"
    except Exception:
        return 1900.0, "fallback"


def run_prefill(args, emit=True):
    """Configuration 4: prefill of one prompt per turn on the 8B shape, the turns rotating over
    the five masks' plans; each prefill fills its plan-shaped KV cache, which then serves 32
    decode steps on the same plan. Reports ms per prompt and tensor TFLOP/s, with the decode
    steps that follow timed separately."""
    import dataclasses

    import torch
    from paper_2609_29499_gb300 import build
    build.build()
    from paper_2609_29499_gb300 import tasp
    tasp.load()
    wl = synth.CFG4
    sh = wl.shape if not args.layers else dataclasses.replace(wl.shape, L=args.layers)
    if args.quant_group:  # the paper's groupwise store
        sh = dataclasses.replace(sh, quant_group=args.quant_group)
    T, K, Wm = args.prompt, args.steps, args.warmup
    dec_steps = wl.steps
    plans, sessions, embs, flops = [], [], [], []
    g = sh.Hq // sh.Hkv
    for i, r in enumerate(wl.masks):
        sc = synth.mask_scores_u32(r.mask_seed, sh.L, sh.n_units)
        tg = synth.layer_target_u24(r.mask_seed, sh.L)
        pl = tasp.Plan(sh, tasp.greedy_mask(sc, tg, r.budget, r.r_lo, r.r_hi))
        dims = [pl.layer_dims(l) for l in range(sh.L)]
        flops.append((pl.info()["launched_flops"] * T,
                      sum(2 * 2 * m * g * sh.dh * T * (T + 1) // 2 for m, _ in dims)))
        plans.append(pl)
        sessions.append(tasp.Session(pl, T + dec_steps + 1))
        embs.append(torch.from_numpy(synth.prompt_bf16(wl.x_seed, i, T, sh.d).view(np.int16))
                    .view(torch.bfloat16).cuda())
    n = len(plans)
    logits = torch.empty(sh.vocab, dtype=torch.float32, device="cuda")
    for i in range(n):  # set-up: each plan's FP16 panels are made on its first prefill
        sessions[i].prefill_into(embs[i], logits)
    for t in range(Wm):
        sessions[t % n].prefill_into(embs[t % n], logits)
    torch.cuda.synchronize()
    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    stream = torch.cuda.current_stream()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for t in range(K):
        sessions[t % n].prefill_into(embs[t % n], logits)
    ev1.record(stream)
    torch.cuda.synchronize()
    ms = ev0.elapsed_time(ev1) / K
    # the 32 decode steps that follow a prefill, on each plan's freshly prefilled cache
    xb = synth.step_inputs_bf16(wl.x_seed + 7, dec_steps, 1, sh.d)
    x = torch.from_numpy(xb.view(np.int16)).view(torch.bfloat16).cuda()
    for i in range(n):
        sessions[i].prefill_into(embs[i], logits)
        tasp.decode_step([sessions[i]], x[0], None, logits.view(1, -1))  # records the step graph
        sessions[i].prefill_into(embs[i], logits)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(n):
        for t in range(dec_steps):
            tasp.decode_step([sessions[i]], x[t], None, logits.view(1, -1))
    e1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    dec_ms = e0.elapsed_time(e1) / (n * dec_steps)
    # end to end: pinned host embeddings in, last-position logits out, every prompt
    e2e = None
    if not args.no_e2e:
        eh = [e.cpu().pin_memory() for e in embs]
        lh = torch.empty(sh.vocab, dtype=torch.float32).pin_memory()
        ed = torch.empty_like(embs[0])
        torch.cuda.synchronize()
        te = time.perf_counter()
        for t in range(K):
            ed.copy_(eh[t % n], non_blocking=True)
            sessions[t % n].prefill_into(ed, logits)
            lh.copy_(logits, non_blocking=True)
        torch.cuda.synchronize()
        e2e = {"value": round((time.perf_counter() - te) * 1e3 / K, 3), "unit": "ms",
               "h2d_bytes_per_step": T * sh.d * 2, "d2h_bytes_per_step": sh.vocab * 4}
    err = sum(s.device_error() for s in sessions)
    gemm_flops = sum(f[0] for f in flops) / n
    attn_flops = sum(f[1] for f in flops) / n
    peak, kind = measured_tensor_peak()
    tflops = (gemm_flops + attn_flops) / (ms * 1e-3) / 1e12
    for s_ in sessions:
        s_.release()
    for p_ in plans:
        p_.release()
    out = {"metric": f"prefill ms/prompt (8B-shape, 5 masks at 0.57 active FLOPs, {T} tokens)", "value": round(ms, 3),
           "unit": "ms", "n_gpus": 1, "steps": K, "warmup": Wm, "ms_per_step": round(ms, 3),
           "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f16xint8-f32acc",
           "data": "synthetic",
           "config": {"workload": f"llama3_8b_prefill_{T}" + (f"_{args.layers}layers" if args.layers else "") +
                                  (f"_int8g{args.quant_group}" if args.quant_group else ""),
                      "masks": n, "tokens_per_s": round(T / (ms * 1e-3), 1),
                      "l2": "inputs larger than L2 (every prefill streams a plan's FP16 panels, ~8 GB)"},
           "roofline": {"bound": "tensor", "achieved": round(tflops, 1), "peak": peak, "unit": "TFLOP/s",
                        "frac": round(tflops / peak, 4), "peak_source": f"{kind} bf16_tflops (FP16 runs at the same rate)",
                        "flops_gemm": int(gemm_flops), "flops_attention": int(attn_flops), "traffic": None},
           "decode_after_prefill": {"steps_per_plan": dec_steps, "ms_per_token": round(dec_ms, 4),
                                    "context": T + dec_steps},
           "e2e": e2e, "clocks": clocks, "device_error": err,
           "paper_context": {"prefill_ms_2048_sparse": 1326, "prefill_ms_2048_dense": 1814, "hardware": "A100, 70B"}}
    if emit:
        print(json.dumps(out), flush=True)
    return out


def run_mixed(args, emit=True):
    """Mixed-turn serving on the 70B shape: 16 turns, each bound to the dense plan (p = 0.1)
    or one of five masks (seeded), prompts of U[256, 2048] synthetic prior tokens; every
    step decodes one token for every turn, grouped per plan (up to four sessions share a
    weight pass). Reports aggregate tokens/s."""
    import dataclasses

    import torch
    from paper_2609_29499_gb300 import build
    build.build()
    from paper_2609_29499_gb300 import tasp
    tasp.load()
    wl = synth.CFG5
    sh = wl.shape if not args.layers else dataclasses.replace(wl.shape, L=args.layers)
    if args.quant_group:  # the paper's groupwise store
        sh = dataclasses.replace(sh, quant_group=args.quant_group)
    K, Wm = args.steps, args.warmup
    turns = synth.turn_assignment(wl.x_seed, wl.n_turns, len(wl.masks), wl.p_dense, *wl.prompt_lens)
    n = len(turns)
    mode = tasp.PANELS_ROW_INDEXED if args.panels == "row-indexed" else tasp.PANELS_COMPACT
    t0 = time.perf_counter()
    plans = {}
    for pi, _ in turns:
        if pi in plans:
            continue
        if pi == len(wl.masks):
            plans[pi] = tasp.Plan(sh, tasp.all_keep_mask())
        else:
            r = wl.masks[pi]
            sc = synth.mask_scores_u32(r.mask_seed, sh.L, sh.n_units)
            tg = synth.layer_target_u24(r.mask_seed, sh.L)
            plans[pi] = tasp.Plan(sh, tasp.greedy_mask(sc, tg, r.budget, r.r_lo, r.r_hi, mode))
    setup_s = time.perf_counter() - t0
    e2e_steps = 0 if args.no_e2e else K
    sessions = []
    for i, (pi, T) in enumerate(turns):
        s = tasp.Session(plans[pi], T + Wm + K + e2e_steps + 2)
        s.fill_synthetic(T, wl.kv_seed + i)
        sessions.append(s)
    groups = {}
    for i, (pi, _) in enumerate(turns):
        groups.setdefault(pi, []).append(i)
    xb = synth.step_inputs_bf16(wl.x_seed, Wm + K + 1, n, sh.d)
    xg = {pi: torch.from_numpy(np.ascontiguousarray(xb[:, idx]).view(np.int16)).view(torch.bfloat16).cuda()
          for pi, idx in groups.items()}
    lg = {pi: torch.empty((len(idx), sh.vocab), dtype=torch.float32, device="cuda") for pi, idx in groups.items()}
    gs = {pi: [sessions[i] for i in idx] for pi, idx in groups.items()}
    stream = torch.cuda.current_stream()
    if args.union:
        return run_mixed_union(args, tasp, wl, sh, turns, plans, sessions, xb, setup_s, emit)

    def step(t):
        for pi in groups:
            tasp.decode_step(gs[pi], xg[pi][t], None, lg[pi])

    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    for t in range(Wm):
        step(t)
    torch.cuda.synchronize()
    ctx0 = [s.position for s in sessions]
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for t in range(K):
        step(Wm + t)
    ev1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = ev0.elapsed_time(ev1) / K
    tok_s = n / (ms * 1e-3)
    errs = sum(s.device_error() for s in sessions)

    # roofline: per-kernel times of one eager step of every group, bytes from each plan's ledger
    prof_tot, bytes_tot = {}, {}
    step_bytes = 0
    per_group = {}
    for pi, idx in groups.items():
        dims = [plans[pi].layer_dims(l) for l in range(sh.L)]
        passes = (len(idx) + 3) // 4
        gb = gemv_bytes(sh, dims)
        prof = tasp.profile_step(gs[pi], xg[pi][Wm + K], lg[pi])
        for k, (msk, cnt) in prof.items():
            a = prof_tot.setdefault(k, [0.0, 0])
            a[0] += msk
            a[1] += cnt
            if k in gb:
                bytes_tot[k] = bytes_tot.get(k, 0) + gb[k] * passes
        wbytes = plans[pi].info()["weight_bytes_per_token"] * passes
        kvb = sum(kv_bytes(dims, sh.dh, ctx0[i] + K // 2 + 1) for i in idx)
        step_bytes += wbytes + kvb
        per_group[("dense" if pi == len(wl.masks) else f"mask{pi}")] = {"sessions": len(idx),
                                                                         "weight_passes": passes}
    peak, peak_kind = measured_peak()
    kinds = {k: v for k, v in prof_tot.items() if v[1] > 0}
    dominant = max(kinds, key=lambda k: kinds[k][0])
    dur_ms, launches = kinds[dominant]
    per_launch = bytes_tot.get(dominant, 0) / max(1, launches)
    achieved = per_launch / (dur_ms / launches * 1e-3) / 1e9 if dominant in bytes_tot else None
    roofline = {"bound": "hbm", "kernel": dominant, "achieved": round(achieved, 1) if achieved else None,
                "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 4) if achieved else None,
                "peak_source": f"{peak_kind} hbm_gbs (copy bandwidth)", "bytes_per_launch": int(per_launch),
                "launch_us": round(dur_ms / launches * 1e3, 2), "traffic": None}
    step_gbs = step_bytes / (ms * 1e-3) / 1e9

    e2e = None
    if not args.no_e2e:
        xh = {pi: torch.from_numpy(np.ascontiguousarray(xb[:, idx]).view(np.int16)).view(torch.bfloat16).pin_memory()
              for pi, idx in groups.items()}
        lh = {pi: torch.empty((len(idx), sh.vocab), dtype=torch.float32).pin_memory() for pi, idx in groups.items()}
        for pi in groups:
            tasp.decode_step_host(gs[pi], xh[pi][0], None, lh[pi])  # records the host-path graphs once
        te = time.perf_counter()
        for t in range(1, K):
            for pi in groups:
                tasp.decode_step_host(gs[pi], xh[pi][t], None, lh[pi])
        e2e_ms = (time.perf_counter() - te) * 1e3 / max(1, K - 1)
        e2e = {"value": round(n / (e2e_ms * 1e-3), 2), "unit": "tokens/s", "h2d_bytes_per_step": n * sh.d * 2,
               "d2h_bytes_per_step": n * sh.vocab * 4}
    launches = sum(tasp.step_launches(gs[pi], with_logits=True) for pi in groups)
    for s in sessions:
        s.release()
    for p in plans.values():
        p.release()

    cpu = None
    if not args.no_cpu_baseline:
        mean_T = int(round(np.mean([T for _, T in turns])))
        wl_c = dataclasses.replace(wl, t_prior=mean_T)
        per_step, cinfo = cpu_oracle_sample(sh, wl.masks[0], wl_c, 3)
        cinfo["value"] = round(1e3 / float(np.mean(per_step)), 4)
        cinfo["unit"] = "tokens/s"
        cinfo["sample"] += "; the oracle decodes the turns one after another, so tokens/s = 1 / (s per token)"
        cpu = cinfo

    out = {"metric": "mixed-turn decode tokens/s (70B-shape, 16 turns over dense + 5 masks, grouped per plan)",
           "value": round(tok_s, 2), "unit": "tokens/s", "n_gpus": 1, "steps": K, "warmup": Wm,
           "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "int8w-f32", "data": "synthetic",
           "config": {"workload": wl.name + (f"_{args.layers}layers" if args.layers else "") +
                                  (f"_int8g{args.quant_group}" if args.quant_group else ""), "turns": n,
                      "plans": {("dense" if pi == len(wl.masks) else f"mask{pi}"): len(idx)
                                for pi, idx in groups.items()},
                      "prompt_tokens": [T for _, T in turns], "panels": args.panels,
                      "l2": "inputs larger than L2 (each step streams every plan's weights)"},
           "groups": per_group,
           "roofline": roofline,
           "step_roofline": {"bytes_per_step": int(step_bytes), "achieved": round(step_gbs, 1), "peak": peak,
                             "unit": "GB/s", "frac": round(step_gbs / peak, 4)},
           "e2e": e2e, "gpu_launches": launches * K, "clocks": clocks, "cpu_baseline": cpu,
           "device_error": errs, "setup_s": round(setup_s, 1)}
    if emit:
        print(json.dumps(out), flush=True)
    return out


def run_mixed_union(args, tasp, wl, sh, turns, plans, sessions, xb, setup_s, emit=True):
    """The mixed-turn step as one union-of-masks step over all turns: each layer's dense
    panels are read once for every session (tensor-core skinny GEMMs), each session's mask
    applied where its units meet it; the LM head (BF16) is one more skinny GEMM for all turns."""
    import torch
    K, Wm = args.steps, args.warmup
    n = len(turns)
    x = torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).view(torch.bfloat16).cuda()
    lg = torch.empty((n, sh.vocab), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    for t in range(Wm):
        tasp.decode_step_union(sessions, x[t], None, lg)
    torch.cuda.synchronize()
    ctx0 = [s.position for s in sessions]
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for t in range(K):
        tasp.decode_step_union(sessions, x[Wm + t], None, lg)
    ev1.record(stream)
    torch.cuda.synchronize()
    clocks = sampler.stop()
    ms = ev0.elapsed_time(ev1) / K
    tok_s = n / (ms * 1e-3)
    err, launches = tasp.union_status(sessions)
    errs = err + sum(s.device_error() for s in sessions)
    # bytes of one step: every dense panel byte (and row scale) once, the LM head once, every
    # turn's KV cache
    d, qd, df = sh.d, sh.Hq * sh.dh, sh.df
    qkv_rows = (sh.Hq + 2 * sh.Hkv) * sh.dh
    layer_w = qkv_rows * d + d * qd + 2 * df * d + d * df + 4 * (qkv_rows + d + 2 * df + d)
    G = getattr(sh, "quant_group", 0)
    if G:  # BF16 group scales: 2 bytes per G weights
        layer_w += 2 * (qkv_rows * d + d * qd + 2 * df * d + d * df) // G
    lm = sh.vocab * d * 2
    kvb = 0
    for i, (pi, _) in enumerate(turns):
        dims = [plans[pi].layer_dims(l) for l in range(sh.L)]
        kvb += kv_bytes(dims, sh.dh, ctx0[i] + K // 2 + 1)
    step_bytes = sh.L * layer_w + lm + kvb
    peak, peak_kind = measured_peak()
    step_gbs = step_bytes / (ms * 1e-3) / 1e9
    e2e = None
    if not args.no_e2e:
        xh = torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).view(torch.bfloat16).pin_memory()
        lh = torch.empty((n, sh.vocab), dtype=torch.float32).pin_memory()
        xd = torch.empty((n, sh.d), dtype=torch.bfloat16, device="cuda")
        te = time.perf_counter()
        for t in range(K):
            xd.copy_(xh[t], non_blocking=True)
            tasp.decode_step_union(sessions, xd, None, lg)
            lh.copy_(lg, non_blocking=True)
            torch.cuda.current_stream().synchronize()
        e2e_ms = (time.perf_counter() - te) * 1e3 / K
        e2e = {"value": round(n / (e2e_ms * 1e-3), 2), "unit": "tokens/s", "h2d_bytes_per_step": n * sh.d * 2,
               "d2h_bytes_per_step": n * sh.vocab * 4}
    for s in sessions:
        s.release()
    for p in plans.values():
        p.release()
    groups = {}
    for pi, _ in turns:
        groups[pi] = groups.get(pi, 0) + 1
    out = {"metric": "mixed-turn decode tokens/s (70B-shape, 16 turns over dense + 5 masks, union-of-masks step)",
           "value": round(tok_s, 2), "unit": "tokens/s", "n_gpus": 1, "steps": K, "warmup": Wm,
           "ms_per_step": round(ms, 3), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
           "dtype": "int8w-f16", "data": "synthetic",
           "config": {"workload": wl.name + (f"_{args.layers}layers" if args.layers else "") +
                                  (f"_int8g{args.quant_group}" if args.quant_group else "") + "_union", "turns": n,
                      "plans": {("dense" if pi == len(wl.masks) else f"mask{pi}"): c for pi, c in groups.items()},
                      "prompt_tokens": [T for _, T in turns],
                      "l2": "inputs larger than L2 (each step streams the dense panels)"},
           "roofline": None,
           "step_roofline": {"bytes_per_step": int(step_bytes), "achieved": round(step_gbs, 1), "peak": peak,
                             "unit": "GB/s", "frac": round(step_gbs / peak, 4), "peak_source": peak_kind},
           "e2e": e2e, "gpu_launches": launches * K, "clocks": clocks, "cpu_baseline": None,
           "device_error": errs, "setup_s": round(setup_s, 1)}
    if emit:
        print(json.dumps(out), flush=True)
    return out


def run_spectral(args, emit=True):
    """The spectral descriptors of every candidate unit of one 70B-shape layer (64 heads of
    [512, 8192] blocks, 28 channel groups of [3072, 8192]): ms per layer, and the Gram step's
    tensor rate against the measured bf16 peak (FP16 operands run at the same rate)."""
    import torch
    from paper_2609_29499_gb300 import build
    build.build()
    from paper_2609_29499_gb300 import tasp
    tasp.load()
    sh = synth.LLAMA3_70B
    layer = 0
    nh, nc, nu = 4 * sh.dh, 3 * sh.chan_unit, sh.df // sh.chan_unit
    gram_flops = 2 * sh.d * (sh.Hq * nh * nh + nu * nc * nc)
    for _ in range(max(1, args.warmup)):
        tasp.spectral_layer(sh, layer)
    K = max(1, args.steps)
    ph = np.zeros(4)
    t_tot = 0.0
    sampler = ClockSampler(torch.cuda.current_device())
    sampler.start()
    for _ in range(K):
        p = np.zeros(4)
        t0 = time.perf_counter()
        feat, _ = tasp.spectral_layer(sh, layer, phase_ms=p)
        t_tot += time.perf_counter() - t0
        ph += p
    clocks = sampler.stop()
    ph /= K
    ms = t_tot * 1e3 / K
    peak, kind = measured_tensor_peak()
    gram_tf = gram_flops / (ph[1] * 1e-3) / 1e12
    out = {"metric": "spectral descriptors ms/layer (70B-shape, 64 head + 28 channel-group candidates)",
           "value": round(ms, 2), "unit": "ms", "n_gpus": 1, "steps": K, "warmup": args.warmup,
           "higher_is_better": False, "data": "synthetic", "dtype": "f16-gram-f32acc, f32 eigensolver, f64 statistics",
           "config": {"workload": "llama3_70b_spectral_layer", "candidates": int(feat.shape[0])},
           "phases_ms": {"blocks": round(ph[0], 3), "gram": round(ph[1], 3), "eigensolver": round(ph[2], 3),
                         "statistics": round(ph[3], 3)},
           "roofline": {"bound": "tensor", "kernel": "gram (gemm_persist_kernel)", "achieved": round(gram_tf, 1),
                        "peak": peak, "unit": "TFLOP/s", "frac": round(gram_tf / peak, 4),
                        "peak_source": f"{kind} bf16_tflops", "flops": int(gram_flops), "traffic": None,
                        "note": "Gram FLOPs over the Gram launches' summed device time while eight worker "
                                "streams share the GPU (the eigensolver, a library routine, sets the layer time)"},
           "clocks": clocks}
    if emit:
        print(json.dumps(out), flush=True)
    return out


def other_workloads(args):
    """Configurations 4 and 5 measured in the same run as the headline decode (short, bounded):
    the prefill of 2,048-token prompts on the 8B shape over the five masks, and the 16 mixed
    turns on the 70B shape in one union-of-masks step per token. Each entry is the summary of
    that workload's own line (`--workload prefill` / `--workload mixed --union`)."""
    import copy
    res = {}
    for name, fn, kw in (("prefill_8b_2048", run_prefill, dict(workload="prefill", prompt=2048)),
                         ("mixed_70b_16turns_union", run_mixed, dict(workload="mixed", union=True))):
        a = copy.copy(args)
        a.steps, a.warmup, a.no_cpu_baseline, a.layers = 10, 3, True, 0
        for k, v in kw.items():
            setattr(a, k, v)
        t0 = time.perf_counter()
        try:
            d = fn(a, emit=False)
            res[name] = {k: d.get(k) for k in ("metric", "value", "unit", "higher_is_better", "ms_per_step",
                                                 "roofline", "step_roofline", "e2e", "clocks", "config",
                                                 "decode_after_prefill", "device_error") if d.get(k) is not None}
        except Exception as e:  # the headline line must still print
            res[name] = {"error": repr(e)[:300]}
        res[name]["wall_s"] = round(time.perf_counter() - t0, 1)
    return res


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.workload == "prefill":
        run_prefill(args)
    elif args.workload == "mixed":
        run_mixed(args)
    elif args.workload == "spectral":
        run_spectral(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
