#!/usr/bin/env python
"""Training throughput (tokens/s: forward + backward + AdamW) of a FAL decoder
stack on GB300 through libfal's C ABI, with the same library's sequential GPT
baseline, the GEMM roofline fraction, and the fp64 oracle on the host cores.

Default workload: the 1.3B-shaped FAL stack (24 layers, d_model 2048, 16 heads
of 128, d_ff 8192, seq 2048, batch 4, vocab 50257), bf16 with fp32
accumulation, seeded synthetic tokens.  Every step reads > 2.6 GB of bf16
weights plus activations, far above the 129 MB L2, so no flush is needed.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload gpt_1p3b|gpt2_small|gpt2_medium|gpt2_xl] [--variant fal|falplus|gpt]

With N > 1 (torchrun) every rank trains an independent replica on its own GPU
(the path has no data-path collective); value = all ranks' tokens / max time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2510_14614_gb300 import synth  # noqa: E402

METRIC = "train tokens/s on 1 GB300 (FAL vs own GPT baseline); % of dense BF16 peak"
UNIT = "tokens/s"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="gpt_1p3b", choices=[k for k in synth.SHAPES if k != "tiny"])
    ap.add_argument("--variant", default="fal", choices=list(synth.VARIANTS))
    ap.add_argument("--schedule", default="two_stream", choices=["serial", "two_stream"])
    ap.add_argument("--no-baseline", action="store_true", help="skip the same-library GPT baseline")
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--layers", type=int, default=None, help="override depth (small profiling cases only)")
    ap.add_argument("--batch", type=int, default=None, help="override batch (small profiling cases only)")
    return ap.parse_args()


def shape_of(args):
    s = synth.SHAPES[args.workload]
    if args.layers:
        s = s.replace(layers=args.layers, name=f"{s.name}_L{args.layers}")
    if args.batch:
        s = s.replace(batch=args.batch, name=f"{s.name}_B{args.batch}")
    return s


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x, world, torch):
    """The slowest rank's time: replicas run independent steps, the job takes
    as long as its slowest member (max all-reduce; identity on one rank)."""
    if world <= 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank, n, seconds):
    """Whole-job tokens/s of n replicas that each processed tokens_per_rank in
    `seconds` (the max over ranks): weak scaling, no data-path exchange."""
    return tokens_per_rank * n / seconds


def workload_config(s, variant, schedule, n):
    return {
        "workload": f"{s.name} {variant.upper() if variant != 'falplus' else 'FAL+'}: L={s.layers} d_model={s.d_model} "
                    f"heads={s.heads} (head_dim {s.head_dim}) d_ff={s.d_ff} seq={s.seq} batch={s.batch} vocab={s.vocab}",
        "variant": variant,
        "schedule": schedule,
        "global_batch": s.batch * n,
        "seq_len": s.seq,
        "parallelism": f"replicas x{n}" if n > 1 else "single GPU",
        "l2": "inputs larger than L2 (>2.6 GB of weights read per step), no flush",
    }


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return j, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


def gemm_traffic(workload, variant, schedule):
    """DRAM bytes per tcgen05 GEMM launch from the committed ncu launch-list
    summary of this workload (profiles/launches_<workload>_<variant>.md), or
    None when there is none or when the GEMM sources changed since it was
    captured (their SHA-256 is recorded next to the figure)."""
    import hashlib
    import re
    if schedule != "two_stream":
        return None
    path = os.path.join(ROOT, "profiles", f"launches_{workload}_{variant}.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    mb = re.search(r"^gemm_dram_bytes_per_launch:\s*(\d+)", text, re.M)
    mh = re.search(r"^gemm_sources_sha256:\s*([0-9a-f]{64})", text, re.M)
    if not mb or not mh:
        return None
    h = hashlib.sha256()
    for f in ("gemm_tc.cu", "gemm_epi.cuh", "tc_ptx.cuh", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2510_14614_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return int(mb.group(1)) if h.hexdigest() == mh.group(1) else None


# ------------------------------------------------------------------ oracle arm
def oracle_step_sample(s, variant, seed=1234):
    """One fp64 oracle training step (forward, backward, AdamW) on a bounded
    sample of the workload: full width and sequence, one layer, batch 1.
    Returns (seconds, scale) where scale converts the sample's time into the
    time of one full step by the ratio of algorithmic FLOPs."""
    import numpy as np
    from oracle import fal_oracle as O
    sample = s.replace(layers=1, batch=1)
    params = synth.init_params(variant, sample, seed)
    tok, tgt = synth.make_tokens(sample, seed)
    cfg = O.Config.from_shape(variant, sample)
    hp = synth.adamw_hparams()
    decayed = {n for n, _, dec in synth.param_specs(variant, sample) if dec}
    zeros = {k: np.zeros(v.shape) for k, v in params.items()}
    t0 = time.perf_counter()
    _, cache = O.forward(params, cfg, tok, tgt)
    grads = O.backward(params, cfg, cache)
    O.adamw_step(params, grads, zeros, zeros, 1, hp["lr"], hp["beta1"], hp["beta2"], hp["eps"], hp["weight_decay"],
                 decayed)
    dt = time.perf_counter() - t0
    scale = synth.model_flops_per_step(s) / synth.model_flops_per_step(sample)
    return dt, scale


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def run_reference(args, n):
    s = shape_of(args)
    for _ in range(args.warmup):
        oracle_step_sample(s, args.variant)
    times = []
    scale = 1.0
    for _ in range(args.steps):
        dt, scale = oracle_step_sample(s, args.variant)
        times.append(dt * scale)
    ms = statistics.mean(times) * 1e3
    value = s.tokens / (ms / 1e3)
    sample = (f"one step of the fp64 oracle per timed step on 1 of {s.layers} layers, batch 1 of {s.batch}, full width "
              f"and seq; time scaled to the full step by the algorithmic FLOP ratio {scale:.1f}")
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": n, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": workload_config(s, args.variant, args.schedule, n),
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": sample},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# ------------------------------------------------------------------ GPU arm
class ClockSampler:
    """nvidia-smi samples (200 ms) of SM clock and throttle reasons while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.proc = None
        self.index = index

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc:
            time.sleep(0.3)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out = ""
        else:
            self.out = ""

    def summary(self):
        rows = []
        for line in self.out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[4:8]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, r in rows for i in range(4) if r[i].lower().startswith("active")})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


def init_flat_params(model, s, variant, seed, torch):
    """Seeded weights drawn on the device with the recipe of the synthetic-input
    module (N(0, 0.02), out-projections scaled when the shape asks for it,
    LN gamma = 1, beta = 0, zero biases)."""
    import math
    gen = torch.Generator(device=model.device)
    gen.manual_seed(seed)
    flat = torch.zeros(model.n_params, dtype=torch.float32, device=model.device)
    for name, off, n, shape, _ in model.tensors:
        leaf = name.rsplit(".", 1)[-1]
        view = flat[off:off + n]
        if name in ("wte", "wpe") or leaf.startswith("w_"):
            sd = 0.02
            if s.scale_out_proj and leaf in ("w_o", "w_down"):
                sd = 0.02 / math.sqrt(2 * s.layers)
            view.normal_(0.0, sd, generator=gen)
        elif leaf == "g":
            view.fill_(1.0)
    model.set_params(flat)


def time_variant(args, s, variant, schedule, torch, fal, dev, n, world, rank, peaks, with_e2e):
    hp = synth.adamw_hparams()
    cfg = fal.make_config(variant, s.layers, s.d_model, s.heads, s.d_ff, s.seq, s.batch, s.vocab, precision="bf16",
                          schedule=schedule, **hp)
    m = fal.Model(cfg, device=dev)
    init_flat_params(m, s, variant, 1234 + rank, torch)
    tok_np, tgt_np = synth.make_tokens(s, 1234 + rank)
    tok = torch.from_numpy(tok_np).to(dev)
    tgt = torch.from_numpy(tgt_np).to(dev)
    for _ in range(args.warmup):
        m.train_step(tok, tgt, sync=False)
    loss0 = m.loss()
    stream = m.stream_main
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(dev)
    m.profile_enable(True)
    n0 = fal.launch_count()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clk:
        ev0.record(stream)
        for _ in range(args.steps):
            m.train_step(tok, tgt, sync=False)
        ev1.record(stream)
        torch.cuda.synchronize(dev)
    launches = fal.launch_count() - n0
    m.profile_enable(False)
    prof = m.profile_read()
    ms = max_over_ranks(ev0.elapsed_time(ev1) / args.steps, world, torch)
    if world > 1:
        torch.distributed.barrier()
    loss1 = m.loss()
    res = {"ms": ms, "launches": launches / args.steps * args.steps, "prof": prof, "clocks": clk.summary(),
           "loss_first": loss0, "loss_last": loss1}
    if with_e2e:
        # Through the public C ABI with host buffers: pinned token upload, the
        # step, and the loss read back every step.
        tok_h = torch.from_numpy(tok_np).pin_memory()
        tgt_h = torch.from_numpy(tgt_np).pin_memory()
        m.train_step(tok_h, tgt_h, sync=True)
        if world > 1:
            torch.distributed.barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            m.train_step(tok_h, tgt_h, sync=True)
        e2e_s = max_over_ranks((time.perf_counter() - t0) / args.steps, world, torch)
        res["e2e_s"] = e2e_s
        res["h2d"] = tok_h.numel() * 4 * 2
        res["d2h"] = 4
    m.close()
    del m
    torch.cuda.empty_cache()
    return res


def main():
    args = parse()
    world, rank, local = dist_env()
    n = max(world, 1)
    if world > 1:
        import torch.distributed as td
        import torch
        td.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    if args.impl == "reference":
        if rank == 0:
            run_reference(args, n)
        return

    import torch
    from paper_2510_14614_gb300 import fal
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA device (the library has no CPU path)")
    torch.cuda.set_device(local)
    dev = torch.device(f"cuda:{local}")
    fal.lib()
    peaks, peak_kind = measured_peaks()
    s = shape_of(args)
    main_res = time_variant(args, s, args.variant, args.schedule, torch, fal, dev, n, world, rank, peaks, True)
    base = None
    if not args.no_baseline and args.variant != "gpt":
        base = time_variant(args, s, "gpt", "serial", torch, fal, dev, n, world, rank, peaks, False)

    tokens = s.tokens * n
    ms = main_res["ms"]
    value = job_throughput(s.tokens, n, ms / 1e3)
    flops = synth.model_flops_per_step(s)
    peak_burst = peaks.get("bf16_tflops", 1900.0)
    peak_sus = peaks.get("bf16_tflops_sustained", 1700.0)
    mfu = flops / (ms / 1e3) / 1e12
    prof = main_res["prof"]
    gemm_tflops = prof["gemm_flops"] / (prof["gemm_ms"] / 1e3) / 1e12 if prof["gemm_ms"] > 0 else None
    attn_tflops = prof["attn_flops"] / (prof["attn_ms"] / 1e3) / 1e12 if prof["attn_ms"] > 0 else None
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": n, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded uniform token ids, N(0,0.02) weights)",
        "config": workload_config(s, args.variant, args.schedule, n),
        "model_tflops": mfu,
        "frac_of_peak": {"burst": mfu / peak_burst, "sustained": mfu / peak_sus, "peak_kind": peak_kind},
        "roofline": {
            "kernel": "gemm_tc2_kernel (tcgen05 GEMM on CTA pairs, all launches of the timed steps)",
            "bound": "tensor", "achieved": gemm_tflops, "peak": peak_sus, "unit": "TFLOP/s",
            "frac": (gemm_tflops / peak_sus) if gemm_tflops else None,
            "traffic": gemm_traffic(args.workload if args.layers is None and args.batch is None else "",
                                    args.variant, args.schedule),
            "traffic_unit": "DRAM bytes per launch (ncu launch list of this workload, profiles/)",
            "peak_kind": f"{peak_kind} bf16_tflops_sustained (kernel timed inside a long step)",
            "launches_per_step": prof["gemm_launches"] / args.steps,
            "time_share_of_step": prof["gemm_ms"] / (ms * args.steps),
        },
        "attention": {"achieved_tflops": attn_tflops, "ms_per_step": prof["attn_ms"] / args.steps,
                      "launches_per_step": prof["attn_launches"] / args.steps},
        "gpu_launches": int(main_res["launches"]),
        "clocks": main_res["clocks"],
        "loss": {"after_warmup": main_res["loss_first"], "after_timed": main_res["loss_last"]},
    }
    e2e_s = main_res.get("e2e_s")
    out["e2e"] = {"value": tokens / e2e_s, "unit": UNIT, "h2d_bytes_per_step": main_res["h2d"],
                  "d2h_bytes_per_step": main_res["d2h"]}
    if base is not None:
        gv = tokens / (base["ms"] / 1e3)
        out["gpt_baseline"] = {"value": gv, "ms_per_step": base["ms"], "model_tflops": flops / (base["ms"] / 1e3) / 1e12,
                               "schedule": "serial"}
        out["speedup_vs_gpt"] = value / gv
    if rank == 0 and n == 1 and not args.no_cpu:
        dt, scale = oracle_step_sample(s, args.variant)
        cpu_val = s.tokens / (dt * scale)
        out["cpu_baseline"] = {
            "value": cpu_val, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
            "sample": f"one fp64 oracle step (forward, backward, AdamW) on 1 of {s.layers} layers, batch 1, full width "
                      f"and seq ({dt:.1f} s), scaled to the full step by the algorithmic FLOP ratio {scale:.1f}"}
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as td
        td.barrier()
        td.destroy_process_group()


if __name__ == "__main__":
    main()
