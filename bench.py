#!/usr/bin/env python
"""Training throughput (tokens/s: forward + backward + AdamW) of FAL / FAL+
decoder stacks on GB300 through libfal's C ABI, beside the same library's
sequential GPT baseline, with the fraction of the dense BF16 peak, the GEMM
roofline, and the fp64 oracle timed on the host cores.

Headline workload: the 1.3B-shaped FAL stack (24 layers, d_model 2048, 16 heads
of 128, d_ff 8192, seq 2048, batch 4, vocab 50257), two-stream schedule, bf16
operands with fp32 accumulation, seeded synthetic tokens.  Every step reads
> 2.6 GB of bf16 weights plus activations, far above the 129 MB L2, so no
flush is needed between steps.

One JSON line carries, besides the headline (timed with profiling off):
  e2e           the same step through fal_train_step with host token buffers
                and the loss read back every step;
  roofline      the tcgen05 GEMMs' algorithmic FLOPs over their CUDA-event time
                in a separate profiled pass;
  fal_serial    the same FAL stack with both branches on one stream (isolates
                the branch concurrency of Sec. 4.2 from the fused residual GEMM);
  gpt_baseline  the same library's sequential GPT stack on the same shape;
  chunked_head  the headline step with the chunked LM head (head_chunk
                vocabulary columns per chunk: the logits are never stored
                whole), its workspace beside the stored-logits one;
  configs       the other benchmark shapes (GPT-2 small / medium / XL): FAL or
                FAL+ beside GPT, tokens/s and fraction of peak;
  attention_isolated  forward and backward attention kernels timed alone on one
                layer of the headline shape;
  inference     forward-only prefill (App. E: forward step without gradients,
                the time to first token) of FAL and GPT at the headline shape
                and for single requests of 2048 and 1024 tokens;
  cpu_baseline  a measured sample of one fp64 oracle training step (OracleSample).

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
# The other benchmark shapes and the variants each is reported with.
CONFIG_ARMS = (("gpt2_small", ("fal", "gpt")), ("gpt2_medium", ("falplus", "gpt")),
               ("gpt2_xl", ("fal", "falplus", "gpt")))
REF_SEQ = 128          # tokens per timed step of the reference (oracle) arm
CPU_SEQ = 512          # tokens of the oracle step timed for cpu_baseline
HEAD_CHUNK = 8192      # vocabulary columns per chunk of the chunked-LM-head arm


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="gpt_1p3b", choices=[k for k in synth.SHAPES if k != "tiny"])
    ap.add_argument("--variant", default="fal", choices=list(synth.VARIANTS))
    ap.add_argument("--schedule", default="two_stream", choices=["serial", "two_stream"])
    ap.add_argument("--no-baseline", action="store_true", help="skip the GPT and FAL-serial arms of the headline shape")
    ap.add_argument("--no-configs", action="store_true", help="skip the other benchmark shapes")
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle CPU baseline")
    ap.add_argument("--no-inference", action="store_true", help="skip the forward-only prefill arms")
    ap.add_argument("--arm-steps", type=int, default=5, help="timed steps of each extra arm")
    ap.add_argument("--layers", type=int, default=None, help="override depth (small profiling cases only)")
    ap.add_argument("--batch", type=int, default=None, help="override batch (small profiling cases only)")
    return ap.parse_args(argv)


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


def variant_name(v):
    return {"fal": "FAL", "falplus": "FAL+", "gpt": "GPT"}[v]


def workload_config(s, variant, schedule, n):
    return {
        "workload": f"{s.name} {variant_name(variant)}: L={s.layers} d_model={s.d_model} heads={s.heads} "
                    f"(head_dim {s.head_dim}) d_ff={s.d_ff} seq={s.seq} batch={s.batch} vocab={s.vocab}",
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
            return json.load(f), "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


def gemm_traffic(s, variant, schedule):
    """Average DRAM bytes per tcgen05 GEMM launch of one full training step of
    this workload, from the committed small-case ncu capture
    (profiles/gemm_traffic_<workload>_<variant>.md: every GEMM launch of one
    step of the same stack at depth 2, scaled to the full depth there), or None
    when there is none, when the workload is not the one captured, or when the
    GEMM sources changed since (their SHA-256 is recorded next to the figure)."""
    import hashlib
    import re
    path = os.path.join(ROOT, "profiles", f"gemm_traffic_{s.name}_{variant}.md")
    if schedule != "two_stream" or not os.path.exists(path):
        return None
    text = open(path).read()
    mb = re.search(r"^gemm_dram_bytes_per_launch_full_step:\s*(\d+)", text, re.M)
    mh = re.search(r"^gemm_sources_sha256:\s*([0-9a-f]{64})", text, re.M)
    if not mb or not mh:
        return None
    h = hashlib.sha256()
    for f in ("gemm_tc.cu", "gemm_epi.cuh", "tc_ptx.cuh", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2510_14614_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return int(mb.group(1)) if h.hexdigest() == mh.group(1) else None


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ------------------------------------------------------------------ oracle
class OracleSample:
    """A measured, bounded sample of one training step of the stack `s`, run by
    the fp64 oracle as it stands: forward and backward of `batch` sequences of
    `seq` tokens at the full depth and width, plus AdamW on the same fraction
    f = (batch * seq) / (s.batch * s.seq) of every parameter tensor (a
    different slice of rows each call).  Every part of the step is thus timed
    on f of its work, so tokens / time is the oracle's throughput on the
    workload, apart from the causal attention, whose per-token cost grows with
    the sequence (under 2 % of the FLOPs at the benchmark sequences).  The
    seeded inputs are drawn once, and the parameters are held in fp64 so the
    oracle's own conversion is the identity."""

    def __init__(self, s, variant, batch, seq, seed=1234):
        import numpy as np
        from oracle import fal_oracle as O
        self.O, self.np = O, np
        self.sample = s.replace(batch=batch, seq=seq)
        self.frac = self.sample.tokens / s.tokens
        self.params = {k: v.astype(np.float64) for k, v in synth.init_params(variant, self.sample, seed).items()}
        self.tok, self.tgt = synth.make_tokens(self.sample, seed)
        self.cfg = O.Config.from_shape(variant, self.sample)
        self.hp = synth.adamw_hparams()
        self.decayed = {n for n, _, dec in synth.param_specs(variant, self.sample) if dec}
        self.calls = 0

    def __call__(self):
        """Runs the sample; returns its wall time in seconds."""
        O, hp, np = self.O, self.hp, self.np
        nslices = max(1, round(1.0 / self.frac))
        j = self.calls % nslices
        self.calls += 1
        t0 = time.perf_counter()
        _, cache = O.forward(self.params, self.cfg, self.tok, self.tgt)
        grads = O.backward(self.params, self.cfg, cache)
        del cache
        part = {}
        for k, v in self.params.items():
            r = v.shape[0]
            lo, hi = j * r // nslices, (j + 1) * r // nslices
            part[k] = slice(lo, hi)
        sub = lambda d: {k: d[k][part[k]] for k in d}
        zeros = {k: np.zeros_like(v) for k, v in sub(self.params).items()}
        O.adamw_step(sub(self.params), sub(grads), zeros, zeros, 1, hp["lr"], hp["beta1"], hp["beta2"], hp["eps"],
                     hp["weight_decay"], self.decayed)
        return time.perf_counter() - t0

    def describe(self, sec):
        return (f"fp64 oracle on the host cores, measured: forward and backward of the full {self.sample.layers}-layer "
                f"stack at full width on {self.sample.batch} sequence(s) of {self.sample.seq} tokens plus AdamW on the "
                f"same fraction ({self.frac:.4g}) of every parameter tensor: {sec:.2f} s per sample")


def run_reference(args, n):
    """The reference arm: the fp64 oracle on the host cores.  Each step is a
    measured OracleSample of the workload's step on one sequence of REF_SEQ
    tokens; throughput = those tokens over the measured time."""
    s = shape_of(args)
    step = OracleSample(s, args.variant, 1, min(REF_SEQ, s.seq))
    for _ in range(args.warmup):
        step()
    times = [step() for _ in range(args.steps)]
    sec = statistics.mean(times)
    value = step.sample.tokens / sec
    desc = "each timed step: " + step.describe(sec)
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": n, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": workload_config(s, args.variant, args.schedule, n),
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": desc},
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
        self.out = ""

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


def init_flat_params(model, s, seed, torch):
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


class Arm:
    """One model of the library on the device with its resident inputs."""

    def __init__(self, s, variant, schedule, torch, fal, dev, rank, head_chunk=0):
        # The weights are drawn with torch's device RNG, whose kernels torch
        # loads lazily on first use.  When that load happened after the model's
        # ~39 GB workspace had been allocated, every later step of that model ran
        # about 2 % slower (same kernels and launch shapes; 110 W more power, so
        # lower clocks); CUDA_MODULE_LOADING=EAGER removed the difference too.
        # One draw on a tiny tensor before the workspace exists loads them first.
        warm = torch.Generator(device=dev)
        warm.manual_seed(0)
        torch.empty(16, device=dev).normal_(0.0, 1.0, generator=warm)
        hp = synth.adamw_hparams()
        cfg = fal.make_config(variant, s.layers, s.d_model, s.heads, s.d_ff, s.seq, s.batch, s.vocab,
                              precision="bf16", schedule=schedule, head_chunk=head_chunk, **hp)
        self.workspace_bytes = fal.workspace_size(cfg)
        self.s, self.variant, self.schedule, self.torch, self.fal, self.dev = s, variant, schedule, torch, fal, dev
        self.m = fal.Model(cfg, device=dev)
        init_flat_params(self.m, s, 1234 + rank, torch)
        self.tok_np, self.tgt_np = synth.make_tokens(s, 1234 + rank)
        self.tok = torch.from_numpy(self.tok_np).to(dev)
        self.tgt = torch.from_numpy(self.tgt_np).to(dev)

    @staticmethod
    def workspace_of(s, variant, schedule, fal, head_chunk):
        return fal.workspace_size(fal.make_config(variant, s.layers, s.d_model, s.heads, s.d_ff, s.seq, s.batch,
                                                  s.vocab, precision="bf16", schedule=schedule,
                                                  head_chunk=head_chunk, **synth.adamw_hparams()))

    def steps(self, k):
        for _ in range(k):
            self.m.train_step(self.tok, self.tgt, sync=False)

    def timed(self, steps, warmup, world, clocks=False):
        """W untimed steps, then K steps between CUDA events on the library's
        main stream (barrier + synchronize on both sides); max over ranks."""
        torch = self.torch
        self.steps(warmup)
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(self.dev)
        n0 = self.fal.launch_count()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        stream = self.m.stream_main
        clk = ClockSampler(torch.cuda.current_device()) if clocks else None
        if clk:
            clk.__enter__()
        ev0.record(stream)
        self.steps(steps)
        ev1.record(stream)
        torch.cuda.synchronize(self.dev)
        if clk:
            clk.__exit__(None, None, None)
        launches = self.fal.launch_count() - n0
        ms = max_over_ranks(ev0.elapsed_time(ev1) / steps, world, torch)
        if world > 1:
            torch.distributed.barrier()
        out = {"ms": ms, "launches": launches, "loss": self.m.loss()}
        if clk:
            out["clocks"] = clk.summary()
        return out

    def prefill_ms(self, steps, warmup):
        """Forward-only prefill (no loss, no backward state), CUDA events on the
        library's main stream."""
        torch = self.torch
        for _ in range(warmup):
            self.m.prefill(self.tok, sync=False)
        torch.cuda.synchronize(self.dev)
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(self.m.stream_main)
        for _ in range(steps):
            self.m.prefill(self.tok, sync=False)
        ev1.record(self.m.stream_main)
        torch.cuda.synchronize(self.dev)
        return ev0.elapsed_time(ev1) / steps

    def e2e(self, steps, world):
        """Through the public C ABI with host buffers: pinned token upload, the
        step, and the loss read back to the host every step."""
        torch = self.torch
        tok_h = torch.from_numpy(self.tok_np).pin_memory()
        tgt_h = torch.from_numpy(self.tgt_np).pin_memory()
        self.m.train_step(tok_h, tgt_h, sync=True)
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(self.dev)
        t0 = time.perf_counter()
        for _ in range(steps):
            self.m.train_step(tok_h, tgt_h, sync=True)
        sec = max_over_ranks((time.perf_counter() - t0) / steps, world, torch)
        return {"s": sec, "h2d": tok_h.numel() * 4 * 2, "d2h": 4}

    def profiled(self, steps):
        """GEMM and attention launches bracketed by CUDA events on their own
        streams, over `steps` steps (a pass of its own, not the headline's)."""
        self.torch.cuda.synchronize(self.dev)
        self.m.profile_read()
        self.m.profile_enable(True)
        self.steps(steps)
        prof = self.m.profile_read()
        self.m.profile_enable(False)
        return prof

    def shares(self):
        """Every launch of one step on its own CUDA events: time per kind."""
        self.torch.cuda.synchronize(self.dev)
        self.m.profile_read()
        self.m.profile_enable(True, every_launch=True)
        self.steps(1)
        recs = self.m.profile_timeline()
        self.m.profile_read()
        self.m.profile_enable(False)
        per = {}
        for r in recs:
            key = r["label"] or str(r["kind"])
            e = per.setdefault(key, {"launches": 0, "ms": 0.0})
            e["launches"] += 1
            e["ms"] += r["end_ms"] - r["start_ms"]
        span = (max(r["end_ms"] for r in recs) - min(r["start_ms"] for r in recs)) if recs else 0.0
        return {"step_span_ms": span, "per_label": {k: {"launches": v["launches"], "ms": round(v["ms"], 4)}
                                                    for k, v in sorted(per.items(), key=lambda kv: -kv[1]["ms"])}}

    def close(self):
        self.m.close()
        del self.m
        self.torch.cuda.empty_cache()


def arm_summary(s, res, n, peaks):
    flops = synth.model_flops_per_step(s)
    tf = flops / (res["ms"] / 1e3) / 1e12
    return {"value": job_throughput(s.tokens, n, res["ms"] / 1e3), "ms_per_step": res["ms"], "model_tflops": tf,
            "frac_of_burst": tf / peaks.get("bf16_tflops", 1900.0),
            "frac_of_sustained": tf / peaks.get("bf16_tflops_sustained", 1700.0)}


def attention_isolated(s, torch, fal, dev):
    """The attention kernels alone on one layer of the headline shape (CUDA
    events, 3 warm-up and 10 timed launches each)."""
    B, T, H, hd = s.batch, s.seq, s.heads, s.head_dim
    g = torch.Generator(device=dev)
    g.manual_seed(7)
    qkv = torch.randn((B * T, 3 * H * hd), generator=g, device=dev).to(torch.bfloat16)
    dctx = torch.randn((B * T, H * hd), generator=g, device=dev).to(torch.bfloat16)
    ctx, lse = fal.attention_fwd(qkv, B, T, H, hd)

    def clock(fn):
        for _ in range(3):
            fn()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        a.record()
        for _ in range(10):
            fn()
        b.record()
        torch.cuda.synchronize(dev)
        return a.elapsed_time(b) / 10

    fwd_ms = clock(lambda: fal.attention_fwd(qkv, B, T, H, hd))
    bwd_ms = clock(lambda: fal.attention_bwd(qkv, ctx, lse, dctx, B, T, H, hd))
    f_fwd = 2.0 * B * H * T * T * hd  # causal half of 4*B*H*T^2*hd
    return {"shape": f"B={B} T={T} H={H} hd={hd}", "fwd_us": fwd_ms * 1e3, "bwd_us": bwd_ms * 1e3,
            "fwd_tflops": f_fwd / (fwd_ms / 1e3) / 1e12, "bwd_tflops": 2 * f_fwd / (bwd_ms / 1e3) / 1e12,
            "note": "backward includes its D = rowsum(dO*O) pre-pass; FLOPs algorithmic (backward = 2x forward)"}


def main():
    args = parse()
    world, rank, local = dist_env()
    n = max(world, 1)
    if world > 1:
        import torch
        import torch.distributed as td
        td.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    if args.impl == "reference":
        if rank == 0:
            run_reference(args, n)
        if world > 1:
            import torch.distributed as td
            td.destroy_process_group()
        return

    import torch
    from paper_2510_14614_gb300 import fal
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA device (the library has no CPU path)")
    torch.cuda.set_device(local)
    dev = torch.device(f"cuda:{local}")
    fal.lib()
    peaks, peak_kind = measured_peaks()
    peak_burst = peaks.get("bf16_tflops", 1900.0)
    peak_sus = peaks.get("bf16_tflops_sustained", 1700.0)
    s = shape_of(args)
    flops = synth.model_flops_per_step(s)

    # ---- headline (profiling off), end to end, then a separate profiled pass
    arm = Arm(s, args.variant, args.schedule, torch, fal, dev, rank)
    head = arm.timed(args.steps, args.warmup, world, clocks=True)
    e2e = arm.e2e(args.steps, world)
    prof = arm.profiled(min(args.steps, 3))
    shares = arm.shares() if world == 1 else None
    arm.close()
    ms = head["ms"]
    value = job_throughput(s.tokens, n, ms / 1e3)
    mfu = flops / (ms / 1e3) / 1e12
    gemm_tflops = prof["gemm_flops"] / (prof["gemm_ms"] / 1e3) / 1e12 if prof["gemm_ms"] > 0 else None
    psteps = min(args.steps, 3)
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": n, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded uniform token ids, N(0,0.02) weights)",
        "config": workload_config(s, args.variant, args.schedule, n),
        "model_tflops": mfu,
        "frac_of_peak": {"burst": mfu / peak_burst, "sustained": mfu / peak_sus, "peak_kind": peak_kind},
        "roofline": {
            "kernel": "gemm_tc2_kernel (tcgen05 GEMM on CTA pairs, every launch of the profiled steps)",
            "bound": "tensor", "achieved": gemm_tflops, "peak": peak_sus, "unit": "TFLOP/s",
            "frac": (gemm_tflops / peak_sus) if gemm_tflops else None,
            "frac_of_burst": (gemm_tflops / peak_burst) if gemm_tflops else None,
            "traffic": gemm_traffic(s, args.variant, args.schedule),
            "traffic_unit": "DRAM bytes per launch, average over one full step (small-case ncu capture, profiles/)",
            "peak_kind": f"{peak_kind} bf16_tflops_sustained (kernel timed inside a long step); "
                         f"frac_of_burst against bf16_tflops",
            "launches_per_step": prof["gemm_launches"] / psteps,
            "gemm_ms_per_step": prof["gemm_ms"] / psteps,
            "profiled_steps": psteps,
        },
        "attention_in_step": {"ms_per_step": prof["attn_ms"] / psteps, "launches_per_step": prof["attn_launches"] / psteps,
                              "note": "event time on the side stream while other kernels share the SMs"},
        "gpu_launches": int(head["launches"]),
        "clocks": head["clocks"],
        "loss": {"after_timed": head["loss"]},
        "e2e": {"value": job_throughput(s.tokens, n, e2e["s"]), "unit": UNIT, "h2d_bytes_per_step": e2e["h2d"],
                "d2h_bytes_per_step": e2e["d2h"]},
    }
    if shares:
        out["step_shares"] = shares
    extra = world == 1
    if extra:
        out["attention_isolated"] = attention_isolated(s, torch, fal, dev)
    k, w = args.arm_steps, min(args.warmup, 3)
    if not args.no_baseline and extra:
        if args.variant != "gpt":
            a = Arm(s, args.variant, "serial", torch, fal, dev, rank)
            r = a.timed(k, w, world)
            a.close()
            out["fal_serial" if args.variant == "fal" else f"{args.variant}_serial"] = dict(
                arm_summary(s, r, n, peaks), schedule="serial")
            if args.variant == "fal" and args.schedule == "two_stream":
                out["two_stream_gain"] = r["ms"] / ms
        a = Arm(s, "gpt", "serial", torch, fal, dev, rank)
        r = a.timed(k, w, world)
        a.close()
        out["gpt_baseline"] = dict(arm_summary(s, r, n, peaks), schedule="serial")
        out["speedup_vs_gpt"] = out["gpt_baseline"]["ms_per_step"] / ms
        # the same step with the chunked LM head (logits never stored whole)
        ws_stored = Arm.workspace_of(s, args.variant, args.schedule, fal, 0)
        a = Arm(s, args.variant, args.schedule, torch, fal, dev, rank, head_chunk=HEAD_CHUNK)
        r = a.timed(k, w, world)
        a.close()
        out["chunked_head"] = dict(arm_summary(s, r, n, peaks), schedule=args.schedule, head_chunk=HEAD_CHUNK,
                                   workspace_gib=a.workspace_bytes / 2**30, stored_logits_workspace_gib=ws_stored / 2**30,
                                   vs_stored_logits=ms / r["ms"])
    if not args.no_configs and extra and args.layers is None and args.batch is None:
        cfgs = {}
        for name, variants in CONFIG_ARMS:
            if name == s.name:
                continue
            cs = synth.SHAPES[name]
            row = {}
            for v in variants:
                sched = "two_stream" if v == "fal" else "serial"
                a = Arm(cs, v, sched, torch, fal, dev, rank)
                r = a.timed(k, w, world)
                a.close()
                row[variant_name(v)] = dict(arm_summary(cs, r, n, peaks), schedule=sched)
            for v in variants:
                if v != "gpt":
                    row[f"{variant_name(v)}/GPT"] = row["GPT"]["ms_per_step"] / row[variant_name(v)]["ms_per_step"]
            row["shape"] = (f"L={cs.layers} d_model={cs.d_model} heads={cs.heads} d_ff={cs.d_ff} seq={cs.seq} "
                            f"batch={cs.batch} vocab={cs.vocab}")
            cfgs[name] = row
        out["configs"] = cfgs
        out["configs_note"] = f"{w} warm-up and {k} timed steps per arm; fractions against measured burst / sustained"
    if not args.no_inference and extra and args.layers is None and args.batch is None:
        inf = {}
        for label, shp in (("batch", s), ("request_T2048", s.replace(batch=1, seq=min(2048, s.seq))),
                           ("request_T1024", s.replace(batch=1, seq=min(1024, s.seq)))):
            row = {}
            for v, sched in ((args.variant, args.schedule), ("gpt", "serial")):
                if v in row:
                    continue
                a = Arm(shp, v, sched, torch, fal, dev, rank)
                ms_pf = a.prefill_ms(10, 3)
                a.close()
                row[variant_name(v)] = {"ms": ms_pf, "tokens_per_s": shp.tokens / (ms_pf / 1e3), "schedule": sched}
            if "GPT" in row and variant_name(args.variant) in row and args.variant != "gpt":
                row[f"{variant_name(args.variant)}/GPT"] = row["GPT"]["ms"] / row[variant_name(args.variant)]["ms"]
            row["shape"] = f"batch={shp.batch} seq={shp.seq}"
            inf[label] = row
        out["inference"] = inf
        out["inference_note"] = ("fal_prefill: embedding, every block, final LN and the LM head of each sequence's "
                                 "last position; 3 warm-up and 10 timed calls, CUDA events")
    if rank == 0 and n == 1 and not args.no_cpu:
        cpu = OracleSample(s, args.variant, 1, min(CPU_SEQ, s.seq))
        sec = cpu()
        out["cpu_baseline"] = {"value": cpu.sample.tokens / sec, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                               "sample": cpu.describe(sec)}
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as td
        td.barrier()
        td.destroy_process_group()


if __name__ == "__main__":
    main()
