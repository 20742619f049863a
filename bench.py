#!/usr/bin/env python
"""Benchmark of the UniF-MoE layer forward pass on GB300.

One step = one forward of the whole layer (router, permute, grouped up and
down GEMMs, combine; Sec. III, Eqs. 16-30) over one batch of seeded
synthetic tokens. Default workload: ViT-S-like vision tokens (64 images x 197
tokens, d=384, H=1536 in 8 blocks, 8 upcycled residual experts + 1 shared
expert, bf16), the stand-in for the paper's DeiT-S/DomainBed setting.

Prints one JSON line (rank 0). Multi-GPU (torchrun): every rank runs its own
batch (weak scaling, no data-path collective); value = tokens of all ranks /
max over ranks of the timed device time.

--impl reference times the CPU oracle (the plain fp64 restatement of the
paper) on the host cores instead, on bounded token samples of the same
workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "UniF-MoE layer fwd tokens/s & activated TFLOP/s (% of GB300 bf16 peak), 1 GPU"
UNIT = "tokens/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# Routing variants (the ablations of Table IV and the fixed cumulative-mass
# thresholds): overrides of the layer's thresholds.
ROUTINGS = {
    "adaptive": {},
    "alpha0.4": {"alpha_fixed": 0.4},
    "top2": {"topk_fixed": 2},
    "prefix": {"prefix_blocks": 1},
    "theta0.5": {"beta_fixed": 0.5},
    "theta0.7": {"beta_fixed": 0.7},
    "theta0.9": {"beta_fixed": 0.9},
}


def routing_desc(s):
    parts = []
    if not math.isnan(s.alpha_fixed):
        parts.append("alpha fixed %.2f" % s.alpha_fixed)
    if not math.isnan(s.beta_fixed):
        parts.append("beta fixed %.2f" % s.beta_fixed)
    if s.topk_fixed:
        parts.append("top-%d residual experts" % s.topk_fixed)
    if s.prefix_blocks:
        parts.append("prefix block selection")
    return ", ".join(parts) if parts else "adaptive (Eqs. 18-27)"


def workload_desc(s, T_valid):
    return {"workload": "%s: %d tokens (%d valid), d=%d, H=%d in B=%d blocks of %d, K=%d residual "
                        "experts + 1 shared, %s" % (s.name, s.tokens, T_valid, s.d_model, s.d_ff,
                                                    s.n_blocks, s.block_width, s.n_experts, s.dtype),
            "tokens": s.tokens, "valid_tokens": T_valid, "d_model": s.d_model, "d_ff": s.d_ff,
            "n_blocks": s.n_blocks, "n_experts": s.n_experts,
            "thresholds": routing_desc(s)}


# ----------------------------------------------------------------- ranks

def rank_token_seed(s, rank):
    """Token seed of a rank: rank 0 draws the workload's own batch; every other
    rank an independent batch of the same shape (weak scaling: each rank owns
    its tokens, the layer weights are the same everywhere)."""
    return None if rank == 0 else s.index * 1000 + 1 + 7919 * rank


def max_over_ranks(value, dist=None, device="cpu"):
    """The largest value over all ranks (the slowest rank sets the job time)."""
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value, dist=None, device="cpu"):
    """The sum of a per-rank count over all ranks."""
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def job_throughput(total_tokens, ms_per_step):
    """Whole-job tokens/s: the valid tokens all ranks processed in one step
    over the slowest rank's step time."""
    return total_tokens / (ms_per_step / 1e3)


def measured_traffic(workload, kernel):
    """DRAM bytes per launch of `kernel` from the committed ncu capture, or
    None when there is none or the kernel sources changed since it was taken."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    rec = json.load(open(path)).get(workload, {})
    if isinstance(rec.get(kernel), dict):  # a kernel with its own record and sources
        rec = dict(rec[kernel], **{kernel: rec[kernel].get("bytes")})
    csrc = os.path.join(ROOT, "paper_2608_10392_gb300", "csrc")
    h = hashlib.sha1()
    for f in rec.get("sources", []):
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(fh.read())
    if rec.get("kernel_source_sha1") != h.hexdigest():
        return None
    return rec.get(kernel)


# ----------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, interval_ms=50):
        import tempfile
        self.proc = None
        fd, self.path = tempfile.mkstemp(prefix="unif_moe_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", str(interval_ms)],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self, gpu_index=0):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        with open(self.path) as f:
            lines = f.read().splitlines()
        os.unlink(self.path)
        for line in lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9 or not parts[0].isdigit() or int(parts[0]) != gpu_index:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, v in zip(("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                                "sw_power_cap"), parts[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ----------------------------------------------------------------- oracle

class OracleRunner:
    """The CPU oracle, as it stands, on the first `tokens` token slots of a
    workload (inputs converted to fp64 once, outside the timing)."""

    def __init__(self, wl, train=False):
        import oracle
        s = wl.spec
        self.o, self.wl, self.s = oracle, wl, s
        self.train = train
        if train:  # a training step: the backward too, for a seeded dL/dy
            import numpy as np
            self.dy = np.random.default_rng(17).standard_normal((s.tokens, s.d_model))
        self.rm = oracle.ROUND_BF16 if s.dtype == "bf16" else oracle.ROUND_F32
        self.th = oracle.Thresholds(s.tau, s.alpha_fixed, s.beta_fixed, s.topk_fixed,
                                    s.prefix_blocks)
        self.wu, self.wd = oracle._f64(wl.w_up), oracle._f64(wl.w_down)
        self.wr, self.xa = oracle._f64(wl.w_router), oracle._f64(wl.x)

    def time(self, tokens, repeat=1):
        m = None if self.wl.mask is None else self.wl.mask[:tokens]
        x = self.xa[:tokens]
        t0 = time.perf_counter()
        for _ in range(repeat):
            _, r = self.o.layer(x, self.wr, self.wu, self.wd, self.s.n_blocks, self.th, m,
                                self.wl.router_bias, self.rm)
            if self.train:
                self.o.backward(x, self.wr, self.wu, self.wd, r.shr_mask, r.expert_mask(),
                                self.s.n_blocks, self.dy[:tokens], self.th, m,
                                self.wl.router_bias)
                self.o.diversity(self.wr)
        dt = time.perf_counter() - t0
        valid = tokens if m is None else int(m.sum())
        return valid * repeat / dt, dt, valid * repeat

    def sample(self, target_s=12.0):
        """At least `target_s` seconds of oracle work: passes over the first
        `tokens` token slots (the whole workload when a pass fits in
        `target_s`, sized from a short probe pass) until the time is spent."""
        T = self.xa.shape[0]
        probe = min(T, 256)
        rate, _, _ = self.time(probe)
        tokens = int(min(T, max(probe, rate * target_s)))
        dt, n, repeat = 0.0, 0, 0
        while dt < target_s:
            _, t, k = self.time(tokens)
            dt, n, repeat = dt + t, n + k, repeat + 1
        return n / dt, dt, n, tokens, repeat


def decision_check(wl, gpu, tokens):
    """The oracle's decisions on the first `tokens` token slots against the
    GPU's (b, k, shared block set, residual expert set): near-ties (oracle
    margin <= 1e-3), tokens whose decisions differ, and those among them
    with a margin above 1e-3."""
    import numpy as np
    import oracle
    s = wl.spec
    rm = oracle.ROUND_BF16 if s.dtype == "bf16" else oracle.ROUND_F32
    th = oracle.Thresholds(s.tau, s.alpha_fixed, s.beta_fixed, s.topk_fixed, s.prefix_blocks)
    m = None if wl.mask is None else wl.mask[:tokens]
    mu = oracle.prototypes(wl.w_up, s.n_blocks, rm)
    r = oracle.route(wl.x[:tokens], wl.w_router, mu, s.n_experts, s.n_blocks, th, m,
                     wl.router_bias)
    valid = np.ones(tokens, bool) if m is None else m.numpy() != 0
    same = ((gpu["b"][:tokens] == r.b) & (gpu["k"][:tokens] == r.k) &
            (gpu["shr"][:tokens] == r.shr_mask) & (gpu["em"][:tokens] == r.expert_mask()))
    near = r.margin.min(axis=1) <= 1e-3
    return {"tokens": int(valid.sum()), "near_ties_margin_le_1e-3": int((near & valid).sum()),
            "decisions_differ": int((~same).sum()),
            "differ_with_margin_gt_1e-3": int((~same & ~near).sum())}


def oracle_cores():
    import oracle
    return oracle.threads()


# ----------------------------------------------------------------- main

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="vit_s")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=50)
    ap.add_argument("--gemm-kernels", default="auto",
                    choices=["auto", "grouped", "streaming", "expert_tile"],
                    help="expert GEMM kernel family (unif_moe_options.gemm_kernels)")
    ap.add_argument("--routing", default="adaptive", choices=sorted(ROUTINGS),
                    help="routing variant (Table IV ablations, fixed thresholds)")
    ap.add_argument("--train", action="store_true",
                    help="time a training step: the forward, then the backward pass with the "
                         "Gram regulariser (Sec. III-E, lambda_div 0.01)")
    ap.add_argument("--sublayer", default="none", choices=["none", "pre", "post"],
                    help="time the layer inside a Transformer sublayer: x + F(LN(x)) (pre) or "
                         "LN(x + F(x)) (post), seeded LayerNorm parameters")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    import torch
    import workloads

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    s = workloads.spec(args.workload, **ROUTINGS[args.routing])

    if args.impl == "reference":
        if rank != 0:
            return 0
        run_reference(args, s)
        return 0

    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_10392_gb300 import FEATURE_BACKWARD, FEATURES_DEFAULT, Layer
    if args.train and args.sublayer != "none":
        raise SystemExit("--train times the layer alone")

    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)

    # every rank draws its own batch of tokens (same layer weights)
    w_router, w_up, w_down, bias = workloads.make_weights(s)
    x, mask = workloads.make_tokens(s, w_router, seed=rank_token_seed(s, rank))
    T = s.tokens
    T_valid = T if mask is None else int(mask.sum())
    layer = Layer(s.d_model, s.d_ff, s.n_experts, s.n_blocks, dtype=s.dtype, max_tokens=T,
                  tau=s.tau, alpha_fixed=s.alpha_fixed, beta_fixed=s.beta_fixed,
                  topk_fixed=s.topk_fixed, prefix_blocks=s.prefix_blocks,
                  features=FEATURES_DEFAULT | (FEATURE_BACKWARD if args.train else 0),
                  gemm_kernels=args.gemm_kernels)
    layer.load_weights(w_router.to(dev), w_up.to(dev), w_down.to(dev),
                       None if bias is None else bias.to(dev))
    xd = x.to(dev)
    md = None if mask is None else mask.to(dev)
    out = torch.empty_like(xd)
    bcnt = torch.empty(T, dtype=torch.int32, device=dev)
    kcnt = torch.empty(T, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    # L2 flush between steps: a 512 MB write evicts everything, then a 256 MB
    # read evicts the written (dirty) lines, so each step starts on a cold,
    # clean L2 (both outside the timed events).
    flush = torch.empty(512 * 1024 * 1024, dtype=torch.uint8, device=dev)
    flush_r = torch.zeros(256 * 1024 * 1024, dtype=torch.uint8, device=dev)

    bwd_ev = None
    if args.train:
        gen = torch.Generator().manual_seed(rank + 17)
        dy = torch.randn(T, s.d_model, generator=gen).to(xd.dtype).to(dev)
        grads = {}

        def step():
            layer.forward(xd, out=out, mask=md, shared_counts=bcnt, residual_counts=kcnt)
            if bwd_ev is not None:
                bwd_ev[0].record(stream)
            grads.update(layer.backward(xd, dy, mask=md, lambda_div=0.01, want_bias=True,
                                        out=grads or None))
            if bwd_ev is not None:
                bwd_ev[1].record(stream)
    elif args.sublayer == "none":
        def step():
            layer.forward(xd, out=out, mask=md, shared_counts=bcnt, residual_counts=kcnt)
    else:
        gen = torch.Generator().manual_seed(7)
        ln_g = (0.5 + torch.rand(s.d_model, generator=gen)).to(xd.dtype).to(dev)
        ln_b = (0.1 * torch.randn(s.d_model, generator=gen)).to(xd.dtype).to(dev)

        def step():
            layer.sublayer_forward(xd, ln_g, ln_b, 1e-5, args.sublayer == "pre", out=out,
                                   mask=md, shared_counts=bcnt, residual_counts=kcnt)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    if layer.sync_status() != 0:
        raise RuntimeError("device status word set during warm-up")
    b_h, k_h = bcnt.cpu().long(), kcnt.cpu().long()
    rt = layer.routing()
    gpu_dec = {"b": bcnt.cpu().numpy(), "k": kcnt.cpu().numpy(),
               "shr": rt["shared_mask"].cpu().numpy().view("uint64"),
               "em": rt["expert_mask"].cpu().numpy().view("uint64")}
    B, M, d = s.n_blocks, s.block_width, s.d_model
    cb = b_h + k_h * (B - b_h)
    if mask is not None:
        cb = cb * mask.long()
    sum_cb = int(cb.sum())
    gemm_flops = 2.0 * d * M * sum_cb  # one of the two grouped GEMMs (Eq. 16)
    act_flops = 2.0 * gemm_flops       # activated FLOPs of the layer (Eq. 35 blocks)
    # a forward of more than pass_tokens tokens runs in passes; the stage
    # events of the per-kernel pass time the last one, tokens [last0, T)
    P = layer.pass_tokens()
    n_pass = (T + P - 1) // P
    last0 = (n_pass - 1) * P
    T_last = T - last0
    cb_last = int(cb[last0:].sum())
    stage_flops = 2.0 * d * M * cb_last  # one grouped GEMM launch of the last pass

    K = args.steps
    mk = lambda: torch.cuda.Event(enable_timing=True)
    starts = [mk() for _ in range(K)]
    ends = [mk() for _ in range(K)]
    stage_ev = [[mk() for _ in range(6)] for _ in range(K)]
    for evs in stage_ev:  # create the CUDA events
        for e in evs:
            e.record(stream)
    torch.cuda.synchronize(dev)

    if dist:
        dist.barrier()
    torch.cuda.synchronize(dev)
    sampler = ClockSampler() if rank == 0 else None
    for i in range(K):
        flush.zero_()  # L2 flush between steps (outside the timed events)
        flush_r.max()
        starts[i].record(stream)
        step()
        ends[i].record(stream)
    torch.cuda.synchronize(dev)
    if dist:
        dist.barrier()
    clocks = sampler.stop(0) if sampler else None
    if layer.sync_status() != 0:
        raise RuntimeError("device status word set during the timed region")
    # Per-kernel durations: the same K steps again with an event between
    # consecutive kernels. Those events serialise the kernels (no dependent
    # launch overlaps its predecessor), so each duration is the kernel's own
    # launch; the timed steps above run without them.
    bwd_pairs = [(mk(), mk()) for _ in range(K)] if args.train else None
    for i in range(K):
        flush.zero_()
        flush_r.max()
        layer.set_stage_events(stage_ev[i])
        if args.train:
            bwd_ev = bwd_pairs[i]
        step()
    torch.cuda.synchronize(dev)
    layer.set_stage_events(None)
    bwd_ev = None
    if layer.sync_status() != 0:
        raise RuntimeError("device status word set during the per-kernel pass")

    step_ms = [starts[i].elapsed_time(ends[i]) for i in range(K)]
    total_ms = sum(step_ms)
    names = ["router", "permute", "up_gemm", "down_gemm", "combine"]
    stage_ms = {n: statistics.fmean(stage_ev[i][j].elapsed_time(stage_ev[i][j + 1]) for i in range(K))
                for j, n in enumerate(names)}
    total_ms = max_over_ranks(total_ms, dist, dev)
    total_valid = sum_over_ranks(T_valid, dist, dev)

    # e2e through the C ABI with host buffers (copies inside the timed region)
    xh = x.pin_memory()
    oh = torch.empty_like(xh).pin_memory()
    mh = None if mask is None else mask.pin_memory()
    bh = torch.empty(T, dtype=torch.int32).pin_memory()
    kh = torch.empty(T, dtype=torch.int32).pin_memory()
    # (the host-buffer entry points run the layer alone: no end-to-end line
    # for a sublayer run or a training step)
    n_e2e = args.e2e_steps if args.sublayer == "none" and not args.train else 0
    # pipelined calls (unif_moe_forward_host_async: a call's input copy runs
    # under the previous call's kernels, its output copy under the next
    # call's), timed on the host clock from the first call to the return of
    # the wait after the last, launch overhead included
    for _ in range(3):
        layer.forward_host_async(xh, oh, mh, bh, kh)
    layer.forward_host_wait()
    e2e_pipe_s = None
    if n_e2e:
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(n_e2e):
            layer.forward_host_async(xh, oh, mh, bh, kh)
        layer.forward_host_wait()
        e2e_pipe_s = (time.perf_counter() - t0) / n_e2e
    # one synchronous call at a time (unif_moe_forward_host), event-timed
    for _ in range(3):
        layer.forward_host(xh, oh, mh, bh, kh)
    e2e_ms = []
    for _ in range(n_e2e):
        a, b = mk(), mk()
        a.record(stream)
        layer.forward_host(xh, oh, mh, bh, kh)
        b.record(stream)
        b.synchronize()
        e2e_ms.append(a.elapsed_time(b))
    elt = 2 if s.dtype == "bf16" else 4
    h2d = T * d * elt + (0 if mask is None else T)
    d2h = T * d * elt + 2 * 4 * T

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return 0

    peaks, peak_kind = load_peaks()
    ms = total_ms / K
    value = job_throughput(total_valid, ms)
    tflops = act_flops / (ms / 1e3) / 1e12
    # the per-kernel pass times each kernel alone (events between kernels):
    # the burst bf16 peak applies to the GEMMs; the whole step is set
    # against the sustained one
    peak_tf = peaks["bf16_tflops"]
    peak_tf_sus = peaks["bf16_tflops_sustained"]
    hbm = peaks["hbm_gbs"]
    hbm_nominal = 8000.0
    # roofline of the dominant kernel (the larger grouped GEMM), timed in the
    # per-kernel pass
    # the expert-tile FFN (three kernels per forward) runs both projections
    # in one launch: its stage is the up stage (the down stage is the empty
    # gap between two events), its work the activated flops of both
    # projections, 4 d M C_B per token (Eq. 35); the masked blocks it also
    # computes are not counted
    expert_tile = layer.kernels_per_forward() == 3
    if expert_tile:
        dom = "ffn"
        ffn_ms = stage_ms["up_gemm"] + stage_ms["down_gemm"]
        ach = 2.0 * stage_flops / (ffn_ms / 1e3) / 1e12
    else:
        dom = "up_gemm" if stage_ms["up_gemm"] >= stage_ms["down_gemm"] else "down_gemm"
        ach = stage_flops / (stage_ms[dom] / 1e3) / 1e12
    traffic = measured_traffic(s.name, dom)
    # algorithmic bytes of the memory-bound kernels (per forward): the router
    # reads x and writes each token's records (alpha, b, k, two masks, K
    # affinities; b and k also to the caller) and, when it groups the pairs,
    # one (token, weight) row per pair; the permute writes those rows; the
    # combine reads the fp32 accumulator and writes the output
    fused = layer.kernels_per_forward() <= 5 and s.dtype == "bf16"
    # (grouped by expert: one row per (token, expert), 1[b > 0] + k per token)
    n_rows_last = cb_last
    if expert_tile:
        rows_t = (b_h > 0).long() + k_h
        if mask is not None:
            rows_t = rows_t * mask.long()
        n_rows_last = int(rows_t[last0:].sum())
    exec_tf = (4.0 * d * s.d_ff * n_rows_last / (ffn_ms / 1e3) / 1e12) if expert_tile else None
    router_bytes = (T_last * d * elt + T_last * (4 * 3 + 8 * 2 + 4 * s.n_experts + 8) +
                    (8 * n_rows_last if fused else 0))
    combine_bytes = T_last * d * (4 + elt)
    permute_bytes = cb_last * 8

    def hbm_stage(ms_, nbytes):
        gbs = nbytes / ms_ / 1e6
        return {"ms": ms_, "bytes": nbytes, "GB/s": gbs, "frac_of_measured_hbm": gbs / hbm,
                "frac_of_nominal_8tbs": gbs / hbm_nominal}

    stages = {
        "router": hbm_stage(stage_ms["router"], router_bytes),
        "permute": (hbm_stage(stage_ms["permute"], permute_bytes) if not fused else
                    {"ms": 0.0, "fused_into": "router", "event_gap_ms": stage_ms["permute"]}),
        **({"ffn": {"ms": ffn_ms, "TFLOP/s": ach, "frac_of_burst_bf16": ach / peak_tf,
                    "kernel": "expert-tile FFN (both projections, rows grouped by expert)",
                    # the tensor work the kernel issues: both projections over
                    # all H channels of every (token, expert) row, the blocks
                    # the row does not run included (masked)
                    "executed_TFLOP/s": exec_tf,
                    "executed_frac_of_burst_bf16": exec_tf / peak_tf,
                    "event_gap_ms": stage_ms["down_gemm"]}} if expert_tile else {
            "up_gemm": {"ms": stage_ms["up_gemm"],
                        "TFLOP/s": stage_flops / stage_ms["up_gemm"] / 1e9,
                        "frac_of_burst_bf16": stage_flops / stage_ms["up_gemm"] / 1e9 / peak_tf},
            "down_gemm": {"ms": stage_ms["down_gemm"],
                          "TFLOP/s": stage_flops / stage_ms["down_gemm"] / 1e9,
                          "frac_of_burst_bf16":
                              stage_flops / stage_ms["down_gemm"] / 1e9 / peak_tf}}),
        "timed_pass": {"passes_per_forward": n_pass, "pass_tokens": P,
                       "tokens": [last0, T]},
        "combine": hbm_stage(stage_ms["combine"], combine_bytes),
    }
    import numpy as np
    valid = np.ones(T, bool) if mask is None else mask.numpy() != 0
    cb_np = cb.numpy()

    def hist(v):
        vals, counts = np.unique(v[valid], return_counts=True)
        return {str(int(a)): int(c) for a, c in zip(vals, counts)}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": s.dtype, "data": "synthetic (seeded; stands in for DeiT-S "
        "tokens on DomainBed, which are not available)",
        "config": dict(workload_desc(s, T_valid), parallelism="dp%d (independent batches)" % world,
                       sublayer={"none": "no (the layer alone)",
                                 "pre": "x + F(LN(x)), LN eps 1e-5",
                                 "post": "LN(x + F(x)), LN eps 1e-5"}[args.sublayer],
                       l2="flushed between steps (512 MB write + 256 MB read, outside the "
                          "timed events)"),
        "activated_tflops": tflops,
        "activated_frac_of_bf16_peak": tflops / peak_tf_sus,
        "activated_frac_kind": "%s bf16 sustained (whole step)" % peak_kind,
        "mean_C_B": sum_cb / T_valid,
        "decisions": {"hist_b": hist(b_h.numpy()), "hist_k": hist(k_h.numpy()),
                      "hist_C_B": hist(cb_np)},
        "roofline": {"bound": "tensor", "kernel": dom, "achieved": ach, "peak": peak_tf,
                     "unit": "TFLOP/s", "frac": ach / peak_tf, "traffic": traffic,
                     "peak_kind": "%s bf16 burst (kernel timed alone)" % peak_kind,
                     "frac_of_sustained": ach / peak_tf_sus},
        "stages": stages,
        "hbm_peak_gbs": hbm,
        "e2e": None if e2e_pipe_s is None else {
            "value": T_valid / e2e_pipe_s, "unit": UNIT,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": e2e_pipe_s * 1e3, "steps": n_e2e,
            "kind": "unif_moe_forward_host_async from pinned host buffers, pipelined "
                    "(copies of one call under the kernels of its neighbours), host clock "
                    "from the first call to the end of unif_moe_forward_host_wait"},
        "e2e_sync": None if not e2e_ms else {
            "value": T_valid / (statistics.fmean(e2e_ms) / 1e3), "unit": UNIT,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": statistics.fmean(e2e_ms),
            "kind": "unif_moe_forward_host, one synchronous call at a time, CUDA events"},
        # (a norm-first sublayer adds its layer-normalisation kernel)
        # (a norm-first sublayer adds its layer-normalisation kernel; a
        # training step the backward's seven kernels)
        "gpu_launches": (layer.kernels_per_forward() * n_pass + (args.sublayer == "pre") +
                         (7 if args.train else 0)) * K,
        "clocks": clocks,
    }
    if args.train:
        bwd_ms = statistics.fmean(a.elapsed_time(b) for a, b in bwd_pairs)
        # backward GEMM work: the hidden kernel's two products, dL/dx and the
        # two weight gradients, each 2 d M flops per (token, pair)
        line["config"]["step"] = ("training: forward, then backward with the Gram regulariser "
                                  "(Sec. III-E, lambda_div 0.01)")
        line["train"] = {"backward_ms": bwd_ms,
                         "backward_TFLOP/s": 5.0 * gemm_flops / bwd_ms / 1e9,
                         "step_activated_TFLOP/s": 7.0 * gemm_flops / ms / 1e9,
                         "backward_kind": "timed in the per-kernel pass (events around the "
                                          "backward call)"}
    if not args.no_cpu_baseline and world >= 1:
        wl = workloads.Workload(s, w_router, w_up, w_down, bias, x, mask)
        v, dt, n, tokens, repeat = OracleRunner(wl, train=args.train).sample()
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": oracle_cores(), "kind": "oracle",
                                "sample": "first %d of the workload's %d token slots, %d passes "
                                          "(%d valid tokens in all, %.1f s)"
                                          % (tokens, T, repeat, n, dt),
                                # the oracle's decisions on every token against the GPU's
                                "parity_check": decision_check(wl, gpu_dec, T)}
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


def run_reference(args, s):
    """The reference arm: the CPU oracle as it stands, on the host cores, each
    step a bounded token sample of the same workload."""
    import workloads
    wl = workloads.make_workload(s)
    runner = OracleRunner(wl)
    # size the per-step sample so that warm-up + steps stay within ~2 minutes
    probe_tokens = 64
    v, dt, _ = runner.time(probe_tokens)
    budget = 120.0 / (args.steps + args.warmup)
    tokens = int(max(16, min(s.tokens, probe_tokens * budget / max(dt, 1e-6))))
    for _ in range(args.warmup):
        runner.time(tokens)
    total_t, total_n = 0.0, 0
    for _ in range(args.steps):
        _, dt, n = runner.time(tokens)
        total_t += dt
        total_n += n
    value = total_n / total_t
    T_valid = s.tokens if wl.mask is None else int(wl.mask.sum())
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total_t / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded)",
        "config": dict(workload_desc(s, T_valid), parallelism="host cores"),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle_cores(), "kind": "oracle",
                         "sample": "first %d token slots of the workload per step" % tokens},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


if __name__ == "__main__":
    sys.exit(main())
