"""Shared helpers for the GPU parity tests: run the CUDA layer through the C
ABI and compare it with the CPU oracle on the same seeded inputs.

Parity rules (Sec. III decisions are discrete, the outputs continuous):
  - routing decisions (b, k, shared block set, residual expert set) must be
    identical on every token whose oracle near-tie margin exceeds 1e-3;
  - tokens whose decisions differ are counted; they must be fewer than 0.1%
    of all tokens, and for each the oracle is re-run on the GPU's decisions;
  - outputs: per-token max |y_gpu - y_ref| / max |y_ref| within 2e-2 (bf16
    layers, fp32 accumulation) or 1e-4 (fp32 layers).
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np
import torch

import oracle
from oracle import Routing, Thresholds

TOL = {"bf16": 2e-2, "f32": 1e-4}
NEAR_TIE = 1e-3


def thresholds_of(s) -> Thresholds:
    return Thresholds(tau=s.tau, alpha_fixed=s.alpha_fixed, beta_fixed=s.beta_fixed,
                      topk_fixed=s.topk_fixed, prefix_blocks=s.prefix_blocks)


def round_mode(s) -> int:
    return oracle.ROUND_BF16 if s.dtype == "bf16" else oracle.ROUND_F32


@dataclass
class GpuRun:
    y: np.ndarray          # [T][d] float64
    b: np.ndarray
    k: np.ndarray
    shr: np.ndarray        # uint64
    em: np.ndarray         # uint64
    alpha: np.ndarray
    q: np.ndarray
    p: np.ndarray
    layer: object


def make_layer(s, max_tokens=None):
    from paper_2608_10392_gb300 import Layer
    return Layer(s.d_model, s.d_ff, s.n_experts, s.n_blocks, dtype=s.dtype,
                 max_tokens=max_tokens or s.tokens, tau=s.tau, alpha_fixed=s.alpha_fixed,
                 beta_fixed=s.beta_fixed, topk_fixed=s.topk_fixed, prefix_blocks=s.prefix_blocks)


def run_gpu(wl, layer=None, x=None, mask="default") -> GpuRun:
    s = wl.spec
    dev = torch.device("cuda")
    if layer is None:
        layer = make_layer(s, max_tokens=max(s.tokens, 1))
        bias = None if wl.router_bias is None else wl.router_bias.to(dev)
        layer.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev), bias)
    x = wl.x if x is None else x
    m = wl.mask if isinstance(mask, str) else mask
    T = x.shape[0]
    xd = x.to(dev)
    md = None if m is None else m.to(dev)
    b = torch.full((T,), -7, dtype=torch.int32, device=dev)
    k = torch.full((T,), -7, dtype=torch.int32, device=dev)
    y = layer.forward(xd, mask=md, shared_counts=b, residual_counts=k)
    torch.cuda.synchronize()
    st = layer.sync_status()
    assert st == 0, "device status %d" % st
    r = layer.routing()
    return GpuRun(y=y.float().cpu().numpy().astype(np.float64), b=b.cpu().numpy(),
                  k=k.cpu().numpy(), shr=r["shared_mask"].cpu().numpy().view(np.uint64),
                  em=r["expert_mask"].cpu().numpy().view(np.uint64),
                  alpha=r["alpha"].cpu().numpy(), q=r["q"].cpu().numpy(), p=r["p"].cpu().numpy(),
                  layer=layer)


def oracle_routing(wl, x=None, mask="default") -> Routing:
    s = wl.spec
    x = wl.x if x is None else x
    m = wl.mask if isinstance(mask, str) else mask
    mu = oracle.prototypes(wl.w_up, s.n_blocks, round_mode(s))
    return oracle.route(x, wl.w_router, mu, s.n_experts, s.n_blocks, thresholds_of(s), m,
                        wl.router_bias)


def subset(r: Routing, idx) -> Routing:
    return Routing(**{f: getattr(r, f)[idx] for f in r.__dataclass_fields__})


@dataclass
class Report:
    n_tokens: int
    n_near: int
    n_mismatch: int
    n_mismatch_clear: int
    max_rel: float
    checked: int


def compare(wl, g: GpuRun, sample=None, x=None, mask="default", seed=0) -> Report:
    """Decisions on all tokens, outputs on `sample` tokens (None = all)."""
    s = wl.spec
    x = wl.x if x is None else x
    m = wl.mask if isinstance(mask, str) else mask
    r = oracle_routing(wl, x, m)
    T = x.shape[0]
    em_ref = r.expert_mask()
    same = ((g.b == r.b) & (g.k == r.k) & (g.shr == r.shr_mask) & (g.em == em_ref))
    near = r.margin.min(axis=1) <= NEAR_TIE
    mism = ~same
    rep_clear = int((mism & ~near).sum())
    # outputs
    if sample is None or sample >= T:
        idx = np.arange(T)
    else:
        rng = np.random.default_rng(seed)
        idx = np.unique(np.concatenate([[0, T - 1], rng.choice(T, sample, replace=False),
                                        np.nonzero(mism)[0]]))
    rs = subset(r, idx)
    # tokens whose decisions differ: re-run the oracle on the GPU's decisions
    mi = np.nonzero(mism[idx])[0]
    if len(mi):
        forced = oracle.with_decisions(subset(rs, mi), g.shr[idx][mi], g.em[idx][mi], s.n_blocks)
        for f in ("alpha", "b", "k", "shr_mask", "q", "p"):
            arr = getattr(rs, f).copy()
            arr[mi] = getattr(forced, f)
            setattr(rs, f, arr)
    xs = x[idx]
    ms = None if m is None else m[idx]
    y_ref = oracle.forward(xs, wl.w_up, wl.w_down, rs, s.n_blocks, ms)
    yg = g.y[idx]
    denom = np.abs(y_ref).max(axis=1)
    err = np.abs(yg - y_ref).max(axis=1)
    valid = denom > 0
    rel = np.where(valid, err / np.where(valid, denom, 1.0), err)
    return Report(n_tokens=T, n_near=int(near.sum()), n_mismatch=int(mism.sum()),
                  n_mismatch_clear=rep_clear, max_rel=float(rel.max()) if len(rel) else 0.0,
                  checked=len(idx))


def assert_parity(wl, g: GpuRun, rep: Report):
    tol = TOL[wl.spec.dtype]
    assert rep.n_mismatch_clear == 0, rep
    assert rep.n_mismatch <= max(1, math.floor(1e-3 * rep.n_tokens)), rep
    assert rep.max_rel <= tol, rep
