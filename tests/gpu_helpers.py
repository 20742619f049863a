"""Shared helpers for the GPU parity tests: run the CUDA layer through the C
ABI and compare it with the CPU oracle on the same seeded inputs.

Parity rules (Sec. III decisions are discrete, the outputs continuous):
  - routing decisions (b, k, shared block set, residual expert set) must be
    identical on every token whose oracle near-tie margin exceeds 1e-3;
  - tokens whose decisions differ are counted; they must be at most 0.1% of
    the valid tokens (none at all below 1000 tokens), and for each the
    oracle is re-run on the GPU's decisions;
  - near-ties (margin <= 1e-3) are counted and reported, by the margin that
    is smallest;
  - outputs: per-token max |y_gpu - y_ref| / max |y_ref| within 2e-2 (bf16
    layers, fp32 accumulation) or 1e-4 (fp32 layers), on every token.

With UNIF_MOE_PARITY_REPORT set to a path, every comparison appends one JSON
line there (counts, errors, histograms of b, k and C_B); conftest.py renders
the lines as a table at the end of the session.
"""
from __future__ import annotations

import json
import math
import os
from dataclasses import asdict, dataclass, field

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


def make_layer(s, max_tokens=None, **kw):
    from paper_2608_10392_gb300 import Layer
    return Layer(s.d_model, s.d_ff, s.n_experts, s.n_blocks, dtype=s.dtype,
                 max_tokens=max_tokens or s.tokens, tau=s.tau, alpha_fixed=s.alpha_fixed,
                 beta_fixed=s.beta_fixed, topk_fixed=s.topk_fixed, prefix_blocks=s.prefix_blocks,
                 **kw)


def run_gpu(wl, layer=None, x=None, mask="default", **layer_kw) -> GpuRun:
    s = wl.spec
    dev = torch.device("cuda")
    if layer is None:
        layer = make_layer(s, max_tokens=max(s.tokens, 1), **layer_kw)
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
    n_valid: int
    n_near: int
    n_mismatch: int
    n_mismatch_clear: int
    max_rel: float
    checked: int
    # near-ties by the margin that is smallest: (i) rounding of B alpha,
    # (ii) prototype TopK, (iii) cumulative-mass cutoff, (iv) expert order
    near_by_margin: list = field(default_factory=list)
    n_margin_below_1e5: int = 0
    mean_cb: float = 0.0
    hist_b: dict = field(default_factory=dict)
    hist_k: dict = field(default_factory=dict)
    hist_cb: dict = field(default_factory=dict)


def _hist(v) -> dict:
    vals, counts = np.unique(np.asarray(v), return_counts=True)
    return {int(a): int(c) for a, c in zip(vals, counts)}


def record(rep: Report, wl, label: str = ""):
    """Appends the comparison to the parity report, if one is requested."""
    path = os.environ.get("UNIF_MOE_PARITY_REPORT")
    if not path:
        return
    s = wl.spec
    test = os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0]
    line = dict(test=test, label=label, workload=s.name, dtype=s.dtype, d=s.d_model, H=s.d_ff,
                K=s.n_experts, B=s.n_blocks, thresholds=dict(
                    tau=None if math.isnan(s.tau) else s.tau,
                    alpha_fixed=None if math.isnan(s.alpha_fixed) else s.alpha_fixed,
                    beta_fixed=None if math.isnan(s.beta_fixed) else s.beta_fixed,
                    topk_fixed=s.topk_fixed, prefix_blocks=s.prefix_blocks),
                tol=TOL[s.dtype], **asdict(rep))
    with open(path, "a") as f:
        f.write(json.dumps(line) + "\n")


def compare(wl, g: GpuRun, x=None, mask="default", label: str = "") -> Report:
    """Decisions and outputs of the GPU run against the oracle, on every
    token."""
    s = wl.spec
    x = wl.x if x is None else x
    m = wl.mask if isinstance(mask, str) else mask
    r = oracle_routing(wl, x, m)
    T = x.shape[0]
    valid = np.ones(T, bool) if m is None else (np.asarray(m) != 0)
    em_ref = r.expert_mask()
    same = ((g.b == r.b) & (g.k == r.k) & (g.shr == r.shr_mask) & (g.em == em_ref))
    mmin = r.margin.min(axis=1)
    near = mmin <= NEAR_TIE
    mism = ~same
    rep_clear = int((mism & ~near).sum())
    which = np.argmin(r.margin, axis=1)
    near_by = [int((near & valid & (which == i)).sum()) for i in range(4)]
    idx = np.arange(T)
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
    nz = denom > 0
    rel = np.where(nz, err / np.where(nz, denom, 1.0), err)
    cb = (g.b.astype(np.int64) + g.k.astype(np.int64) * (s.n_blocks - g.b.astype(np.int64)))
    rep = Report(n_tokens=T, n_valid=int(valid.sum()), n_near=int((near & valid).sum()),
                 n_mismatch=int(mism.sum()), n_mismatch_clear=rep_clear,
                 max_rel=float(rel.max()) if len(rel) else 0.0, checked=len(idx),
                 near_by_margin=near_by, n_margin_below_1e5=int(((mmin <= 1e-5) & valid).sum()),
                 mean_cb=float(cb[valid].mean()) if valid.any() else 0.0,
                 hist_b=_hist(g.b[valid]), hist_k=_hist(g.k[valid]), hist_cb=_hist(cb[valid]))
    record(rep, wl, label)
    return rep


def assert_parity(wl, g: GpuRun, rep: Report):
    tol = TOL[wl.spec.dtype]
    assert rep.checked == rep.n_tokens, rep  # outputs compared on every token
    assert rep.n_mismatch_clear == 0, rep
    assert rep.n_mismatch <= math.floor(1e-3 * rep.n_valid), rep
    assert rep.max_rel <= tol, rep
