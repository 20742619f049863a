"""The layer as a Transformer sublayer (pre- or post-norm, the paper's DeiT-S
and BERT backbones, Appendix A) and experts upcycled from one dense FFN
(Sec. III), on the GPU against the oracle. Decisions are compared as for the
layer itself: bit-exact away from near-ties, with the oracle re-run on the
GPU's decisions where they differ; outputs within the layer's tolerance."""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads
from gpu_helpers import (NEAR_TIE, TOL, GpuRun, Report, _hist, make_layer, oracle_routing,
                         record, round_mode, subset)

pytestmark = pytest.mark.gpu

EPS = 1e-5


def ln_params(d, dtype, seed=7):
    """Seeded LayerNorm scale and shift (gamma ~ U(0.5, 1.5), beta ~ N(0, 0.1)),
    rounded to the layer dtype; float64 copies for the oracle."""
    g = torch.Generator().manual_seed(seed)
    gamma = (0.5 + torch.rand(d, generator=g)).to(dtype)
    beta = (0.1 * torch.randn(d, generator=g)).to(dtype)
    return gamma, beta


def run_sublayer(wl, gamma, beta, norm_first, layer=None):
    s = wl.spec
    dev = torch.device("cuda")
    if layer is None:
        layer = make_layer(s)
        bias = None if wl.router_bias is None else wl.router_bias.to(dev)
        layer.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev), bias)
    T = wl.x.shape[0]
    xd = wl.x.to(dev)
    md = None if wl.mask is None else wl.mask.to(dev)
    b = torch.full((T,), -7, dtype=torch.int32, device=dev)
    k = torch.full((T,), -7, dtype=torch.int32, device=dev)
    out = layer.sublayer_forward(xd, gamma.to(dev), beta.to(dev), EPS, norm_first, mask=md,
                                 shared_counts=b, residual_counts=k)
    torch.cuda.synchronize()
    assert layer.sync_status() == 0
    r = layer.routing()
    return GpuRun(y=out.float().cpu().numpy().astype(np.float64), b=b.cpu().numpy(),
                  k=k.cpu().numpy(), shr=r["shared_mask"].cpu().numpy().view(np.uint64),
                  em=r["expert_mask"].cpu().numpy().view(np.uint64),
                  alpha=r["alpha"].cpu().numpy(), q=r["q"].cpu().numpy(),
                  p=r["p"].cpu().numpy(), layer=layer)


def check_sublayer(wl, g: GpuRun, gamma, beta, norm_first, label=""):
    """Decisions and outputs on every token; returns the oracle's routing."""
    s = wl.spec
    m = wl.mask
    xa = oracle._f64(wl.x)
    ga, be = oracle._f64(gamma), oracle._f64(beta)
    # the layer's input: LN(x) in the layer dtype (norm first), else x
    xin = oracle.layernorm(xa, ga, be, EPS, m, round_mode(s)) if norm_first else xa
    r = oracle_routing(wl, x=xin, mask=m)
    T = xa.shape[0]
    valid = np.ones(T, bool) if m is None else (np.asarray(m) != 0)
    same = ((g.b == r.b) & (g.k == r.k) & (g.shr == r.shr_mask) & (g.em == r.expert_mask()))
    mmin = r.margin.min(axis=1)
    near = mmin <= NEAR_TIE
    mism = ~same
    idx = np.arange(T)
    rs = subset(r, idx)
    mi = np.nonzero(mism[idx])[0]
    if len(mi):
        forced = oracle.with_decisions(subset(rs, mi), g.shr[idx][mi], g.em[idx][mi], s.n_blocks)
        for f in ("alpha", "b", "k", "shr_mask", "q", "p"):
            arr = getattr(rs, f).copy()
            arr[mi] = getattr(forced, f)
            setattr(rs, f, arr)
    ms = None if m is None else m[idx]
    y = oracle.forward(xin[idx], wl.w_up, wl.w_down, rs, s.n_blocks, ms)
    with np.errstate(invalid="ignore"):
        ref = xa[idx] + y if norm_first else oracle.layernorm(xa[idx] + y, ga, be, EPS, ms)
    if ms is not None:
        ref[oracle._u8(ms) == 0] = 0.0
    out = g.y[idx]
    assert np.isfinite(out).all()
    denom = np.abs(ref).max(axis=1)
    err = np.abs(out - ref).max(axis=1)
    rel = np.where(denom > 0, err / np.where(denom > 0, denom, 1.0), err)
    which = np.argmin(r.margin, axis=1)
    cb = g.b.astype(np.int64) + g.k.astype(np.int64) * (s.n_blocks - g.b.astype(np.int64))
    rep = Report(n_tokens=T, n_valid=int(valid.sum()), n_near=int((near & valid).sum()),
                 n_mismatch=int(mism.sum()), n_mismatch_clear=int((mism & ~near).sum()),
                 max_rel=float(rel.max()), checked=len(idx),
                 near_by_margin=[int((near & valid & (which == i)).sum()) for i in range(4)],
                 n_margin_below_1e5=int(((mmin <= 1e-5) & valid).sum()),
                 mean_cb=float(cb[valid].mean()), hist_b=_hist(g.b[valid]),
                 hist_k=_hist(g.k[valid]), hist_cb=_hist(cb[valid]))
    record(rep, wl, label or ("sublayer, norm first" if norm_first else "sublayer, norm after"))
    assert rep.n_mismatch_clear == 0, rep
    assert rep.n_mismatch <= math.floor(1e-3 * rep.n_valid), rep
    assert rep.max_rel <= TOL[s.dtype], rep
    return r


@pytest.mark.parametrize("norm_first", [True, False])
def test_sublayer_vit_s(norm_first):
    """ViT-S layer inside a DeiT-style (norm first) or BERT-style (norm after)
    sublayer, all 12,608 tokens decided and checked."""
    wl = workloads.make_workload(workloads.spec("vit_s"))
    gamma, beta = ln_params(wl.spec.d_model, torch.bfloat16)
    g = run_sublayer(wl, gamma, beta, norm_first)
    check_sublayer(wl, g, gamma, beta, norm_first)


@pytest.mark.parametrize("norm_first", [True, False])
def test_sublayer_bert_padding(norm_first):
    """BERT-base-shaped layer with NaN-filled padding slots: padding gives 0,
    its NaNs reach neither the norm nor the residual."""
    wl = workloads.make_workload(workloads.spec("bert_base"))
    gamma, beta = ln_params(wl.spec.d_model, torch.bfloat16, seed=8)
    g = run_sublayer(wl, gamma, beta, norm_first)
    check_sublayer(wl, g, gamma, beta, norm_first)


@pytest.mark.parametrize("norm_first", [True, False])
def test_sublayer_in_passes(norm_first):
    """A sublayer forward that runs in two passes (d = 1024: 32,768 tokens per
    pass) adds the residual of each pass's own tokens."""
    s = workloads.spec("bert_base").with_(tokens=33468, d_model=1024, d_ff=1024, n_experts=2,
                                          n_blocks=4)
    wl = workloads.make_workload(s)
    gamma, beta = ln_params(s.d_model, torch.bfloat16, seed=10)
    g = run_sublayer(wl, gamma, beta, norm_first)
    assert g.layer.pass_tokens() == 32768
    check_sublayer(wl, g, gamma, beta, norm_first,
                   label="two passes, " + ("norm first" if norm_first else "norm after"))


@pytest.mark.parametrize("norm_first", [True, False])
def test_sublayer_f32(norm_first):
    wl = workloads.make_workload(workloads.spec("tiny_f32"))
    gamma, beta = ln_params(wl.spec.d_model, torch.float32, seed=9)
    g = run_sublayer(wl, gamma, beta, norm_first)
    check_sublayer(wl, g, gamma, beta, norm_first)


def test_upcycled_experts():
    """Loading one dense FFN into every expert equals loading the K + 1 copies
    explicitly, and matches the oracle on the upcycled weights (whose output is
    alpha times the shared blocks plus the selected residual mass times the
    complementary blocks of the dense FFN)."""
    s = workloads.spec("vit_s", tokens=3000)
    wl = workloads.make_workload(s)
    dev = torch.device("cuda")
    w1, w2 = wl.w_up[0].clone(), wl.w_down[0].clone()  # a dense FFN: [H][d], [d][H]
    up = make_layer(s)
    up.load_upcycled(wl.w_router.to(dev), w1.to(dev), w2.to(dev))
    K = s.n_experts
    rep = make_layer(s)
    rep.load_weights(wl.w_router.to(dev), w1.expand(K + 1, -1, -1).contiguous().to(dev),
                     w2.expand(K + 1, -1, -1).contiguous().to(dev))
    x = wl.x.to(dev)
    y_up = up.forward(x).float()
    y_rep = rep.forward(x).float()
    torch.cuda.synchronize()
    assert up.sync_status() == 0 and rep.sync_status() == 0
    # the same weights and kernels: equal up to the order of the fp32 sums
    rel = (y_up - y_rep).abs().amax(1) / y_rep.abs().amax(1).clamp_min(1e-6)
    assert float(rel.max()) < 1e-2
    # against the oracle on the upcycled weights
    wu, wd = oracle.upcycle(w1, w2, K)
    y_ref, _ = oracle.layer(wl.x[:500], wl.w_router, wu, wd, s.n_blocks,
                            round_mode=round_mode(s))
    out = y_up[:500].cpu().numpy().astype(np.float64)
    denom = np.abs(y_ref).max(axis=1)
    err = np.abs(out - y_ref).max(axis=1)
    assert float((err / np.maximum(denom, 1e-12)).max()) <= TOL["bf16"]


def test_sublayer_argument_errors():
    """Misaligned LayerNorm parameters and a bad eps are refused before any
    launch, and the handle stays usable."""
    from paper_2608_10392_gb300 import UnifMoeError
    wl = workloads.make_workload(workloads.spec("vit_s", tokens=256))
    s = wl.spec
    dev = torch.device("cuda")
    layer = make_layer(s)
    layer.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    gamma, beta = ln_params(s.d_model, torch.bfloat16)
    gd, bd = gamma.to(dev), beta.to(dev)
    x = wl.x.to(dev)
    shifted = torch.empty(s.d_model + 1, dtype=torch.bfloat16, device=dev)[1:]  # 2-byte offset
    shifted.copy_(gd)
    with pytest.raises(UnifMoeError) as e:
        layer.sublayer_forward(x, shifted, bd, EPS, True)
    assert e.value.code == -1
    for eps in (-1.0, float("nan")):
        with pytest.raises(UnifMoeError) as e:
            layer.sublayer_forward(x, gd, bd, eps, False)
        assert e.value.code == -1
    out = layer.sublayer_forward(x, gd, bd, EPS, True)
    torch.cuda.synchronize()
    assert layer.sync_status() == 0 and torch.isfinite(out.float()).all()
