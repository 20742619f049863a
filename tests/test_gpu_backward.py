"""Backward pass on the GPU (training, Sec. III-E) against the oracle.

The gradients are defined with the forward's discrete decisions held fixed,
so the oracle's backward runs on the GPU's own decisions (their parity with
the oracle's is the forward tests' subject); alpha and s are the oracle's,
recomputed in fp64 from the same bf16 inputs and weights.

Tolerance: the GPU keeps dL/da and w GeLU(a) in bf16 (8 significant bits,
2^-8 relative) between its GEMMs and accumulates in fp32, as the forward
keeps h; every gradient is compared at the forward's bf16 bound of 2e-2:
dL/dx per token (max |err| / max |ref| over the token's features), each
weight gradient over the whole tensor (max |err| / max |ref|)."""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads
from gpu_helpers import make_layer, thresholds_of

pytestmark = pytest.mark.gpu

TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def run_case(spec, lambda_div=0.0, seed=11):
    from paper_2608_10392_gb300 import FEATURE_BACKWARD, FEATURES_DEFAULT
    wl = workloads.make_workload(spec)
    dev = torch.device("cuda")
    L = make_layer(spec, features=FEATURES_DEFAULT | FEATURE_BACKWARD)
    bias = None if wl.router_bias is None else wl.router_bias.to(dev)
    L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev), bias)
    x = wl.x.to(dev)
    md = None if wl.mask is None else wl.mask.to(dev)
    L.forward(x, mask=md)
    r = L.routing()
    g = torch.Generator().manual_seed(seed)
    dy = torch.randn(spec.tokens, spec.d_model, generator=g).to(torch.bfloat16)
    grads = L.backward(x, dy.to(dev), mask=md, lambda_div=lambda_div, want_bias=True)
    torch.cuda.synchronize()
    assert L.sync_status() == 0
    got = {k: (None if v is None else v.double().cpu().numpy()) for k, v in grads.items()}
    shr = r["shared_mask"].cpu().numpy().view(np.uint64)
    em = r["expert_mask"].cpu().numpy().view(np.uint64)
    ref = oracle.backward(wl.x, wl.w_router, wl.w_up, wl.w_down, shr, em, spec.n_blocks, dy,
                          thresholds_of(spec), wl.mask, wl.router_bias)
    return wl, got, ref, L


def rel_tensor(got, ref):
    return float(np.abs(got - ref).max() / max(np.abs(ref).max(), 1e-30))


def rel_rows(got, ref, valid):
    den = np.abs(ref).max(axis=1)
    err = np.abs(got - ref).max(axis=1)
    ok = valid & (den > 0)
    return float((err[ok] / den[ok]).max()) if ok.any() else 0.0


def check(wl, got, ref, lambda_div=0.0):
    T = wl.x.shape[0]
    valid = np.ones(T, bool) if wl.mask is None else wl.mask.numpy() != 0
    assert np.isfinite(got["dx"]).all()
    assert (got["dx"][~valid] == 0).all()
    errs = {"dx": rel_rows(got["dx"], ref.dx, valid),
            "dw_up": rel_tensor(got["dw_up"], ref.dw_up),
            "dw_down": rel_tensor(got["dw_down"], ref.dw_down),
            "dbias": rel_tensor(got["dbias"], ref.dbias)}
    wr_ref = ref.dw_router
    if lambda_div:
        _, gdiv = oracle.diversity(wl.w_router)
        wr_ref = wr_ref + lambda_div * gdiv
    errs["dw_router"] = rel_tensor(got["dw_router"], wr_ref)
    print(errs)
    for k, v in errs.items():
        assert v <= TOL, (k, v, errs)
    return errs


def small(**kw):
    base = dict(tokens=300, d_model=128, d_ff=512, n_experts=4, n_blocks=4)
    base.update(kw)
    return workloads.spec("vit_s").with_(**base)


def test_backward_small_ragged():
    """300 tokens: the last tile of every group is ragged."""
    wl, got, ref, _ = run_case(small())
    check(wl, got, ref)


def test_backward_vit_s_full_size():
    wl, got, ref, _ = run_case(workloads.spec("vit_s"))
    check(wl, got, ref)


def test_backward_bert_padding_two_subtiles():
    """BERT-base: block width 384 runs as two 192-channel sub-tiles in both
    backward GEMM kernels; padding tokens (NaN inputs) get dx = 0."""
    wl, got, ref, _ = run_case(workloads.spec("bert_base"))
    check(wl, got, ref)


def test_backward_router_bias_many_experts():
    """The stress layer's shapes (K = 32, B = 16, d = 1024) and Zipf router
    bias on its first 2,048 tokens: the bias gradient and 33 router columns."""
    wl, got, ref, _ = run_case(workloads.spec("stress", tokens=2048))
    check(wl, got, ref)


def test_backward_sixteen_experts():
    """K = 16 residual experts (17 router columns, as ViT-B's layer), 300
    tokens: the router gradients' kernel instance for up to 32 columns."""
    wl, got, ref, _ = run_case(small(tokens=300, n_experts=16))
    check(wl, got, ref)


def test_backward_gram_regulariser():
    """lambda_div = 0.01 (the paper's choice): dW* gains lambda dL_div/dW*,
    and L_div itself is returned."""
    lam = 0.01
    wl, got, ref, _ = run_case(small(tokens=500), lambda_div=lam)
    check(wl, got, ref, lambda_div=lam)
    L, _ = oracle.diversity(wl.w_router)
    assert got["l_div"][0] == pytest.approx(L, rel=1e-4)


def test_backward_fixed_alpha_has_no_shared_router_gradient():
    wl, got, ref, _ = run_case(small(tokens=400, alpha_fixed=0.4))
    check(wl, got, ref)
    assert (got["dw_router"][:, 0] == 0).all()


def test_backward_argument_errors():
    from paper_2608_10392_gb300 import FEATURE_BACKWARD, FEATURES_DEFAULT, UnifMoeError
    s = small(tokens=256)
    wl = workloads.make_workload(s)
    dev = torch.device("cuda")
    x = wl.x.to(dev)
    dy = torch.zeros_like(x)
    plain = make_layer(s)
    plain.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    plain.forward(x)
    with pytest.raises(UnifMoeError) as e:  # no backward workspace
        plain.backward(x, dy)
    assert e.value.code == -6
    L = make_layer(s, features=FEATURES_DEFAULT | FEATURE_BACKWARD)
    L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    with pytest.raises(UnifMoeError) as e:  # no forward yet
        L.backward(x, dy)
    assert e.value.code == -6
    L.forward(x)
    with pytest.raises(UnifMoeError) as e:  # another T than the forward's
        L.backward(x[:100], dy[:100])
    assert e.value.code == -6
    torch.cuda.synchronize()
    assert L.sync_status() == 0
