"""The diagnostics of Sec. II-B on the GPU (value alignment, ridge functional
demand) against the oracle (`oracle/diagnostics.py`, fp64).

The GPU computes the cosines and expert outputs in fp32 (from the layer's
bf16 or fp32 weights) and the ridge fits in fp64. Channels whose cosine lies
within 1e-5 of delta, pairs whose top-2 logits tie within 1e-5, and tokens
with an e_m within 1e-3 of eps are decided by rounding: they are counted and
excluded from the exact comparisons; e_m itself is compared within 2e-3
absolute (the errors are relative to |y_orig|)."""
import math

import numpy as np
import pytest
import torch

import workloads
from gpu_helpers import make_layer

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def diag_layer(dtype="bf16", T=256, d=128, H=512, K=4, B=4, spread=0.12, seed=5):
    """Experts copied from one FFN, then perturbed (relative size `spread`
    on the values, so that the value cosines straddle delta = 0.98)."""
    s = workloads.spec("tiny_f32" if dtype == "f32" else "vit_s").with_(
        tokens=T, d_model=d, d_ff=H, n_experts=K, n_blocks=B)
    wl = workloads.make_workload(s)
    g = torch.Generator().manual_seed(seed)
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    wd = wl.w_down.float().clone()
    base = wd[1].clone()
    for e in range(1, K + 1):
        wd[e] = base + spread * (0.5 + e / K) * torch.randn(base.shape, generator=g) / math.sqrt(H)
    w_res = (torch.randn(d, K, generator=g) * 0.2).to(tdt)
    return s, wl, wd.to(tdt), w_res


def load(s, wl, w_down):
    from paper_2608_10392_gb300 import FEATURE_DIAGNOSTICS
    dev = torch.device("cuda")
    L = make_layer(s, features=FEATURE_DIAGNOSTICS)
    L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), w_down.to(dev))
    return L


def cosines(w_down):
    V = np.transpose(w_down.double().numpy()[1:], (0, 2, 1))  # [K][H][d]
    n = np.linalg.norm(V, axis=2)
    return np.einsum("ihd,jhd->ijh", V, V) / (n[:, None, :] * n[None, :, :])


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_value_alignment(dtype):
    from oracle import diagnostics as dg
    s, wl, wd, _ = diag_layer(dtype)
    L = load(s, wl, wd)
    delta = 0.98
    rho = L.value_alignment(delta).cpu().numpy()
    torch.cuda.synchronize()
    rho_ref, S_ref = dg.value_alignment(wd, delta)
    near = np.abs(cosines(wd) - delta) < 1e-5
    H = s.d_ff
    off = rho_ref[~np.eye(s.n_experts, dtype=bool)]
    assert ((off > 0.05) & (off < 0.95)).any()  # delta splits the channels of some pair
    # rho may differ only by channels at the threshold
    assert (np.abs(rho - rho_ref) * H <= near.sum(axis=2) + 1e-6).all()
    assert np.allclose(np.diag(rho), 1.0)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_functional_demand(dtype):
    from oracle import diagnostics as dg
    s, wl, wd, w_res = diag_layer(dtype)
    L = load(s, wl, wd)
    dev = torch.device("cuda")
    delta, eps = 0.98, 0.05
    out = L.functional_demand(wl.x.to(dev), w_res.to(dev), delta, eps)
    torch.cuda.synchronize()
    k_ref, e_ref, pair_ref = dg.functional_demand(wl.x, wl.w_router, wl.w_up, wd, w_res, delta,
                                                  eps)
    k, e, pair = (out[n].cpu().numpy() for n in ("k_eps", "err", "pair"))
    z = wl.x.double().numpy() @ wl.w_router.double().numpy()[:, 1:]
    zs = np.sort(z, axis=1)
    tie = (zs[:, -2] - zs[:, -3] < 1e-5) | (zs[:, -1] - zs[:, -2] < 1e-5)
    same_pair = (pair == pair_ref).all(axis=1)
    assert (same_pair | tie).all(), np.nonzero(~(same_pair | tie))[0]
    ok = same_pair
    assert np.abs(e[ok] - e_ref[ok]).max() < 2e-3, np.abs(e[ok] - e_ref[ok]).max()
    edge = (np.abs(e_ref - eps) < 1e-3).any(axis=1)
    exact = ok & ~edge
    assert (k[exact] == k_ref[exact]).all()
    print("tokens", len(k), "compared exactly", int(exact.sum()), "k_eps histogram",
          np.bincount(k, minlength=s.n_experts + 2).tolist())
    assert len(set(k_ref.tolist())) > 1  # the tolerance separates tokens


def test_identical_experts_need_one_expert():
    """Experts copied from one FFN (no perturbation): every channel aligned
    (rho = 1), the shared part is the whole output, k_eps = 1."""
    s, wl, wd, w_res = diag_layer(spread=0.0)
    L = load(s, wl, wd)
    dev = torch.device("cuda")
    assert (L.value_alignment(0.98).cpu().numpy() == 1.0).all()
    out = L.functional_demand(wl.x.to(dev), w_res.to(dev), 0.98, 0.05)
    torch.cuda.synchronize()
    assert (out["k_eps"].cpu() == 1).all()
    assert float(out["err"].abs().max()) < 1e-6


def test_diagnostics_need_the_feature():
    from paper_2608_10392_gb300 import UnifMoeError
    s, wl, wd, w_res = diag_layer()
    L = make_layer(s)
    dev = torch.device("cuda")
    L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wd.to(dev))
    with pytest.raises(UnifMoeError) as e:
        L.value_alignment(0.98)
    assert e.value.code == -6
