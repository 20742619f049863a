"""GPU parity: the CUDA layer (through the C ABI) against the CPU oracle on
the five seeded workloads, on ragged and edge-case shapes, and on the
ablation switches of Table IV. Rules in tests/gpu_helpers.py."""
import math

import numpy as np
import pytest
import torch

import oracle
import workloads
from gpu_helpers import assert_parity, compare, make_layer, run_gpu, subset

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def small(dtype="bf16", **kw):
    base = dict(tokens=300, d_model=128, d_ff=512, n_experts=4, n_blocks=4)
    base.update(kw)
    name = "tiny_f32" if dtype == "f32" else "vit_s"
    return workloads.spec(name).with_(**base)


# ---------------------------------------------------------------- workloads

def test_tiny_f32_full():
    wl = workloads.make_workload(workloads.spec("tiny_f32"))
    g = run_gpu(wl)
    rep = compare(wl, g)
    assert_parity(wl, g, rep)


def test_vit_s_full_size():
    wl = workloads.make_workload(workloads.spec("vit_s"))
    g = run_gpu(wl)
    rep = compare(wl, g)
    print(rep)
    assert_parity(wl, g, rep)


def test_bert_base_padding():
    wl = workloads.make_workload(workloads.spec("bert_base"))
    g = run_gpu(wl)
    m = wl.mask.numpy()
    assert (g.b[m == 0] == 0).all() and (g.k[m == 0] == 0).all()
    assert (g.y[m == 0] == 0).all()
    assert np.isfinite(g.y).all()
    rep = compare(wl, g)
    print(rep)
    assert_parity(wl, g, rep)


@pytest.mark.parametrize("theta", [math.nan, 0.5, 0.7, 0.9])
def test_vit_b_thresholds(theta):
    wl = workloads.make_workload(workloads.spec("vit_b", beta_fixed=theta))
    g = run_gpu(wl)
    rep = compare(wl, g, label="theta %s" % theta)
    print(theta, rep)
    assert_parity(wl, g, rep)


def test_stress_full_size():
    wl = workloads.make_workload(workloads.spec("stress"))
    g = run_gpu(wl)
    rep = compare(wl, g)
    print(rep, "b range", g.b.min(), g.b.max(), "k range", g.k.min(), g.k.max())
    assert g.b.min() == 1 and g.b.max() == 15  # the mixture spans every shared count
    assert_parity(wl, g, rep)


def test_forward_in_passes():
    """d = 4096: the fp32 accumulator of 8,192 tokens fills the 128 MiB a pass
    may use, so 8,969 tokens (text batch with padding, NaN-filled) run in two
    passes, the second ragged. Decisions, counts and outputs of every token
    match the oracle; the routing records cover both passes; the group table
    is that of the last pass, with absolute token indices."""
    s = workloads.spec("bert_base").with_(tokens=8969, d_model=4096, d_ff=1024, n_experts=2,
                                          n_blocks=4)
    wl = workloads.make_workload(s)
    g = run_gpu(wl)
    assert g.layer.pass_tokens() == 8192
    m = wl.mask.numpy()
    assert (g.y[m == 0] == 0).all() and np.isfinite(g.y).all()
    assert_parity(wl, g, compare(wl, g, label="two passes"))
    counts, offsets, tok, w = g.layer.groups()
    real = tok.numpy()[tok.numpy() >= 0]
    assert real.min() >= 8192 and real.max() < 8969
    cb = g.b[8192:] + g.k[8192:] * (s.n_blocks - g.b[8192:])
    assert int(counts.sum()) == int(cb[m[8192:] == 1].sum())


# ------------------------------------------------------------- ragged sizes

@pytest.mark.parametrize("T", [1, 7, 64, 129, 255, 257, 1000])
def test_ragged_token_counts(T):
    wl = workloads.make_workload(small(tokens=T))
    g = run_gpu(wl)
    assert_parity(wl, g, compare(wl, g))


def _router_rows(T, n_sm):
    """Tokens per router CTA the library picks for T tokens: the smallest
    multiple of 32 whose grid fits on the SMs, else 128."""
    for r in (32, 64, 96):
        if (T + r - 1) // r <= n_sm:
            return r
    return 128


@pytest.mark.parametrize("where", ["R32-last", "R64-first", "R64-last", "R96-first",
                                   "R96-last", "R128-first"])
def test_router_tile_heights(where):
    """Token counts at each switch of the tensor-core router's tokens per CTA
    (32, 64, 96, 128 with the grid in one wave): every token's decisions and
    output against the oracle, with a ragged last CTA on both sides."""
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    R, side = where.split("-")
    R = int(R[1:])
    prev = {32: 0, 64: 32, 96: 64, 128: 96}[R]
    T = prev * n_sm + 1 if side == "first" else R * n_sm - 5
    assert _router_rows(T, n_sm) == R
    wl = workloads.make_workload(small(tokens=T, d_model=128, d_ff=256, n_experts=4, n_blocks=4))
    g = run_gpu(wl)
    assert_parity(wl, g, compare(wl, g))


def test_zero_tokens_is_noop():
    wl = workloads.make_workload(small(tokens=16))
    layer = make_layer(wl.spec)
    dev = torch.device("cuda")
    layer.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    x = torch.empty(0, wl.spec.d_model, dtype=torch.bfloat16, device=dev)
    y = layer.forward(x)
    assert y.shape == (0, wl.spec.d_model)


def test_all_tokens_masked():
    wl = workloads.make_workload(small(tokens=200))
    mask = torch.zeros(200, dtype=torch.uint8)
    g = run_gpu(wl, mask=mask)
    assert (g.y == 0).all() and (g.b == 0).all() and (g.k == 0).all()


def test_max_tokens_and_reuse():
    """T = max_tokens, then a smaller T on the same handle (workspace reuse)."""
    wl = workloads.make_workload(small(tokens=1000))
    g = run_gpu(wl)
    assert_parity(wl, g, compare(wl, g))
    x2 = wl.x[:333].clone()
    g2 = run_gpu(wl, layer=g.layer, x=x2, mask=None)
    np.testing.assert_allclose(g2.y, g.y[:333], rtol=1e-2, atol=1e-6)  # one bf16 ulp


def test_smaller_then_larger_forward_on_one_handle():
    """A small forward, then the full one: the accumulator rows and the
    group counters the first forward used are clean for the second."""
    wl = workloads.make_workload(small(tokens=1000))
    g1 = run_gpu(wl, x=wl.x[:200].clone(), mask=None)
    g = run_gpu(wl, layer=g1.layer)
    assert_parity(wl, g, compare(wl, g))


def test_kernels_per_forward():
    s = small(tokens=500)
    assert make_layer(s).kernels_per_forward() == 3   # router, expert-tile FFN, combine
    assert make_layer(s, gemm_kernels="expert_tile").kernels_per_forward() == 3
    assert make_layer(s, gemm_kernels="grouped").kernels_per_forward() == 4  # up, down
    assert make_layer(small(tokens=500, d_model=192, d_ff=768),
                      gemm_kernels="expert_tile").kernels_per_forward() == 4  # d % 128 != 0
    assert make_layer(small("f32", tokens=64)).kernels_per_forward() == 6


def test_kernels_per_forward_streaming():
    L = make_layer(small(tokens=500), gemm_kernels="streaming")
    assert L.kernels_per_forward() == 5   # + tile list


@pytest.mark.parametrize("shape", [
    dict(d_model=64, d_ff=256, n_experts=2, n_blocks=2),     # B = 2: b = 1 always
    dict(d_model=192, d_ff=768, n_experts=6, n_blocks=4),
    dict(d_model=256, d_ff=2048, n_experts=3, n_blocks=8),   # M = 256
    dict(d_model=384, d_ff=3072, n_experts=5, n_blocks=8),   # M = 384: two N sub-tiles
    dict(d_model=320, d_ff=1280, n_experts=4, n_blocks=5),   # d = 5 x 64
])
def test_shapes(shape):
    wl = workloads.make_workload(small(tokens=700, **shape))
    g = run_gpu(wl)
    if shape["n_blocks"] == 2:
        assert (g.b == 1).all()
    assert_parity(wl, g, compare(wl, g))


# ------------------------------------------------- ablation switches (Table IV)

@pytest.mark.parametrize("kw", [
    dict(alpha_fixed=0.4),
    dict(topk_fixed=2),
    dict(prefix_blocks=1),
    dict(beta_fixed=0.7),
    dict(tau=0.05),
])
def test_threshold_variants(kw):
    wl = workloads.make_workload(small(tokens=900, n_experts=6, n_blocks=8, d_ff=1024, **kw))
    g = run_gpu(wl)
    assert_parity(wl, g, compare(wl, g))


def test_alpha_one_is_dense_ffn():
    """alpha = 1: every block shared, y = E_shr(x) (Eq. 4)."""
    wl = workloads.make_workload(small(tokens=500, alpha_fixed=1.0))
    g = run_gpu(wl)
    assert (g.b == wl.spec.n_blocks).all()
    x = wl.x.double().numpy()
    wu = wl.w_up[0].double().numpy()
    wd = wl.w_down[0].double().numpy()
    from scipy.stats import norm
    a = x @ wu.T
    dense = (a * norm.cdf(a)) @ wd.T
    rel = np.abs(g.y - dense).max(axis=1) / np.abs(dense).max(axis=1)
    assert rel.max() < 2e-2


def test_alpha_zero_all_experts_is_soft_moe():
    wl = workloads.make_workload(small(tokens=400, alpha_fixed=0.0, beta_fixed=1.0))
    g = run_gpu(wl)
    assert (g.b == 0).all() and (g.k == wl.spec.n_experts).all()
    assert_parity(wl, g, compare(wl, g))


def test_f32_variants():
    wl = workloads.make_workload(workloads.spec("tiny_f32", tokens=1000, topk_fixed=2))
    g = run_gpu(wl)
    assert_parity(wl, g, compare(wl, g))


# ------------------------------------------------------------ group table

@pytest.mark.parametrize("kernels", ["expert_tile", "grouped"])
def test_group_table_matches_oracle(kernels):
    """The (expert, block) group table: read from the device grouping
    ("grouped"), or derived from the routing records when the device
    grouped the rows by expert (the expert-tile FFN)."""
    wl = workloads.make_workload(small(tokens=1500, n_experts=6, n_blocks=8, d_ff=1024))
    g = run_gpu(wl, gemm_kernels=kernels)
    counts, offsets, tok, w = g.layer.groups()
    r = oracle.with_decisions(compare_routing(wl), g.shr, g.em, wl.spec.n_blocks)
    c_ref, tok_ref, w_ref = oracle.groups(r, wl.spec.n_experts, wl.spec.n_blocks)
    assert counts.numpy().tolist() == c_ref.tolist()
    offs = offsets.numpy()
    assert (offs[1:] - offs[:-1]).tolist() == [(c + 127) // 128 * 128 for c in c_ref]
    start = np.concatenate([[0], np.cumsum(c_ref)])
    for gi in range(len(c_ref)):
        got = tok.numpy()[offs[gi]:offs[gi] + c_ref[gi]]
        assert got.tolist() == tok_ref[start[gi]:start[gi + 1]].tolist()
        np.testing.assert_allclose(w.numpy()[offs[gi]:offs[gi] + c_ref[gi]],
                                   w_ref[start[gi]:start[gi + 1]], rtol=1e-5, atol=1e-7)
        assert (tok.numpy()[offs[gi] + c_ref[gi]:offs[gi + 1]] == -1).all()


def compare_routing(wl):
    from gpu_helpers import oracle_routing
    return oracle_routing(wl)


def test_permuting_tokens_permutes_outputs():
    wl = workloads.make_workload(small(tokens=600))
    g = run_gpu(wl)
    perm = torch.from_numpy(np.random.default_rng(1).permutation(600))
    g2 = run_gpu(wl, layer=g.layer, x=wl.x[perm], mask=None)
    pn = perm.numpy()
    assert np.array_equal(g2.b, g.b[pn]) and np.array_equal(g2.shr, g.shr[pn])
    assert np.array_equal(g2.em, g.em[pn])
    np.testing.assert_allclose(g2.y, g.y[pn], rtol=1e-2, atol=1e-6)  # one bf16 ulp


# ------------------------------------------------------------- ABI behaviour

def test_errors_are_reported():
    from paper_2608_10392_gb300 import UnifMoeError
    wl = workloads.make_workload(small(tokens=64))
    layer = make_layer(wl.spec)
    dev = torch.device("cuda")
    x = wl.x.to(dev)
    with pytest.raises(UnifMoeError) as e:
        layer.forward(x)  # no weights yet
    assert e.value.code == -6
    layer.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    big = torch.zeros(65, wl.spec.d_model, dtype=torch.bfloat16, device=dev)
    with pytest.raises(UnifMoeError) as e:
        layer.forward(big)
    assert e.value.code == -3
    raw = torch.zeros(64 * wl.spec.d_model + 8, dtype=torch.bfloat16, device=dev)
    mis = raw[1:1 + 64 * wl.spec.d_model].view(64, wl.spec.d_model)
    with pytest.raises(UnifMoeError) as e:
        layer.forward(mis)
    assert e.value.code == -1
    with pytest.raises(UnifMoeError):
        make_layer(wl.spec.with_(d_ff=500))  # H % B != 0
    with pytest.raises(UnifMoeError):
        make_layer(wl.spec.with_(d_model=96))  # bf16 needs d % 64 == 0


def test_forward_calls_allocate_nothing():
    """Every buffer a forward-family call needs is allocated at create time:
    the device's free memory does not move across a fresh handle's first
    forward, norm-first and norm-after sublayer forwards and host-buffer
    forwards (kernel modules loaded beforehand by another handle; every
    torch output allocated beforehand)."""
    s = workloads.spec("vit_s")
    wl = workloads.make_workload(s)
    dev = torch.device("cuda")
    d = s.d_model
    x = wl.x.to(dev)
    out = torch.empty_like(x)
    b = torch.empty(s.tokens, dtype=torch.int32, device=dev)
    k = torch.empty_like(b)
    gamma = torch.ones(d, dtype=torch.bfloat16, device=dev)
    beta = torch.zeros(d, dtype=torch.bfloat16, device=dev)
    xh = wl.x.pin_memory()
    oh = torch.empty_like(xh).pin_memory()
    xp, op = wl.x.clone(), torch.empty_like(wl.x)  # pageable: staging buffers and copies
    bh = torch.empty(s.tokens, dtype=torch.int32)

    def every_call(L):
        L.forward(x, out=out, shared_counts=b, residual_counts=k)
        L.sublayer_forward(x, gamma, beta, 1e-5, True, out=out)
        L.sublayer_forward(x, gamma, beta, 1e-5, False, out=out)
        L.forward_host(xh, oh, shared_counts_host=bh)
        L.forward_host(xp, op, shared_counts_host=bh)
        torch.cuda.synchronize()
        assert L.sync_status() == 0

    def fresh():
        L = make_layer(s)
        L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
        torch.cuda.synchronize()
        return L

    every_call(fresh())  # loads every kernel the calls launch
    L = fresh()
    free0 = torch.cuda.mem_get_info()[0]
    every_call(L)
    assert torch.cuda.mem_get_info()[0] == free0


def test_features_left_out_are_refused():
    """A handle created without the optional workspaces refuses the calls
    that need them (ERR_STATE) and runs the rest."""
    from paper_2608_10392_gb300 import UnifMoeError
    wl = workloads.make_workload(small(tokens=256))
    dev = torch.device("cuda")
    L = make_layer(wl.spec, features=0)
    L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    x = wl.x.to(dev)
    d = wl.spec.d_model
    gamma = torch.ones(d, dtype=torch.bfloat16, device=dev)
    beta = torch.zeros(d, dtype=torch.bfloat16, device=dev)
    with pytest.raises(UnifMoeError) as e:
        L.sublayer_forward(x, gamma, beta, 1e-5, True)
    assert e.value.code == -6
    with pytest.raises(UnifMoeError) as e:
        L.forward_host(wl.x.clone(), torch.empty_like(wl.x))
    assert e.value.code == -6
    y = L.forward(x)
    z = L.sublayer_forward(x, gamma, beta, 1e-5, False)
    torch.cuda.synchronize()
    assert L.sync_status() == 0
    assert torch.isfinite(y.float()).all() and torch.isfinite(z.float()).all()


def test_output_guard_bands():
    wl = workloads.make_workload(small(tokens=257))
    layer = make_layer(wl.spec)
    dev = torch.device("cuda")
    layer.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    d = wl.spec.d_model
    buf = torch.full((257 + 4, d), 7.0, dtype=torch.bfloat16, device=dev)
    out = buf[2:2 + 257]
    layer.forward(wl.x.to(dev), out=out)
    torch.cuda.synchronize()
    assert (buf[:2] == 7.0).all() and (buf[-2:] == 7.0).all()


def test_timeout_status_path():
    """A bounded wait that runs out is reported, and the context stays usable."""
    wl = workloads.make_workload(small(tokens=128))
    layer = make_layer(wl.spec)
    assert layer.sync_status() == 0
    layer.selftest_timeout(2000)
    assert layer.sync_status() == -5
    assert layer.sync_status() == 0  # cleared
    g = run_gpu(wl, layer=None)
    assert_parity(wl, g, compare(wl, g))


def test_forward_host_matches_device():
    wl = workloads.make_workload(small(tokens=500))
    g = run_gpu(wl)
    xh = wl.x.pin_memory()
    out = torch.empty_like(xh).pin_memory()
    b = torch.empty(500, dtype=torch.int32).pin_memory()
    k = torch.empty(500, dtype=torch.int32).pin_memory()
    g.layer.forward_host(xh, out, shared_counts_host=b, residual_counts_host=k)
    np.testing.assert_allclose(out.float().numpy(), g.y, rtol=1e-2, atol=1e-6)  # one bf16 ulp
    assert np.array_equal(b.numpy(), g.b) and np.array_equal(k.numpy(), g.k)


def test_forward_host_pageable_buffers():
    """Pageable host buffers go through the staging buffers and copies."""
    wl = workloads.make_workload(small(tokens=500))
    g = run_gpu(wl)
    xh = wl.x.clone()
    out = torch.empty_like(xh)
    b = torch.empty(500, dtype=torch.int32)
    k = torch.empty(500, dtype=torch.int32)
    g.layer.forward_host(xh, out, shared_counts_host=b, residual_counts_host=k)
    np.testing.assert_allclose(out.float().numpy(), g.y, rtol=1e-2, atol=1e-6)  # one bf16 ulp
    assert np.array_equal(b.numpy(), g.b) and np.array_equal(k.numpy(), g.k)


def test_forward_host_async_pipeline():
    """Pipelined host-buffer forwards: four different batches (different
    sizes, a padding mask on two) enqueued back to back, so that both staging
    slots are refilled while earlier calls' kernels and copies are in flight;
    each call's output and counts match the device forward of its batch, and
    a synchronous host-buffer forward afterwards is unaffected."""
    base = workloads.make_workload(small(tokens=700))
    layer = run_gpu(base).layer
    dev = torch.device("cuda")
    gen = torch.Generator().manual_seed(5)
    batches = []
    for i, T in enumerate([700, 513, 640, 128]):
        idx = torch.randperm(700, generator=gen)[:T]
        x = (base.x[idx].float() * (1.0 + 0.1 * i)).to(base.x.dtype)
        m = None if i % 2 == 0 else (torch.rand(T, generator=gen) > 0.2).to(torch.uint8)
        b = torch.empty(T, dtype=torch.int32, device=dev)
        k = torch.empty(T, dtype=torch.int32, device=dev)
        y = layer.forward(x.to(dev), mask=None if m is None else m.to(dev), shared_counts=b,
                          residual_counts=k)
        torch.cuda.synchronize()
        batches.append((x, m, y.float().cpu(), b.cpu(), k.cpu()))
    pending = []
    for x, m, *_ in batches:
        T = x.shape[0]
        xh = x.pin_memory()
        mh = None if m is None else m.pin_memory()
        oh = torch.full_like(xh, float("nan")).pin_memory()
        bh = torch.full((T,), -7, dtype=torch.int32).pin_memory()
        kh = torch.full((T,), -7, dtype=torch.int32).pin_memory()
        layer.forward_host_async(xh, oh, mh, bh, kh)
        pending.append((xh, mh, oh, bh, kh))
    layer.forward_host_wait()
    torch.cuda.synchronize()
    assert layer.sync_status() == 0
    for (x, m, y, b, k), (_, _, oh, bh, kh) in zip(batches, pending):
        np.testing.assert_allclose(oh.float().numpy(), y.numpy(), rtol=1e-2, atol=1e-6)
        assert np.array_equal(bh.numpy(), b.numpy()) and np.array_equal(kh.numpy(), k.numpy())
    x, m, y, b, k = batches[1]
    out = torch.empty_like(x).pin_memory()
    bh = torch.empty(x.shape[0], dtype=torch.int32).pin_memory()
    layer.forward_host(x.pin_memory(), out, m.pin_memory(), shared_counts_host=bh)
    np.testing.assert_allclose(out.float().numpy(), y.numpy(), rtol=1e-2, atol=1e-6)
    assert np.array_equal(bh.numpy(), b.numpy())


# ------------------------------------------- GEMM kernel variants

GEMM_FAMILY = {"expert_tile": "expert_tile", "weight_stationary": "grouped",
               "streaming": "streaming"}


@pytest.mark.parametrize("kernels", list(GEMM_FAMILY))
def test_gemm_variants_many_group_runs(kernels):
    """Enough tiles that every CTA walks several group runs (weight slabs
    reloaded mid-run; several expert tiles per CTA), on every GEMM kernel
    family."""
    wl = workloads.make_workload(small(tokens=6000, d_model=128, d_ff=512, n_experts=8,
                                       n_blocks=4))
    g = run_gpu(wl, gemm_kernels=GEMM_FAMILY[kernels])
    assert_parity(wl, g, compare(wl, g, label=kernels))


@pytest.mark.parametrize("shape", [
    dict(d_model=128, d_ff=384, n_experts=3, n_blocks=6),     # M = 64: two blocks per chunk
    dict(d_model=256, d_ff=1536, n_experts=8, n_blocks=8),    # M = 192: blocks across chunks
    dict(d_model=384, d_ff=1024, n_experts=2, n_blocks=16),   # M = 64, B = 16
])
def test_expert_tile_shapes(shape):
    """The expert-tile FFN where blocks and 128-channel chunks do not line
    up, on ragged token counts (partial last tiles of every expert)."""
    wl = workloads.make_workload(small(tokens=1111, **shape))
    g = run_gpu(wl, gemm_kernels="expert_tile")
    assert g.layer.kernels_per_forward() == 3
    assert_parity(wl, g, compare(wl, g, label="expert_tile"))


def test_expert_tile_padding_mask():
    """Text-style batch (valid lengths uniform per sequence, padding tokens
    NaN-filled and masked) through the expert-tile FFN: padding tokens get no
    rows, their outputs are exactly zero, the NaNs reach no valid token, and
    every valid token's decisions and output match the oracle."""
    s = workloads.spec("bert_base").with_(tokens=2048, d_model=256, d_ff=1024, n_experts=8,
                                          n_blocks=8)
    wl = workloads.make_workload(s)
    g = run_gpu(wl)
    assert g.layer.kernels_per_forward() == 3
    m = wl.mask.numpy()
    assert 0 < int(m.sum()) < s.tokens
    assert (g.b[m == 0] == 0).all() and (g.k[m == 0] == 0).all()
    assert (g.y[m == 0] == 0).all() and np.isfinite(g.y).all()
    assert_parity(wl, g, compare(wl, g, label="expert_tile, padding"))


def test_vit_s_streaming_kernels():
    """The ViT-S layer through the streaming GEMMs agrees with the oracle too."""
    wl = workloads.make_workload(workloads.spec("vit_s", tokens=4000))
    g = run_gpu(wl, gemm_kernels="streaming")
    assert_parity(wl, g, compare(wl, g, label="streaming"))


def test_repeated_forwards_match_streaming_kernels():
    """Ten forwards of the ViT-S layer through the expert-tile FFN, and ten
    through the weight-stationary kernels, agree with the streaming kernels
    token by token (the two differ only in
    the order of the fp32 additions into the accumulator): catches
    synchronisation races that corrupt a tile now and then."""
    s = workloads.spec("vit_s")
    wl = workloads.make_workload(s)
    dev = torch.device("cuda")

    def layer(kernels):
        L = make_layer(s, gemm_kernels=kernels)
        L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
        return L

    x = wl.x.to(dev)
    ref = layer("streaming").forward(x).float()
    for kernels in ("expert_tile", "grouped"):
        L = layer(kernels)
        for _ in range(10):
            y = L.forward(x).float()
            torch.cuda.synchronize()
            assert L.sync_status() == 0
            rel = (y - ref).abs().amax(1) / ref.abs().amax(1).clamp_min(1e-6)
            assert float(rel.max()) < 1e-2, (kernels, int((rel >= 1e-2).sum()))


def test_repeated_forwards_sliced_down_projection():
    """A ViT-B-shaped layer (d = 768: the weight-stationary down projection
    runs in three 256-column slices) agrees with the streaming kernels over
    repeated forwards, and with the oracle on every token."""
    s = workloads.spec("vit_b", tokens=3000)
    wl = workloads.make_workload(s)
    dev = torch.device("cuda")

    def layer(kernels):
        L = make_layer(s, gemm_kernels=kernels)
        L.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
        return L

    x = wl.x.to(dev)
    ref = layer("streaming").forward(x).float()
    L = layer("auto")
    for _ in range(5):
        y = L.forward(x).float()
        torch.cuda.synchronize()
        assert L.sync_status() == 0
        rel = (y - ref).abs().amax(1) / ref.abs().amax(1).clamp_min(1e-6)
        assert float(rel.max()) < 1e-2, int((rel >= 1e-2).sum())
    g = run_gpu(wl, layer=L)
    assert_parity(wl, g, compare(wl, g, label="sliced down projection"))

