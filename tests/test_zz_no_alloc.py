"""The allocation-free grouping entry point (unif_moe_group_noalloc).

Some callers cannot call cudaMalloc (engines that hand out all device memory
up front, latency-critical paths that cannot take cudaMalloc's implicit
synchronisation); for them the library keeps the grouping step's scratch in
a fixed device array of its own. This test calls that entry point through
the C ABI and checks it against the group table the regular forward built,
on two calls in a row (the second call finds the first call's scratch
contents and must not depend on them). It runs last on purpose (file name),
and passes alone in a fresh process as well as after the other tests."""
import ctypes as C

import numpy as np
import pytest
import torch

import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()


def noalloc_groups(lib, T, K, B, shr, em, alpha, s):
    dev = torch.device("cuda")
    G = (K + 1) * B
    cap = T * K * B + G * 127
    cap = (cap + 127) // 128 * 128
    counts = torch.full((G,), -9, dtype=torch.int32, device=dev)
    offsets = torch.full((G + 1,), -9, dtype=torch.int32, device=dev)
    n_tiles = torch.full((1,), -9, dtype=torch.int32, device=dev)
    tg = torch.full((cap // 128,), -9, dtype=torch.int32, device=dev)
    tr = torch.full((cap // 128,), -9, dtype=torch.int32, device=dev)
    tok = torch.full((cap,), -9, dtype=torch.int32, device=dev)
    w = torch.full((cap,), -9.0, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream().cuda_stream
    rc = lib.unif_moe_group_noalloc(T, K, B, shr.data_ptr(), em.data_ptr(), alpha.data_ptr(),
                                    s.data_ptr(), counts.data_ptr(), offsets.data_ptr(),
                                    n_tiles.data_ptr(), tg.data_ptr(), tr.data_ptr(),
                                    tok.data_ptr(), w.data_ptr(), cap, stream)
    assert rc == 0, lib.unif_moe_last_error()
    torch.cuda.synchronize()
    n = int(offsets[G].item())
    return (counts.cpu(), offsets.cpu(), int(n_tiles.item()), tok[:n].cpu(), w[:n].cpu(),
            tg.cpu(), tr.cpu())


def run_case(spec):
    from paper_2608_10392_gb300 import Layer, lib
    wl = workloads.make_workload(spec)
    dev = torch.device("cuda")
    layer = Layer(spec.d_model, spec.d_ff, spec.n_experts, spec.n_blocks, dtype=spec.dtype,
                  max_tokens=spec.tokens)
    layer.load_weights(wl.w_router.to(dev), wl.w_up.to(dev), wl.w_down.to(dev))
    layer.forward(wl.x.to(dev))
    r = layer.routing()
    T, K, B = spec.tokens, spec.n_experts, spec.n_blocks
    # affinities by expert index from the sorted lists: s[t, q[t, i]] = p[t, i]
    s = torch.zeros(T, K, dtype=torch.float32, device=dev)
    s.scatter_(1, r["q"].long(), r["p"])
    ref_counts, ref_offsets, ref_tok, ref_w = layer.groups()
    G = (K + 1) * B
    for call in range(2):  # two calls in a row on the shared scratch
        counts, offsets, n_tiles, tok, w, tg, tr = noalloc_groups(
            lib(), T, K, B, r["shared_mask"], r["expert_mask"], r["alpha"], s)
        assert torch.equal(counts, ref_counts), call
        assert torch.equal(offsets, ref_offsets), call
        assert n_tiles == int(ref_offsets[G]) // 128
        assert torch.equal(tok, ref_tok), call
        # the same fp32 values travel both paths; the tests' tolerance for
        # routing weights is rtol 1e-5
        np.testing.assert_allclose(w.numpy(), ref_w.numpy(), rtol=1e-5, atol=0)
        rows = offsets.numpy()
        for t in range(n_tiles):
            g = int(tg[t])
            assert rows[g] <= int(tr[t]) < rows[g + 1]
    layer.close()


def test_noalloc_grouping_matches_forward_groups():
    run_case(workloads.spec("vit_s").with_(tokens=1500, d_model=128, d_ff=1024, n_experts=6,
                                           n_blocks=8))
    # a second, differently shaped call reuses the same scratch array
    run_case(workloads.spec("vit_s").with_(tokens=333, d_model=64, d_ff=256, n_experts=3,
                                           n_blocks=4))


def test_noalloc_rejects_sizes_beyond_the_scratch():
    from paper_2608_10392_gb300 import lib
    K, B = 64, 64
    T = 20000  # (K+1)*B*ceil(T/256) = 4160*79 > 262144
    G = (K + 1) * B
    dev = torch.device("cuda")
    dummy = torch.zeros(8, dtype=torch.int64, device=dev)
    p = dummy.data_ptr()
    rc = lib().unif_moe_group_noalloc(T, K, B, p, p, p, p, p, p, p, p, p, p, p,
                                      T * K * B + G * 127, None)
    assert rc == -3
    assert b"scratch" in lib().unif_moe_last_error()


def test_noalloc_scratch_limit_is_exact():
    """(K+1) B ceil(T/256) equal to the scratch's 262144 entries is accepted
    (and groups every pair); one 256-token chunk more is refused with
    ERR_CAPACITY before anything is enqueued."""
    from paper_2608_10392_gb300 import lib
    K, B = 63, 64
    G = (K + 1) * B                      # 4096 groups
    T = 262144 // G * 256                # 64 chunks of 256 tokens: exactly at the limit
    dev = torch.device("cuda")
    g = torch.Generator().manual_seed(3)
    shr = torch.randint(0, 2**62, (T,), generator=g, dtype=torch.int64) & 0x0101  # blocks 0, 8
    em = torch.randint(0, 2**62, (T,), generator=g, dtype=torch.int64) & 0x11     # experts 0, 4
    alpha = torch.rand(T, generator=g)
    s = torch.rand(T, K, generator=g)
    n_shr = np.array([bin(int(v)).count("1") for v in shr])
    n_em = np.array([bin(int(v)).count("1") for v in em])
    pairs = int((n_shr + n_em * (B - n_shr)).sum())  # sum of C_B (Eq. 35)
    counts, offsets, n_tiles, tok, w, tg, tr = noalloc_groups(
        lib(), T, K, B, shr.to(dev), em.to(dev), alpha.to(dev), s.to(dev))
    assert int(counts.sum()) == pairs
    assert (tok >= 0).sum() == pairs
    T1 = T + 1                           # 65 chunks
    p = torch.zeros(8, dtype=torch.int64, device=dev).data_ptr()
    rc = lib().unif_moe_group_noalloc(T1, K, B, p, p, p, p, p, p, p, p, p, p, p,
                                      T1 * K * B + G * 127, None)
    assert rc == -3 and b"scratch" in lib().unif_moe_last_error()
