"""Host-side logic on the CPU: the seeded workload generators (shapes, value
distributions and structure the parity tests and the bench rely on) and the
multi-rank bookkeeping of bench.py, run as two gloo ranks."""
import math
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import workloads


# ------------------------------------------------------------ generators

def test_generators_are_deterministic():
    s = workloads.spec("tiny_f32")
    a, b = workloads.make_workload(s), workloads.make_workload(s)
    for u, v in ((a.x, b.x), (a.w_up, b.w_up), (a.w_down, b.w_down), (a.w_router, b.w_router)):
        assert torch.equal(u, v)


@pytest.mark.parametrize("name", list(workloads.CONFIGS))
def test_weight_shapes_and_dtypes(name):
    s = workloads.spec(name)
    wr, wu, wd, bias = workloads.make_weights(s.with_(d_model=64, d_ff=s.n_blocks * 64))
    K, B = s.n_experts, s.n_blocks
    dt = torch.float32 if s.dtype == "f32" else torch.bfloat16
    assert wr.shape == (64, K + 1) and wr.dtype == dt
    assert wu.shape == (K + 1, B * 64, 64) and wu.dtype == dt
    assert wd.shape == (K + 1, 64, B * 64) and wd.dtype == dt
    assert (bias is None) == (s.zipf_s == 0)


def test_upcycled_experts_are_close_to_one_base():
    s = workloads.spec("vit_s", d_model=128, d_ff=512)
    _, wu, wd, _ = workloads.make_weights(s)
    wu = wu.float()
    # every expert = base + 5% perturbation: pairwise differences are ~7% of the weights
    rel = (wu[1] - wu[2]).norm() / wu[1].norm()
    assert 0.04 < rel < 0.11
    assert abs(wu.std().item() - 1 / math.sqrt(128)) < 0.1 / math.sqrt(128)
    assert abs(wd.float().std().item() - 1 / math.sqrt(512)) < 0.1 / math.sqrt(512)


def test_text_padding_structure():
    s = workloads.spec("bert_base", d_model=64, d_ff=512)
    wl = workloads.make_workload(s)
    m = wl.mask.view(-1, s.seq_len)
    lens = m.sum(1)
    assert lens.min() >= s.min_len and lens.max() <= s.seq_len
    # valid tokens form a prefix of each sequence; padding rows are NaN
    assert (m[:, :-1] >= m[:, 1:]).all()
    assert torch.isnan(wl.x[wl.mask == 0].float()).all()
    assert torch.isfinite(wl.x[wl.mask == 1].float()).all()


def test_stress_clusters_and_zipf_prior():
    s = workloads.spec("stress", tokens=4096, d_model=128, d_ff=512)
    wl = workloads.make_workload(s)
    bias = wl.router_bias
    assert bias[0] == 0 and torch.all(bias[1:-1] > bias[2:])
    assert torch.allclose(bias[2], torch.tensor(-1.2 * math.log(2.0)))
    # the shared logit x . W_shr separates into the four cluster levels
    w = wl.w_router.float()[:, 0]
    proj = wl.x.float() @ w
    lv = proj.sort().values
    q = [lv[int(f * len(lv))].item() for f in (0.1, 0.35, 0.65, 0.9)]
    assert q[0] < -4 and -4 < q[1] < 0 and 0 < q[2] < 4 and q[3] > 4


def test_rank_batches_are_independent():
    s = workloads.spec("vit_s", tokens=256, d_model=64, d_ff=512)
    wr = workloads.make_weights(s)[0]
    x0, _ = workloads.make_tokens(s, wr, seed=bench.rank_token_seed(s, 0))
    x0b, _ = workloads.make_tokens(s, wr)
    x1, _ = workloads.make_tokens(s, wr, seed=bench.rank_token_seed(s, 1))
    assert torch.equal(x0, x0b)          # rank 0 runs the workload's own batch
    assert not torch.equal(x0, x1)       # other ranks draw their own tokens


def test_single_rank_bookkeeping():
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.sum_over_ranks(7) == 7.0
    assert bench.job_throughput(12608, 0.5) == pytest.approx(12608 / 0.5e-3)


# ------------------------------------------------------------ two gloo ranks

def _free_port():
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        return sk.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each rank times its own batch: the job time is the slowest rank's,
        # the job's tokens the sum of every rank's valid tokens
        ms = [0.25, 0.40][rank]
        valid = [1000, 900][rank]
        t = bench.max_over_ranks(ms, dist)
        n = bench.sum_over_ranks(valid, dist)
        q.put((rank, t, n, bench.job_throughput(n, t)))
    finally:
        dist.destroy_process_group()


def test_two_rank_weak_scaling_bookkeeping():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, t, n, v in res:
        assert t == 0.40 and n == 1900.0
        assert v == pytest.approx(1900 / 0.40e-3)
