"""Pins for the CPU oracle: checks against facts the paper and the mathematics
fix, computed here by other means than the oracle's own code (dense matrix
products, exhaustive search over subsets, a hand derivation, library routines
for the normal CDF and the logistic function).

Each test names the passage it pins. None needs a GPU.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
from scipy.special import expit, softmax
from scipy.stats import norm

import oracle
from oracle import Thresholds

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def gelu_ref(v):
    # GeLU(v) = v * Phi(v), Phi the standard normal CDF (library routine).
    return v * norm.cdf(v)


def rand_layer(rng, d, H, K, B, router_scale=1.0, T=64):
    x = rng.standard_normal((T, d))
    w_router = rng.standard_normal((d, K + 1)) * router_scale / math.sqrt(d)
    w_up = rng.standard_normal((K + 1, H, d)) / math.sqrt(d)
    w_down = rng.standard_normal((K + 1, d, H)) / math.sqrt(H)
    return x, w_router, w_up, w_down


def block_outputs_dense(x, w_up, w_down, B):
    """All (K+1)*B block outputs E_e^(b)(x) for every token, by dense matrix
    products: [T][K+1][B][d] (Eq. 16)."""
    T = x.shape[0]
    E1, H, d = w_up.shape
    M = H // B
    out = np.zeros((T, E1, B, d))
    for e in range(E1):
        act = gelu_ref(x @ w_up[e].T)  # [T][H]
        for blk in range(B):
            sl = slice(blk * M, (blk + 1) * M)
            out[:, e, blk, :] = act[:, sl] @ w_down[e][:, sl].T
    return out


# --------------------------------------------------------------------------
# Hand-derived example (Sec. III, Eqs. 16-30 and 35)
# --------------------------------------------------------------------------

def _num(v):
    if isinstance(v, str):
        return {"ln3/2": math.log(3) / 2}[v]
    return float(v)


def load_hand():
    g = json.load(open(os.path.join(GOLDEN, "hand_example.json")))
    x = np.array(g["x"], dtype=np.float64)
    w_router = np.array([[_num(v) for v in row] for row in g["w_router"]])
    w_up = np.array(g["w_up"], dtype=np.float64)
    vr = np.array(g["value_rows"], dtype=np.float64)  # [K+1][H][d]
    w_down = np.ascontiguousarray(vr.transpose(0, 2, 1))  # [K+1][d][H]
    mask = np.array(g["mask"], dtype=np.uint8)
    return g, x, w_router, w_up, w_down, mask


def test_hand_example_decisions_and_output(oracle_mod):
    g, x, w_router, w_up, w_down, mask = load_hand()
    B = g["B"]
    y, r = oracle.layer(x, w_router, w_up, w_down, B, mask=mask)
    exp = g["expected"]
    assert r.b.tolist() == exp["b"]
    assert r.k.tolist() == exp["k"]
    for t in range(3):
        blocks = [blk for blk in range(B) if (int(r.shr_mask[t]) >> blk) & 1]
        assert blocks == exp["shared_blocks"][t]
        experts = sorted(int(r.q[t, i]) + 1 for i in range(r.k[t]))
        assert experts == exp["experts"][t]
    assert r.cb(B).tolist() == exp["C_B"]
    alpha = [0.5, 0.25 + expit(-3.0) / 2, 0.0]
    np.testing.assert_allclose(r.alpha, alpha, rtol=0, atol=1e-15)
    s = {0: (0.75, 0.25), 1: (math.sqrt(3) / (1 + math.sqrt(3)), 1 / (1 + math.sqrt(3)))}
    for t in range(3):
        want = np.zeros(2)
        for coef, pre, val in exp["output_terms"][t]:
            c = {"alpha": alpha[t], "s1": s.get(t, (0, 0))[0], "s2": s.get(t, (0, 0))[1]}[coef]
            want += c * gelu_ref(pre) * np.array(val, dtype=np.float64)
        np.testing.assert_allclose(y[t], want, rtol=1e-13, atol=1e-15)


def test_hand_example_groups(oracle_mod):
    g, x, w_router, w_up, w_down, mask = load_hand()
    B, K = g["B"], g["K"]
    _, r = oracle.layer(x, w_router, w_up, w_down, B, mask=mask)
    counts, tok, w = oracle.groups(r, K, B, mask)
    assert counts.tolist() == g["expected"]["groups"]["counts"]
    assert tok.tolist() == g["expected"]["groups"]["tokens"]
    # weights: alpha on shared groups, p on residual groups
    sA, sB = 0.75, math.sqrt(3) / (1 + math.sqrt(3))
    np.testing.assert_allclose(w, [0.5, 0.25 + expit(-3.0) / 2, sB, sA, 1 - sB], atol=1e-15)


# --------------------------------------------------------------------------
# Exhaustive search on tiny layers (Eqs. 18-30 by enumeration)
# --------------------------------------------------------------------------

def brute_force(x, w_router, w_up, w_down, B, th: Thresholds, bias=None):
    """Decisions by exhaustive search and the output as a masked sum of dense
    block outputs. No sorting: the shared set is the b-subset with the
    largest total priority (with prefix selection, Table IV, the blocks
    0..b-1), the residual set the smallest subset of experts whose affinity
    mass reaches beta (largest mass among subsets of that size; with a fixed
    top-k, the k-subset of largest mass). `bias` is added to the router
    logits x W* column by column."""
    T, d = x.shape
    K = w_up.shape[0] - 1
    H = w_up.shape[1]
    M = H // B
    tau = (B - 1) / B**2 if math.isnan(th.tau) else th.tau
    mu = np.stack([w_up[0, blk * M:(blk + 1) * M, :].mean(axis=0) for blk in range(B)])
    blocks = block_outputs_dense(x, w_up, w_down, B)
    ys, bs, ks, shr_sets, exp_sets = [], [], [], [], []
    for t in range(T):
        z = x[t] @ w_router + (0.0 if bias is None else bias)
        alpha = tau + (1 - 2 * tau) * expit(z[0]) if math.isnan(th.alpha_fixed) else th.alpha_fixed
        b = int(np.rint(B * alpha))
        u = mu @ x[t]
        if th.prefix_blocks:
            shr = set(range(b))
        else:
            best = max(itertools.combinations(range(B), b), key=lambda S: sum(u[i] for i in S))
            shr = set(best)
        s = softmax(z[1:])
        beta = 1 - alpha if math.isnan(th.beta_fixed) else th.beta_fixed
        chosen = None
        for n in range(1, K + 1):
            S = max(itertools.combinations(range(K), n), key=lambda S: sum(s[j] for j in S))
            if th.topk_fixed:
                if n == th.topk_fixed:
                    chosen = S
                    break
            elif sum(s[j] for j in S) >= beta or n == K:
                chosen = S
                break
        y = alpha * sum(blocks[t, 0, blk] for blk in shr) if shr else np.zeros(d)
        for j in chosen:
            y = y + s[j] * sum((blocks[t, 1 + j, blk] for blk in range(B) if blk not in shr),
                               np.zeros(d))
        ys.append(y)
        bs.append(b)
        ks.append(len(chosen))
        shr_sets.append(shr)
        exp_sets.append(set(chosen))
    return np.array(ys), np.array(bs), np.array(ks), shr_sets, exp_sets


@pytest.mark.parametrize("d,H,K,B", [(4, 8, 3, 2), (8, 16, 4, 4), (5, 12, 2, 4), (6, 16, 4, 2)])
@pytest.mark.parametrize("seed", [0, 1])
def test_brute_force_tiny(oracle_mod, d, H, K, B, seed):
    rng = np.random.default_rng(100 * seed + d)
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, router_scale=3.0, T=48)
    th = Thresholds()
    y, r = oracle.layer(x, w_router, w_up, w_down, B, th)
    yb, bb, kb, shr, exps = brute_force(x, w_router, w_up, w_down, B, th)
    assert r.b.tolist() == bb.tolist()
    assert r.k.tolist() == kb.tolist()
    em = r.expert_mask()
    for t in range(x.shape[0]):
        assert {blk for blk in range(B) if (int(r.shr_mask[t]) >> blk) & 1} == shr[t]
        assert {j for j in range(K) if (int(em[t]) >> j) & 1} == exps[t]
    np.testing.assert_allclose(y, yb, rtol=1e-11, atol=1e-13)


@pytest.mark.parametrize("th", [Thresholds(beta_fixed=0.7), Thresholds(alpha_fixed=0.4),
                                Thresholds(tau=0.1), Thresholds(prefix_blocks=1),
                                Thresholds(topk_fixed=2),
                                Thresholds(prefix_blocks=1, topk_fixed=3, alpha_fixed=0.3)])
def test_brute_force_threshold_variants(oracle_mod, th):
    """The Table IV ablation switches (fixed alpha, fixed top-k, prefix block
    selection) and the fixed thresholds, against exhaustive search."""
    rng = np.random.default_rng(7)
    x, w_router, w_up, w_down = rand_layer(rng, 6, 16, 4, 4, router_scale=3.0, T=40)
    y, r = oracle.layer(x, w_router, w_up, w_down, 4, th)
    yb, bb, kb, shr, exps = brute_force(x, w_router, w_up, w_down, 4, th)
    assert r.b.tolist() == bb.tolist() and r.k.tolist() == kb.tolist()
    em = r.expert_mask()
    for t in range(x.shape[0]):
        assert {blk for blk in range(4) if (int(r.shr_mask[t]) >> blk) & 1} == shr[t]
        assert {j for j in range(4) if (int(em[t]) >> j) & 1} == exps[t]
    np.testing.assert_allclose(y, yb, rtol=1e-11, atol=1e-13)


def test_prefix_selection_ignores_priorities(oracle_mod):
    """Prefix block selection (Table IV) shares blocks 0..b-1 even when the
    priorities rank the last blocks highest; the default TopK picks those."""
    d, H, K, B = 4, 8, 2, 8
    x = np.array([[1.0, 0.0, 0.0, 0.0]])
    w_router = np.zeros((d, K + 1))
    w_up = np.zeros((K + 1, H, d))
    w_up[0, :, 0] = np.arange(H, dtype=np.float64)  # M = 1: u_b = b, last blocks first
    w_down = np.zeros((K + 1, d, H))
    th = Thresholds(alpha_fixed=0.375)  # b = 3
    _, r = oracle.layer(x, w_router, w_up, w_down, B, th)
    assert r.b[0] == 3 and int(r.shr_mask[0]) == 0b11100000
    _, rp = oracle.layer(x, w_router, w_up, w_down, B,
                         Thresholds(alpha_fixed=0.375, prefix_blocks=1))
    assert rp.b[0] == 3 and int(rp.shr_mask[0]) == 0b00000111


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_router_bias_brute_force(oracle_mod, seed):
    """A bias per router column enters the logits before Eqs. 18 and 24:
    decisions and output against exhaustive search with the bias added to
    x W* by a dense product."""
    rng = np.random.default_rng(40 + seed)
    K, B = 4, 4
    x, w_router, w_up, w_down = rand_layer(rng, 6, 16, K, B, router_scale=2.0, T=40)
    bias = rng.normal(0.0, 1.5, K + 1)
    y, r = oracle.layer(x, w_router, w_up, w_down, B, bias=bias)
    yb, bb, kb, shr, exps = brute_force(x, w_router, w_up, w_down, B, Thresholds(), bias=bias)
    assert r.b.tolist() == bb.tolist() and r.k.tolist() == kb.tolist()
    em = r.expert_mask()
    for t in range(x.shape[0]):
        assert {j for j in range(K) if (int(em[t]) >> j) & 1} == exps[t]
    np.testing.assert_allclose(y, yb, rtol=1e-11, atol=1e-13)
    # the bias changes decisions here (it is not a no-op on this layer)
    _, r0 = oracle.layer(x, w_router, w_up, w_down, B)
    assert (r0.k != r.k).any() or (r0.b != r.b).any()


@pytest.mark.parametrize("j", [0, 2])
def test_router_bias_closed_form(oracle_mod, j):
    """A large bias on one residual expert's column makes its affinity 1 (to
    rounding), so it alone is selected: k = 1, q_1 = j (Eqs. 24-27). A large
    bias on the shared column drives alpha to its bounds tau and 1 - tau
    (Eq. 18): with B = 4, tau = 3/16, b = round(4 * 13/16) = 3 or
    round(4 * 3/16) = 1."""
    rng = np.random.default_rng(3)
    K, B = 3, 4
    x, w_router, w_up, w_down = rand_layer(rng, 8, 16, K, B, T=30)
    for sign, b_want in ((1.0, 3), (-1.0, 1)):
        bias = np.zeros(K + 1)
        bias[0] = 60.0 * sign
        bias[1 + j] = 60.0
        _, r = oracle.layer(x, w_router, w_up, w_down, B, bias=bias)
        assert (r.k == 1).all() and (r.q[:, 0] == j).all()
        np.testing.assert_allclose(r.p[:, 0], 1.0, rtol=0, atol=1e-15)
        assert (r.b == b_want).all()
        alpha_bound = 13 / 16 if sign > 0 else 3 / 16
        np.testing.assert_allclose(r.alpha, alpha_bound, rtol=0, atol=1e-15)


def test_with_decisions_hand_case(oracle_mod):
    """with_decisions keeps this oracle's scores and takes the given discrete
    decisions: q lists the given residual experts by decreasing affinity
    (ties to the lower index), then the rest; p follows q; k counts the given
    experts; b counts the given shared blocks (hand example)."""
    s = np.array([[0.1, 0.5, 0.4], [0.25, 0.5, 0.25]])
    T, K, B = 2, 3, 4
    r = oracle.Routing(alpha=np.array([0.6, 0.3]), beta=np.array([0.4, 0.7]),
                       b=np.array([2, 1], np.int32), k=np.array([1, 2], np.int32),
                       shr_mask=np.array([0b0011, 0b0001], np.uint64),
                       q=np.zeros((T, K), np.int32), p=np.zeros((T, K)), s=s,
                       u=np.zeros((T, B)), margin=np.zeros((T, 4)))
    f = oracle.with_decisions(r, np.array([0b1010, 0b0111], np.uint64),
                              np.array([0b101, 0b101], np.uint64), B)
    assert f.q.tolist() == [[2, 0, 1], [0, 2, 1]]
    np.testing.assert_array_equal(f.p, [[0.4, 0.1, 0.5], [0.25, 0.25, 0.5]])
    assert f.k.tolist() == [2, 2] and f.b.tolist() == [2, 3]
    assert f.shr_mask.tolist() == [0b1010, 0b0111]
    np.testing.assert_array_equal(f.alpha, r.alpha)


def test_with_decisions_output_matches_brute_force(oracle_mod):
    """The layer output for given decisions (other than the oracle's own)
    equals the masked sum of dense block outputs with those sets (Eq. 30),
    and the oracle's own decisions reproduce its own output."""
    rng = np.random.default_rng(21)
    K, B = 4, 4
    x, w_router, w_up, w_down = rand_layer(rng, 6, 16, K, B, router_scale=3.0, T=30)
    y, r = oracle.layer(x, w_router, w_up, w_down, B)
    same = oracle.with_decisions(r, r.shr_mask, r.expert_mask(), B)
    np.testing.assert_array_equal(oracle.forward(x, w_up, w_down, same, B), y)
    shr = rng.integers(0, 2**B, 30).astype(np.uint64)
    em = rng.integers(1, 2**K, 30).astype(np.uint64)
    f = oracle.with_decisions(r, shr, em, B)
    yf = oracle.forward(x, w_up, w_down, f, B)
    blocks = block_outputs_dense(x, w_up, w_down, B)
    for t in range(30):
        want = np.zeros(x.shape[1])
        for blk in range(B):
            if (int(shr[t]) >> blk) & 1:
                want += r.alpha[t] * blocks[t, 0, blk]
            else:
                for j in range(K):
                    if (int(em[t]) >> j) & 1:
                        want += r.s[t, j] * blocks[t, 1 + j, blk]
        np.testing.assert_allclose(yf[t], want, rtol=1e-12, atol=1e-13)


# --------------------------------------------------------------------------
# Special cases that reduce to textbook layers
# --------------------------------------------------------------------------

@pytest.mark.parametrize("B", [2, 4, 8])
def test_alpha_one_is_dense_ffn(oracle_mod, B):
    """alpha fixed at 1: b = B, every block shared, I_res empty (Eqs. 19,
    22-23), so y = E_shr(x), the plain FFN of Eq. 4."""
    rng = np.random.default_rng(B)
    x, w_router, w_up, w_down = rand_layer(rng, 16, 64, 4, B)
    y, r = oracle.layer(x, w_router, w_up, w_down, B, Thresholds(alpha_fixed=1.0))
    assert (r.b == B).all()
    dense = gelu_ref(x @ w_up[0].T) @ w_down[0].T
    np.testing.assert_allclose(y, dense, rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("th", [Thresholds(alpha_fixed=0.0, beta_fixed=1.0),
                                Thresholds(alpha_fixed=0.0, topk_fixed=5)])
def test_alpha_zero_all_experts_is_soft_moe(oracle_mod, th):
    """alpha = 0 and all K experts selected: y = sum_j s_j E_j(x), the
    conventional MoE output of Eq. 5 with k = K (softmax gate of Eq. 2)."""
    rng = np.random.default_rng(3)
    K, B = 5, 4
    x, w_router, w_up, w_down = rand_layer(rng, 12, 32, K, B, router_scale=4.0)
    y, r = oracle.layer(x, w_router, w_up, w_down, B, th)
    assert (r.b == 0).all() and (r.k == K).all()
    s = softmax(x @ w_router[:, 1:], axis=1)
    want = sum(s[:, [j]] * (gelu_ref(x @ w_up[1 + j].T) @ w_down[1 + j].T) for j in range(K))
    np.testing.assert_allclose(y, want, rtol=1e-12, atol=1e-13)


def test_two_blocks_share_exactly_one(oracle_mod):
    """B = 2 gives tau = 1/4, alpha in (1/4, 3/4), so b = 1 always (Eqs. 18-19)."""
    rng = np.random.default_rng(11)
    x, w_router, w_up, w_down = rand_layer(rng, 8, 16, 3, 2, router_scale=6.0, T=400)
    _, r = oracle.layer(x, w_router, w_up, w_down, 2)
    assert (r.alpha > 0.25).all() and (r.alpha < 0.75).all()
    assert r.alpha.min() < 0.27 and r.alpha.max() > 0.73  # the range is exercised
    assert (r.b == 1).all()


def test_top1_covers_one_full_ffn(oracle_mod):
    """k = 1: shared plus residual blocks are exactly one FFN's B blocks,
    C_B = B (Eq. 35 and the remark after it)."""
    rng = np.random.default_rng(5)
    x, w_router, w_up, w_down = rand_layer(rng, 8, 32, 4, 8)
    _, r = oracle.layer(x, w_router, w_up, w_down, 8, Thresholds(topk_fixed=1))
    assert (r.k == 1).all() and (r.cb(8) == 8).all()


# --------------------------------------------------------------------------
# Invariants stated in the paper, on realistic random layers
# --------------------------------------------------------------------------

@pytest.mark.parametrize("B,K", [(4, 4), (8, 8), (16, 16), (16, 32)])
def test_invariants(oracle_mod, B, K):
    rng = np.random.default_rng(B * 100 + K)
    d = 32
    x, w_router, w_up, w_down = rand_layer(rng, d, 16 * B, K, B, router_scale=8.0, T=500)
    y, r = oracle.layer(x, w_router, w_up, w_down, B)
    T = x.shape[0]
    # Eq. 19 remark: b in {1..B-1}
    assert r.b.min() >= 1 and r.b.max() <= B - 1
    pc = np.array([bin(int(v)).count("1") for v in r.shr_mask])
    assert (pc == r.b).all()  # |I_shr| = b (Eq. 22)
    for t in range(T):
        inside = [r.u[t, blk] for blk in range(B) if (int(r.shr_mask[t]) >> blk) & 1]
        outside = [r.u[t, blk] for blk in range(B) if not (int(r.shr_mask[t]) >> blk) & 1]
        assert min(inside) >= max(outside)  # TopK of priorities (Eq. 22)
        # p sorted, a permutation of s (Eq. 25)
        assert (np.diff(r.p[t]) <= 0).all()
        np.testing.assert_allclose(np.sort(r.s[t]), np.sort(r.p[t]), rtol=0, atol=0)
        kk = r.k[t]
        Pk = r.p[t, :kk].sum()
        Pk1 = r.p[t, :kk - 1].sum()
        # Eq. 31-32: beta <= P_k < beta + p_k, and 1 <= alpha + P_k < 1 + p_k
        assert r.beta[t] <= Pk + 1e-15 and Pk < r.beta[t] + r.p[t, kk - 1] + 1e-15
        assert 1 - 1e-15 <= r.alpha[t] + Pk < 1 + r.p[t, kk - 1] + 1e-15
        assert Pk1 < r.beta[t]  # minimality (Eq. 27)
    np.testing.assert_allclose(r.alpha + r.beta, 1.0, atol=1e-15)  # Eq. 26
    # The spread of decisions is exercised
    assert len(set(r.b.tolist())) > 1 and len(set(r.k.tolist())) > 1


def test_priorities_are_block_mean_preactivations(oracle_mod):
    """u_b = x mu_b equals the mean over block b of the shared expert's
    pre-activations x K_shr[:, h] (Eqs. 20-21)."""
    rng = np.random.default_rng(9)
    B, K, d, H = 8, 4, 24, 96
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, T=50)
    mu = oracle.prototypes(w_up, B, oracle.ROUND_NONE)
    r = oracle.route(x, w_router, mu, K, B)
    pre = x @ w_up[0].T
    want = pre.reshape(50, B, H // B).mean(axis=2)
    np.testing.assert_allclose(r.u, want, rtol=1e-12, atol=1e-14)


def test_block_decomposition_sums_to_expert(oracle_mod):
    """E_j = sum_b E_j^(b) (Eq. 16): with every block shared and alpha = 1 the
    oracle's blockwise sum equals the full FFN for every B dividing H."""
    rng = np.random.default_rng(2)
    x, w_router, w_up, w_down = rand_layer(rng, 8, 48, 2, 2, T=16)
    outs = [oracle.layer(x, w_router, w_up, w_down, B, Thresholds(alpha_fixed=1.0))[0]
            for B in (2, 3, 4, 6, 8, 12)]
    for o in outs[1:]:
        np.testing.assert_allclose(o, outs[0], rtol=1e-12, atol=1e-14)


def test_permuting_tokens_permutes_outputs(oracle_mod):
    rng = np.random.default_rng(4)
    x, w_router, w_up, w_down = rand_layer(rng, 16, 64, 4, 4, router_scale=4.0, T=80)
    y, r = oracle.layer(x, w_router, w_up, w_down, 4)
    perm = rng.permutation(80)
    y2, r2 = oracle.layer(x[perm], w_router, w_up, w_down, 4)
    assert np.array_equal(y2, y[perm])
    assert np.array_equal(r2.shr_mask, r.shr_mask[perm]) and np.array_equal(r2.k, r.k[perm])


def test_padding_tokens(oracle_mod):
    rng = np.random.default_rng(6)
    x, w_router, w_up, w_down = rand_layer(rng, 8, 32, 4, 4, T=20)
    mask = (np.arange(20) % 3 != 0).astype(np.uint8)
    x[mask == 0] = np.nan
    y, r = oracle.layer(x, w_router, w_up, w_down, 4, mask=mask)
    assert np.isfinite(y).all()
    assert (y[mask == 0] == 0).all() and (r.b[mask == 0] == 0).all() and (r.k[mask == 0] == 0).all()
    counts, tok, _ = oracle.groups(r, 4, 4, mask)
    assert not set(tok.tolist()) & set(np.nonzero(mask == 0)[0].tolist())
    assert counts.sum() == r.cb(4)[mask == 1].sum()


def test_group_table_matches_decisions(oracle_mod):
    """Each token appears in exactly C_B(t) groups (Eq. 35): the b shared
    blocks of expert 0 and the B-b residual blocks of each of its k experts."""
    rng = np.random.default_rng(8)
    B, K = 8, 6
    x, w_router, w_up, w_down = rand_layer(rng, 16, 64, K, B, router_scale=6.0, T=200)
    _, r = oracle.layer(x, w_router, w_up, w_down, B)
    counts, tok, w = oracle.groups(r, K, B)
    assert np.bincount(tok, minlength=200).tolist() == r.cb(B).tolist()
    start = np.concatenate([[0], np.cumsum(counts)])
    em = r.expert_mask()
    for g in range(len(counts)):
        e, blk = divmod(g, B)
        rows = tok[start[g]:start[g + 1]]
        assert (np.diff(rows) > 0).all()  # increasing token order
        for t, wt in zip(rows, w[start[g]:start[g + 1]]):
            shared = (int(r.shr_mask[t]) >> blk) & 1
            if e == 0:
                assert shared and wt == r.alpha[t]
            else:
                assert not shared and (int(em[t]) >> (e - 1)) & 1
                assert wt == r.s[t, e - 1]


# --------------------------------------------------------------------------
# Readings: ties, rounding of Eq. 19 and of the stored prototypes
# --------------------------------------------------------------------------

def test_ties_break_to_lower_index(oracle_mod):
    d, K, B = 4, 4, 4
    x = np.array([[1.0, 0.0, 0.0, 0.0]])
    w_router = np.zeros((d, K + 1))
    w_router[0, 2] = w_router[0, 3] = 1.0  # experts 1 and 2 tie on top
    w_up = np.zeros((K + 1, 16, d))
    w_up[0, :, 0] = 1.0  # all block priorities equal
    w_down = np.zeros((K + 1, d, 16))
    _, r = oracle.layer(x, w_router, w_up, w_down, B, Thresholds(alpha_fixed=0.5))
    assert r.q[0, :2].tolist() == [1, 2] and r.q[0, 2:].tolist() == [0, 3]
    assert int(r.shr_mask[0]) == 0b0011  # b = 2 of 4 equal priorities: blocks 0, 1


@pytest.mark.parametrize("alpha,b", [(0.3125, 2), (0.4375, 4), (0.5625, 4), (0.6875, 6)])
def test_round_half_to_even(oracle_mod, alpha, b):
    """B alpha exactly halfway between integers (B = 8): round half to even."""
    rng = np.random.default_rng(0)
    x, w_router, w_up, w_down = rand_layer(rng, 4, 16, 2, 8, T=1)
    _, r = oracle.layer(x, w_router, w_up, w_down, 8, Thresholds(alpha_fixed=alpha))
    assert r.b[0] == b


def test_prototype_rounding(oracle_mod):
    """With M = 1 the prototype is the key itself, so the rounding to the
    router's storage precision is seen directly: bf16 keeps 8 significant
    bits, ties go to the even neighbour; fp32 is the IEEE single rounding."""
    vals = np.array([1 + 2**-8, 1 + 3 * 2**-8, 1 + 2**-8 + 2**-30, -(1 + 2**-8),
                     3.0, 0.1, 2**-130 * 1.5])
    want_bf16 = np.array([1.0, 1 + 2**-6, 1 + 2**-7, -1.0, 3.0, 0.10009765625,
                          2**-130 * 1.5])
    w = np.zeros((len(vals), 1))
    w[:, 0] = vals
    mu = oracle.prototypes(w, len(vals), oracle.ROUND_BF16)[:, 0]
    np.testing.assert_array_equal(mu, want_bf16)
    mu32 = oracle.prototypes(w, len(vals), oracle.ROUND_F32)[:, 0]
    np.testing.assert_array_equal(mu32, vals.astype(np.float32).astype(np.float64))
    # The mean over a block is exact before the single rounding.
    w2 = np.array([[1.0], [2**-9], [0.0], [0.0]])  # mean of first block = (1 + 2^-9)/2
    mu2 = oracle.prototypes(w2, 2, oracle.ROUND_BF16)[:, 0]
    assert mu2[0] == 0.5  # (1+2^-9)/2 = 0.5 + 2^-10, below the halfway point 0.5 + 2^-9


def test_margins_hand_case(oracle_mod):
    """All four margins on two hand-built tokens. M = 1, so the priority of
    block b is key b of the shared expert; x is a unit vector, so the logits
    are one row of W*: residual logits ln(0.5, 0.3, 0.2) and ln(0.65, 0.25,
    0.1) give those affinities exactly (to rounding). alpha fixed at 0.5
    (B = 4: b = 2, margin (i) not applicable), beta fixed at 0.6.
      token 0: u = (0.9, 0.5, 0.45, 0.1): (ii) = 0.5 - 0.45 = 0.05;
               P = 0.5, 0.8: k = 2, (iii) = min(0.8 - 0.6, 0.6 - 0.5) = 0.1;
               (iv) = p_2 - p_3 = 0.1
      token 1: u = (0.2, 0.8, 0.1, 0.3): (ii) = 0.3 - 0.2 = 0.1;
               P_1 = 0.65: k = 1, (iii) = min(0.65 - 0.6, 0.6 - 0) = 0.05;
               (iv) = 0.65 - 0.25 = 0.4"""
    d, H, K, B = 4, 4, 3, 4
    x = np.eye(d)[:2]
    w_router = np.zeros((d, K + 1))
    w_router[0, 1:] = np.log([0.5, 0.3, 0.2])
    w_router[1, 1:] = np.log([0.65, 0.25, 0.1])
    w_up = np.zeros((K + 1, H, d))
    w_up[0, :, 0] = [0.9, 0.5, 0.45, 0.1]
    w_up[0, :, 1] = [0.2, 0.8, 0.1, 0.3]
    w_down = np.zeros((K + 1, d, H))
    _, r = oracle.layer(x, w_router, w_up, w_down, B, Thresholds(alpha_fixed=0.5, beta_fixed=0.6))
    assert r.b.tolist() == [2, 2] and r.k.tolist() == [2, 1]
    assert np.isinf(r.margin[:, 0]).all()
    np.testing.assert_allclose(r.margin[:, 1], [0.05, 0.1], rtol=0, atol=1e-15)
    np.testing.assert_allclose(r.margin[:, 2], [0.1, 0.05], rtol=0, atol=1e-15)
    np.testing.assert_allclose(r.margin[:, 3], [0.1, 0.4], rtol=0, atol=1e-15)
    # a fixed top-k has no cutoff margin; prefix selection no priority margin
    _, r2 = oracle.layer(x, w_router, w_up, w_down, B,
                         Thresholds(alpha_fixed=0.5, topk_fixed=2, prefix_blocks=1))
    assert np.isinf(r2.margin[:, 1]).all() and np.isinf(r2.margin[:, 2]).all()


def test_margins_flag_near_ties(oracle_mod):
    """Margin (iv) is p_k - p_{k+1}; margin (i) is the distance of B alpha to
    the nearest half-integer, divided by B."""
    rng = np.random.default_rng(12)
    x, w_router, w_up, w_down = rand_layer(rng, 16, 64, 8, 8, router_scale=2.0, T=300)
    _, r = oracle.layer(x, w_router, w_up, w_down, 8)
    for t in range(300):
        kk = r.k[t]
        if kk < 8:
            assert r.margin[t, 3] == pytest.approx(r.p[t, kk - 1] - r.p[t, kk], abs=1e-15)
        frac = 8 * r.alpha[t] - math.floor(8 * r.alpha[t])
        assert r.margin[t, 0] == pytest.approx(abs(frac - 0.5) / 8, abs=1e-15)
        assert (r.margin[t] >= 0).all()


# --------------------------------------------------------------------------
# The layer as a Transformer sublayer (Appendix A, Architecture details) and upcycled experts
# (Sec. III)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("eps", [0.0, 1e-5, 0.3])
def test_layernorm_moments(oracle_mod, eps):
    """With gamma = 1, beta = 0 every normalised row has mean 0 and variance
    var / (var + eps), var the row's biased variance (closed form)."""
    rng = np.random.default_rng(11)
    d = 48
    v = rng.standard_normal((40, d)) * rng.uniform(0.2, 3.0, (40, 1)) + rng.normal(0, 2, (40, 1))
    out = oracle_mod.layernorm(v, np.ones(d), np.zeros(d), eps)
    var = v.var(axis=1)  # numpy's default is the biased (1/d) variance
    np.testing.assert_allclose(out.mean(axis=1), 0.0, atol=1e-12)
    np.testing.assert_allclose(out.var(axis=1), var / (var + eps), rtol=1e-12)


def test_layernorm_affine_constant_padding_rounding(oracle_mod):
    """gamma and beta act after the normalisation; a constant row normalises
    to beta; padding rows give 0; round_mode rounds to bf16 values."""
    rng = np.random.default_rng(12)
    d = 32
    v = rng.standard_normal((6, d))
    v[3] = 2.5  # constant row
    g = rng.uniform(0.5, 2.0, d)
    b = rng.standard_normal(d)
    unit = oracle_mod.layernorm(v, np.ones(d), np.zeros(d), 1e-5)
    out = oracle_mod.layernorm(v, g, b, 1e-5)
    np.testing.assert_allclose(out, unit * g + b, rtol=1e-13, atol=1e-13)
    np.testing.assert_array_equal(out[3], b)
    mask = np.array([1, 1, 0, 1, 1, 1], np.uint8)
    np.testing.assert_array_equal(oracle_mod.layernorm(v, g, b, 1e-5, mask)[2], 0.0)
    r = oracle_mod.layernorm(v, g, b, 1e-5, round_mode=oracle_mod.ROUND_BF16)
    import torch
    as_bf16 = torch.tensor(out).to(torch.bfloat16).double().numpy()  # library rounding
    np.testing.assert_array_equal(r, as_bf16)


@pytest.mark.parametrize("norm_first", [True, False])
def test_sublayer_with_silent_experts(oracle_mod, norm_first):
    """Experts with zero up-projections output nothing (GeLU(0) = 0), so the
    sublayer reduces to the residual path: x itself when normalised first,
    LN(x) when normalised after the sum. Padding rows give 0."""
    rng = np.random.default_rng(13)
    d, H, K, B = 16, 32, 3, 4
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, T=20)
    w_up[:] = 0.0
    g = rng.uniform(0.5, 2.0, d)
    b = rng.standard_normal(d)
    mask = np.ones(20, np.uint8)
    mask[[4, 9]] = 0
    out, _ = oracle_mod.sublayer(x, w_router, w_up, w_down, B, g, b, 1e-5, norm_first, mask=mask)
    ref = x if norm_first else oracle_mod.layernorm(x, g, b, 1e-5)
    keep = mask == 1
    np.testing.assert_allclose(out[keep], ref[keep], rtol=1e-13, atol=1e-13)
    np.testing.assert_array_equal(out[~keep], 0.0)


def test_sublayer_order_of_norm_and_residual(oracle_mod):
    """Normalised first, the residual adds the raw input to the layer's output
    on the normalised input; normalised after, the norm sees the sum. Both
    against the layer oracle composed by hand."""
    rng = np.random.default_rng(14)
    d, H, K, B = 16, 32, 3, 4
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, T=24)
    g = rng.uniform(0.5, 2.0, d)
    b = rng.standard_normal(d)
    pre, _ = oracle_mod.sublayer(x, w_router, w_up, w_down, B, g, b, 1e-5, True)
    xn = oracle_mod.layernorm(x, g, b, 1e-5)
    np.testing.assert_allclose(pre, x + oracle_mod.layer(xn, w_router, w_up, w_down, B)[0],
                               rtol=1e-13, atol=1e-13)
    post, _ = oracle_mod.sublayer(x, w_router, w_up, w_down, B, g, b, 1e-5, False)
    y = oracle_mod.layer(x, w_router, w_up, w_down, B)[0]
    np.testing.assert_allclose(post, oracle_mod.layernorm(x + y, g, b, 1e-5), rtol=1e-13,
                               atol=1e-13)


def test_upcycled_experts_closed_form(oracle_mod):
    """Sec. III: experts upcycled from one dense FFN are identical, so the
    layer output is alpha times the dense FFN's shared blocks plus P_k (the
    selected residual mass) times its complementary blocks, whatever experts
    were selected (block outputs by dense matrix products, GeLU from the
    normal CDF)."""
    rng = np.random.default_rng(15)
    d, H, K, B = 24, 48, 4, 4
    x, w_router, _, _ = rand_layer(rng, d, H, K, B, T=40)
    w1 = rng.standard_normal((H, d)) / math.sqrt(d)
    w2 = rng.standard_normal((d, H)) / math.sqrt(H)
    wu, wd = oracle_mod.upcycle(w1, w2, K)
    assert wu.shape == (K + 1, H, d) and wd.shape == (K + 1, d, H)
    y, r = oracle_mod.layer(x, w_router, wu, wd, B)
    Eb = block_outputs_dense(x, w1[None], w2[None], B)[:, 0]  # [T][B][d]
    for t in range(x.shape[0]):
        shr = [(int(r.shr_mask[t]) >> blk) & 1 for blk in range(B)]
        Pk = float(np.sum(r.p[t, :r.k[t]]))
        ref = sum(r.alpha[t] * Eb[t, blk] if shr[blk] else Pk * Eb[t, blk] for blk in range(B))
        np.testing.assert_allclose(y[t], ref, rtol=1e-12, atol=1e-12)


# --------------------------------------------------------------------------
# Training (Sec. III-E): gradients through Eq. 30 and the Gram regulariser
# --------------------------------------------------------------------------

def fixed_decision_loss(x, w_router, w_up, w_down, bias, B, th, shr, em, dy, mask=None):
    """<dy, y> with y the oracle's forward for the given discrete decisions
    (shared block sets, selected experts) and alpha, s recomputed from the
    perturbed parameters: a smooth function of every parameter."""
    K = w_up.shape[0] - 1
    mu = oracle.prototypes(w_up, B, oracle.ROUND_NONE)
    r = oracle.route(x, w_router, mu, K, B, th, mask, bias)
    y = oracle.forward(x, w_up, w_down, oracle.with_decisions(r, shr, em, B), B, mask)
    return float(np.sum(dy * y))


def central_differences(f, arrays, eps=1e-6):
    """dL/da for every entry of every array by (f(a + eps) - f(a - eps)) / 2 eps."""
    out = []
    for a in arrays:
        g = np.zeros_like(a)
        flat, gf = a.reshape(-1), g.reshape(-1)
        for i in range(flat.size):
            keep = flat[i]
            flat[i] = keep + eps
            fp = f()
            flat[i] = keep - eps
            fm = f()
            flat[i] = keep
            gf[i] = (fp - fm) / (2 * eps)
        out.append(g)
    return out


@pytest.mark.parametrize("th,masked", [(Thresholds(), False), (Thresholds(), True),
                                       (Thresholds(alpha_fixed=0.4, topk_fixed=2), False),
                                       (Thresholds(beta_fixed=0.8, prefix_blocks=1), True)])
def test_backward_matches_finite_differences(oracle_mod, th, masked):
    """Every gradient of the oracle's backward (x, keys, values, router
    columns, router bias) against central differences of the pinned forward,
    the discrete decisions held at the unperturbed ones."""
    rng = np.random.default_rng(31)
    T, d, H, K, B = 7, 4, 8, 3, 4
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, router_scale=3.0, T=T)
    bias = rng.normal(0.0, 0.5, K + 1)
    dy = rng.standard_normal((T, d))
    mask = np.array([1, 0, 1, 1, 0, 1, 1], np.uint8) if masked else None
    _, r = oracle.layer(x, w_router, w_up, w_down, B, th, mask=mask, bias=bias)
    shr, em = r.shr_mask.copy(), r.expert_mask()
    g = oracle.backward(x, w_router, w_up, w_down, shr, em, B, dy, th, mask, bias)
    f = lambda: fixed_decision_loss(x, w_router, w_up, w_down, bias, B, th, shr, em, dy, mask)
    num = central_differences(f, [x, w_up, w_down, w_router, bias])
    for got, want in zip([g.dx, g.dw_up, g.dw_down, g.dw_router, g.dbias], num):
        np.testing.assert_allclose(got, want, rtol=1e-6, atol=1e-8)
    if masked:
        assert (g.dx[mask == 0] == 0).all()
    if not math.isnan(th.alpha_fixed):
        assert (g.dw_router[:, 0] == 0).all()  # alpha fixed: no gradient to W_shr


def test_backward_dense_ffn_closed_form(oracle_mod):
    """alpha fixed at 1: y = GeLU(x K_shr) V_shr (every block shared), so
    dV = dy^T GeLU(A), dA = (dy V) * GeLU'(A) with GeLU'(a) = Phi(a) + a phi(a)
    (normal CDF and density from the library), dK = dA^T x, dx = dA K; the
    router gets nothing (alpha fixed; the residual expert runs no block)."""
    rng = np.random.default_rng(32)
    T, d, H, K, B = 30, 12, 32, 3, 4
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, T=T)
    dy = rng.standard_normal((T, d))
    th = Thresholds(alpha_fixed=1.0)
    _, r = oracle.layer(x, w_router, w_up, w_down, B, th)
    g = oracle.backward(x, w_router, w_up, w_down, r.shr_mask, r.expert_mask(), B, dy, th)
    A = x @ w_up[0].T
    gA = (dy @ w_down[0]) * (norm.cdf(A) + A * norm.pdf(A))
    np.testing.assert_allclose(g.dw_down[0], dy.T @ gelu_ref(A), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(g.dw_up[0], gA.T @ x, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(g.dx, gA @ w_up[0], rtol=1e-12, atol=1e-12)
    assert (g.dw_up[1:] == 0).all() and (g.dw_down[1:] == 0).all()
    assert (g.dw_router == 0).all() and (g.dbias == 0).all()


@pytest.mark.parametrize("c", [0.5, 1.0, 1.7])
def test_diversity_closed_form(oracle_mod, c):
    """W* = c Q with Q's K+1 columns orthonormal: W*^T W* - I = (c^2 - 1) I, so
    L_div = |c^2 - 1| sqrt(K+1) and dL_div/dW* = 2 c sign(c^2 - 1) Q / sqrt(K+1)
    (Eq. diversity-loss); orthonormal columns (c = 1) give 0."""
    rng = np.random.default_rng(33)
    d, K1 = 16, 5
    Q, _ = np.linalg.qr(rng.standard_normal((d, K1)))
    L, grad = oracle.diversity(c * Q)
    np.testing.assert_allclose(L, abs(c * c - 1) * math.sqrt(K1), rtol=1e-12, atol=1e-13)
    if c == 1.0:
        return  # the norm has no gradient at 0 (L is rounding noise here)
    want = 2 * c * np.sign(c * c - 1) * Q / math.sqrt(K1)
    np.testing.assert_allclose(grad, want, rtol=1e-11, atol=1e-12)


def test_diversity_finite_differences(oracle_mod):
    rng = np.random.default_rng(34)
    W = rng.standard_normal((6, 4)) * 0.7
    L, grad = oracle.diversity(W)
    G = np.linalg.norm(W.T @ W - np.eye(4))  # Frobenius norm, library routine
    assert L == pytest.approx(G, rel=1e-13)
    num, = central_differences(lambda: oracle.diversity(W)[0], [W])
    np.testing.assert_allclose(grad, num, rtol=1e-7, atol=1e-9)


# --------------------------------------------------------------------------
# Diagnostics of Sec. II-B: value alignment and functional demand
# --------------------------------------------------------------------------

def test_value_alignment_closed_forms(oracle_mod):
    """Eq. shared-set on constructed value rows (d = 2): identical rows have
    c = 1, opposite rows c = -1, rows (3, 4) and (4, 3) have c = 24/25
    exactly (an exact cosine counts at delta = 0.96, the set uses >=), and a
    zero row is aligned with nothing."""
    from oracle import diagnostics as dg
    d, H, K = 2, 8, 3
    wd = np.zeros((K + 1, d, H))
    v1 = np.array([[3.0, 4.0], [1.0, 0.0], [0.0, 2.0], [5.0, 1.0],
                   [1.0, 1.0], [2.0, -1.0], [0.0, 0.0], [1.0, 3.0]])  # [H][d]
    v2 = v1.copy()
    v2[0] = [4.0, 3.0]          # c = 24/25
    v2[1] = [-1.0, 0.0]         # c = -1
    v2[2] = [0.0, 7.0]          # c = 1 (positive scale)
    v2[3] = [-1.0, 5.0]         # orthogonal: c = 0
    v3 = -v1                    # every row opposite
    for e, v in ((1, v1), (2, v2), (3, v3)):
        wd[e] = v.T
    rho, S = dg.value_alignment(wd, 0.96)
    # expert 1 vs 2: rows 0 (24/25), 2, 4, 5, 7 aligned; 1 (opposite), 3 (orthogonal), 6 (zero) not
    assert S[0, 1].tolist() == [True, False, True, False, True, True, False, True]
    assert rho[0, 1] == pytest.approx(5 / 8) and rho[1, 0] == pytest.approx(5 / 8)
    assert rho[0, 2] == 0.0
    assert rho[0, 0] == pytest.approx(7 / 8)  # every nonzero row with itself
    _, S2 = dg.value_alignment(wd, 0.96 + 1e-12)
    assert not S2[0, 1, 0] and S2[0, 1, 2]


def test_expert_outputs_match_layer_oracle(oracle_mod):
    """E_e(x) of the diagnostic equals the layer oracle's dense FFN of that
    expert (alpha fixed at 1 with expert e as the shared one); E^S with every
    channel is E, with none is 0."""
    from oracle import diagnostics as dg
    rng = np.random.default_rng(41)
    T, d, H, K, B = 20, 8, 16, 3, 4
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, T=T)
    E, ES = dg.expert_outputs(x, w_up, w_down, np.ones((T, H), bool))
    _, ES0 = dg.expert_outputs(x, w_up, w_down, np.zeros((T, H), bool))
    np.testing.assert_array_equal(ES, E)
    assert (ES0 == 0).all()
    for e in range(1, K + 1):
        wu = w_up.copy()
        wd = w_down.copy()
        wu[0], wd[0] = w_up[e], w_down[e]
        y, _ = oracle.layer(x, w_router, wu, wd, B, Thresholds(alpha_fixed=1.0))
        np.testing.assert_allclose(E[:, e - 1], y, rtol=1e-12, atol=1e-13)


def test_functional_demand_identical_experts(oracle_mod):
    """Experts copied from one FFN align at every channel (rho = 1), so the
    shared response is the whole output, r = 0 and k_eps = 1 for every token."""
    from oracle import diagnostics as dg
    rng = np.random.default_rng(42)
    T, d, H, K, B = 16, 8, 16, 4, 4
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, router_scale=3.0, T=T)
    w_up[:] = w_up[0]
    w_down[:] = w_down[0]
    rho, _ = dg.value_alignment(w_down, 0.98)
    assert (rho == 1).all()
    k, err, _ = dg.functional_demand(x, w_router, w_up, w_down, rng.standard_normal((d, K)),
                                     0.98, 0.05)
    assert (k == 1).all() and np.abs(err).max() < 1e-12


def test_functional_demand_nothing_shared(oracle_mod):
    """delta above 1 shares nothing: r = y_orig. With the residual order of
    the original router the first two residual rows are E_i and E_j, which
    span r: e_2 is the ridge's own (1e-6-relative) residual; e_1 is the
    distance of r from the line of E_i, from the normal equations by hand."""
    from oracle import diagnostics as dg
    rng = np.random.default_rng(43)
    T, d, H, K, B = 12, 10, 16, 4, 4
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, router_scale=3.0, T=T)
    k, err, pair = dg.functional_demand(x, w_router, w_up, w_down, w_router[:, 1:], 2.0, 1e-3)
    E, _ = dg.expert_outputs(x, w_up, w_down, np.zeros((T, H), bool))
    i, j, ti, tj = dg.top2_pairs(x, w_router)
    assert (pair[:, 0] == i).all() and (pair[:, 1] == j).all()
    for t in range(T):
        r = ti[t] * E[t, i[t]] + tj[t] * E[t, j[t]]
        Ei = E[t, i[t]]
        g = Ei @ Ei
        a = (Ei @ r) / (g * (1 + 1e-6))
        assert err[t, 0] == pytest.approx(np.linalg.norm(r - a * Ei) / np.linalg.norm(r),
                                          rel=1e-9, abs=1e-12)
        assert err[t, 1] < 1e-5
    assert (k <= 2).all()
    k0, _, _ = dg.functional_demand(x, w_router, w_up, w_down, w_router[:, 1:], 2.0, -1.0)
    assert (k0 == K + 1).all()  # no prefix reaches a negative tolerance: the sentinel


def test_functional_demand_ridge_by_augmented_least_squares(oracle_mod):
    """Every e_m against the ridge solved another way: least squares on the
    stacked system [R^T; sqrt(gamma) I] a = [r; 0] (scipy.linalg.lstsq)."""
    import scipy.linalg
    from oracle import diagnostics as dg
    rng = np.random.default_rng(44)
    T, d, H, K, B, delta = 10, 12, 32, 5, 4, 0.8
    x, w_router, w_up, w_down = rand_layer(rng, d, H, K, B, router_scale=3.0, T=T)
    w_down[2:] = w_down[1] + 0.8 * rng.standard_normal(w_down[2:].shape) / math.sqrt(H)
    w_res = rng.standard_normal((d, K))
    k, err, pair = dg.functional_demand(x, w_router, w_up, w_down, w_res, delta, 0.1)
    _, S = dg.value_alignment(w_down, delta)
    i, j, ti, tj = dg.top2_pairs(x, w_router)
    E, ES = dg.expert_outputs(x, w_up, w_down, S[i, j])
    q = np.argsort(-(x @ w_res), axis=1, kind="stable")
    assert 0 < S[i, j].sum() < T * H  # some channels shared, some not
    for t in range(T):
        y = ti[t] * E[t, i[t]] + tj[t] * E[t, j[t]]
        sb = ti[t] * ES[t, i[t]] + tj[t] * ES[t, j[t]]
        for m in range(1, K + 1):
            R = (E - ES)[t, q[t, :m]]
            gam = 1e-6 * np.sum(R * R) / m
            A = np.vstack([R.T, math.sqrt(gam) * np.eye(m)])
            a = scipy.linalg.lstsq(A, np.concatenate([y - sb, np.zeros(m)]))[0]
            want = np.linalg.norm(sb + a @ R - y) / np.linalg.norm(y)
            assert err[t, m - 1] == pytest.approx(want, rel=1e-7, abs=1e-12)
        hit = np.nonzero(err[t] <= 0.1)[0]
        assert k[t] == (hit[0] + 1 if len(hit) else K + 1)
