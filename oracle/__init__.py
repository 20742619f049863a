"""CPU oracle for the UniF-MoE layer forward pass (fp64, plain C).

TEST INFRASTRUCTURE ONLY: the tests, the smoke check and the benchmark's CPU
baseline leg are the only callers. The CUDA library never loads, links or
calls anything here, and nothing here imports the CUDA package.

The arithmetic lives in `unif_moe_oracle.c`, which follows Sec. III of the
paper equation by equation (Eqs. 16-30); this module only compiles it, moves
arrays in and out with ctypes, and chains the steps:
    prototypes (Eq. 20) -> route (Eqs. 17-27) -> forward (Eqs. 16, 28-30).
`groups` lists the (expert, block) pairs the output sums over, grouped by
pair (the bookkeeping behind Eq. 35). `backward` and `diversity` are the
training side (Sec. III-E): gradients through Eq. 30 with the discrete
decisions held fixed, and the Gram regulariser of the router embeddings.
`upcycle` and `sublayer` place the layer the way the paper's backbones use
it (Sec. III: experts initialised from one dense FFN; Appendix A,
Architecture details: converted FFN layers of DeiT-S, normalised first, and
of BERT, normalised after the residual sum).
"""
from __future__ import annotations

import ctypes as C
import math
import os
import subprocess
import threading
from dataclasses import dataclass
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "unif_moe_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

ROUND_NONE, ROUND_F32, ROUND_BF16 = 0, 1, 2


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (IEEE fp64, no contraction into FMA, so
    results do not depend on the host CPU)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp%d" % os.getpid()
        cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-shared",
               "-fPIC", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            # A test may point the wrapper at a deliberately broken build of
            # the same source (mutation check of the pins).
            path = os.environ.get("UNIF_MOE_ORACLE_LIB") or build()
            lib = C.CDLL(path)
            P = C.c_void_p
            lib.oracle_max_threads.restype = C.c_int
            lib.oracle_prototypes.argtypes = [P, C.c_int, C.c_int, C.c_int, C.c_int, P]
            lib.oracle_route.argtypes = [C.c_int] * 4 + [P] * 16
            lib.oracle_forward.argtypes = [C.c_int] * 5 + [P] * 10
            lib.oracle_groups.argtypes = [C.c_int] * 3 + [P] * 9 + [C.c_longlong]
            lib.oracle_groups.restype = C.c_longlong
            lib.oracle_layernorm.argtypes = [C.c_int, C.c_int, P, P, P, P, C.c_double, C.c_int, P]
            lib.oracle_backward.argtypes = [C.c_int] * 5 + [P] * 15
            lib.oracle_diversity.argtypes = [C.c_int, C.c_int, P, P]
            lib.oracle_diversity.restype = C.c_double
            _lib = lib
    return _lib


def threads() -> int:
    return _load().oracle_max_threads()


def _f64(a) -> np.ndarray:
    if hasattr(a, "detach"):  # torch tensor
        import torch
        a = a.detach().to("cpu", torch.float64).numpy()
    return np.ascontiguousarray(a, dtype=np.float64)


def _u8(a) -> Optional[np.ndarray]:
    if a is None:
        return None
    if hasattr(a, "detach"):
        a = a.detach().cpu().numpy()
    return np.ascontiguousarray(a, dtype=np.uint8)


def _p(a) -> Optional[int]:
    return None if a is None else a.ctypes.data


@dataclass
class Thresholds:
    tau: float = math.nan
    alpha_fixed: float = math.nan
    beta_fixed: float = math.nan
    topk_fixed: int = 0
    prefix_blocks: int = 0

    def array(self) -> np.ndarray:
        return np.array([self.tau, self.alpha_fixed, self.beta_fixed,
                         float(self.topk_fixed), float(self.prefix_blocks)], dtype=np.float64)


@dataclass
class Routing:
    alpha: np.ndarray      # [T]
    beta: np.ndarray       # [T]
    b: np.ndarray          # [T] int32, shared block count (Eq. 19)
    k: np.ndarray          # [T] int32, residual expert count (Eq. 27)
    shr_mask: np.ndarray   # [T] uint64, bit blk = block blk in I_shr (Eq. 22)
    q: np.ndarray          # [T][K] int32, experts by decreasing affinity (Eq. 25)
    p: np.ndarray          # [T][K] sorted affinities
    s: np.ndarray          # [T][K] affinities (Eq. 24)
    u: np.ndarray          # [T][B] block priorities (Eq. 21)
    margin: np.ndarray     # [T][4] near-tie margins (i)-(iv)

    def expert_mask(self) -> np.ndarray:
        """[T] uint64 set of selected residual experts {q_1..q_k}."""
        T, K = self.q.shape
        out = np.zeros(T, dtype=np.uint64)
        for i in range(K):
            sel = self.k > i
            out[sel] |= (np.uint64(1) << self.q[sel, i].astype(np.uint64))
        return out

    def cb(self, B: int) -> np.ndarray:
        """C_B = b + k (B - b) (Eq. 35)."""
        return self.b.astype(np.int64) + self.k.astype(np.int64) * (B - self.b.astype(np.int64))


def prototypes(w_up, B: int, round_mode: int) -> np.ndarray:
    """Eq. 20 on the shared expert (w_up[0]), rounded once to the router's
    storage precision (ROUND_F32 / ROUND_BF16) or kept exact (ROUND_NONE)."""
    w = _f64(w_up)
    if w.ndim == 3:
        w = np.ascontiguousarray(w[0])
    H, d = w.shape
    mu = np.empty((B, d), dtype=np.float64)
    rc = _load().oracle_prototypes(_p(w), d, H, B, round_mode, _p(mu))
    if rc != 0:
        raise ValueError("oracle_prototypes: bad shape")
    return mu


def route(x, w_router, mu, K: int, B: int, th: Optional[Thresholds] = None,
          mask=None, bias=None) -> Routing:
    xa = _f64(x)
    T, d = xa.shape
    wr = _f64(w_router)
    mu = _f64(mu)
    bias_a = None if bias is None else _f64(bias)
    m = _u8(mask)
    th = th or Thresholds()
    r = Routing(alpha=np.empty(T), beta=np.empty(T), b=np.empty(T, np.int32),
                k=np.empty(T, np.int32), shr_mask=np.empty(T, np.uint64),
                q=np.empty((T, K), np.int32), p=np.empty((T, K)), s=np.empty((T, K)),
                u=np.empty((T, B)), margin=np.empty((T, 4)))
    rc = _load().oracle_route(T, d, K, B, _p(xa), _p(m), _p(wr), _p(bias_a), _p(mu),
                              _p(th.array()), _p(r.alpha), _p(r.beta), _p(r.b), _p(r.k),
                              _p(r.shr_mask), _p(r.q), _p(r.p), _p(r.s), _p(r.u),
                              _p(r.margin))
    if rc != 0:
        raise ValueError("oracle_route: bad arguments")
    return r


def forward(x, w_up, w_down, r: Routing, B: int, mask=None) -> np.ndarray:
    """Eqs. 16, 28-30 for the decisions in `r` (any decisions may be passed,
    e.g. another implementation's, with this oracle's alpha and p)."""
    xa = _f64(x)
    T, d = xa.shape
    wu = _f64(w_up)
    wd = _f64(w_down)
    K = wu.shape[0] - 1
    H = wu.shape[1]
    m = _u8(mask)
    y = np.empty((T, d), dtype=np.float64)
    alpha = np.ascontiguousarray(r.alpha, dtype=np.float64)
    shr = np.ascontiguousarray(r.shr_mask, dtype=np.uint64)
    k = np.ascontiguousarray(r.k, dtype=np.int32)
    q = np.ascontiguousarray(r.q, dtype=np.int32)
    p = np.ascontiguousarray(r.p, dtype=np.float64)
    rc = _load().oracle_forward(T, d, H, K, B, _p(xa), _p(m), _p(wu), _p(wd), _p(alpha),
                                _p(shr), _p(k), _p(q), _p(p), _p(y))
    if rc != 0:
        raise ValueError("oracle_forward: bad arguments (%d)" % rc)
    return y


def layer(x, w_router, w_up, w_down, B: int, th: Optional[Thresholds] = None, mask=None,
          bias=None, round_mode: int = ROUND_NONE):
    """The whole layer: returns (y [T][d], Routing)."""
    wu = _f64(w_up)
    K = wu.shape[0] - 1
    mu = prototypes(wu, B, round_mode)
    r = route(x, w_router, mu, K, B, th, mask, bias)
    return forward(x, wu, w_down, r, B, mask), r


def groups(r: Routing, K: int, B: int, mask=None):
    """Group table: counts [(K+1)B] and, group after group, the rows
    (token, weight) in increasing token order. Group g = e*B + blk with e=0
    the shared expert and e=1+j residual expert j."""
    T = r.alpha.shape[0]
    m = _u8(mask)
    cap = int(np.sum(r.cb(B))) + 1
    counts = np.empty((K + 1) * B, np.int32)
    tok = np.empty(cap, np.int32)
    w = np.empty(cap, np.float64)
    alpha = np.ascontiguousarray(r.alpha, dtype=np.float64)
    n = _load().oracle_groups(T, K, B, _p(m), _p(alpha), _p(r.shr_mask), _p(r.k), _p(r.q),
                              _p(r.p), _p(counts), _p(tok), _p(w), cap)
    if n < 0:
        raise ValueError("oracle_groups: capacity")
    return counts, tok[:n].copy(), w[:n].copy()


def with_decisions(r: Routing, shr_mask: np.ndarray, expert_mask: np.ndarray, B: int) -> Routing:
    """This oracle's scores (alpha, s) combined with given discrete decisions
    (a shared block set and a residual expert set per token): q lists the
    given experts by decreasing affinity, p their affinities, k their count."""
    T, K = r.s.shape
    q = np.empty((T, K), np.int32)
    p = np.zeros((T, K))
    k = np.zeros(T, np.int32)
    for t in range(T):
        sel = [j for j in range(K) if (int(expert_mask[t]) >> j) & 1]
        sel.sort(key=lambda j: (-r.s[t, j], j))
        rest = [j for j in range(K) if j not in sel]
        order = sel + rest
        q[t] = order
        p[t] = r.s[t, order]
        k[t] = len(sel)
    b = np.array([bin(int(v)).count("1") for v in shr_mask], np.int32)
    return Routing(alpha=r.alpha.copy(), beta=r.beta.copy(), b=b, k=k,
                   shr_mask=np.asarray(shr_mask, np.uint64).copy(), q=q, p=p, s=r.s.copy(),
                   u=r.u.copy(), margin=r.margin.copy())


def layernorm(v, gamma, beta, eps: float, mask=None, round_mode: int = ROUND_NONE) -> np.ndarray:
    """Layer normalisation of each token over its d features (biased variance,
    eps inside the square root), rounded per round_mode; padding rows give 0."""
    va = _f64(v)
    T, d = va.shape
    g = _f64(gamma).reshape(d)
    b = _f64(beta).reshape(d)
    m = _u8(mask)
    out = np.empty((T, d), dtype=np.float64)
    rc = _load().oracle_layernorm(T, d, _p(va), _p(m), _p(g), _p(b), float(eps), round_mode,
                                  _p(out))
    if rc != 0:
        raise ValueError("oracle_layernorm: bad arguments")
    return out


def upcycle(w_up_dense, w_down_dense, K: int):
    """Sec. III: every expert (the shared one and the K residual ones) starts
    as the same dense FFN: K+1 copies of its up projection [H][d] and down
    projection [d][H]."""
    wu = _f64(w_up_dense)
    wd = _f64(w_down_dense)
    return (np.ascontiguousarray(np.broadcast_to(wu, (K + 1,) + wu.shape)),
            np.ascontiguousarray(np.broadcast_to(wd, (K + 1,) + wd.shape)))


def sublayer(x, w_router, w_up, w_down, B: int, gamma, beta, eps: float, norm_first: bool,
             th: Optional[Thresholds] = None, mask=None, bias=None,
             round_mode: int = ROUND_NONE):
    """The layer as a Transformer sublayer (backbones of Appendix A, Architecture details):
    norm_first (DeiT-S): out = x + F(LN(x)), LN(x) kept in the layer's input
    precision (round_mode); otherwise (BERT): out = LN(x + F(x)). Padding
    tokens give 0. Returns (out [T][d], Routing)."""
    xa = _f64(x)
    if norm_first:
        xn = layernorm(xa, gamma, beta, eps, mask, round_mode)
        y, r = layer(xn, w_router, w_up, w_down, B, th, mask, bias, round_mode)
        out = xa + y
    else:
        y, r = layer(xa, w_router, w_up, w_down, B, th, mask, bias, round_mode)
        out = layernorm(xa + y, gamma, beta, eps, mask, ROUND_NONE)
    if mask is not None:
        out[_u8(mask) == 0] = 0.0
    return out, r


@dataclass
class Grads:
    dx: np.ndarray         # [T][d]
    dw_up: np.ndarray      # [K+1][H][d]
    dw_down: np.ndarray    # [K+1][d][H]
    dw_router: np.ndarray  # [d][K+1]
    dbias: np.ndarray      # [K+1]


def backward(x, w_router, w_up, w_down, shr_mask, expert_mask, B: int, dy,
             th: Optional[Thresholds] = None, mask=None, bias=None) -> Grads:
    """dL/d(inputs, parameters) given dL/dy, through Eq. 30 with the given
    discrete decisions (shared block set and selected residual experts per
    token) held fixed; alpha and s are recomputed from x and the router."""
    xa = _f64(x)
    T, d = xa.shape
    wr = _f64(w_router)
    wu = _f64(w_up)
    wd = _f64(w_down)
    g = _f64(dy)
    K1, H = wu.shape[0], wu.shape[1]
    th = th or Thresholds()
    m = _u8(mask)
    bias_a = None if bias is None else _f64(bias)
    shr = np.ascontiguousarray(shr_mask, dtype=np.uint64)
    em = np.ascontiguousarray(expert_mask, dtype=np.uint64)
    out = Grads(dx=np.empty((T, d)), dw_up=np.empty((K1, H, d)), dw_down=np.empty((K1, d, H)),
                dw_router=np.empty((d, K1)), dbias=np.empty(K1))
    rc = _load().oracle_backward(T, d, H, K1 - 1, B, _p(xa), _p(m), _p(wr), _p(bias_a), _p(wu),
                                 _p(wd), _p(th.array()), _p(shr), _p(em), _p(g), _p(out.dx),
                                 _p(out.dw_up), _p(out.dw_down), _p(out.dw_router), _p(out.dbias))
    if rc != 0:
        raise ValueError("oracle_backward: bad arguments (%d)" % rc)
    return out


def diversity(w_router):
    """Eq. diversity-loss: (L_div, dL_div/dW*) for W* = w_router [d][K+1]."""
    wr = _f64(w_router)
    d, K1 = wr.shape
    grad = np.empty((d, K1))
    L = _load().oracle_diversity(d, K1, _p(wr), _p(grad))
    return float(L), grad
