"""CPU oracle of the diagnostic analyses of Sec. II-B (fp64, numpy).

TEST INFRASTRUCTURE ONLY, like the rest of `oracle/`: the tests are the only
callers; nothing here imports the CUDA package.

The analyses run on the K residual experts of a layer (experts 1..K of the
weight arrays; the diagnosis in the paper is of a standard top-2 MoE whose
experts were copied from one dense FFN) and its residual router W_g:

  value alignment (Eq. shared-set): for experts i, j and channel h,
      c_ijh = V_i[h,:] . V_j[h,:] / (|V_i[h,:]| |V_j[h,:]|),
      S_ij(delta) = {h : c_ijh >= delta},  rho_ij = |S_ij| / H;
  functional demand (Eqs. diagnostic-original .. functional-demand): for a
  token x with top-2 pair (i, j) of s = softmax(x W_g) and normalised
  weights s~_e = s_e / (s_i + s_j),
      y_orig = sum_{e in {i,j}} s~_e E_e(x),  S_bar = sum s~_e E_e^{S_ij}(x),
      r = y_orig - S_bar,
      R_m = the residual outputs E_{q_1}^{R_ij}, ..., E_{q_m}^{R_ij} (rows),
            q the expert order of a residual router W_r (x W_r, decreasing),
      a* = argmin_a |a^T R_m - r|^2 + gamma_m |a|^2,
            gamma_m = 1e-6 tr(R_m R_m^T) / m,
      e_m = |S_bar + a*^T R_m - y_orig| / max(|y_orig|, 1e-12),
      k_eps = min({m : e_m <= eps} u {K+1}),
  with E_e^{S}(x) = sum_{h in S} GeLU(x K_e[:,h]) V_e[h,:] and R the
  complement of S.

Readings where the paper is silent: ties (top-2 pair, residual order) go to
the lower index; a value row of zero norm is aligned with nothing (c = 0);
with R_m = 0 the fit is a = 0; the residual router W_r is given (the paper
trains one on the residual positions, which needs data).
"""
from __future__ import annotations

import numpy as np
from scipy.special import erf

from . import _f64


def _gelu(v):
    return 0.5 * v * (1.0 + erf(v / np.sqrt(2.0)))


def value_alignment(w_down, delta: float):
    """(rho [K][K], S [K][K][H] bool) over the residual experts 1..K of
    w_down [K+1][d][H] (Eq. shared-set)."""
    wd = _f64(w_down)
    V = np.transpose(wd[1:], (0, 2, 1))  # [K][H][d]: value rows
    K, H, _ = V.shape
    norms = np.sqrt(np.einsum("khd,khd->kh", V, V))
    S = np.zeros((K, K, H), dtype=bool)
    for i in range(K):
        for j in range(K):
            dots = np.einsum("hd,hd->h", V[i], V[j])
            den = norms[i] * norms[j]
            c = np.where(den > 0, dots / np.where(den > 0, den, 1.0), 0.0)
            S[i, j] = c >= delta
    return S.sum(axis=2) / H, S


def top2_pairs(x, w_router, bias=None):
    """Each token's top-2 residual experts (i < j not required: i has the
    larger affinity) and their normalised weights, from s = softmax(x W_g)
    (Eq. 24), ties to the lower index."""
    xa = _f64(x)
    wr = _f64(w_router)
    z = xa @ wr[:, 1:]
    if bias is not None:
        z = z + _f64(bias)[1:]
    z = z - z.max(axis=1, keepdims=True)
    s = np.exp(z)
    s /= s.sum(axis=1, keepdims=True)
    order = np.argsort(-s, axis=1, kind="stable")
    i, j = order[:, 0], order[:, 1]
    si, sj = s[np.arange(len(s)), i], s[np.arange(len(s)), j]
    return i, j, si / (si + sj), sj / (si + sj)


def expert_outputs(x, w_up, w_down, mask):
    """E_e(x) and E_e^S(x) (Eq. ffn-kv restricted to channel sets) of the
    residual experts e = 1..K for every token: ([T][K][d], [T][K][d]);
    mask [T][H] bool is each token's channel set S."""
    xa = _f64(x)
    wu = _f64(w_up)[1:]            # [K][H][d] keys (rows)
    wd = _f64(w_down)[1:]          # [K][d][H]
    K, H, d = wu.shape
    T = xa.shape[0]
    m = np.asarray(mask, dtype=np.float64)
    E = np.empty((T, K, d))
    ES = np.empty((T, K, d))
    for e in range(K):
        G = _gelu(xa @ wu[e].T)       # [T][H]
        E[:, e] = G @ wd[e].T
        ES[:, e] = (G * m) @ wd[e].T
    return E, ES


def functional_demand(x, w_router, w_up, w_down, w_res, delta: float, eps: float, bias=None):
    """(k_eps [T], e [T][K], pair [T][2]) for every token (the equations of
    the module docstring)."""
    xa = _f64(x)
    K = _f64(w_up).shape[0] - 1
    T = xa.shape[0]
    _, S = value_alignment(w_down, delta)
    i, j, ti, tj = top2_pairs(xa, w_router, bias)
    q = np.argsort(-(xa @ _f64(w_res)), axis=1, kind="stable")  # residual order
    E, ES = expert_outputs(xa, w_up, w_down, S[i, j])  # S the token's pair set
    ER = E - ES
    rows = np.arange(T)
    y = ti[:, None] * E[rows, i] + tj[:, None] * E[rows, j]
    s_bar = ti[:, None] * ES[rows, i] + tj[:, None] * ES[rows, j]
    r = y - s_bar
    errs = np.empty((T, K))
    k_eps = np.full(T, K + 1, dtype=np.int32)
    for t in range(T):
        ynorm = max(np.linalg.norm(y[t]), 1e-12)
        for m in range(1, K + 1):
            R = ER[t, q[t, :m]]          # [m][d]
            Gm = R @ R.T
            tr = np.trace(Gm)
            if tr > 0:
                a = np.linalg.solve(Gm + 1e-6 * tr / m * np.eye(m), R @ r[t])
            else:
                a = np.zeros(m)
            errs[t, m - 1] = np.linalg.norm(s_bar[t] + a @ R - y[t]) / ynorm
            if errs[t, m - 1] <= eps and k_eps[t] == K + 1:
                k_eps[t] = m
    return k_eps, errs, np.stack([i, j], axis=1).astype(np.int32)
