"""Generates the polynomial used by the tensor-core path's GeLU epilogue.

GeLU(x) = x Phi(x) with Phi the standard normal CDF (the exact erf form).
The epilogue writes Phi(x) = (1 + tanh(g(x))) / 2, where g(x) =
atanh(2 Phi(x) - 1) is odd and smooth, and approximates g by x P(x^2) with P
a degree-4 polynomial. The coefficients minimise the largest error of
Phi on [0, 8] (Gauss-Newton steps with Lawson reweighting towards the
minimax solution, numpy/scipy); g then increases monotonically for all x, so
tanh saturates to +-1 beyond the fitted range.

On the GPU, tanh is the hardware approximation tanh.approx.f32, whose error
(about 2^-11) dominates the polynomial's (below 2e-6 on Phi): the GeLU
error stays a small fraction of the bf16 rounding that h receives next.

Run:  python tests/gelu_fit.py   (prints the constants the epilogue in
csrc/tc_common.cuh holds; tests/test_gelu_epilogue.py checks them)
"""
import struct

import numpy as np
from scipy.stats import norm

DEG, X_MAX = 4, 8.0


def _phi_err(c, x):
    return 0.5 * np.tanh(x * np.polyval(c[::-1], x * x)) - (norm.cdf(x) - 0.5)


def fit():
    x = np.linspace(1e-4, X_MAX, 40001)
    c = np.zeros(DEG + 1)
    c[0], c[1] = np.sqrt(2.0 / np.pi), 0.0356774  # tanh-form starting point
    w = np.ones_like(x)
    for _ in range(300):
        e = _phi_err(c, x)
        u = x * x
        t = np.tanh(x * np.polyval(c[::-1], u))
        jac = np.stack([0.5 * (1.0 - t * t) * x * u ** k for k in range(DEG + 1)], 1)
        sw = np.sqrt(w)
        c = c + 0.5 * np.linalg.lstsq(jac * sw[:, None], -e * sw, rcond=None)[0]
        e = _phi_err(c, x)
        w = w * (np.abs(e) / np.abs(e).max() + 1e-3)
        w /= w.mean()
    return c.astype(np.float32)


def gelu_fp32(x, coef):
    """The epilogue's arithmetic in fp32, with an exact tanh."""
    x = x.astype(np.float32)
    u = x * x
    r = np.full_like(u, coef[-1])
    for c in coef[-2::-1]:
        r = (r * u + c).astype(np.float32)
    g = (x * r).astype(np.float32)
    hx = np.float32(0.5) * x
    return (hx * np.tanh(g).astype(np.float32) + hx).astype(np.float32)


if __name__ == "__main__":
    coef = fit()
    x = np.linspace(-12, 12, 480001)
    ref = x * norm.cdf(x)
    g = gelu_fp32(x, coef).astype(np.float64)
    phi_err = np.abs(_phi_err(coef.astype(np.float64), np.linspace(1e-4, X_MAX, 40001))).max()
    gg = np.linspace(0, 1e3, 100001)
    mono = bool(np.all(np.diff(gg * np.polyval(coef[::-1].astype(np.float64), gg * gg)) > 0))
    print("// max |Phi err| %.2e, max |GeLU err| / max(|x|, 1) %.2e, g monotone: %s"
          % (phi_err, (np.abs(g - ref) / np.maximum(np.abs(x), 1)).max(), mono))
    for i, c in enumerate(coef):
        bits = struct.unpack("<I", struct.pack("<f", float(c)))[0]
        print("  0x%08x  // c%d = %.9g" % (bits, i, c))
