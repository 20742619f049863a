"""Generates the polynomial used by the tensor-core path's GeLU epilogue.

GeLU(x) = x Phi(x) = max(x, 0) - |x| Q(|x|), with Q(a) = Phi(-a), the upper
tail of the standard normal. Writing Q(a) = exp(-a^2/2) R(a) leaves
R(a) = erfcx(a / sqrt 2) / 2, a smooth, slowly varying function on [0, 5]
(from 1/2 down to about 0.076). R is fitted by least squares in the Chebyshev
basis (numpy) on [0, 5], mapped to s = 0.4 a - 1 in [-1, 1], and converted to
the power basis for Horner evaluation in fp32. Beyond |x| = 5 the argument is
clamped; there Q < 3e-7 and the absolute GeLU error stays below 5e-7.

Run:  python paper_2608_10392_gb300/csrc/gelu_coeffs.py
"""
import struct

import numpy as np
from scipy.special import erfcx
from scipy.stats import norm

A, DEG = 5.0, 12


def fit():
    a = np.linspace(0.0, A, 400001)
    r = 0.5 * erfcx(a / np.sqrt(2.0))
    cheb = np.polynomial.chebyshev.Chebyshev.fit(a, r, DEG, domain=[0.0, A])
    return np.polynomial.chebyshev.cheb2poly(cheb.coef).astype(np.float32)


def gelu_fp32(x, coef):
    ax = np.abs(x).astype(np.float32)
    s = (np.minimum(ax, np.float32(A)) * np.float32(2.0 / A) - np.float32(1.0)).astype(np.float32)
    v = np.full_like(s, coef[-1])
    for c in coef[-2::-1]:
        v = (v * s + c).astype(np.float32)
    q = np.exp(-(ax.astype(np.float64) ** 2) / 2.0).astype(np.float32) * v
    return np.maximum(x.astype(np.float32), np.float32(0)) - ax * q


if __name__ == "__main__":
    coef = fit()
    x = np.linspace(-10, 10, 400001)
    g = gelu_fp32(x, coef)
    ref = x * norm.cdf(x)
    inner = np.abs(x) <= A
    rel = np.abs(g - ref)[inner] / np.maximum(np.abs(ref[inner]), 1e-30)
    print("// max rel err |x|<=5: %.2e, max abs err: %.2e" % (rel.max(), np.abs(g - ref).max()))
    for i, c in enumerate(coef):
        bits = struct.unpack("<I", struct.pack("<f", float(c)))[0]
        print("  0x%08xu,  // c%d = %.9g" % (bits, i, c))
