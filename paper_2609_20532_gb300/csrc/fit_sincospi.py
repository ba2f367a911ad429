"""Derivation of the sin(pi y) / cos(pi y) polynomial coefficients in philox.cuh.

sin(pi y) = y * P(y^2) and cos(pi y) = Q(y^2) on |y| <= 1/4, with P and Q of
degree 4, fitted by iteratively reweighted least squares (Lawson's method
toward the minimax fit) on Chebyshev nodes, relative error for sin and absolute
for cos.  The script then evaluates the float32-rounded coefficients with
float32 FMA Horner steps (emulated in numpy) on every fp32 value of y in
[0, 1/4) with spacing 2^-24 and prints the largest relative error against
numpy's float64 sin / cos: the "4 4" line is the one the kernel uses.

Run:  python paper_2609_20532_gb300/csrc/fit_sincospi.py
"""
import numpy as np
from numpy.polynomial import chebyshev as Ch
N = 20001
x = 0.25 * np.cos(np.pi * (np.arange(N) + 0.5) / N)   # Chebyshev nodes on [-1/4, 1/4]
x = x[x > 0]
def fit_sin(deg):   # sin(pi y) = y * P(y^2), P degree deg
    t = x * x
    V = np.stack([t ** k for k in range(deg + 1)], 1)
    target = np.sin(np.pi * x) / x
    # minimise relative error of sin: weight 1/target (target ~ pi)
    c, *_ = np.linalg.lstsq(V / target[:, None], np.ones_like(target), rcond=None)
    for _ in range(30):   # iteratively reweighted toward minimax (Lawson)
        err = (V @ c - target) / target
        w = np.abs(err) + 1e-30
        w = w / w.max()
        Wt = np.sqrt(w)[:, None]
        c, *_ = np.linalg.lstsq(Wt * V / target[:, None], Wt[:, 0] * np.ones_like(target), rcond=None)
    return c
def fit_cos(deg):   # cos(pi y) = Q(y^2)
    t = x * x
    V = np.stack([t ** k for k in range(deg + 1)], 1)
    target = np.cos(np.pi * x)
    c, *_ = np.linalg.lstsq(V, target, rcond=None)
    for _ in range(30):
        err = V @ c - target
        w = np.abs(err) + 1e-30; w /= w.max(); Wt = np.sqrt(w)[:, None]
        c, *_ = np.linalg.lstsq(Wt * V, Wt[:, 0] * target, rcond=None)
    return c
for ds, dc in [(4, 4), (5, 5), (4, 5)]:
    cs = fit_sin(ds).astype(np.float32); cc = fit_cos(dc).astype(np.float32)
    # evaluate in float32 Horner with fma emulated by fp64 rounding to fp32 each step
    ys = (np.arange(0, 2**22) / 2**24).astype(np.float32)   # y in [0, 1/4): exact fp32 grid
    y = ys.astype(np.float64)
    t = (ys * ys).astype(np.float32).astype(np.float64)
    def horner(c, t):
        acc = np.float64(c[-1]) * np.ones_like(t)
        for k in range(len(c) - 2, -1, -1):
            acc = (acc * t + np.float64(c[k])).astype(np.float32).astype(np.float64)
        return acc
    s = (horner(cs, t) * y).astype(np.float32).astype(np.float64)
    co = horner(cc, t)
    es = np.max(np.abs(s[1:] - np.sin(np.pi * y[1:])) / np.abs(np.sin(np.pi * y[1:])))
    ec = np.max(np.abs(co - np.cos(np.pi * y)) / np.abs(np.cos(np.pi * y)))
    print(ds, dc, "sin rel", es, "cos rel", ec, "ulp~", es / 2**-24, ec / 2**-24)
    print("  sin coeffs", [float(v) for v in cs]); print("  cos coeffs", [float(v) for v in cc])
