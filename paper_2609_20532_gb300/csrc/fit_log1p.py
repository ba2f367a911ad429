"""Derivation of the log1p polynomial coefficients of ln_u0() in philox.cuh.

The Box-Muller radius needs ln(u0) for u0 in [2^-32, 1].  The kernel splits
u0 = 2^e m with m in [2/3, 4/3) (from the float's bits), so f = m - 1 is exact
and |f| <= 1/3, and forms ln(u0) = e ln2 + log1p(f) with
log1p(f) = f + f^2 R(f), R a polynomial of degree 7.  R is fitted here by
iteratively reweighted least squares (Lawson's method toward the minimax fit)
on Chebyshev nodes, weighted for the relative error of log1p(f).  The script
then rounds the coefficients to float32, evaluates the kernel's float32 steps
(Horner with FMA, emulated by one rounding of the exact fp64 result per step)
for every float32 m in [2/3, 4/3) and for u0 across all 33 binades, and
prints the largest relative error against numpy's float64 log.  The printed
"deg 7" coefficients are the ones the kernel uses.

Run:  python paper_2609_20532_gb300/csrc/fit_log1p.py
"""
import numpy as np

N = 40001
lo, hi = -1.0 / 3.0, 1.0 / 3.0
x = 0.5 * (hi + lo) + 0.5 * (hi - lo) * np.cos(np.pi * (np.arange(N) + 0.5) / N)
x = x[np.abs(x) > 1e-9]


def fit(deg):
    target = (np.log1p(x) - x) / x ** 2  # R(f)
    V = np.stack([x ** k for k in range(deg + 1)], 1)
    wgt = x ** 2 / np.abs(np.log1p(x))  # error of R scaled into relative error of log1p
    c, *_ = np.linalg.lstsq(V * wgt[:, None], target * wgt, rcond=None)
    for _ in range(40):
        err = (V @ c - target) * wgt
        w = np.abs(err) + 1e-30
        w /= w.max()
        W = np.sqrt(w)
        c, *_ = np.linalg.lstsq(V * (wgt * W)[:, None], target * wgt * W, rcond=None)
    return c


def f32(a):
    return np.asarray(a, dtype=np.float64).astype(np.float32).astype(np.float64)


def fma32(a, b, c):
    return f32(a * b + c)  # products of two floats are exact in fp64; one rounding


def ln_u0(u, c):
    """The kernel's steps on float32 values u (numpy emulation)."""
    i = np.asarray(u, dtype=np.float32).view(np.int32).astype(np.int64)
    e = (i - 0x3F2AAAAB) >> 23
    m = (i - (e << 23)).astype(np.int32).view(np.float32).astype(np.float64)
    f = f32(m - 1.0)
    r = np.full_like(f, c[-1])
    for k in range(len(c) - 2, -1, -1):
        r = fma32(r, f, c[k])
    p = fma32(f32(f * f), r, f)
    return fma32(e.astype(np.float64), f32(np.log(2.0)), p)


if __name__ == "__main__":
    m_all = np.arange(np.float32(2.0 / 3.0).view(np.int32), np.float32(4.0 / 3.0).view(np.int32),
                      dtype=np.int32).view(np.float32)
    for deg in (6, 7, 8):
        c = f32(fit(deg))
        # every float32 m in [2/3, 4/3) (e = 0: u0 in [2/3, 1] is the part near ln = 0)
        got = ln_u0(m_all[m_all <= 1.0], c)
        ref = np.log(m_all[m_all <= 1.0].astype(np.float64))
        nz = ref != 0
        e0 = np.max(np.abs(got[nz] - ref[nz]) / np.abs(ref[nz]))
        # u0 in every binade of [2^-32, 1): 2^20 random float32 values per binade
        rng = np.random.default_rng(0)
        worst = 0.0
        for b in range(1, 33):
            u = (rng.integers(0, 1 << 23, 1 << 20) | ((127 - b) << 23)).astype(np.int32).view(np.float32)
            g = ln_u0(u, c)
            rf = np.log(u.astype(np.float64))
            worst = max(worst, float(np.max(np.abs(g - rf) / np.abs(rf))))
        print(f"deg {deg}: max rel err {max(e0, worst):.3e} ({max(e0, worst) / 2 ** -24:.2f} x 2^-24)")
        print("  coeffs (R_0 .. R_deg)", [float(v) for v in c])
