"""CPU checks of the device noise generator's own math (csrc/philox.cuh).

The kernels evaluate ln(u0) and sin/cos(pi x) with fitted polynomials instead
of the CUDA math library.  These tests read the coefficients out of the
header, replay the kernel's float32 steps in numpy (each fmaf as one rounding
of the exact product-sum) and bound the error against float64 references:
the natural log, and the oracle's sincospi (exact argument reduction, so its
zeros are exact).  The GPU parity tests compare the whole generator with the
oracle; these pin the two approximations on their own, without a GPU.
"""
import os
import re

import numpy as np
import pytest

from oracle import dp_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "paper_2609_20532_gb300", "csrc", "philox.cuh")
FLOAT = r"(-?\d+\.\d+(?:e[-+]?\d+)?)f"


def _body(name):
    src = open(HEADER).read()
    start = src.index(f"__device__ __forceinline__ {name}")
    return src[start:src.index("\n}\n", start)]


def _f32(a):
    return np.asarray(a, dtype=np.float64).astype(np.float32).astype(np.float64)


def _fma(a, b, c):
    return _f32(np.asarray(a, np.float64) * b + c)


def _ln_u0(u):
    body = _body("float ln_u0")
    horner = body[body.index("float r ="):body.index("const float p")]
    r_coef = [float(v) for v in re.findall(FLOAT, horner)]  # R, highest degree first
    ln2 = float(re.findall(FLOAT, body[body.index("return"):])[0])
    assert len(r_coef) == 8
    i = np.asarray(u, np.float32).view(np.int32).astype(np.int64)
    e = (i - 0x3F2AAAAB) >> 23
    m = (i - (e << 23)).astype(np.int32).view(np.float32).astype(np.float64)
    f = _f32(m - 1.0)
    r = np.full_like(f, r_coef[0])
    for c in r_coef[1:]:
        r = _fma(r, f, c)
    p = _fma(_f32(f * f), r, f)
    return _fma(e.astype(np.float64), ln2, p)


def _sincospi_0_2(X):
    """The kernel's steps on X = RN(x_odd), the float of the word; they give
    sin / cos(pi x) for x = X 2^-31."""
    body = _body("void sincospi_0_2")
    ps_body = body[body.index("const float ps"):body.index("const float pc")]
    pc_body = body[body.index("const float pc"):body.index("const bool odd")]
    cs = [float(v) for v in re.findall(FLOAT, ps_body)]
    cc = [float(v) for v in re.findall(FLOAT, pc_body)]
    assert len(cs) == 5 and len(cc) == 5
    X = _f32(X)
    sh = _fma(X, 2.0 ** -30, 12582912.0)         # 2x + 1.5 * 2^23, rounded once
    mk = _fma(sh, -0.5, 6291456.0)               # -k / 2, exact
    q = sh.astype(np.float32).view(np.int32)
    y = _fma(X, 2.0 ** -31, mk)                  # x - k / 2
    # the folded steps equal the plain ones: k = sh - 1.5 * 2^23, y = x - k / 2
    k = _f32(sh - 12582912.0)
    assert np.array_equal(mk, -0.5 * k)
    assert np.array_equal(y, _fma(-0.5, k, _f32(X) * 2.0 ** -31))
    t = _f32(y * y)
    ps = np.full_like(t, cs[0])
    for c in cs[1:]:
        ps = _fma(ps, t, c)
    ps = _f32(ps * y)
    pc = np.full_like(t, cc[0])
    for c in cc[1:]:
        pc = _fma(pc, t, c)
    odd = (q & 1) != 0
    a, b = np.where(odd, pc, ps), np.where(odd, ps, pc)
    s = np.where((q & 2) != 0, -a, a)
    c = np.where(((q + 1) & 2) != 0, -b, b)
    return s, c


def _u0_from_words(w):
    """The kernel's u0 = RN_fp32((w + 1) / 2^32), 1 for w = 2^32 - 1."""
    w = np.asarray(w, np.uint64)
    return np.where(w == 0xFFFFFFFF, 1.0, _f32((w + 1).astype(np.float64)) * 2.0 ** -32)


def test_ln_u0_error_bound_over_its_domain():
    # every float32 in [2/3, 1] (the binade where ln u0 is near 0), then
    # sampled u0 in each binade down to 2^-32, and the generator's extremes
    m = np.arange(np.float32(2.0 / 3.0).view(np.int32), np.float32(1.0).view(np.int32),
                  dtype=np.int32).view(np.float32)
    rng = np.random.default_rng(0)
    parts = [m]
    for b in range(1, 33):
        mant = rng.integers(0, 1 << 23, 1 << 14)
        parts.append((mant | ((127 - b) << 23)).astype(np.int32).view(np.float32))
    parts.append(_u0_from_words([0, 1, 2, 0xFFFFFFFE]).astype(np.float32))
    u = np.concatenate(parts)
    u = u[u != 1.0]            # words near 2^32 - 1 round to u0 = 1 (checked below)
    got = _ln_u0(u)
    ref = np.log(u.astype(np.float64))
    rel = np.abs(got - ref) / np.abs(ref)
    assert rel.max() <= 1.6 * 2.0 ** -24, rel.max()
    assert _ln_u0(np.float32([1.0]))[0] == 0.0   # u0 = 1 gives z = 0 exactly


@pytest.mark.parametrize("seed", [0, 1])
def test_sincospi_error_bound_and_exact_zeros(seed):
    rng = np.random.default_rng(seed)
    words = rng.integers(0, 1 << 32, 1 << 20, dtype=np.uint64)
    edges = np.array([0, 1, 1 << 30, 1 << 31, 3 << 30, (1 << 32) - 1, (1 << 29), (5 << 29)],
                     dtype=np.uint64)
    words = np.concatenate([words, edges])
    X = _f32(words.astype(np.float64))                     # RN(x_odd)
    two_u1 = X * 2.0 ** -31                                  # 2 u1 = RN(x_odd) 2^-31
    s, c = _sincospi_0_2(X)
    s_ref, c_ref = O.sincospi(two_u1)
    for got, ref in ((s, s_ref), (c, c_ref)):
        zero = ref == 0
        assert np.all(got[zero] == 0)
        rel = np.abs(got[~zero] - ref[~zero]) / np.abs(ref[~zero])
        assert rel.max() <= 2.5 * 2.0 ** -24, rel.max()
