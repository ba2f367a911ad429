"""Pins of the fp64 oracle against things other than itself (CPU only).

Each pin is chosen so that a plausible mistake in the oracle (a dropped term,
a wrong sign or index, a transposed operand, a wrong constant) fails at least
one of them; ``test_planted_mistakes_are_caught`` plants such mistakes in
copies of oracle functions and checks that the pin helpers reject them.
"""

import json
import math
import os
import shutil
import subprocess

import numpy as np
import pytest

import workloads as W
from oracle import dp_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------
# helpers (pin checks, written so the planted-mistake test can reuse them)
# ---------------------------------------------------------------------------

def brute_force_grads(A, D):
    """Pure-Python triple loop: G[i][j][k] = sum_t A[i][t][j] * D[i][t][k]."""
    B, T, din = A.shape
    dout = D.shape[2]
    Al, Dl = A.tolist(), D.tolist()
    G = [[[0.0] * dout for _ in range(din)] for _ in range(B)]
    for i in range(B):
        for t in range(T):
            for j in range(din):
                a = Al[i][t][j]
                for k in range(dout):
                    G[i][j][k] += a * Dl[i][t][k]
    return np.array(G)


def _tiny(rng, B, T, din, dout):
    return rng.standard_normal((B, T, din)), rng.standard_normal((B, T, dout))


def check_grads_brute(grads_fn, sqnorm_fn, seeds=range(6)) -> bool:
    for sd in seeds:
        rng = np.random.default_rng(sd)
        B, T = int(rng.integers(1, 5)), int(rng.integers(1, 4))
        din, dout = int(rng.integers(1, 6)), int(rng.integers(1, 6))
        A, D = _tiny(rng, B, T, din, dout)
        Gb = brute_force_grads(A, D)
        G = grads_fn(A, D)
        if G.shape != Gb.shape or not np.allclose(G, Gb, rtol=1e-12, atol=1e-12):
            return False
        nb = np.array([sum(x * x for x in Gb[i].ravel().tolist()) for i in range(B)])
        if not np.allclose(sqnorm_fn(A, D), nb, rtol=1e-12, atol=1e-14):
            return False
    return True


def check_clip_defining_properties(clip_fn) -> bool:
    """Clipped examples end up with norm exactly C; unclipped keep c = 1."""
    rng = np.random.default_rng(7)
    C = 0.7
    L, B = 3, 64
    scales = np.logspace(-3, 3, B)          # straddles the clip boundary
    n = rng.random((L, B)) * scales[None, :] ** 2
    s, c = clip_fn(n, C)
    if not np.allclose(s, n.sum(0), rtol=1e-14):
        return False
    norm = np.sqrt(s)
    clipped = norm > C
    if not (clipped.any() and (~clipped).any()):
        return False
    if not np.all((c > 0) & (c <= 1)):
        return False
    if not np.all(c * norm <= C * (1 + 1e-6)):
        return False
    if not np.allclose(c[clipped] * norm[clipped], C, rtol=1e-12):
        return False
    return bool(np.all(c[~clipped] == 1.0))


def check_box_muller_identities(bm_fn) -> bool:
    rng = np.random.default_rng(3)
    u0 = rng.random(10000) * (1 - 1e-9) + 1e-9
    u1 = rng.random(10000)
    z0, z1 = bm_fn(u0, u1)
    r2 = -2.0 * np.log(u0)
    if not np.allclose(z0 * z0 + z1 * z1, r2, rtol=1e-12, atol=1e-300):
        return False
    ang = np.mod(np.arctan2(z1, z0), 2 * np.pi)
    d = np.abs(ang - 2 * np.pi * u1)
    d = np.minimum(d, 2 * np.pi - d)
    return bool(np.all(d < 1e-9))


_PHILOX_BIN = None


def _philox_torch_bin(tmp_dir):
    """Build the PyTorch-header Philox reference once per session."""
    global _PHILOX_BIN
    if _PHILOX_BIN and os.path.exists(_PHILOX_BIN):
        return _PHILOX_BIN
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not available")
    import torch
    inc = os.path.join(os.path.dirname(torch.__file__), "include")
    if not os.path.exists(os.path.join(inc, "ATen", "core", "PhiloxRNGEngine.h")):
        pytest.skip("PyTorch C++ headers not installed")
    src = os.path.join(os.path.dirname(__file__), "philox_torch_ref.cpp")
    out = os.path.join(tmp_dir, "philox_torch_ref")
    subprocess.run([gxx, "-O1", "-std=c++17", "-I", inc, src, "-o", out], check=True)
    _PHILOX_BIN = out
    return out


def _philox_cases():
    M64 = (1 << 64) - 1
    seeds = [0, 1, 0xFFFFFFFF, 1 << 32, M64, 0x123456789ABCDEF0]
    steps = [0, 1, 0xFFFFFFFF, 1 << 32, M64, 987654321]
    quads = [0, 1, 2, 0xFFFFFFFF, 1 << 32, M64, 35_126_000]
    rng = np.random.default_rng(11)
    cases = [(s, t, q) for s in seeds for t in steps for q in quads]
    for _ in range(300):
        cases.append(tuple(int(x) for x in rng.integers(0, 1 << 63, size=3, dtype=np.int64)))
    return cases


def check_philox_vs_torch(quads_fn, binpath) -> bool:
    cases = _philox_cases()
    inp = "\n".join(f"{s} {t} {q}" for s, t, q in cases) + "\n"
    res = subprocess.run([binpath], input=inp, capture_output=True, text=True, check=True)
    ref = np.array([[int(x) for x in ln.split()] for ln in res.stdout.strip().splitlines()],
                   dtype=np.uint64)
    got = np.array([quads_fn(s, t, q, 1)[0] for s, t, q in cases], dtype=np.uint64)
    return got.shape == ref.shape and bool(np.all(got == ref))


# ---------------------------------------------------------------------------
# per-example gradients and norms
# ---------------------------------------------------------------------------

def test_grads_and_norms_match_brute_force():
    assert check_grads_brute(O.per_example_grads, O.layer_sqnorms_materialised)
    assert check_grads_brute(O.per_example_grads, O.layer_sqnorms_ghost)


def test_rank1_closed_form():
    rng = np.random.default_rng(5)
    A, D = _tiny(rng, 9, 1, 37, 11)
    expect = np.einsum("bj,bj->b", A[:, 0], A[:, 0]) * np.einsum("bk,bk->b", D[:, 0], D[:, 0])
    np.testing.assert_allclose(O.layer_sqnorms_materialised(A, D), expect, rtol=1e-13)
    np.testing.assert_allclose(O.layer_sqnorms_ghost(A, D), expect, rtol=1e-13)


@pytest.mark.parametrize("T,din,dout", [(2, 3, 5), (17, 40, 9), (64, 96, 128), (130, 33, 70)])
def test_ghost_equals_materialised(T, din, dout):
    rng = np.random.default_rng(T * 1000 + din)
    A, D = _tiny(rng, 3, T, din, dout)
    np.testing.assert_allclose(O.layer_sqnorms_ghost(A, D),
                               O.layer_sqnorms_materialised(A, D), rtol=1e-12)


@pytest.mark.parametrize("name", ["single_fp32", "mlp_fp32", "block_bf16", "llm_bf16"])
def test_ghost_equals_materialised_on_workload_first_example(name):
    w = W.get(name)
    for l in range(len(w.layers)):
        A, D = W.make_layer(w, l, seed=0, B=1)
        A, D = W.to_f64(A), W.to_f64(D)
        np.testing.assert_allclose(O.layer_sqnorms_ghost(A, D),
                                   O.layer_sqnorms_materialised(A, D), rtol=1e-12)


# ---------------------------------------------------------------------------
# clip factors
# ---------------------------------------------------------------------------

def test_clip_defining_properties():
    assert check_clip_defining_properties(O.clip_factors)


def test_clip_special_cases():
    # zero gradient: c = 1 (reading of min(1, C/0))
    s, c = O.clip_factors(np.zeros((2, 3)), 1.0)
    assert np.all(c == 1.0) and np.all(s == 0.0)
    # tie ||g|| = C exactly: c = 1
    s, c = O.clip_factors(np.array([[0.25], [0.75]]), 1.0)
    assert s[0] == 1.0 and c[0] == 1.0
    # just above the tie: clipped, c < 1
    s, c = O.clip_factors(np.array([[0.25], [0.75 + 1e-12]]), 1.0)
    assert c[0] < 1.0
    with pytest.raises(ValueError):
        O.clip_factors(np.array([[np.nan]]), 1.0)
    with pytest.raises(ValueError):
        O.clip_factors(np.array([[1.0]]), 0.0)


def test_scaled_example_law():
    """Scaling one example's D by lambda scales its clip factor by 1/lambda."""
    rng = np.random.default_rng(9)
    A, D = _tiny(rng, 4, 3, 6, 5)
    C = 0.01                                   # all examples clipped
    _, c0 = O.clip_factors(O.layer_sqnorms(A, D)[None], C)
    lam = 3.7
    D2 = D.copy()
    D2[2] *= lam
    _, c1 = O.clip_factors(O.layer_sqnorms(A, D2)[None], C)
    np.testing.assert_allclose(c1[2], c0[2] / lam, rtol=1e-13)
    np.testing.assert_array_equal(np.delete(c1, 2), np.delete(c0, 2))


def test_clipped_examples_and_aggregate_respect_bounds():
    """||c_i g_i|| <= C(1+1e-6) per example; ||S/B|| <= C(1+1e-4) (Sec. 6.2)."""
    rng = np.random.default_rng(21)
    B = 12
    layers = []
    for din, dout in [(7, 5), (5, 3)]:
        A, D = _tiny(rng, B, 4, din, dout)
        D *= np.logspace(-2, 2, B)[:, None, None]
        layers.append((A, D))
    C = 1.3
    n = np.stack([O.layer_sqnorms(A, D) for A, D in layers])
    s, c = O.clip_factors(n, C)
    per = np.zeros(B)
    for A, D in layers:
        G = O.per_example_grads(A, D)
        per += np.sum((c[:, None, None] * G) ** 2, axis=(1, 2))
    assert np.all(np.sqrt(per) <= C * (1 + 1e-6))
    agg = math.sqrt(sum(np.sum(O.clipped_sum(A, D, c) ** 2) for A, D in layers))
    assert agg / B <= C * (1 + 1e-4)


# ---------------------------------------------------------------------------
# clipped sum
# ---------------------------------------------------------------------------

def test_clipped_sum_reduces_to_plain_matmul_when_nothing_clips():
    rng = np.random.default_rng(4)
    A, D = _tiny(rng, 5, 7, 13, 9)
    _, c = O.clip_factors(O.layer_sqnorms(A, D)[None], 1e30)
    assert np.all(c == 1.0)
    S = O.clipped_sum(A, D, c)
    ref = np.matmul(A.reshape(-1, 13).T, D.reshape(-1, 9))
    np.testing.assert_allclose(S, ref, rtol=1e-12, atol=1e-12)


def test_clipped_sum_is_sum_of_scaled_brute_force_grads():
    rng = np.random.default_rng(6)
    A, D = _tiny(rng, 3, 2, 4, 3)
    c = np.array([0.5, 1.0, 0.125])
    Gb = brute_force_grads(A, D)
    ref = sum(c[i] * Gb[i] for i in range(3))
    np.testing.assert_allclose(O.clipped_sum(A, D, c), ref, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(O.clipped_sum(A, D, 3 * c), 3 * ref, rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------------------
# Philox, uniforms, Box-Muller, Gaussian noise
# ---------------------------------------------------------------------------

def test_philox_matches_pytorch_reference(tmp_path_factory):
    binpath = _philox_torch_bin(str(tmp_path_factory.mktemp("philox")))
    assert check_philox_vs_torch(O.philox_quads, binpath)


def test_philox_avalanche():
    """One flipped counter bit flips about half of the 128 output bits."""
    rng = np.random.default_rng(2)
    base = rng.integers(0, 1 << 32, size=(4, 4096), dtype=np.uint64)
    out0 = np.stack(O.philox4x32_10(list(base), (123, 456)))
    flips = []
    for word in range(4):
        for bit in (0, 13, 31):
            ctr = base.copy()
            ctr[word] ^= np.uint64(1 << bit)
            out1 = np.stack(O.philox4x32_10(list(ctr), (123, 456)))
            x = (out0 ^ out1).astype(np.uint64)
            cnt = sum(int(np.sum((x >> np.uint64(b)) & np.uint64(1))) for b in range(32))
            flips.append(cnt / (4096 * 128))
    assert all(abs(f - 0.5) < 0.01 for f in flips), flips


def test_uniform_edges_golden():
    g = json.load(open(os.path.join(GOLDEN, "uniform_edges.json")))
    xs0 = np.array([e["x"] for e in g["u0"]], dtype=np.uint64)
    xs1 = np.array([e["x"] for e in g["u1"]], dtype=np.uint64)
    u0, _ = O.uniforms_from_words(xs0, np.zeros_like(xs0))
    _, u1 = O.uniforms_from_words(np.zeros_like(xs1), xs1)
    np.testing.assert_array_equal(u0, [e["u"] for e in g["u0"]])
    np.testing.assert_array_equal(u1, [e["u"] for e in g["u1"]])
    for e in g["box_muller"]:
        z0, z1 = O.box_muller(np.array([e["u0"]]), np.array([e["u1"]]))
        assert abs(z0[0] - e["z0"]) <= 1e-15 * max(1, abs(e["z0"]))
        assert abs(z1[0] - e["z1"]) <= 1e-15 * max(1, abs(e["z1"]))


def test_box_muller_identities():
    assert check_box_muller_identities(O.box_muller)


def test_sincospi_exact_zeros():
    s, c = O.sincospi(np.array([0.0, 0.5, 1.0, 1.5, 2.0]))
    np.testing.assert_array_equal(np.abs(s[[0, 2, 4]]), 0.0)
    np.testing.assert_array_equal(np.abs(c[[1, 3]]), 0.0)


def test_noise_statistics():
    from scipy import stats
    n = 1 << 24
    z = O.gaussian_noise(0, 0, 0, n)
    assert abs(z.mean()) <= 5 / math.sqrt(n)
    assert abs(z.var() - 1) <= 5 * math.sqrt(2 / n)
    assert stats.kstest(z[: 1 << 22], "norm").pvalue > 1e-4
    # tails reach beyond 5 sigma only rarely, and never beyond sqrt(64 ln 2)
    assert np.max(np.abs(z)) <= math.sqrt(64 * math.log(2)) + 1e-12


def test_noise_scale_matches_paper_table():
    g = json.load(open(os.path.join(GOLDEN, "noise_scale_table.json")))
    n = 1 << 21
    z = O.gaussian_noise(1, 0, 0, n)
    for row in g["rows"]:
        sd = np.std(row["sigma"] * g["C"] * z / row["B"])
        # printed to 3 significant figures; statistical error of the sample std
        tol = 0.5 * 10 ** (math.floor(math.log10(row["sigmaC_over_B"])) - 2)
        tol += 5 * sd / math.sqrt(2 * n)
        assert abs(sd - row["sigmaC_over_B"]) <= tol, (row, sd)


def test_noise_indexing_is_slice_invariant():
    full = O.gaussian_noise(42, 7, 0, 1001)
    for a, b in [(0, 1001), (1, 10), (3, 4), (4, 8), (5, 999), (1000, 1001)]:
        np.testing.assert_array_equal(O.gaussian_noise(42, 7, a, b - a), full[a:b])


def test_noise_keying():
    a = O.gaussian_noise(0, 0, 0, 4096)
    assert np.array_equal(a, O.gaussian_noise(0, 0, 0, 4096))
    assert not np.any(a == O.gaussian_noise(0, 1, 0, 4096))
    assert not np.any(a == O.gaussian_noise(1, 0, 0, 4096))


# ---------------------------------------------------------------------------
# whole step and audit
# ---------------------------------------------------------------------------

def test_dp_step_sigma_zero_is_clipped_sum():
    w = W.get("single_fp32")
    layers = [(W.to_f64(A), W.to_f64(D)) for A, D in W.make_inputs(w)]
    r = O.dp_step(layers, w.C, 0.0, 0, 0, out_scale=1.0 / w.B)
    r0 = O.dp_step(layers, w.C, w.sigma, 0, 0, out_scale=1.0 / w.B, noise=False)
    np.testing.assert_array_equal(r["out"][0], r0["out"][0])
    np.testing.assert_allclose(r["out"][0], r["S"][0] / w.B, rtol=1e-15)


def test_dp_step_noise_offsets_follow_layer_order():
    w = W.get("mlp_fp32")
    rng = np.random.default_rng(0)
    layers = [(rng.standard_normal((4, 1, i)), rng.standard_normal((4, 1, o)))
              for i, o in [(5, 3), (3, 7), (7, 2)]]
    r = O.dp_step(layers, 1.0, 2.0, 5, 9)
    z = O.gaussian_noise(5, 9, 0, 15 + 21 + 14)
    off = 0
    for S, out in zip(r["S"], r["out"]):
        np.testing.assert_allclose(out - S, 2.0 * z[off:off + S.size].reshape(S.shape),
                                   rtol=1e-12, atol=1e-12)
        off += S.size


def test_audit_records():
    rng = np.random.default_rng(1)
    n = rng.random((3, 10))
    s, c = O.clip_factors(n, 0.5)
    recs = O.audit_records(n, s, c, [7, 2])
    assert [r["example"] for r in recs] == [7, 2]
    np.testing.assert_array_equal(recs[0]["layer_sqnorm"], n[:, 7])
    assert recs[1]["clip_factor"] == c[2] and recs[1]["total_sqnorm"] == s[2]


# ---------------------------------------------------------------------------
# planted mistakes: each must be rejected by a pin helper above
# ---------------------------------------------------------------------------

def test_planted_mistakes_are_caught(tmp_path_factory):
    # transposed per-example gradient (D^T A instead of A^T D)
    def grads_transposed(A, D):
        return np.stack([D[i].T @ A[i] for i in range(A.shape[0])])
    assert not check_grads_brute(grads_transposed, O.layer_sqnorms_materialised)

    # norm without squaring one factor
    def sqnorm_dropped_square(A, D):
        return np.array([np.sum(np.abs(A[i].T @ D[i])) for i in range(A.shape[0])])
    assert not check_grads_brute(O.per_example_grads, sqnorm_dropped_square)

    # ghost norm with one Gram transposed into the wrong contraction
    def ghost_wrong(A, D):
        return np.array([np.sum((A[i] @ A[i].T) * (D[i] @ D[i].T).sum(0)) for i in range(A.shape[0])])
    assert not check_grads_brute(O.per_example_grads, ghost_wrong)

    # clip factor C/s instead of C/sqrt(s)
    def clip_no_sqrt(n, C):
        s = np.sum(n, axis=0)
        c = np.where(s > C * C, C / np.maximum(s, 1e-300), 1.0)
        return s, c
    assert not check_clip_defining_properties(clip_no_sqrt)

    # clip that never clips (min dropped)
    def clip_no_min(n, C):
        s = np.sum(n, axis=0)
        return s, C / np.sqrt(s)
    assert not check_clip_defining_properties(clip_no_min)

    # Box-Muller with sin and cos swapped, or the wrong log argument
    def bm_swapped(u0, u1):
        z0, z1 = O.box_muller(u0, u1)
        return z1, z0
    assert not check_box_muller_identities(bm_swapped)

    def bm_wrong_log(u0, u1):
        return O.box_muller(u1 * 0.5 + 0.25, u0)
    assert not check_box_muller_identities(bm_wrong_log)

    # Philox with a wrong multiplier, wrong number of rounds, or the key bump
    # applied before the first round
    binpath = _philox_torch_bin(str(tmp_path_factory.mktemp("philox_m")))

    def make_quads(mutant):
        def quads(seed, step, q0, n):
            q = np.arange(n, dtype=np.uint64) + np.uint64(q0)
            M = np.uint64(0xFFFFFFFF)
            ctr = (q & M, q >> np.uint64(32), np.uint64(step & 0xFFFFFFFF), np.uint64(step >> 32))
            return np.stack(mutant(ctr, (seed & 0xFFFFFFFF, seed >> 32)), axis=1)
        return quads

    def philox_variant(m0=O.PHILOX_M0, rounds=10, bump_first=False):
        def f(ctr, key):
            M = np.uint64(0xFFFFFFFF)
            x = [np.asarray(w, dtype=np.uint64) & M for w in ctr]
            k0, k1 = np.uint64(key[0]), np.uint64(key[1])
            for r in range(rounds):
                if r or bump_first:
                    k0 = (k0 + np.uint64(O.PHILOX_W0)) & M
                    k1 = (k1 + np.uint64(O.PHILOX_W1)) & M
                p0 = np.uint64(m0) * x[0]
                p1 = np.uint64(O.PHILOX_M1) * x[2]
                x = [(p1 >> np.uint64(32)) ^ x[1] ^ k0, p1 & M, (p0 >> np.uint64(32)) ^ x[3] ^ k1, p0 & M]
            return [w.astype(np.uint32) for w in x]
        return f

    assert check_philox_vs_torch(make_quads(philox_variant()), binpath)
    assert not check_philox_vs_torch(make_quads(philox_variant(m0=0xD2511F55)), binpath)
    assert not check_philox_vs_torch(make_quads(philox_variant(rounds=7)), binpath)
    assert not check_philox_vs_torch(make_quads(philox_variant(bump_first=True)), binpath)


# ---------------------------------------------------------------------------
# AdamW after the seed release (App. A one-step map; Algorithm 2 OptStep)
# ---------------------------------------------------------------------------

def adamw_scalar_loop(theta, m, v, g, lr, b1, b2, eps, wd, t):
    out = []
    for th, mm, vv, gg in zip(theta.tolist(), m.tolist(), v.tolist(), g.tolist()):
        m2 = b1 * mm + (1 - b1) * gg
        v2 = b2 * vv + (1 - b2) * gg * gg
        mh = m2 / (1 - b1 ** t)
        vh = v2 / (1 - b2 ** t)
        out.append((th - lr * (mh / (math.sqrt(vh) + eps) + wd * th), m2, v2))
    return [np.array(x) for x in zip(*out)]


def check_adamw_golden(step_fn) -> bool:
    g = json.load(open(os.path.join(GOLDEN, "adamw_hand.json")))
    for c in g["cases"]:
        th, m, v = step_fn(np.array([c["theta"]]), np.array([c["m"]]), np.array([c["v"]]),
                           np.array([c["g"]]), c["lr"], c["beta1"], c["beta2"], c["eps"],
                           c["wd"], c["t"])
        if not (np.isclose(th[0], c["theta_new"], rtol=1e-14, atol=1e-15)
                and np.isclose(m[0], c["m_new"], rtol=1e-14, atol=1e-15)
                and np.isclose(v[0], c["v_new"], rtol=1e-14, atol=1e-15)):
            return False
    return True


def test_adamw_golden_cases():
    assert check_adamw_golden(O.adamw_step)


def test_adamw_matches_scalar_loop():
    rng = np.random.default_rng(17)
    n = 257
    theta, m, g = rng.standard_normal((3, n))
    v = rng.random(n)
    for t in (1, 2, 10, 1000):
        got = O.adamw_step(theta, m, v, g, 3e-4, 0.9, 0.999, 1e-8, 0.01, t)
        ref = adamw_scalar_loop(theta, m, v, g, 3e-4, 0.9, 0.999, 1e-8, 0.01, t)
        for a, b in zip(got, ref):
            np.testing.assert_allclose(a, b, rtol=1e-14, atol=1e-16)
    with pytest.raises(ValueError):
        O.adamw_step(theta, m, v, g, 1e-3, 0.9, 0.999, 1e-8, 0.0, 0)


def test_noise_adamw_composes_noise_and_step():
    rng = np.random.default_rng(3)
    shape = (7, 9)
    committed, theta, m = rng.standard_normal((3,) + shape)
    v = rng.random(shape)
    g, th, m2, v2 = O.noise_adamw(committed, theta, m, v, 4, 6, 100, 1.1, 0.5, 0.25,
                                  1e-3, 0.9, 0.99, 1e-8, 0.02, 5)
    z = O.gaussian_noise(4, 6, 100, 63).reshape(shape)
    np.testing.assert_allclose(g, committed + 0.25 * 1.1 * 0.5 * z, rtol=1e-15)
    ref = O.adamw_step(theta, m, v, g, 1e-3, 0.9, 0.99, 1e-8, 0.02, 5)
    for a, b in zip((th, m2, v2), ref):
        np.testing.assert_array_equal(a, b)


def test_planted_adamw_mistakes_are_caught():
    def no_bias_correction(theta, m, v, g, lr, b1, b2, eps, wd, t):
        m2 = b1 * m + (1 - b1) * g
        v2 = b2 * v + (1 - b2) * g * g
        return theta - lr * (m2 / (np.sqrt(v2) + eps) + wd * theta), m2, v2

    def coupled_decay(theta, m, v, g, lr, b1, b2, eps, wd, t):
        return O.adamw_step(theta, m, v, g + wd * theta, lr, b1, b2, eps, 0.0, t)

    def eps_inside_sqrt(theta, m, v, g, lr, b1, b2, eps, wd, t):
        m2 = b1 * m + (1 - b1) * g
        v2 = b2 * v + (1 - b2) * g * g
        mh, vh = m2 / (1 - b1 ** t), v2 / (1 - b2 ** t)
        return theta - lr * (mh / np.sqrt(vh + eps) + wd * theta), m2, v2

    assert check_adamw_golden(O.adamw_step)
    assert not check_adamw_golden(no_bias_correction)
    assert not check_adamw_golden(coupled_decay)
    assert not check_adamw_golden(eps_inside_sqrt)


# ---------------------------------------------------------------------------
# 2-D convolutions (CIFAR-10 WideResNet of App. B)
# ---------------------------------------------------------------------------

CONV_GEOMS = [
    # (B, H, W, C_in, C_out, kh, kw, stride, pad)
    (2, 5, 6, 3, 4, 3, 3, (1, 1), (1, 1)),
    (2, 7, 5, 2, 3, 3, 3, (2, 2), (1, 1)),
    (1, 6, 6, 4, 2, 1, 1, (2, 2), (0, 0)),
    (2, 4, 5, 2, 3, 2, 3, (1, 2), (0, 1)),
]


def _conv_inputs(geom, seed=0):
    B, H, W_, Cin, Cout, kh, kw, st, pd = geom
    Ho, Wo = O.conv2d_out_hw(H, W_, kh, kw, st, pd)
    r = np.random.default_rng(seed)
    return r.standard_normal((B, H, W_, Cin)), r.standard_normal((B, Ho, Wo, Cout))


def brute_force_conv_grads(X, Dy, kh, kw, stride, pad):
    """Pure-Python loops over examples, taps, channels and output positions,
    reading padded positions as zero."""
    B, H, W_, Cin = X.shape
    _, Ho, Wo, Cout = Dy.shape
    Xl, Dl = X.tolist(), Dy.tolist()
    G = [[[[[0.0] * Cout for _ in range(Cin)] for _ in range(kw)] for _ in range(kh)]
         for _ in range(B)]
    for i in range(B):
        for ki in range(kh):
            for kj in range(kw):
                for h in range(Ho):
                    for w in range(Wo):
                        y = h * stride[0] + ki - pad[0]
                        x = w * stride[1] + kj - pad[1]
                        if not (0 <= y < H and 0 <= x < W_):
                            continue
                        for c in range(Cin):
                            a = Xl[i][y][x][c]
                            for o in range(Cout):
                                G[i][ki][kj][c][o] += a * Dl[i][h][w][o]
    return np.array(G)


def check_conv_grads(fn):
    """fn(X, Dy, kh, kw, stride, pad) against brute force and PyTorch's own
    weight-gradient routine, one example at a time."""
    import torch
    for g in CONV_GEOMS:
        B, H, W_, Cin, Cout, kh, kw, st, pd = g
        X, Dy = _conv_inputs(g, seed=B + H)
        G = fn(X, Dy, kh, kw, st, pd)
        if G.shape != (B, kh, kw, Cin, Cout):
            return False
        if not np.allclose(G, brute_force_conv_grads(X, Dy, kh, kw, st, pd), rtol=1e-12, atol=1e-12):
            return False
        for i in range(B):
            x = torch.from_numpy(X[i:i + 1]).permute(0, 3, 1, 2)
            dy = torch.from_numpy(Dy[i:i + 1]).permute(0, 3, 1, 2)
            gw = torch.nn.grad.conv2d_weight(x, (Cout, Cin, kh, kw), dy, stride=st, padding=pd)
            if not np.allclose(G[i], gw.permute(2, 3, 1, 0).numpy(), rtol=1e-10, atol=1e-10):
                return False
    return True


def check_unfold(fn):
    """fn(X, kh, kw, stride, pad) against torch.nn.functional.unfold (columns
    (c, ki, kj), permuted to (ki, kj, c)) and hand-placed values."""
    import torch
    for g in CONV_GEOMS:
        B, H, W_, Cin, Cout, kh, kw, st, pd = g
        X, _ = _conv_inputs(g, seed=3)
        A = fn(X, kh, kw, st, pd)
        Ho, Wo = O.conv2d_out_hw(H, W_, kh, kw, st, pd)
        u = torch.nn.functional.unfold(torch.from_numpy(X).permute(0, 3, 1, 2), (kh, kw),
                                       padding=pd, stride=st)          # [B, C*kh*kw, L]
        u = u.reshape(B, Cin, kh, kw, Ho * Wo).permute(0, 4, 2, 3, 1).reshape(B, Ho * Wo, -1)
        if A.shape != u.shape or not np.array_equal(A, u.numpy()):
            return False
    # hand-placed: X[0, y, x, c] = 100 y + 10 x + c on a 3x3x2 image, 3x3
    # kernel, pad 1: output position (0, 0) reads rows -1..1 and columns -1..1
    X = np.array([[[[100 * y + 10 * x + c for c in range(2)] for x in range(3)] for y in range(3)]],
                 dtype=np.float64)
    A = fn(X, 3, 3, (1, 1), (1, 1))
    row = A[0, 0].reshape(3, 3, 2)
    want = np.zeros((3, 3, 2))
    for ki in range(3):
        for kj in range(3):
            y, x = ki - 1, kj - 1
            if 0 <= y < 3 and 0 <= x < 3:
                want[ki, kj] = [100 * y + 10 * x, 100 * y + 10 * x + 1]
    return bool(np.array_equal(row, want) and A[0, 4].reshape(3, 3, 2)[1, 1, 1] == 111)


def test_conv2d_weight_grads_pins():
    assert check_conv_grads(O.conv2d_weight_grads)


def test_conv2d_unfold_pins():
    assert check_unfold(O.conv2d_unfold)


def test_unfold_product_is_the_conv_gradient():
    for g in CONV_GEOMS:
        B, H, W_, Cin, Cout, kh, kw, st, pd = g
        X, Dy = _conv_inputs(g, seed=7)
        A = O.conv2d_unfold(X, kh, kw, st, pd)
        G = O.per_example_grads(A, Dy.reshape(B, -1, Cout))
        np.testing.assert_allclose(G.reshape(B, kh, kw, Cin, Cout),
                                   O.conv2d_weight_grads(X, Dy, kh, kw, st, pd), rtol=0, atol=1e-12)


def test_1x1_conv_is_the_dense_layer_on_pixels():
    r = np.random.default_rng(11)
    X, Dy = r.standard_normal((3, 4, 5, 6)), r.standard_normal((3, 4, 5, 7))
    G = O.conv2d_weight_grads(X, Dy, 1, 1)
    np.testing.assert_allclose(G[:, 0, 0], O.per_example_grads(X.reshape(3, 20, 6), Dy.reshape(3, 20, 7)),
                               rtol=0, atol=1e-12)


def test_step_from_grads_equals_dense_step():
    r = np.random.default_rng(12)
    layers = [(r.standard_normal((5, 4, 6)), r.standard_normal((5, 4, 3))),
              (r.standard_normal((5, 4, 3)), 0.1 * r.standard_normal((5, 4, 2)))]
    a = O.dp_step(layers, 0.7, 1.3, seed=5, step=2, out_scale=0.2)
    b = O.dp_step_from_grads([O.per_example_grads(A, D) for A, D in layers], 0.7, 1.3, seed=5,
                             step=2, out_scale=0.2)
    for k in ("n", "s", "c"):
        np.testing.assert_allclose(a[k], b[k], rtol=1e-13, atol=0)
    for x, y in zip(a["out"], b["out"]):
        np.testing.assert_allclose(x, y, rtol=1e-12, atol=1e-15)


def test_planted_conv_mistakes_are_caught():
    # a true convolution (kernel flipped) instead of the cross-correlation
    def flipped(X, Dy, kh, kw, st, pd):
        return O.conv2d_weight_grads(X, Dy, kh, kw, st, pd)[:, ::-1, ::-1]
    assert not check_conv_grads(flipped)

    # stride ignored in the input taps
    def no_stride(X, Dy, kh, kw, st, pd):
        Xp = np.pad(X, ((0, 0), (pd[0], pd[0]), (pd[1], pd[1]), (0, 0)))
        Ho, Wo = Dy.shape[1:3]
        G = np.zeros((X.shape[0], kh, kw, X.shape[3], Dy.shape[3]))
        for ki in range(kh):
            for kj in range(kw):
                G[:, ki, kj] = np.einsum("bhwc,bhwo->bco", Xp[:, ki:ki + Ho, kj:kj + Wo], Dy)
        return G
    assert not check_conv_grads(no_stride)

    # padding applied on one side only
    def one_side(X, Dy, kh, kw, st, pd):
        Xs = np.pad(X, ((0, 0), (2 * pd[0], 0), (2 * pd[1], 0), (0, 0)))
        return O.conv2d_weight_grads(Xs, Dy, kh, kw, st, (0, 0))
    assert not check_conv_grads(one_side)

    # unfold columns in (c, ki, kj) order
    def unfold_c_major(X, kh, kw, st, pd):
        A = O.conv2d_unfold(X, kh, kw, st, pd)
        B, T, K = A.shape
        return A.reshape(B, T, kh, kw, -1).transpose(0, 1, 4, 2, 3).reshape(B, T, K)
    assert not check_unfold(unfold_c_major)
