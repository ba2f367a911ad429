"""The trusted-side verifier (Algorithm 1, Sec. 6.2) on the CPU: its frozen
parameters against the paper's table, its fp64 recomputation against the
oracle, every path of the algorithm with constructed submissions, and the
audit-record check."""

import json
import math
import os

import numpy as np
import pytest

import workloads as W
from oracle import dp_oracle as O
from paper_2609_20532_gb300 import verifier as V

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "verifier_params.json")))


def test_frozen_parameters_match_the_paper_table():
    for fam, g in GOLD.items():
        if fam == "citation":
            continue
        p = V.FAMILIES[fam]
        assert (p.p, p.tau_abs, p.K_sub, p.K_amb, p.slack) == (g["p"], g["tau_abs"], g["K_sub"],
                                                                  g["K_amb"], g["slack"])
        if "tau_num" in g:
            assert p.fp64_layer and p.tau_num == g["tau_num"]
        else:
            assert not p.fp64_layer and p.rho_ill == g["rho"]


def test_table_internal_relations():
    """rho_amb = 2 tau_num / B reproduces the table's rho column (RoBERTa at
    its calibration batch 256, GPT-2 at B = 64 and B = 32), and CIFAR-10's
    rho_ill is 2 tau_abs, all to the table's printed digits."""
    r = V.FAMILIES["roberta"]
    assert r.rho_amb(256) == pytest.approx(GOLD["roberta"]["rho"], abs=5e-6)
    g = V.FAMILIES["gpt2"]
    assert g.rho_amb(64) == pytest.approx(GOLD["gpt2"]["rho"], abs=5e-7)
    assert 2 * GOLD["gpt2"]["tau_num_B32"] / 32 == pytest.approx(GOLD["gpt2"]["rho"], abs=5e-6)
    c = V.FAMILIES["cifar10"]
    assert 2 * c.tau_abs == pytest.approx(c.rho_ill, abs=5e-6)


def _layers(name, seed=0):
    w = W.get(name)
    return w, W.make_inputs(w, seed=seed)


@pytest.mark.parametrize("name", ["single_fp32", "mlp_fp32"])
def test_fp64_recomputation_equals_the_oracle(name):
    w, layers = _layers(name)
    C = float(np.float32(w.C))
    got, s, c = V.recompute_average(layers, C, np.float64)
    ref = O.dp_step([(W.to_f64(A), W.to_f64(D)) for A, D in layers], C, 0.0, 0, 0,
                    out_scale=1.0 / w.B, noise=False)
    assert np.allclose(s, ref["s"], rtol=1e-12, atol=0)
    assert np.allclose(c, ref["c"], rtol=1e-12, atol=0)
    for a, b in zip(got, ref["out"]):
        assert np.linalg.norm(a - b) <= 1e-12 * np.linalg.norm(b)


def test_fp64_recomputation_equals_the_oracle_bf16_block():
    w = W.custom("vblock", [(96, 40), (40, 72)], 4, 24, "bf16", C=0.05, sigma=1.0, d_std=0.2,
                 wid=701)
    layers = W.make_inputs(w)
    got, s, c = V.recompute_average(layers, w.C, np.float64)
    ref = O.dp_step([(W.to_f64(A), W.to_f64(D)) for A, D in layers], w.C, 0.0, 0, 0,
                    out_scale=1.0 / w.B, noise=False)
    assert np.allclose(s, ref["s"], rtol=1e-12, atol=0)
    assert np.any(c < 1) and np.allclose(c, ref["c"], rtol=1e-12, atol=0)
    for a, b in zip(got, ref["out"]):
        assert np.linalg.norm(a - b) <= 1e-12 * np.linalg.norm(b)


def _honest(name="mlp_fp32"):
    w, layers = _layers(name)
    C = float(np.float32(w.C))
    g64, _, _ = V.recompute_average(layers, C, np.float64)
    g32, _, _ = V.recompute_average(layers, C, np.float32)
    return w, layers, C, g64, g32


def _unit(shape_list, seed):
    rng = np.random.default_rng(seed)
    v = np.concatenate([rng.standard_normal(int(np.prod(s))) for s in shape_list])
    return v / np.linalg.norm(v)


def test_body_path_accepts_and_charges_the_ledger():
    w, layers, C, g64, g32 = _honest()
    ver = V.Verifier(V.FAMILIES["roberta"], C, w.B, coin_seed=1)
    sub = np.concatenate([x.reshape(-1) for x in g64]).astype(np.float32)
    r = ver.step(sub, lambda: g32, lambda: g64, checked=True)
    assert r.verdict == V.ACCEPT and r.path == "body"
    assert r.z32 <= 1e-5 and ver.Z_sub == pytest.approx(r.z32)


def test_structural_bound():
    C = 0.5
    ver = V.Verifier(V.FAMILIES["roberta"], C, 16, coin_seed=0)
    d = np.zeros(1000)
    d[3] = C * (1 + 2e-4)
    assert ver.step(d, None, checked=True).path == "structural"
    d[3] = C * (1 + 0.5e-4)
    boom = lambda: (_ for _ in ()).throw(AssertionError("an unchecked step recomputes nothing"))
    assert ver.step(d, boom, checked=False).verdict == V.ACCEPT
    d[5] = np.nan
    assert ver.step(d, None, checked=True).path == "structural"


def test_ledger_exhaustion_under_tau_abs():
    """Deviations of 0.9 tau_abs on every checked step pass the body path
    until their sum exceeds K_sub (Sec. 6.2: no accepted deviation is free)."""
    w, layers, C, g64, g32 = _honest()
    prm = V.FAMILIES["roberta"]
    ver = V.Verifier(prm, C, w.B, coin_seed=0)
    base = np.concatenate([x.reshape(-1) for x in g32]).astype(np.float64)
    u = _unit([x.shape for x in g32], 3)
    dev = base + 0.9 * prm.tau_abs * C * u
    n_ok = 0
    while True:
        r = ver.step(dev, lambda: g32, checked=True)
        if r.verdict == V.ABORT:
            break
        assert r.path == "body"
        n_ok += 1
    assert r.path == "ledger"
    assert n_ok == math.floor(prm.K_sub / (0.9 * prm.tau_abs))


def test_ambiguity_counter_and_hard_rejection():
    w, layers, C, g64, g32 = _honest()
    prm = V.FAMILIES["roberta"]
    u = _unit([x.shape for x in g64], 4)
    base = np.concatenate([x.reshape(-1) for x in g64])
    rho = prm.rho_amb(w.B)
    assert 2 * prm.tau_abs < rho
    ver = V.Verifier(prm, C, w.B, coin_seed=0)
    amb = base + 2 * prm.tau_abs * C * u           # escalates, within rho_amb
    for k in range(prm.K_amb):
        r = ver.step(amb, lambda: g32, lambda: g64, checked=True)
        assert r.verdict == V.ACCEPT and r.path == "ambiguity" and ver.S_amb == k + 1
        assert r.n_t == pytest.approx(w.B / 2 * 2 * prm.tau_abs, rel=1e-3)
    r = ver.step(amb, lambda: g32, lambda: g64, checked=True)
    assert r.verdict == V.ABORT and r.path == "ledger"
    ver2 = V.Verifier(prm, C, w.B, coin_seed=0)
    bad = base + 2 * rho * C * u
    r = ver2.step(bad, lambda: g32, lambda: g64, checked=True)
    assert r.verdict == V.ABORT and r.path == "hard_reject" and r.n_t > prm.tau_num


def test_cifar_variant_caps_without_fp64():
    w, layers, C, g64, g32 = _honest()
    prm = V.FAMILIES["cifar10"]
    u = _unit([x.shape for x in g32], 5)
    base = np.concatenate([x.reshape(-1) for x in g32]).astype(np.float64)
    ver = V.Verifier(prm, C, w.B, coin_seed=0)
    r = ver.step(base + 1.5 * prm.tau_abs * C * u, lambda: g32, checked=True)
    assert r.verdict == V.ACCEPT and r.path == "ambiguity" and r.z64 is None
    r = ver.step(base + 3 * prm.tau_abs * C * u, lambda: g32, checked=True)
    assert r.verdict == V.ABORT and r.path == "hard_reject"


def test_secret_coins():
    prm = V.FAMILIES["gpt2"]
    C = 1.0
    d = np.zeros(10)
    a = V.Verifier(prm, C, 64, coin_seed=11)
    b = V.Verifier(prm, C, 64, coin_seed=11)
    ca = [a.draw_coin() for _ in range(20000)]
    assert ca == [b.draw_coin() for _ in range(20000)]
    k = sum(ca)
    # binomial(20000, 0.1): mean 2000, sd 42.4; 5 sd
    assert abs(k - 2000) < 5 * math.sqrt(20000 * 0.1 * 0.9)


def _records_from_oracle(layers, C, idx):
    n = np.stack([O.layer_sqnorms_materialised(W.to_f64(A), W.to_f64(D)) for A, D in layers])
    s, c = O.clip_factors(n, C)
    rec = np.zeros(len(idx), dtype=[("example", "<i4"), ("total_sqnorm", "<f4"),
                                    ("clip_factor", "<f4"), ("layer_sqnorm", "<f4", (len(layers),))])
    rec["example"] = idx
    rec["total_sqnorm"] = s[idx]
    rec["clip_factor"] = c[idx]
    rec["layer_sqnorm"] = n[:, idx].T
    return rec


def test_audit_records_check():
    w, layers = _layers("mlp_fp32")
    C = float(np.float32(w.C))
    idx = [0, 17, 255]
    rec = _records_from_oracle(layers, C, idx)
    rep = V.check_audit_records(rec, layers, C, rtol=1e-6)
    assert rep.ok and rep.examples == idx
    bad = rec.copy()
    bad["layer_sqnorm"][1, 2] *= 1.01
    assert not V.check_audit_records(bad, layers, C, rtol=1e-5).ok
    bad = rec.copy()
    bad["clip_factor"][0] = min(1.0, bad["clip_factor"][0] * 1.01)
    bad["clip_factor"][1] = bad["clip_factor"][1] * 1.01
    assert not V.check_audit_records(bad, layers, C, rtol=1e-5).ok
    assert V.check_audit_records(rec[:0], layers, C, rtol=1e-6).ok
