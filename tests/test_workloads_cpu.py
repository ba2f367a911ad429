"""The synthetic inputs follow their stated recipe (CPU only).

Every workload draws A and D from numpy generators seeded by
SeedSequence([seed, workload id, layer, kind]) with the distribution, scale
and dtype of its description; these tests pin the recipe of the named
workloads (shapes, B, T, C, sigma, distributions and scales), the
distributions' observable properties on samples, the seeding, and the audit
subset size.
"""
import math

import numpy as np
import pytest
import torch

import workloads as W


@pytest.mark.parametrize("name,layers,B,T,dtype,C,sigma,a_dist,d_var", [
    ("single_fp32", [(64, 32)], 8, 1, "f32", 1.0, 1.0, ("normal",), 1.0),
    ("mlp_fp32", [(784, 512), (512, 512), (512, 10)], 256, 1, "f32", 1.0, 1.1,
     ("uniform", "relu_normal", "relu_normal"), 0.01),
    ("block_bf16", [(768, 2304), (768, 768), (768, 3072), (3072, 768)], 32, 128, "bf16",
     1.0, 0.8, ("normal",) * 4, 1e-4),
    ("llm_bf16", [(4096, 11008), (11008, 4096), (4096, 12288)], 16, 512, "bf16", 0.5, 1.0,
     ("normal",) * 3, 1e-5),
])
def test_named_workload_recipe(name, layers, B, T, dtype, C, sigma, a_dist, d_var):
    w = W.get(name)
    assert [tuple(x) for x in w.layers] == layers
    assert (w.B, w.T, w.dtype, w.C, w.sigma) == (B, T, dtype, C, sigma)
    assert tuple(w.a_dist) == a_dist and w.a_std == 1.0
    assert w.d_std == pytest.approx(math.sqrt(d_var), rel=1e-12)   # "N(0, v)" is a variance


def test_sweep_points():
    pts = sorted((w.B, w.T) for w in W.SWEEP)
    assert pts == sorted((b, t) for b in (8, 32, 128) for t in (1, 64, 512, 2048))
    assert all([tuple(x) for x in w.layers] == [(4096, 4096)] and w.dtype == "bf16"
               for w in W.SWEEP)


def test_distributions_on_samples():
    w = W.get("mlp_fp32")
    A0, D0 = W.make_layer(w, 0)
    A1, _ = W.make_layer(w, 1)
    a0 = A0.numpy().ravel()
    assert a0.dtype == np.float32 and a0.min() >= 0.0 and a0.max() < 1.0
    assert abs(a0.mean() - 0.5) < 0.01                        # U[0, 1)
    a1 = A1.numpy().ravel()
    assert a1.min() == 0.0 and abs((a1 == 0).mean() - 0.5) < 0.01   # ReLU of N(0, 1)
    assert abs(a1[a1 > 0].mean() - math.sqrt(2 / math.pi)) < 0.01    # half-normal mean
    d0 = D0.numpy().ravel()
    assert abs(d0.std() / 0.1 - 1) < 0.01 and abs(d0.mean()) < 0.005
    # bf16 workloads: stored as bf16, scales as stated
    w = W.get("llm_bf16")
    A, D = W.make_layer(w, 0, B=1)
    assert A.dtype == torch.bfloat16 and D.dtype == torch.bfloat16
    assert tuple(A.shape) == (1, 512, 4096) and tuple(D.shape) == (1, 512, 11008)
    a = A.double().numpy().ravel()
    d = D.double().numpy().ravel()
    assert abs(a.std() - 1) < 0.01 and abs(a.mean()) < 0.01
    assert abs(d.std() / math.sqrt(1e-5) - 1) < 0.01


def test_seeding_is_per_layer_and_kind():
    w = W.get("block_bf16")
    A1, D1 = W.make_layer(w, 1, seed=0)
    A1b, D1b = W.make_layer(w, 1, seed=0)
    assert torch.equal(A1, A1b) and torch.equal(D1, D1b)     # reproducible
    A1c, _ = W.make_layer(w, 1, seed=1)
    assert not torch.equal(A1, A1c)                           # the seed matters
    A0, D0 = W.make_layer(w, 0, seed=0)
    assert not torch.equal(A0[:, :, :768], A1[:, :, :768])    # layers draw independently
    assert not torch.equal(A1[0, :, :768].float(), D1[0, :, :768].float() / w.d_std)  # kinds


def test_convolution_and_bias_inputs():
    w = W.get("wrn16_4_cifar10_bf16")
    assert w.a_dist[0] == "normal" and w.a_dist[-1] == "ones"
    assert all(d == "relu_normal" for d in w.a_dist[1:-1])
    A, D = W.make_layer(w, 1, B=2)          # 3x3 conv 32x32x16 -> 64: NHWC input
    H, W_, cin = w.conv_of(1)[:3]
    assert tuple(A.shape) == (2, H, W_, cin) and tuple(D.shape) == (2, w.T_of(1), 64)
    Ab, _ = W.make_layer(w, len(w.layers) - 1, B=2)   # the classifier's bias row
    assert torch.all(Ab == 1)


def test_audit_subset_sizes():
    assert len(W.audit_indices(W.get("llm_bf16"))) == 1       # ceil(0.05 * 16)
    idx = W.audit_indices(W.get("wrn16_4_cifar10_bf16"))
    assert len(idx) == math.ceil(0.05 * 2048) == 103
    assert np.all(np.diff(idx) > 0) and idx.min() >= 0 and idx.max() < 2048
    np.testing.assert_array_equal(idx, W.audit_indices(W.get("wrn16_4_cifar10_bf16")))
