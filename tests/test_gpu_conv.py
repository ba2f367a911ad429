"""GPU parity of convolution layers (the CIFAR-10 WideResNet of App. B).

A convolution enters the step as a dense layer whose A is its patch rows,
written by the library's dp_conv2d_unfold.  The unfold is copy work and must
match the oracle's bit for bit; the step's norms, clip factors and outputs
are compared with the oracle's per-example gradients taken from the
definition of the convolution (not through patch rows), within the bf16 /
fp32 tolerances of the dense tests.
"""

import numpy as np
import pytest
import torch

import paper_2609_20532_gb300 as dp
import workloads as W
from oracle import dp_oracle as O

from gpu_harness import (TOL, assert_step_matches, f32, oracle_grads, rel_err_elementwise,
                         rel_err_normwise, run_gpu_step)

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.fail("CUDA GPU required for -m gpu tests")
    dp.lib()


UNFOLD_CASES = [
    # (B, H, W, C_in, kh, kw, stride, pad, dtype)
    (2, 5, 6, 3, 3, 3, (2, 2), (1, 1), "bf16"),      # C_in = 3: element path
    (3, 8, 8, 16, 3, 3, (1, 1), (1, 1), "bf16"),     # 16-byte channel vectors
    (2, 9, 7, 8, 2, 3, (1, 2), (0, 1), "bf16"),      # asymmetric kernel, stride, padding
    (2, 8, 8, 64, 1, 1, (2, 2), (0, 0), "bf16"),     # 1x1 shortcut, stride 2
    (2, 6, 6, 4, 3, 3, (1, 1), (2, 2), "f32"),       # fp32 vectors, padding wider than 1
    (2, 5, 5, 3, 3, 3, (1, 1), (1, 1), "f32"),       # fp32 element path
    (2, 8, 8, 256, 3, 3, (1, 1), (1, 1), "bf16"),    # K = 2304 (a WideResNet group-3 row)
    (1, 3, 3, 8, 3, 3, (1, 1), (0, 0), "bf16"),      # one output position
]


@pytest.mark.parametrize("case", range(len(UNFOLD_CASES)))
def test_unfold_bit_exact(case):
    B, H, W_, C, kh, kw, st, pd, dtype = UNFOLD_CASES[case]
    rng = np.random.default_rng(40 + case)
    x = torch.from_numpy(rng.standard_normal((B, H, W_, C), dtype=np.float32))
    if dtype == "bf16":
        x = x.to(torch.bfloat16)
    conv = dp.make_conv(H, W_, C, kh, kw, st, pd)
    T, K = dp.dp_conv2d_dims(conv)
    Ho, Wo = O.conv2d_out_hw(H, W_, kh, kw, st, pd)
    assert (T, K) == (Ho * Wo, kh * kw * C)
    a = torch.full((B, T, K), float("nan"), dtype=x.dtype, device=DEV)
    dp.dp_conv2d_unfold(conv, B, dtype, x.to(DEV), a)
    torch.cuda.synchronize()
    ref = O.conv2d_unfold(x.to(torch.float64).numpy(), kh, kw, st, pd)
    assert np.array_equal(a.cpu().to(torch.float64).numpy(), ref)


def test_unfold_argument_errors():
    conv = dp.make_conv(8, 8, 16, 3, 3, (1, 1), (1, 1))
    x = torch.zeros((2, 8, 8, 16), dtype=torch.bfloat16, device=DEV)
    a = torch.zeros((2, 64, 144), dtype=torch.bfloat16, device=DEV)
    n0 = dp.dp_kernel_launches()
    for bad, status in ((dict(B=0), 1), (dict(x=x.view(-1)[1:]), 1), (dict(a_out=x), 1),
                        (dict(conv=dp.make_conv(2, 2, 16, 5, 5)), 2),
                        (dict(conv=dp.make_conv(8, 8, 16, 3, 3, (0, 1))), 2)):
        kw = dict(conv=conv, B=2, dtype="bf16", x=x, a_out=a)
        kw.update(bad)
        with pytest.raises(dp.DPError) as ei:
            dp.dp_conv2d_unfold(kw["conv"], kw["B"], kw["dtype"], kw["x"], kw["a_out"])
        assert ei.value.status == status, bad
    assert dp.dp_kernel_launches() == n0   # refused on the host, nothing launched


def oracle_conv_step(w, layers, seed=0, step=0, out_scale=1.0, noise=True):
    return O.dp_step_from_grads(oracle_grads(w, layers), f32(w.C), f32(w.sigma), seed, step,
                                out_scale=f32(out_scale), noise=noise)


CONV_NETS = [
    # (convs (H, W, C_in, C_out, kh, kw, stride, pad), head (d_in, d_out, T), B, dtype)
    ([(16, 16, 3, 16, 3, 3, 1, 1),      # K = 27: thin, multiply-add kernel
      (16, 16, 16, 64, 3, 3, 1, 1),     # K = 144, T = 256: materialised norm, split GEMM
      (16, 16, 64, 64, 3, 3, 2, 1),     # K = 576, T = 64: Gram norm, split GEMM
      (16, 16, 16, 64, 1, 1, 2, 0)],    # 1x1 shortcut: thin, warp MMAs
     [(64, 10, 1), (1, 10, 1)], 8, "bf16"),
    ([(6, 6, 4, 8, 3, 3, 1, 1), (6, 6, 8, 8, 3, 3, 2, 1)], [(8, 3, 1)], 5, "f32"),
    # channels in multiples of 64: patch rows read in place by the tensor-core
    # kernels (W_out = 16, 8 and 128), a 1x1 identity, strided convolutions
    # (four parity maps of the input)
    ([(16, 16, 64, 64, 3, 3, 1, 1),       # T = 256, W_out = 16
      (8, 8, 128, 128, 3, 3, 1, 1),       # T = 64, W_out = 8
      (4, 128, 64, 64, 3, 3, 1, 1),       # W_out = 128: boxes are half rows
      (16, 16, 64, 128, 1, 1, 1, 0),      # 1x1 stride 1: the input is the patch rows
      (16, 16, 64, 128, 3, 3, 2, 1)],     # stride 2
     [], 6, "bf16"),
    # stride 2 read in place: odd input sizes (parity maps of unequal size),
    # no padding, a 5x5 kernel (tap offsets -2 .. 2), a 4x4 kernel (offsets
    # -1 .. 2: parities 1, 0, 1, 0), all with 8 x 8 outputs
    ([(15, 15, 64, 64, 3, 3, 2, 1),
      (17, 17, 64, 128, 3, 3, 2, 0),
      (16, 16, 128, 64, 5, 5, 2, 2),
      (16, 16, 64, 64, 4, 4, 2, 1)],
     [], 5, "bf16"),
]


@pytest.mark.parametrize("conv_mode", ["explicit", "library"])
@pytest.mark.parametrize("case", range(len(CONV_NETS)))
def test_conv_net_step_matches_oracle(case, conv_mode):
    convs, head, B, dtype = CONV_NETS[case]
    dists = ("normal",) + ("relu_normal",) * (len(convs) - 1) + ("normal",) * len(head)
    if head and head[-1][0] == 1:
        dists = dists[:-1] + ("ones",)
    w = W.custom_conv(f"convnet{case}", convs, B, dtype, C=0.5, sigma=0.8, d_std=0.05,
                      wid=950 + case, a_dist=dists, head=head)
    layers = W.make_inputs(w)
    res = run_gpu_step(w, layers, seed=3, step=11, out_scale=1.0 / B, conv_mode=conv_mode)
    ref = oracle_conv_step(w, layers, seed=3, step=11, out_scale=1.0 / B)
    ref["out"] = [o.reshape(i, d) for o, (i, d) in zip(ref["out"], w.layers)]
    assert_step_matches(res, ref, dtype)


@pytest.mark.parametrize("conv,launches", [
    ((16, 16, 64, 64, 3, 3, 1, 1), 1),    # read in place: the norm kernel alone
    ((16, 16, 64, 128, 3, 3, 2, 1), 1),   # stride 2, read in place through parity maps
    ((15, 15, 64, 64, 3, 3, 2, 1), 1),    # the same with odd input sizes
    ((16, 16, 64, 128, 3, 3, 3, 1), 2),   # stride 3: unfold into scratch, then the norm
    ((16, 16, 64, 128, 1, 1, 1, 0), 1),   # 1x1 identity: the input is the patch rows
    ((16, 16, 3, 16, 3, 3, 1, 1), 1),     # thin, 3 channels: gradients straight from the input
    ((20, 21, 5, 12, 3, 2, 1, 1), 1),     # thin, 3x2 kernel, odd sizes
    ((16, 16, 3, 16, 3, 3, 2, 1), 1),     # thin, stride 2
])
def test_library_conv_paths_and_launches(conv, launches):
    """A DP_LAYER_CONV2D layer: how many kernels its norm call issues shows
    whether its patch rows are read in place, and its outputs match the
    caller-unfolded dense layer within the bf16 tolerance."""
    w = W.custom_conv("libconv", [conv], 4, "bf16", C=0.5, sigma=0.5, d_std=0.05, wid=970,
                      a_dist=("relu_normal",))
    layers = W.make_inputs(w)
    H, W_, cin, cout, kh, kw, st, pd = conv
    cv = dp.make_conv(H, W_, cin, kh, kw, (st, st), (pd, pd))
    cfg = dp.make_config(w.specs, w.B, w.T, "bf16", w.C, w.sigma, audit_capacity=w.B, convs=[cv])
    ctx = dp.dp_step_init(cfg)
    try:
        x, d = layers[0][0].to(DEV), layers[0][1].to(DEV)
        n0 = dp.dp_kernel_launches()
        dp.dp_layer_norms(ctx, 0, x, d)
        assert dp.dp_kernel_launches() - n0 == launches
        dp.dp_clip_factors(ctx)
        out = torch.zeros(w.layers[0], device=DEV)
        dp.dp_clipped_sum_noise(ctx, 0, x, d, out, dp.DP_NO_NOISE)
        recs = dp.dp_audit_emit(ctx, range(w.B), 1)
    finally:
        dp.dp_step_destroy(ctx)
    ref = oracle_conv_step(w, layers, noise=False)
    assert rel_err_elementwise(recs["layer_sqnorm"].astype(np.float64).T, ref["n"]) <= TOL["bf16"]
    assert rel_err_normwise(out.cpu().numpy(), ref["out"][0].reshape(w.layers[0])) <= TOL["bf16"]


def test_wrn16_4_full_size_sampled():
    """WideResNet-16-4 at B = 2048, the bench's configuration.  The oracle
    recomputes every layer's per-example norm, s_i and c_i for sampled
    examples; with C so large that nothing is clipped (c_i = 1), sampled
    weights of every layer's noiseless sum are the oracle's sums over all
    2048 examples, one kernel tap and channel pair at a time."""
    w = W.get("wrn16_4_cifar10_bf16")
    layers = W.make_inputs(w)
    tol = TOL[w.dtype]
    res = run_gpu_step(w, layers, seed=1, step=5, out_scale=1.0 / w.B, conv_mode="library")
    rng = np.random.default_rng(77)
    ex = np.sort(rng.choice(w.B, size=3, replace=False))
    sub = [(A[ex], D[ex]) for A, D in layers]
    wsub = W.Workload(w.name, w.wid, w.layers, len(ex), w.T, w.dtype, w.a_dist, w.a_std,
                      w.d_std, w.C, w.sigma, layer_T=w.layer_T, convs=w.convs)
    G = oracle_grads(wsub, sub)
    n_ref = np.stack([np.sum(g.reshape(len(ex), -1) ** 2, axis=1) for g in G])
    s_ref, c_ref = O.clip_factors(n_ref, f32(w.C))
    assert rel_err_elementwise(res["n"][:, ex], n_ref) <= tol
    assert rel_err_elementwise(res["s"][ex], s_ref) <= tol
    assert rel_err_elementwise(res["c"][ex], c_ref) <= tol
    assert np.all(res["c"] <= 1.0) and np.all(res["c"] > 0.0)
    # nothing clipped: the commitment is the plain sum over the batch
    wbig = W.Workload(w.name, w.wid, w.layers, w.B, w.T, w.dtype, w.a_dist, w.a_std, w.d_std,
                      1e30, w.sigma, layer_T=w.layer_T, convs=w.convs)
    big = run_gpu_step(wbig, layers, flags=dp.DP_NO_NOISE, audit=False, conv_mode="library")
    assert np.all(big["c"] == 1.0)
    for l, (A, D) in enumerate(layers):
        d_in, d_out = w.layers[l]
        out = big["out"][l]
        picks = [(int(rng.integers(d_in)), int(rng.integers(d_out))) for _ in range(4)]
        cv = w.conv_of(l)
        for k, o in picks:
            if cv:
                H, W_, cin, kh, kw, st, pd = cv
                tap, c = divmod(k, cin)
                ki, kj = divmod(tap, kw)
                Ho, Wo = O.conv2d_out_hw(H, W_, kh, kw, (st, st), (pd, pd))
                x = W.to_f64(A[..., c:c + 1])
                dy = W.to_f64(D[..., o:o + 1]).reshape(w.B, Ho, Wo, 1)
                ref = O.conv2d_weight_grads(x, dy, kh, kw, (st, st), (pd, pd))[:, ki, kj, 0, 0].sum()
            else:
                ref = float(np.sum(W.to_f64(A[..., k]) * W.to_f64(D[..., o])))
            scale = max(np.max(np.abs(out)), 1e-30)
            assert abs(out[k, o] - ref) <= tol * scale, (l, k, o, out[k, o], ref)
