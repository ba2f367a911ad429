"""GPU parity: the CUDA path through the C ABI against the fp64 oracle.

Tolerances: Philox words bit-exact; Gaussian numbers within 1e-6 relative
elementwise; per-example norms, s_i and c_i within 2e-3 (bf16 inputs) or
1e-5 (fp32 inputs) relative elementwise; clipped sums and noisy outputs
within the same bounds normwise per layer.
"""

import math
import time

import numpy as np
import pytest
import torch

import paper_2609_20532_gb300 as dp
import workloads as W
from oracle import dp_oracle as O

from gpu_harness import (TOL, assert_step_matches, f32, rel_err_elementwise, rel_err_normwise,
                         run_gpu_step)

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.fail("CUDA GPU required for -m gpu tests")
    dp.lib()  # fails loudly if the library was not built


def is_thin(d_in, d_out, T, dtype):
    """The library's rule for layers whose per-example gradients the norm pass
    stores (include/dp_step.h, dp_clipped_sum_noise)."""
    elem = 2 if dtype == "bf16" else 4
    return min(d_in, d_out) <= 32 and (T == 1 or 8 * d_in * d_out < T * (d_in + d_out) * elem)


def oracle_step(w, layers, seed=0, step=0, out_scale=1.0, noise=True, norm="materialised"):
    return O.dp_step([(W.to_f64(A), W.to_f64(D)) for A, D in layers], f32(w.C), f32(w.sigma),
                     seed, step, out_scale=f32(out_scale), noise=noise, norm=norm)


# ---------------------------------------------------------------------------
# generator
# ---------------------------------------------------------------------------

M64 = (1 << 64) - 1


@pytest.mark.parametrize("seed,step,q0,n", [
    (0, 0, 0, 1 << 22),
    (0x123456789ABCDEF0, 7, (1 << 32) - 1000, 1 << 16),     # crosses the 32-bit counter carry
    (M64, M64, M64 - 4095, 4096),                             # wraps the 64-bit quad counter
    (1, 1 << 32, 35_000_000, 1 << 16),
])
def test_philox_words_bit_exact(seed, step, q0, n):
    out = torch.empty(4 * n, dtype=torch.int32, device=DEV)
    dp.dp_debug_philox(seed, step, q0, n, out)
    got = out.cpu().numpy().view(np.uint32).reshape(n, 4)
    if q0 + n - 1 > M64:  # the oracle's quad range is defined modulo 2^64
        ref = np.concatenate([O.philox_quads(seed, step, q0, M64 - q0 + 1),
                              O.philox_quads(seed, step, 0, q0 + n - 1 - M64)])
    else:
        ref = O.philox_quads(seed, step, q0, n)
    assert np.array_equal(got, ref)


@pytest.mark.parametrize("seed,step,p0,n", [
    (0, 0, 0, 1 << 22), (5, 9, 3, 100_003), (M64, 2, (1 << 34) + 1, 1 << 16)])
def test_gaussian_within_1e6(seed, step, p0, n):
    out = torch.empty(n, dtype=torch.float32, device=DEV)
    dp.dp_debug_gaussian(seed, step, p0, n, out)
    got = out.cpu().numpy().astype(np.float64)
    ref = O.gaussian_noise(seed, step, p0, n)
    e = rel_err_elementwise(got, ref)
    assert e <= 1e-6, e


# ---------------------------------------------------------------------------
# whole-step parity on the workloads
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name", ["single_fp32", "mlp_fp32", "block_bf16"])
@pytest.mark.parametrize("out_scale", ["sum", "mean"])
def test_step_matches_oracle(name, out_scale):
    w = W.get(name)
    layers = W.make_inputs(w, seed=0)
    scale = 1.0 if out_scale == "sum" else 1.0 / w.B
    res = run_gpu_step(w, layers, seed=0, step=0, out_scale=scale)
    ref = oracle_step(w, layers, seed=0, step=0, out_scale=scale)
    assert_step_matches(res, ref, w.dtype)
    assert np.array_equal(res["rec_i"], np.arange(w.B))


@pytest.mark.parametrize("name", ["single_fp32", "mlp_fp32", "block_bf16"])
def test_commitment_is_noiseless_clipped_sum(name):
    """DP_NO_NOISE writes the commitment of Algorithm 2: S_l (times out_scale)."""
    w = W.get(name)
    layers = W.make_inputs(w, seed=0)
    res = run_gpu_step(w, layers, flags=dp.DP_NO_NOISE, audit=False)
    ref = oracle_step(w, layers, noise=False)
    for l, (o, r) in enumerate(zip(res["out"], ref["out"])):
        assert rel_err_normwise(o, r) <= TOL[w.dtype], l
    # the structural check of Sec. 6.2 on the averaged commitment
    agg = math.sqrt(sum(float(np.sum(o.astype(np.float64) ** 2)) for o in res["out"])) / w.B
    assert agg <= f32(w.C) * (1 + 1e-4)


def _llm_sample_check(w, layers, res, sample_rows=24, seed=0, step=0):
    """Full-size check at the LLM workload: every per-example norm from the
    oracle's Gram form (pinned equal to the materialised one), clip factors,
    and sampled rows of the clipped sum and of the noisy output."""
    L = len(w.layers)
    n_ref = np.stack([O.layer_sqnorms_ghost(W.to_f64(A), W.to_f64(D)) for A, D in layers])
    s_ref, c_ref = O.clip_factors(n_ref, f32(w.C))
    tol = TOL[w.dtype]
    assert rel_err_elementwise(res["n"], n_ref) <= tol
    assert rel_err_elementwise(res["c"], c_ref) <= tol
    rng = np.random.default_rng(123)
    off = 0
    for l, (A, D) in enumerate(layers):
        d_in, d_out = w.layers[l]
        rows = np.sort(rng.choice(d_in, size=sample_rows, replace=False))
        A64 = W.to_f64(A[:, :, rows])
        S_rows = O.clipped_sum(A64, W.to_f64(D), c_ref)          # = S_l[rows, :]
        z = np.stack([O.gaussian_noise(seed, step, off + int(j) * d_out, d_out) for j in rows])
        ref = S_rows + f32(w.sigma) * f32(w.C) * z
        got = res["out"][l][rows]
        assert rel_err_normwise(got, ref) <= tol, l
        off += d_in * d_out


def test_llm_workload_sampled():
    w = W.get("llm_bf16")
    layers = W.make_inputs(w, seed=0)
    res = run_gpu_step(w, layers)
    _llm_sample_check(w, layers, res)


def test_widest_layers_sampled():
    """Layers at the widest size the library accepts (2^20 on one side): two
    thin layers at T = 1 (per-example gradients stored) and a tensor-core
    layer at T = 64 whose output has 2^26 parameters.  Every norm and clip
    factor against the oracle, and sampled rows of every noisy output."""
    M = 1 << 20
    shapes = [(M, 8, 1), (8, M, 1), (64, M, 64)]
    w = W.custom("widest", shapes, 2, 64, "bf16", C=0.5, sigma=0.7, d_std=0.05, wid=640)
    layers = W.make_inputs(w, seed=0)
    res = run_gpu_step(w, layers, seed=6, step=2)
    # the cost model prefers the Gram form for the last layer, but its 2^20-long
    # feature reductions exceed the tensor cores' accumulation bound: the
    # materialised form on tensor cores (reductions of length T) serves it
    assert [p[0] for p in res["paths"]] == [2, 2, 1], res["paths"]
    assert res["modes"][2] == dp.DP_NORM_MATERIALISED
    n_ref = np.stack([O.layer_sqnorms_ghost(W.to_f64(A), W.to_f64(D)) for A, D in layers])
    s_ref, c_ref = O.clip_factors(n_ref, f32(w.C))
    assert rel_err_elementwise(res["n"], n_ref) <= TOL["bf16"]
    assert rel_err_elementwise(res["c"], c_ref) <= TOL["bf16"]
    rng = np.random.default_rng(7)
    off = 0
    for l, (A, D) in enumerate(layers):
        d_in, d_out = w.layers[l]
        rows = np.sort(rng.choice(d_in, size=min(6, d_in), replace=False))
        S_rows = O.clipped_sum(W.to_f64(A[:, :, rows]), W.to_f64(D), c_ref)
        z = np.stack([O.gaussian_noise(6, 2, off + int(j) * d_out, d_out) for j in rows])
        ref = S_rows + f32(w.sigma) * f32(w.C) * z
        assert rel_err_normwise(res["out"][l][rows], ref) <= TOL["bf16"], l
        off += d_in * d_out
    # the Gram form forced on the wide layer runs on CUDA cores, also in bound
    w1 = W.custom("widest_g", [(64, M)], 2, 64, "bf16", C=0.5, sigma=0.7, d_std=0.05, wid=641)
    l1 = W.make_inputs(w1, seed=0)
    g = run_gpu_step(w1, l1, norm_mode=dp.DP_NORM_GHOST, flags=dp.DP_NO_NOISE)
    assert g["paths"][0][0] == 0 and g["modes"][0] == dp.DP_NORM_GHOST
    n1 = O.layer_sqnorms_ghost(W.to_f64(l1[0][0]), W.to_f64(l1[0][1]))
    assert rel_err_elementwise(g["n"][0], n1) <= TOL["bf16"]


def test_long_reductions_leave_the_tensor_cores():
    """Paths whose tensor-core reduction would exceed 2^16 terms run on CUDA
    cores: T = 2^17 positions (an example's product), a 2^17-wide Gram side,
    and a pre-scaled T < 32 batch of more than 2^15 rows."""
    cases = [([(64, 64)], 1, 1 << 17, dp.DP_NORM_MATERIALISED, (0, 0)),
             ([(64, 1 << 17)], 2, 64, dp.DP_NORM_GHOST, (0, 1)),
             ([(64, 64)], 1 << 12, 16, dp.DP_NORM_MATERIALISED, (0, 0)),
             ([(64, 64)], 1 << 10, 16, dp.DP_NORM_MATERIALISED, (0, 1))]
    for shapes, B, T, mode, want in cases:
        cfg = dp.make_config(shapes, B, T, "bf16", 1.0, 1.0, norm_mode=mode)
        ctx = dp.dp_step_init(cfg)
        try:
            assert dp.dp_layer_path(ctx, 0) == want, (shapes, B, T)
        finally:
            dp.dp_step_destroy(ctx)


# ---------------------------------------------------------------------------
# norm modes, edge shapes and flags
# ---------------------------------------------------------------------------

EDGE = [
    # (layers, B, T, dtype)
    ([(8, 8)], 1, 1, "bf16"),
    ([(136, 72), (64, 200)], 3, 80, "bf16"),
    ([(24, 264)], 2, 129, "bf16"),
    ([(130, 70), (70, 3)], 5, 3, "f32"),
    ([(1, 1)], 1, 1, "f32"),
    ([(5, 7)], 4, 65, "f32"),
    ([(256, 128)], 2, 256, "bf16"),
    # FFMA clipped sum: 64-wide tiles walked by four K groups over 21 chunks
    # (the last one partial), ragged in both directions; and the 128-wide
    # tiles of a grid large enough for them (20 x 16 tiles)
    ([(200, 136)], 9, 37, "f32"),
    ([(2560, 2048)], 2, 3, "f32"),
]


@pytest.mark.parametrize("case", range(len(EDGE)))
@pytest.mark.parametrize("mode", [dp.DP_NORM_AUTO, dp.DP_NORM_GHOST, dp.DP_NORM_MATERIALISED])
def test_edge_shapes_and_norm_modes(case, mode):
    layers_shape, B, T, dtype = EDGE[case]
    w = W.custom(f"edge{case}", layers_shape, B, T, dtype, C=0.3, sigma=0.9, d_std=0.5,
                 wid=500 + case)
    layers = W.make_inputs(w, seed=1)
    res = run_gpu_step(w, layers, seed=11, step=3, norm_mode=mode)
    ref = oracle_step(w, layers, seed=11, step=3)
    assert_step_matches(res, ref, dtype)
    if mode != dp.DP_NORM_AUTO:
        assert all(m == mode for m in res["modes"])


def test_zero_example_keeps_clip_factor_one():
    w = W.custom("zero", [(64, 48)], 4, 16, "bf16", C=1e-3, sigma=0.0, wid=600)
    layers = W.make_inputs(w)
    A, D = layers[0]
    A = A.clone()
    A[2].zero_()
    layers = [(A, D)]
    res = run_gpu_step(w, layers)
    assert res["c"][2] == 1.0 and res["n"][0, 2] == 0.0
    ref = oracle_step(w, layers)
    assert_step_matches(res, ref, "bf16")


def test_nonfinite_input_is_reported():
    w = W.custom("nan", [(32, 16)], 3, 4, "f32", wid=601)
    layers = W.make_inputs(w)
    A, D = layers[0]
    A = A.clone()
    A[1, 2, 5] = float("nan")
    dev = torch.device(DEV)
    Ad, Dd = A.to(dev), D.to(dev)
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, audit_capacity=w.B)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.dp_layer_norms(ctx, 0, Ad, Dd)
        c = torch.empty(w.B, device=dev)
        dp.dp_clip_factors(ctx, None, c)
        with pytest.raises(dp.DPError) as ei:
            dp.dp_audit_emit(ctx, [0, 1], 1)
        assert ei.value.status == 5
        cc = c.cpu().numpy()
        assert np.isnan(cc[1]) and np.isfinite(cc[0]) and np.isfinite(cc[2])
        # a re-keyed step with clean inputs clears the flag
        dp.dp_step_init(cfg, ctx=ctx)
        A2 = layers[0][0].to(dev)
        dp.dp_layer_norms(ctx, 0, A2, Dd)
        dp.dp_clip_factors(ctx)
        dp.dp_audit_emit(ctx, [1], 1)
    finally:
        dp.dp_step_destroy(ctx)


def test_call_order_errors():
    w = W.custom("order", [(32, 16), (16, 8)], 2, 3, "f32", wid=602)
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    out = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, audit_capacity=1)
    ctx = dp.dp_step_init(cfg)
    try:
        def status(fn, *a):
            with pytest.raises(dp.DPError) as ei:
                fn(*a)
            return ei.value.status
        assert status(dp.dp_clipped_sum_noise, ctx, 0, Ad[0], Dd[0], out[0]) == 4
        assert status(dp.dp_audit_emit, ctx, [0], 2) == 4
        dp.dp_layer_norms(ctx, 0, Ad[0], Dd[0])
        assert status(dp.dp_clip_factors, ctx) == 4          # layer 1 missing
        dp.dp_layer_norms(ctx, 1, Ad[1], Dd[1])
        dp.dp_clip_factors(ctx)
        assert status(dp.dp_layer_norms, ctx, 0, Ad[0], Dd[0]) == 4
        assert status(dp.dp_clip_factors, ctx) == 4
        assert status(dp.dp_audit_emit, ctx, [0, 1], 2) == 1  # over capacity
        assert status(dp.dp_audit_emit, ctx, [5], 2) == 1     # index out of range
        assert status(dp.dp_layer_norms, ctx, 2, Ad[0], Dd[0]) == 1
        assert status(dp.dp_clipped_sum_noise, ctx, 0, Ad[0], Dd[0], out[0],
                      dp.DP_NO_NOISE | dp.DP_NOISE_ONLY) == 1
        misaligned = out[0].view(-1)[1:]
        assert status(dp.dp_clipped_sum_noise, ctx, 0, Ad[0], Dd[0], misaligned.data_ptr()) == 1
        dp.dp_clipped_sum_noise(ctx, 0, Ad[0], Dd[0], out[0])
        # re-key with other shapes is refused, the context stays usable
        bad = dp.make_config([(32, 16)], w.B, w.T, w.dtype, w.C, w.sigma)
        assert status(dp.dp_step_init, bad, None, ctx) == 2
        dp.dp_audit_emit(ctx, [1], 2)
    finally:
        dp.dp_step_destroy(ctx)


def test_bounded_wait_that_runs_out_is_reported_and_context_stays_usable():
    """The failure path of every pipeline wait: a device wait that nothing
    satisfies gives up after its limit (1 ms here), the call and the step's
    dp_audit_emit report DP_ERR_TIMEOUT, and after a re-key the same context
    runs a correct step (Algorithm 1's checker would reject the failed one)."""
    w = W.custom("timeout", [(136, 72), (64, 200)], 3, 80, "bf16", C=0.05, sigma=0.7,
                 d_std=0.1, wid=611)
    layers = W.make_inputs(w, seed=2)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    out = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, seed=3, step=5,
                         audit_capacity=w.B)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.run_step(ctx, Ad, Dd, out)
        t0 = time.perf_counter()
        assert dp.dp_debug_bounded_wait(ctx, 1_000_000) == 7          # DP_ERR_TIMEOUT
        assert time.perf_counter() - t0 < 5.0
        with pytest.raises(dp.DPError) as ei:
            dp.dp_audit_emit(ctx, range(w.B), len(w.layers))
        assert ei.value.status == 7
        assert "gave up" in str(ei.value)
        # a wait that is satisfied in time reports nothing: out of range is an argument error
        assert dp.lib().dp_debug_bounded_wait(ctx, 0) == 1
        # re-key: the flag is cleared and the next step is correct
        dp.dp_step_init(cfg, None, ctx)
        dp.run_step(ctx, Ad, Dd, out)
        recs = dp.dp_audit_emit(ctx, range(w.B), len(w.layers))
        torch.cuda.synchronize()
    finally:
        dp.dp_step_destroy(ctx)
    ref = O.dp_step([(W.to_f64(A), W.to_f64(D)) for A, D in layers], f32(w.C), f32(w.sigma),
                    3, 5)
    assert rel_err_elementwise(recs["layer_sqnorm"].astype(np.float64).T, ref["n"]) <= TOL["bf16"]
    for o, r in zip(out, ref["out"]):
        assert rel_err_normwise(o.double().cpu().numpy(), r) <= TOL["bf16"]


def test_commit_then_noise_equals_one_shot():
    """Commit (DP_NO_NOISE), re-key with the released seed, DP_NOISE_ONLY:
    equals the one-shot noisy output (Algorithm 2 commit-then-release)."""
    w = W.get("block_bf16")
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    one = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    two = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    scale = 1.0 / w.B
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=scale,
                         seed=77, step=4)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.run_step(ctx, Ad, Dd, one)
        cfg0 = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=scale,
                              seed=0, step=4)   # seed not released yet
        dp.dp_step_init(cfg0, ctx=ctx)
        dp.run_step(ctx, Ad, Dd, two, flags=dp.DP_NO_NOISE)
        dp.dp_step_init(cfg, ctx=ctx)           # released seed
        for l in range(len(layers)):
            dp.dp_clipped_sum_noise(ctx, l, None, None, two[l], dp.DP_NOISE_ONLY)
    finally:
        dp.dp_step_destroy(ctx)
    for a, b in zip(one, two):
        assert rel_err_normwise(b.cpu().numpy(), a.cpu().numpy()) <= 1e-6


def test_accumulate_over_microbatches():
    """Two micro-batches with DP_ACCUMULATE | DP_NO_NOISE sum their clipped sums."""
    w = W.custom("micro", [(96, 40)], 6, 32, "bf16", C=0.05, sigma=1.0, d_std=0.2, wid=603)
    layers = W.make_inputs(w)
    A, D = layers[0]
    dev = torch.device(DEV)
    out = torch.zeros(96, 40, device=dev)
    halves = [(A[:3], D[:3]), (A[3:], D[3:])]
    ref = np.zeros((96, 40))
    for Ah, Dh in halves:
        wh = W.custom("micro_h", [(96, 40)], 3, 32, "bf16", C=0.05, sigma=1.0, wid=603)
        cfg = dp.make_config(wh.layers, 3, 32, "bf16", wh.C, wh.sigma)
        ctx = dp.dp_step_init(cfg)
        try:
            dp.run_step(ctx, [Ah.contiguous().to(dev)], [Dh.contiguous().to(dev)], [out],
                        flags=dp.DP_NO_NOISE | dp.DP_ACCUMULATE)
        finally:
            dp.dp_step_destroy(ctx)
        r = oracle_step(wh, [(Ah, Dh)], noise=False)
        ref += r["out"][0]
    assert rel_err_normwise(out.cpu().numpy(), ref) <= 2e-3


def test_accumulate_large_layer():
    """DP_ACCUMULATE on a layer of 13 x 16 pair tiles (reduce-add stores)."""
    w = W.custom("micro_cl4", [(4096, 3320)], 4, 64, "bf16", C=0.05, sigma=1.0, d_std=0.2,
                 wid=604)
    layers = W.make_inputs(w)
    A, D = layers[0]
    dev = torch.device(DEV)
    out = torch.zeros(4096, 3320, device=dev)
    ref = np.zeros((4096, 3320))
    for h in range(2):
        Ah, Dh = A[2 * h:2 * h + 2].contiguous(), D[2 * h:2 * h + 2].contiguous()
        wh = W.custom("micro_cl4_h", [(4096, 3320)], 2, 64, "bf16", C=0.05, sigma=1.0, wid=604)
        cfg = dp.make_config(wh.layers, 2, 64, "bf16", wh.C, wh.sigma)
        ctx = dp.dp_step_init(cfg)
        try:
            dp.run_step(ctx, [Ah.to(dev)], [Dh.to(dev)], [out],
                        flags=dp.DP_NO_NOISE | dp.DP_ACCUMULATE)
        finally:
            dp.dp_step_destroy(ctx)
        ref += oracle_step(wh, [(Ah, Dh)], noise=False)["out"][0]
    assert rel_err_normwise(out.cpu().numpy(), ref) <= 2e-3


def test_eager_rekey_does_not_reach_a_queued_step():
    """Two steps enqueued back to back behind a long queue, re-keyed in
    between with no synchronisation: each uses its own key (the eager key
    is fixed when its launch is enqueued)."""
    w = W.get("block_bf16")
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    s = torch.cuda.Stream()
    outs = [[torch.zeros(i, o, device=dev) for i, o in w.layers] for _ in range(2)]
    x = torch.randn(8192, 8192, device=dev, dtype=torch.bfloat16)
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, seed=7, step=1)
    ctx = dp.dp_step_init(cfg, s)
    try:
        torch.cuda.synchronize()
        with torch.cuda.stream(s):
            for _ in range(8):
                x = (x @ x) * 1e-4          # milliseconds of queued work
            for k, t in enumerate((1, 2)):
                cfg.step = t
                dp.dp_step_init(cfg, s, ctx)
                dp.run_step(ctx, Ad, Dd, outs[k])
        torch.cuda.synchronize()
    finally:
        dp.dp_step_destroy(ctx)
    for k, t in enumerate((1, 2)):
        ref = run_gpu_step(w, layers, seed=7, step=t)
        for a, b in zip(outs[k], ref["out"]):
            assert np.array_equal(a.cpu().numpy(), b)


def test_deterministic_and_step_keyed():
    w = W.get("block_bf16")
    layers = W.make_inputs(w)
    r1 = run_gpu_step(w, layers, seed=3, step=10)
    r2 = run_gpu_step(w, layers, seed=3, step=10)
    r3 = run_gpu_step(w, layers, seed=3, step=11)
    for a, b, c in zip(r1["out"], r2["out"], r3["out"]):
        assert np.array_equal(a, b)
        assert not np.array_equal(a, c)
    assert np.array_equal(r1["n"], r2["n"]) and np.array_equal(r1["c"], r2["c"])


@pytest.mark.parametrize("p_first,n", [(0, 4096), (3, 1001), (140_000_001, 77), (1 << 40, 4099)])
def test_noise_add_range_matches_oracle(p_first, n):
    """dp_noise_add_range adds out_scale * sigma * C * z_{p_first + e} to any
    range of global parameter indices (a rank's slice of the commitment):
    elementwise against the oracle to 1e-6, with unaligned starts and ragged
    ends; n = 0 launches nothing."""
    w = W.custom("range", [(8, 8)], 2, 1, "f32", C=0.7, sigma=1.3, wid=612)
    dev = torch.device(DEV)
    scale = 0.25
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=scale,
                         seed=(1 << 62) + 9, step=17)
    ctx = dp.dp_step_init(cfg)
    g = torch.Generator().manual_seed(n)
    init = torch.randn(n + 8, generator=g)
    buf = init.clone().to(dev)
    try:
        n0 = dp.dp_kernel_launches()
        dp.dp_noise_add_range(ctx, p_first, 0, buf)
        assert dp.dp_kernel_launches() == n0
        dp.dp_noise_add_range(ctx, p_first, n, buf)
        torch.cuda.synchronize()
    finally:
        dp.dp_step_destroy(ctx)
    got = buf.double().cpu().numpy()
    z = O.gaussian_noise((1 << 62) + 9, 17, p_first, n)
    want = scale * f32(w.sigma) * f32(w.C) * z
    added = got[:n] - init.double().numpy()[:n]
    bound = 1e-6 * np.abs(want) + 2 * 2.0 ** -24 * np.abs(got[:n])
    assert np.all(np.abs(added - want) <= bound)
    assert np.array_equal(got[n:], init.double().numpy()[n:])   # nothing past the range


def test_noise_statistics_on_device():
    """Noise-only output over a large layer: mean ~ 0, variance ~ (out_scale sigma C)^2."""
    w = W.custom("stat", [(4096, 4096)], 2, 1, "bf16", C=0.5, sigma=1.3, wid=604)
    dev = torch.device(DEV)
    out = torch.zeros(4096, 4096, device=dev)
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=0.5, seed=9)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.dp_clipped_sum_noise(ctx, 0, None, None, out, dp.DP_NOISE_ONLY)
    finally:
        dp.dp_step_destroy(ctx)
    x = out.double().cpu().numpy().ravel()
    sd = 0.5 * f32(1.3) * f32(0.5)
    n = x.size
    assert abs(x.mean()) <= 5 * sd / math.sqrt(n)
    assert abs(x.var() / sd ** 2 - 1) <= 5 * math.sqrt(2 / n)


def test_noise_only_batch_one_launch():
    """DP_NOISE_ONLY over several layers in one batched call: one launch, the
    same bits as per-layer calls, and scale * z of the oracle to 1e-6.  The
    layer sizes are not multiples of 4, so most layers start inside a Philox
    quad, and the largest spans several 4096-quad blocks with a ragged end."""
    shapes = [(3, 5), (64, 33), (7, 1), (300, 257), (1, 3), (128, 128)]
    w = W.custom("noise_batch", shapes, 2, 1, "f32", C=0.7, sigma=1.3, wid=611)
    dev = torch.device(DEV)
    scale = 0.25
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=scale,
                         seed=(1 << 63) + 5, step=11)
    ctx = dp.dp_step_init(cfg)
    g = torch.Generator().manual_seed(3)
    init = [torch.randn(i, o, generator=g) for i, o in shapes]
    one = [x.clone().to(dev) for x in init]
    per = [x.clone().to(dev) for x in init]
    zero = [torch.zeros(i, o, device=dev) for i, o in shapes]
    try:
        n0 = dp.dp_kernel_launches()
        dp.dp_clipped_sum_noise_batch(ctx, list(range(len(shapes))), None, None, one,
                                      dp.DP_NOISE_ONLY)
        assert dp.dp_kernel_launches() - n0 == 1
        for l in range(len(shapes)):
            dp.dp_clipped_sum_noise(ctx, l, None, None, per[l], dp.DP_NOISE_ONLY)
        # listed out of order: each layer still takes its own global indices
        dp.dp_clipped_sum_noise_batch(ctx, list(range(len(shapes)))[::-1], None, None,
                                      zero[::-1], dp.DP_NOISE_ONLY)
    finally:
        dp.dp_step_destroy(ctx)
    torch.cuda.synchronize()
    for a, b in zip(one, per):
        assert torch.equal(a, b)
    z = O.gaussian_noise((1 << 63) + 5, 11, 0, sum(i * o for i, o in shapes))
    want = z * (scale * float(np.float32(w.sigma)) * float(np.float32(w.C)))
    got = np.concatenate([x.double().cpu().numpy().ravel() for x in zero])
    assert rel_err_elementwise(got, want) <= 1e-6


# ---------------------------------------------------------------------------
# tensor-core paths: ragged tiles, persistence across many tiles, both norms
# ---------------------------------------------------------------------------

TC_CASES = [
    # (layers, B, T): bf16 layers whose clipped sum and norms run on tcgen05
    ([(200, 264)], 3, 64),               # ragged M and N tiles
    ([(40, 48), (48, 56)], 2, 64),       # tiles far smaller than one MMA (not thin)
    ([(520, 1000), (1000, 136)], 2, 128),
    ([(4096, 4096)], 2, 64),             # 512 tiles > SM count: persistent loop
    ([(384, 512)], 5, 192),              # 3 K-blocks per example, T not a power of 2
    ([(200, 520)], 3, 45),               # T padded to 64 per example (3-D maps)
    ([(264, 136), (64, 8)], 4, 97),      # padded, ragged
    ([(3320, 3320)], 2, 64),             # 13 x 13 pair tiles, ragged in M and N
    ([(3320, 4096)], 2, 96),             # 13 x 16 pair tiles, 3-D maps
    # stages of two K blocks loaded as 128-row boxes (pairs, T % 128 == 0),
    # beside a single-CTA layer of the same step that keeps 64-row boxes
    ([(264, 520), (120, 296)], 3, 256),
    ([(704, 136)], 2, 384),              # six K blocks per example, ragged M and N
]

SMALL_T_CASES = [
    # T < 32: the clipped sum runs on the pre-scaled hi+lo operand
    ([(264, 136)], 7, 3),
    ([(3320, 264)], 5, 31),
    ([(4096, 1024)], 16, 1),
    ([(136, 72), (72, 8)], 33, 31),
]


@pytest.mark.parametrize("case", range(len(TC_CASES)))
@pytest.mark.parametrize("mode", [dp.DP_NORM_GHOST, dp.DP_NORM_MATERIALISED])
def test_tensor_core_paths(case, mode):
    shapes, B, T = TC_CASES[case]
    w = W.custom(f"tc{case}", shapes, B, T, "bf16", C=0.2, sigma=0.5, d_std=0.05,
                 wid=700 + case)
    layers = W.make_inputs(w, seed=2)
    res = run_gpu_step(w, layers, seed=5, step=1, norm_mode=mode)
    for (di, do), path in zip(shapes, res["paths"]):
        thin = mode != dp.DP_NORM_GHOST and is_thin(di, do, T, "bf16")
        assert path == ((2, 0) if thin else (1, 1)), (shapes, res["paths"])
    ref = oracle_step(w, layers, seed=5, step=1)
    assert_step_matches(res, ref, "bf16")


def test_tail_split_of_the_last_round():
    """A 2304 x 2304 layer is 81 CTA-pair tiles of 256 x 256.  On a GPU of
    76 resident pairs the last round holds 5 tiles; they run as 5 x 15
    pieces of 1-2 examples on 75 pairs, the clipped sums' pieces are added
    by one more launch (the tail reduce, which also adds the noise), the
    materialised norm's pieces write their examples' partials directly.
    Full output, norms and factors against the oracle for both norm forms;
    DP_ACCUMULATE adds the same bits again."""
    units = torch.cuda.get_device_properties(0).multi_processor_count // 2
    tiles = 81
    r = tiles % units
    tail = tiles > units and r > 0 and units // r >= 2
    # B T = 4096: the GEMM adds the noise itself (the tail reduce for its pieces)
    w = W.custom("tail81", [(2304, 2304)], 16, 256, "bf16", C=0.2, sigma=0.5, d_std=0.05,
                 wid=771)
    layers = W.make_inputs(w, seed=4)
    ref = oracle_step(w, layers, seed=6, step=3, norm="ghost")
    for mode in (dp.DP_NORM_GHOST, dp.DP_NORM_MATERIALISED):
        res = run_gpu_step(w, layers, seed=6, step=3, norm_mode=mode)
        assert res["paths"] == [(1, 1)]
        assert_step_matches(res, ref, "bf16")
    dev = torch.device(DEV)
    A, D = [t.to(dev) for t in layers[0]]
    cfg = dp.make_config(w.layers, w.B, w.T, "bf16", w.C, w.sigma, seed=6, step=3)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.dp_layer_norms(ctx, 0, A, D)
        dp.dp_clip_factors(ctx)
        out = torch.zeros(2304, 2304, device=dev)
        n0 = dp.dp_kernel_launches()
        dp.dp_clipped_sum_noise(ctx, 0, A, D, out, 0)
        assert dp.dp_kernel_launches() - n0 == (2 if tail else 1)
        twice = out.clone()
        dp.dp_clipped_sum_noise(ctx, 0, A, D, twice, dp.DP_ACCUMULATE)
        torch.cuda.synchronize()
    finally:
        dp.dp_step_destroy(ctx)
    assert torch.equal(twice, 2 * out)
    assert rel_err_normwise(out.cpu().numpy(), ref["out"][0]) <= TOL["bf16"]


@pytest.mark.parametrize("B,T", [(8, 64), (16, 64), (128, 1)])
def test_noise_added_after_a_short_gemm(B, T):
    """With B T <= 1024 the tensor-core clipped sum writes the noiseless sum
    and the noise-add kernel adds the noise (one more launch): the output
    against the oracle, and two DP_ACCUMULATE calls against twice the
    oracle's step."""
    w = W.custom(f"nafter{B}_{T}", [(1024, 1536)], B, T, "bf16", C=0.3, sigma=0.7, d_std=0.05,
                 wid=780 + B + T)
    layers = W.make_inputs(w, seed=6)
    res = run_gpu_step(w, layers, seed=2, step=5)
    assert res["paths"][0][1] == 1   # tensor cores (direct, or pre-scaled at T < 32)
    ref = oracle_step(w, layers, seed=2, step=5, norm="ghost")
    assert_step_matches(res, ref, "bf16")
    dev = torch.device(DEV)
    A, D = [t.to(dev) for t in layers[0]]
    cfg = dp.make_config(w.layers, w.B, w.T, "bf16", w.C, w.sigma, seed=2, step=5)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.dp_layer_norms(ctx, 0, A, D)
        dp.dp_clip_factors(ctx)
        out = torch.zeros(1024, 1536, device=dev)
        n0 = dp.dp_kernel_launches()
        dp.dp_clipped_sum_noise(ctx, 0, A, D, out, dp.DP_ACCUMULATE)
        gemm_launches = dp.dp_kernel_launches() - n0
        dp.dp_clipped_sum_noise(ctx, 0, A, D, out, dp.DP_ACCUMULATE)
        torch.cuda.synchronize()
    finally:
        dp.dp_step_destroy(ctx)
    # the GEMM (with its pre-scale pass or split reduce), then the noise
    assert gemm_launches in (2, 3)
    assert rel_err_normwise(out.cpu().numpy(), 2 * ref["out"][0]) <= TOL["bf16"]


@pytest.mark.parametrize("case", range(len(SMALL_T_CASES)))
def test_small_T_prescaled_clipped_sum(case):
    shapes, B, T = SMALL_T_CASES[case]
    w = W.custom(f"smallT{case}", shapes, B, T, "bf16", C=0.2, sigma=0.5, d_std=0.05,
                 wid=750 + case)
    layers = W.make_inputs(w, seed=3)
    res = run_gpu_step(w, layers, seed=8, step=2)
    for (di, do), (npath, spath) in zip(shapes, res["paths"]):
        assert (npath, spath) == (2, 0) if is_thin(di, do, T, "bf16") else spath, res["paths"]
    ref = oracle_step(w, layers, seed=8, step=2)
    assert_step_matches(res, ref, "bf16")
    nz = run_gpu_step(w, layers, flags=dp.DP_NO_NOISE, audit=False)
    r0 = oracle_step(w, layers, noise=False)
    for o, r in zip(nz["out"], r0["out"]):
        assert rel_err_normwise(o, r) <= 1e-4   # hi+lo split keeps c_i a to ~2^-16


def test_workload_paths_use_tensor_cores():
    for name, expect in [("block_bf16", True), ("llm_bf16", True), ("mlp_fp32", False)]:
        w = W.get(name)
        cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma)
        ctx = dp.dp_step_init(cfg)
        try:
            paths = [dp.dp_layer_path(ctx, l) for l in range(len(w.layers))]
        finally:
            dp.dp_step_destroy(ctx)
        for (i, o), p in zip(w.layers, paths):
            assert p == ((2, 0) if is_thin(i, o, w.T, w.dtype) else (expect, expect)), (name, paths)


@pytest.mark.parametrize("T", [200, 300, 450, 512, 640, 800, 1000, 1100, 2000])
def test_gram_strips_cover_every_block_pair(T):
    """Tensor-core Gram norms at 2 to 16 blocks of 128 positions: the strips
    must cover every block pair of the upper triangle once (diagonal pairs
    weighted 1, the others 2), with ragged last blocks."""
    shapes = [(64, 72), (136, 32)]
    w = W.custom(f"gram{T}", shapes, 2, T, "bf16", C=1e6, sigma=0.0, wid=960 + T % 97)
    layers = W.make_inputs(w, seed=1)
    res = run_gpu_step(w, layers, norm_mode=dp.DP_NORM_GHOST, flags=dp.DP_NO_NOISE, audit=True)
    assert res["modes"] == [dp.DP_NORM_GHOST] * 2 and all(p[0] == 1 for p in res["paths"])
    for l, (A, D) in enumerate(layers):
        ref = O.layer_sqnorms_materialised(W.to_f64(A), W.to_f64(D))
        assert rel_err_elementwise(res["n"][l], ref) <= TOL["bf16"]


@pytest.mark.parametrize("B,T,layers,want", [
    (8, 64, [(4096, 4096)], dp.DP_NORM_MATERIALISED),   # 8 Gram items: one item's latency decides
    (32, 64, [(4096, 4096)], dp.DP_NORM_GHOST),         # materialised work grows with B
    (128, 64, [(4096, 4096)], dp.DP_NORM_GHOST),        # enough items to fill the GPU
    (8, 512, [(4096, 4096)], dp.DP_NORM_GHOST),         # CTA-pair items, arithmetic decides
    (32, 128, [(768, 2304), (768, 768), (768, 3072), (3072, 768)], dp.DP_NORM_GHOST),
])
def test_auto_norm_form_latency_term(B, T, layers, want):
    """DP_NORM_AUTO's choice where the Gram form's few work items leave the
    GPU mostly idle: at B = 8, T = 64 on the 4096 x 4096 layer the
    materialised form is faster up to the clip factors (measured 0.033
    against 0.038 ms) and AUTO takes it; at larger B, longer examples or
    several layers sharing the Gram launch (block_bf16) it keeps the Gram
    form."""
    cfg = dp.make_config(layers, B, T, "bf16", 1.0, 1.0)
    ctx = dp.dp_step_init(cfg)
    try:
        assert all(dp.dp_layer_norm_mode(ctx, l) == want for l in range(len(layers)))
    finally:
        dp.dp_step_destroy(ctx)


def test_ghost_and_materialised_agree_on_block_workload():
    w = W.get("block_bf16")
    layers = W.make_inputs(w)
    g = run_gpu_step(w, layers, norm_mode=dp.DP_NORM_GHOST, flags=dp.DP_NO_NOISE)
    m = run_gpu_step(w, layers, norm_mode=dp.DP_NORM_MATERIALISED, flags=dp.DP_NO_NOISE)
    assert rel_err_elementwise(g["n"], m["n"]) <= 1e-4


# ---------------------------------------------------------------------------
# the 4096 x 4096 sweep at full size (sampled against the oracle)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name", [w.name for w in W.SWEEP])
def test_sweep_point_full_size(name):
    w = W.get(name)
    A, D = W.make_layer(w, 0, seed=0)
    res = run_gpu_step(w, [(A, D)], seed=4, step=9)
    rng = np.random.default_rng(w.wid)
    ex = np.sort(rng.choice(w.B, size=min(3, w.B), replace=False))
    n_ref = O.layer_sqnorms_ghost(W.to_f64(A[ex]), W.to_f64(D[ex]))
    assert rel_err_elementwise(res["n"][0, ex], n_ref) <= TOL["bf16"]
    # c_i of the sampled examples (one layer: s_i = n_i)
    _, c_ref = O.clip_factors(n_ref[None, :], f32(w.C))
    assert rel_err_elementwise(res["c"][ex], c_ref) <= TOL["bf16"]
    # unclipped, noiseless sum on sampled rows: S[rows] = sum_i A_i[:, rows]^T D_i
    wu = W.custom(name + "_unclipped", w.layers, w.B, w.T, "bf16", C=1e30, sigma=0.0,
                  wid=w.wid)
    resu = run_gpu_step(wu, [(A, D)], flags=dp.DP_NO_NOISE, audit=False)
    rows = np.sort(rng.choice(4096, size=16, replace=False))
    ones = np.ones(1)
    S = np.zeros((rows.size, 4096))
    for i in range(w.B):                     # the oracle's sum, one example at a time
        S += O.clipped_sum(W.to_f64(A[i:i + 1, :, rows]), W.to_f64(D[i:i + 1]), ones)
    assert rel_err_normwise(resu["out"][0][rows], S) <= TOL["bf16"]
    # the clipped, noisy output of the first run on the same rows, with the
    # clip factors the GPU formed (checked above on the sampled examples)
    c_gpu = res["c"].astype(np.float64)
    Sc = np.zeros((rows.size, 4096))
    for i in range(w.B):
        Sc += O.clipped_sum(W.to_f64(A[i:i + 1, :, rows]), W.to_f64(D[i:i + 1]), c_gpu[i:i + 1])
    z = np.stack([O.gaussian_noise(4, 9, int(j) * 4096, 4096) for j in rows])
    ref = Sc + f32(w.sigma) * f32(w.C) * z
    assert rel_err_normwise(res["out"][0][rows], ref) <= TOL["bf16"]


def test_fused_noise_of_the_tensor_core_sum_elementwise():
    """The noise the tensor-core clipped sum adds inside its main loop, alone:
    with D = 0 every S_l is exactly 0, so out = out_scale * sigma * C * z and
    each element must be within 1e-6 of the oracle's z (llm_bf16 shapes and
    batch, sampled rows of every layer).  Then, on the real inputs, the noisy
    output minus the noiseless commitment is that noise to 1e-6 plus the
    fp32 rounding of the sums (a few ulp of each output)."""
    w = W.get("llm_bf16")
    dev = torch.device(DEV)
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    Ad = [torch.randn(w.B, w.T, i, generator=g, device=dev).to(torch.bfloat16)
          for i, _ in w.layers]
    Z = [torch.zeros(w.B, w.T, o, device=dev, dtype=torch.bfloat16) for _, o in w.layers]
    outs = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    scale, seed, step = 1.0 / w.B, 17, 4
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=scale, seed=seed,
                         step=step)
    ctx = dp.dp_step_init(cfg)
    try:
        assert all(dp.dp_layer_path(ctx, l)[1] == 1 for l in range(len(w.layers)))
        dp.run_step(ctx, Ad, Z, outs)
        torch.cuda.synchronize()
        rng = np.random.default_rng(8)
        k = scale * f32(w.sigma) * f32(w.C)
        off = 0
        for l, (d_in, d_out) in enumerate(w.layers):
            rows = np.sort(rng.choice(d_in, size=6, replace=False))
            z = np.stack([O.gaussian_noise(seed, step, off + int(j) * d_out, d_out) for j in rows])
            got = outs[l][torch.as_tensor(rows, device=dev)].double().cpu().numpy()
            assert rel_err_elementwise(got, k * z) <= 1e-6, l
            off += d_in * d_out
        # real inputs: noisy minus noiseless
        Dd = [(torch.randn(w.B, w.T, o, generator=g, device=dev) * w.d_std).to(torch.bfloat16)
              for _, o in w.layers]
        noisy = [torch.zeros(i, o, device=dev) for i, o in w.layers]
        clean = [torch.zeros(i, o, device=dev) for i, o in w.layers]
        dp.dp_step_init(cfg, None, ctx)
        dp.run_step(ctx, Ad, Dd, noisy)
        dp.dp_step_init(cfg, None, ctx)
        dp.run_step(ctx, Ad, Dd, clean, flags=dp.DP_NO_NOISE)
        torch.cuda.synchronize()
        off = 0
        for l, (d_in, d_out) in enumerate(w.layers):
            rows = torch.as_tensor(np.sort(rng.choice(d_in, size=4, replace=False)), device=dev)
            a = noisy[l][rows].double().cpu().numpy()
            b = clean[l][rows].double().cpu().numpy()
            z = np.stack([O.gaussian_noise(seed, step, off + int(j) * d_out, d_out)
                          for j in rows.cpu().numpy()])
            want = k * z
            # each of the B folds into the fp32 accumulator rounds once, and the
            # noisy run adds the noise before the folds, the clean one does not
            bound = 1e-6 * np.abs(want) + w.B * 2.0 ** -24 * (np.abs(a) + np.abs(b))
            assert np.all(np.abs((a - b) - want) <= bound), l
            off += d_in * d_out
    finally:
        dp.dp_step_destroy(ctx)


def test_batched_norms_equal_per_layer_calls():
    """dp_layer_norms_batch gives the same norms as one dp_layer_norms per layer."""
    w = W.get("block_bf16")
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    outs = []
    for batched in (False, True):
        cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, audit_capacity=w.B)
        ctx = dp.dp_step_init(cfg)
        try:
            if batched:
                order = [2, 0, 3, 1]
                dp.dp_layer_norms_batch(ctx, order, [Ad[l] for l in order], [Dd[l] for l in order])
            else:
                for l in range(len(layers)):
                    dp.dp_layer_norms(ctx, l, Ad[l], Dd[l])
            dp.dp_clip_factors(ctx)
            recs = dp.dp_audit_emit(ctx, range(w.B), len(layers))
        finally:
            dp.dp_step_destroy(ctx)
        outs.append(recs["layer_sqnorm"].astype(np.float64))
    assert np.array_equal(outs[0], outs[1])
    ref = oracle_step(w, layers, noise=False)
    assert rel_err_elementwise(outs[1].T, ref["n"]) <= 2e-3
    # invalid batch: duplicate layer, nothing launched, context still usable
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma)
    ctx = dp.dp_step_init(cfg)
    try:
        with pytest.raises(dp.DPError) as ei:
            dp.dp_layer_norms_batch(ctx, [0, 0], [Ad[0], Ad[0]], [Dd[0], Dd[0]])
        assert ei.value.status == 1
        dp.dp_layer_norms_batch(ctx, [0, 1, 2, 3], Ad, Dd)
        dp.dp_clip_factors(ctx)
    finally:
        dp.dp_step_destroy(ctx)


def test_batched_clipped_sum_equals_per_layer_calls():
    """dp_clipped_sum_noise_batch writes the same outputs as per-layer calls."""
    w = W.get("block_bf16")
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    res = []
    for batched in (False, True):
        outs = [torch.zeros(i, o, device=dev) for i, o in w.layers]
        cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, seed=3, step=1)
        ctx = dp.dp_step_init(cfg)
        try:
            dp.dp_layer_norms_batch(ctx, [0, 1, 2, 3], Ad, Dd)
            dp.dp_clip_factors(ctx)
            if batched:
                order = [3, 1, 0, 2]
                dp.dp_clipped_sum_noise_batch(ctx, order, [Ad[l] for l in order],
                                              [Dd[l] for l in order], [outs[l] for l in order])
            else:
                for l in range(4):
                    dp.dp_clipped_sum_noise(ctx, l, Ad[l], Dd[l], outs[l])
        finally:
            dp.dp_step_destroy(ctx)
        res.append([o.cpu().numpy() for o in outs])
    for a, b in zip(*res):
        assert np.array_equal(a, b)
    ref = oracle_step(w, layers, seed=3, step=1)
    for o, r in zip(res[1], ref["out"]):
        assert rel_err_normwise(o, r) <= 2e-3


# ---------------------------------------------------------------------------
# the paper's own acceptance test on the commitment (Sec. 6.2, Algorithm 1)
# ---------------------------------------------------------------------------

TAU_ABS = 1.60e-3   # tightest LLM routing threshold of the verifier table (App. E), units of C


@pytest.mark.parametrize("name", ["single_fp32", "mlp_fp32", "block_bf16"])
def test_commitment_passes_the_verifier_body_path(name):
    """The averaged commitment g = S/B passes the always-on structural check
    ||g|| <= C(1 + 1e-4) and lands in the FP32 body path of Algorithm 1:
    z = ||g_GPU - g_ref||_2 / C <= tau_abs against the fp64 recomputation."""
    w = W.get(name)
    layers = W.make_inputs(w, seed=0)
    res = run_gpu_step(w, layers, out_scale=1.0 / w.B, flags=dp.DP_NO_NOISE, audit=False)
    ref = oracle_step(w, layers, out_scale=1.0 / w.B, noise=False)
    g_gpu = np.concatenate([o.astype(np.float64).ravel() for o in res["out"]])
    g_ref = np.concatenate([r.ravel() for r in ref["out"]])
    C = f32(w.C)
    assert np.linalg.norm(g_gpu) <= C * (1 + 1e-4)
    z = np.linalg.norm(g_gpu - g_ref) / C
    assert z <= TAU_ABS, z


def test_cuda_graph_replay_matches_eager_steps():
    """A step captured once in a CUDA graph and replayed under new keys
    (dp_set_noise_key between replays) writes exactly the eager outputs."""
    w = W.custom("graph", [(264, 520), (520, 136)], 6, 64, "bf16", C=0.1, sigma=0.7, d_std=0.2,
                 wid=900)
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    s = torch.cuda.Stream()
    outs_g = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, seed=5, step=0,
                         audit_capacity=w.B)
    ctx = dp.dp_step_init(cfg, s)
    try:
        with torch.cuda.stream(s):
            dp.run_step(ctx, Ad, Dd, outs_g)            # eager warm-up (one-time set-up)
            dp.dp_audit_emit(ctx, [0], len(layers))
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=s):
                dp.dp_step_init(cfg, s, ctx)
                dp.run_step(ctx, Ad, Dd, outs_g)
            for step in (3, 4):
                dp.dp_set_noise_key(ctx, 5, step)
                graph.replay()
                recs = dp.dp_audit_emit(ctx, range(w.B), len(layers))
                got = [o.cpu().numpy().copy() for o in outs_g]
                eager = run_gpu_step(w, layers, seed=5, step=step)
                for a, b in zip(got, eager["out"]):
                    assert np.array_equal(a, b)
                assert np.array_equal(recs["layer_sqnorm"].astype(np.float64).T, eager["n"])
    finally:
        dp.dp_step_destroy(ctx)


SPLIT_CASES = [
    # (layers, B, T): tensor-core layers with few output tiles and many
    # examples, so each tile's examples are split into ranges and reduced
    ([(256, 64)], 64, 256),                 # one CTA-pair tile, 32 ranges
    ([(576, 64), (1152, 128)], 48, 100),    # conv-like widths, T % 64 != 0, 12 ranges
]


@pytest.mark.parametrize("mode", [dp.DP_NORM_AUTO, dp.DP_NORM_MATERIALISED])
@pytest.mark.parametrize("case", range(len(SPLIT_CASES)))
def test_split_batch_tensor_core_layers(case, mode):
    """Few tiles, many examples: the clipped sum splits each tile's examples
    into ranges, stores their partial sums and adds them in order with the
    noise (a second launch); the materialised norm splits the same way."""
    shapes, B, T = SPLIT_CASES[case]
    w = W.custom(f"split{case}", shapes, B, T, "bf16", C=0.2, sigma=0.6, d_std=0.1,
                 wid=880 + case)
    assert not any(is_thin(i, o, T, "bf16") for i, o in shapes)
    layers = W.make_inputs(w)
    res = run_gpu_step(w, layers, seed=8, step=3, out_scale=1.0 / B, norm_mode=mode)
    assert all(sum_tc == 1 for _, sum_tc in res["paths"])
    ref = oracle_step(w, layers, seed=8, step=3, out_scale=1.0 / B)
    assert_step_matches(res, ref, "bf16")
    # the split path runs (GEMM + reduce) and DP_ACCUMULATE adds exactly
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    cfg = dp.make_config(w.layers, B, T, "bf16", w.C, w.sigma, out_scale=1.0 / B,
                         norm_mode=mode)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.dp_layer_norms_batch(ctx, list(range(len(shapes))), Ad, Dd)
        dp.dp_clip_factors(ctx)
        once = torch.zeros(shapes[0], device=dev)
        twice = torch.zeros(shapes[0], device=dev)
        n0 = dp.dp_kernel_launches()
        dp.dp_clipped_sum_noise(ctx, 0, Ad[0], Dd[0], once, dp.DP_NO_NOISE)
        assert dp.dp_kernel_launches() - n0 == 2
        for _ in range(2):
            dp.dp_clipped_sum_noise(ctx, 0, Ad[0], Dd[0], twice, dp.DP_NO_NOISE | dp.DP_ACCUMULATE)
        torch.cuda.synchronize()
        assert torch.equal(twice, 2 * once)
    finally:
        dp.dp_step_destroy(ctx)


ODD_BASE_CASES = [
    # (layers, B, T): a tensor-core layer whose first global parameter index
    # is not a multiple of 4, so its noise groups straddle two Philox quads
    ([(1, 3), (264, 136)], 6, 128),     # direct tiles, p_base = 3
    ([(1, 5), (256, 64)], 64, 256),     # split ranges + reduce, p_base = 5
    ([(1, 3), (256, 256)], 16, 8),      # pre-scaled operand (T < 32), p_base = 3
]


@pytest.mark.parametrize("case", range(len(ODD_BASE_CASES)))
def test_tensor_core_layer_after_odd_sized_layer(case):
    shapes, B, T = ODD_BASE_CASES[case]
    w = W.custom(f"oddbase{case}", shapes, B, T, "bf16", C=0.3, sigma=0.9, d_std=0.1,
                 wid=890 + case, a_dist=("ones", "normal"))
    layers = W.make_inputs(w)
    res = run_gpu_step(w, layers, seed=9, step=7, out_scale=1.0 / B)
    assert res["paths"][1][1] == 1 and is_thin(*shapes[0], T, "bf16")
    ref = oracle_step(w, layers, seed=9, step=7, out_scale=1.0 / B)
    assert_step_matches(res, ref, "bf16")
    # the noise part alone equals the oracle's noise to 1e-6
    noiseless = run_gpu_step(w, layers, seed=9, step=7, out_scale=1.0 / B, flags=dp.DP_NO_NOISE,
                             audit=False)
    z = O.gaussian_noise(9, 7, 0, sum(i * o for i, o in shapes))
    got = np.concatenate([(a - b).ravel() for a, b in zip(res["out"], noiseless["out"])])
    want = z * (float(np.float32(w.C)) * float(np.float32(w.sigma)) / B)
    assert np.max(np.abs(got - want)) <= 1e-5 * np.max(np.abs(want))


def test_launch_counts_of_a_step():
    """The library's own launch count: 33 thin layers of one width bucket and
    T take two norm launches and two clipped-sum launches (32 layers per
    launch), the re-key, clip and audit one each, a call refused on the host
    none; a captured step counts its kernels once, at capture, and replays
    add nothing."""
    w = W.custom("launch33", [(64, 8)] * 33, 4, 64, "bf16", C=0.5, sigma=0.5, wid=870)
    assert is_thin(64, 8, w.T, w.dtype)
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    outs = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    ids = list(range(len(layers)))
    n = dp.dp_kernel_launches
    s = torch.cuda.Stream()
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, audit_capacity=w.B)
    ctx = dp.dp_step_init(cfg, s)
    try:
        with torch.cuda.stream(s):
            counts = []
            for call in (lambda: dp.dp_step_init(cfg, s, ctx),
                         lambda: dp.dp_layer_norms_batch(ctx, ids, Ad, Dd),
                         lambda: dp.dp_clip_factors(ctx),
                         lambda: dp.dp_clipped_sum_noise_batch(ctx, ids, Ad, Dd, outs, 0),
                         lambda: dp.dp_audit_emit(ctx, range(w.B), len(layers))):
                c0 = n()
                call()
                counts.append(n() - c0)
            assert counts == [1, 2, 1, 2, 1]
            c0 = n()
            with pytest.raises(dp.DPError):
                dp.dp_clip_factors(ctx)          # twice in one step: refused on the host
            assert n() == c0
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=s):
                dp.dp_step_init(cfg, s, ctx)
                dp.run_step(ctx, Ad, Dd, outs)
            assert n() - c0 == 6
            c0 = n()
            for _ in range(3):
                graph.replay()
            s.synchronize()
            assert n() == c0
    finally:
        dp.dp_step_destroy(ctx)


# ---------------------------------------------------------------------------
# the GPU's update after the seed release (Algorithm 2, OptStep = AdamW, App. A)
# ---------------------------------------------------------------------------

U32 = 2.0 ** -24          # fp32 unit roundoff
Z_REL = 1e-6              # elementwise relative error of the device Gaussian (test above)


def adamw_error_bound(committed, theta, m, v, z, s, hp):
    """First-order forward error of the fp32 kernel, per element, from the
    fp64 values: every fp32 operation rounds once (relative U32), z carries
    Z_REL, and the errors propagate through m', v', the bias corrections,
    sqrt, the division and the final update.  Returned with a 4x margin."""
    b1, b2, lr, eps, wd, t = hp["beta1"], hp["beta2"], hp["lr"], hp["eps"], hp["wd"], hp["t"]
    g = committed + s * z
    e_g = s * np.abs(z) * (Z_REL + 3 * U32) + np.abs(g) * U32
    m2 = b1 * m + (1 - b1) * g
    e_m = (1 - b1) * (e_g + np.abs(g) * U32) + np.abs(m2) * U32
    v2 = b2 * v + (1 - b2) * g * g
    e_v = (1 - b2) * (2 * np.abs(g) * e_g + 2 * g * g * U32) + np.abs(v2) * U32
    bc1 = 1.0 / (1.0 - b1 ** t)
    bc2 = 1.0 / (1.0 - b2 ** t)
    mh, vh = m2 * bc1, v2 * bc2
    e_mh = bc1 * e_m + np.abs(mh) * 2 * U32
    e_vh = bc2 * e_v + vh * 2 * U32
    sq = np.sqrt(vh)
    with np.errstate(divide="ignore", invalid="ignore"):
        e_sq = np.minimum(np.where(sq > 0, e_vh / (2 * sq), np.inf), np.sqrt(e_vh)) + sq * U32
    den = sq + eps
    e_den = e_sq + den * U32
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(den > 0, mh / den, 0.0)
        e_r = np.where(den > 0, e_mh / den + np.abs(r) * (e_den / den + U32), 0.0)
    upd = r + wd * theta
    e_upd = e_r + (np.abs(upd) + np.abs(wd * theta)) * U32
    th2 = theta - lr * upd
    e_th = abs(lr) * (e_upd + np.abs(upd) * U32) + np.abs(th2) * U32
    return {"g": 4 * e_g, "m": 4 * e_m, "v": 4 * e_v, "theta": 4 * e_th}


ADAMW_LAYERS = [(4, 5), (264, 520), (3, 7), (128, 1001)]   # aligned, vector+tail, unaligned


def _adamw_inputs(layers, seed, zero_state):
    rng = np.random.default_rng(seed)
    out = []
    for i, o in layers:
        c = rng.normal(0.0, 1e-3, (i, o)).astype(np.float32)
        th = rng.normal(0.0, 0.05, (i, o)).astype(np.float32)
        if zero_state:
            m = np.zeros((i, o), np.float32)
            v = np.zeros((i, o), np.float32)
        else:
            m = rng.normal(0.0, 1e-3, (i, o)).astype(np.float32)
            v = (rng.normal(0.0, 1e-3, (i, o)) ** 2).astype(np.float32)
        out.append((c, th, m, v))
    return out


@pytest.mark.parametrize("flags", [0, dp.DP_WRITE_GRAD, dp.DP_NO_NOISE | dp.DP_WRITE_GRAD])
@pytest.mark.parametrize("hpi", [0, 1, 2])
def test_noise_adamw_matches_oracle(flags, hpi):
    """theta', m', v' (and g~ when written back) against oracle.noise_adamw,
    elementwise within the propagated fp32 error bound, on layers whose
    parameter ranges start aligned, with a ragged tail, and unaligned."""
    hps = [dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, wd=0.0, t=1, zero=True),
           dict(lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-6, wd=0.1, t=1000, zero=False),
           dict(lr=-2e-2, beta1=0.0, beta2=0.5, eps=0.0, wd=0.01, t=3, zero=False)]
    hp = {k: (f32(x) if isinstance(x, float) else x) for k, x in hps[hpi].items()}
    B, C, sigma, seed, step = 64, 0.25, 1.1, 123, 9
    scale = 1.0 / B
    data = _adamw_inputs(ADAMW_LAYERS, 40 + hpi, hp["zero"])
    dev = torch.device(DEV)
    cfg = dp.make_config(ADAMW_LAYERS, B, 16, "f32", C, sigma, out_scale=scale, seed=seed,
                         step=step)
    ctx = dp.dp_step_init(cfg)
    got = []
    try:
        for l, (c, th, m, v) in enumerate(data):
            t_c, t_th, t_m, t_v = (torch.from_numpy(x.copy()).to(dev) for x in (c, th, m, v))
            dp.dp_noise_adamw(ctx, l, t_c, t_th, t_m, t_v, hp["lr"], hp["beta1"], hp["beta2"],
                              hp["eps"], hp["wd"], hp["t"], flags)
            got.append([x.cpu().numpy().astype(np.float64) for x in (t_c, t_th, t_m, t_v)])
    finally:
        dp.dp_step_destroy(ctx)
    s = 0.0 if flags & dp.DP_NO_NOISE else f32(scale) * f32(sigma) * f32(C)
    p0 = 0
    for (c, th, m, v), (g_g, th_g, m_g, v_g), (i, o) in zip(data, got, ADAMW_LAYERS):
        g_r, th_r, m_r, v_r = O.noise_adamw(c, th, m, v, seed, step, p0, s, 1.0, 1.0,
                                            hp["lr"], hp["beta1"], hp["beta2"], hp["eps"],
                                            hp["wd"], hp["t"])
        z = O.gaussian_noise(seed, step, p0, i * o).reshape(i, o)
        bound = adamw_error_bound(c.astype(np.float64), th.astype(np.float64),
                                  m.astype(np.float64), v.astype(np.float64), z, s, hp)
        for name, a, r in (("theta", th_g, th_r), ("m", m_g, m_r), ("v", v_g, v_r)):
            bad = np.abs(a - r) > bound[name] + 1e-37
            assert not bad.any(), (name, np.argwhere(bad)[:5], a[bad][:5], r[bad][:5])
        if flags & dp.DP_WRITE_GRAD:
            assert not (np.abs(g_g - g_r) > bound["g"] + 1e-37).any()
        else:
            assert np.array_equal(g_g, c.astype(np.float64))     # input left untouched
        p0 += i * o


def test_noise_adamw_gradient_equals_noise_only_path():
    """The noisy gradient written back by dp_noise_adamw is bit-identical to
    DP_NOISE_ONLY on the same committed buffer: the released update and the
    commit-then-noise path draw the same z with the same scale."""
    layers = [(136, 72), (64, 203)]
    B = 8
    rng = np.random.default_rng(5)
    dev = torch.device(DEV)
    cfg = dp.make_config(layers, B, 16, "f32", 0.3, 0.8, out_scale=1.0 / B, seed=99, step=17)
    ctx = dp.dp_step_init(cfg)
    try:
        for l, (i, o) in enumerate(layers):
            c = torch.from_numpy(rng.normal(0, 1e-2, (i, o)).astype(np.float32)).to(dev)
            a = c.clone()
            dp.dp_clipped_sum_noise(ctx, l, None, None, a, dp.DP_NOISE_ONLY)
            th = torch.zeros(i, o, device=dev)
            m = torch.zeros(i, o, device=dev)
            v = torch.zeros(i, o, device=dev)
            dp.dp_noise_adamw(ctx, l, c, th, m, v, 1e-3, 0.9, 0.999, 1e-8, 0.0, 1,
                              dp.DP_WRITE_GRAD)
            assert torch.equal(a, c)
    finally:
        dp.dp_step_destroy(ctx)


def test_noise_adamw_argument_errors():
    cfg = dp.make_config([(8, 8)], 2, 4, "f32", 1.0, 1.0)
    ctx = dp.dp_step_init(cfg)
    dev = torch.device(DEV)
    x = [torch.zeros(8, 8, device=dev) for _ in range(4)]
    try:
        hp = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0, t=1)
        for bad in (dict(beta1=1.0), dict(beta2=-0.1), dict(eps=-1.0), dict(t=0),
                    dict(lr=float("nan"))):
            h = dict(hp, **bad)
            with pytest.raises(dp.DPError):
                dp.dp_noise_adamw(ctx, 0, *x, h["lr"], h["beta1"], h["beta2"], h["eps"],
                                  h["weight_decay"], h["t"])
        with pytest.raises(dp.DPError):
            dp.dp_noise_adamw(ctx, 1, *x, **hp)
        with pytest.raises(dp.DPError):
            dp.dp_noise_adamw(ctx, 0, *x, **hp, flags=dp.DP_NOISE_ONLY)
        flat = torch.zeros(8 * 8 + 1, device=dev)
        with pytest.raises(dp.DPError):
            dp.dp_noise_adamw(ctx, 0, flat[1:], *x[1:], **hp)
    finally:
        dp.dp_step_destroy(ctx)


# ---------------------------------------------------------------------------
# the trusted side consumes the GPU's commitment and audit records (Algorithm 1)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name,fam", [("mlp_fp32", "roberta"), ("block_bf16", "gpt2"),
                                      ("mlp_fp32", "cifar10")])
def test_verifier_accepts_gpu_commitment_and_rejects_tampering(name, fam):
    from paper_2609_20532_gb300 import verifier as V
    w = W.get(name)
    layers = W.make_inputs(w, seed=0)
    res = run_gpu_step(w, layers, out_scale=1.0 / w.B, flags=dp.DP_NO_NOISE, audit=True)
    C = f32(w.C)
    prm = V.FAMILIES[fam]
    g32 = V.recompute_average(layers, C, np.float32)[0]
    g64 = V.recompute_average(layers, C, np.float64)[0]
    ver = V.Verifier(prm, C, w.B, coin_seed=9)
    r = ver.step(res["out"], lambda: g32, lambda: g64, checked=True)
    assert r.verdict == V.ACCEPT and r.path == "body", r
    assert r.z32 <= prm.tau_abs / 4
    # the audit records of every example check against the fp64 recomputation
    recs = np.zeros(w.B, dtype=dp.audit_dtype(len(layers)))
    recs["example"] = res["rec_i"]
    recs["total_sqnorm"] = res["rec_s"]
    recs["clip_factor"] = res["rec_c"]
    recs["layer_sqnorm"] = res["n"].T
    rep = V.check_audit_records(recs, layers, C, rtol=TOL[w.dtype])
    assert rep.ok, rep
    # one layer's commitment nudged by 3 tau_abs C: the body path cannot hold it
    bad = [o.copy() for o in res["out"]]
    bad[0].reshape(-1)[0] += 3 * prm.tau_abs * C
    r = V.Verifier(prm, C, w.B, coin_seed=9).step(bad, lambda: g32, lambda: g64, checked=True)
    assert r.path in ("hard_reject", "ambiguity") and r.z32 > prm.tau_abs
    if fam == "cifar10":
        assert r.verdict == V.ABORT      # 3 tau_abs > rho_ill = 2 tau_abs


# ---------------------------------------------------------------------------
# thin layers (LoRA factors, heads, bias rows): per-example gradients stored
# by the norm pass, summed by the clipped-sum pass
# ---------------------------------------------------------------------------

THIN_CASES = [
    # (layers, B, T, dtype)
    ([(256, 8), (8, 520)], 5, 64, "bf16"),        # LoRA-like down / up factors
    ([(1000, 4), (4, 1000)], 3, 100, "bf16"),     # r = 4, ragged wide side, T % 64 != 0
    ([(300, 3), (3, 300)], 4, 96, "bf16"),        # odd widths (6-byte bf16 rows)
    ([(1024, 32), (17, 600)], 2, 256, "f32"),     # widest bucket, r = 17 in it
    ([(1, 512)], 6, 80, "f32"),                   # a bias row (d_in = 1)
    ([(256, 8), (264, 136)], 3, 64, "bf16"),      # thin next to a tensor-core layer
    ([(1000, 12), (24, 1000)], 3, 101, "bf16"),   # MMA kernel, padded n-tiles, ragged chunk and T
    ([(16, 1536), (2048, 32)], 2, 150, "bf16"),   # MMA kernel, copied narrow rows, 3 and 4 chunks
    ([(1001, 6)], 3, 40, "bf16"),                 # bf16 r > 4 with unaligned rows: multiply-adds
]


@pytest.mark.parametrize("case", range(len(THIN_CASES)))
def test_thin_layers_match_oracle(case):
    shapes, B, T, dtype = THIN_CASES[case]
    w = W.custom(f"thin{case}", shapes, B, T, dtype, C=0.3, sigma=0.7, d_std=0.1,
                 wid=800 + case)
    layers = W.make_inputs(w)
    res = run_gpu_step(w, layers, seed=4, step=2, out_scale=1.0 / B)
    for (i, o), (npath, spath) in zip(shapes, res["paths"]):
        thin = is_thin(i, o, T, dtype)
        assert (npath == 2) == thin and (not thin or spath == 0), (shapes, res["paths"])
    ref = oracle_step(w, layers, seed=4, step=2, out_scale=1.0 / B)
    assert_step_matches(res, ref, dtype)
    # the batched calls (one launch per bucket) give the same bits
    dev = torch.device(DEV)
    outs = [torch.zeros(i, o, device=dev) for i, o in shapes]
    cfg = dp.make_config(w.layers, B, T, dtype, w.C, w.sigma, out_scale=1.0 / B, seed=4, step=2)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.run_step(ctx, [A.to(dev) for A, _ in layers], [D.to(dev) for _, D in layers], outs)
    finally:
        dp.dp_step_destroy(ctx)
    for a, b in zip(outs, res["out"]):
        assert np.array_equal(a.cpu().numpy(), b)


def test_thin_accumulate_and_commit_then_noise():
    """DP_ACCUMULATE and the commit-then-noise order on the stored-gradient path."""
    w = W.custom("thin_acc", [(512, 8), (8, 512)], 4, 128, "bf16", C=0.2, sigma=0.9,
                 d_std=0.1, wid=820)
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    one = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    two = [torch.zeros(i, o, device=dev) for i, o in w.layers]
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, seed=8, step=3)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.run_step(ctx, Ad, Dd, one)
        dp.dp_step_init(cfg, ctx=ctx)
        dp.run_step(ctx, Ad, Dd, two, flags=dp.DP_NO_NOISE)
        for l in range(2):
            dp.dp_clipped_sum_noise(ctx, l, None, None, two[l], dp.DP_NOISE_ONLY)
        acc = [torch.zeros(i, o, device=dev) for i, o in w.layers]
        for _ in range(2):
            dp.dp_step_init(cfg, ctx=ctx)
            dp.run_step(ctx, Ad, Dd, acc, flags=dp.DP_NO_NOISE | dp.DP_ACCUMULATE)
    finally:
        dp.dp_step_destroy(ctx)
    ref = oracle_step(w, layers, noise=False)
    for a, b, c, r in zip(one, two, acc, ref["out"]):
        assert rel_err_normwise(b.cpu().numpy(), a.cpu().numpy()) <= 1e-6
        assert rel_err_normwise(c.cpu().numpy(), 2 * r) <= 2e-3


def test_gpt2_medium_lora_workload_full():
    """The 48 LoRA factor layers of GPT-2-medium (r = 4, B = 64, T = 128)
    against the full oracle, every norm and every output element."""
    w = W.get("gpt2m_lora_e2e_bf16")
    layers = W.make_inputs(w)
    res = run_gpu_step(w, layers, seed=1, step=7, out_scale=1.0 / w.B)
    assert all(n == 2 for n, _ in res["paths"])
    ref = oracle_step(w, layers, seed=1, step=7, out_scale=1.0 / w.B)
    assert_step_matches(res, ref, "bf16")


# ---------------------------------------------------------------------------
# layers with their own T: a classification head and bias rows on the first
# token next to LoRA factors over the whole sequence
# ---------------------------------------------------------------------------

MIXED_T_CASES = [
    # (layers (d_in, d_out, T), a_dist, dtype)
    ([(256, 8, 64), (8, 256, 64), (64, 32, 1), (1, 32, 1), (264, 136, 64), (40, 48, 3)],
     ("normal", "normal", "normal", "ones", "normal", "normal"), "bf16"),
    ([(128, 4, 96), (4, 300, 96), (300, 5, 1), (1, 5, 1)],
     ("normal", "normal", "normal", "ones"), "f32"),
]


@pytest.mark.parametrize("case", range(len(MIXED_T_CASES)))
def test_per_layer_T_matches_oracle(case):
    specs, a_dist, dtype = MIXED_T_CASES[case]
    w = W.custom(f"mixT{case}", specs, 6, 64, dtype, C=0.3, sigma=0.8, d_std=0.1,
                 wid=850 + case, a_dist=a_dist)
    layers = W.make_inputs(w)
    assert [A.shape[1] for A, _ in layers] == [t for _, _, t in specs]
    res = run_gpu_step(w, layers, seed=6, step=4, out_scale=1.0 / w.B)
    ref = oracle_step(w, layers, seed=6, step=4, out_scale=1.0 / w.B)
    assert_step_matches(res, ref, dtype)
    dev = torch.device(DEV)
    outs = [torch.zeros(i, o, device=dev) for i, o, _ in specs]
    cfg = dp.make_config(w.specs, w.B, w.T, dtype, w.C, w.sigma, out_scale=1.0 / w.B, seed=6,
                         step=4)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.run_step(ctx, [A.to(dev) for A, _ in layers], [D.to(dev) for _, D in layers], outs)
    finally:
        dp.dp_step_destroy(ctx)
    for a, b in zip(outs, res["out"]):
        assert np.array_equal(a.cpu().numpy(), b)


def test_roberta_adapters_with_head_reduced():
    """Two blocks of RoBERTa-style rank-8 query/value adapters (T = 128) and
    the 3-class head with its biases on the first token (T = 1), B = 64."""
    specs = [(1024, 8, 128), (8, 1024, 128)] * 4 + [(1024, 1024, 1), (1, 1024, 1),
                                                     (1024, 3, 1), (1, 3, 1)]
    a_dist = ("normal",) * 8 + ("normal", "ones", "normal", "ones")
    w = W.custom("rob_head", specs, 64, 128, "bf16", C=1.0, sigma=0.6407, d_std=0.01,
                 wid=860, a_dist=a_dist)
    layers = W.make_inputs(w)
    res = run_gpu_step(w, layers, seed=2, step=9, out_scale=1.0 / w.B)
    assert [n for n, _ in res["paths"][:8]] == [2] * 8
    ref = oracle_step(w, layers, seed=2, step=9, out_scale=1.0 / w.B)
    assert_step_matches(res, ref, "bf16")


def test_data_parallel_step_on_one_rank():
    """data_parallel_step through the library on a one-rank NCCL group: the
    commitment, the (trivial) reduce-scatter, the noise of the rank's slice
    (all of it) and the all-gather give the same bits as an eager step of the
    same context."""
    import socket
    import torch.distributed as dist
    from paper_2609_20532_gb300.data_parallel import FlatOutputs, data_parallel_step
    w = W.custom("dp1", [(136, 72), (64, 200)], 5, 64, "bf16", C=0.05, sigma=0.7, d_std=0.1,
                 wid=612)
    layers = W.make_inputs(w)
    dev = torch.device(DEV)
    Ad = [A.to(dev) for A, _ in layers]
    Dd = [D.to(dev) for _, D in layers]
    with socket.socket() as s_:
        s_.bind(("127.0.0.1", 0))
        port = s_.getsockname()[1]
    dist.init_process_group("nccl", init_method=f"tcp://127.0.0.1:{port}", rank=0, world_size=1)
    try:
        stream = torch.cuda.current_stream()
        cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=1.0 / w.B,
                             seed=21, step=3)
        fo = FlatOutputs(w.layers, 1, dev)
        ref = [torch.zeros(i, o, device=dev) for i, o in w.layers]
        ctx = dp.dp_step_init(cfg, stream)
        try:
            data_parallel_step(ctx, Ad, Dd, fo)
            dp.dp_step_init(cfg, stream, ctx)
            dp.run_step(ctx, Ad, Dd, ref, flags=dp.DP_NO_NOISE)
            dp.dp_clipped_sum_noise_batch(ctx, list(range(len(layers))), None, None, ref,
                                          dp.DP_NOISE_ONLY)
        finally:
            dp.dp_step_destroy(ctx)
        torch.cuda.synchronize()
    finally:
        dist.destroy_process_group()
    for a, b in zip(fo.views, ref):
        assert torch.equal(a, b)
    r = oracle_step(w, layers, seed=21, step=3, out_scale=1.0 / w.B)
    for o, rr in zip(fo.views, r["out"]):
        assert rel_err_normwise(o.cpu().numpy(), rr) <= TOL["bf16"]


DP2_SHAPES = [(136, 72), (64, 200), (96, 48)]
DP2_B, DP2_T = 6, 64


def _dp2_worker(rank, world, port, kind, out):
    """One rank of a two-process step on cuda:0 through the real library;
    the collectives run over gloo on host copies.  The ranks' kernels never
    wait on each other: only the host-side collectives join them."""
    import os
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch
    import torch.distributed as dist
    import paper_2609_20532_gb300 as dp
    import workloads as W
    from paper_2609_20532_gb300 import data_parallel as P
    torch.cuda.set_device(0)
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        w = W.custom("dp2", DP2_SHAPES, DP2_B, DP2_T, "bf16", C=0.05, sigma=0.7, d_std=0.1,
                     wid=613)
        layers = W.make_inputs(w)
        dev = torch.device("cuda:0")
        stream = torch.cuda.current_stream()
        if kind == "example":
            start, count = P.shard_examples(w.B, world, rank)
            Ad = [A[start:start + count].to(dev) for A, _ in layers]
            Dd = [D[start:start + count].to(dev) for _, D in layers]
            cfg = dp.make_config(w.layers, count, w.T, w.dtype, w.C, w.sigma,
                                 out_scale=1.0 / w.B, seed=21, step=3)
            fo = P.FlatOutputs(w.layers, world, dev)
            ctx = dp.dp_step_init(cfg, stream)
            try:
                P.data_parallel_step(ctx, Ad, Dd, fo, host_staging=True)
                torch.cuda.synchronize()
            finally:
                dp.dp_step_destroy(ctx)
            out[rank] = [v.cpu().numpy() for v in fo.views]
        else:
            first, count, pbase = P.shard_layers(w.layers, world, rank)
            mine = w.layers[first:first + count]
            Ad = [layers[l][0].to(dev) for l in range(first, first + count)]
            Dd = [layers[l][1].to(dev) for l in range(first, first + count)]
            cfg = dp.make_config(mine, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=1.0 / w.B,
                                 seed=21, step=3, param_base=pbase)
            outs = [torch.zeros(i, o, device=dev) for i, o in mine]
            s = torch.zeros(w.B, device=dev)
            ctx = dp.dp_step_init(cfg, stream)
            try:
                P.layer_parallel_step(ctx, Ad, Dd, outs, w.B, host_staging=True, s_total=s)
                torch.cuda.synchronize()
            finally:
                dp.dp_step_destroy(ctx)
            out[rank] = (first, [o.cpu().numpy() for o in outs], s.cpu().numpy())
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("kind", ["example", "layer"])
def test_two_rank_partitions_through_the_library(kind):
    """Both multi-GPU partitions at world size 2 with the real library (two
    processes sharing cuda:0, gloo collectives on host copies): by example,
    every rank ends with the whole-batch oracle step; by layer, every rank's
    outputs are the whole-model oracle step's for its layers and its summed
    squared norms those of the whole model."""
    import socket
    import torch.multiprocessing as mp
    with socket.socket() as s_:
        s_.bind(("127.0.0.1", 0))
        port = s_.getsockname()[1]
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    procs = [ctx.Process(target=_dp2_worker, args=(r, 2, port, kind, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
        assert p.exitcode == 0
    w = W.custom("dp2", DP2_SHAPES, DP2_B, DP2_T, "bf16", C=0.05, sigma=0.7, d_std=0.1, wid=613)
    layers = W.make_inputs(w)
    r = oracle_step(w, layers, seed=21, step=3, out_scale=1.0 / w.B)
    if kind == "example":
        for rank in range(2):
            for o, rr in zip(out[rank], r["out"]):
                assert rel_err_normwise(o, rr) <= TOL["bf16"]
        for a, b in zip(out[0], out[1]):
            assert np.array_equal(a, b)
    else:
        seen = []
        for rank in range(2):
            first, outs, s = out[rank]
            assert rel_err_elementwise(s, r["n"].sum(axis=0)) <= TOL["bf16"]
            for k, o in enumerate(outs):
                assert rel_err_normwise(o, r["out"][first + k]) <= TOL["bf16"]
                seen.append(first + k)
        assert sorted(seen) == list(range(len(DP2_SHAPES)))


def test_bench_data_parallel_path_two_ranks_one_gpu():
    """bench.py's multi-rank path (data_parallel_step under torchrun) at two
    ranks sharing cuda:0 with gloo collectives on host copies: it runs to
    completion and rank 0 prints one JSON line that counts both ranks'
    examples and names the partition."""
    import json
    import os
    import socket
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    with socket.socket() as s_:
        s_.bind(("127.0.0.1", 0))
        port = s_.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--gpus", "2",
           "--steps", "2", "--warmup", "3", "--workload", "block_bf16", "--dist-backend", "gloo",
           "--same-device", "--no-e2e"]
    r = subprocess.run(cmd, cwd=root, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    line = json.loads(lines[0])
    w = W.get("block_bf16")
    assert line["n_gpus"] == 2 and line["config"]["global_batch"] == 2 * w.B
    assert line["config"]["parallelism"] == "data-parallel by example"
    assert line["value"] == pytest.approx(2 * w.B / (line["ms_per_step"] * 1e-3))
    assert line["gpu_launches"] > 0 and line["collective_bytes_per_rank"] > 0
