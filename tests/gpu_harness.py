"""Helpers shared by the GPU tests: run one step through the C ABI and compare
it with the fp64 oracle on the same stored input bits."""

from __future__ import annotations

import math

import numpy as np
import torch

import paper_2609_20532_gb300 as dp
import workloads as W
from oracle import dp_oracle as O

TOL = {"f32": 1e-5, "bf16": 2e-3}


def f32(x: float) -> float:
    """The fp32 value the library receives for a config scalar."""
    return float(np.float32(x))


def conv_struct(w: W.Workload, l: int):
    """The library's description of layer l's convolution (None if dense)."""
    cv = w.conv_of(l)
    if not cv:
        return None
    H, W_, cin, kh, kw, st, pd = cv
    return dp.make_conv(H, W_, cin, kh, kw, (st, st), (pd, pd))


def device_inputs(w: W.Workload, layers, dev="cuda:0", conv_mode="explicit"):
    """A and D of every layer on the device.  conv_mode "explicit": a
    convolution's A becomes its patch rows through dp_conv2d_unfold; "library":
    it stays the NHWC input and the step forms the patch rows itself (the
    layer is declared DP_LAYER_CONV2D, see conv_structs)."""
    Ad, Dd = [], []
    for l, (A, D) in enumerate(layers):
        x = A.to(dev)
        conv = conv_struct(w, l)
        if conv is not None and conv_mode == "explicit":
            T, K = dp.dp_conv2d_dims(conv)
            a = torch.empty((w.B, T, K), dtype=x.dtype, device=dev)
            dp.dp_conv2d_unfold(conv, w.B, w.dtype, x, a)
            x = a
        Ad.append(x)
        Dd.append(D.to(dev))
    return Ad, Dd


def oracle_grads(w: W.Workload, layers):
    """fp64 per-example gradients of every layer from the oracle: a dense
    layer's A_i^T D_i, a convolution's from its definition (not through the
    patch rows), laid out [B, d_in, d_out] as the library's outputs are."""
    G = []
    for l, (A, D) in enumerate(layers):
        cv = w.conv_of(l)
        if cv:
            H, W_, cin, kh, kw, st, pd = cv
            Ho, Wo = O.conv2d_out_hw(H, W_, kh, kw, (st, st), (pd, pd))
            Dy = W.to_f64(D).reshape(w.B, Ho, Wo, -1)
            g = O.conv2d_weight_grads(W.to_f64(A), Dy, kh, kw, (st, st), (pd, pd))
            G.append(g.reshape(w.B, kh * kw * cin, -1))
        else:
            G.append(O.per_example_grads(W.to_f64(A), W.to_f64(D)))
    return G


def conv_structs(w: W.Workload, conv_mode: str):
    """make_config's convs argument: the geometries in "library" mode."""
    if conv_mode != "library" or not w.convs:
        return None
    return [conv_struct(w, l) for l in range(len(w.layers))]


def run_gpu_step(w: W.Workload, layers, seed=0, step=0, out_scale=1.0, flags=0,
                 norm_mode=dp.DP_NORM_AUTO, audit=True, conv_mode="explicit"):
    """Run norms -> clip -> clipped sum (+noise) on cuda:0.

    layers: list of (A, D) CPU tensors.  Returns dict with n [L,B], s, c
    (from the audit records of every example), out (list of fp32 numpy) and
    the chosen norm modes."""
    dev = torch.device("cuda:0")
    Ad, Dd = device_inputs(w, layers, dev, conv_mode)
    outs = [torch.zeros(i, o, device=dev, dtype=torch.float32) for i, o in w.layers]
    s_dev = torch.empty(w.B, device=dev)
    c_dev = torch.empty(w.B, device=dev)
    cfg = dp.make_config(w.specs, w.B, w.T, w.dtype, w.C, w.sigma, out_scale=out_scale,
                         seed=seed, step=step, norm_mode=norm_mode, audit_capacity=w.B,
                         convs=conv_structs(w, conv_mode))
    ctx = dp.dp_step_init(cfg)
    try:
        for l in range(len(layers)):
            dp.dp_layer_norms(ctx, l, Ad[l], Dd[l])
        dp.dp_clip_factors(ctx, s_dev, c_dev)
        for l in range(len(layers)):
            dp.dp_clipped_sum_noise(ctx, l, Ad[l], Dd[l], outs[l], flags)
        recs = dp.dp_audit_emit(ctx, range(w.B), len(layers)) if audit else None
        modes = [dp.dp_layer_norm_mode(ctx, l) for l in range(len(layers))]
        paths = [dp.dp_layer_path(ctx, l) for l in range(len(layers))]
    finally:
        dp.dp_step_destroy(ctx)
    torch.cuda.synchronize()
    res = {"out": [o.cpu().numpy() for o in outs], "s": s_dev.cpu().numpy(),
           "c": c_dev.cpu().numpy(), "modes": modes, "paths": paths}
    if recs is not None:
        res["n"] = recs["layer_sqnorm"].astype(np.float64).T
        res["rec_s"] = recs["total_sqnorm"].astype(np.float64)
        res["rec_c"] = recs["clip_factor"].astype(np.float64)
        res["rec_i"] = recs["example"].astype(np.int64)
    return res


def rel_err_elementwise(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.max(np.abs(got - ref) / np.maximum(np.abs(ref), 1e-30)))


def rel_err_normwise(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    den = np.linalg.norm(ref)
    return float(np.linalg.norm(got - ref) / den) if den > 0 else float(np.linalg.norm(got))


def assert_step_matches(res, ref, dtype: str, what=("n", "s", "c", "out")):
    tol = TOL[dtype]
    if "n" in what:
        e = rel_err_elementwise(res["n"], ref["n"])
        assert e <= tol, f"per-layer norms rel err {e:.3e} > {tol}"
    if "s" in what:
        e = rel_err_elementwise(res["s"], ref["s"])
        assert e <= tol, f"s rel err {e:.3e}"
        assert np.array_equal(res["rec_s"].astype(np.float32), res["s"].astype(np.float32))
    if "c" in what:
        e = rel_err_elementwise(res["c"], ref["c"])
        assert e <= tol, f"clip factor rel err {e:.3e}"
        assert np.all(res["c"] <= 1.0) and np.all(res["c"] > 0)
    if "out" in what:
        for l, (o, r) in enumerate(zip(res["out"], ref["out"])):
            e = rel_err_normwise(o, r)
            assert e <= tol, f"layer {l} output normwise rel err {e:.3e} > {tol}"
