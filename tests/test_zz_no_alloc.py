"""GPU test of dp_layer_sqnorms_noalloc, the entry point that allocates nothing.

Some callers cannot call cudaMalloc where they need per-example norms (inside
a CUDA stream capture in global mode, under a device-memory budget fixed at
start-up, or where the synchronisation an allocation may cause is not
allowed), so they cannot create a step context.  This test calls the
allocation-free entry point through the C ABI twice in a row and checks each
result against the existing context-based entry point (dp_layer_norms with
the Gram form) and against the fp64 oracle, within the tolerances of the
parity tests; then it captures a call into a CUDA graph in global capture
mode after a first, eager call has done the per-device set-up.  It lives in
a file collected last so that a stop-at-first-failure run has already run
every other test; it also passes alone in a fresh process.
"""

import ctypes

import numpy as np
import pytest
import torch

import paper_2609_20532_gb300 as dp
import workloads as W
from oracle import dp_oracle as O

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
TOL = {"f32": 1e-5, "bf16": 2e-3}


def _context_norms(w, A, D):
    """Per-example norms from the existing entry point (context, Gram form)."""
    cfg = dp.make_config(w.layers, w.B, w.T, w.dtype, w.C, w.sigma,
                         norm_mode=dp.DP_NORM_GHOST)
    s = torch.empty(w.B, device=DEV)
    ctx = dp.dp_step_init(cfg)
    try:
        dp.dp_layer_norms(ctx, 0, A, D)
        dp.dp_clip_factors(ctx, s, None)   # one layer: s_i = n_i
    finally:
        dp.dp_step_destroy(ctx)
    return s.cpu().numpy().astype(np.float64)


def _rel(got, ref):
    return float(np.max(np.abs(got - ref) / np.maximum(np.abs(ref), 1e-30)))


CASES = [
    ("bf16", [(264, 136)], 5, 200),   # tensor-core Gram, CTA pairs (2 blocks of 128)
    ("bf16", [(64, 200)], 3, 300),    # tensor-core Gram, single-CTA strips (3 blocks)
    ("f32", [(40, 24)], 3, 70),       # CUDA-core Gram kernel
]


@pytest.mark.parametrize("dtype,layers,B,T", CASES)
def test_noalloc_matches_context_entry_point_twice(dtype, layers, B, T):
    torch.cuda.set_device(0)
    outs = []
    for call, seed in enumerate((0, 1)):      # two calls in a row, different inputs
        w = W.custom(f"noalloc{call}", layers, B, T, dtype, d_std=0.3, wid=800 + call)
        A_cpu, D_cpu = W.make_layer(w, 0, seed=seed)
        A, D = A_cpu.to(DEV), D_cpu.to(DEV)
        ref = _context_norms(w, A, D)
        out = torch.full((B,), float("nan"), device=DEV)
        torch.cuda.synchronize()
        free_before = torch.cuda.mem_get_info()[0]
        dp.dp_layer_sqnorms_noalloc(A, D, B, T, layers[0][0], layers[0][1], dtype, out)
        torch.cuda.synchronize()
        free_after = torch.cuda.mem_get_info()[0]
        got = out.cpu().numpy().astype(np.float64)
        assert _rel(got, ref) <= TOL[dtype], (call, _rel(got, ref))
        # and against the plain definition (fp64 oracle on the same stored bits)
        n_ref = O.layer_sqnorms_materialised(W.to_f64(A_cpu), W.to_f64(D_cpu))
        assert _rel(got, n_ref) <= TOL[dtype], (call, _rel(got, n_ref))
        if call == 1:
            # the second call on this device allocates nothing at all
            assert free_after == free_before
        outs.append(got)
    assert not np.array_equal(outs[0][: min(map(len, outs))], outs[1][: min(map(len, outs))])


def test_noalloc_inside_global_mode_graph_capture():
    """After one eager call, a call captured in global mode (where allocation
    calls are refused) replays to the same norms as the context path, for
    both tensor-core Gram kernels and the CUDA-core one."""
    torch.cuda.set_device(0)
    shapes = [("bf16", (264, 136), 4, 256), ("bf16", (64, 200), 3, 300),
              ("f32", (40, 24), 3, 70)]
    inputs = []
    for k, (dtype, (di, do), B, T) in enumerate(shapes):
        w = W.custom(f"noalloc_graph{k}", [(di, do)], B, T, dtype, d_std=0.3, wid=830 + k)
        A, D = W.make_layer(w, 0, seed=7)
        inputs.append((w, A.to(DEV), D.to(DEV), torch.full((B,), float("nan"), device=DEV)))
    s = torch.cuda.Stream()
    # one eager call (the first call on the device does the set-up), on the first shape only
    w0, A0, D0, o0 = inputs[0]
    with torch.cuda.stream(s):
        dp.dp_layer_sqnorms_noalloc(A0, D0, w0.B, w0.T, w0.layers[0][0], w0.layers[0][1],
                                    w0.dtype, o0, stream=s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s, capture_error_mode="global"):
        for w, A, D, o in inputs:
            dp.dp_layer_sqnorms_noalloc(A, D, w.B, w.T, w.layers[0][0], w.layers[0][1],
                                        w.dtype, o, stream=s)
    for w, A, D, o in inputs:
        o.fill_(float("nan"))
    torch.cuda.synchronize()
    g.replay()
    torch.cuda.synchronize()
    for w, A, D, o in inputs:
        ref = _context_norms(w, A, D)
        got = o.cpu().numpy().astype(np.float64)
        assert _rel(got, ref) <= TOL[w.dtype], (w.name, _rel(got, ref))


def test_noalloc_rejects_requests_beyond_its_scratch():
    A = torch.zeros(16, device=DEV, dtype=torch.bfloat16)
    out = torch.zeros(1, device=DEV)
    st = dp.lib().dp_layer_sqnorms_noalloc(
        ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(A.data_ptr()), 4096, 1 << 17, 8, 8,
        dp.DP_BF16, ctypes.c_void_p(out.data_ptr()), None)
    assert st == 2  # DP_ERR_SHAPE, before any launch
    assert "scratch" in dp.dp_last_error()
