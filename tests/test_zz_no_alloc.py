"""GPU test of dp_layer_sqnorms_noalloc, the entry point that allocates nothing.

Some callers cannot call cudaMalloc where they need per-example norms (inside
a CUDA stream capture in global mode, under a device-memory budget fixed at
start-up, or where the synchronisation an allocation may cause is not
allowed), so they cannot create a step context.  This test calls the
allocation-free entry point through the C ABI twice in a row and checks each
result against the existing context-based entry point (dp_layer_norms with
the Gram form) within the tolerances of the parity tests.  It lives in a file
collected last so that a stop-at-first-failure run has already run every
other test; it also passes alone in a fresh process.
"""

import ctypes

import numpy as np
import pytest
import torch

import paper_2609_20532_gb300 as dp
import workloads as W

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


CASES = [
    ("bf16", [(264, 136)], 5, 200),   # tensor-core Gram kernel, ragged tiles
    ("f32", [(40, 24)], 3, 70),       # CUDA-core Gram kernel
]


@pytest.mark.parametrize("dtype,layers,B,T", CASES)
def test_noalloc_matches_context_entry_point_twice(dtype, layers, B, T):
    torch.cuda.set_device(0)
    outs = []
    for call, seed in enumerate((0, 1)):      # two calls in a row, different inputs
        w = W.custom(f"noalloc{call}", layers, B, T, dtype, d_std=0.3, wid=800 + call)
        A, D = W.make_layer(w, 0, seed=seed)
        A, D = A.to(DEV), D.to(DEV)
        ref = _context_norms(w, A, D)
        out = torch.full((B,), float("nan"), device=DEV)
        torch.cuda.synchronize()
        free_before = torch.cuda.mem_get_info()[0]
        dp.dp_layer_sqnorms_noalloc(A, D, B, T, layers[0][0], layers[0][1], dtype, out)
        torch.cuda.synchronize()
        free_after = torch.cuda.mem_get_info()[0]
        got = out.cpu().numpy().astype(np.float64)
        rel = np.max(np.abs(got - ref) / np.maximum(np.abs(ref), 1e-30))
        assert rel <= TOL[dtype], (call, rel)
        if call == 1:
            # the second call on this device allocates nothing at all
            assert free_after == free_before
        outs.append(got)
    assert not np.array_equal(outs[0][: min(map(len, outs))], outs[1][: min(map(len, outs))])


def test_noalloc_rejects_requests_beyond_its_scratch():
    A = torch.zeros(16, device=DEV, dtype=torch.bfloat16)
    out = torch.zeros(1, device=DEV)
    st = dp.lib().dp_layer_sqnorms_noalloc(
        ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(A.data_ptr()), 4096, 1 << 17, 8, 8,
        dp.DP_BF16, ctypes.c_void_p(out.data_ptr()), None)
    assert st == 2  # DP_ERR_SHAPE, before any launch
    assert "scratch" in dp.dp_last_error()
