"""C-ABI checks that need no GPU: the library loads, exports every symbol the
header declares, and rejects bad arguments on the host before touching the
device."""

import ctypes
import os
import re

import pytest

import paper_2609_20532_gb300 as dp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dp_step.h")


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(dp.lib_path):
        from paper_2609_20532_gb300 import build
        build.build()
    return dp.lib()


def header_functions():
    txt = open(HEADER).read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    return sorted(set(re.findall(r"\b(dp_[a-z_0-9]+)\s*\(", txt)))


def test_header_and_binding_agree():
    assert header_functions() == sorted(dp.EXPORTED_SYMBOLS)


def test_library_exports_every_declared_symbol(L):
    for name in header_functions():
        assert hasattr(L, name), name


def _cfg(**kw):
    base = dict(layers=[(64, 32)], B=8, T=1, dtype="f32", C=1.0, sigma=1.0)
    base.update(kw)
    return dp.make_config(**base)


def _init_status(L, cfg):
    h = ctypes.c_void_p(None)
    st = L.dp_step_init(ctypes.byref(h), ctypes.byref(cfg) if cfg is not None else None, None)
    return st, h.value


@pytest.mark.parametrize("kw,status", [
    (dict(B=0), 2), (dict(T=0), 2), (dict(layers=[(0, 4)]), 2),
    (dict(layers=[(1 << 21, 4)]), 2), (dict(layers=[(8, 8)] * 1025), 2), (dict(layers=[(8, 8, -1)]), 1),
    (dict(C=0.0), 1), (dict(C=float("inf")), 1), (dict(sigma=-1.0), 1),
    (dict(sigma=float("nan")), 1), (dict(out_scale=float("inf")), 1),
    (dict(norm_mode=7), 1), (dict(norm_mode=dp.DP_NORM_RANK1, T=4), 2),
    (dict(audit_capacity=9), 1), (dict(audit_capacity=-1), 1),
])
def test_init_rejects_bad_config_on_host(L, kw, status):
    st, h = _init_status(L, _cfg(**kw))
    assert st == status, dp.dp_last_error()
    assert h is None
    assert dp.dp_last_error()


def test_init_rejects_null_and_bad_dtype(L):
    st, _ = _init_status(L, None)
    assert st == 1
    cfg = _cfg()
    cfg.dtype = 5
    st, _ = _init_status(L, cfg)
    assert st == 3
    cfg = _cfg()
    cfg.n_layers = 0
    st, _ = _init_status(L, cfg)
    assert st == 2
    assert L.dp_step_init(None, ctypes.byref(_cfg()), None) == 1


def test_calls_reject_null_context(L):
    assert L.dp_layer_norms(None, 0, 16, 16) == 1
    assert L.dp_layer_norms_batch(None, 1, None, None, None) == 1
    assert L.dp_clip_factors(None, None, None) == 1
    assert L.dp_clipped_sum_noise(None, 0, 16, 16, 16, 0) == 1
    assert L.dp_audit_emit(None, None, 0, None) == 1
    m = ctypes.c_int32()
    assert L.dp_layer_norm_mode(None, 0, ctypes.byref(m)) == 1
    assert L.dp_set_noise_key(None, 0, 0) == 1
    assert L.dp_noise_adamw(None, 0, 16, 16, 16, 16, None, 0) == 1
    L.dp_step_destroy(None)  # no-op


def test_misc_exports(L):
    assert L.dp_audit_record_bytes(3) == 24
    assert L.dp_status_string(5) == b"DP_ERR_NONFINITE"
    assert L.dp_debug_philox(0, 0, 0, -1, None, None) == 1
    assert L.dp_debug_gaussian(0, 0, 0, -1, None, None) == 1
    # zero-length requests launch nothing
    assert L.dp_debug_philox(0, 0, 0, 0, None, None) == 0


def test_kernel_launch_count_is_a_host_query(L):
    """dp_kernel_launches reads a host counter: no device is touched, a NULL
    output is rejected, and calls that fail on the host launch nothing."""
    n0 = dp.dp_kernel_launches()
    assert isinstance(n0, int) and n0 >= 0
    assert L.dp_kernel_launches(None) == 1
    st, h = _init_status(L, _cfg(B=0))
    assert st == 2 and not h
    assert dp.dp_kernel_launches() == n0


def test_conv2d_dims_on_host(L):
    """dp_conv2d_dims: T and K of a convolution, and its host-side refusals."""
    from oracle import dp_oracle as O
    for H, W_, C, kh, kw, st, pd in [(32, 32, 3, 3, 3, (1, 1), (1, 1)), (32, 32, 64, 1, 1, (2, 2), (0, 0)),
                                     (9, 7, 8, 2, 3, (1, 2), (0, 1)), (3, 3, 8, 3, 3, (1, 1), (0, 0))]:
        T, K = dp.dp_conv2d_dims(dp.make_conv(H, W_, C, kh, kw, st, pd))
        Ho, Wo = O.conv2d_out_hw(H, W_, kh, kw, st, pd)
        assert (T, K) == (Ho * Wo, kh * kw * C)
    for bad in [dp.make_conv(0, 8, 3, 3, 3), dp.make_conv(8, 8, 3, 3, 3, (0, 1)),
                dp.make_conv(8, 8, 3, 3, 3, (1, 1), (-1, 0)), dp.make_conv(2, 2, 3, 5, 5),
                dp.make_conv(8, 8, 1 << 18, 3, 3)]:
        with pytest.raises(dp.DPError) as ei:
            dp.dp_conv2d_dims(bad)
        assert ei.value.status == 2


def test_conv_layer_config_checked_on_host(L):
    """DP_LAYER_CONV2D layers: geometry present and consistent with d_in, T."""
    cv = dp.make_conv(8, 8, 16, 3, 3, (1, 1), (1, 1))      # T = 64, K = 144
    ok = dp.make_config([(144, 32)], 2, 1, "bf16", 1.0, 1.0, convs=[cv])
    assert ok.layers[0].kind == dp.DP_LAYER_CONV2D
    for layers, convs, status in [
        ([(144, 32)], None, None),                 # dense: fine without geometry
        ([(143, 32)], [cv], 2),                    # d_in is not kh*kw*C_in
        ([(144, 32, 63)], [cv], 2),                # T is not H_out*W_out
        ([(144, 32)], [dp.make_conv(2, 2, 16, 5, 5)], 2),
    ]:
        cfg = dp.make_config(layers, 2, 1, "bf16", 1.0, 1.0, convs=convs)
        st, h = _init_status(L, cfg)
        if status is None:
            assert st in (0, 6, 9), st   # no GPU here: the host checks passed
            if h:
                L.dp_step_destroy(h)
        else:
            assert st == status and not h
    bad = dp.make_config([(144, 32)], 2, 1, "bf16", 1.0, 1.0)
    bad.layers[0].kind = 7
    assert _init_status(L, bad)[0] == 1
    nogeom = dp.make_config([(144, 32)], 2, 1, "bf16", 1.0, 1.0)
    nogeom.layers[0].kind = dp.DP_LAYER_CONV2D
    assert _init_status(L, nogeom)[0] == 1


def test_header_is_plain_c_and_cpp():
    """include/dp_step.h is a C ABI: it compiles as C99 and as C++17 with
    warnings as errors, and a C translation unit can take the address of
    every declared entry point."""
    import shutil
    import subprocess
    import tempfile
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    inc = os.path.join(ROOT, "include")
    with tempfile.TemporaryDirectory() as td:
        src = os.path.join(td, "use.c")
        with open(src, "w") as f:
            f.write('#include "dp_step.h"\n')
            f.write("void* const entry_points[] = {\n")
            f.write("".join(f"  (void*)&{n},\n" for n in header_functions()))
            f.write("};\n")
        for lang, std in (("c", "-std=c99"), ("c++", "-std=c++17")):
            r = subprocess.run([gcc, "-fsyntax-only", std, "-Wall", "-Wextra", "-Werror",
                                "-x", lang, "-I", inc, src], capture_output=True, text=True)
            assert r.returncode == 0, (lang, r.stderr)


@pytest.mark.parametrize("dtype,B,T,d", [
    (dp.DP_BF16, 1, 1 << 22, 8),     # ~T^2/8192 partial sums would overflow 32-bit counts
    (dp.DP_F32, 1, 1 << 22, 8),
    (dp.DP_BF16, 1, 4_194_304, 4096),
    (dp.DP_BF16, 4096, 1 << 17, 8),  # fits 32 bits, exceeds the 2^20-float scratch
])
def test_noalloc_rejects_long_examples_on_host(L, dtype, B, T, d):
    """dp_layer_sqnorms_noalloc counts the Gram form's partial sums in 64 bits
    and refuses requests beyond its static scratch on the host.  The pointers
    are never dereferenced: the check comes before any CUDA call, so this
    runs without a GPU and launches nothing."""
    n0 = dp.dp_kernel_launches()
    fake = ctypes.c_void_p(1 << 20)   # 16-byte aligned, never touched
    st = L.dp_layer_sqnorms_noalloc(fake, fake, B, T, d, d, dtype, fake, None)
    assert st == 2, (st, dp.dp_last_error())
    assert "scratch" in dp.dp_last_error()
    assert dp.dp_kernel_launches() == n0


@pytest.mark.parametrize("mode,T,d", [
    (dp.DP_NORM_GHOST, 1 << 22, 8),  # forced Gram form on very long examples
])
def test_init_rejects_gram_form_beyond_its_partials(L, mode, T, d):
    """A forced Gram form whose partial sums per example exceed the norm
    scratch's bound is refused on the host with DP_ERR_SHAPE (the count is
    formed in 64 bits, so it cannot wrap into a small or negative number)."""
    cfg = _cfg(layers=[(d, d)], B=1, T=T, dtype="bf16", norm_mode=mode)
    st, h = _init_status(L, cfg)
    assert st == 2 and not h, (st, dp.dp_last_error())
    assert "partial sums" in dp.dp_last_error()
