"""Seeded synthetic inputs for the DP-SGD step, shared by tests, smoke and bench.

This module holds only shapes, value distributions and the random draws; it
contains none of the DP-SGD arithmetic, so both the CUDA path and the CPU
oracle can be fed from it without sharing any of the method's code.

Recipe (stated once, used everywhere):
  * every array comes from ``numpy.random.default_rng(SeedSequence([seed,
    workload_id, layer, kind]))`` with kind 0 = activations A, 1 = output
    gradients D, 2 = audit indices;
  * draws are fp32 (numpy's float32 samplers), scaled by the distribution's
    standard deviation in fp32, then rounded to nearest-even into the
    workload's dtype (fp32: unchanged; bf16: one RNE rounding);
  * "N(0, v)" in a workload description is read as variance v (std sqrt(v));
    "ReLU-sparse N(0,1)" is max(0, x) with x ~ N(0,1) (about half exact zeros);
  * layouts: A [B, T, d_in], D [B, T, d_out], row-major, example-major; for
    a convolution layer A is its NHWC input [B, H, W, C_in] (the patch rows
    the layer's dense form needs are built from it by each side on its own)
    and D its output gradient [B, H_out * W_out, C_out].

The paper trains LoRA adapters of GPT-2 / RoBERTa, an MLP on Purchase and a
WideResNet on CIFAR-10 (App. B); none of those datasets or checkpoints is
available here, so these seeded dense-layer workloads stand in for them.
"""

from __future__ import annotations

import dataclasses
import math
from typing import List, Sequence, Tuple

import numpy as np
import torch

__all__ = ["Workload", "WORKLOADS", "SWEEP", "get", "make_layer", "make_inputs",
           "audit_indices", "to_f64"]


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    wid: int                       # id folded into the seed sequence
    layers: Tuple[Tuple[int, int], ...]
    B: int
    T: int
    dtype: str                     # "f32" or "bf16"
    a_dist: Tuple[str, ...]        # per layer: "normal", "uniform", "relu_normal"
    a_std: float
    d_std: float
    C: float
    sigma: float
    audit_frac: float = 0.0
    layer_T: Tuple[int, ...] = ()  # per-layer positions (empty: every layer has T)
    # per layer: None for a dense layer, else the convolution
    # (H, W, C_in, kh, kw, stride, pad) whose dense form is layers[l]
    convs: Tuple = ()

    @property
    def n_params(self) -> int:
        return sum(i * o for i, o in self.layers)

    def T_of(self, layer: int) -> int:
        return self.layer_T[layer] if self.layer_T else self.T

    def conv_of(self, layer: int):
        return self.convs[layer] if self.convs else None

    @property
    def specs(self) -> Tuple[Tuple[int, int, int], ...]:
        """(d_in, d_out, T) of every layer, as the C ABI's dp_layer takes them."""
        return tuple((i, o, self.T_of(l)) for l, (i, o) in enumerate(self.layers))

    def describe(self) -> str:
        def one(l, i, o):
            cv = self.conv_of(l)
            if cv:
                H, W_, cin, kh, kw, st, pd = cv
                return f"conv{kh}x{kw}s{st}:{H}x{W_}x{cin}->{o}"
            return f"{i}x{o}" if self.T_of(l) == self.T else f"{i}x{o}@T{self.T_of(l)}"
        dims = ",".join(one(l, i, o) for l, (i, o) in enumerate(self.layers))
        return f"{self.name}: layers[{dims}] B={self.B} T={self.T} {self.dtype}"


def _normal_all(n):
    return tuple("normal" for _ in range(n))


WORKLOADS = {
    # single linear layer, fp32, the small case the oracle finishes instantly
    "single_fp32": Workload("single_fp32", 1, ((64, 32),), 8, 1, "f32",
                            _normal_all(1), 1.0, 1.0, 1.0, 1.0),
    # 3-layer MLP 784-512-512-10, fp32; U[0,1) inputs, ReLU-sparse hidden
    # activations, D ~ N(0, 0.01)
    "mlp_fp32": Workload("mlp_fp32", 2, ((784, 512), (512, 512), (512, 10)), 256, 1,
                         "f32", ("uniform", "relu_normal", "relu_normal"),
                         1.0, math.sqrt(0.01), 1.0, 1.1),
    # transformer-block linears: QKV, out-proj, FFN up, FFN down; bf16
    "block_bf16": Workload("block_bf16", 3,
                           ((768, 2304), (768, 768), (768, 3072), (3072, 768)),
                           32, 128, "bf16", _normal_all(4), 1.0, math.sqrt(1e-4),
                           1.0, 0.8),
    # LLM-scale projections d_model=4096: FFN up/down and fused QKV; bf16
    "llm_bf16": Workload("llm_bf16", 4,
                         ((4096, 11008), (11008, 4096), (4096, 12288)),
                         16, 512, "bf16", _normal_all(3), 1.0, math.sqrt(1e-5),
                         0.5, 1.0, audit_frac=0.05),
}

# the FFN-up layer of the LLM workload alone (profiling case: 247 MB of
# inputs, larger than L2, a few hundred MB on the device)
WORKLOADS["llm_ffn_up_bf16"] = Workload("llm_ffn_up_bf16", 5, ((4096, 11008),), 16, 512, "bf16",
                                        _normal_all(1), 1.0, math.sqrt(1e-5), 0.5, 1.0,
                                        audit_frac=0.05)

# The paper's LoRA fine-tuning shapes (table of forged-gradient experiment
# parameters, App. B): GPT-2-medium (24 blocks, d = 1024) with rank-4 adapters
# on the fused QKV projection 1024 -> 3072, and RoBERTa-large (24 blocks,
# d = 1024) with rank-8 adapters on the query and value projections.  Each
# adapter is two dense layers: the down factor (d_in x r, inputs = the
# block's hidden states, output gradients of width r) and the up factor
# (r x d_out, inputs of width r).  Seeded N(0,1) activations and N(0,1e-4)
# output gradients stand in for the real ones; C = 1 and the noise
# multipliers are the table's.
def _lora(blocks: int, targets: Sequence[Tuple[int, int]], r: int):
    out = []
    for _ in range(blocks):
        for d_in, d_out in targets:
            out += [(d_in, r), (r, d_out)]
    return tuple(out)


WORKLOADS["gpt2m_lora_e2e_bf16"] = Workload(
    "gpt2m_lora_e2e_bf16", 6, _lora(24, [(1024, 3072)], 4), 64, 128, "bf16",
    _normal_all(48), 1.0, math.sqrt(1e-4), 1.0, 0.6679, audit_frac=0.05)
WORKLOADS["gpt2m_lora_webnlg_bf16"] = Workload(
    "gpt2m_lora_webnlg_bf16", 7, _lora(24, [(1024, 3072)], 4), 32, 256, "bf16",
    _normal_all(48), 1.0, math.sqrt(1e-4), 1.0, 0.6827, audit_frac=0.05)
WORKLOADS["roberta_l_lora_mnli_bf16"] = Workload(
    "roberta_l_lora_mnli_bf16", 8, _lora(24, [(1024, 1024), (1024, 1024)], 8), 256, 128,
    "bf16", _normal_all(96), 1.0, math.sqrt(1e-4), 1.0, 0.6407, audit_frac=0.05)
# one RoBERTa-large block's query and value adapters alone (profiling case for
# the thin-layer kernels: 270 MB of inputs, larger than L2)
WORKLOADS["roberta_l_lora_block_bf16"] = Workload(
    "roberta_l_lora_block_bf16", 10, _lora(1, [(1024, 1024), (1024, 1024)], 8), 256, 128,
    "bf16", _normal_all(4), 1.0, math.sqrt(1e-4), 1.0, 0.6407, audit_frac=0.05)
# ... with the trainable classification head of a 3-class task (MNLI): dense
# 1024 x 1024 and its bias, out_proj 1024 x 3 and its bias, all applied to the
# first token only (T = 1); a bias row is a layer with d_in = 1 and ones as A
_HEAD = ((1024, 1024), (1, 1024), (1024, 3), (1, 3))
WORKLOADS["roberta_l_lora_head_mnli_bf16"] = Workload(
    "roberta_l_lora_head_mnli_bf16", 9, _lora(24, [(1024, 1024), (1024, 1024)], 8) + _HEAD,
    256, 128, "bf16", _normal_all(96) + ("normal", "ones", "normal", "ones"), 1.0,
    math.sqrt(1e-4), 1.0, 0.6407, audit_frac=0.05, layer_T=(128,) * 96 + (1, 1, 1, 1))

def conv_out(H: int, k: int, stride: int, pad: int) -> int:
    return (H + 2 * pad - k) // stride + 1


def _conv_net(specs, head=()):
    """Dense forms, per-layer T and geometries of a list of convolutions
    (H, C_in, C_out, k, stride) on square inputs with pad k // 2, followed by
    dense head layers (d_in, d_out, T)."""
    layers, Ts, convs = [], [], []
    for H, cin, cout, k, st in specs:
        pad = k // 2
        Ho = conv_out(H, k, st, pad)
        layers.append((k * k * cin, cout))
        Ts.append(Ho * Ho)
        convs.append((H, H, cin, k, k, st, pad))
    for d_in, d_out, T in head:
        layers.append((d_in, d_out))
        Ts.append(T)
        convs.append(None)
    return tuple(layers), tuple(Ts), tuple(convs)


# WideResNet-16-4 on CIFAR-10 (App. B): 32x32x3 images, a 3x3 stem to 16
# channels, three groups of two basic blocks of widths 64, 128, 256 (the
# first block of groups 2 and 3 strides by 2; a 1x1 convolution is the
# shortcut where the width changes), then the 256 -> 10 classifier and its
# bias on the pooled features (T = 1).  The normalisation layers' scale and
# shift are not part of it: their per-example gradients are per-channel dot
# products, not dense products.  Batch 2048 in one pass (the paper's batch;
# it trains it as 4 micro-batches of 512), C = 1, sigma from the
# accountant for epsilon = 2, delta = 1e-5, 5000 steps at q = 2048/40000.
_WRN = [(32, 3, 16, 3, 1),
        (32, 16, 64, 3, 1), (32, 64, 64, 3, 1), (32, 16, 64, 1, 1),
        (32, 64, 64, 3, 1), (32, 64, 64, 3, 1),
        (32, 64, 128, 3, 2), (16, 128, 128, 3, 1), (32, 64, 128, 1, 2),
        (16, 128, 128, 3, 1), (16, 128, 128, 3, 1),
        (16, 128, 256, 3, 2), (8, 256, 256, 3, 1), (16, 128, 256, 1, 2),
        (8, 256, 256, 3, 1), (8, 256, 256, 3, 1)]
_wl, _wT, _wc = _conv_net(_WRN, head=((256, 10, 1), (1, 10, 1)))
WORKLOADS["wrn16_4_cifar10_bf16"] = Workload(
    "wrn16_4_cifar10_bf16", 11, _wl, 2048, 1024, "bf16",
    ("normal",) + ("relu_normal",) * 16 + ("ones",), 1.0, math.sqrt(1e-4), 1.0, 9.11,
    audit_frac=0.05, layer_T=_wT, convs=_wc)
# its first group alone at the paper's micro-batch of 512 (profiling case)
_gl, _gT, _gc = _conv_net(_WRN[1:6])
WORKLOADS["wrn16_4_group1_bf16"] = Workload(
    "wrn16_4_group1_bf16", 12, _gl, 512, 1024, "bf16", ("relu_normal",) * 5, 1.0,
    math.sqrt(1e-4), 1.0, 9.11, audit_frac=0.05, layer_T=_gT, convs=_gc)

# one 4096x4096 bf16 layer over B x T
SWEEP = [Workload(f"sweep_B{b}_T{t}", 100 + 10 * bi + ti, ((4096, 4096),), b, t,
                  "bf16", _normal_all(1), 1.0, 1.0, 1.0, 1.0)
         for bi, b in enumerate((8, 32, 128)) for ti, t in enumerate((1, 64, 512, 2048))]


def get(name: str) -> Workload:
    if name in WORKLOADS:
        return WORKLOADS[name]
    for w in SWEEP:
        if w.name == name:
            return w
    raise KeyError(name)


def custom(name: str, layers: Sequence[Sequence[int]], B: int, T: int, dtype: str,
           C: float = 1.0, sigma: float = 1.0, a_std: float = 1.0, d_std: float = 1.0,
           wid: int = 999, a_dist=None) -> Workload:
    """An ad-hoc workload (tests use these for ragged and edge shapes).  A
    layer is (d_in, d_out) or (d_in, d_out, T)."""
    a_dist = tuple(a_dist) if a_dist else _normal_all(len(layers))
    lt = tuple(int(x[2]) if len(x) > 2 else T for x in layers)
    return Workload(name, wid, tuple((int(x[0]), int(x[1])) for x in layers), B, T, dtype,
                    a_dist, a_std, d_std, C, sigma,
                    layer_T=lt if any(t != T for t in lt) else ())


def custom_conv(name: str, convs: Sequence[Sequence[int]], B: int, dtype: str, C: float = 1.0,
                sigma: float = 1.0, d_std: float = 1.0, wid: int = 999, a_dist=None,
                head: Sequence[Sequence[int]] = ()) -> Workload:
    """An ad-hoc convolution workload: convolutions (H, W, C_in, C_out, kh,
    kw, stride, pad), then dense head layers (d_in, d_out, T)."""
    layers, Ts, cv = [], [], []
    for H, W_, cin, cout, kh, kw, st, pd in convs:
        Ho, Wo = (H + 2 * pd - kh) // st + 1, (W_ + 2 * pd - kw) // st + 1
        layers.append((kh * kw * cin, cout))
        Ts.append(Ho * Wo)
        cv.append((H, W_, cin, kh, kw, st, pd))
    for d_in, d_out, T in head:
        layers.append((d_in, d_out))
        Ts.append(T)
        cv.append(None)
    a_dist = tuple(a_dist) if a_dist else _normal_all(len(layers))
    return Workload(name, wid, tuple(layers), B, max(Ts), dtype, a_dist, 1.0, d_std, C, sigma,
                    layer_T=tuple(Ts), convs=tuple(cv))


def _draw(rng: np.random.Generator, dist: str, shape, std: float) -> np.ndarray:
    if dist == "normal":
        x = rng.standard_normal(shape, dtype=np.float32)
    elif dist == "uniform":
        x = rng.random(shape, dtype=np.float32)
    elif dist == "relu_normal":
        x = rng.standard_normal(shape, dtype=np.float32)
        np.maximum(x, np.float32(0.0), out=x)
    elif dist == "ones":  # the input of a bias row
        return np.ones(shape, dtype=np.float32)
    else:
        raise ValueError(dist)
    if std != 1.0:
        x *= np.float32(std)
    return x


def _to_dtype(x: np.ndarray, dtype: str) -> torch.Tensor:
    t = torch.from_numpy(x)
    if dtype == "bf16":
        return t.to(torch.bfloat16)
    if dtype == "f32":
        return t
    raise ValueError(dtype)


def make_layer(w: Workload, layer: int, seed: int = 0, B: int | None = None):
    """(A, D) CPU tensors of layer ``layer`` in the workload's dtype.

    ``B`` may ask for only the first B examples (the draws of example i do not
    depend on how many examples are drawn after it only when B is the full
    batch, so callers that sample examples pass the full B)."""
    B = w.B if B is None else B
    d_in, d_out = w.layers[layer]
    T = w.T_of(layer)
    ra = np.random.default_rng(np.random.SeedSequence([seed, w.wid, layer, 0]))
    rd = np.random.default_rng(np.random.SeedSequence([seed, w.wid, layer, 1]))
    cv = w.conv_of(layer)
    a_shape = (B, cv[0], cv[1], cv[2]) if cv else (B, T, d_in)
    A = _draw(ra, w.a_dist[layer], a_shape, w.a_std)
    D = _draw(rd, "normal", (B, T, d_out), w.d_std)
    return _to_dtype(A, w.dtype), _to_dtype(D, w.dtype)


def make_inputs(w: Workload, seed: int = 0) -> List[Tuple[torch.Tensor, torch.Tensor]]:
    return [make_layer(w, l, seed) for l in range(len(w.layers))]


def audit_indices(w: Workload, seed: int = 0, frac: float | None = None) -> np.ndarray:
    """ceil(frac * B) distinct example indices (sorted), drawn with kind 2;
    frac defaults to the workload's audit fraction, else 5%.

    In the paper the TEE picks what to audit from hidden randomness; here the
    caller's seeded draw stands in for it."""
    if frac is None:
        frac = w.audit_frac if w.audit_frac > 0 else 0.05
    k = max(1, math.ceil(frac * w.B)) if frac > 0 else w.B
    rng = np.random.default_rng(np.random.SeedSequence([seed, w.wid, 0, 2]))
    return np.sort(rng.choice(w.B, size=min(k, w.B), replace=False)).astype(np.int32)


def to_f64(t: torch.Tensor) -> np.ndarray:
    """Exact upcast of fp32 / bf16 tensor values to a float64 numpy array."""
    return t.detach().cpu().to(torch.float64).numpy()
