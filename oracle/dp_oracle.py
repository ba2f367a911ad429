"""fp64 CPU oracle of the DP-SGD gradient step for dense layers.

TEST INFRASTRUCTURE ONLY -- see ``oracle/__init__.py``.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py`` (its ``cpu_baseline`` leg and its
``--impl reference`` arm) may import it.  It is slow on purpose: every
quantity is its plain definition, in the order the paper states it.

What is computed (paper: Sec. 2.2 "DP-SGD", and the GPU loop of Algorithm 2):

* per-example gradient of a dense layer with activations ``A_i`` [T, d_in]
  and output gradients ``D_i`` [T, d_out]:  ``G_i = A_i^T D_i``  (the
  gradient ``g_t(x_i)`` of Sec. 2.2 restricted to one weight matrix, laid out
  [d_in, d_out]);
* per-example squared L2 norm over all layers ``s_i = sum_l ||G_{i,l}||_F^2``;
* clip factor ``c_i = min(1, C / ||g_i||_2)``  (Sec. 2.2 clipping equation;
  Algorithm 2, the per-example clip);
* clipped sum ``S_l = sum_i c_i G_{i,l}`` -- the commitment of Algorithm 2
  before the 1/B average;
* Gaussian noise ``z ~ N(0, sigma^2 C^2 I)`` drawn from a counter-based
  generator keyed by (seed, step) and indexed by the global parameter offset
  (``Noise(s_noise_t; sigma C)`` of Algorithms 2 and 3; the paper does not name
  the generator, so this oracle fixes Philox4x32-10 from Salmon et al., SC'11,
  and Box--Muller, 1958);
* output ``out_l = out_scale * (S_l + sigma*C*z_l)``; ``out_scale = 1/B`` is the
  paper's average ``(1/|B_t|)(sum + z)`` of Sec. 2.2, ``out_scale = 1`` the
  plain sum;
* per-example weight gradients of 2-D convolutions (the CIFAR-10 WideResNet
  of App. B) from the definition of the convolution, and the patch rows
  (unfold) that turn a convolution into the dense form above; the step on
  per-example gradients given directly (:func:`dp_step_from_grads`);
* audit records (example, per-layer squared norms, total, clip factor) for a
  caller-chosen subset of examples, the material a CPU checker recomputes when
  it partially re-executes a step (Sec. 7, "recomputes, or partially
  recomputes");
* the update that follows the seed release in Algorithm 2,
  g~ = committed average + (1/B) Noise(s; sigma C), then OptStep = AdamW as the
  paper writes its one-step map (App. A): m = b1 m + (1-b1) g,
  v = b2 v + (1-b2) g*g, bias corrections 1 - b^t, and
  theta <- theta - lr (m^/(sqrt(v^) + eps) + wd theta).

Readings where the paper is silent (each also listed with its reason in the
design notes): c_i = 1 when s_i <= C^2, including s_i = 0; no stabiliser
epsilon in C/||g||; non-finite inputs raise; the uint32 -> uniform mapping of
:func:`uniforms_from_words`; noise word order of :func:`gaussian_noise`.

Pins (tests/test_oracle_pins.py, all ``-m "not gpu"``):

* per_example_grads / layer_sqnorms: pure-Python triple-loop brute force on
  tiny inputs; rank-1 closed form ||a||^2 ||d||^2 at T = 1; ghost (Gram)
  identity equals the materialised norm.
* clip_factors: invariants ||c_i g_i|| <= C(1+1e-6), c_i in (0, 1]; the
  scaled-example law c(lambda D_i) = c(D_i)/lambda once clipped; the zero and
  tie special cases; aggregate ||S/B|| <= C(1+1e-4) (Sec. 6.2 structural check).
* clipped_sum: C -> infinity reduces it to the textbook product
  reshape(A)^T reshape(D) (numpy.matmul); linearity in c.
* philox4x32_10: bit-exact against PyTorch's independent C++ implementation
  (``at::philox_engine``) compiled from its header; counter/key sensitivity.
* uniforms_from_words: hand-derived edge values (tests/golden/uniform_edges.json).
* box_muller: the identities z0^2 + z1^2 = -2 ln u0, atan2(z1, z0) = 2 pi u1.
* adamw_step: pure-Python scalar loop of the App. A equations; the t = 1 and
  b1 = b2 = 0 special cases where the step is lr (g/(|g| + eps) + wd theta)
  (tests/golden/adamw_hand.json, worked by hand); g = 0 leaves theta
  changed by weight decay only.
* conv2d_weight_grads: a pure-Python six-fold loop on tiny inputs; PyTorch's
  independent ``torch.nn.grad.conv2d_weight`` per example (NCHW, strides and
  padding); a 1x1 stride-1 convolution is the dense layer on the pixels.
* conv2d_unfold: ``torch.nn.functional.unfold`` with its (c, ki, kj) column
  order permuted; hand-placed values including the zero padding; its dense
  product equals conv2d_weight_grads.
* dp_step_from_grads: equals dp_step on dense layers.
* gaussian_noise: sample mean / variance / Kolmogorov-Smirnov against
  N(0, 1); per-coordinate std of the averaged noise against the sigma*C/B
  column printed in the paper's attack-parameter table (App. B.1).
"""

from __future__ import annotations

import math
from typing import Sequence

import numpy as np

__all__ = [
    "per_example_grads",
    "layer_sqnorms_materialised",
    "layer_sqnorms_ghost",
    "layer_sqnorms",
    "clip_factors",
    "clipped_sum",
    "philox4x32_10",
    "philox_quads",
    "uniforms_from_words",
    "box_muller",
    "sincospi",
    "gaussian_noise",
    "dp_step",
    "dp_step_from_grads",
    "conv2d_out_hw",
    "conv2d_weight_grads",
    "conv2d_unfold",
    "audit_records",
    "adamw_step",
    "noise_adamw",
    "PHILOX_M0",
    "PHILOX_M1",
    "PHILOX_W0",
    "PHILOX_W1",
]


def _as_f64(x) -> np.ndarray:
    a = np.asarray(x, dtype=np.float64)
    if not np.all(np.isfinite(a)):
        # Reading: the paper defines no behaviour for non-finite gradients;
        # the oracle refuses them instead of propagating NaN.
        raise ValueError("non-finite input to the DP-SGD oracle")
    return a


# ---------------------------------------------------------------------------
# Per-example gradients and their norms (Sec. 2.2; Algorithm 2 inner loop)
# ---------------------------------------------------------------------------

def per_example_grads(A, D) -> np.ndarray:
    """G_i = A_i^T D_i for every example i.

    A: [B, T, d_in], D: [B, T, d_out] -> G: [B, d_in, d_out] (fp64).
    A dense layer y_t = W^T a_t summed over the T positions of one example has
    weight gradient sum_t a_t d_t^T, the per-example gradient g_t(x_i) of
    Sec. 2.2 for that weight matrix.
    """
    A = _as_f64(A)
    D = _as_f64(D)
    if A.ndim != 3 or D.ndim != 3 or A.shape[:2] != D.shape[:2]:
        raise ValueError("A and D must be [B, T, d] with matching B, T")
    B = A.shape[0]
    G = np.empty((B, A.shape[2], D.shape[2]), dtype=np.float64)
    for i in range(B):
        G[i] = A[i].T @ D[i]
    return G


def layer_sqnorms_materialised(A, D) -> np.ndarray:
    """n_i = ||A_i^T D_i||_F^2, with the per-example gradient materialised."""
    A = _as_f64(A)
    D = _as_f64(D)
    B = A.shape[0]
    n = np.empty(B, dtype=np.float64)
    for i in range(B):
        G = A[i].T @ D[i]
        n[i] = np.sum(G * G)
    return n


def layer_sqnorms_ghost(A, D) -> np.ndarray:
    """n_i = sum_{t,s} (a_t . a_s)(d_t . d_s) = <A_i A_i^T, D_i D_i^T>_F.

    The same number as the materialised norm: ||sum_t a_t d_t^T||_F^2 expands
    to sum_{t,s} (a_t^T a_s)(d_t^T d_s).  The oracle keeps it only as an
    internal cross-check of :func:`layer_sqnorms_materialised`.
    """
    A = _as_f64(A)
    D = _as_f64(D)
    B = A.shape[0]
    n = np.empty(B, dtype=np.float64)
    for i in range(B):
        GA = A[i] @ A[i].T
        GD = D[i] @ D[i].T
        n[i] = np.sum(GA * GD)
    return n


def layer_sqnorms(A, D) -> np.ndarray:
    """The oracle's per-example squared norm of one layer (materialised)."""
    return layer_sqnorms_materialised(A, D)


# ---------------------------------------------------------------------------
# Clip factors (Sec. 2.2 clipping equation; Algorithm 2)
# ---------------------------------------------------------------------------

def clip_factors(n_layers, C: float):
    """s_i = sum_l n_{l,i};  c_i = min(1, C / sqrt(s_i)).

    n_layers: [L, B] per-layer squared norms.  Returns (s [B], c [B]).
    Readings: c_i = 1 whenever s_i <= C^2 (this covers s_i = 0, where
    C/||g|| is undefined but any factor leaves the zero gradient unchanged,
    and the tie ||g_i|| = C); no stabilising epsilon is added to the norm.
    """
    n = _as_f64(n_layers)
    if n.ndim == 1:
        n = n[None, :]
    if not C > 0:
        raise ValueError("clip norm C must be positive")
    s = np.sum(n, axis=0)
    c = np.ones_like(s)
    big = s > C * C
    c[big] = C / np.sqrt(s[big])
    return s, c


# ---------------------------------------------------------------------------
# Clipped sum (Algorithm 2: sum of the clipped per-example gradients)
# ---------------------------------------------------------------------------

def clipped_sum(A, D, c) -> np.ndarray:
    """S = sum_i c_i A_i^T D_i  ([d_in, d_out], fp64), no noise.

    This is B times the committed average gradient of Algorithm 2.
    """
    A = _as_f64(A)
    D = _as_f64(D)
    c = _as_f64(c)
    S = np.zeros((A.shape[2], D.shape[2]), dtype=np.float64)
    for i in range(A.shape[0]):
        S += c[i] * (A[i].T @ D[i])
    return S


# ---------------------------------------------------------------------------
# Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) -- the counter-based
# generator used for Noise(s; sigma C); the paper names none.
# ---------------------------------------------------------------------------

PHILOX_M0 = 0xD2511F53  # round multiplier for counter word 0
PHILOX_M1 = 0xCD9E8D57  # round multiplier for counter word 2
PHILOX_W0 = 0x9E3779B9  # Weyl increment of key word 0 (golden ratio)
PHILOX_W1 = 0xBB67AE85  # Weyl increment of key word 1 (sqrt(3) - 1)
_MASK32 = np.uint64(0xFFFFFFFF)


def philox4x32_10(ctr: Sequence, key: Sequence):
    """Ten Philox rounds on 4x32-bit counters with a 2x32-bit key.

    ctr: four uint32 arrays (broadcastable), key: two uint32 scalars or arrays.
    One round maps (x0, x1, x2, x3) to
        (hi(M1*x2) ^ x1 ^ k0,  lo(M1*x2),  hi(M0*x0) ^ x3 ^ k1,  lo(M0*x0))
    and the key is bumped by the Weyl constants between rounds.
    Returns four uint32 arrays.
    """
    x = [np.asarray(w, dtype=np.uint64) & _MASK32 for w in ctr]
    k0 = np.asarray(key[0], dtype=np.uint64) & _MASK32
    k1 = np.asarray(key[1], dtype=np.uint64) & _MASK32
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    for rnd in range(10):
        if rnd:
            k0 = (k0 + np.uint64(PHILOX_W0)) & _MASK32
            k1 = (k1 + np.uint64(PHILOX_W1)) & _MASK32
        p0 = m0 * x[0]          # < 2^64, exact in uint64
        p1 = m1 * x[2]
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK32
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK32
        x = [hi1 ^ x[1] ^ k0, lo1, hi0 ^ x[3] ^ k1, lo0]
    return [w.astype(np.uint32) for w in x]


def philox_quads(seed: int, step: int, first_quad: int, n_quads: int) -> np.ndarray:
    """Philox blocks for quads q = first_quad .. first_quad+n_quads-1.

    Key = (lo32(seed), hi32(seed)); counter = (lo32(q), hi32(q), lo32(step),
    hi32(step)).  Reading of Derive(s_noise, t) in Algorithm 3: the per-step
    stream is the generator evaluated with the step in the upper counter words,
    so every (seed, step) pair owns its own 2^64-quad stream.
    Returns uint32 [n_quads, 4].
    """
    q = np.arange(n_quads, dtype=np.uint64) + np.uint64(first_quad)
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    step = int(step) & 0xFFFFFFFFFFFFFFFF
    ctr = (q & _MASK32, q >> np.uint64(32),
           np.uint64(step & 0xFFFFFFFF), np.uint64(step >> 32))
    key = (seed & 0xFFFFFFFF, seed >> 32)
    w = philox4x32_10(ctr, key)
    return np.stack(w, axis=1)


def uniforms_from_words(x_even, x_odd):
    """Map one pair of uint32 words to the Box--Muller uniforms (fp32 values).

    u0 = RN_fp32((x_even + 1) / 2^32)  in (0, 1]   (never 0, so ln u0 is finite)
    u1 = RN_fp32(x_odd / 2^32)         in [0, 1]
    Both are round-to-nearest-even fp32 numbers of an exact rational; the
    GPU computes the same fp32 values, so the comparison of the Gaussians does
    not depend on how either side rounds the integers.
    Returns fp64 arrays holding those fp32 values.
    """
    xe = np.asarray(x_even, dtype=np.float64)       # exact: < 2^53
    xo = np.asarray(x_odd, dtype=np.float64)
    u0 = ((xe + 1.0) * 2.0 ** -32).astype(np.float32).astype(np.float64)
    u1 = (xo * 2.0 ** -32).astype(np.float32).astype(np.float64)
    return u0, u1


def sincospi(x):
    """(sin(pi x), cos(pi x)) in fp64 with exact argument reduction.

    x is split as x = y + k/2 with |y| <= 1/4 (exact for the fp32-valued
    arguments used here), then the quarter-turn identities
    sin(pi(y + k/2)), cos(pi(y + k/2)) are applied.  This keeps the relative
    accuracy of the result near the zeros of sin and cos.
    """
    x = np.asarray(x, dtype=np.float64)
    k = np.rint(2.0 * x)
    y = x - 0.5 * k
    sy = np.sin(np.pi * y)
    cy = np.cos(np.pi * y)
    q = np.mod(k, 4).astype(np.int64)
    s = np.choose(q, [sy, cy, -sy, -cy])
    c = np.choose(q, [cy, -sy, -cy, sy])
    return s, c


def box_muller(u0, u1):
    """Box & Muller (1958): r = sqrt(-2 ln u0); (r cos 2 pi u1, r sin 2 pi u1)."""
    u0 = np.asarray(u0, dtype=np.float64)
    u1 = np.asarray(u1, dtype=np.float64)
    r = np.sqrt(-2.0 * np.log(u0))
    s, c = sincospi(2.0 * u1)
    return r * c, r * s


def gaussian_noise(seed: int, step: int, first_index: int, n: int) -> np.ndarray:
    """Standard normal draws z_p for global parameter indices p in [first, first+n).

    Parameter p uses Philox quad q = p >> 2 and slot p & 3:
      slots 0, 1 <- Box-Muller of words (x0, x1): (r cos, r sin)
      slots 2, 3 <- Box-Muller of words (x2, x3): (r cos, r sin)
    The global index runs over all layers in the order they were declared
    (layer l starts at the running sum of the earlier d_in*d_out), so the
    noise of a parameter does not depend on tiling, launch shape or layer
    order of the calls.
    """
    if n <= 0:
        return np.zeros(0, dtype=np.float64)
    q0 = first_index >> 2
    q1 = (first_index + n - 1) >> 2
    w = philox_quads(seed, step, q0, q1 - q0 + 1)
    ua0, ua1 = uniforms_from_words(w[:, 0], w[:, 1])
    ub0, ub1 = uniforms_from_words(w[:, 2], w[:, 3])
    z0, z1 = box_muller(ua0, ua1)
    z2, z3 = box_muller(ub0, ub1)
    z = np.stack([z0, z1, z2, z3], axis=1).reshape(-1)
    start = first_index - 4 * q0
    return z[start:start + n].copy()


# ---------------------------------------------------------------------------
# One whole step (Algorithm 2 up to the noisy gradient) and its audit record
# ---------------------------------------------------------------------------

def dp_step(layers, C: float, sigma: float, seed: int, step: int,
            out_scale: float = 1.0, noise: bool = True, norm: str = "materialised"):
    """Run the DP-SGD gradient step over L dense layers.

    layers: sequence of (A [B,T,d_in], D [B,T,d_out]).
    Returns dict with n [L,B], s [B], c [B], S (list of clipped sums) and out
    (list of out_scale * (S + sigma*C*z), or out_scale * S when noise=False).
    """
    fn = layer_sqnorms_materialised if norm == "materialised" else layer_sqnorms_ghost
    n = np.stack([fn(A, D) for A, D in layers])
    s, c = clip_factors(n, C)
    S_list, out = [], []
    offset = 0
    for A, D in layers:
        S = clipped_sum(A, D, c)
        S_list.append(S)
        o = S.copy()
        if noise:
            z = gaussian_noise(seed, step, offset, S.size).reshape(S.shape)
            o = o + sigma * C * z
        out.append(out_scale * o)
        offset += S.size
    return {"n": n, "s": s, "c": c, "S": S_list, "out": out}


def dp_step_from_grads(grads, C: float, sigma: float, seed: int, step: int,
                       out_scale: float = 1.0, noise: bool = True):
    """The same step on per-example gradients given directly.

    grads: sequence of [B, ...] arrays, one per layer (any layer kind whose
    per-example gradient is known, e.g. :func:`conv2d_weight_grads`); each
    layer's parameters are its trailing dimensions in C order, which fixes
    their global noise indices.  n_{l,i} = ||G_{l,i}||^2, then clip, clipped
    sum and noise exactly as :func:`dp_step` (Sec. 2.2, Algorithm 2).
    """
    grads = [_as_f64(G) for G in grads]
    B = grads[0].shape[0]
    if any(G.shape[0] != B for G in grads):
        raise ValueError("every layer needs the same B")
    n = np.stack([np.sum(G.reshape(B, -1) ** 2, axis=1) for G in grads])
    s, c = clip_factors(n, C)
    S_list, out = [], []
    offset = 0
    for G in grads:
        S = np.tensordot(c, G, axes=(0, 0))
        S_list.append(S)
        o = S.copy()
        if noise:
            z = gaussian_noise(seed, step, offset, S.size).reshape(S.shape)
            o = o + sigma * C * z
        out.append(out_scale * o)
        offset += S.size
    return {"n": n, "s": s, "c": c, "S": S_list, "out": out}


# ---------------------------------------------------------------------------
# 2-D convolution layers (the CIFAR-10 WideResNet of App. B)
# ---------------------------------------------------------------------------
# A convolution without bias, NHWC activations x [H, W, C_in] and weight
# W [kh, kw, C_in, C_out]:
#   y[h, w, o] = sum_{ki, kj, c} xp[h*sh + ki, w*sw + kj, c] * W[ki, kj, c, o]
# where xp is x with pad rows / columns of zeros on every side.  Its weight
# gradient for one example is the sum over output positions of the input
# patch times the output gradient.

def conv2d_out_hw(H: int, W: int, kh: int, kw: int, stride=(1, 1), pad=(0, 0)):
    """(H_out, W_out) of the convolution above."""
    sh, sw = stride
    ph, pw = pad
    Ho = (H + 2 * ph - kh) // sh + 1
    Wo = (W + 2 * pw - kw) // sw + 1
    if Ho < 1 or Wo < 1:
        raise ValueError("kernel larger than the padded input")
    return Ho, Wo


def _padded(X, pad):
    ph, pw = pad
    return np.pad(X, ((0, 0), (ph, ph), (pw, pw), (0, 0)))


def conv2d_weight_grads(X, Dy, kh: int, kw: int, stride=(1, 1), pad=(0, 0)) -> np.ndarray:
    """Per-example weight gradients G_i[ki, kj, c, o] = sum_{h, w}
    xp_i[h*sh + ki, w*sw + kj, c] * dy_i[h, w, o].

    X: [B, H, W, C_in], Dy: [B, H_out, W_out, C_out] -> [B, kh, kw, C_in, C_out].
    One contraction per kernel tap (ki, kj) over the output positions.
    """
    X = _as_f64(X)
    Dy = _as_f64(Dy)
    B, H, W_, Cin = X.shape
    Ho, Wo = conv2d_out_hw(H, W_, kh, kw, stride, pad)
    if Dy.shape[:3] != (B, Ho, Wo):
        raise ValueError("Dy must be [B, H_out, W_out, C_out]")
    sh, sw = stride
    Xp = _padded(X, pad)
    G = np.zeros((B, kh, kw, Cin, Dy.shape[3]))
    for ki in range(kh):
        for kj in range(kw):
            tap = Xp[:, ki:ki + sh * (Ho - 1) + 1:sh, kj:kj + sw * (Wo - 1) + 1:sw, :]
            G[:, ki, kj] = np.einsum("bhwc,bhwo->bco", tap, Dy)
    return G


def conv2d_unfold(X, kh: int, kw: int, stride=(1, 1), pad=(0, 0)) -> np.ndarray:
    """Input patches as rows: A[i, h*W_out + w, (ki*kw + kj)*C_in + c] =
    xp_i[h*sh + ki, w*sw + kj, c]  ->  [B, H_out*W_out, kh*kw*C_in].

    With it a convolution's weight gradient is the dense A_i^T D_i of
    :func:`per_example_grads` with D_i = dy_i as [H_out*W_out, C_out], laid out
    [(ki, kj, c), o].  The values are copies of inputs and zeros, so the
    result is exact in any precision.
    """
    X = np.asarray(X)
    B, H, W_, Cin = X.shape
    Ho, Wo = conv2d_out_hw(H, W_, kh, kw, stride, pad)
    sh, sw = stride
    Xp = _padded(X, pad)
    A = np.empty((B, Ho, Wo, kh, kw, Cin), dtype=X.dtype)
    for ki in range(kh):
        for kj in range(kw):
            A[:, :, :, ki, kj, :] = Xp[:, ki:ki + sh * (Ho - 1) + 1:sh,
                                       kj:kj + sw * (Wo - 1) + 1:sw, :]
    return A.reshape(B, Ho * Wo, kh * kw * Cin)


def audit_records(n, s, c, idx):
    """Records (example, n_{1..L}, s, c) for the examples listed in idx."""
    n = np.asarray(n, dtype=np.float64)
    recs = []
    for i in idx:
        i = int(i)
        recs.append({"example": i, "layer_sqnorm": n[:, i].copy(),
                     "total_sqnorm": float(s[i]), "clip_factor": float(c[i])})
    return recs


# ---------------------------------------------------------------------------
# After the seed release: noisy gradient and OptStep = AdamW (Algorithm 2;
# the one-step AdamW map of App. A)
# ---------------------------------------------------------------------------

def adamw_step(theta, m, v, g, lr: float, beta1: float, beta2: float, eps: float,
               weight_decay: float, t: int):
    """One AdamW step at step count t >= 1 (bias corrections 1 - beta^t).

    m' = b1 m + (1 - b1) g;  v' = b2 v + (1 - b2) g*g;
    m^ = m' / (1 - b1^t);    v^ = v' / (1 - b2^t);
    theta' = theta - lr (m^ / (sqrt(v^) + eps) + wd theta).
    Returns (theta', m', v') in fp64."""
    if t < 1:
        raise ValueError("step count t must be >= 1")
    theta = _as_f64(theta)
    m = _as_f64(m)
    v = _as_f64(v)
    g = _as_f64(g)
    m2 = beta1 * m + (1.0 - beta1) * g
    v2 = beta2 * v + (1.0 - beta2) * g * g
    mh = m2 / (1.0 - beta1 ** t)
    vh = v2 / (1.0 - beta2 ** t)
    theta2 = theta - lr * (mh / (np.sqrt(vh) + eps) + weight_decay * theta)
    return theta2, m2, v2


def noise_adamw(committed, theta, m, v, seed: int, step: int, first_index: int,
                sigma: float, C: float, out_scale: float, lr: float, beta1: float,
                beta2: float, eps: float, weight_decay: float, t: int):
    """The GPU's update after the seed is released (Algorithm 2):
    g~ = committed + out_scale * sigma * C * z  (committed = out_scale * S, the
    noiseless commitment), then AdamW.  z uses the parameters' global indices
    first_index .. first_index + size - 1.  Returns (g~, theta', m', v')."""
    committed = _as_f64(committed)
    z = gaussian_noise(seed, step, first_index, committed.size).reshape(committed.shape)
    g = committed + out_scale * sigma * C * z
    th, m2, v2 = adamw_step(theta, m, v, g, lr, beta1, beta2, eps, weight_decay, t)
    return g, th, m2, v2
