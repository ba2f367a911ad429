"""Trusted-side verification of a committed DP-SGD gradient (Algorithm 1,
Sec. 6.2) and of the audit records the GPU step emits.

This is the CPU side of the protocol, not part of the GPU path. A trusted
host (the TEE of the paper) holds the batch, receives the GPU's committed
clipped average g_GPU = (1/B) sum_i c_i G_i (``dp_clipped_sum_noise`` with
``DP_NO_NOISE`` and out_scale = 1/B) and decides Accept or Abort:

* every step: the structural bound ||g_GPU||_2 <= C (1 + slack), since an
  average of vectors of norm <= C has norm <= C (slack 1e-4 covers fp32
  rounding of the norm);
* with a secret coin V_t ~ Bernoulli(p) the step is checked: the host
  recomputes the clipped average in fp32, z32 = ||g_GPU - g32|| / C;
  - body path, z32 <= tau_abs: the discrepancy is charged to the ledger
    Z_sub (abort once Z_sub > K_sub);
  - otherwise the host recomputes in fp64, n_t = (B / 2C) ||g_GPU - g64||
    (equivalently z64 = ||g_GPU - g64|| / C against rho_amb = 2 tau_num / B);
    n_t > tau_num aborts (hard rejection), else the accepted fallback is
    counted in S_amb (abort once S_amb > K_amb);
  - families without the fp64 layer (CIFAR-10 in the paper's table) accept an
    escalated step only under the same-metric cap z32 <= rho_ill = 2 tau_abs,
    counted by the same K_amb counter.

The recomputation follows the paper's statement of DP-SGD (Sec. 2.2): per-
example squared norms of every layer (Gram form, which is the same number as
the Frobenius norm of A_i^T D_i), s_i = sum over layers, c_i = 1 if
s_i <= C^2 else C / sqrt(s_i), and the clipped sum A^T diag(c) D, all in the
working precision (numpy BLAS), divided by B.

``check_audit_records`` recomputes, in fp64, only the examples a record set
names (the partial recomputation of Sec. 7) and compares norms, totals and
clip factors with the GPU's records.

The frozen parameters per model family are the paper's table of verifier
parameters at p = 0.1 (App. E).
"""

from __future__ import annotations

import dataclasses
import math
from typing import Callable, Dict, Iterable, List, Optional, Sequence, Tuple

import numpy as np

ACCEPT, ABORT = "accept", "abort"


@dataclasses.dataclass(frozen=True)
class VerifierParams:
    """Thresholds of Algorithm 1.  z-thresholds are in clipping-norm units.

    tau_num is in the accountant's units (times B / 2C); rho_amb = 2 tau_num
    / B.  fp64_layer = False selects the same-metric cap rho_ill instead of
    the fp64 escalation."""
    p: float
    tau_abs: float
    K_sub: float
    K_amb: int
    tau_num: Optional[float] = None
    rho_ill: Optional[float] = None
    slack: float = 1e-4
    fp64_layer: bool = True

    def rho_amb(self, B: int) -> float:
        if self.tau_num is None:
            raise ValueError("no fp64 layer: this family has no tau_num")
        return 2.0 * self.tau_num / B


# The paper's frozen verifier parameters per model family (table of verifier
# parameters, App. E).  GPT-2's tau_num is stated for B = 64 (0.0783 at
# B = 32); CIFAR-10 has no fp64 layer and caps at rho_ill = 2 tau_abs.
FAMILIES: Dict[str, VerifierParams] = {
    "roberta": VerifierParams(p=0.1, tau_abs=1.60e-3, K_sub=0.088, K_amb=25, tau_num=1.5169),
    "gpt2": VerifierParams(p=0.1, tau_abs=1.74e-3, K_sub=0.72, K_amb=17, tau_num=0.1565),
    "cifar10": VerifierParams(p=0.1, tau_abs=7.30e-4, K_sub=0.20, K_amb=5, rho_ill=1.459e-3,
                              fp64_layer=False),
}


# ---------------------------------------------------------------------------
# trusted recomputation of the committed clipped average
# ---------------------------------------------------------------------------

def _as(x, dtype):
    """Host array of the stored input values in the working precision (the
    stored bf16 / fp32 bits are exact in both fp32 and fp64)."""
    if hasattr(x, "detach"):  # a torch tensor: read its stored values
        x = x.detach().to("cpu")
        if str(x.dtype) == "torch.bfloat16":
            x = x.float()
        x = x.numpy()
    return np.asarray(x).astype(dtype, copy=False)


def per_example_sqnorms(A, D, dtype=np.float64) -> np.ndarray:
    """n_i = ||A_i^T D_i||_F^2 for every example of one layer, in Gram form:
    sum_{t,s} (A_i A_i^T)_{ts} (D_i D_i^T)_{ts}.  A [B,T,d_in], D [B,T,d_out]."""
    A = _as(A, dtype)
    D = _as(D, dtype)
    if A.ndim == 2:
        A, D = A[:, None, :], D[:, None, :]
    ga = np.matmul(A, np.swapaxes(A, 1, 2))
    gd = np.matmul(D, np.swapaxes(D, 1, 2))
    return np.einsum("bts,bts->b", ga, gd).astype(dtype, copy=False)


def clip_factors(s: np.ndarray, C: float) -> np.ndarray:
    """c_i = 1 if s_i <= C^2 (including s_i = 0), else C / sqrt(s_i), in the
    precision of s."""
    s = np.asarray(s)
    C = s.dtype.type(C)
    with np.errstate(divide="ignore", invalid="ignore"):
        c = np.where(s <= C * C, s.dtype.type(1), C / np.sqrt(s))
    return c.astype(s.dtype, copy=False)


def recompute_average(layers: Sequence[Tuple[object, object]], C: float, dtype=np.float64
                      ) -> Tuple[List[np.ndarray], np.ndarray, np.ndarray]:
    """The prescribed clipped average (1/B) A^T diag(c) D of every layer in
    the working precision (np.float32 or np.float64).

    layers: (A [B,T,d_in], D [B,T,d_out]) per layer.  Returns (the per-layer
    averages [d_in, d_out], s [B], c [B])."""
    n = np.stack([per_example_sqnorms(A, D, dtype) for A, D in layers])
    s = n.sum(axis=0, dtype=dtype)
    c = clip_factors(s, C)
    out = []
    for A, D in layers:
        A = _as(A, dtype)
        D = _as(D, dtype)
        B = A.shape[0]
        Ac = (A * c[:, None, None]).reshape(-1, A.shape[-1])
        S = Ac.T @ D.reshape(-1, D.shape[-1])
        out.append((S / dtype(B)).astype(dtype, copy=False))
    return out, s, c


def _flat(xs) -> np.ndarray:
    if isinstance(xs, np.ndarray):
        return xs.reshape(-1).astype(np.float64)
    return np.concatenate([_as(x, np.float64).reshape(-1) for x in xs])


# ---------------------------------------------------------------------------
# Algorithm 1
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class StepResult:
    verdict: str              # ACCEPT or ABORT
    path: str                 # structural | unchecked | body | ambiguity | hard_reject | ledger
    z32: Optional[float] = None
    z64: Optional[float] = None
    n_t: Optional[float] = None


class Verifier:
    """One run's verification state: the ledgers Z_sub and S_amb and the
    secret coin stream.  ``coin_seed`` is the trusted side's secret; the GPU
    never sees the coins."""

    def __init__(self, params: VerifierParams, C: float, B: int, coin_seed: int):
        self.params = params
        self.C = float(C)
        self.B = int(B)
        self._coins = np.random.default_rng(coin_seed)
        self.Z_sub = 0.0
        self.S_amb = 0
        self.aborted = False
        self.log: List[StepResult] = []

    def draw_coin(self) -> bool:
        """V_t ~ Bernoulli(p), drawn after the GPU has committed."""
        return bool(self._coins.random() < self.params.p)

    def step(self, g_gpu, recompute32: Callable[[], object],
             recompute64: Optional[Callable[[], object]] = None,
             checked: Optional[bool] = None) -> StepResult:
        """Verify one committed average g_GPU (flat array or list of layer
        arrays).  recompute32 / recompute64 return the host's fp32 / fp64
        recomputation (called only when needed).  ``checked`` overrides the
        coin (for replaying a known schedule)."""
        r = self._step(g_gpu, recompute32, recompute64, checked)
        if r.verdict == ABORT:
            self.aborted = True
        self.log.append(r)
        return r

    def _step(self, g_gpu, recompute32, recompute64, checked) -> StepResult:
        prm, C = self.params, self.C
        g = _flat(g_gpu)
        if not np.all(np.isfinite(g)) or np.linalg.norm(g) > C * (1.0 + prm.slack):
            return StepResult(ABORT, "structural")
        v = self.draw_coin() if checked is None else bool(checked)
        if not v:
            return StepResult(ACCEPT, "unchecked")
        z32 = float(np.linalg.norm(g - _flat(recompute32())) / C)
        if z32 <= prm.tau_abs:
            self.Z_sub += z32
            return StepResult(ABORT if self.Z_sub > prm.K_sub else ACCEPT,
                              "ledger" if self.Z_sub > prm.K_sub else "body", z32=z32)
        if prm.fp64_layer:
            if recompute64 is None:
                raise ValueError("an escalated step needs the fp64 recomputation")
            z64 = float(np.linalg.norm(g - _flat(recompute64())) / C)
            n_t = self.B / 2.0 * z64
            if n_t > prm.tau_num:
                return StepResult(ABORT, "hard_reject", z32=z32, z64=z64, n_t=n_t)
            self.S_amb += 1
            return StepResult(ABORT if self.S_amb > prm.K_amb else ACCEPT,
                              "ledger" if self.S_amb > prm.K_amb else "ambiguity",
                              z32=z32, z64=z64, n_t=n_t)
        if z32 > prm.rho_ill:
            return StepResult(ABORT, "hard_reject", z32=z32)
        self.S_amb += 1
        return StepResult(ABORT if self.S_amb > prm.K_amb else ACCEPT,
                          "ledger" if self.S_amb > prm.K_amb else "ambiguity", z32=z32)


# ---------------------------------------------------------------------------
# audit records (partial recomputation of the emitted per-example values)
# ---------------------------------------------------------------------------

@dataclasses.dataclass
class AuditReport:
    ok: bool
    max_rel_norm: float          # largest relative error of n_{l,i}
    max_rel_total: float         # of s_i
    max_rel_clip: float          # of c_i
    examples: List[int]


def check_audit_records(records, layers: Sequence[Tuple[object, object]], C: float,
                        rtol: float) -> AuditReport:
    """Recompute, in fp64, the examples named by ``records`` (a structured
    array with fields example, total_sqnorm, clip_factor, layer_sqnorm, as
    returned by the binding's dp_audit_emit) and compare elementwise with
    relative tolerance rtol.  The record's own c_i must also follow from its
    own s_i (c_i = min(1, C / sqrt(s_i)) to rtol)."""
    idx = [int(i) for i in records["example"]]
    if not idx:
        return AuditReport(True, 0.0, 0.0, 0.0, [])
    sub = [(_as(A, np.float64)[idx], _as(D, np.float64)[idx]) for A, D in layers]
    n = np.stack([per_example_sqnorms(A, D, np.float64) for A, D in sub])  # [L, n]
    s = n.sum(axis=0)
    c = clip_factors(s, C)

    def rel(got, ref):
        got = np.asarray(got, np.float64)
        return float(np.max(np.abs(got - ref) / np.maximum(np.abs(ref), 1e-300))) if got.size else 0.0

    rn = rel(np.asarray(records["layer_sqnorm"], np.float64).T, n)
    rs = rel(records["total_sqnorm"], s)
    rc = rel(records["clip_factor"], c)
    own = clip_factors(np.asarray(records["total_sqnorm"], np.float64), C)
    r_own = rel(records["clip_factor"], own)
    ok = (rn <= rtol and rs <= rtol and rc <= rtol and r_own <= rtol
          and bool(np.all(np.asarray(records["clip_factor"]) <= 1.0)))
    return AuditReport(ok, rn, rs, max(rc, r_own), idx)
