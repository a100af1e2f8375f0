"""Plain CPU oracle for the Muon step -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s baseline legs may import this
module. The CUDA path never imports, links or calls it, and it shares no code with the CUDA path.

What it computes: Alg. "Muon" of the paper (momentum orthogonalized by Newton-Schulz, with
decoupled weight decay), literally, step by step:

  M <- beta1 M + (1 - beta1) G                          (momentum EMA)
  X_0 = M / max(||M||_F, eps)                           (normalised momentum)
  for i = 1..n:  A = X X^T,  B = b_i A + c_i A^2,  X <- a_i X + B X
  dW = X_n * sqrt(max(in, out))                         (update RMS matching)
  W <- (1 - lr * wd) W - lr * dW                        (decoupled weight decay)

The coefficient schedule {(a_i, b_i, c_i)} is an input (the paper's schedule is published
elsewhere and not restated here).

Readings of points the paper leaves open:
  * Orientation: the algorithm forms X X^T as printed, whatever the shape. An odd polynomial
    step satisfies (a + b X X^T + c (X X^T)^2) X = X (a + b X^T X + c (X^T X)^2), so the
    result does not depend on the orientation; a faster implementation may work on the
    transpose of a tall matrix.
  * Precision: the paper runs the Newton-Schulz iterations in bf16 (products of bf16 operands
    accumulated in fp32). ``ns_bf16=True`` rounds X_0 and every product's result to bf16 at
    the points a bf16 implementation stores them (X_0, A, B, X_i); the default is plain fp64.
    The momentum and the weight update stay in the state's precision.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


@dataclass
class MuonParams:
    """Hyper-parameters of Alg. Muon and its table (beta1 0.9, wd 0.1, n 16, eps 1e-7)."""
    lr: float = 3e-3
    beta1: float = 0.9
    weight_decay: float = 0.1
    eps: float = 1e-7
    coeffs: list = field(default_factory=list)  # [(a_i, b_i, c_i)] for i = 1..n
    ns_bf16: bool = False


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round an array to the nearest bfloat16 value (ties to even), returned as float64.

    bfloat16 keeps the top 16 bits of the float32 encoding; the rounding adds half of the
    dropped part (plus the kept part's lowest bit, for ties to even) before truncating."""
    f = np.asarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32).astype(np.float64)
    return np.where(np.isfinite(f), out, f.astype(np.float64))


def newton_schulz(M: np.ndarray, coeffs, eps: float, bf16: bool = False) -> np.ndarray:
    """X_n of Alg. Muon's orthogonalization from the momentum M (fp64 arithmetic; with
    ``bf16`` the stored intermediates are rounded to bfloat16)."""
    rnd = bf16_round if bf16 else (lambda a: a)
    M = np.asarray(M, dtype=np.float64)
    X = rnd(M / max(np.linalg.norm(M), eps))
    for a, b, c in coeffs:
        A = rnd(X @ X.T)
        B = rnd(b * A + c * (A @ A))
        X = rnd(a * X + B @ X)
    return X


@dataclass
class MuonState:
    """Per-matrix state of Alg. Muon: the momentum M (rows x cols, zero at t = 0) and the step count."""
    rows: int
    cols: int
    dtype: type = np.float64
    t: int = 0
    M: np.ndarray = field(default=None)

    def __post_init__(self):
        if self.M is None:
            self.M = np.zeros((self.rows, self.cols), self.dtype)


def muon_step(st: MuonState, W: np.ndarray, G: np.ndarray, hp: MuonParams):
    """One step of Alg. Muon for one matrix. Mutates ``st``; returns (W_new, dW)."""
    d = st.dtype
    W = np.asarray(W, dtype=d)
    G = np.asarray(G, dtype=d)
    st.t += 1
    st.M = d(hp.beta1) * st.M + d(1 - hp.beta1) * G
    O = newton_schulz(st.M, hp.coeffs, hp.eps, hp.ns_bf16)
    dW = (O * np.sqrt(max(st.rows, st.cols))).astype(d)
    return (d(1 - hp.lr * hp.weight_decay) * W - d(hp.lr) * dW), dW
