"""Plain CPU oracle for one SOAP optimizer step -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s ``cpu_baseline`` /
``--impl reference`` legs may import this module. The CUDA path never imports,
links or calls it, and it shares no code with the CUDA path.

What it computes: the SOAP step of the paper's Alg. 1 ("KL-SOAP used in
experiments"), run literally, step by step, in the order the algorithm gives,
with the Kronecker factors accumulated in the standard Shampoo form of the primer
(section 2, the L_t / R_t equations) using the current gradient (section 5,
"Mitigating Staleness: Real-Time Eigenbasis Updates"):

  S1  L <- b L + (1-b) G G^T,  R <- b R + (1-b) G^T G          (section 2, Shampoo EMAs)
  S4a M_hat = Q_L m Q_R^T            (old basis)                (Alg. 1, re-projection)
  S2  P_L = L Q_L,  P_R = R Q_R                                 (Alg. 1, power step)
  S3  Q_L <- QR(P_L).Q,  Q_R <- QR(P_R).Q, diag(R) >= 0          (Alg. 1; appendix on eigh vs QR)
  S4b m = Q_L^T M_hat Q_R            (new basis)                (Alg. 1, re-projection)
  S5  G' = Q_L^T G Q_R                                          (Alg. 1, rotate gradient)
  S6  m <- b1 m + (1-b1) G',  v <- b2 v + (1-b2) G'*G',  N = m / (sqrt(v) + eps)
                                                                (Alg. 1 Adam block, primer convention)
  S7  dW = Q_L N Q_R^T                                          (Alg. 1, rotate update out)
  S8  W <- (1 - lr*wd) W - lr*dW                                (Alg. 1, weight decay and update)

Readings of points the paper leaves open:
  * EMA convention: the coefficient multiplies the OLD state (primer, section 2).
    Alg. 1 prints (1-beta) old + beta new; with beta = 0.95 for every EMA here the
    primer's form is used.
  * Initial state: L = R = 0, Q = I, m = v = 0, t = 1 on the first call, and the
    first call applies an update (Alg. 1 has no warm-up branch).
  * Only m is re-projected when the basis changes; v is not (Alg. 1).
  * No bias correction unless ``bias_correction`` is set (section 2's AdamW primer leaves
    it out; Alg. 1 has none).
  * eps is added outside the square root (Alg. 1).
  * A side whose dimension is not preconditioned keeps Q = I and stores no factor.
  * QR of a rank-deficient P: a Householder column whose remaining norm is at most
    ``qr_tol * ||P||_F`` is treated as exactly zero (no reflector, R_kk = 0, sign +1),
    which is what Householder QR does in exact arithmetic on an exactly zero column.
  * Noise-floor guard (``guard=True``): rows of N whose Q_L column was such a zero
    column, and columns of N whose Q_R column was, are set to 0. In exact arithmetic
    G' is exactly 0 there, so N = 0 there too; in finite precision G' holds rounding
    noise that Adam's normalisation would blow up to O(1).
  * ``refresh="eigh"`` (the appendix's alternative to QR, which it finds equivalent at
    F = 1): Q <- the factor's eigenvectors ordered by decreasing eigenvalue, each column's
    sign chosen so that q_new . q_old >= 0. That order is the one the QR refresh converges
    to (subspace iteration orders by decreasing eigenvalue), and that sign rule is the one it
    follows near its fixed point (R_kk = q_new . L q_old > 0 becomes lambda_k q_new . q_old > 0),
    so v's coordinates stay aligned from step to step. An eigenvalue at most ``qr_tol * ||F||_F`` counts as a
    zero direction for the guard, as a zero QR column does (||P||_F = ||F Q||_F = ||F||_F).
    The CUDA path has no eigh refresh (not built); this reading serves the oracle's pins.

Precision: every array is held in ``dtype`` (float64 by default). ``dtype=np.float32``
gives the "fp32 twin" used to measure the error any faithful fp32 implementation
makes against the float64 result.
"""
from __future__ import annotations

import ctypes
import os
import platform
import subprocess
import threading
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD_DIR = os.path.join(_HERE, "_build", platform.machine())
_LIB_PATH = os.path.join(_BUILD_DIR, "libsoap_oracle.so")
_lib = None
_lib_lock = threading.Lock()


def build_oracle(force: bool = False) -> str:
    """Compile oracle/householder.c with gcc into oracle/_build/libsoap_oracle.so."""
    src = os.path.join(_HERE, "householder.c")
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(src)):
        return _LIB_PATH
    os.makedirs(_BUILD_DIR, exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-o", tmp, src, "-lm"],
                   check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lib_lock:
        if _lib is None:
            lib = ctypes.CDLL(build_oracle())
            for name, ct in (("oracle_householder_q_f64", ctypes.c_double),
                             ("oracle_householder_q_f32", ctypes.c_float)):
                f = getattr(lib, name)
                f.restype = ctypes.c_int
                f.argtypes = [ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p,
                              ctypes.c_void_p, ctypes.c_void_p, ctypes.c_double]
            _lib = lib
    return _lib


def householder_q(P: np.ndarray, tol: float = 0.0):
    """Q of P = QR with diag(R) >= 0 (Alg. 1 "QR(...).Q"; sign convention of the step).

    Returns (Q, skipped, rdiag): ``skipped[k]`` marks the columns treated as exactly
    zero under the ``tol`` reading, ``rdiag`` is diag(R) after the sign fix.
    Works in P's dtype (float64 or float32).
    """
    P = np.ascontiguousarray(P)
    n = P.shape[0]
    assert P.ndim == 2 and P.shape[1] == n
    if P.dtype == np.float64:
        fn = _load().oracle_householder_q_f64
    elif P.dtype == np.float32:
        fn = _load().oracle_householder_q_f32
    else:
        raise TypeError(P.dtype)
    Q = np.empty_like(P)
    skipped = np.zeros(n, dtype=np.uint8)
    rdiag = np.empty(n, dtype=P.dtype)
    rc = fn(n, P.ctypes.data, Q.ctypes.data, skipped.ctypes.data, rdiag.ctypes.data,
            float(tol))
    if rc != 0:
        raise MemoryError("oracle QR: allocation failed")
    return Q, skipped.astype(bool), rdiag


@dataclass
class HParams:
    """Hyper-parameters of Alg. 1 and its table; defaults follow the 256x512 workload."""
    lr: float = 3e-3
    beta1: float = 0.95
    beta2: float = 0.95
    factor_beta: float = 0.95
    eps: float = 1e-8
    weight_decay: float = 0.1
    eig_every: int = 1            # F: refresh the basis when t mod F == 0
    bias_correction: bool = False
    guard: bool = True
    qr_tol: float = 2e-5
    kl: bool = False              # KL-Shampoo factor form (Alg. 1's "Accumulate Kronecker Factors")
    stale: bool = False           # factors updated after the refresh (the stale variant of section 5)
    refresh: str = "qr"           # "qr" (Alg. 1) or "eigh" (the appendix's alternative)


@dataclass
class MatrixState:
    """Per-matrix optimizer state of Alg. 1: m, v (rows x cols), L, Q_L, R, Q_R."""
    rows: int
    cols: int
    left: bool
    right: bool
    dtype: type = np.float64
    t: int = 0
    m: np.ndarray = field(default=None)
    v: np.ndarray = field(default=None)
    L: np.ndarray = field(default=None)
    QL: np.ndarray = field(default=None)
    R: np.ndarray = field(default=None)
    QR: np.ndarray = field(default=None)
    skipL: np.ndarray = field(default=None)
    skipR: np.ndarray = field(default=None)

    def __post_init__(self):
        d = self.dtype
        if self.m is None:
            self.m = np.zeros((self.rows, self.cols), d)
            self.v = np.zeros((self.rows, self.cols), d)
            if self.left:
                self.L = np.zeros((self.rows, self.rows), d)
                self.QL = np.eye(self.rows, dtype=d)
                self.skipL = np.zeros(self.rows, bool)
            if self.right:
                self.R = np.zeros((self.cols, self.cols), d)
                self.QR = np.eye(self.cols, dtype=d)
                self.skipR = np.zeros(self.cols, bool)

    def copy(self) -> "MatrixState":
        c = MatrixState(self.rows, self.cols, self.left, self.right, self.dtype, self.t,
                        self.m.copy(), self.v.copy())
        for name in ("L", "QL", "R", "QR", "skipL", "skipR"):
            a = getattr(self, name)
            setattr(c, name, None if a is None else a.copy())
        return c


# ---- sub-steps, each a plain transcription of one line group of Alg. 1 ----------

def eigh_basis(F: np.ndarray, Q_old: np.ndarray, tol: float):
    """The eigh refresh (appendix on eigh vs QR): eigenvectors of the symmetric factor F by
    decreasing eigenvalue, signs aligned with the previous basis; zero directions flagged as
    eigenvalues at most tol * ||F||_F. Returns (Q, skipped)."""
    lam, U = np.linalg.eigh((F + F.T) / 2)
    order = np.argsort(-lam, kind="stable")
    lam, U = lam[order], U[:, order]
    sign = np.where(np.sum(U * Q_old, axis=0) < 0, -1.0, 1.0).astype(F.dtype)
    return (U * sign).astype(F.dtype), lam <= tol * np.linalg.norm(F)


def approx_eigenvalues(F: np.ndarray, Q: np.ndarray) -> np.ndarray:
    """lambda = diag(Q^T F Q): Alg. 1's approximate eigenvalues of a factor in its current basis."""
    return np.diag(Q.T @ F @ Q).copy()


def factor_ema_kl(st: "MatrixState", G: np.ndarray, b: float, eps: float):
    """KL-Shampoo factor EMAs (Alg. 1, "Accumulate Kronecker Factors (KL-Shampoo)"; section
    on the SVD view of KL-Shampoo):

        L <- b L + (1-b)/out * G S_R^-1 G^T,   R <- b R + (1-b)/in * G^T S_L^-1 G,

    with S^-1 = Q diag(1/(lambda + eps)) Q^T, lambda = diag(Q^T F Q) taken from the factors and
    bases before this step's update (the exponent is read as -1, the inverse of the other
    factor; beta weights the old state as in the standard form). A side without a factor
    (identity side) counts as S = I, i.e. lambda = 1 and Q = I. The factor is positive
    semi-definite, so lambda >= 0 in exact arithmetic; a lambda that rounding made negative is
    taken as 0, which keeps every weight 1/(lambda + eps) positive and finite for eps > 0.
    Returns (L_new, R_new)."""
    rows, cols = G.shape
    d = G.dtype.type
    if st.right:
        wR = 1.0 / (np.maximum(approx_eigenvalues(st.R, st.QR), 0) + eps)
        SR_inv = st.QR @ np.diag(wR) @ st.QR.T
    else:
        SR_inv = np.eye(cols, dtype=G.dtype) / d(1.0 + eps)
    if st.left:
        wL = 1.0 / (np.maximum(approx_eigenvalues(st.L, st.QL), 0) + eps)
        SL_inv = st.QL @ np.diag(wL) @ st.QL.T
    else:
        SL_inv = np.eye(rows, dtype=G.dtype) / d(1.0 + eps)
    L = b * st.L + (1 - b) / cols * (G @ SR_inv @ G.T) if st.left else None
    R = b * st.R + (1 - b) / rows * (G.T @ SL_inv @ G) if st.right else None
    return L, R


def factor_ema(F: np.ndarray, G: np.ndarray, b: float, side: str) -> np.ndarray:
    """S1: L <- b L + (1-b) G G^T (side 'L') or R <- b R + (1-b) G^T G (side 'R').

    Standard Shampoo factor EMAs (section 2) with the current gradient (section 5).
    """
    if side == "L":
        return b * F + (1 - b) * (G @ G.T)
    return b * F + (1 - b) * (G.T @ G)


def rotate_in(QL, G, QR):
    """S5: G' = Q_L^T G Q_R (Alg. 1, "Rotate gradient into eigenbasis")."""
    X = G if QL is None else QL.T @ G
    return X if QR is None else X @ QR


def rotate_out(QL, N, QR):
    """S7: dW = Q_L N Q_R^T (Alg. 1, "Rotate update out of eigenbasis")."""
    X = N if QL is None else QL @ N
    return X if QR is None else X @ QR.T


def adam_in_basis(m, v, Gp, hp: HParams, t: int, skipL=None, skipR=None):
    """S6: m, v EMAs in the rotated basis and N = m / (sqrt(v) + eps) (Alg. 1 Adam block).

    With ``hp.guard`` the rows/cols of N belonging to zero QR columns are 0.
    Returns (m, v, N).
    """
    m = hp.beta1 * m + (1 - hp.beta1) * Gp
    v = hp.beta2 * v + (1 - hp.beta2) * Gp * Gp
    if hp.bias_correction:
        mh = m / (1 - hp.beta1 ** t)
        vh = v / (1 - hp.beta2 ** t)
    else:
        mh, vh = m, v
    N = mh / (np.sqrt(vh) + m.dtype.type(hp.eps))
    if hp.guard:
        if skipL is not None:
            N[skipL, :] = 0
        if skipR is not None:
            N[:, skipR] = 0
    return m, v, N


def weight_update(W, dW, lr, wd):
    """S8: W <- (1 - lr*wd) W - lr*dW (Alg. 1, "Weight decay and update")."""
    return (1 - lr * wd) * W - lr * dW


def soap_step(st: MatrixState, W: np.ndarray, G: np.ndarray, hp: HParams,
              lr: float | None = None, wd: float | None = None):
    """One SOAP step of Alg. 1 for one matrix. Mutates ``st``; returns (W_new, dW).

    ``W`` and ``G`` are converted to the state's dtype. ``dW`` is the back-rotated
    Adam direction Q_L N Q_R^T before the learning rate is applied.
    """
    d = st.dtype
    W = np.asarray(W, dtype=d)
    G = np.asarray(G, dtype=d)
    lr = hp.lr if lr is None else lr
    wd = hp.weight_decay if wd is None else wd
    st.t += 1
    t = st.t
    if hp.stale:
        # section 5's "stale preconditioner" variant: the refresh sees the factors of the earlier
        # steps only, and the current gradient enters them after the update. Its zero QR
        # columns are not null directions of the current gradient, so the guard does not apply.
        if hp.kl or hp.guard:
            raise ValueError("the stale variant is defined for the standard factors without the guard")
        W_new, dW = _rotate_adam_update(st, W, G, hp, t, d, lr, wd)
        if st.left:
            st.L = factor_ema(st.L, G, hp.factor_beta, "L")
        if st.right:
            st.R = factor_ema(st.R, G, hp.factor_beta, "R")
        return W_new, dW
    # S1: accumulate the Kronecker factors with the current gradient
    if hp.kl:
        L, R = factor_ema_kl(st, G, d(hp.factor_beta), d(hp.eps))
        if st.left:
            st.L = L
        if st.right:
            st.R = R
    else:
        if st.left:
            st.L = factor_ema(st.L, G, hp.factor_beta, "L")
        if st.right:
            st.R = factor_ema(st.R, G, hp.factor_beta, "R")
    return _rotate_adam_update(st, W, G, hp, t, d, lr, wd)


def _rotate_adam_update(st: MatrixState, W, G, hp: HParams, t: int, d, lr, wd):
    """S2-S8 of one step (the factors as they stand): refresh every F steps, re-projection,
    rotation, Adam in the basis, back-rotation and update. Returns (W_new, dW)."""
    if hp.refresh not in ("qr", "eigh"):
        raise ValueError(f"unknown basis refresh {hp.refresh!r}")
    # S2-S4: eigenbasis re-computation every F steps
    if t % hp.eig_every == 0:
        M_hat = rotate_out(st.QL if st.left else None, st.m, st.QR if st.right else None)
        if hp.refresh == "eigh":
            if st.left:
                st.QL, st.skipL = eigh_basis(st.L, st.QL, hp.qr_tol)
            if st.right:
                st.QR, st.skipR = eigh_basis(st.R, st.QR, hp.qr_tol)
        else:
            if st.left:
                st.QL, st.skipL, _ = householder_q(st.L @ st.QL, hp.qr_tol)
            if st.right:
                st.QR, st.skipR, _ = householder_q(st.R @ st.QR, hp.qr_tol)
        st.m = rotate_in(st.QL if st.left else None, M_hat, st.QR if st.right else None)
    # S5: rotate the gradient with the (new) basis
    QL = st.QL if st.left else None
    QR = st.QR if st.right else None
    Gp = rotate_in(QL, G, QR)
    # S6: Adam in the eigenbasis
    st.m, st.v, N = adam_in_basis(st.m, st.v, Gp, hp, t,
                                  st.skipL if st.left else None,
                                  st.skipR if st.right else None)
    # S7: rotate back; S8: decoupled weight decay and update
    dW = rotate_out(QL, N, QR)
    return weight_update(W, dW, d(lr), d(wd)), dW
