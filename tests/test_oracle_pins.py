"""Pins of the fp64 oracle against facts fixed by the paper or by mathematics.

Each test compares the oracle with something other than itself: a closed form, an
invariant, a library routine solving the same textbook problem, or brute force.
"""
import numpy as np
import pytest

from oracle.soap_ref import (HParams, MatrixState, eigh_basis, factor_ema, householder_q, rotate_in,
                             rotate_out, soap_step)

RNG = np.random.default_rng(1234)


# ---- S3: the QR refresh ------------------------------------------------------------

@pytest.mark.parametrize("n", [1, 2, 5, 33, 128])
def test_qr_matches_library_qr_with_positive_diagonal(n):
    """Full-rank P: Q with diag(R) > 0 is unique, so it equals LAPACK's after its sign fix."""
    P = RNG.standard_normal((n, n))
    Q, skipped, rdiag = householder_q(P, 0.0)
    Ql, Rl = np.linalg.qr(P)
    s = np.sign(np.diag(Rl))
    s[s == 0] = 1
    assert not skipped.any()
    np.testing.assert_allclose(Q, Ql * s, atol=1e-12)
    np.testing.assert_allclose(rdiag, np.abs(np.diag(Rl)), rtol=1e-12)


@pytest.mark.parametrize("n", [3, 64, 200])
def test_qr_orthogonal_and_triangular(n):
    """Q^T Q = I and Q^T P is upper triangular with a non-negative diagonal."""
    P = RNG.standard_normal((n, n))
    Q, _, rdiag = householder_q(P, 0.0)
    assert np.abs(Q.T @ Q - np.eye(n)).max() < 1e-13
    R = Q.T @ P
    assert np.abs(np.tril(R, -1)).max() < 1e-12 * np.abs(P).max() * n
    np.testing.assert_allclose(np.diag(R), rdiag, atol=1e-12 * np.linalg.norm(P))
    assert (np.diag(R) > 0).all()


def test_qr_exactly_rank_deficient_columns_are_skipped():
    """Dependent columns (exact integer combinations) get no reflector, Q stays orthogonal,
    P = Q R still holds with R upper triangular and R_kk = 0 at the skipped columns."""
    a = np.array([1.0, 2.0, 0.0, -1.0, 3.0])
    b = np.array([0.0, 1.0, 1.0, 2.0, -2.0])
    c = np.array([4.0, 0.0, 1.0, 1.0, 1.0])
    P = np.stack([a, 2 * a, b, a - b, c], axis=1)
    Q, skipped, rdiag = householder_q(P, 1e-10)
    assert skipped.tolist() == [False, True, False, True, False]
    assert np.abs(Q.T @ Q - np.eye(5)).max() < 1e-14
    R = Q.T @ P
    assert np.abs(np.tril(R, -1)).max() < 1e-12
    assert np.abs(np.diag(R)[[1, 3]]).max() < 1e-12
    assert (rdiag[[0, 2, 4]] > 0).all()


def test_qr_zero_matrix_gives_identity():
    Q, skipped, _ = householder_q(np.zeros((7, 7)), 0.0)
    assert skipped.all()
    np.testing.assert_array_equal(Q, np.eye(7))


def test_qr_float32_twin_is_orthogonal():
    P = RNG.standard_normal((96, 96)).astype(np.float32)
    Q, _, _ = householder_q(P, 0.0)
    assert Q.dtype == np.float32
    assert np.abs(Q.T.astype(np.float64) @ Q - np.eye(96)).max() < 2e-6


def test_subspace_iteration_converges_to_planted_eigenvectors():
    """Repeated refreshes Q <- QR(L Q).Q are subspace iteration (Golub & Van Loan 8.2.4): with a
    planted spectrum the k-th column converges to the k-th eigenvector at rate lambda_k+1/lambda_k."""
    n = 24
    U, _ = np.linalg.qr(RNG.standard_normal((n, n)))
    lam = 2.0 ** -np.arange(n)          # ratio 1/2 between neighbours
    L = (U * lam) @ U.T
    Q = np.eye(n)
    for _ in range(80):
        Q, _, _ = householder_q(L @ Q, 0.0)
    cos = np.abs(np.sum(Q[:, :12] * U[:, :12], axis=0))
    assert cos.min() > 1 - 1e-10
    # every leading prefix spans the planted invariant subspace (principal angles ~ 0)
    for k in (1, 4, 8, 12):
        s = np.linalg.svd(U[:, :k].T @ Q[:, :k], compute_uv=False)
        assert s.min() > 1 - 1e-10


# ---- S1: factor EMAs --------------------------------------------------------------

def test_factor_ema_closed_form():
    """L_t = sum_s (1-b) b^(t-s) G_s G_s^T and R_t likewise (section 2 Shampoo EMAs, unrolled)."""
    b = 0.95
    Gs = [RNG.standard_normal((6, 9)) for _ in range(7)]
    L = np.zeros((6, 6))
    R = np.zeros((9, 9))
    for G in Gs:
        L = factor_ema(L, G, b, "L")
        R = factor_ema(R, G, b, "R")
    T = len(Gs)
    Lc = sum((1 - b) * b ** (T - 1 - s) * np.einsum("ik,jk->ij", Gs[s], Gs[s]) for s in range(T))
    Rc = sum((1 - b) * b ** (T - 1 - s) * np.einsum("ki,kj->ij", Gs[s], Gs[s]) for s in range(T))
    np.testing.assert_allclose(L, Lc, rtol=1e-13)
    np.testing.assert_allclose(R, Rc, rtol=1e-13)


# ---- S6/S8: reduction to AdamW when Q = I -----------------------------------------

@pytest.mark.parametrize("sides", [(False, False), (True, True), (True, False)])
@pytest.mark.parametrize("bias_correction", [False, True])
def test_constant_gradient_reduces_to_adam_closed_form(sides, bias_correction):
    """With Q = I (section 2: identity eigenvectors recover AdamW) and a constant gradient g,
    the EMAs sum to m_t = (1-b1^t) g and v_t = (1-b2^t) g^2, so
    N_t = (1-b1^t) g / (sqrt(1-b2^t) |g| + eps), or g / (|g| + eps) with bias correction.
    One entry has |g| = 2e-8 ~ eps, where eps inside the root would change N by 1e3x.
    A diagonal gradient keeps L, R diagonal, so preconditioned sides stay at Q = I."""
    n = 5
    gd = np.array([0.3, -0.2, 0.5, -0.7, 2e-8])
    g = np.diag(gd)
    hp = HParams(lr=1e-2, weight_decay=0.0, bias_correction=bias_correction, qr_tol=0.0)
    st = MatrixState(n, n, sides[0], sides[1])
    W0 = np.full((n, n), 0.25)
    W = W0.copy()
    expected = W0.copy()
    for t in range(1, 9):
        W, _ = soap_step(st, W, g, hp)
        if bias_correction:
            N = gd / (np.abs(gd) + 1e-8)
        else:
            N = (1 - 0.95 ** t) * gd / (np.sqrt(1 - 0.95 ** t) * np.abs(gd) + 1e-8)
        expected = expected - hp.lr * np.diag(N)
        np.testing.assert_allclose(W, expected, rtol=0, atol=1e-15)
    if sides[0]:
        np.testing.assert_allclose(st.QL, np.eye(n), atol=1e-15)


def test_zero_gradient_is_pure_weight_decay():
    """G = 0: every EMA stays 0, N = 0/(0+eps) = 0, so W_t = (1 - lr*wd)^t W_0 (Alg. 1 last line)."""
    hp = HParams(lr=3e-3, weight_decay=0.1)
    st = MatrixState(4, 6, True, True)
    W0 = RNG.standard_normal((4, 6))
    W = W0.copy()
    for _ in range(5):
        W, dW = soap_step(st, W, np.zeros((4, 6)), hp)
        assert np.all(dW == 0)
    np.testing.assert_allclose(W, (1 - 3e-4) ** 5 * W0, rtol=1e-14)
    assert st.skipL.all() and st.skipR.all()


def test_basis_frequency_refreshes_only_every_f_steps():
    """Eigenbasis frequency F = 4 (Alg. 1 refreshes when t mod F = 0): steps 1-3 keep Q = I and
    are AdamW in closed form for any gradients; step 4 takes Q from the library QR of L_4 Q = L_4
    (and R_4) with the sign fix, re-projects m but not v (Alg. 1 re-projects only m), and rotates;
    steps 5-7 keep that basis while the factors move on."""
    rows, cols, F = 6, 5, 4
    b, b1, b2, eps, lr, wd = 0.95, 0.9, 0.99, 1e-8, 1e-2, 0.1
    hp = HParams(lr=lr, weight_decay=wd, beta1=b1, beta2=b2, factor_beta=b, eps=eps, eig_every=F)
    rng = np.random.default_rng(77)
    st = MatrixState(rows, cols, True, True)
    W = rng.standard_normal((rows, cols))
    m, v = np.zeros((rows, cols)), np.zeros((rows, cols))
    L, R = np.zeros((rows, rows)), np.zeros((cols, cols))
    QL, QR = np.eye(rows), np.eye(cols)

    def signed_q(P):
        q, r = np.linalg.qr(P)
        return q * np.where(np.diag(r) < 0, -1.0, 1.0)

    for t in range(1, 8):
        G = rng.standard_normal((rows, cols))
        L = b * L + (1 - b) * G @ G.T
        R = b * R + (1 - b) * G.T @ G
        if t % F == 0:
            newL, newR = signed_q(L @ QL), signed_q(R @ QR)
            m = newL.T @ (QL @ m @ QR.T) @ newR
            QL, QR = newL, newR
        Gp = QL.T @ G @ QR
        m = b1 * m + (1 - b1) * Gp
        v = b2 * v + (1 - b2) * Gp * Gp
        want = (1 - lr * wd) * W - lr * QL @ (m / (np.sqrt(v) + eps)) @ QR.T
        W, _ = soap_step(st, W, G, hp)
        np.testing.assert_allclose(W, want, rtol=0, atol=1e-12)
        np.testing.assert_allclose(st.QL, QL, atol=1e-12)
        np.testing.assert_allclose(st.QR, QR, atol=1e-12)
        np.testing.assert_allclose(st.v, v, atol=1e-14)
        if t < F:
            assert np.array_equal(st.QL, np.eye(rows)) and np.array_equal(st.QR, np.eye(cols))
    assert not st.skipL.any() and not st.skipR.any()
    assert not np.allclose(QL, np.eye(rows))


# ---- S7: update-RMS invariance ------------------------------------------------------

def test_update_norm_equals_adam_norm():
    """||dW||_F = ||N||_F because Q_L, Q_R are orthogonal (section 5, update RMS matching)."""
    hp = HParams()
    st = MatrixState(12, 20, True, True)
    W = RNG.standard_normal((12, 20))
    for t in range(4):
        G = RNG.standard_normal((12, 20))
        W, dW = soap_step(st, W, G, hp)
        N = st.m / (np.sqrt(st.v) + hp.eps)
        N[st.skipL, :] = 0
        N[:, st.skipR] = 0
        assert abs(np.linalg.norm(dW) - np.linalg.norm(N)) < 1e-12 * np.linalg.norm(N)


# ---- S4: first-moment re-projection -------------------------------------------------

def test_reprojection_preserves_momentum_in_original_space():
    """With beta1 = 1 the Adam block leaves m unchanged, so across a basis change
    Q_L,new m_new Q_R,new^T must equal Q_L,old m_old Q_R,old^T (Alg. 1 re-projection)."""
    hp = HParams(beta1=0.95)
    st = MatrixState(8, 10, True, True)
    W = np.zeros((8, 10))
    for _ in range(3):
        W, _ = soap_step(st, W, RNG.standard_normal((8, 10)), hp)
    before = st.QL @ st.m @ st.QR.T
    QL_old = st.QL.copy()
    hp1 = HParams(beta1=1.0)
    soap_step(st, W, RNG.standard_normal((8, 10)), hp1)
    assert np.abs(st.QL - QL_old).max() > 1e-3  # the basis really changed
    after = st.QL @ st.m @ st.QR.T
    np.testing.assert_allclose(after, before, atol=1e-13)


def test_rotations_are_the_two_sided_products():
    QL, _ = np.linalg.qr(RNG.standard_normal((4, 4)))
    QR, _ = np.linalg.qr(RNG.standard_normal((6, 6)))
    G = RNG.standard_normal((4, 6))
    Gp = rotate_in(QL, G, QR)
    np.testing.assert_allclose(np.einsum("ki,kl,lj->ij", QL, G, QR), Gp, atol=1e-14)
    np.testing.assert_allclose(rotate_out(QL, Gp, QR), G, atol=1e-14)


# ---- S1-S3 against a brute-force eigendecomposition ---------------------------------

@pytest.mark.parametrize("shape", [(4, 6), (6, 3), (5, 5)])
def test_constant_gradient_basis_converges_to_eigh(shape):
    """Constant G: L_t -> G G^T and R_t -> G^T G, and the refreshed bases converge to their
    eigenvectors, ordered by decreasing eigenvalue (Q_0 = I is generic), up to sign --
    checked against the library's symmetric eigensolver."""
    m, n = shape
    G = RNG.standard_normal(shape)
    st = MatrixState(m, n, True, True)
    hp = HParams(factor_beta=0.5, qr_tol=1e-10)
    W = np.zeros(shape)
    for _ in range(300):
        W, _ = soap_step(st, W, G, hp)
    for Q, F, skip in ((st.QL, G @ G.T, st.skipL), (st.QR, G.T @ G, st.skipR)):
        w, U = np.linalg.eigh(F)
        order = np.argsort(-w)
        w, U = w[order], U[:, order]
        r = int(np.sum(w > 1e-10 * w[0]))
        cos = np.abs(np.sum(Q[:, :r] * U[:, :r], axis=0))
        assert cos.min() > 1 - 1e-8, cos


# ---- S1-S7: the SVD view with the EMAs switched off ---------------------------------

def test_emas_off_gives_polar_factor():
    """Appendix (SVD view of SOAP): with b = beta1 = beta2 = 0 and a constant full-rank G, the
    bases converge to U, V of G = U S V^T, G' -> S (diagonal), N -> sign(S) = I and the update
    direction dW -> U V^T, the polar factor; compared with the library SVD."""
    n = 6
    G = RNG.standard_normal((n, n))
    hp = HParams(beta1=0.0, beta2=0.0, factor_beta=0.0, lr=0.0, weight_decay=0.0, qr_tol=1e-12)
    st = MatrixState(n, n, True, True)
    W = np.zeros((n, n))
    for _ in range(400):
        W, dW = soap_step(st, W, G, hp)
    U, s, Vt = np.linalg.svd(G)
    np.testing.assert_allclose(dW, U @ Vt, atol=1e-6)
    Gp = rotate_in(st.QL, G, st.QR)
    np.testing.assert_allclose(np.abs(np.diag(Gp)), s, rtol=1e-8)
    assert np.abs(Gp - np.diag(np.diag(Gp))).max() < 1e-8 * s[0]


# ---- guard and rank deficiency -----------------------------------------------------

def test_first_step_of_rectangular_matrix_is_null_space_free():
    """At t = 1 R = (1-b) G^T G has rank = rows < cols; the zero QR columns span G's null
    space, so G Q_R is exactly 0 there and the guarded N is 0 there (exact arithmetic)."""
    G = RNG.standard_normal((5, 9))
    st = MatrixState(5, 9, True, True)
    soap_step(st, np.zeros((5, 9)), G, HParams(qr_tol=1e-9))
    assert st.skipR.sum() == 4
    assert np.abs(G @ st.QR[:, st.skipR]).max() < 1e-12
    assert np.abs(G @ st.QR[:, ~st.skipR]).min(axis=0).max() > 1e-3


# ---- KL-Shampoo factor form (Alg. 1 "Accumulate Kronecker Factors (KL-Shampoo)") ----------

def test_kl_first_step_closed_form():
    """From L = R = 0 and Q = I every approximate eigenvalue is 0, so the first KL update is
    the standard one scaled by 1/((in or out) * eps)."""
    rng = np.random.default_rng(31)
    rows, cols = 6, 9
    G = rng.standard_normal((rows, cols))
    hp = HParams(kl=True, eps=1e-3)
    st = MatrixState(rows, cols, True, True)
    soap_step(st, np.zeros((rows, cols)), G, hp)
    b = hp.factor_beta
    L_expect = (1 - b) / (cols * hp.eps) * np.einsum("ik,jk->ij", G, G)
    R_expect = (1 - b) / (rows * hp.eps) * np.einsum("ki,kj->ij", G, G)
    np.testing.assert_allclose(st.L, L_expect, rtol=1e-12)
    np.testing.assert_allclose(st.R, R_expect, rtol=1e-12)


def test_kl_update_uses_the_regularised_inverse_of_the_other_factor():
    """When the basis diagonalises the other factor exactly, Q diag(1/(lambda + eps)) Q^T is
    (F + eps I)^-1, so the KL update equals b L + (1-b)/out G (R + eps I)^-1 G^T computed with
    a library inverse (and likewise for R)."""
    rng = np.random.default_rng(32)
    rows, cols = 5, 7
    G = rng.standard_normal((rows, cols))
    QL = np.linalg.qr(rng.standard_normal((rows, rows)))[0]
    QR = np.linalg.qr(rng.standard_normal((cols, cols)))[0]
    muL = rng.uniform(0.5, 2.0, rows)
    muR = rng.uniform(0.5, 2.0, cols)
    st = MatrixState(rows, cols, True, True)
    st.L, st.QL = QL @ np.diag(muL) @ QL.T, QL
    st.R, st.QR = QR @ np.diag(muR) @ QR.T, QR
    L0, R0 = st.L.copy(), st.R.copy()
    from oracle.soap_ref import factor_ema_kl
    b, eps = 0.9, 0.05
    L, R = factor_ema_kl(st, G, b, eps)
    L_expect = b * L0 + (1 - b) / cols * G @ np.linalg.inv(R0 + eps * np.eye(cols)) @ G.T
    R_expect = b * R0 + (1 - b) / rows * G.T @ np.linalg.inv(L0 + eps * np.eye(rows)) @ G
    np.testing.assert_allclose(L, L_expect, rtol=1e-10)
    np.testing.assert_allclose(R, R_expect, rtol=1e-10)


def test_kl_identity_side_counts_as_identity_factor():
    """A one-sided matrix: the missing factor is S = I (lambda = 1)."""
    rng = np.random.default_rng(33)
    rows, cols = 4, 6
    G = rng.standard_normal((rows, cols))
    st = MatrixState(rows, cols, True, False)
    from oracle.soap_ref import factor_ema_kl
    L, R = factor_ema_kl(st, G, 0.9, 1e-3)
    assert R is None
    np.testing.assert_allclose(L, 0.1 / cols / (1 + 1e-3) * G @ G.T, rtol=1e-12)


def test_kl_factors_track_singular_values_at_the_fixed_point():
    """The appendix's fixed point: for a constant square gradient G = U diag(s) V^T and balanced
    factors, KL-Shampoo's factor eigenvalues settle at s / sqrt(n) (with the 1/out and 1/in
    scalings), not at s^2 / n as Shampoo's do, so kappa(L_KL) = sqrt(kappa(L_Shampoo))."""
    rng = np.random.default_rng(34)
    n = 6
    U = np.linalg.qr(rng.standard_normal((n, n)))[0]
    V = np.linalg.qr(rng.standard_normal((n, n)))[0]
    s = np.array([4.0, 2.5, 1.5, 1.0, 0.6, 0.3])
    G = U @ np.diag(s) @ V.T
    hp = HParams(kl=True, factor_beta=0.5, eps=1e-8, lr=0.0, weight_decay=0.0)
    st = MatrixState(n, n, True, True)
    for _ in range(120):
        soap_step(st, np.zeros((n, n)), G, hp)
    evL = np.sort(np.linalg.eigvalsh(st.L))[::-1]
    evR = np.sort(np.linalg.eigvalsh(st.R))[::-1]
    np.testing.assert_allclose(evL, s / np.sqrt(n), rtol=1e-6)
    np.testing.assert_allclose(evR, s / np.sqrt(n), rtol=1e-6)
    kappa_kl = evL[0] / evL[-1]
    kappa_shampoo = (s[0] / s[-1]) ** 2
    assert abs(kappa_kl - np.sqrt(kappa_shampoo)) < 1e-5 * kappa_kl


def test_kl_rounding_negative_eigenvalue_counts_as_zero():
    """lambda = diag(Q^T F Q) of a positive semi-definite factor is >= 0; a value that rounding
    pushed below 0 is read as 0, so the weight there is 1/eps (positive, finite) rather than a
    negative or unbounded 1/(lambda + eps). Checked against the closed form with F's null
    direction given weight 1/eps and the others 1/(mu + eps)."""
    rng = np.random.default_rng(35)
    rows, cols = 4, 5
    G = rng.standard_normal((rows, cols))
    QR = np.linalg.qr(rng.standard_normal((cols, cols)))[0]
    mu = np.array([3.0, 1.0, 0.5, 0.25, -1e-9])  # the last: a rounding artefact of a null direction
    st = MatrixState(rows, cols, False, True)
    st.R, st.QR = QR @ np.diag(mu) @ QR.T, QR
    st2 = MatrixState(rows, cols, True, True)
    st2.R, st2.QR = st.R, QR
    from oracle.soap_ref import factor_ema_kl
    eps = 1e-8
    L, _ = factor_ema_kl(st2, G, 0.5, eps)
    w = 1.0 / (np.array([3.0, 1.0, 0.5, 0.25, 0.0]) + eps)
    L_expect = 0.5 / cols * G @ QR @ np.diag(w) @ QR.T @ G.T
    np.testing.assert_allclose(L, L_expect, rtol=1e-9)
    assert np.all(np.linalg.eigvalsh(L) > -1e-6 * np.abs(L).max())


# ---- the stale variant (section 5, "Diagnosing the Slingshot Instability") -----------------

def test_stale_first_step_is_plain_adam():
    """With the current gradient left out of the refresh, step 1 factors P = 0 Q = 0: every QR
    column is zero, Q stays I, and (without the guard) the step is elementwise Adam with
    decoupled weight decay; the factors take the gradient only afterwards."""
    rng = np.random.default_rng(41)
    rows, cols = 5, 7
    G = rng.standard_normal((rows, cols))
    W0 = rng.standard_normal((rows, cols))
    hp = HParams(stale=True, guard=False)
    st = MatrixState(rows, cols, True, True)
    W1, _ = soap_step(st, W0, G, hp)
    m = (1 - hp.beta1) * G
    v = (1 - hp.beta2) * G * G
    N = m / (np.sqrt(v) + hp.eps)
    np.testing.assert_allclose(W1, (1 - hp.lr * hp.weight_decay) * W0 - hp.lr * N, rtol=1e-12, atol=1e-15)
    np.testing.assert_array_equal(st.QL, np.eye(rows))
    np.testing.assert_array_equal(st.QR, np.eye(cols))
    np.testing.assert_allclose(st.L, (1 - hp.factor_beta) * G @ G.T, rtol=1e-12)
    np.testing.assert_allclose(st.R, (1 - hp.factor_beta) * G.T @ G, rtol=1e-12)


def test_stale_basis_lags_one_gradient():
    """Step 2 of the stale variant refreshes from L_1 = (1-b) G_1 G_1^T alone: Q_L equals a
    library QR of L_1 (Q_L = I before it) with the sign fix, and differs from the real-time
    basis, which also sees G_2."""
    rng = np.random.default_rng(42)
    rows, cols = 5, 9
    G1, G2 = rng.standard_normal((rows, cols)), rng.standard_normal((rows, cols))
    W = np.zeros((rows, cols))
    hp = HParams(stale=True, guard=False)
    st = MatrixState(rows, cols, True, True)
    soap_step(st, W, G1, hp)
    soap_step(st, W, G2, hp)
    Q, Rm = np.linalg.qr((1 - hp.factor_beta) * G1 @ G1.T)
    Q = Q * np.where(np.diag(Rm) < 0, -1.0, 1.0)
    np.testing.assert_allclose(st.QL, Q, atol=1e-12)
    rt = MatrixState(rows, cols, True, True)
    soap_step(rt, W, G1, HParams(guard=False))
    soap_step(rt, W, G2, HParams(guard=False))
    assert np.abs(rt.QL - st.QL).max() > 1e-3


def test_stale_rejects_kl_and_guard():
    st = MatrixState(3, 4, True, True)
    for hp in (HParams(stale=True), HParams(stale=True, guard=False, kl=True)):
        with pytest.raises(ValueError):
            soap_step(st, np.zeros((3, 4)), np.ones((3, 4)), hp)


# ---- the eigh refresh (appendix on eigh vs QR) ----------------------------------------

def test_eigh_basis_diagonalises_in_decreasing_order_with_aligned_signs():
    """eigh_basis returns an orthogonal Q with Q^T F Q diagonal and its diagonal decreasing, and
    every column has a nonnegative overlap with the previous basis's column."""
    rng = np.random.default_rng(61)
    n = 9
    X = rng.standard_normal((n, 4))
    F = X @ X.T + np.diag(np.linspace(0.1, 0.2, n))
    Q_old = np.linalg.qr(rng.standard_normal((n, n)))[0]
    Q, skip = eigh_basis(F, Q_old, 1e-4)
    assert np.abs(Q.T @ Q - np.eye(n)).max() < 1e-13
    D = Q.T @ F @ Q
    assert np.abs(D - np.diag(np.diag(D))).max() < 1e-12 * np.abs(F).max()
    assert np.all(np.diff(np.diag(D)) <= 1e-14)
    assert np.all(np.sum(Q * Q_old, axis=0) >= 0)
    assert not skip.any()
    # the zero factor: every direction is a zero direction, and the basis stays the old one
    Q0, skip0 = eigh_basis(np.zeros((n, n)), np.eye(n), 1e-4)
    assert skip0.all() and np.array_equal(Q0, np.eye(n))


def test_eigh_and_qr_refreshes_agree_at_the_fixed_point():
    """For a constant gradient the QR refresh is subspace iteration and converges to the
    eigenvectors by decreasing eigenvalue, the basis and order the eigh refresh takes at once
    (the appendix finds the two refreshes equivalent at F = 1). Column signs may differ (each
    path keeps the signs its history gave), and the update does not depend on them: once the
    EMAs have forgotten the steps before convergence, both give the same update. The entries of
    N off the converged diagonal forget slowest, as (beta1 / sqrt(beta2))^k = 0.974^k, about
    1e-5 after the 450 steps here."""
    rng = np.random.default_rng(62)
    n = 5
    U = np.linalg.qr(rng.standard_normal((n, n)))[0]
    V = np.linalg.qr(rng.standard_normal((n, n)))[0]
    G = U @ np.diag([3.0, 2.0, 1.3, 0.8, 0.5]) @ V.T
    runs = {}
    for refresh in ("qr", "eigh"):
        hp = HParams(refresh=refresh, lr=1e-3)
        st = MatrixState(n, n, True, True)
        W = np.zeros((n, n))
        for _ in range(450):
            W, dW = soap_step(st, W, G, hp)
        runs[refresh] = (st, dW)
    (sq, dq), (se, de) = runs["qr"], runs["eigh"]
    for A, B in ((sq.QL, se.QL), (sq.QR, se.QR)):
        s = np.sign(np.sum(A * B, axis=0))
        np.testing.assert_allclose(A, B * s, atol=1e-9)
    np.testing.assert_allclose(dq, de, rtol=0, atol=1e-5 * np.abs(de).max())
    # and the eigenvectors are G's singular vectors, up to sign
    np.testing.assert_allclose(np.abs(se.QL), np.abs(U), atol=1e-9)


def test_unknown_refresh_is_rejected():
    with pytest.raises(ValueError):
        soap_step(MatrixState(2, 2, True, True), np.zeros((2, 2)), np.ones((2, 2)), HParams(refresh="svd"))


def _planted(n, lam, rng):
    U, _ = np.linalg.qr(rng.standard_normal((n, n)))
    return U, (U * lam) @ U.T


def test_guard_zeroes_nothing_on_a_full_rank_factor():
    """Reading R12's zero-column rule on a full-rank factor with kappa = 1e3 (eigenvalues
    log-spaced in [1e-3, 1]): the refresh treats no column as zero, from Q = I and from a random
    basis, over several refreshes, at the default qr_tol."""
    rng = np.random.default_rng(31)
    n = 64
    _, L = _planted(n, np.logspace(-3, 0, n), rng)
    for Q0 in (np.eye(n), np.linalg.qr(rng.standard_normal((n, n)))[0]):
        Q = Q0
        for _ in range(6):
            Q, skip, _ = householder_q(L @ Q, HParams().qr_tol)
            assert not skip.any()


@pytest.mark.parametrize("lo, tol", [(1e-6, 1e-9), (1e-2, None)])
def test_guard_zeroes_exactly_a_planted_null_space(lo, tol):
    """A factor of rank 40 of 64 whose nonzero eigenvalues are log-spaced in [lo, 1]: the refresh
    zeroes exactly 24 columns, and they span the planted null space (the kept ones its
    complement). With nonzero eigenvalues down to 1e-6 this needs a qr_tol below their QR residuals
    (1e-9 here, far above fp64 rounding); the default qr_tol, set just above the fp32 noise floor
    of the step's refresh, does the same on a spectrum in [1e-2, 1]."""
    rng = np.random.default_rng(32)
    n, r = 64, 40
    lam = np.concatenate([np.logspace(np.log10(lo), 0, r), np.zeros(n - r)])
    U, L = _planted(n, lam, rng)
    tol = HParams().qr_tol if tol is None else tol
    for Q0 in (np.eye(n), np.linalg.qr(rng.standard_normal((n, n)))[0]):
        Q, skip, _ = householder_q(L @ Q0, tol)
        assert skip.sum() == n - r
        assert np.abs(U[:, :r].T @ Q[:, skip]).max() <= 1e-8
        assert np.abs(U[:, r:].T @ Q[:, ~skip]).max() <= 1e-8
