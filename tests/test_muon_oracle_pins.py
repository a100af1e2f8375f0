"""Pins of the Muon oracle (Alg. Muon) against closed forms and library routines."""
import numpy as np

from oracle.muon_ref import MuonParams, MuonState, bf16_round, muon_step, newton_schulz


def test_cubic_newton_schulz_converges_to_the_polar_factor():
    """(a, b, c) = (1.5, -0.5, 0) is the classical Newton-Schulz iteration X <- X (3 I - X^T X)/2,
    which converges to the polar factor U V^T of X_0 when its singular values lie in (0, sqrt 3);
    after normalisation by ||M||_F they lie in (0, 1]."""
    rng = np.random.default_rng(51)
    M = rng.standard_normal((6, 9))
    U, s, Vt = np.linalg.svd(M, full_matrices=False)
    M = U @ np.diag(np.linspace(1.0, 0.4, 6)) @ Vt  # well conditioned
    X = newton_schulz(M, [(1.5, -0.5, 0.0)] * 60, 1e-7)
    np.testing.assert_allclose(X, U @ Vt, atol=1e-10)


def test_identity_schedule_and_step_closed_form():
    """With a_i = 1, b_i = c_i = 0 the iterations leave X_0 = M / ||M||_F, so the step is
    W <- (1 - lr wd) W - lr sqrt(max(in, out)) M / ||M||_F with M = (1 - beta1) G at t = 1."""
    rng = np.random.default_rng(52)
    G, W = rng.standard_normal((4, 10)), rng.standard_normal((4, 10))
    hp = MuonParams(coeffs=[(1.0, 0.0, 0.0)] * 3)
    st = MuonState(4, 10)
    W1, dW = muon_step(st, W, G, hp)
    M = (1 - hp.beta1) * G
    np.testing.assert_allclose(dW, M / np.linalg.norm(M) * np.sqrt(10), rtol=1e-12)
    np.testing.assert_allclose(W1, (1 - hp.lr * hp.weight_decay) * W - hp.lr * dW, rtol=1e-12)
    np.testing.assert_allclose(st.M, M, rtol=1e-12)


def test_eps_bounds_the_normalisation():
    """A momentum with ||M||_F < eps is divided by eps, not by its norm."""
    G = np.full((2, 3), 1e-9)
    hp = MuonParams(coeffs=[(1.0, 0.0, 0.0)], beta1=0.0, eps=1e-7)
    st = MuonState(2, 3)
    _, dW = muon_step(st, np.zeros((2, 3)), G, hp)
    np.testing.assert_allclose(dW, G / 1e-7 * np.sqrt(3), rtol=1e-12)


def test_orientation_does_not_change_the_result():
    """An odd polynomial step commutes with transposition: Newton-Schulz on M^T is the
    transpose of Newton-Schulz on M (X X^T and X^T X give the same X_n)."""
    rng = np.random.default_rng(53)
    M = rng.standard_normal((5, 12))
    coeffs = [(3.0, -3.2, 1.2), (2.0, -1.5, 0.5), (1.5, -0.5, 0.0)]
    np.testing.assert_allclose(newton_schulz(M.T, coeffs, 1e-7), newton_schulz(M, coeffs, 1e-7).T, atol=1e-12)


def test_orthogonalized_update_is_orthogonal_after_many_steps():
    """Enough cubic iterations make the rows of X_n orthonormal (rows <= cols)."""
    rng = np.random.default_rng(54)
    M = rng.standard_normal((8, 20))
    X = newton_schulz(M, [(1.5, -0.5, 0.0)] * 80, 1e-7)
    np.testing.assert_allclose(X @ X.T, np.eye(8), atol=1e-9)


def test_bf16_rounding_matches_the_format():
    """bfloat16 keeps 8 significant bits: 1 + 2^-8 rounds to 1 (tie, to even), 1 + 3 * 2^-8 to
    1 + 2^-6, and values already representable stay put."""
    x = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, 1.5, -2.0 ** -20, 3.0e38])
    r = bf16_round(x)
    assert r[0] == 1.0 and r[1] == 1.0 + 2.0 ** -6 and r[2] == 1.5 and r[3] == -2.0 ** -20
    assert abs(r[4] - 3.0e38) / 3.0e38 < 2.0 ** -8
