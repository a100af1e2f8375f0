"""Properties of the Muon oracle's orthogonalization that hold for every coefficient schedule:
each Newton-Schulz step is an odd polynomial in X of the form a X + (b XX^T + c (XX^T)^2) X, so
the result commutes with orthogonal changes of basis on either side, is odd in M, and (through
the normalisation by ||M||_F) does not depend on M's scale. Random cases by hypothesis."""
import numpy as np
import pytest

pytest.importorskip("hypothesis")
from hypothesis import assume, given, settings, strategies as st  # noqa: E402

from oracle.muon_ref import MuonParams, MuonState, muon_step, newton_schulz  # noqa: E402

QUINTIC = (15 / 8, -10 / 8, 3 / 8)
CUBIC = (1.5, -0.5, 0.0)

schedules = st.one_of(
    st.just([CUBIC] * 12),
    st.just([QUINTIC] * 8),
    st.lists(st.tuples(st.floats(-2, 2), st.floats(-2, 2), st.floats(-1, 1)), min_size=1, max_size=4),
)


def _orth(rng, n):
    q, r = np.linalg.qr(rng.standard_normal((n, n)))
    return q * np.sign(np.diag(r))


@settings(max_examples=60, deadline=None)
@given(st.integers(1, 8), st.integers(1, 8), schedules, st.floats(1e-3, 1e3), st.integers(0, 2 ** 31 - 1))
def test_newton_schulz_equivariance_oddness_and_scale(rows, cols, coeffs, scale, seed):
    rng = np.random.default_rng(seed)
    M = rng.standard_normal((rows, cols))
    assume(min(1.0, scale) * np.linalg.norm(M) > 1e-5)   # the eps floor stays inactive
    X = newton_schulz(M, coeffs, 1e-7)
    tol = 1e-9 * max(1.0, np.abs(X).max())
    U, V = _orth(rng, rows), _orth(rng, cols)
    np.testing.assert_allclose(newton_schulz(U @ M @ V.T, coeffs, 1e-7), U @ X @ V.T, rtol=0, atol=tol)
    np.testing.assert_allclose(newton_schulz(-M, coeffs, 1e-7), -X, rtol=0, atol=tol)
    np.testing.assert_allclose(newton_schulz(scale * M, coeffs, 1e-7), X, rtol=0, atol=tol)
    # the orientation: Newton-Schulz of M^T is the transpose of Newton-Schulz of M
    np.testing.assert_allclose(newton_schulz(M.T, coeffs, 1e-7), X.T, rtol=0, atol=tol)


@settings(max_examples=40, deadline=None)
@given(st.integers(1, 8), st.integers(1, 8), st.integers(1, 4), st.integers(0, 2 ** 31 - 1))
def test_step_is_the_decoupled_update_of_the_orthogonalized_momentum(rows, cols, steps, seed):
    rng = np.random.default_rng(seed)
    hp = MuonParams(coeffs=[QUINTIC] * 8)
    s = MuonState(rows, cols)
    W = rng.standard_normal((rows, cols))
    M = np.zeros((rows, cols))
    for _ in range(steps):
        G = rng.standard_normal((rows, cols))
        M = hp.beta1 * M + (1 - hp.beta1) * G
        W_new, dW = muon_step(s, W, G, hp)
        np.testing.assert_allclose(s.M, M, rtol=0, atol=1e-14)
        np.testing.assert_allclose(dW, np.sqrt(max(rows, cols)) * newton_schulz(M, hp.coeffs, hp.eps),
                                   rtol=0, atol=1e-12)
        np.testing.assert_allclose(W_new, (1 - hp.lr * hp.weight_decay) * W - hp.lr * dW, rtol=0, atol=1e-12)
        W = W_new
