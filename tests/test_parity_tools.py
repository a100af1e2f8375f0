"""The parity checker itself, on the host: a stand-in for the GPU handle that steps the oracle's
own fp32 twin passes it on the 256x512 workload (steps beyond fp32 resolution included), and the
same stand-in with a planted mistake in its step fails it."""
import numpy as np
import pytest
import torch

from oracle.soap_ref import HParams, MatrixState, soap_step
from paper_2607_20548_gb300 import soap as S
from paper_2607_20548_gb300.workloads import make_stream

from tests.parity_tools import TeacherForcedCheck


class _TwinHandle:
    """Answers the checker's state_get like a libsoap handle, stepping an fp32 oracle state on the
    host; `plant` alters its update to show that the checker catches a mistake."""

    def __init__(self, rows, cols, hp, plant=None):
        self.shapes = [S.Shape(rows, cols, True, True)]
        self.st = MatrixState(rows, cols, True, True, np.float32)
        self.hp = hp
        self.plant = plant

    @property
    def t(self):
        return self.st.t

    def step(self, W, G):
        Wn, _ = soap_step(self.st, W.numpy(), G.numpy(), self.hp)
        if self.plant == "no_weight_decay":
            Wn = Wn + (self.hp.lr * self.hp.weight_decay) * W.numpy()
        elif self.plant == "transposed_left_basis":
            dW = (W.numpy() * (1 - self.hp.lr * self.hp.weight_decay) - Wn) / self.hp.lr
            Wn = W.numpy() * (1 - self.hp.lr * self.hp.weight_decay) - self.hp.lr * (self.st.QL.T @ self.st.QL.T @ dW)
        W.copy_(torch.from_numpy(np.ascontiguousarray(Wn, np.float32)))

    def state_get(self, idx, which):
        st = self.st
        v = {S.STATE_M: st.m, S.STATE_V: st.v, S.STATE_L: st.L, S.STATE_QL: st.QL, S.STATE_R: st.R,
             S.STATE_QR: st.QR, S.STATE_SKIP_L: st.skipL.astype(np.uint8),
             S.STATE_SKIP_R: st.skipR.astype(np.uint8)}[which]
        return torch.from_numpy(np.ascontiguousarray(v))


def _run(plant, steps):
    hp = HParams()
    s = make_stream("single_256x512", seed=0, device="cpu")
    W = s.weights()[0][0].clone()
    h = _TwinHandle(256, 512, hp, plant)
    chk = TeacherForcedCheck(h, hp)
    for t in range(1, steps + 1):
        G = s.grads(t)[0][0]
        chk.before(0, W, G)
        h.step(W, G)
        chk.after(0, W)
    return chk


def test_checker_accepts_a_faithful_fp32_step():
    chk = _run(None, 4)
    print("\n" + chk.report())
    chk.assert_ok()
    assert chk.rows[1]["amplified"] > 0            # step 2 rotates momentum outside Adam's range
    assert all(r["e_mask"] <= 1e-3 for r in chk.rows)


@pytest.mark.parametrize("plant", ["no_weight_decay", "transposed_left_basis"])
def test_checker_rejects_a_planted_mistake(plant):
    chk = _run(plant, 3)
    with pytest.raises(AssertionError):
        chk.assert_ok()


@pytest.mark.parametrize("b1, b2", [(0.95, 0.95), (0.9, 0.95), (0.5, 0.99)])
def test_adam_normal_range(b1, b2):
    """The checker's normal range: without a basis change, |m| / sqrt(v) never exceeds
    normal_bound (1 for beta1 = beta2), on random gradient sequences including ones that flip
    sign and span six decades; the bound is reached by the worst case it is derived from."""
    from tests.parity_tools import normal_bound
    rng = np.random.default_rng(3)
    hp = HParams(beta1=b1, beta2=b2)
    worst = 0.0
    for _ in range(200):
        g = rng.standard_normal(50) * 10.0 ** rng.uniform(-3, 3, 50)
        m = v = 0.0
        for x in g:
            m = b1 * m + (1 - b1) * x
            v = b2 * v + (1 - b2) * x * x
            worst = max(worst, abs(m) / np.sqrt(v))
    assert worst <= normal_bound(hp)
    # equality case of Cauchy-Schwarz: the gradient of age k proportional to (b1 / b2)^k
    k = np.arange(400)[::-1]
    m = v = 0.0
    for x in (b1 / b2) ** k:
        m = b1 * m + (1 - b1) * x
        v = b2 * v + (1 - b2) * x * x
    assert abs(m) / np.sqrt(v) >= 0.999 * normal_bound(hp)
