"""Workspace waves: a model whose step workspace is capped is stepped in several waves of
matrices, each reusing one workspace arena. The result must not depend on the plan: the
same matrices stepped in one wave and in many give the same weights and state, and both
follow the oracle."""
import numpy as np
import pytest
import torch

from paper_2607_20548_gb300 import soap as S

from tests.parity_tools import TeacherForcedCheck, oracle_hparams

pytestmark = pytest.mark.gpu

# two-sided, left-only (stored transposed), right-only tensor-core classes, a CUDA-core class
# (30 columns) and several matrices per class, so that classes are cut into slices
SHAPES = ([(96, 160, True, True)] * 5 + [(64, 304, True, False)] * 3 + [(300, 64, False, True)] * 2
          + [(32, 30, True, False)] * 2 + [(128, 96, True, True)] * 4)


def _inputs(cuda, steps, seed=17):
    g = torch.Generator(device=cuda).manual_seed(seed)
    W = [(0.02 * torch.randn(r, c, device=cuda, generator=g)).contiguous() for r, c, _, _ in SHAPES]
    A = [torch.randn(r, c, device=cuda, generator=g) / np.sqrt(r * c) for r, c, _, _ in SHAPES]
    Gs = [[(a + 0.3 * torch.randn(a.shape, device=cuda, generator=g) / np.sqrt(a.shape[1])).contiguous() for a in A]
          for _ in range(steps)]
    return W, Gs


def _limit_for_waves(cuda, hp, pipelined):
    """A workspace bound under which the model takes at least 3 waves, pipelined (two waves in
    halves of the workspace) or one after another: found by shrinking the one-wave plan's size."""
    probe = S.SoapOptimizer(SHAPES, hp)
    info = probe.plan_info()
    probe.destroy()
    assert info["waves"] == 1
    for divisor in (2.5, 3, 4, 5, 6, 8, 10, 12, 16, 20, 24, 32):
        limit = int(info["workspace_bytes"] / divisor)
        try:
            opt = S.SoapOptimizer(SHAPES, hp, workspace_limit=limit)
        except S.SoapError:
            break
        plan = opt.plan_info()
        opt.destroy()
        if plan["waves"] >= 3 and plan["pipelined"] == pipelined:
            return limit
    pytest.fail(f"no workspace limit gives >= 3 {'pipelined' if pipelined else 'serial'} waves")


@pytest.mark.parametrize("pipelined", [True, False])
@pytest.mark.parametrize("variant", [dict(), dict(kl=1), dict(stale=1, guard=0), dict(eig_every=2)])
def test_waves_match_one_wave(cuda, variant, pipelined):
    hp = S.default_hparams(**variant)
    steps = 5
    W0, Gs = _inputs(cuda, steps)
    one = S.SoapOptimizer(SHAPES, hp)
    many = S.SoapOptimizer(SHAPES, hp, workspace_limit=_limit_for_waves(cuda, hp, pipelined))
    info = many.plan_info()
    print(f"\nplan: {info}")
    assert info["waves"] >= 3 and info["pipelined"] == pipelined
    Wa = [w.clone() for w in W0]
    Wb = [w.clone() for w in W0]
    for t in range(steps):
        one.step(Wa, Gs[t])
        many.step(Wb, Gs[t])
        torch.cuda.synchronize()
        assert one.status() == 0 and many.status() == 0
        worst = max((a - b).abs().max().item() / max(1e-30, (a - w).abs().max().item())
                    for a, b, w in zip(Wa, Wb, W0))
        print(f"step {t + 1}: largest difference / largest update {worst:.2e}")
        # the same kernels on the same matrices: a plan only regroups the batched launches
        assert worst <= 1e-5
    for i in range(len(SHAPES)):
        for which in (S.STATE_MHAT, S.STATE_V, S.STATE_L, S.STATE_QL, S.STATE_R, S.STATE_QR):
            if one.state_bytes(i, which):
                a, b = one.state_get(i, which), many.state_get(i, which)
                scale = max(1e-30, a.abs().max().item())
                assert (a - b).abs().max().item() <= 1e-5 * scale, (i, which)
    one.destroy()
    many.destroy()


def test_waves_against_oracle(cuda):
    """Matrices of every class, stepped in several waves, teacher-forced against the oracle."""
    hp = S.default_hparams()
    steps = 6
    W, Gs = _inputs(cuda, steps, seed=23)
    opt = S.SoapOptimizer(SHAPES, hp, workspace_limit=_limit_for_waves(cuda, hp, True))
    assert opt.plan_info()["waves"] >= 3 and opt.plan_info()["pipelined"]
    chk = TeacherForcedCheck(opt, oracle_hparams(hp))
    sample = [0, 4, 5, 8, 10, 12, 15]
    for t in range(steps):
        for i in sample:
            chk.before(i, W[i], Gs[t][i])
        opt.step(W, Gs[t])
        torch.cuda.synchronize()
        assert opt.status() == 0, opt.last_error()
        for i in sample:
            chk.after(i, W[i])
    print("\n" + chk.report())
    chk.assert_ok()
    opt.destroy()


def test_workspace_limit_too_small_is_oom(cuda):
    with pytest.raises(S.SoapError) as e:
        S.SoapOptimizer([(256, 512)], S.default_hparams(), workspace_limit=4096)
    assert e.value.code == 3  # SOAP_ERR_OOM


def test_state_round_trip_of_packed_factors(cuda):
    """L and R are stored as packed lower tiles: state_set of a symmetric factor reads back
    exactly, and a ragged size (not a multiple of the 32-wide tile) keeps its edge."""
    opt = S.SoapOptimizer([(100, 68, True, True)])
    g = torch.Generator(device=cuda).manual_seed(3)
    for which, n in ((S.STATE_L, 100), (S.STATE_R, 68)):
        X = torch.randn(n, n, device=cuda, generator=g)
        F = (X @ X.T).contiguous()
        F = 0.5 * (F + F.T)
        opt.state_set(0, which, F)
        back = opt.state_get(0, which)
        torch.cuda.synchronize()
        assert torch.equal(back, torch.tril(F) + torch.tril(F, -1).T)
    opt.destroy()
