"""Alg. Muon on the GPU (include/muon.h) against the oracle (oracle/muon_ref.py).

The Newton-Schulz iterations run in bf16 as the paper runs them (bf16 operands and stored
results, fp32 accumulation), so the GPU is compared with the oracle's bf16 twin, which rounds
to bf16 at the same points (X_0, A, B, X_i) in otherwise exact arithmetic, and with the fp64
oracle. Teacher forcing: before each checked step the GPU's momentum is copied out and the
oracle applies the step to it with the same gradient.

Tolerance (from the arithmetic): a bf16 result carries a relative rounding error of at most
2^-9 per element; each iteration stores three of them, the tensor core's fp32 accumulation
order differs from the oracle's, and an element sitting on a bf16 rounding boundary can round
either way, which the next iterations carry along (Newton-Schulz damps errors along the
singular values it has converged). The update is therefore held to a relative Frobenius error
of 2e-2 (about 10 bf16 units of 2^-9) against the bf16 twin, and against fp64 to the larger
of 2e-2 and twice the twin's own error (where bf16 cannot converge the small singular values,
as for a square matrix, no bf16 implementation gets closer to fp64 than the twin); the
momentum (fp32 arithmetic) to 1e-6.
"""
import numpy as np
import pytest
import torch

from oracle.muon_ref import MuonParams, MuonState, muon_step, newton_schulz
from paper_2607_20548_gb300 import soap as S

pytestmark = pytest.mark.gpu

QUINTIC = [(15 / 8, -10 / 8, 3 / 8)] * 16


def _rel(a, b):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    return np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300)


def _ok(x):
    return x["e16"] <= 2e-2 and x["e64"] <= max(2e-2, 2 * x["e_twin"]) and x["e_m"] <= 1e-6


def _run(cuda, shapes, coeffs, steps, seed=0, check=None):
    g = torch.Generator(device=cuda).manual_seed(seed)
    opt = S.MuonOptimizer(shapes, coeffs=coeffs)
    hp64 = MuonParams(coeffs=list(coeffs))
    hp16 = MuonParams(coeffs=list(coeffs), ns_bf16=True)
    W = [(0.02 * torch.randn(r, c, device=cuda, generator=g)).contiguous() for r, c in shapes]
    A = [torch.randn(r, c, device=cuda, generator=g) / np.sqrt(r * c) for r, c in shapes]
    rows = []
    for t in range(1, steps + 1):
        G = [(a + 0.3 * torch.randn(a.shape, device=cuda, generator=g) / np.sqrt(a.shape[1])).contiguous() for a in A]
        checked = check is None or t in check
        pre = [(opt.state_get(i).cpu().numpy().astype(np.float64), W[i].cpu().numpy().astype(np.float64))
               for i in range(len(shapes))] if checked else None
        opt.step(W, G)
        torch.cuda.synchronize()
        assert opt.status() == 0
        if not checked:
            continue
        for i, (r, c) in enumerate(shapes):
            M0, W0 = pre[i]
            Gh = G[i].cpu().numpy().astype(np.float64)
            W1 = W[i].cpu().numpy().astype(np.float64)
            out = {}
            for name, hp in (("fp64", hp64), ("bf16", hp16)):
                st = MuonState(r, c, np.float64, t - 1, M0.copy())
                Wn, _ = muon_step(st, W0, Gh, hp)
                out[name] = (Wn, st.M)
            e64 = _rel(W1 - W0, out["fp64"][0] - W0)
            e16 = _rel(W1 - W0, out["bf16"][0] - W0)
            e_twin = _rel(out["bf16"][0] - W0, out["fp64"][0] - W0)
            e_m = _rel(opt.state_get(i).cpu().numpy(), out["fp64"][1])
            rows.append(dict(i=i, t=t, shape=(r, c), e64=e64, e16=e16, e_twin=e_twin, e_m=e_m))
    opt.destroy()
    print("\n" + "\n".join(f"{x['shape']} step {x['t']:2d}: gpu vs fp64 {x['e64']:.2e}, vs bf16 twin {x['e16']:.2e}"
                           f" (twin vs fp64 {x['e_twin']:.2e}), momentum {x['e_m']:.1e}" for x in rows))
    return rows


@pytest.mark.parametrize("coeffs", [[(0.0, 1.0, 0.0)], [(0.0, 0.0, 1.0)], [(1.5, -0.5, 0.0)] * 3],
                         ids=["XXtX", "AAX", "cubic3"])
def test_single_products(cuda, coeffs):
    """One to three iterations with schedules that isolate the products: X X^T X (A X), A^2 X
    (the c-term), and three cubic steps; tiles of 128 with ragged edges (136 x 264)."""
    rows = _run(cuda, [(136, 264), (264, 136)], coeffs, 2)
    for x in rows:
        assert _ok(x), x


def test_muon_quintic_16_steps(cuda):
    """The default 16-step quintic schedule on wide, tall (orthogonalized as its transpose),
    flat and square matrices in one batch, 6 steps, every step teacher-forced."""
    shapes = [(256, 512), (512, 256), (64, 2048), (384, 384), (256, 512)]
    rows = _run(cuda, shapes, QUINTIC, 6)
    for x in rows:
        assert _ok(x), x


def test_muon_default_schedule_matches_quintic(cuda):
    """coeffs = None selects the library's quintic schedule: bit-identical to passing it."""
    g = torch.Generator(device=cuda).manual_seed(3)
    G = torch.randn(128, 256, device=cuda, generator=g)
    W0 = torch.randn(128, 256, device=cuda, generator=g)
    Wa, Wb = W0.clone(), W0.clone()
    a = S.MuonOptimizer([(128, 256)], coeffs=None)
    b = S.MuonOptimizer([(128, 256)], coeffs=QUINTIC)
    a.step([Wa], [G])
    b.step([Wb], [G])
    torch.cuda.synchronize()
    assert torch.equal(Wa, Wb)
    a.destroy()
    b.destroy()


def test_muon_orthogonalizes(cuda):
    """With beta1 = 0, lr = 1 and no weight decay the update is X_n sqrt(max(in, out)): after
    the quintic schedule its rows are orthonormal to bf16 accuracy."""
    g = torch.Generator(device=cuda).manual_seed(4)
    G = torch.randn(128, 512, device=cuda, generator=g)
    W = torch.zeros(128, 512, device=cuda)
    opt = S.MuonOptimizer([(128, 512)], lr=1.0, beta1=0.0, weight_decay=0.0, coeffs=QUINTIC)
    opt.step([W], [G])
    torch.cuda.synchronize()
    O = (-W / np.sqrt(512)).double().cpu().numpy()
    err = np.abs(O @ O.T - np.eye(128)).max()
    print(f"\nmax |O O^T - I| = {err:.2e}")
    assert err <= 5e-2
    opt.destroy()


def test_muon_resume_is_bit_exact(cuda):
    """The momentum is Muon's only state: 2 steps, save, 2 more == restore and run the same 2."""
    shapes = [(128, 256), (256, 128)]
    g = torch.Generator(device=cuda).manual_seed(5)
    W = [torch.randn(r, c, device=cuda, generator=g).contiguous() for r, c in shapes]
    Gs = [[torch.randn(r, c, device=cuda, generator=g).contiguous() for r, c in shapes] for _ in range(4)]
    a = S.MuonOptimizer(shapes, coeffs=QUINTIC[:4])
    for t in range(2):
        a.step(W, Gs[t])
    saved = [a.state_get(i).clone() for i in range(2)]
    W2 = [w.clone() for w in W]
    for t in range(2, 4):
        a.step(W, Gs[t])
    b = S.MuonOptimizer(shapes, coeffs=QUINTIC[:4])
    for i in range(2):
        b.state_set(i, saved[i])
    for t in range(2, 4):
        b.step(W2, Gs[t])
    torch.cuda.synchronize()
    for x, y in zip(W, W2):
        assert torch.equal(x, y)
    a.destroy()
    b.destroy()
