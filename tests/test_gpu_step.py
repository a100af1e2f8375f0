"""Whole-step parity of soap_step (through the C ABI) with the fp64 oracle on seeded workloads."""
import numpy as np
import pytest
import torch

from oracle.soap_ref import HParams, MatrixState, soap_step
from paper_2607_20548_gb300 import soap as S
from paper_2607_20548_gb300.workloads import WORKLOADS, make_stream

from tests.parity_tools import TeacherForcedCheck, oracle_hparams, orth_err, rel

pytestmark = pytest.mark.gpu


def _flat(stream, tensors):
    """Per-matrix views of per-group [batch, rows, cols] tensors, in matrix order."""
    out = [None] * sum(len(idx) for _, idx in stream.groups)
    for (spec, idx), t in zip(stream.groups, tensors):
        for b, j in enumerate(idx):
            out[j] = t[b]
    return out


def _run_teacher_forced(cuda, name, steps, sample, hp=None, specs=None, check_steps=None):
    hp = hp or S.default_hparams()
    stream = make_stream(name, seed=0, device=cuda, specs=specs)
    shapes = [(s.rows, s.cols, s.left, s.right) for s in stream.specs]
    opt = S.SoapOptimizer(shapes, hp)
    W = _flat(stream, [w.contiguous() for w in stream.weights()])
    chk = TeacherForcedCheck(opt, oracle_hparams(hp))
    for t in range(1, steps + 1):
        G = _flat(stream, stream.grads(t))
        active = [] if (check_steps is not None and t not in check_steps) else sample
        for i in active:
            chk.before(i, W[i], G[i])
        opt.step(W, G)
        torch.cuda.synchronize()
        assert opt.status() == 0, opt.last_error()
        for i in active:
            chk.after(i, W[i])
    print("\n" + chk.report())
    return opt, chk


def test_single_256x512_20_steps(cuda):
    """The 256x512 workload, 20 steps, every step teacher-forced against the fp64 oracle."""
    opt, chk = _run_teacher_forced(cuda, "single_256x512", 20, [0])
    chk.assert_ok()
    assert all(r["skipL_same"] and r["skipR_same"] for r in chk.rows)
    # every step whose N stays in Adam's normal range meets the 1e-3 bound outright, and on every
    # step the update on that range does
    assert all(r["e_gpu"] <= 1e-3 for r in chk.rows if r["amplified"] == 0)
    assert all(r["e_mask"] <= 1e-3 for r in chk.rows)
    assert sum(r["ill"] for r in chk.rows) <= 2
    opt.destroy()


def _free_running(cuda, name, steps, sample):
    """Every matrix of the workload stepped on the GPU for `steps` steps, and the sampled ones in
    the fp64 oracle and its fp32 twin from the same inputs, all three free-running. Returns per
    (matrix, step) the relative Frobenius errors of the GPU's and the twin's update against fp64."""
    hp = S.default_hparams()
    ohp = oracle_hparams(hp)
    stream = make_stream(name, seed=0, device=cuda)
    shapes = [(s.rows, s.cols, s.left, s.right) for s in stream.specs]
    opt = S.SoapOptimizer(shapes, hp)
    W = _flat(stream, [w.contiguous() for w in stream.weights()])
    ref = {}
    for i in sample:
        r, c, left, right = shapes[i]
        w0 = W[i].cpu().numpy()
        ref[i] = dict(st64=MatrixState(r, c, left, right, np.float64), st32=MatrixState(r, c, left, right, np.float32),
                      W64=w0.astype(np.float64), W32=w0.copy())
    rows = []
    for t in range(1, steps + 1):
        G = _flat(stream, stream.grads(t))
        Wp = {i: W[i].cpu().double().numpy() for i in sample}
        opt.step(W, G)
        torch.cuda.synchronize()
        assert opt.status() == 0, opt.last_error()
        for i in sample:
            x = ref[i]
            Gh = G[i].cpu().numpy()
            W64n, _ = soap_step(x["st64"], x["W64"], Gh, ohp)
            W32n, _ = soap_step(x["st32"], x["W32"], Gh, ohp)
            d64 = W64n - x["W64"]
            rows.append((i, t, rel(W[i].cpu().double().numpy() - Wp[i], d64),
                         rel(W32n.astype(np.float64) - x["W32"], d64)))
            x["W64"], x["W32"] = W64n, W32n
    opt.destroy()
    return rows


def _assert_free_running(rows):
    """Per step and matrix: the GPU's update within 1e-3 of fp64, or within 2x the fp32 twin's
    own free-running error where the twin -- a faithful fp32 implementation -- parts from fp64
    (after a step beyond fp32 resolution both trajectories differ from fp64 by the rounding that
    step amplified)."""
    print("\n" + "\n".join(f"matrix {i:4d} t={t:2d}: gpu {e:.2e} twin {e32:.2e}" for i, t, e, e32 in rows))
    bad = [(i, t, e, e32) for i, t, e, e32 in rows if not e <= max(1e-3, 2.0 * e32)]
    assert not bad, bad


def test_single_256x512_free_running_against_fp64(cuda):
    """Free-running 20 steps on the GPU and in the fp64 oracle from identical inputs: every step's
    update within max(1e-3, 2 x the fp32 twin's free-running error)."""
    rows = _free_running(cuda, "single_256x512", 20, [0])
    _assert_free_running(rows)
    assert rows[0][2] <= 1e-3


def test_moe_layer_free_running_sample(cuda):
    """The fine-grained MoE layer, all 193 matrices stepped on the GPU, free-running for its 20
    steps; the gate of expert 0, the up of expert 5, the down of expert 9 and the router followed
    in the fp64 oracle and its fp32 twin, each step bounded as above."""
    rows = _free_running(cuda, "moe_layer_64x768_h2048", 20, [0, 64 + 5, 128 + 9, 192])
    _assert_free_running(rows)


@pytest.mark.parametrize("shape", [(64, 300, True, False), (300, 64, False, True), (16, 24, False, False),
                                   (48, 40, True, True), (64, 304, True, False), (304, 64, False, True),
                                   (1028, 96, True, False), (96, 1028, False, True), (260, 1028, True, False)])
def test_one_sided_and_identity_matrices(cuda, shape):
    """Identity sides (Q fixed at I, no factor stored), 8 steps against the oracle. Sides
    that are multiples of 4 run on the tensor-core path (a left-only matrix as the
    right-only problem of G^T), the others on CUDA cores; 1028 spans several 128-row
    tiles with a ragged tail."""
    rows, cols, left, right = shape
    hp = S.default_hparams()
    opt = S.SoapOptimizer([shape], hp)
    ohp = oracle_hparams(hp)
    chk = TeacherForcedCheck(opt, ohp)
    g = torch.Generator(device=cuda).manual_seed(3)
    W = (0.02 * torch.randn(rows, cols, device=cuda, generator=g)).contiguous()
    for t in range(8):
        G = torch.randn(rows, cols, device=cuda, generator=g) / np.sqrt(cols)
        chk.before(0, W, G)
        opt.step([W], [G])
        chk.after(0, W)
    print("\n" + chk.report())
    chk.assert_ok()


@pytest.mark.parametrize("variant", [dict(eig_every=3), dict(bias_correction=1), dict(guard=0, qr_tol=0.0),
                                     dict(stale=1, guard=0), dict(stale=1, guard=0, eig_every=3)])
def test_variants_against_oracle(cuda, variant):
    """F > 1 (no refresh on most steps), bias correction, the guard/zero-column reading off, and
    section 5's stale variant (the refresh leaves out the current gradient), every step and every
    third step."""
    hp = S.default_hparams(**variant)
    opt = S.SoapOptimizer([(96, 160)], hp)
    chk = TeacherForcedCheck(opt, oracle_hparams(hp))
    g = torch.Generator(device=cuda).manual_seed(11)
    W = (0.02 * torch.randn(96, 160, device=cuda, generator=g)).contiguous()
    A = torch.randn(96, 160, device=cuda, generator=g) / 8
    for t in range(9):
        G = (A + 0.3 * torch.randn(96, 160, device=cuda, generator=g) / np.sqrt(160)).contiguous()
        chk.before(0, W, G)
        opt.step([W], [G])
        chk.after(0, W)
    print("\n" + chk.report())
    if variant.get("guard", 1) == 0 and not variant.get("stale"):
        # without the guard, fp32 junk in the zero directions decides the update: bound by the twin only
        assert all(np.isfinite(r["e_gpu"]) for r in chk.rows)
    else:
        chk.assert_ok()


def test_moe_layer_all_193_matrices(cuda):
    """The fine-grained MoE layer (128 x 2048x768, 64 x 768x2048, router 2048x64) as one batched
    step for 20 steps; sampled matrices teacher-forced against the oracle on chosen steps."""
    sample = [0, 64 + 5, 128 + 9, 192]  # gate of expert 0, up of expert 5, down of expert 9, router
    opt, chk = _run_teacher_forced(cuda, "moe_layer_64x768_h2048", 20, sample, check_steps={1, 2, 3, 20})
    chk.assert_ok()
    opt.destroy()


@pytest.mark.parametrize("shape", [(64, 304, True, False), (300, 64, False, True), (48, 40, True, True)])
def test_stale_variant_one_sided_and_small(cuda, shape):
    """The stale variant on a left-only tensor-core class (run as the right-only problem of G^T),
    a right-only CUDA-core class and a small two-sided class, 8 steps against the oracle."""
    rows, cols, left, right = shape
    hp = S.default_hparams(stale=1, guard=0)
    opt = S.SoapOptimizer([shape], hp)
    chk = TeacherForcedCheck(opt, oracle_hparams(hp))
    g = torch.Generator(device=cuda).manual_seed(13)
    W = (0.02 * torch.randn(rows, cols, device=cuda, generator=g)).contiguous()
    A = torch.randn(rows, cols, device=cuda, generator=g) / np.sqrt(rows * cols)
    for t in range(8):
        G = (A + 0.3 * torch.randn(rows, cols, device=cuda, generator=g) / np.sqrt(cols)).contiguous()
        chk.before(0, W, G)
        opt.step([W], [G])
        chk.after(0, W)
    print("\n" + chk.report())
    chk.assert_ok()
    opt.destroy()


def test_moe_stack_24x_sample(cuda):
    """The 24-layer MoE stack (4706 matrices) does not fit one GPU's HBM with every matrix's
    state resident, and its matrices are independent, so a deterministic sample is stepped as
    one batch for the workload's 10 steps: layers 0 and 23 (Wq, Wk, Wv, Wo and experts 0, 31, 63
    with gate, up and down each) plus the embedding and the LM head (2048x32768, left side only).
    Teacher-forced against the oracle on steps 1, 2 and 10 for one matrix of each shape class."""
    per_layer = 4 + 192
    sample = []
    for layer in (0, 23):
        base = layer * per_layer
        sample += [base + j for j in range(4)]
        for e in (0, 31, 63):
            sample += [base + 4 + e, base + 4 + 64 + e, base + 4 + 128 + e]
    sample += [24 * per_layer, 24 * per_layer + 1]
    checked = [0, 4, 6, len(sample) - 1]  # Wq of layer 0, gate and down of expert 0, LM head
    opt, chk = _run_teacher_forced(cuda, "moe_stack_24x_h2048", 10, checked, specs=sample,
                                   check_steps={1, 2, 10})
    chk.assert_ok()
    opt.destroy()


def test_dense_block_full_size(cuda):
    """The dense block (hidden 2048, FFN 8192) at full size for 20 steps. Wq is teacher-forced
    against the oracle on steps 1-3 and 20; every matrix's refreshed bases are orthogonal to 1e-5
    on every step (the 8192-sided factors are too large for the oracle's unblocked QR)."""
    hp = S.default_hparams()
    name = "dense_block_h2048_ffn8192"
    stream = make_stream(name, seed=0, device=cuda)
    shapes = [(s.rows, s.cols, s.left, s.right) for s in stream.specs]
    opt = S.SoapOptimizer(shapes, hp)
    W = _flat(stream, [w.contiguous() for w in stream.weights()])
    chk = TeacherForcedCheck(opt, oracle_hparams(hp))
    worst = 0.0
    for t in range(1, 21):
        G = _flat(stream, stream.grads(t))
        if t in (1, 2, 3, 20):
            chk.before(0, W[0], G[0])
        opt.step(W, G)
        torch.cuda.synchronize()
        assert opt.status() == 0, opt.last_error()
        if t in (1, 2, 3, 20):
            chk.after(0, W[0])
        if t in (1, 2, 5, 20):
            for i in (0, 4, 6):
                for which in (S.STATE_QL, S.STATE_QR):
                    worst = max(worst, orth_err(opt.state_get(i, which)))
    print("\n" + chk.report() + f"\nworst ||Q^T Q - I||_max over sampled steps: {worst:.2e}")
    assert worst <= 1e-5
    chk.assert_ok()
    opt.destroy()


def test_checkpoint_resume_is_bit_exact(cuda):
    """state_get/state_set of every piece (M_hat, v, L, Q_L, R, Q_R, skip flags, t) round-trips:
    3 steps, save, 3 more steps == restore into a new handle and run the same 3 steps."""
    # two-sided, left-only and right-only tensor-core classes (the left-only one stores M_hat
    # and v transposed) and a CUDA-core class (30 columns: not a multiple of 4)
    shapes = [(40, 72, True, True), (72, 40, True, False), (44, 36, False, True), (32, 30, True, False)]
    hp = S.default_hparams()
    g = torch.Generator(device=cuda).manual_seed(7)
    Ws = [(0.02 * torch.randn(r, c, device=cuda, generator=g)).contiguous() for r, c, _, _ in shapes]
    Gs = [[torch.randn(r, c, device=cuda, generator=g).contiguous() for r, c, _, _ in shapes] for _ in range(6)]
    a = S.SoapOptimizer(shapes, hp)
    for t in range(3):
        a.step(Ws, Gs[t])
    pieces = (S.STATE_MHAT, S.STATE_V, S.STATE_L, S.STATE_QL, S.STATE_R, S.STATE_QR, S.STATE_SKIP_L, S.STATE_SKIP_R)
    saved = {(i, w): a.state_get(i, w).clone() for i in range(len(shapes)) for w in pieces
             if a.state_bytes(i, w) > 0}
    W_saved = [w.clone() for w in Ws]
    t_saved = a.t
    for t in range(3, 6):
        a.step(Ws, Gs[t])
    b = S.SoapOptimizer(shapes, hp)
    for (i, w), v in saved.items():
        b.state_set(i, w, v)
    b.t = t_saved
    Wb = [w.clone() for w in W_saved]
    for t in range(3, 6):
        b.step(Wb, Gs[t])
    torch.cuda.synchronize()
    for x, y in zip(Ws, Wb):
        assert torch.equal(x, y)
    # the rotated-basis first moment round-trips to fp32 rounding
    for i in range(len(shapes)):
        m = a.state_get(i, S.STATE_M)
        b.state_set(i, S.STATE_M, m)
        assert (b.state_get(i, S.STATE_MHAT) - a.state_get(i, S.STATE_MHAT)).abs().max().item() < 1e-6
    a.destroy()
    b.destroy()


def test_nonfinite_gradient_sets_sticky_status(cuda):
    opt = S.SoapOptimizer([(32, 48)])
    W = torch.zeros(32, 48, device=cuda)
    G = torch.randn(32, 48, device=cuda)
    G[3, 5] = float("nan")
    opt.step([W], [G])
    assert opt.status() == 4  # SOAP_ERR_NONFINITE
    with pytest.raises(S.SoapError):
        opt.step([W], [torch.randn(32, 48, device=cuda)])
    opt.clear_status()
    assert opt.status() == 0
    opt.destroy()


def test_invalid_arguments(cuda):
    opt = S.SoapOptimizer([(32, 48)])
    buf = torch.zeros(32 * 48 + 4, device=cuda)
    W = buf[1:1 + 32 * 48].view(32, 48)  # 4-byte offset: not 16-byte aligned
    G = torch.zeros(32, 48, device=cuda)
    with pytest.raises(S.SoapError) as e:
        opt.step([W], [G])
    assert e.value.code == 1
    with pytest.raises(S.SoapError):
        opt.state_get(0, 99)
    opt.destroy()
    lib = S.load_library()
    assert lib.soap_qr(9000, 1, None, None, None, 0.0, None, 0, None, None) == 1
