"""Sub-step parity on the GPU through the C ABI: the batched GEMM and the QR refresh."""
import numpy as np
import pytest
import torch

from oracle.soap_ref import householder_q
from paper_2607_20548_gb300 import soap as S

pytestmark = pytest.mark.gpu


def _rel(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("ta,tb", [(False, False), (False, True), (True, False), (True, True)])
@pytest.mark.parametrize("M,N,K,batch", [(1, 1, 1, 1), (37, 129, 65, 3), (128, 128, 8, 2), (300, 70, 513, 2),
                                         (33, 2049, 31, 1), (1000, 1000, 1000, 1)])
def test_gemm_matches_fp64(cuda, ta, tb, M, N, K, batch):
    g = torch.Generator().manual_seed(M * 7 + N * 13 + K)
    A = torch.randn(batch, *((K, M) if ta else (M, K)), generator=g)
    B = torch.randn(batch, *((N, K) if tb else (K, N)), generator=g)
    C0 = torch.randn(batch, M, N, generator=g)
    alpha, beta = 0.7, -0.3
    C = C0.clone().to(cuda)
    S.soap_gemm(A.to(cuda), B.to(cuda), ta, tb, alpha, beta, C)
    A64, B64 = A.double().numpy(), B.double().numpy()
    opA = np.transpose(A64, (0, 2, 1)) if ta else A64
    opB = np.transpose(B64, (0, 2, 1)) if tb else B64
    ref = alpha * opA @ opB + beta * C0.double().numpy()
    # fp32 accumulation over K terms: relative error ~ sqrt(K) * 2^-24
    assert _rel(C.cpu().double().numpy(), ref) < 2e-6 * max(1.0, np.sqrt(K) / 8)


def test_gemm_beta_zero_ignores_c(cuda):
    A = torch.randn(64, 64, device=cuda)
    B = torch.randn(64, 64, device=cuda)
    C = torch.full((64, 64), float("nan"), device=cuda)
    S.soap_gemm(A, B, C=C, beta=0.0)
    assert torch.isfinite(C).all()


def _qr_case(n, batch, kind, seed):
    rng = np.random.default_rng(seed)
    if kind == "well":
        return np.stack([np.eye(n) + 0.1 * rng.standard_normal((n, n)) / np.sqrt(n) for _ in range(batch)]).astype(np.float32)
    if kind == "gauss":
        return rng.standard_normal((batch, n, n)).astype(np.float32)
    if kind == "lowrank":
        r = max(1, n // 3)
        X = rng.standard_normal((batch, n, r))
        return (X @ np.transpose(X, (0, 2, 1))).astype(np.float32)  # PSD of rank r, like G G^T at step 1
    raise ValueError(kind)


@pytest.mark.parametrize("n,batch,kind", [(4, 1, "well"), (36, 2, "well"), (32, 1, "gauss"), (36, 3, "gauss"),
                                          (100, 2, "lowrank"), (516, 2, "well"), (1028, 1, "well"),
                                          (768, 2, "lowrank"), (2048, 1, "well"), (2048, 1, "lowrank"),
                                          (200, 2, "lowrank"), (644, 1, "gauss")])
def test_qr_matches_oracle(cuda, n, batch, kind):
    """S3 on identical fp32 inputs: skip flags equal the oracle's, Q^T Q = I to 1e-5, and Q agrees
    with the fp64 oracle to within 4x the oracle's own fp32 twin (the problem's fp32 resolution)."""
    tol = 1e-4
    P = _qr_case(n, batch, kind, seed=n + batch)
    Q, skip = S.soap_qr(torch.from_numpy(P).to(cuda), tol)
    Q = Q.cpu().numpy()
    skip = skip.cpu().numpy().astype(bool)
    for b in range(batch):
        Q64, s64, _ = householder_q(P[b].astype(np.float64), tol)
        Q32, _, _ = householder_q(P[b], tol)
        assert np.array_equal(skip[b], s64)
        orth = np.abs(Q[b].astype(np.float64).T @ Q[b] - np.eye(n)).max()
        assert orth <= 1e-5, orth
        keep = ~s64  # columns of the zero-column completion are compared through orthogonality only
        e_gpu = _rel(Q[b][:, keep], Q64[:, keep])
        e_twin = _rel(Q32[:, keep].astype(np.float64), Q64[:, keep])
        assert e_gpu <= max(1e-5, 4 * e_twin), (e_gpu, e_twin)
        if s64.any():
            # the columns completing a rank-deficient P (H_1 ... H_k-1 e_k) follow the oracle too
            c_gpu = _rel(Q[b][:, s64], Q64[:, s64])
            c_twin = _rel(Q32[:, s64].astype(np.float64), Q64[:, s64])
            assert c_gpu <= max(1e-5, 4 * c_twin), (c_gpu, c_twin)


def test_qr_batched_column_kernel(cuda):
    """A batch of 16 factors of more than 1024 rows takes the panel's column loop as a kernel of
    its own (two CTAs per SM) before the block product, T and the in-block update: the same checks
    as above on three members of the batch (rank-deficient, well-conditioned and Gaussian), and
    orthogonality on all of them."""
    n, batch, tol = 1028, 16, 1e-4
    P = np.concatenate([_qr_case(n, 6, "lowrank", seed=11), _qr_case(n, 5, "well", seed=12),
                        _qr_case(n, 5, "gauss", seed=13)])
    Q, skip = S.soap_qr(torch.from_numpy(P).to(cuda), tol)
    Qd = Q.double()
    eye = torch.eye(n, dtype=torch.float64, device=cuda)
    for b in range(batch):
        assert (Qd[b].T @ Qd[b] - eye).abs().max().item() <= 1e-5, b
    Q = Q.cpu().numpy()
    skip = skip.cpu().numpy().astype(bool)
    for b in (0, 6, 11):
        Q64, s64, _ = householder_q(P[b].astype(np.float64), tol)
        Q32, _, _ = householder_q(P[b], tol)
        assert np.array_equal(skip[b], s64), b
        keep = ~s64
        e_gpu = _rel(Q[b][:, keep], Q64[:, keep])
        e_twin = _rel(Q32[:, keep].astype(np.float64), Q64[:, keep])
        assert e_gpu <= max(1e-5, 4 * e_twin), (b, e_gpu, e_twin)


def test_qr_rejects_sizes_not_multiple_of_4(cuda):
    """The QR's tensor-core products read rows with TMA (16-byte rows): n must be a multiple of 4."""
    with pytest.raises(S.SoapError) as err:
        S.soap_qr(torch.eye(33, device=cuda).unsqueeze(0), 1e-4)
    assert err.value.code == 1


def test_qr_full_size_8192_properties(cuda):
    """n = 8192 (the largest factor of the dense block and the 8192-wide layer), on a PSD factor of
    rank 2048 plus a tiny ridge, like L after a few steps: Q^T Q = I to 1e-5; R = Q^T P is upper
    triangular with diag(R) >= 0 in every Householder column; a column treated as zero keeps its
    unreflected sub-column, whose norm is at most tol * ||P||_F by the zero-column reading."""
    n, tol = 8192, 1e-4
    g = torch.Generator(device=cuda).manual_seed(5)
    X = torch.randn(n, 2048, device=cuda, generator=g)
    P = (X @ X.T + 1e-3 * torch.eye(n, device=cuda)).unsqueeze(0)
    Q, skip = S.soap_qr(P, tol)
    skip = skip[0].bool()
    assert 0 < int(skip.sum()) < n
    Qd = Q[0].double()
    I = torch.eye(n, dtype=torch.float64, device=cuda)
    assert (Qd.T @ Qd - I).abs().max().item() <= 1e-5
    del I
    R = Qd.T @ P[0].double()
    fro = P[0].double().norm().item()
    low = torch.tril(R, -1)
    assert low[:, ~skip].abs().max().item() <= 1e-5 * fro
    assert low[:, skip].norm(dim=0).max().item() <= tol * fro * (1 + 1e-3)
    assert torch.diagonal(R)[~skip].min().item() >= 0.0
    del P, Q, R, Qd, X, low
    torch.cuda.empty_cache()


def test_qr_status_word_reports_breakdown(cuda):
    """soap_qr's status word: 0 for a finite input, the QR-breakdown bit where a pivot norm is
    not finite (no exception: the host reads the word once the stream has passed the call)."""
    g = torch.Generator(device=cuda).manual_seed(9)
    X = torch.randn(2, 128, 128, device=cuda, generator=g)
    P = (X @ X.transpose(1, 2)).contiguous()
    _, _, status = S.soap_qr(P, 1e-4, return_status=True)
    torch.cuda.synchronize()
    assert status.item() == 0
    P[1, 0, 5] = float("inf")
    _, _, status = S.soap_qr(P, 1e-4, return_status=True)
    torch.cuda.synchronize()
    assert status.item() & S.STATUS_QR_BREAKDOWN
