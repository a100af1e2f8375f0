"""soap_qr_static: the QR refresh for callers that cannot give the library device memory.

It takes its workspace from a fixed array inside libsoap.so instead of from the caller.
Its results must equal soap_qr's (the same kernels on the same inputs), on consecutive
calls that reuse the array, and it must refuse work larger than the array. This file is
named to be collected last.
"""
import numpy as np
import pytest
import torch

from paper_2607_20548_gb300 import soap as S

pytestmark = pytest.mark.gpu


def _psd(rng, batch, n, rank):
    X = rng.standard_normal((batch, n, rank))
    return (X @ np.transpose(X, (0, 2, 1)) + 1e-3 * np.eye(n)).astype(np.float32)


def test_static_workspace_qr_matches_soap_qr(cuda):
    rng = np.random.default_rng(21)
    # two calls in a row: the second finds the first one's data left in the array
    for n, batch in ((1024, 1), (512, 3)):
        P = torch.from_numpy(_psd(rng, batch, n, n // 2)).to(cuda)
        Q_ref, skip_ref = S.soap_qr(P, 1e-4)
        Q, skip, status = S.soap_qr_static(P, 1e-4, return_status=True)
        torch.cuda.synchronize()
        assert status.item() == 0
        assert torch.equal(skip, skip_ref)
        assert (Q - Q_ref).abs().max().item() <= 1e-5
        Qd = Q.double()
        eye = torch.eye(n, dtype=torch.float64, device=cuda)
        assert (Qd.transpose(1, 2) @ Qd - eye).abs().max().item() <= 1e-5


def test_static_workspace_refuses_more_than_it_holds(cuda):
    P = torch.zeros(1, 4096, 4096, device=cuda)
    with pytest.raises(S.SoapError) as err:
        S.soap_qr_static(P, 1e-4)
    assert err.value.code == 1  # SOAP_ERR_INVALID_ARG


def test_static_workspace_reports_a_breakdown(cuda):
    """The call's device status reaches the caller: a non-finite input sets the QR-breakdown
    bit in the caller's word, and the next clean call clears it again."""
    rng = np.random.default_rng(5)
    P = torch.from_numpy(_psd(rng, 1, 256, 64)).to(cuda)
    bad = P.clone()
    bad[0, 3, 7] = float("nan")
    _, _, status = S.soap_qr_static(bad, 1e-4, return_status=True)
    torch.cuda.synchronize()
    assert status.item() & S.STATUS_QR_BREAKDOWN
    _, _, status = S.soap_qr_static(P, 1e-4, return_status=True)
    torch.cuda.synchronize()
    assert status.item() == 0
