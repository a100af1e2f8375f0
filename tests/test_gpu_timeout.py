"""Failure detection on the device, without a fault: every wait of the tensor-core products is
bounded. A device flag that nothing sets (soap_wait_limit's `hold`) makes the waits run out; the
kernels then drain what they have in flight, free their tensor memory and return, the status
word reports SOAP_STATUS_TIMEOUT, and the context stays usable for the next call."""
import numpy as np
import pytest
import torch

from paper_2607_20548_gb300 import soap as S

pytestmark = pytest.mark.gpu

LIMIT_NS = 1_000_000  # 1 ms: the bound the waits get in these tests


def _held(fn, cuda):
    hold = torch.zeros(1, dtype=torch.int32, device=cuda)
    try:
        S.soap_wait_limit(LIMIT_NS, hold)
        out = fn()
        torch.cuda.synchronize()
    finally:
        S.soap_wait_limit(0, None)
    return out


@pytest.mark.parametrize("M, N, K", [(256, 384, 512), (128, 32, 2048)])
def test_product_wait_runs_out_and_reports(cuda, M, N, K):
    g = torch.Generator(device=cuda).manual_seed(M + N + K)
    A = torch.randn(M, K, device=cuda, generator=g)
    B = torch.randn(N, K, device=cuda, generator=g)
    status = torch.zeros(1, dtype=torch.int32, device=cuda)
    _held(lambda: S.soap_gemm_tf32x4(A, B, status=status), cuda)
    assert status.item() & S.STATUS_TIMEOUT
    # the same product afterwards: no timeout, and the result of an fp32 product
    status.zero_()
    C = S.soap_gemm_tf32x4(A, B, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    ref = A.double() @ B.double().T
    assert ((C.double() - ref).abs().max() / ref.abs().max()).item() <= 1e-5


def test_step_wait_runs_out_sets_sticky_timeout(cuda):
    shapes = [(64, 96, True, True), (128, 64, True, False)]
    g = torch.Generator(device=cuda).manual_seed(4)
    W = [(0.02 * torch.randn(r, c, device=cuda, generator=g)).contiguous() for r, c, _, _ in shapes]
    G = [torch.randn(r, c, device=cuda, generator=g).contiguous() / np.sqrt(c) for r, c, _, _ in shapes]
    opt = S.SoapOptimizer(shapes)
    _held(lambda: opt.step(W, G), cuda)
    assert opt.status() == 6  # SOAP_ERR_TIMEOUT
    with pytest.raises(S.SoapError) as e:  # sticky: the next step reports it before enqueuing
        opt.step(W, G)
    assert e.value.code == 6
    opt.clear_status()
    assert opt.status() == 0
    opt.destroy()
    # a handle created after the timeout steps normally on the same context
    fresh = S.SoapOptimizer(shapes)
    W2 = [w.clone() for w in W]
    fresh.step(W2, G)
    torch.cuda.synchronize()
    assert fresh.status() == 0
    assert all(torch.isfinite(w).all().item() for w in W2)
    fresh.destroy()
