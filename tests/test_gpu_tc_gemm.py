"""The tcgen05 fp32-accurate product (four TF32 products; C = alpha A B^T + beta C) against fp64,
through the C ABI."""
import numpy as np
import pytest
import torch

from paper_2607_20548_gb300 import soap as S

pytestmark = pytest.mark.gpu


def _ref(A, B, alpha, beta, C0):
    A64 = A.double().cpu().numpy()
    B64 = B.double().cpu().numpy()
    out = alpha * np.einsum("bmk,bnk->bmn", A64, B64 if B64.shape[0] == A64.shape[0] else np.broadcast_to(
        B64, (A64.shape[0],) + B64.shape[1:]))
    if C0 is not None:
        out = out + beta * C0.double().cpu().numpy()
    return out


def _rel(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("M,N,K,batch,bb", [(128, 128, 32, 1, 1), (128, 128, 1024, 2, 2), (200, 130, 100, 3, 3),
                                            (1, 5, 4, 1, 1), (384, 256, 2048, 2, 1), (1000, 520, 260, 1, 1),
                                            (256, 256, 8192, 1, 1)])
def test_tc_gemm_matches_fp64(cuda, M, N, K, batch, bb):
    g = torch.Generator(device=cuda).manual_seed(M + N + K)
    A = torch.randn(batch, M, K, device=cuda, generator=g)
    B = torch.randn(bb, N, K, device=cuda, generator=g)
    C0 = torch.randn(batch, M, N, device=cuda, generator=g)
    status = torch.zeros(1, dtype=torch.int32, device=cuda)
    C = C0.clone()
    S.soap_gemm_tf32x4(A, B, alpha=0.5, beta=-1.25, C=C, status=status)
    torch.cuda.synchronize()
    assert status.item() == 0
    e = _rel(C.double().cpu().numpy(), _ref(A, B, 0.5, -1.25, C0))
    # fp32 level at any K: each 32-wide K block is summed afresh and drained with fp32 adds
    print(f"\nM={M} N={N} K={K}: relative error {e:.2e}")
    assert e < 2e-6, e


def test_tc_gemm_transposed_output_and_lo(cuda):
    M, N, K = 256, 384, 512
    g = torch.Generator(device=cuda).manual_seed(1)
    A = torch.randn(2, M, K, device=cuda, generator=g)
    B = torch.randn(2, N, K, device=cuda, generator=g)
    Ct, lo = S.soap_gemm_tf32x4(A, B, transpose_c=True, with_lo=True)
    ref = _ref(A, B, 1.0, 0.0, None)
    assert Ct.shape == (2, N, M)
    assert _rel(np.transpose(Ct.double().cpu().numpy(), (0, 2, 1)), ref) < 2e-6
    hi, lo2 = S.soap_split_tf32(Ct)
    assert torch.equal(lo, lo2)
    # lo is x - trunc(x) rounded to tf32: hi + lo is x to within 2^-20 |x|
    assert ((hi + lo) - Ct).abs().le(2.0 ** -20 * Ct.abs()).all()


def test_tc_gemm_is_fp32_accurate_where_tf32_is_not(cuda):
    """A product that a single TF32 pass gets wrong at ~1e-3 and the split product gets right at fp32 level."""
    M = N = K = 512
    g = torch.Generator(device=cuda).manual_seed(2)
    A = torch.randn(1, M, K, device=cuda, generator=g)
    B = torch.randn(1, N, K, device=cuda, generator=g)
    ref = _ref(A, B, 1.0, 0.0, None)
    C = S.soap_gemm_tf32x4(A, B)
    e3 = _rel(C.double().cpu().numpy(), ref)
    ahi, alo = S.soap_split_tf32(A)
    bhi, blo = S.soap_split_tf32(B)
    C1 = S.soap_gemm_tf32x4(A, B, A_split=(ahi, torch.zeros_like(alo)), B_split=(bhi, torch.zeros_like(blo)))
    e1 = _rel(C1.double().cpu().numpy(), ref)
    # raw fp32 passed as "hi": shows whether the tensor core truncates tf32 operands
    tr = lambda x: (x.view(torch.int32) & ~0x1FFF).view(torch.float32)
    Craw = S.soap_gemm_tf32x4(A, B, A_split=(A, A - tr(A)), B_split=(B, B - tr(B)))
    eraw = _rel(Craw.double().cpu().numpy(), ref)
    print(f"\nsplit {e3:.2e}  1xTF32 {e1:.2e}  raw-fp32-as-hi {eraw:.2e}")
    assert e1 > 1e-4 and e3 < 2e-6


def test_tc_gemm_throughput_report(cuda):
    """Times an 8192^3 product (one of the dense block's largest) and prints TFLOP/s."""
    n = 8192
    g = torch.Generator(device=cuda).manual_seed(3)
    A = torch.randn(1, n, n, device=cuda, generator=g)
    B = torch.randn(1, n, n, device=cuda, generator=g)
    ah, al = S.soap_split_tf32(A)
    bh, bl = S.soap_split_tf32(B)
    C = torch.empty(1, n, n, device=cuda)
    for _ in range(2):
        S.soap_gemm_tf32x4(A, B, C=C, A_split=(ah, al), B_split=(bh, bl))
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    reps = 5
    for _ in range(reps):
        S.soap_gemm_tf32x4(A, B, C=C, A_split=(ah, al), B_split=(bh, bl))
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    tflops = 2 * n ** 3 / (ms / 1e3) / 1e12
    print(f"\n8192^3 split product: {ms:.2f} ms, {tflops:.1f} fp32-equivalent TFLOP/s ({4 * tflops:.0f} TF32 TFLOP/s)")
    assert tflops > 0
