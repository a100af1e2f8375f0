"""bench.py's FLOP model (the literal Alg. 1 count its effective TFLOP/s divides by) against the
per-workload totals worked out by hand for the synthetic workloads, and its identity-side rule."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2607_20548_gb300.workloads import WORKLOADS  # noqa: E402

# model FLOP per step of each workload, counted by hand from the matrix list (2 per multiply-add;
# S1 as a SYRK m^2 n + m n^2, S2 2(m^3 + n^3), S3 (8/3)(m^3 + n^3), S4 4(m^2 n + m n^2),
# S5 = S7 = 2(m^2 n + m n^2), identity sides dropped), to the digits they were quoted with
HAND_TOTALS = {
    "single_256x512": (1.61e9, 0.005),
    "dense_block_h2048_ffn8192": (13.39e12, 0.001),
    "moe_layer_64x768_h2048": (15.80e12, 0.001),
    "dense_8192_ffn28672": (89.70e12, 0.001),
    "moe_stack_24x_h2048": (403.2e12, 0.001),
}


@pytest.mark.parametrize("name", sorted(HAND_TOTALS))
def test_workload_totals(name):
    specs, _ = WORKLOADS[name]
    total = sum(bench.model_flops(s.rows, s.cols, s.left, s.right) for s in specs)
    want, rel = HAND_TOTALS[name]
    assert abs(total - want) <= rel * want, (total, want)


def test_square_two_sided_is_82_over_3_cubes():
    # 2 (S1) + 4 (S2) + 16/3 (S3) + 8 (S4) + 4 + 4 (S5, S7) = 82/3 n^3
    n = 2048
    assert bench.model_flops(n, n, True, True) == pytest.approx(82.0 / 3.0 * n ** 3, rel=1e-12)


def test_identity_side_drops_its_factor_basis_and_rotation():
    m, n = 4096, 1024
    both = bench.model_flops(m, n, True, True)
    left = bench.model_flops(m, n, True, False)
    right = bench.model_flops(m, n, False, True)
    assert bench.model_flops(m, n, False, False) == 0.0
    # every term belongs to exactly one side
    assert left + right == pytest.approx(both, rel=1e-12)
    # the left side: S1 m^2 n, S2 2 m^3, S3 (8/3) m^3, S4 + S5 + S7 8 m^2 n
    assert left == pytest.approx(9 * m * m * n + (14.0 / 3.0) * m ** 3, rel=1e-12)


def test_kl_form_adds_lambda_products_and_rotations_for_two_sided_only():
    m, n = 2048, 8192
    extra = bench.model_flops(m, n, True, True, kl=True) - bench.model_flops(m, n, True, True)
    assert extra == pytest.approx(2 * m ** 3 + 2 * n ** 3 + 2 * m * n * n + 2 * n * m * m, rel=1e-12)
    assert bench.model_flops(m, n, True, False, kl=True) == bench.model_flops(m, n, True, False)


def test_muon_counts_three_products_per_newton_schulz_step():
    # A = X X^T (2 r^2 k), A A (2 r^3), (bA + cA^2) X (2 r^2 k), on the short side r
    assert bench.muon_flops(2048, 8192, ns=1) == pytest.approx(4 * 2048 ** 2 * 8192 + 2 * 2048 ** 3)
    assert bench.muon_flops(8192, 2048) == bench.muon_flops(2048, 8192)
    assert bench.muon_flops(2048, 2048) == pytest.approx(16 * 6 * 2048 ** 3)
