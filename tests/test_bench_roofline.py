"""bench.py's roofline arithmetic on the host: the bound a family is placed under, and
achieved / peak, from per-family CUDA-event totals and algorithmic FLOPs and bytes."""
import bench

PEAKS = {"hbm_gbs": 6787.2, "bf16_tflops": 1903.2, "bf16_tflops_sustained": 1716.0}


def test_contraction_above_the_ridge_is_tensor_bound():
    # 10 launches, 100 ms in all, 20 TFLOP and 50 GB: 400 FLOP per byte, far above the ridge
    st = {"ms": 100.0, "launches": 10, "flops": 20e12, "bytes": 50e9}
    r = bench.roofline("gemm_tc", st, PEAKS, "measured")
    peak = bench.TF32_TFLOPS["sustained"] / bench.TC_PRODUCTS
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert abs(r["achieved"] - 200.0) < 1e-9 and abs(r["peak"] - peak) < 1e-9
    assert abs(r["frac"] - 200.0 / peak) < 1e-12
    assert abs(r["avg_launch_us"] - 10_000.0) < 1e-9


def test_block_update_below_the_ridge_is_hbm_bound():
    # the K = 128 update: 2 x 128 FLOP per 8 bytes of C = 32 FLOP per byte, just below the ridge
    # of 237.9 TFLOP/s over 6787.2 GB/s (~35 FLOP per byte)
    st = {"ms": 50.0, "launches": 100, "flops": 32 * 100e9, "bytes": 100e9}
    r = bench.roofline("qr_update", st, PEAKS, "measured")
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert abs(r["achieved"] - 2000.0) < 1e-9
    assert abs(r["frac"] - 2000.0 / 6787.2) < 1e-12
    # the traffic estimate scales the algorithmic bytes per launch by the measured ratio
    ratio = bench.TRAFFIC_PER_ALGORITHMIC_BYTE["qr_update"]
    assert abs(r["traffic"] - ratio * 1e9) < 1e-3


def test_elementwise_family_is_hbm_bound():
    st = {"ms": 10.0, "launches": 4, "flops": 1e9, "bytes": 60e9}
    r = bench.roofline("elementwise", st, PEAKS, "measured")
    assert r["bound"] == "hbm" and abs(r["achieved"] - 6000.0) < 1e-9
