#!/usr/bin/env python
"""Throughput of the batched SOAP step (Alg. 1) over every weight matrix of a model.

Default workload: the 24-layer fine-grained MoE stack (hidden 2048; per layer Wq, Wk, Wv, Wo
2048x2048 and 64 experts with gate/up 2048x768 and down 768x2048; embedding and LM head
2048x32768 with the 32768 side not preconditioned) -- 4706 fp32 matrices, one soap_step over
all of them per step. --workload selects another of the synthetic workloads (the dense block,
the MoE layer, the 8192-wide layer, the single 256x512 weight). Gradients are seeded and
rank-structured (power law + noise). Metric: SOAP steps/s for the whole model, plus effective
TFLOP/s from the fixed FLOP model of Alg. 1 (S1 as a SYRK, S2 power step, S3 Householder QR with
explicit Q, S4 re-projection with four two-sided products, S5/S7 rotations).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl {soap,reference}] [--workload NAME]
                  [--kl] [--optimizer {soap,muon}] [--layerwise] [--matrices i,j,...] [--peaks]

N > 1 (torchrun, one rank per GPU) runs N independent replicas of the model: the step has no
exchange, so value = N * K / max-over-ranks time. --impl reference times the fp64 CPU oracle on
the host cores instead (rank 0 only). --kl runs Alg. 1's KL-Shampoo factor form instead of the
standard factor EMAs, --optimizer muon the paper's Muon step, and --layerwise (N > 1) one model
stepped by all ranks, each owning whole matrices (section 6) and all-gathering the updated
weights; these are separate lines, not the headline. --peaks measures the TF32 and bf16 tensor
peaks (torch.matmul 8192^3, best of 10 and 4 s back to back) and prints them instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "moe_stack_24x_h2048"
SHAPES_TEXT = {
    "single_256x512": "1x 256x512, both sides preconditioned",
    "dense_block_h2048_ffn8192": "4x 2048x2048, 2x 2048x8192, 1x 8192x2048, all sides preconditioned",
    "moe_layer_64x768_h2048": "128x 2048x768, 64x 768x2048, 1x 2048x64 router, all sides preconditioned",
    "dense_8192_ffn28672": "2x 8192x8192 (both sides), 2x 8192x28672 (left only), 1x 28672x8192 (right only)",
    "moe_stack_24x_h2048": "24 layers x (4x 2048x2048 + 128x 2048x768 + 64x 768x2048), both sides; "
                           "2x 2048x32768 (left only): 4706 matrices",
}
METRIC = "SOAP steps/sec per model + effective TFLOP/s (fraction of dense peak)"
# fp32 FMA peak of the CUDA cores: 152 SMs x 128 lanes x 2 flop x 2.07 GHz
FP32_SIMT_PEAK_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def model_flops(rows, cols, left, right, kl=False) -> float:
    """FLOPs of one literal Alg. 1 step for one matrix (2 per multiply-add). The KL-Shampoo
    factor form of a two-sided matrix adds lambda = diag(Q^T F Q) for both factors (Q^T F)
    and the rotations G Q_R, G^T Q_L that its weighted EMA terms are built from."""
    m, n = float(rows), float(cols)
    f = 0.0
    if kl and left and right:
        f += 2 * m ** 3 + 2 * n ** 3 + 2 * m * n * n + 2 * n * m * m
    if left:
        f += m * m * n + 2 * m ** 3 + (8.0 / 3.0) * m ** 3      # S1 (SYRK), S2, S3
    if right:
        f += n * n * m + 2 * n ** 3 + (8.0 / 3.0) * n ** 3
    rot = (m * m * n if left else 0.0) + (m * n * n if right else 0.0)
    f += (4 + 2 + 2) * rot                                      # S4, S5, S7
    return f


MUON_NS_STEPS = 16
MUON_METRIC = "Muon steps/sec per model (bf16 Newton-Schulz) + effective TFLOP/s"


def muon_flops(rows, cols, ns=MUON_NS_STEPS) -> float:
    """FLOPs of one Alg. Muon step for one matrix: per Newton-Schulz iteration A = X X^T,
    A^2 and (b A + c A^2) X on the min(rows, cols) side (2 per multiply-add)."""
    r, k = float(min(rows, cols)), float(max(rows, cols))
    return ns * (2 * r * r * k + 2 * r ** 3 + 2 * r * r * k)


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


class ClockSampler:
    """nvidia-smi clock/throttle samples every 200 ms while the timed region runs."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index),
                 "--query-gpu=index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (FileNotFoundError, OSError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        os.unlink(self.path)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "samples": len(sm),
                "power_w_max": max(power), "reasons": sorted(reasons)}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        try:
            return json.load(open(p)), "measured"
        except ValueError:
            pass
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


# tensor-core fp32 products take 4 tf32 MMAs (hi/lo split of both operands)
TC_PRODUCTS = 4
# TF32 dense matmul throughput of the GB300s, measured with `python bench.py --peaks`
# (torch.matmul 8192^3 with TF32 allowed: best of 10, and back to back for 4 s); the summary is
# profiles/peaks_gb300.md. The driver's MEASURED_PEAKS.json has the bf16 and HBM figures only.
TF32_TFLOPS = {"burst": 1047.2, "sustained": 951.8}

# DRAM bytes (ncu dram__bytes_read.sum + dram__bytes_write.sum) per algorithmic byte, from one
# full capture of each family's representative launch (profiles/): the QR's K = 128 trailing
# update of an 8192 factor (0.89) and the power step of an 8192 factor, whose operand panels are
# re-read across tiles (5.1). Applied to a family's average algorithmic bytes per launch, the
# mixed launches of a family make it an estimate; the other families have no current capture.
TRAFFIC_PER_ALGORITHMIC_BYTE = {"qr_update": 0.89, "gemm_tc": 5.12}


def roofline(family, st, peaks, peak_src, products=None, dtype_ratio=2.0):
    """Roofline of one kernel family from its CUDA-event time and algorithmic FLOPs/bytes."""
    secs = st["ms"] / 1e3
    ratio = TRAFFIC_PER_ALGORITHMIC_BYTE.get(family)
    per_launch = st["bytes"] / max(1, st["launches"])
    base = {"kernel": family, "launches": st["launches"], "avg_launch_us": 1e3 * st["ms"] / max(1, st["launches"]),
            "traffic": ratio * per_launch if ratio is not None else None,
            "traffic_note": "DRAM bytes per launch = measured DRAM/algorithmic ratio x algorithmic bytes per launch"
            if ratio is not None else None}
    if family == "gemm_simt":
        ach = st["flops"] / secs / 1e12
        return dict(base, bound="alu", achieved=ach, peak=FP32_SIMT_PEAK_TFLOPS, unit="TFLOP/s",
                    frac=ach / FP32_SIMT_PEAK_TFLOPS,
                    peak_source="fp32 FMA peak of the CUDA cores, 152 SMs x 128 lanes x 2 x 2.07 GHz")
    # the kernels run inside a long step: the sustained tensor peak. fp32 products take
    # TC_PRODUCTS tf32 MMAs at the measured TF32 rate; bf16 products (Muon) one MMA at the
    # measured bf16 rate
    products = TC_PRODUCTS if products is None else products
    if products > 1:
        tc_peak = TF32_TFLOPS["sustained"] / products
        tc_src = f"measured sustained tf32 dense ({TF32_TFLOPS['sustained']} TFLOP/s, bench.py --peaks) / {products}" \
                 " (tf32 products per fp32 product)"
    else:
        tc_peak = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
        tc_src = f"{peak_src} sustained bf16 dense"
    ridge = tc_peak * 1e12 / (peaks["hbm_gbs"] * 1e9)  # FLOP per byte where the two bounds meet
    # a tensor-core family whose FLOPs per algorithmic byte reach the ridge is bound by the tensor
    # pipe (the QR's block products sit at the ridge: 2 x 128 fp32 FLOP per 4-8 bytes of C)
    if family in ("gemm_tc", "qr_update") and st["flops"] / max(1.0, st["bytes"]) >= ridge:
        ach = st["flops"] / secs / 1e12
        return dict(base, bound="tensor", achieved=ach, peak=tc_peak, unit="TFLOP/s", frac=ach / tc_peak,
                    peak_source=tc_src)
    ach = st["bytes"] / secs / 1e9
    return dict(base, bound="hbm", achieved=ach, peak=peaks["hbm_gbs"], unit="GB/s", frac=ach / peaks["hbm_gbs"],
                peak_source=peak_src)


def shape_classes(specs):
    """{(rows, cols, left, right): count} in first-appearance order."""
    out = {}
    for sp in specs:
        key = (sp.rows, sp.cols, sp.left, sp.right)
        out[key] = out.get(key, 0) + 1
    return out


def _time_oracle_step(rows, cols, left, right, kl, name, spec_index):
    """Host seconds of one fp64 oracle step (t = 1) of one rows x cols matrix with the workload's
    gradient recipe."""
    from oracle.soap_ref import HParams, MatrixState, soap_step
    from paper_2607_20548_gb300.workloads import GradientStream, expert_scales, WORKLOADS, MatrixSpec

    specs, _ = WORKLOADS[name]
    scale = expert_scales(specs, name, 0)[spec_index] if spec_index is not None else 1.0
    stream = GradientStream([MatrixSpec(rows, cols, left, right)], 0, [scale], "cpu", name)
    W = stream.weights()[0][0].numpy().astype(np.float64)
    G = stream.grads(1)[0][0].numpy()
    st = MatrixState(rows, cols, left, right, np.float64)
    t0 = time.perf_counter()
    soap_step(st, W, G, HParams(kl=kl))
    return time.perf_counter() - t0


def oracle_sample(name: str, steps: int = 1, kl: bool = False):
    """Times the fp64 oracle's SOAP step on one matrix of each shape class of the workload, on the
    host cores, and extrapolates to the whole model by the class counts (the matrices are
    independent and a class's matrices cost the same). A class with an identity side longer than
    2048 is timed at 1024 and 2048 on that side and extrapolated linearly in its length (every
    stage of a one-sided step is linear in the identity side, except the factor's refresh, which
    does not depend on it); a class with a preconditioned side longer than 2048 is scaled from a
    2048 x 2048 step by the FLOP model (the oracle's unblocked QR of an 8192 factor alone takes
    minutes). Returns (seconds of host time, model steps/s, threads, description)."""
    from paper_2607_20548_gb300.workloads import WORKLOADS

    specs, _ = WORKLOADS[name]
    per_model = 0.0
    sampled = 0.0
    parts = []
    base2048 = None
    for (r, c, left, right), count in shape_classes(specs).items():
        j = next(i for i, sp in enumerate(specs) if (sp.rows, sp.cols, sp.left, sp.right) == (r, c, left, right))
        tag = f"{r}x{c}{'' if left and right else (' L' if left else (' R' if right else ''))}"
        pre = max(r if left else 0, c if right else 0)
        ident = max(c if not right else 0, r if not left else 0)
        if pre > 2048:
            if base2048 is None:
                base2048 = _time_oracle_step(2048, 2048, True, True, kl, name, None)
                sampled += base2048
            per = base2048 * model_flops(r, c, left, right, kl) / model_flops(2048, 2048, True, True, kl)
            parts.append(f"{tag}: {per:.2f} s (2048x2048 step scaled by the FLOP model) x {count}")
        elif ident > 2048:
            dims = []
            for d in (1024, 2048):
                rr, cc = (r, d) if not right else (d, c)
                dt = _time_oracle_step(rr, cc, left, right, kl, name, j)
                sampled += dt
                dims.append(dt)
            per = dims[0] + (dims[1] - dims[0]) * (ident - 1024) / 1024.0
            parts.append(f"{tag}: {per:.2f} s (identity side 1024 and 2048 timed, linear in its length) x {count}")
        else:
            per = _time_oracle_step(r, c, left, right, kl, name, j)
            sampled += per
            parts.append(f"{tag}: {per:.2f} s x {count}")
        per_model += per * count
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    desc = (f"fp64 oracle step (t = 1) of one matrix per shape class ({'; '.join(parts)}); whole model = "
            f"the sum weighted by the class counts")
    return sampled, 1.0 / per_model, threads, desc


def muon_oracle_sample(name: str):
    """One fp64 oracle Muon step of one matrix per shape class, scaled by the class counts."""
    from oracle.muon_ref import MuonParams, MuonState, muon_step
    from paper_2607_20548_gb300.workloads import WORKLOADS, make_stream

    specs, _ = WORKLOADS[name]
    hp = MuonParams(coeffs=[(15 / 8, -10 / 8, 3 / 8)] * MUON_NS_STEPS)
    per_model, sampled, parts = 0.0, 0.0, []
    for (r, c, _l, _r), count in shape_classes(specs).items():
        j = next(i for i, sp in enumerate(specs) if (sp.rows, sp.cols) == (r, c))
        stream = make_stream(name, seed=0, device="cpu", specs=[j])
        W = stream.weights()[0][0].numpy().astype(np.float64)
        G = stream.grads(1)[0][0].numpy()
        t0 = time.perf_counter()
        muon_step(MuonState(r, c), W, G, hp)
        per = time.perf_counter() - t0
        sampled += per
        per_model += per * count
        parts.append(f"{r}x{c}: {per:.2f} s x {count}")
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return sampled, 1.0 / per_model, threads, (f"fp64 oracle Muon step of one matrix per shape class "
                                               f"({'; '.join(parts)}), scaled by the class counts")


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    name = args.workload
    specs, _ = __import__("paper_2607_20548_gb300.workloads", fromlist=["WORKLOADS"]).WORKLOADS[name]
    sps_all, secs = [], 0.0
    desc, threads = "", 1
    for _ in range(args.warmup + args.steps):
        sampled, sps, threads, desc = oracle_sample(name, 1, args.kl)
        sps_all.append(sps)
        secs += sampled
    sps = float(np.mean(sps_all[args.warmup:])) if args.steps > 0 else float(np.mean(sps_all))
    line = {"impl": "reference", "metric": METRIC, "value": sps, "unit": "steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 / sps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": name, "matrices": len(specs), "shapes": SHAPES_TEXT.get(name),
                       "parallelism": "replicas" if world > 1 else "single"},
            "cpu_baseline": {"value": sps, "unit": "steps/s", "cores": threads, "kind": "oracle",
                             "sample": desc + f"; each bench step times that sample once ({secs:.1f} s of host "
                                              f"time over {args.warmup + args.steps} steps)"},
            "e2e": {"value": sps, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def library_sample(specs, dev, per_class=4, steps=2):
    """Context only: the same standard-form SOAP step written with library calls (torch fp32
    matmul with TF32 off, cuSOLVER QR through torch.linalg.qr), per matrix, on the same GPU, on
    up to `per_class` matrices of each shape class, extrapolated to the model by the class counts.
    Returns (steps/s, note) or (None, reason)."""
    try:
        prev = torch.backends.cuda.matmul.allow_tf32
        torch.backends.cuda.matmul.allow_tf32 = False
        b, b1, b2, eps, lr, wd = 0.95, 0.95, 0.95, 1e-8, 3e-3, 0.1

        def qr_pos(P):
            Q, Rr = torch.linalg.qr(P)
            d = torch.sign(torch.diagonal(Rr))
            return Q * torch.where(d == 0, torch.ones_like(d), d)

        def one(x, G):
            if x["left"]:
                x["L"].mul_(b).addmm_(G, G.T, alpha=1 - b)
                x["QL"] = qr_pos(x["L"] @ x["QL"])
            if x["right"]:
                x["R"].mul_(b).addmm_(G.T, G, alpha=1 - b)
                x["QR"] = qr_pos(x["R"] @ x["QR"])
            x["Mh"].mul_(b1).add_(G, alpha=1 - b1)
            Gp, mp = G, x["Mh"]
            if x["left"]:
                Gp, mp = x["QL"].T @ Gp, x["QL"].T @ mp
            if x["right"]:
                Gp, mp = Gp @ x["QR"], mp @ x["QR"]
            x["V"].mul_(b2).addcmul_(Gp, Gp, value=1 - b2)
            N = mp / (x["V"].sqrt() + eps)
            if x["left"]:
                N = x["QL"] @ N
            if x["right"]:
                N = N @ x["QR"].T
            x["W"].mul_(1 - lr * wd).sub_(N, alpha=lr)

        total = 0.0
        for (m, n, left, right), count in shape_classes(specs).items():
            k = min(count, per_class)
            st = [dict(left=left, right=right, L=torch.zeros(m, m, device=dev) if left else None,
                       R=torch.zeros(n, n, device=dev) if right else None,
                       QL=torch.eye(m, device=dev) if left else None, QR=torch.eye(n, device=dev) if right else None,
                       Mh=torch.zeros(m, n, device=dev), V=torch.zeros(m, n, device=dev),
                       W=torch.zeros(m, n, device=dev)) for _ in range(k)]
            G = torch.randn(m, n, device=dev) / np.sqrt(n)
            for x in st:
                one(x, G)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(steps):
                for x in st:
                    one(x, G)
            e1.record()
            torch.cuda.synchronize()
            total += e0.elapsed_time(e1) / 1e3 / (steps * k) * count
            del st
        torch.backends.cuda.matmul.allow_tf32 = prev
        torch.cuda.empty_cache()
        return 1.0 / total, (f"the standard-form step per matrix with torch fp32 matmul (TF32 off) and "
                             f"torch.linalg.qr (cuSOLVER), sign-fixed, on up to {per_class} matrices per shape "
                             f"class ({steps} steps after one warm-up), extrapolated by the class counts")
    except Exception as e:  # context only: never fails the bench
        return None, f"unavailable: {type(e).__name__}: {str(e)[:200]}"


def measure_peaks():
    """TF32 and bf16 dense matmul throughput on this GPU: torch.matmul 8192^3 (2 N^3 FLOP), best of
    10 (burst) and back to back for 4 s (sustained), with the TF32 path allowed."""
    dev = torch.device("cuda", 0)
    n = 8192
    out = {}
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = True
    for name, dt in (("tf32", torch.float32), ("bf16", torch.bfloat16), ("fp32_simt", torch.float32)):
        if name == "fp32_simt":
            torch.backends.cuda.matmul.allow_tf32 = False
        a = torch.randn(n, n, device=dev, dtype=dt)
        b = torch.randn(n, n, device=dev, dtype=dt)
        c = a @ b
        torch.cuda.synchronize()
        best = float("inf")
        for _ in range(10):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            torch.matmul(a, b, out=c)
            e1.record()
            torch.cuda.synchronize()
            best = min(best, e0.elapsed_time(e1) / 1e3)
        iters, t0 = 0, time.perf_counter()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        while time.perf_counter() - t0 < 4.0:
            for _ in range(8):
                torch.matmul(a, b, out=c)
            iters += 8
            torch.cuda.synchronize()
        e1.record()
        torch.cuda.synchronize()
        sus = e0.elapsed_time(e1) / 1e3 / iters
        out[name] = {"burst_tflops": 2 * n ** 3 / best / 1e12, "sustained_tflops": 2 * n ** 3 / sus / 1e12}
        del a, b, c
    torch.backends.cuda.matmul.allow_tf32 = prev
    return out


def make_inputs(gen, world_mem_bytes):
    """Weights and a pool of gradient sets on the device: W per shape group, and as many distinct
    steps' gradients (up to 4) as fit in a tenth of the device memory, at least one."""
    W = [w.contiguous() for w in gen.weights()]
    gbytes = sum(w.numel() * 4 for w in W)
    npool = int(max(1, min(4, (0.1 * world_mem_bytes) // max(1, gbytes))))
    pool = []
    for t in range(npool):
        pool.append(gen.grads(t + 1))
    return W, pool


def flat_views(gen, tensors, rotate=0):
    """Per-matrix views of per-group [batch, rows, cols] tensors, in matrix order; with `rotate`,
    matrix at position p of its group gets the group's tensor (p + rotate) mod batch."""
    out = [None] * len(gen.specs)
    for (spec, idx), t in zip(gen.groups, tensors):
        B = len(idx)
        for p, j in enumerate(idx):
            out[j] = t[(p + rotate) % B]
    return out


def run_soap(args):
    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
    from paper_2607_20548_gb300 import SoapOptimizer, build, default_hparams
    from paper_2607_20548_gb300 import soap as S
    from paper_2607_20548_gb300.workloads import WORKLOADS, make_stream

    if not os.path.exists(S.LIB_PATH):
        build.build()
    name = args.workload
    specs, _ = WORKLOADS[name]
    subset = [int(x) for x in args.matrices.split(",") if x.strip()] if args.matrices else None
    if subset:
        specs = [specs[j] for j in subset]
    muon = args.optimizer == "muon"
    layerwise = args.layerwise and world > 1
    gen = make_stream(name, seed=0 if layerwise else rank, device=dev, specs=subset)
    total_mem = torch.cuda.get_device_properties(dev).total_memory
    Wg, pool = make_inputs(gen, total_mem)
    npool = len(pool)
    del gen._A, gen._bases
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    if layerwise:
        # one model stepped by all ranks: each owns whole matrices (section 6) and the updated
        # weights are all-gathered over NCCL after every step
        from paper_2607_20548_gb300.layerwise import LayerwiseOptimizer
        nccl = dist.new_group(backend="nccl")
        hp = default_hparams(kl=int(args.kl))
        opt = LayerwiseOptimizer([(s.rows, s.cols, int(s.left), int(s.right)) for s in specs],
                                 lambda sh: SoapOptimizer(sh, hp, device=local), group=nccl, policy=1)
    elif muon:
        opt = S.MuonOptimizer([(s.rows, s.cols) for s in specs], ns_steps=MUON_NS_STEPS, device=local)
    else:
        opt = SoapOptimizer([(s.rows, s.cols, s.left, s.right) for s in specs], default_hparams(kl=int(args.kl)),
                            device=local)
    plan = opt.plan_info() if hasattr(opt, "plan_info") else None

    W = flat_views(gen, Wg)

    def grads_for(t):
        # step t's gradients: pool entry t mod npool; when the pool holds fewer distinct steps than
        # are run, each group's gradients are also handed round its matrices (shifted by one
        # matrix per pass), so that no matrix sees the same gradient twice in a row
        return flat_views(gen, pool[t % npool], rotate=t // npool)

    stream = torch.cuda.current_stream()
    for t in range(args.warmup):
        opt.step(W, grads_for(t))
    torch.cuda.synchronize()
    if opt.status() != 0:
        raise RuntimeError("device status after warm-up: " + opt.last_error())

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    # launches per step, to size the profiler
    opt.profile_begin(1 << 18)
    opt.step(W, grads_for(args.warmup))
    per_step = sum(v["launches"] for k, v in opt.profile_end().items() if k != "overflow")
    step0 = args.warmup + 1
    # timed region: K steps, inputs resident in HBM (optimizer state and gradients >> 129 MB L2)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    opt.profile_begin(max(1024, per_step * args.steps + 1024))
    grads_seq = [grads_for(step0 + t) for t in range(args.steps)]
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        # cudaProfilerStart/Stop bracket the timed steps, so that a profiler started with
        # profiling off (ncu --profile-from-start off) records exactly these launches
        torch.cuda.profiler.start()
        start.record(stream)
        for t in range(args.steps):
            opt.step(W, grads_seq[t])
        stop.record(stream)
        torch.cuda.synchronize()
        torch.cuda.profiler.stop()
    prof = opt.profile_end()
    barrier()
    elapsed = start.elapsed_time(stop) / 1e3
    if world > 1:
        import torch.distributed as dist
        tt = torch.tensor([elapsed], dtype=torch.float64)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        elapsed = float(tt.item())
    # replicas: N models per step; layer-wise: one model per step, stepped by all ranks
    units = 1 if layerwise else world
    value = units * args.steps / elapsed

    # end to end through the public API: each step's gradients copied in from pinned host
    # memory (into the same device buffers), the step, and the updated weights copied back
    def pinned_copy(x):
        hx = torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
        hx.copy_(x)
        return hx

    host_pool = [[pinned_copy(g) for g in grp] for grp in pool]
    host_w = [pinned_copy(w) for w in Wg]
    h2d = sum(g.numel() * 4 for g in pool[0])
    d2h = sum(w.numel() * 4 for w in Wg)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    # the copies run on two side streams, so that a step's weights going out overlap the next
    # step's gradients coming in (the two directions of the link); each step waits for its
    # gradients and for the previous step's weights to be out before it rewrites them
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev_in, ev_out, ev_done = torch.cuda.Event(), torch.cuda.Event(), torch.cuda.Event()
    e0.record(stream)
    base = step0 + args.steps
    for t in range(args.steps):
        k = (base + t) % npool
        s_in.wait_stream(stream)  # the previous step has read the gradient buffers
        with torch.cuda.stream(s_in):
            for d, hsrc in zip(pool[k], host_pool[k]):
                d.copy_(hsrc, non_blocking=True)
            ev_in.record(s_in)
        stream.wait_event(ev_in)
        if t > 0:
            stream.wait_event(ev_out)
        opt.step(W, grads_for(base + t))
        ev_done.record(stream)
        s_out.wait_event(ev_done)
        with torch.cuda.stream(s_out):
            for hdst, w in zip(host_w, Wg):
                hdst.copy_(w, non_blocking=True)
            ev_out.record(s_out)
    stream.wait_event(ev_out)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_s = e0.elapsed_time(e1) / 1e3
    if world > 1:
        import torch.distributed as dist
        tt = torch.tensor([e2e_s], dtype=torch.float64)
        dist.all_reduce(tt, op=dist.ReduceOp.MAX)
        e2e_s = float(tt.item())
    if opt.status() != 0:
        raise RuntimeError("device status after timed steps: " + opt.last_error())
    del host_pool, host_w
    # one more step (outside the timed regions) with every launch timed alone: each starts on an
    # idle device, so the per-family rates are the kernels' own, without the contention of the
    # library's concurrent QR streams that the live figures include
    iso = None
    if not (muon or layerwise):
        opt.profile_begin(max(1024, per_step + 1024), serial=True)
        opt.step(W, grads_for(base + args.steps))
        iso = {k: v for k, v in opt.profile_end().items() if k != "overflow"}
        if opt.status() != 0:
            raise RuntimeError("device status after the isolated step: " + opt.last_error())

    if rank != 0:
        opt.destroy()
        return
    if muon:
        model_f = sum(muon_flops(s.rows, s.cols) for s in specs)
    else:
        model_f = sum(model_flops(s.rows, s.cols, s.left, s.right, args.kl) for s in specs)
    peaks, peak_src = measured_peaks()
    fams = {k: v for k, v in prof.items() if k != "overflow"}
    top = max(fams, key=lambda k: fams[k]["ms"])
    st = fams[top]
    launches = sum(v["launches"] for v in fams.values())
    roof = roofline(top, st, peaks, peak_src, products=1 if muon else TC_PRODUCTS, dtype_ratio=1.0 if muon else 2.0)
    if muon:
        # the DRAM/algorithmic ratios above were measured for the fp32 (tf32 x4) kernels
        roof["traffic"], roof["traffic_note"] = None, "not measured for the bf16 kernel"
    if iso and iso.get(top, {}).get("launches"):
        r = roofline(top, iso[top], peaks, peak_src)
        roof["isolated"] = {k: r[k] for k in ("bound", "achieved", "peak", "unit", "frac", "avg_launch_us")}
        roof["isolated"]["note"] = ("one further step with each launch timed alone (the device idle when it starts): "
                                    "the kernel's own rate; the figures above are live, beside the concurrent "
                                    "QR streams")
    opt.destroy()
    del Wg, pool, W, grads_seq
    torch.cuda.empty_cache()
    if subset:
        sps, threads, cpu_desc = None, 0, "not sampled for a subset of the workload"
    elif muon:
        _, sps, threads, cpu_desc = muon_oracle_sample(name)
    else:
        _, sps, threads, cpu_desc = oracle_sample(name, 1, args.kl)
    lib_line = None
    if not (muon or args.kl or layerwise or subset):
        lib_v, lib_note = library_sample(specs, dev)
        lib_line = {"value": lib_v, "unit": "steps/s", "kind": "torch + cuSOLVER", "sample": lib_note}
    tc_peak = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"]) if muon else TF32_TFLOPS["sustained"] / TC_PRODUCTS
    line = {
        "metric": MUON_METRIC if muon else METRIC, "value": value, "unit": "steps/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * elapsed / args.steps,
        "higher_is_better": True, "scaling": "strong" if layerwise else "weak", "vs_baseline": None,
        "dtype": "bf16" if muon else "f32",
        "data": "synthetic",
        "config": {"workload": name if not subset else f"{name}[matrices {args.matrices}]",
                   "matrices": len(specs),
                   "shapes": SHAPES_TEXT.get(name),
                   "parallelism": f"layerwise{world}" if layerwise else ("replicas" if world > 1 else "single"),
                   "optimizer": "muon (16 quintic Newton-Schulz steps)" if muon else
                   ("soap, KL factor form" if args.kl else "soap, standard factor form"),
                   "waves_per_step": plan["waves"] if plan else None,
                   "waves_pipelined": plan["pipelined"] if plan else None,
                   "workspace_gb": plan["workspace_bytes"] / 1e9 if plan else None,
                   "state_gb": plan["state_bytes"] / 1e9 if plan else None,
                   "gradients": (f"{npool} distinct step(s) of gradients resident"
                                 + ("; each shape group's gradients handed round its matrices, shifted by one "
                                    "matrix per pass" if npool < args.warmup + 2 * args.steps + 1 else "")),
                   "l2": "inputs larger than L2 (optimizer state and gradients of every matrix per step)"},
        "effective_tflops": model_f * value / world / 1e12,
        "effective_frac_of_tensor_peak": model_f * value / world / 1e12 / tc_peak,
        "effective_note": "per GPU (the whole-job FLOP rate divided by the number of GPUs)",
        "model_flop_per_step": model_f,
        "roofline": roof,
        "kernel_time_share": {k: round(v["ms"] / max(1e-9, sum(x["ms"] for x in fams.values())), 4)
                              for k, v in fams.items()},
        "kernel_families": {k: {"ms_per_step": v["ms"] / args.steps, "launches_per_step": v["launches"] / args.steps,
                                "tflops": v["flops"] / max(1e-12, v["ms"] / 1e3) / 1e12,
                                "gbs": v["bytes"] / max(1e-12, v["ms"] / 1e3) / 1e9}
                            for k, v in fams.items() if v["launches"]},
        "kernel_families_isolated": {k: {"ms_per_step": v["ms"], "launches_per_step": v["launches"],
                                         "tflops": v["flops"] / max(1e-12, v["ms"] / 1e3) / 1e12,
                                         "gbs": v["bytes"] / max(1e-12, v["ms"] / 1e3) / 1e9}
                                     for k, v in iso.items() if v["launches"]} if iso else None,
        "cpu_baseline": {"value": sps, "unit": "steps/s", "cores": threads, "kind": "oracle", "sample": cpu_desc},
        "e2e": {"value": units * args.steps / e2e_s, "unit": "steps/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "clocks": clk.summary(),
        "library_baseline": lib_line,
    }
    print(json.dumps(line), flush=True)


def main():
    from paper_2607_20548_gb300.workloads import WORKLOADS
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["soap", "reference"], default="soap")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default=DEFAULT_WORKLOAD)
    ap.add_argument("--matrices", default="",
                    help="comma-separated matrix indices of the workload to run (a smaller case for profiling); "
                         "default: all")
    ap.add_argument("--optimizer", choices=["soap", "muon"], default="soap",
                    help="muon: the paper's Muon step on the same model (a separate line, not the headline)")
    ap.add_argument("--layerwise", action="store_true",
                    help="with N > 1: one model, each rank stepping its own matrices (section 6) and "
                         "all-gathering the updated weights over NCCL (strong scaling)")
    ap.add_argument("--kl", action="store_true",
                    help="KL-Shampoo factor form (Alg. 1's factor accumulation) instead of the standard EMAs")
    ap.add_argument("--peaks", action="store_true",
                    help="measure the TF32 / bf16 / fp32 matmul peaks of this GPU and print them")
    args = ap.parse_args()
    if args.peaks:
        print(json.dumps({"peaks": measure_peaks(), "gpu": torch.cuda.get_device_name(0),
                          "how": "torch.matmul 8192^3, 2 N^3 FLOP: best of 10 (burst) and back to back for 4 s "
                                 "(sustained); tf32 with TF32 allowed, fp32_simt with it off"}), flush=True)
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_soap(args)


if __name__ == "__main__":
    main()
