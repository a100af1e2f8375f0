#!/usr/bin/env python
"""Throughput of the batched SOAP step (Alg. 1) on one dense transformer block.

Workload: hidden 2048, 16 heads, SwiGLU FFN 8192 -- Wq, Wk, Wv, Wo 2048x2048, W_gate and
W_up 2048x8192, W_down 8192x2048, fp32 master weights, every side preconditioned, seeded
synthetic gradients (rank-structured power law + noise). One "step" = one soap_step over
all 7 matrices. Metric: SOAP steps/s for the whole block, plus effective TFLOP/s from the
fixed FLOP model of Alg. 1 (S1 as a SYRK, S2 power step, S3 Householder QR with explicit
Q, S4 re-projection with four two-sided products, S5/S7 rotations).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl {soap,reference}] [--kl]
                  [--optimizer {soap,muon}] [--layerwise] [--matrices i,j,...]

N > 1 (torchrun, one rank per GPU) runs N independent replicas of the block: the step
has no exchange, so value = N * K / max-over-ranks time. --impl reference times the
fp64 CPU oracle on the host cores instead (rank 0 only). --kl runs Alg. 1's KL-Shampoo
factor form instead of the standard factor EMAs, --optimizer muon the paper's Muon step,
and --layerwise (N > 1) one block stepped by all ranks, each owning whole matrices
(section 6) and all-gathering the updated weights; these are separate lines, not the
headline.
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

WORKLOAD = "dense_block_h2048_ffn8192"
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


# tensor-core fp32 products take 4 tf32 MMAs (hi/lo split of both operands); TF32 runs at
# half the bf16 rate on this part
TC_PRODUCTS = 4

# DRAM bytes (ncu dram__bytes_read.sum + dram__bytes_write.sum) per algorithmic byte of each
# kernel family, measured with ncu over one step of the block's 2048x8192 matrix alone
# (both of its QR sizes) for the current kernels. The QR products read their small operands
# from L2 across tiles and write split-K partial sums (ratio about 1); the large contractions
# re-read operand panels (ratio > 1); the panel kernel keeps its panel on chip.
TRAFFIC_PER_ALGORITHMIC_BYTE = {"qr_update": 1.059, "qr_panel": 0.383, "gemm_tc": 1.617}


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
    # the kernels run inside a long step: the sustained tensor peak; fp32 products take
    # TC_PRODUCTS tf32 MMAs at half the bf16 rate, bf16 products (Muon) one MMA at the bf16 rate
    products = TC_PRODUCTS if products is None else products
    tc_peak = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"]) / dtype_ratio / products
    ridge = tc_peak * 1e12 / (peaks["hbm_gbs"] * 1e9)  # FLOP per byte where the two bounds meet
    # a tensor-core family whose FLOPs per algorithmic byte reach the ridge is bound by the tensor
    # pipe (the QR's block products sit at the ridge: 2 x 128 fp32 FLOP per 4-8 bytes of C)
    if family in ("gemm_tc", "qr_update") and st["flops"] / max(1.0, st["bytes"]) >= ridge:
        ach = st["flops"] / secs / 1e12
        return dict(base, bound="tensor", achieved=ach, peak=tc_peak, unit="TFLOP/s", frac=ach / tc_peak,
                    peak_source=f"{peak_src} sustained bf16 dense" + (
                        f" / 2 (tf32) / {products} (tf32 products per fp32 product)" if products > 1 else ""))
    ach = st["bytes"] / secs / 1e9
    return dict(base, bound="hbm", achieved=ach, peak=peaks["hbm_gbs"], unit="GB/s", frac=ach / peaks["hbm_gbs"],
                peak_source=peak_src)


def oracle_sample(steps: int, warmup: int, kl: bool = False):
    """Times the fp64 oracle's SOAP step on Wq (2048x2048) of the block, on the host cores.
    Returns (seconds per sampled step, block steps/s extrapolated by the FLOP model, threads)."""
    from oracle.soap_ref import HParams, MatrixState, soap_step
    from paper_2607_20548_gb300.workloads import WORKLOADS, make_stream

    specs, _ = WORKLOADS[WORKLOAD]
    stream = make_stream(WORKLOAD, seed=0, device="cpu", specs=[0])
    W = stream.weights()[0][0].numpy().astype(np.float64)
    st = MatrixState(2048, 2048, True, True, np.float64)
    hp = HParams(kl=kl)
    times = []
    for t in range(1, steps + warmup + 1):
        G = stream.grads(t)[0][0].numpy()
        t0 = time.perf_counter()
        W, _ = soap_step(st, W, G, hp)
        if t > warmup:
            times.append(time.perf_counter() - t0)
    per = float(np.mean(times))
    block = sum(model_flops(s.rows, s.cols, s.left, s.right, kl) for s in specs)
    scale = block / model_flops(2048, 2048, True, True, kl)
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return per, 1.0 / (per * scale), threads, scale


def muon_oracle_sample():
    """One fp64 oracle Muon step of Wq (2048x2048) on the host cores, scaled to the block."""
    from oracle.muon_ref import MuonParams, MuonState, muon_step
    from paper_2607_20548_gb300.workloads import WORKLOADS, make_stream

    specs, _ = WORKLOADS[WORKLOAD]
    stream = make_stream(WORKLOAD, seed=0, device="cpu", specs=[0])
    W = stream.weights()[0][0].numpy().astype(np.float64)
    G = stream.grads(1)[0][0].numpy()
    hp = MuonParams(coeffs=[(15 / 8, -10 / 8, 3 / 8)] * MUON_NS_STEPS)
    t0 = time.perf_counter()
    muon_step(MuonState(2048, 2048), W, G, hp)
    per = time.perf_counter() - t0
    scale = sum(muon_flops(s.rows, s.cols) for s in specs) / muon_flops(2048, 2048)
    threads = int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
    return per, 1.0 / (per * scale), threads, scale


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    per, sps, threads, scale = oracle_sample(args.steps, args.warmup)
    sample = (f"oracle fp64 step of Wq (2048x2048) timed over {args.steps} steps after {args.warmup} warm-up; "
              f"whole-block time = {scale:.1f}x by the FLOP model")
    line = {"impl": "reference", "metric": METRIC, "value": sps, "unit": "steps/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 / sps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "matrices": 7, "parallelism": "replicas"},
            "cpu_baseline": {"value": sps, "unit": "steps/s", "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": sps, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def library_sample(specs, pool, dev, steps=2):
    """Context only: the same standard-form SOAP step written with library calls (torch fp32
    matmul with TF32 off, cuSOLVER QR through torch.linalg.qr), per matrix, on the same GPU.
    Returns (steps/s, note) or (None, reason)."""
    try:
        prev = torch.backends.cuda.matmul.allow_tf32
        torch.backends.cuda.matmul.allow_tf32 = False
        b, b1, b2, eps, lr, wd = 0.95, 0.95, 0.95, 1e-8, 3e-3, 0.1
        st = []
        for s_ in specs:
            m, n = s_.rows, s_.cols
            st.append(dict(L=torch.zeros(m, m, device=dev), R=torch.zeros(n, n, device=dev),
                           QL=torch.eye(m, device=dev), QR=torch.eye(n, device=dev),
                           Mh=torch.zeros(m, n, device=dev), V=torch.zeros(m, n, device=dev),
                           W=torch.zeros(m, n, device=dev)))

        def qr_pos(P):
            Q, Rr = torch.linalg.qr(P)
            d = torch.sign(torch.diagonal(Rr))
            return Q * torch.where(d == 0, torch.ones_like(d), d)

        def one(G_all):
            for x, G in zip(st, G_all):
                x["L"].mul_(b).addmm_(G, G.T, alpha=1 - b)
                x["R"].mul_(b).addmm_(G.T, G, alpha=1 - b)
                x["Mh"].mul_(b1).add_(G, alpha=1 - b1)
                x["QL"] = qr_pos(x["L"] @ x["QL"])
                x["QR"] = qr_pos(x["R"] @ x["QR"])
                Gp = x["QL"].T @ G @ x["QR"]
                mp = x["QL"].T @ x["Mh"] @ x["QR"]
                x["V"].mul_(b2).addcmul_(Gp, Gp, value=1 - b2)
                N = mp / (x["V"].sqrt() + eps)
                x["W"].mul_(1 - lr * wd).sub_(x["QL"] @ N @ x["QR"].T, alpha=lr)

        one(pool[0])
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for t in range(steps):
            one(pool[(t + 1) % len(pool)])
        e1.record()
        torch.cuda.synchronize()
        torch.backends.cuda.matmul.allow_tf32 = prev
        del st
        torch.cuda.empty_cache()
        return steps / (e0.elapsed_time(e1) / 1e3), (
            f"the standard-form step per matrix with torch fp32 matmul (TF32 off) and torch.linalg.qr "
            f"(cuSOLVER), sign-fixed; {steps} steps after one warm-up, same GPU and gradients")
    except Exception as e:  # context only: never fails the bench
        return None, f"unavailable: {type(e).__name__}: {str(e)[:200]}"


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
    specs, _ = WORKLOADS[WORKLOAD]
    subset = [int(x) for x in args.matrices.split(",") if x.strip()] if args.matrices else None
    if subset:
        specs = [specs[j] for j in subset]
    gen = make_stream(WORKLOAD, seed=rank, device=dev, specs=subset)
    muon = args.optimizer == "muon"
    layerwise = args.layerwise and world > 1
    if layerwise:
        # one model stepped by all ranks: each owns whole matrices (section 6) and the updated
        # weights are all-gathered over NCCL after every step
        from paper_2607_20548_gb300.layerwise import LayerwiseOptimizer
        nccl = dist.new_group(backend="nccl")
        gen = make_stream(WORKLOAD, seed=0, device=dev, specs=subset)
        hp = default_hparams(kl=int(args.kl))
        opt = LayerwiseOptimizer([(s.rows, s.cols, int(s.left), int(s.right)) for s in specs],
                                 lambda sh: SoapOptimizer(sh, hp, device=local), group=nccl, policy=1)
    elif muon:
        opt = S.MuonOptimizer([(s.rows, s.cols) for s in specs], ns_steps=MUON_NS_STEPS, device=local)
    else:
        opt = SoapOptimizer([(s.rows, s.cols, s.left, s.right) for s in specs], default_hparams(kl=int(args.kl)),
                            device=local)

    def flat(tensors):
        out = [None] * len(specs)
        for (spec, idx), t in zip(gen.groups, tensors):
            for b, j in enumerate(idx):
                out[j] = t[b]
        return out

    W = flat([w.contiguous() for w in gen.weights()])
    npool = min(args.steps + args.warmup, 4)
    pool = [flat(gen.grads(t + 1)) for t in range(npool)]
    stream = torch.cuda.current_stream()
    for t in range(args.warmup):
        opt.step(W, pool[t % npool])
    torch.cuda.synchronize()
    if opt.status() != 0:
        raise RuntimeError("device status after warm-up: " + opt.last_error())

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    # timed region: K steps, inputs resident in HBM (state 3 GB >> 129 MB L2)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    opt.profile_begin(1 << 18)
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        # cudaProfilerStart/Stop bracket the timed steps, so that a profiler started with
        # profiling off (ncu --profile-from-start off) records exactly these launches
        torch.cuda.profiler.start()
        start.record(stream)
        for t in range(args.steps):
            opt.step(W, pool[(args.warmup + t) % npool])
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

    # end to end through the public API: pinned host gradients in, updated weights out
    host_g = [[g.cpu().pin_memory() for g in pool[i]] for i in range(npool)]
    host_w = [w.cpu().pin_memory() for w in W]
    dev_g = [torch.empty_like(g) for g in pool[0]]
    h2d = sum(g.numel() * 4 for g in dev_g)
    d2h = sum(w.numel() * 4 for w in W)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    e0.record(stream)
    for t in range(args.steps):
        for d, h in zip(dev_g, host_g[t % npool]):
            d.copy_(h, non_blocking=True)
        opt.step(W, dev_g)
        for h, w in zip(host_w, W):
            h.copy_(w, non_blocking=True)
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

    if rank != 0:
        opt.destroy()
        return
    if muon:
        block_flops = sum(muon_flops(s.rows, s.cols) for s in specs)
    else:
        block_flops = sum(model_flops(s.rows, s.cols, s.left, s.right, args.kl) for s in specs)
    peaks, peak_src = measured_peaks()
    fams = {k: v for k, v in prof.items() if k != "overflow"}
    top = max(fams, key=lambda k: fams[k]["ms"])
    st = fams[top]
    launches = sum(v["launches"] for v in fams.values())
    roof = roofline(top, st, peaks, peak_src, products=1 if muon else TC_PRODUCTS, dtype_ratio=1.0 if muon else 2.0)
    if muon:
        # the DRAM/algorithmic ratios above were measured for the fp32 (tf32 x4) kernels
        roof["traffic"], roof["traffic_note"] = None, "not measured for the bf16 kernel"
    per, sps, threads, scale = muon_oracle_sample() if muon else oracle_sample(1, 0, args.kl)
    lib_line = None
    if not (muon or args.kl or layerwise or subset):
        lib_v, lib_note = library_sample(specs, pool, dev)
        lib_line = {"value": lib_v, "unit": "steps/s", "kind": "torch + cuSOLVER", "sample": lib_note}
    tc_peak = peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"]) / (1.0 if muon else 2.0 * TC_PRODUCTS)
    line = {
        "metric": MUON_METRIC if muon else METRIC, "value": value, "unit": "steps/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * elapsed / args.steps,
        "higher_is_better": True, "scaling": "strong" if layerwise else "weak", "vs_baseline": None,
        "dtype": "bf16" if muon else "f32",
        "data": "synthetic",
        "config": {"workload": WORKLOAD if not subset else f"{WORKLOAD}[matrices {args.matrices}]",
                   "matrices": len(specs),
                   "shapes": "4x 2048x2048, 2x 2048x8192, 1x 8192x2048, all sides preconditioned",
                   "parallelism": f"layerwise{world}" if layerwise else ("replicas" if world > 1 else "single"),
                   "optimizer": "muon (16 quintic Newton-Schulz steps)" if muon else
                   ("soap, KL factor form" if args.kl else "soap, standard factor form"),
                   "l2": "inputs larger than L2 (3 GB of optimizer state per step)"},
        "effective_tflops": block_flops * value / world / 1e12,
        "effective_frac_of_tensor_peak": block_flops * value / world / 1e12 / tc_peak,
        "effective_note": "per GPU (the whole-job FLOP rate divided by the number of GPUs)",
        "model_flop_per_step": block_flops,
        "roofline": roof,
        "kernel_time_share": {k: round(v["ms"] / max(1e-9, sum(x["ms"] for x in fams.values())), 4)
                              for k, v in fams.items()},
        "kernel_families": {k: {"ms_per_step": v["ms"] / args.steps, "launches_per_step": v["launches"] / args.steps,
                                "tflops": v["flops"] / max(1e-12, v["ms"] / 1e3) / 1e12,
                                "gbs": v["bytes"] / max(1e-12, v["ms"] / 1e3) / 1e9}
                            for k, v in fams.items() if v["launches"]},
        "cpu_baseline": {"value": sps, "unit": "steps/s", "cores": threads, "kind": "oracle",
                         "sample": f"one fp64 oracle {'Muon' if muon else 'SOAP'} step of Wq (2048x2048) took "
                                   f"{per:.1f} s; whole block = {scale:.1f}x that by the FLOP model"},
        "e2e": {"value": units * args.steps / e2e_s, "unit": "steps/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches,
        "clocks": clk.summary(),
        "library_baseline": lib_line,
    }
    print(json.dumps(line), flush=True)
    opt.destroy()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["soap", "reference"], default="soap")
    ap.add_argument("--matrices", default="",
                    help="comma-separated matrix indices of the block to run (a smaller case for profiling); "
                         "default: all 7")
    ap.add_argument("--optimizer", choices=["soap", "muon"], default="soap",
                    help="muon: the paper's Muon step on the same block (a separate line, not the headline)")
    ap.add_argument("--layerwise", action="store_true",
                    help="with N > 1: one model, each rank stepping its own matrices (section 6) and "
                         "all-gathering the updated weights over NCCL (strong scaling)")
    ap.add_argument("--kl", action="store_true",
                    help="KL-Shampoo factor form (Alg. 1's factor accumulation) instead of the standard EMAs")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_soap(args)


if __name__ == "__main__":
    main()
